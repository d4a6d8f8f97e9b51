// generate.cu -- syn_generate kernels: seeded synthesis of isolated test data
// (CUDA-Harness Sec. 4.2.1), sm_103a.
//
//   gen_kernel    persistent, one contiguous slice of weighted work units per
//                 CTA; per 4-element quantum: base values, special values,
//                 then the clean output and (after the element-wise
//                 perturbation) the perturbed twin, as 16-byte stores.
//   fixup_kernel  one thread per exact-count edit (or swapped pair).
//   dot_kernel    persistent; 64 x 128 output tiles of the dot-like values,
//                 factors streamed through shared memory by cp.async; same
//                 epilogue per quantum.
//
// Bound: HBM writes for cheap maps; the Philox/Box-Muller ALU work for
// normals; FP32 FMA for the dot-like values.
#include <algorithm>

#include "sv_device.cuh"
#include "sv_kernels.h"

namespace sv {

struct GenParams {
  const DevSpec* tab;  // device table, or nullptr: use inl
  DevSpec inl[SV_INLINE_ENTRIES];
  int n;
  uint64_t total;  // weighted units (gen) or edits (fixup)
  uint64_t chunk;  // units per CTA (gen)
  uint8_t* arena;
};

__device__ __forceinline__ const DevSpec* entry(const GenParams& p, int i) { return p.tab ? p.tab + i : p.inl + i; }

// last entry whose first fixup edit is <= t (entries with no edits share their
// successor's start, so this lands on the entry owning t)
__device__ int find_fix_entry(const GenParams& p, uint64_t t) {
  int lo = 0, hi = p.n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    const uint64_t b = entry(p, mid)->fix_begin;
    if (b <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// stage one table entry in shared memory (all threads take part)
__device__ __forceinline__ void stage_entry(const DevSpec* src, DevSpec* dst) {
  static_assert(sizeof(DevSpec) % 4 == 0, "DevSpec is copied as words");
  const uint32_t* s = reinterpret_cast<const uint32_t*>(src);
  uint32_t* d = reinterpret_cast<uint32_t*>(dst);
  for (int i = threadIdx.x; i < (int)(sizeof(DevSpec) / 4); i += blockDim.x) d[i] = s[i];
}

template <int DT>
__device__ __forceinline__ void store4(uint8_t* base, uint64_t i, const typename Store<DT>::T v[4], uint32_t valid) {
  if constexpr (elem_bytes(DT) == 4) {
    uint32_t* p = reinterpret_cast<uint32_t*>(base) + i;
    if (valid == 4) *reinterpret_cast<uint4*>(p) = make_uint4(v[0], v[1], v[2], v[3]);
    else for (uint32_t j = 0; j < valid; ++j) p[j] = v[j];
  } else if constexpr (elem_bytes(DT) == 2) {
    uint16_t* p = reinterpret_cast<uint16_t*>(base) + i;
    if (valid == 4) *reinterpret_cast<uint2*>(p) = make_uint2(v[0] | (v[1] << 16), v[2] | (v[3] << 16));
    else for (uint32_t j = 0; j < valid; ++j) p[j] = (uint16_t)v[j];
  } else {
    uint64_t* p = reinterpret_cast<uint64_t*>(base) + i;
    if (valid == 4 && (reinterpret_cast<uintptr_t>(p) & 31) == 0) {
      // one 256-bit store: a warp writes 1 KiB contiguously in one instruction
      // (two 128-bit stores would each cover every other 16 bytes of it)
      asm volatile("st.global.v4.u64 [%0], {%1, %2, %3, %4};" ::"l"(p), "l"(v[0]), "l"(v[1]), "l"(v[2]), "l"(v[3])
                   : "memory");
    } else if (valid == 4) {
      reinterpret_cast<ulonglong2*>(p)[0] = make_ulonglong2(v[0], v[1]);
      reinterpret_cast<ulonglong2*>(p)[1] = make_ulonglong2(v[2], v[3]);
    } else {
      for (uint32_t j = 0; j < valid; ++j) p[j] = v[j];
    }
  }
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// one quantum (QB bytes: 8, 16 or 32) from global to shared memory by cp.async;
// both addresses aligned to min(QB, 16)
template <int QB>
__device__ __forceinline__ void copy_quantum_async(uint8_t* dst, const uint8_t* src) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  if constexpr (QB == 8) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(d), "l"(src) : "memory");
  } else if constexpr (QB == 16) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src) : "memory");
  } else {
    static_assert(QB == 32, "quantum bytes");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src) : "memory");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d + 16), "l"(src + 16) : "memory");
  }
}

// the four elements of a quantum from its bytes (in shared memory)
template <int DT>
__device__ __forceinline__ void unpack_quantum(const uint8_t* p, typename Store<DT>::T v[4]) {
  using T = typename Store<DT>::T;
  if constexpr (elem_bytes(DT) == 4) {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    v[0] = (T)w.x, v[1] = (T)w.y, v[2] = (T)w.z, v[3] = (T)w.w;
  } else if constexpr (elem_bytes(DT) == 2) {
    const uint2 w = *reinterpret_cast<const uint2*>(p);
    v[0] = (T)(w.x & 0xFFFFu), v[1] = (T)(w.x >> 16), v[2] = (T)(w.y & 0xFFFFu), v[3] = (T)(w.y >> 16);
  } else {
    const ulonglong2 a = reinterpret_cast<const ulonglong2*>(p)[0], b = reinterpret_cast<const ulonglong2*>(p)[1];
    v[0] = (T)a.x, v[1] = (T)a.y, v[2] = (T)b.x, v[3] = (T)b.y;
  }
}

#ifndef SV_GEN_MINB
#define SV_GEN_MINB 2  // resident CTAs per SM the register budget must allow
#endif
#ifndef SV_ARENA_RING_BYTES
#define SV_ARENA_RING_BYTES 64  // shared-memory ring bytes per thread for arena-source quanta
#endif
#ifndef SV_GEN_PIPELINE
#define SV_GEN_PIPELINE 1  // draw the next iteration's VALUE blocks before this iteration's maps (0: after)
#endif

// ---------------------------------------------------------------------------
// exact-count perturbations: the index of stratum st of [0, N) cut into k
// strata is drawn on the INDEX purpose of the perturbation's stream
// (stratum_index); a COUNT edit sets or offsets the candidate value there,
// SWAP_PAIRS exchanges the candidate values of strata 2j and 2j + 1.
// ---------------------------------------------------------------------------
// candidate bits at g after a COUNT_SET / COUNT_ADD edit
template <int DT, int DIST>
__device__ uint64_t count_edit_bits(const Ctx& c, const sv_perturb& pc, uint64_t g) {
  const uint64_t v2 = value_at<DT, DIST>(c, g, 1);
  if constexpr (is_float(DT)) {
    const float f = __double2float_rn(pc.value);
    if (pc.kind == SV_PERT_COUNT_SET) return from_f32<DT>(f);
    const uint32_t b = (uint32_t)v2;
    return finite_bits<DT>(b) ? from_f32<DT>(__fadd_rn(to_f32<DT>(b), f)) : from_f32<DT>(f);
  } else {
    return pc.kind == SV_PERT_COUNT_SET ? ((uint64_t)pc.ivalue & width_mask(DT))
                                        : ((v2 + (uint64_t)pc.ivalue) & width_mask(DT));
  }
}

// the edits of the strata that meet logical range [g0, g1), which this CTA
// has just generated: thread t < m takes stratum sf + t and overwrites the
// candidate element if the stratum's index falls in the range (m <=
// kMaxFusedEdits, which the host guarantees for fused specs).  The caller's
// __syncthreads() orders these stores after the CTA's own generating stores;
// no other CTA writes [g0, g1).  The values equal what the fixup kernel writes.
template <int DT, int DIST>
__device__ __noinline__ void fused_edits(const Ctx& c, const syn_spec& s, uint64_t g0, uint64_t g1, uint8_t* arena) {
  using T = typename Store<DT>::T;
  const sv_perturb& pc = s.pcount;
  const uint64_t k = fix_strata(s);
  const uint64_t sf = stratum_of(g0, k, c.N), sl = stratum_of(g1 - 1, k, c.N);
  const uint64_t m = umin(sl - sf + 1, kMaxFusedEdits);
  if (threadIdx.x >= m) return;
  const uint64_t st = sf + threadIdx.x;
  const uint64_t g = stratum_index(c, pc.stream, P_INDEX, k, st);
  if (g < g0 || g >= g1) return;
  const uint64_t bits = pc.kind == SV_PERT_SWAP_PAIRS
                            ? value_at<DT, DIST>(c, stratum_index(c, pc.stream, P_INDEX, k, st ^ 1), 1)
                            : count_edit_bits<DT, DIST>(c, pc, g);
  uint8_t* cand = arena + s.cand_offset;
  if constexpr (elem_bytes(DT) == 2) reinterpret_cast<uint16_t*>(cand)[g - s.elem_offset] = (uint16_t)bits;
  else reinterpret_cast<T*>(cand)[g - s.elem_offset] = (T)bits;
}

// one element of a spec's output, index i of the output (not the logical index)
template <int DT>
__device__ __forceinline__ void put_elem(uint8_t* out, uint64_t i, uint64_t bits) {
  using T = typename Store<DT>::T;
  if constexpr (elem_bytes(DT) == 2) reinterpret_cast<uint16_t*>(out)[i] = (uint16_t)bits;
  else reinterpret_cast<T*>(out)[i] = (T)bits;
}

// the candidate's final bits at logical index g: the exact-count edit or
// swap when g is one of their indices, else the value after the element-wise
// perturbation (what the generator and the edits together leave there)
template <int DT, int DIST>
__device__ uint64_t final_cand_bits(const Ctx& c, const syn_spec& s, uint64_t g) {
  const sv_perturb& pc = s.pcount;
  if (pc.kind == SV_PERT_COUNT_SET || pc.kind == SV_PERT_COUNT_ADD || pc.kind == SV_PERT_SWAP_PAIRS) {
    const uint64_t k = fix_strata(s), st = stratum_of(g, k, c.N);
    if (stratum_index(c, pc.stream, P_INDEX, k, st) == g)
      return pc.kind == SV_PERT_SWAP_PAIRS ? value_at<DT, DIST>(c, stratum_index(c, pc.stream, P_INDEX, k, st ^ 1), 1)
                                           : count_edit_bits<DT, DIST>(c, pc, g);
  }
  return value_at<DT, DIST>(c, g, 1);
}

// exact-count special values in the logical range [g0, g1) that this CTA has
// just generated: thread t takes strata sf + t, sf + t + kThreads, ...; where
// a stratum's drawn index falls in the range, the clean output gets the
// special value and the twin its final value (the element-wise perturbation
// and any exact-count edit applied).  The caller's __syncthreads() orders
// these stores after the CTA's generating stores; no other CTA writes
// [g0, g1).  A range meets about k (g1 - g0) / N strata.
template <int DT, int DIST>
__device__ __noinline__ void exact_specials_pass(const Ctx& c, const syn_spec& s, uint64_t g0, uint64_t g1,
                                                 uint8_t* arena) {
  const uint64_t k = c.sp_k;
  const uint64_t sf = stratum_of(g0, k, c.N), sl = stratum_of(g1 - 1, k, c.N);
  uint8_t* ref = s.ref_offset == SV_NO_OUTPUT ? nullptr : arena + s.ref_offset;
  uint8_t* cand = s.cand_offset == SV_NO_OUTPUT ? nullptr : arena + s.cand_offset;
  for (uint64_t st = sf + threadIdx.x; st <= sl; st += kThreads) {
    const uint64_t g = stratum_index(c, c.stream, P_SPECIAL_SEL, k, st);
    if (g < g0 || g >= g1) continue;
    if (ref) put_elem<DT>(ref, g - s.elem_offset, value_at<DT, DIST>(c, g, 0));
    if (cand) put_elem<DT>(cand, g - s.elem_offset, final_cand_bits<DT, DIST>(c, s, g));
  }
}

// base values and special values of the quantum g .. g+3
template <int DT, int DIST>
__device__ __forceinline__ void gen_quantum(const Ctx& c, const Ctx& cold, uint64_t g, typename Store<DT>::T v[4]) {
  if (one_block_dist<DT, DIST>() && c.sp_thr) {
    // the quantum's VALUE and SPECIAL_SEL blocks as two interleaved chains
    const uint64_t blk = g >> 2;
    uint4 wv = make_uint4((uint32_t)blk, (uint32_t)(blk >> 32), c.stream, P_VALUE);
    uint4 ws = make_uint4((uint32_t)blk, (uint32_t)(blk >> 32), c.stream, P_SPECIAL_SEL);
    philox2_rk(wv, ws, c.rk);
    base4_words<DT, DIST>(c, wv, v);
    specials4_words<DT, DIST>(c, cold, g, ws, v);
  } else {
    base4<DT, DIST>(c, g, v);
    if (c.sp_thr) specials4<DT, DIST>(c, cold, g, v);
  }
}

// the clean output and, after the element-wise perturbation, the twin
template <int DT>
__device__ __forceinline__ void store_quantum(const Ctx& c, const Ctx& cold, uint8_t* ref, uint8_t* cand, uint64_t g,
                                              uint64_t i, typename Store<DT>::T v[4], uint32_t valid) {
  if (ref) store4<DT>(ref, i, v, valid);
  if (cand) {
    if (c.pe_kind != SV_PERT_NONE) pelem4<DT>(c, cold, g, v);
    store4<DT>(cand, i, v, valid);
  }
}

// elements [i0, i1) of one spec, by 4-element quanta spread over the CTA:
// the full quanta in a loop with no per-quantum bounds, then at most one
// ragged last quantum.  `cold` is the spec's context in shared memory; the
// hot fields are copied to registers.
template <int DT, int DIST>
__device__ void gen_run(const Ctx& cold, const syn_spec& s, uint64_t i0, uint64_t i1, uint8_t* arena) {
  using T = typename Store<DT>::T;
  const Ctx c = cold;
  uint8_t* ref = s.ref_offset == SV_NO_OUTPUT ? nullptr : arena + s.ref_offset;
  uint8_t* cand = s.cand_offset == SV_NO_OUTPUT ? nullptr : arena + s.cand_offset;
  const uint64_t eo = s.elem_offset, n = s.n;
  const uint64_t q0 = i0 >> 2, q1 = (i1 + 3) >> 2, qfull = umin(q1, n >> 2);
  uint64_t q = q0 + threadIdx.x;
  if constexpr (DIST == SV_FROM_ARENA) {
    // values read from memory, two quanta per iteration: their relative noise
    // (the usual perturbation of such twins) runs as two interleaved chains.
    // The source quanta of the next kArenaAhead iterations are in flight as
    // cp.async copies into this thread's own slots of a shared-memory ring (no
    // registers held across the arithmetic, no barrier: a thread reads only
    // what it copied); iteration i waits for its own copies, reads them, and
    // after its arithmetic refills its slot with iteration i + kArenaAhead.
    constexpr int QB = 4 * elem_bytes(DT);  // bytes of a quantum
    constexpr int kArenaAhead = SV_ARENA_RING_BYTES / (2 * QB) > 0 ? SV_ARENA_RING_BYTES / (2 * QB) : 1;
    __shared__ __align__(16) uint8_t ring[kArenaAhead * 2 * kThreads * QB];
    const uint8_t* src = reinterpret_cast<const uint8_t*>(c.A) + eo * elem_bytes(DT);  // 16-byte aligned; quanta on QB
    const int tid = (int)threadIdx.x;
    auto slot_of = [&](uint64_t it, int k) { return ring + (((int)(it % kArenaAhead) * 2 + k) * kThreads + tid) * QB; };
    auto fill = [&](uint64_t it, uint64_t qi) {  // the two quanta of iteration it (qi: its first)
      if (qi < qfull) copy_quantum_async<QB>(slot_of(it, 0), src + (qi << 2) * elem_bytes(DT));
      if (qi + kThreads < qfull) copy_quantum_async<QB>(slot_of(it, 1), src + ((qi + kThreads) << 2) * elem_bytes(DT));
      cp_async_commit();  // one group per iteration, empty past the end: uniform counting
    };
#pragma unroll
    for (int a = 0; a < kArenaAhead; ++a) fill((uint64_t)a, q + 2ull * kThreads * a);
    for (uint64_t it = 0; q < qfull; q += 2ull * kThreads, ++it) {
      const uint64_t q2 = q + kThreads, ia = q << 2, ib = q2 << 2;
      const bool two = q2 < qfull;
      cp_async_wait<kArenaAhead - 1>();  // this thread's copies of iteration it have landed
      T va[4], vb[4];
      unpack_quantum<DT>(slot_of(it, 0), va);
      if (two) unpack_quantum<DT>(slot_of(it, 1), vb);
      if (c.sp_thr) {
        specials4<DT, DIST>(c, cold, eo + ia, va);
        if (two) specials4<DT, DIST>(c, cold, eo + ib, vb);
      }
      bool done = false;
      if constexpr (is_float(DT)) {
        if (two && cand && c.pe_kind == SV_PERT_REL_NOISE) {
          if (ref) {
            store4<DT>(ref, ia, va, 4);
            store4<DT>(ref, ib, vb, 4);
          }
          rel_noise4x2<DT>(c, eo + ia, va, eo + ib, vb);
          store4<DT>(cand, ia, va, 4);
          store4<DT>(cand, ib, vb, 4);
          done = true;
        }
      }
      if (!done) {
        store_quantum<DT>(c, cold, ref, cand, eo + ia, ia, va, 4);
        if (two) store_quantum<DT>(c, cold, ref, cand, eo + ib, ib, vb, 4);
      }
      fill(it + kArenaAhead, q + 2ull * kThreads * kArenaAhead);  // the slot's values are consumed
    }
    cp_async_wait<0>();
  } else {
    if constexpr (one_block_dist<DT, DIST>()) {
      if (!c.sp_thr) {
        // no per-element special selection (none, or the exact mode): one
        // VALUE block per quantum, so two quanta per iteration keep two
        // independent Philox chains in flight
#if SV_GEN_PIPELINE
        // and the next iteration's blocks are drawn before this iteration's
        // value maps, so the multiply-bound Philox rounds and the
        // issue-bound maps interleave (the last iteration's look-ahead draw
        // is for counters past the range: computed, never stored)
        const uint64_t b0 = (eo >> 2) + q;
        uint4 wa = make_uint4((uint32_t)b0, (uint32_t)(b0 >> 32), c.stream, P_VALUE);
        uint4 wb = make_uint4((uint32_t)(b0 + kThreads), (uint32_t)((b0 + kThreads) >> 32), c.stream, P_VALUE);
        philox2_rk(wa, wb, c.rk);
        for (; q + kThreads < qfull; q += 2ull * kThreads) {
          const uint64_t ia = q << 2, ib = (q + kThreads) << 2;
          const uint64_t bn = (eo >> 2) + q + 2ull * kThreads;
          uint4 na = make_uint4((uint32_t)bn, (uint32_t)(bn >> 32), c.stream, P_VALUE);
          uint4 nb = make_uint4((uint32_t)(bn + kThreads), (uint32_t)((bn + kThreads) >> 32), c.stream, P_VALUE);
          philox2_rk(na, nb, c.rk);
          T va[4], vb[4];
          base4_words<DT, DIST>(c, wa, va);
          base4_words<DT, DIST>(c, wb, vb);
          store_quantum<DT>(c, cold, ref, cand, eo + ia, ia, va, 4);
          store_quantum<DT>(c, cold, ref, cand, eo + ib, ib, vb, 4);
          wa = na;
          wb = nb;
        }
#else
        for (; q + kThreads < qfull; q += 2ull * kThreads) {
          const uint64_t ia = q << 2, ib = (q + kThreads) << 2;
          const uint64_t ba = (eo + ia) >> 2, bb = (eo + ib) >> 2;
          uint4 wa = make_uint4((uint32_t)ba, (uint32_t)(ba >> 32), c.stream, P_VALUE);
          uint4 wb = make_uint4((uint32_t)bb, (uint32_t)(bb >> 32), c.stream, P_VALUE);
          philox2_rk(wa, wb, c.rk);
          T va[4], vb[4];
          base4_words<DT, DIST>(c, wa, va);
          base4_words<DT, DIST>(c, wb, vb);
          store_quantum<DT>(c, cold, ref, cand, eo + ia, ia, va, 4);
          store_quantum<DT>(c, cold, ref, cand, eo + ib, ib, vb, 4);
        }
#endif
      }
    }
    for (; q < qfull; q += kThreads) {
      T v[4];
      const uint64_t i = q << 2;
      gen_quantum<DT, DIST>(c, cold, eo + i, v);
      store_quantum<DT>(c, cold, ref, cand, eo + i, i, v, 4);
    }
  }
  // the spec's last quantum, with n % 4 elements, goes to the thread whose
  // stride it falls on (q1 - 1 = n / 4 when it exists)
  if (q1 > qfull && (q1 - 1 - q0) % kThreads == threadIdx.x) {
    T v[4];
    const uint64_t i = (q1 - 1) << 2;
    gen_quantum<DT, DIST>(c, cold, eo + i, v);
    store_quantum<DT>(c, cold, ref, cand, eo + i, i, v, (uint32_t)(n - i));
  }
}

#define SV_COMBO(dt, dist) ((dt) * 8 + (dist))

// one instantiation per dtype x distribution; the host groups the specs so
// that a launch only sees its own kind
template <int DT, int DIST>
__global__ void __launch_bounds__(kThreads, SV_GEN_MINB) gen_kernel(const __grid_constant__ GenParams p) {
  pdl_wait();
  pdl_trigger();
  // two slots for the entry in use and its context: an entry is staged into
  // the slot its predecessor did not use, so one barrier per entry suffices
  // (a slot's previous user is two entries back, which every thread finished
  // before passing the last entry's barrier)
  __shared__ DevSpec cur[2];
  __shared__ Ctx ctx[2];
  __shared__ uint64_t staged[kStagedStarts];
  const uint64_t u0 = (uint64_t)blockIdx.x * p.chunk;
  const uint64_t u1 = umin(u0 + p.chunk, p.total);
  if (u0 >= u1) return;
  int slot = 0;
  for (int e = find_start(entry(p, 0), p.n, u0, staged); e < p.n; ++e) {
    // the entry's place in the units, read from the table by every thread
    const DevSpec* te = entry(p, e);
    const uint64_t wb = te->work_begin;
    if (wb >= u1) break;
    // this entry's quanta occupy units [wb + overhead, wb + gen_units)
    const uint64_t q_base = wb + kGenEntryUnits;
    const uint64_t lo = umax(u0, q_base), hi = umin(u1, wb + gen_units(te->s));
    if (hi <= lo) continue;
    stage_entry(te, &cur[slot]);
    if (threadIdx.x == 0) ctx[slot] = make_ctx(te->s, p.arena);
    __syncthreads();
    const DevSpec& d = cur[slot];
    const Ctx& cx = ctx[slot];
    const uint64_t i0 = (lo - q_base) * 4, i1 = umin((hi - q_base) * 4, d.s.n);
    gen_run<DT, DIST>(cx, d.s, i0, i1, p.arena);
    if (cx.sp_k) {  // exact-count special values inside this CTA's range
      __syncthreads();
      exact_specials_pass<DT, DIST>(cx, d.s, d.s.elem_offset + i0, d.s.elem_offset + i1, p.arena);
    }
    if (d.fused) {  // uniform: the spec's exact-count edits inside this CTA's range
      __syncthreads();
      fused_edits<DT, DIST>(cx, d.s, d.s.elem_offset + i0, d.s.elem_offset + i1, p.arena);
    }
    slot ^= 1;
  }
}

// every (dtype, distribution) the streaming generator handles
#define SV_GEN_COMBOS(X)                                                                        \
  X(SV_F32, SV_UNIFORM) X(SV_F32, SV_NORMAL) X(SV_F32, SV_RAW_BITS) X(SV_F32, SV_CONSTANT)         \
  X(SV_F16, SV_UNIFORM) X(SV_F16, SV_NORMAL) X(SV_F16, SV_RAW_BITS) X(SV_F16, SV_CONSTANT)         \
  X(SV_BF16, SV_UNIFORM) X(SV_BF16, SV_NORMAL) X(SV_BF16, SV_RAW_BITS) X(SV_BF16, SV_CONSTANT)     \
  X(SV_I32, SV_INT_RANGE) X(SV_I32, SV_PERMUTATION) X(SV_I32, SV_RAW_BITS) X(SV_I32, SV_CONSTANT)  \
  X(SV_U32, SV_INT_RANGE) X(SV_U32, SV_PERMUTATION) X(SV_U32, SV_RAW_BITS) X(SV_U32, SV_CONSTANT)  \
  X(SV_I64, SV_INT_RANGE) X(SV_I64, SV_PERMUTATION) X(SV_I64, SV_RAW_BITS) X(SV_I64, SV_CONSTANT)             \
  X(SV_F32, SV_FROM_ARENA) X(SV_F16, SV_FROM_ARENA) X(SV_BF16, SV_FROM_ARENA) X(SV_I32, SV_FROM_ARENA)         \
  X(SV_U32, SV_FROM_ARENA) X(SV_I64, SV_FROM_ARENA)

static const void* gen_kernel_for(uint32_t dtype, uint32_t dist) {
  switch (SV_COMBO(dtype, dist)) {
#define SV_CASE(DT, DIST) \
  case SV_COMBO(DT, DIST): return reinterpret_cast<const void*>(&gen_kernel<DT, DIST>);
    SV_GEN_COMBOS(SV_CASE)
#undef SV_CASE
    default: return nullptr;
  }
}

// ---------------------------------------------------------------------------
// exact-count perturbations: one thread per selected element (per swapped
// pair for SWAP_PAIRS); the index of stratum s of [0, N) cut into k strata is
// floor(s N / k) + mulhi64(x, len), x from INDEX block s.
// ---------------------------------------------------------------------------

template <int DT, int DIST>
__device__ void fix_one(const Ctx& c, const syn_spec& s, uint64_t u, uint8_t* arena) {
  using T = typename Store<DT>::T;
  const uint64_t nsp = fix_special_units(s);
  if (u < nsp) {  // dot-like values: the exact-count special value of stratum u
    const uint64_t g = stratum_index(c, c.stream, P_SPECIAL_SEL, c.sp_k, u);
    if (g < s.elem_offset || g >= s.elem_offset + s.n) return;
    if (s.ref_offset != SV_NO_OUTPUT) put_elem<DT>(arena + s.ref_offset, g - s.elem_offset, value_at<DT, DIST>(c, g, 0));
    if (s.cand_offset != SV_NO_OUTPUT)
      put_elem<DT>(arena + s.cand_offset, g - s.elem_offset, final_cand_bits<DT, DIST>(c, s, g));
    return;
  }
  u -= nsp;
  const sv_perturb& pc = s.pcount;
  uint8_t* cand = arena + s.cand_offset;
  const uint64_t lo = s.elem_offset, hi = s.elem_offset + s.n;
  T* out = reinterpret_cast<T*>(cand);
  auto put = [&](uint64_t g, uint64_t v) {
    if (g < lo || g >= hi) return;
    const uint64_t i = g - lo;
    if constexpr (elem_bytes(DT) == 2) reinterpret_cast<uint16_t*>(cand)[i] = (uint16_t)v;
    else out[i] = (T)v;
  };
  if (pc.kind == SV_PERT_SWAP_PAIRS) {
    const uint64_t k = 2 * pc.count;
    const uint64_t a = stratum_index(c, pc.stream, P_INDEX, k, 2 * u);
    const uint64_t b = stratum_index(c, pc.stream, P_INDEX, k, 2 * u + 1);
    const uint64_t va = value_at<DT, DIST>(c, a, 1), vb = value_at<DT, DIST>(c, b, 1);
    put(a, vb);
    put(b, va);
    return;
  }
  const uint64_t g = stratum_index(c, pc.stream, P_INDEX, pc.count, u);
  if (g < lo || g >= hi) return;
  put(g, count_edit_bits<DT, DIST>(c, pc, g));
}

__device__ void fix_dispatch(const Ctx& c, const syn_spec& s, uint64_t u, uint8_t* arena) {
  switch (SV_COMBO(s.dtype, s.dist)) {
#define SV_CASE(DT, DIST) \
  case SV_COMBO(DT, DIST): fix_one<DT, DIST>(c, s, u, arena); break;
    SV_CASE(SV_F32, SV_UNIFORM) SV_CASE(SV_F32, SV_NORMAL) SV_CASE(SV_F32, SV_RAW_BITS) SV_CASE(SV_F32, SV_CONSTANT)
    SV_CASE(SV_F32, SV_DOTLIKE)
    SV_CASE(SV_F16, SV_UNIFORM) SV_CASE(SV_F16, SV_NORMAL) SV_CASE(SV_F16, SV_RAW_BITS) SV_CASE(SV_F16, SV_CONSTANT)
    SV_CASE(SV_F16, SV_DOTLIKE)
    SV_CASE(SV_BF16, SV_UNIFORM) SV_CASE(SV_BF16, SV_NORMAL) SV_CASE(SV_BF16, SV_RAW_BITS)
    SV_CASE(SV_BF16, SV_CONSTANT) SV_CASE(SV_BF16, SV_DOTLIKE)
    SV_CASE(SV_I32, SV_INT_RANGE) SV_CASE(SV_I32, SV_PERMUTATION) SV_CASE(SV_I32, SV_RAW_BITS)
    SV_CASE(SV_I32, SV_CONSTANT)
    SV_CASE(SV_U32, SV_INT_RANGE) SV_CASE(SV_U32, SV_PERMUTATION) SV_CASE(SV_U32, SV_RAW_BITS)
    SV_CASE(SV_U32, SV_CONSTANT)
    SV_CASE(SV_I64, SV_INT_RANGE) SV_CASE(SV_I64, SV_PERMUTATION) SV_CASE(SV_I64, SV_RAW_BITS)
    SV_CASE(SV_I64, SV_CONSTANT)
    SV_CASE(SV_F32, SV_FROM_ARENA) SV_CASE(SV_F16, SV_FROM_ARENA) SV_CASE(SV_BF16, SV_FROM_ARENA)
    SV_CASE(SV_I32, SV_FROM_ARENA) SV_CASE(SV_U32, SV_FROM_ARENA) SV_CASE(SV_I64, SV_FROM_ARENA)
#undef SV_CASE
    default: break;
  }
}

__global__ void __launch_bounds__(kThreads) fixup_kernel(const __grid_constant__ GenParams p) {
  pdl_wait();
  pdl_trigger();
  const uint64_t u = (uint64_t)blockIdx.x * kThreads + threadIdx.x;
  if (u >= p.total) return;
  const DevSpec* e = entry(p, find_fix_entry(p, u));
  const syn_spec s = e->s;
  const Ctx c = make_ctx(s, p.arena);
  fix_dispatch(c, s, u - e->fix_begin, p.arena);
}

// ---------------------------------------------------------------------------
// dot-like values: persistent CTAs, each a contiguous run of 64 x 128 output
// tiles (row-block major, so consecutive tiles share their A rows).  The
// factors stream through a ring of kDotStages shared-memory slots, one
// kDotK-deep k chunk of A (64 rows x kDotK, row-major) and B (kDotK x 128) per
// slot (64 deep, 2 slots: a whole K = 64 tile per slot, one barrier per tile),
// filled by cp.async while earlier chunks are multiplied; every output is the
// k-ascending chain of fused multiply-adds over exactly its K steps.  Thread
// layout: warp w owns rows 8w..8w+7 of the tile, lane l columns 4l..4l+3 (one
// quantum per row), so a warp's A reads are broadcasts and its B reads and
// output stores are contiguous.
// ---------------------------------------------------------------------------
#ifndef SV_DOT_STAGES
#define SV_DOT_STAGES 2
#endif
#ifndef SV_DOT_MINB
#define SV_DOT_MINB 2
#endif
#ifndef SV_DOT_THREADS
#define SV_DOT_THREADS 256  // threads per CTA: one warp per 8 rows of the tile
#endif
#ifndef SV_DOT_K
#define SV_DOT_K 64  // k depth of one shared-memory slot (a multiple of 16)
#endif
constexpr int kDotThreads = SV_DOT_THREADS;
constexpr int kDotRows = kDotThreads / 32 * 8, kDotCols = 128, kDotK = SV_DOT_K, kDotStages = SV_DOT_STAGES;
static_assert(kDotThreads % 32 == 0 && kDotK % 16 == 0, "dot-like tile shape");
// every thread issues the same number of copies and together they cover a slot
static_assert(kDotThreads % (kDotK / 4) == 0 && (kDotRows * kDotK / 4) % kDotThreads == 0 &&
                  kDotThreads % kDotK == 0 && (kDotK * kDotCols / 4) % kDotThreads == 0,
              "dot-like slot copies");
constexpr int kDotSlotFloats = kDotRows * kDotK + kDotK * kDotCols;
constexpr size_t kDotSmem = (size_t)kDotStages * kDotSlotFloats * sizeof(float);

struct DotParams {
  DevSpec spec;
  uint8_t* arena;
  uint64_t row0;   // first row of the chunk
  uint64_t tiles;  // row blocks x column blocks
  uint32_t n_cb;   // column blocks
};

__device__ __forceinline__ void cp_async16(float* dst, const float* src, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 4 : 0) : "memory");
}

// position in a CTA's run of (tile, k chunk) steps, advanced without division
struct DotCursor {
  uint64_t rb, cb, kc;  // row block (relative to row0), column block, first k of the chunk
  __device__ __forceinline__ void advance(uint64_t K, uint32_t n_cb) {
    kc += kDotK;
    if (kc >= K) {
      kc = 0;
      if (++cb == n_cb) cb = 0, ++rb;
    }
  }
};

// A16: the A rows are 16-byte aligned (K % 4 == 0) and move in 16-byte pieces
template <int DT, bool A16>
__global__ void __launch_bounds__(kDotThreads, SV_DOT_MINB) dot_kernel(const __grid_constant__ DotParams p) {
  using T = typename Store<DT>::T;
  extern __shared__ __align__(128) float dsm[];
  __shared__ Ctx cold;
  const syn_spec& s = p.spec.s;
  if (threadIdx.x == 0) cold = make_ctx(s, p.arena);
  __syncthreads();
  const Ctx c = cold;
  const uint64_t rows = s.rows, cols = s.cols, K = s.dot_k;
  const int tid = threadIdx.x, cg = tid & 31, rg = tid >> 5;
  const uint64_t t_begin = p.tiles * blockIdx.x / gridDim.x, t_end = p.tiles * (blockIdx.x + 1) / gridDim.x;
  const uint64_t nk = (K + kDotK - 1) / kDotK;
  const uint64_t steps = (t_end - t_begin) * nk;
  const DotCursor first{t_begin / p.n_cb, t_begin % p.n_cb, 0};

  // step i of this CTA goes to slot i % kDotStages; the copy of step i is
  // issued at iteration i - (kDotStages - 1), so `ic` runs that far ahead
  DotCursor ic = first;
  uint64_t issued = 0;
  uint32_t islot = 0;
  auto issue = [&]() {
    if (issued < steps) {
      const uint64_t r0 = p.row0 + ic.rb * kDotRows, c0 = ic.cb * kDotCols, kc = ic.kc;
      float* As = dsm + islot * kDotSlotFloats;
      float* Bs = As + kDotRows * kDotK;
      if constexpr (A16) {
#pragma unroll
        for (int it = 0; it < kDotRows * kDotK / 4 / kDotThreads; ++it) {
          const int r = tid / (kDotK / 4) + it * (kDotThreads / (kDotK / 4)), q = tid % (kDotK / 4);
          const uint64_t gr = r0 + r, gk = kc + 4 * q;
          const bool ok = gr < rows && gk < K;  // K % 4 == 0: the whole piece is in range
          cp_async16(As + r * kDotK + 4 * q, ok ? c.A + gr * K + gk : c.A, ok);
        }
      } else {
#pragma unroll
        for (int it = 0; it < kDotRows * kDotK / kDotThreads; ++it) {
          const int r = tid / kDotK + it * (kDotThreads / kDotK), k = tid % kDotK;
          const uint64_t gr = r0 + r, gk = kc + k;
          const bool ok = gr < rows && gk < K;
          cp_async4(As + r * kDotK + k, ok ? c.A + gr * K + gk : c.A, ok);
        }
      }
#pragma unroll
      for (int it = 0; it < kDotK * kDotCols / 4 / kDotThreads; ++it) {
        const int k = (tid >> 5) + it * (kDotThreads / 32), q = tid & 31;
        const uint64_t gk = kc + k, gc = c0 + 4 * q;
        const bool ok = gk < K && gc < cols;  // cols % 4 == 0
        cp_async16(Bs + k * kDotCols + 4 * q, ok ? c.B + gk * cols + gc : c.B, ok);
      }
      ic.advance(K, p.n_cb);
      ++issued;
      islot = islot + 1 == kDotStages ? 0 : islot + 1;
    }
    cp_async_commit();  // one group per step, empty past the end: uniform counting
  };

  for (int i = 0; i < kDotStages - 1; ++i) issue();

  uint8_t* ref = s.ref_offset == SV_NO_OUTPUT ? nullptr : p.arena + s.ref_offset;
  uint8_t* cand = s.cand_offset == SV_NO_OUTPUT ? nullptr : p.arena + s.cand_offset;
  const uint64_t lo = s.elem_offset, hi = s.elem_offset + s.n;
  float acc[8][4];
#pragma unroll
  for (int r = 0; r < 8; ++r)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[r][j] = 0.0f;

  DotCursor cc = first;
  uint32_t cslot = 0;
  for (uint64_t i = 0; i < steps; ++i) {
    cp_async_wait<kDotStages - 2>();
    __syncthreads();  // chunk i landed for every thread; slot (i - 1) % kDotStages is free
    issue();
    const float* As = dsm + cslot * kDotSlotFloats + (8 * rg) * kDotK;
    const float* Bs = dsm + cslot * kDotSlotFloats + kDotRows * kDotK + 4 * cg;
    cslot = cslot + 1 == kDotStages ? 0 : cslot + 1;
    const int kn = (int)umin(kDotK, K - cc.kc);
    int k = 0;
    for (; k + 4 <= kn; k += 4) {
      float4 a[8], b[4];
#pragma unroll
      for (int r = 0; r < 8; ++r) a[r] = *reinterpret_cast<const float4*>(As + r * kDotK + k);
#pragma unroll
      for (int q = 0; q < 4; ++q) b[q] = *reinterpret_cast<const float4*>(Bs + (k + q) * kDotCols);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
#pragma unroll
        for (int r = 0; r < 8; ++r) {
          const float ar = q == 0 ? a[r].x : q == 1 ? a[r].y : q == 2 ? a[r].z : a[r].w;
          acc[r][0] = __fmaf_rn(ar, b[q].x, acc[r][0]);
          acc[r][1] = __fmaf_rn(ar, b[q].y, acc[r][1]);
          acc[r][2] = __fmaf_rn(ar, b[q].z, acc[r][2]);
          acc[r][3] = __fmaf_rn(ar, b[q].w, acc[r][3]);
        }
      }
    }
    for (; k < kn; ++k) {  // K % 4 != 0: exactly the remaining steps, no zero padding
      const float4 b = *reinterpret_cast<const float4*>(Bs + k * kDotCols);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const float ar = As[r * kDotK + k];
        acc[r][0] = __fmaf_rn(ar, b.x, acc[r][0]);
        acc[r][1] = __fmaf_rn(ar, b.y, acc[r][1]);
        acc[r][2] = __fmaf_rn(ar, b.z, acc[r][2]);
        acc[r][3] = __fmaf_rn(ar, b.w, acc[r][3]);
      }
    }
    const DotCursor at = cc;
    cc.advance(K, p.n_cb);
    if (cc.kc != 0) continue;  // the tile has more k chunks

    // epilogue of the tile: rounding, specials, clean store, perturbation, twin store
    const uint64_t r0 = p.row0 + at.rb * kDotRows, col = at.cb * kDotCols + 4 * cg;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const uint64_t row = r0 + 8 * rg + r;
      const uint64_t g = row * cols + col;  // multiple of 4 (cols % 4 == 0)
      if (col < cols && row < rows && g + 4 > lo && g < hi) {
        T v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] = (T)from_f32<DT>(acc[r][j]);
        if (c.sp_thr) specials4<DT, SV_DOTLIKE>(c, cold, g, v);
        // chunk bounds fall on quanta (elem_offset % 4 == 0); n may end mid-quantum
        const uint64_t e = g - lo;
        const uint32_t valid = (uint32_t)umin(4, hi - g);
        if (ref) store4<DT>(ref, e, v, valid);
        if (cand) {
          if (c.pe_kind != SV_PERT_NONE) pelem4<DT>(c, cold, g, v);
          store4<DT>(cand, e, v, valid);
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[r][j] = 0.0f;
    }
  }
  cp_async_wait<0>();
}

// ---------------------------------------------------------------------------
// the Box-Muller step alone, on caller words (syn_box_muller): pair i of
// words gives the two normals the generator makes from the same words.
// Pairs 2j and 2j + 1 go through box_muller4 together, as the generator's
// pairs do; an odd last pair goes through the single-pair box_muller, whose
// values the packed form reproduces bit for bit.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) box_muller_kernel(const uint2* w, uint64_t n_pairs, float2* z) {
  const uint64_t n2 = (n_pairs + 1) / 2;
  for (uint64_t j = (uint64_t)blockIdx.x * kThreads + threadIdx.x; j < n2; j += (uint64_t)gridDim.x * kThreads) {
    const uint64_t i = 2 * j;
    const uint2 a = w[i];
    if (i + 1 < n_pairs) {
      const uint2 b = w[i + 1];
      float v[4];
      box_muller4(make_uint4(a.x, a.y, b.x, b.y), v);
      z[i] = make_float2(v[0], v[1]);
      z[i + 1] = make_float2(v[2], v[3]);
    } else {
      float z0, z1;
      box_muller(a.x, a.y, z0, z1);
      z[i] = make_float2(z0, z1);
    }
  }
}

// ---------------------------------------------------------------------------
// host launchers
// ---------------------------------------------------------------------------
static void fill_params(GenParams& gp, const DevSpec* host, const DevSpec* dev, int n) {
  gp.tab = dev;
  gp.n = n;
  if (!dev)
    for (int i = 0; i < n; ++i) gp.inl[i] = host[i];
}

LaunchShape generate_shape(uint32_t dtype, uint32_t dist, uint64_t units, uint64_t tiles) {
  const void* k = gen_kernel_for(dtype, dist);
  return shape_for(units, tiles, k ? grid_cap_for(k) : 1, (uint64_t)kThreads);
}

cudaError_t launch_generate_group(uint32_t dtype, uint32_t dist, const DevSpec* host, const DevSpec* dev, int n,
                                  uint64_t units, LaunchShape sh, uint8_t* arena, cudaStream_t st) {
  if (units == 0 || n == 0) return cudaSuccess;
  GenParams gp;
  fill_params(gp, host, dev, n);
  gp.total = units;
  gp.chunk = sh.chunk;
  gp.arena = arena;
  cudaError_t e = cudaSuccess;
  switch (SV_COMBO(dtype, dist)) {
#define SV_CASE(DT, DIST) \
  case SV_COMBO(DT, DIST): e = launch_chained(gen_kernel<DT, DIST>, sh.grid, launch_block(), st, gp); break;
    SV_GEN_COMBOS(SV_CASE)
#undef SV_CASE
    default: return cudaErrorInvalidValue;
  }
  count_launch();
  return e;
}

cudaError_t launch_fixup(const DevSpec* host, const DevSpec* dev, int n, uint64_t total_units, uint8_t* arena,
                         cudaStream_t st) {
  if (total_units == 0) return cudaSuccess;
  GenParams gp;
  fill_params(gp, host, dev, n);
  gp.total = total_units;
  gp.chunk = 0;
  gp.arena = arena;
  const uint64_t blocks = (total_units + kThreads - 1) / kThreads;
  const cudaError_t e = launch_chained(fixup_kernel, (unsigned)blocks, launch_block(), st, gp);
  count_launch();
  return e;
}

template <int DT, bool A16>
static cudaError_t launch_dot(const DotParams& dp, uint64_t tiles, cudaStream_t st) {
  const void* fn = reinterpret_cast<const void*>(dot_kernel<DT, A16>);
  const uint32_t cap = grid_cap_for(fn, kDotSmem, kDotThreads);
  const unsigned grid = (unsigned)std::min<uint64_t>(tiles, cap);
  dot_kernel<DT, A16><<<grid, launch_block() ? kDotThreads : 0u, kDotSmem, st>>>(dp);
  count_launch();
  return cudaGetLastError();
}

cudaError_t launch_box_muller(const uint32_t* words, uint64_t n_pairs, float* z, cudaStream_t st) {
  if (n_pairs == 0) return cudaSuccess;
  const void* fn = reinterpret_cast<const void*>(box_muller_kernel);
  const uint64_t blocks = std::min<uint64_t>(((n_pairs + 1) / 2 + kThreads - 1) / kThreads, grid_cap_for(fn));
  box_muller_kernel<<<(unsigned)blocks, launch_block(), 0, st>>>(reinterpret_cast<const uint2*>(words), n_pairs,
                                                            reinterpret_cast<float2*>(z));
  count_launch();
  return cudaGetLastError();
}

cudaError_t launch_dotlike(const DevSpec& spec, uint8_t* arena, cudaStream_t st) {
  const syn_spec& s = spec.s;
  if (s.n == 0) return cudaSuccess;
  DotParams dp;
  dp.spec = spec;
  dp.arena = arena;
  const uint64_t first_row = s.elem_offset / s.cols, last_row = (s.elem_offset + s.n - 1) / s.cols;
  dp.row0 = first_row;
  dp.n_cb = (uint32_t)((s.cols + kDotCols - 1) / kDotCols);
  dp.tiles = (last_row - first_row + kDotRows) / kDotRows * dp.n_cb;
  const bool a16 = s.dot_k % 4 == 0;
  switch (s.dtype) {
    case SV_F32: return a16 ? launch_dot<SV_F32, true>(dp, dp.tiles, st) : launch_dot<SV_F32, false>(dp, dp.tiles, st);
    case SV_F16: return a16 ? launch_dot<SV_F16, true>(dp, dp.tiles, st) : launch_dot<SV_F16, false>(dp, dp.tiles, st);
    default: return a16 ? launch_dot<SV_BF16, true>(dp, dp.tiles, st) : launch_dot<SV_BF16, false>(dp, dp.tiles, st);
  }
}

}  // namespace sv
