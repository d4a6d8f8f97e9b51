/*
 * synverify.h -- C ABI of the GB300 (sm_103a) library for the data-parallel
 * path of Synthesis-Based Verification (CUDA-Harness, Sec. 4.2):
 *
 *   syn_generate        seeded synthesis of isolated test data (Sec. 4.2.1)
 *   verify_compare      functional validation, Eq. 1, per segment (Sec. 4.2.1)
 *   verify_progressive  size-ascending stages with fail-fast exit (Sec. 4.2.2)
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Plain C types only.  Device buffers are raw device pointers with a byte
 *   size; spec/pair tables are HOST arrays, read during the call only.
 * - Ownership: the caller owns every buffer.  The library allocates no device
 *   memory.  It keeps two kinds of state between calls: a per-device cache of
 *   the SM count and occupancy, and pinned host staging buffers for entry
 *   tables (allocated on first need, at most 64 buffers of at most 16 MiB,
 *   kept for the life of the process).
 * - Execution: every call enqueues work on `stream` and returns without
 *   waiting; results are written to device memory.  Calls on different streams
 *   are independent when their workspaces and outputs do not overlap.  A table
 *   larger than SV_INLINE_ENTRIES entries is built in a pinned staging buffer
 *   and copied to the workspace with cudaMemcpyAsync; a staging buffer is
 *   reused only after the copy issued from it has completed.  (If no staging
 *   buffer can be had, the table goes from ordinary host memory, and the
 *   driver may then wait for the stream before that copy.)  The generator,
 *   compare and combine kernels are launched as programmatic dependent
 *   launches: one may be scheduled while the previous kernel of the stream
 *   still runs, and it waits on the device for that kernel to complete before
 *   it reads or writes memory, so stream order holds as for plain launches.
 * - Errors: 0 on success, a negative SV_E* status otherwise.  All arguments are
 *   validated on the host before anything is enqueued, so a validation error
 *   leaves device memory untouched.  SV_ECUDA reports a CUDA launch or copy
 *   error (cudaGetLastError after the launches).
 * - Layout: all byte offsets of element data must be multiples of 16; arrays
 *   are dense and little-endian; fp16 is IEEE binary16, bf16 the top half of
 *   an fp32.
 */
#ifndef SYNVERIFY_H
#define SYNVERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SV_ABI_VERSION 1

/* The stream type: identical to cudaStream_t (NULL = legacy default stream). */
typedef struct CUstream_st* sv_stream_t;

/* ---- element types ---- */
enum { SV_F32 = 0, SV_F16 = 1, SV_BF16 = 2, SV_I32 = 3, SV_I64 = 4, SV_U32 = 5 };

/* ---- base value distributions (syn_spec.dist) ----
 * Every random quantity is a Philox-4x32-10 draw (Salmon et al., SC'11) with
 * counter (block lo, block hi, stream, purpose) and key = the 64-bit seed.
 * Element g (its logical index) of a 16/32-bit type uses word g%4 of block
 * g/4; a 64-bit element uses words 2(g%2), 2(g%2)+1 (high, low) of block g/2.
 *   SV_UNIFORM     float types: a + (b-a)*u, u = (w>>8)*2^-24; a=p0, b=p1,
 *                  a, b, b-a rounded to fp32, two fp32 roundings.
 *   SV_NORMAL      float types: mu + sigma*z (p0=mu, p1=sigma, fp32), z by
 *                  Box-Muller on words (w0,w1) -> elements 4b, 4b+1 and
 *                  (w2,w3) -> 4b+2, 4b+3: u1 = ((w0>>8)+1)*2^-24,
 *                  z = sqrt(-2 ln u1) * (cos, sin)(2 pi (w1>>8) 2^-24).
 *                  Computed in fp32 on the GPU (within 4 ulp of fp64).
 *   SV_INT_RANGE   integer types: [i0, i1] by multiply-high of the word (two
 *                  words for i64), no rejection.
 *   SV_PERMUTATION integer types: a keyed bijection of [0, logical_n).
 *   SV_DOTLIKE     float types: element (i, j) of a rows x cols matrix is
 *                  sum_k A[i,k]*B[k,j], k ascending, one fused multiply-add
 *                  per step in fp32, A (rows x dot_k) and B (dot_k x cols)
 *                  fp32 row-major at a_offset / b_offset of the same arena
 *                  (written by an earlier call).  cols % 4 == 0.
 *   SV_RAW_BITS    the words themselves (16-bit types: the word's top half).
 *   SV_CONSTANT    p0 (float types) or i0 (integer types) everywhere.
 *   SV_FROM_ARENA  any type: element g of the existing array of logical_n
 *                  elements of the same type at a_offset of the same arena
 *                  (written earlier; 16-byte aligned; must not overlap this
 *                  spec's outputs).  Special values and perturbations apply
 *                  as to drawn values, so an existing output (a trusted
 *                  reference's, say) gets perturbed twins.
 */
enum {
  SV_UNIFORM = 0, SV_NORMAL = 1, SV_INT_RANGE = 2, SV_PERMUTATION = 3,
  SV_DOTLIKE = 4, SV_RAW_BITS = 5, SV_CONSTANT = 6, SV_FROM_ARENA = 7
};

/* ---- special values (syn_spec.special_mask, OR of these) ----
 * Selection, Bernoulli mode (SV_SP_EXACT clear): element g is special iff
 * its SPECIAL_SEL word is < floor(rate * 2^32).  Exact mode (SV_SP_EXACT
 * set): exactly k = round(rate * N) elements of the logical array of N
 * elements are special (k <= SV_MAX_COUNT, else SV_ERANGE), one per stratum
 * of [0, N) cut into k equal strata, at floor(s N / k) + mulhi64(x, len) for
 * stratum s, x = the first two words of SPECIAL_SEL block s.  The exact mode
 * draws nothing per element, so a generator pass costs one Philox block less
 * per 4-element quantum (a reading of "0.01% injected" as a count; the paper
 * only asks for broad, special-laden inputs, Sec. 4.2.1).
 * Kind, in both modes: the j-th set kind bit of the mask (ascending), j =
 * mulhi(w0, #kinds), from SPECIAL_KIND block g.  NaN is the canonical quiet
 * NaN; DENORM has a random sign and a random nonzero fraction; DUP copies the
 * base value of a uniformly drawn index of the logical array.  Float types
 * take NAN, PINF, NINF, DENORM, ZERO, DUP; integer types ZERO, IMIN, IMAX,
 * DUP.  A mask with no kind bit selects nothing. */
enum {
  SV_SP_NAN = 1u << 0, SV_SP_PINF = 1u << 1, SV_SP_NINF = 1u << 2,
  SV_SP_DENORM = 1u << 3, SV_SP_ZERO = 1u << 4, SV_SP_IMIN = 1u << 5,
  SV_SP_IMAX = 1u << 6, SV_SP_DUP = 1u << 7
};
#define SV_SP_KINDS 0xFFu
#define SV_SP_EXACT (1u << 31)

/* ---- candidate perturbations ----
 * Element-wise kinds (syn_spec.pelem):
 *   SV_PERT_RATE_ADD_PM  Bernoulli(rate) elements move by +-value (float) or
 *                        +-ivalue (integer, wrapping); non-finite stay.
 *   SV_PERT_REL_NOISE    x + (value*|x|)*z, z ~ N(0,1) (float types only).
 * Exact-count kinds (syn_spec.pcount), on `count` elements chosen one per
 * stratum of [0, logical_n) cut into `count` equal strata:
 *   SV_PERT_COUNT_SET    set to value (float) / ivalue (integer).
 *   SV_PERT_COUNT_ADD    finite x -> x + value; non-finite -> value
 *                        (integers: + ivalue, wrapping).
 *   SV_PERT_SWAP_PAIRS   `count` pairs from 2*count strata exchange values. */
enum {
  SV_PERT_NONE = 0, SV_PERT_RATE_ADD_PM = 1, SV_PERT_REL_NOISE = 2,
  SV_PERT_COUNT_SET = 3, SV_PERT_COUNT_ADD = 4, SV_PERT_SWAP_PAIRS = 5
};

/* ---- compare flags, stage states ---- */
enum { SV_EQUAL_NAN = 1u };
enum { SV_STAGE_RUN = 1u, SV_STAGE_SKIPPED = 2u };

/* ---- status codes ---- */
enum {
  SV_OK = 0,
  SV_EINVAL = -1,     /* bad enum, count, tolerance or dtype/dist pairing   */
  SV_EALIGN = -2,     /* an offset or elem_offset breaks the alignment rule */
  SV_ERANGE = -3,     /* data beyond the buffer, or a size beyond the limits */
  SV_EWORKSPACE = -4, /* workspace missing or smaller than *_workspace_bytes */
  SV_ECUDA = -5       /* a CUDA call failed                                   */
};

#define SV_NO_OUTPUT UINT64_MAX        /* syn_spec.ref_offset / cand_offset   */
#define SV_INLINE_ENTRIES 8            /* tables up to this size need no copy */
#define SV_MAX_ENTRIES (1 << 20)       /* specs / pairs / stages per call     */
#define SV_MAX_LOGICAL_N (1ull << 40)  /* elements of one logical array       */
#define SV_MAX_COUNT (1ull << 20)      /* exact-count perturbation size       */

typedef struct sv_perturb {
  uint32_t kind;   /* SV_PERT_* */
  uint32_t stream; /* Philox counter word 2 of this perturbation's draws */
  double rate;     /* RATE_ADD_PM: Bernoulli rate in [0, 1] */
  uint64_t count;  /* COUNT_*: elements; SWAP_PAIRS: pairs */
  double value;    /* float types: delta, target or noise scale */
  int64_t ivalue;  /* integer types: delta or target */
} sv_perturb;

/* One generator spec: n elements of one logical array (Sec. 4.2.1).
 * The clean output (base value, then special values) goes to ref_offset; the
 * perturbed twin (clean value, then pelem, then pcount) to cand_offset.  Either
 * may be SV_NO_OUTPUT, not both.  Element i of this spec is logical element
 * elem_offset + i of an array of logical_n elements (0 = elem_offset + n):
 * generating an array in chunks gives the same bytes as generating it whole. */
typedef struct syn_spec {
  uint32_t dtype;        /* SV_F32 ... SV_U32 */
  uint32_t dist;         /* SV_UNIFORM ... SV_FROM_ARENA */
  uint64_t n;            /* elements written per output */
  uint64_t seed;         /* Philox key */
  uint32_t stream;       /* Philox counter word 2 of base and special draws */
  uint32_t special_mask; /* OR of SV_SP_* */
  double special_rate;   /* in [0, 1] */
  uint64_t ref_offset;   /* byte offset in the arena, multiple of 16 */
  uint64_t cand_offset;  /* byte offset in the arena, multiple of 16 */
  uint64_t elem_offset;  /* multiple of 4 */
  uint64_t logical_n;    /* 0 -> elem_offset + n; at most SV_MAX_LOGICAL_N */
  double p0, p1;         /* float parameters (see SV_UNIFORM ...) */
  int64_t i0, i1;        /* integer parameters */
  uint64_t rows, cols, dot_k;  /* SV_DOTLIKE shape */
  uint64_t a_offset, b_offset; /* SV_DOTLIKE factors / SV_FROM_ARENA source (a_offset), multiples of 16 */
  sv_perturb pelem;      /* NONE, RATE_ADD_PM or REL_NOISE */
  sv_perturb pcount;     /* NONE, COUNT_SET, COUNT_ADD or SWAP_PAIRS */
} syn_spec;

/* One compare segment: n elements of candidate (K(x)) and reference (y). */
typedef struct vc_pair {
  uint32_t dtype;        /* both operands have this type */
  uint32_t flags;        /* SV_EQUAL_NAN: two NaNs match */
  uint64_t n;
  uint64_t cand_offset;  /* byte offset in the candidate buffer, multiple of 16 */
  uint64_t ref_offset;   /* byte offset in the reference buffer, multiple of 16 */
  double atol, rtol;     /* >= 0; rounded once to fp32; ignored for integers */
} vc_pair;

/* Per-segment verdict of Eq. 1, written to device memory.
 * Float types: the rule |x - y| <= atol + rtol*|y| in fp32 (no fused
 * operations) applies where both values are finite; equal values match
 * (same infinity, +0/-0); two NaNs match under SV_EQUAL_NAN.  Integer types:
 * exact equality, |x - y| as an unsigned 64-bit number. */
typedef struct vc_result {
  uint64_t mismatches;
  uint64_t nan_disagree;   /* exactly one side NaN */
  uint64_t inf_disagree;   /* an infinity on a side, no NaN, x != y */
  uint64_t n_finite;       /* elements with both sides finite (integers: n) */
  int64_t first_mismatch;  /* lowest mismatching index, -1 if none */
  uint64_t max_abs_u64;    /* integer types: max |x - y|; float types: 0 */
  double max_abs;          /* max |x - y| over both-finite elements */
  double max_rel;          /* max |x - y| / |y| over both-finite, y != 0 */
  double rms;              /* sqrt(sum |x - y|^2 / n_finite), 0 if none */
  uint32_t pass;           /* mismatches == 0 */
  uint32_t state;          /* SV_STAGE_RUN or SV_STAGE_SKIPPED */
} vc_result;

/* One shaped output compared tile by tile (CUDA-Harness Sec. 4.1.1: the
 * manifest gives every output's shape and type; Eq. 1 per element).  A
 * rows x cols output, row-major; the rows of each operand start cand_pitch /
 * ref_pitch elements apart (>= cols), so a padded or sub-matrix view works.
 * Tiles of tile_rows x tile_cols cover it in row-major order; the last tile
 * row and column may be smaller.  A tile of one row and all columns gives
 * per-row verdicts; a block tile localises an error to the part of the output
 * that one block of the kernel under test wrote. */
typedef struct vc_tiles {
  uint32_t dtype;        /* SV_F32 ... SV_U32 */
  uint32_t flags;        /* SV_EQUAL_NAN */
  uint64_t rows, cols;
  uint64_t cand_offset;  /* byte offset of element (0, 0), multiple of 16 */
  uint64_t ref_offset;
  uint64_t cand_pitch;   /* elements from one row start to the next, >= cols;
                            pitch * size a multiple of 16 when rows > 1 */
  uint64_t ref_pitch;
  uint64_t tile_rows;    /* >= 1 */
  uint64_t tile_cols;    /* >= 1; tile_cols * size a multiple of 16 when
                            tile_cols < cols */
  double atol, rtol;     /* as vc_pair */
} vc_tiles;

#define SV_MAX_TILES ((1ull << 31) - 1)  /* tiles of one call */

/* ---- workspace sizes (host only; no device needed) ----
 * Bytes of device workspace the matching call needs for these tables, 0 for
 * an invalid table.  The workspace must be 256-byte aligned. */
size_t sv_generate_workspace_bytes(const syn_spec* specs, int n_specs);
size_t sv_compare_workspace_bytes(const vc_pair* pairs, int n_pairs);
size_t sv_progressive_workspace_bytes(const vc_pair* stages, int n_stages);

/* ---- host-only validation (no CUDA call; usable without a GPU) ---- */
int sv_check_specs(const syn_spec* specs, int n_specs, size_t arena_bytes);
int sv_check_pairs(const vc_pair* pairs, int n_pairs, size_t cand_bytes, size_t ref_bytes);
/* also returns the number of tiles (0 on an error) in *n_tiles when not null */
int sv_check_tiles(const vc_tiles* tiles, size_t cand_bytes, size_t ref_bytes, uint64_t* n_tiles);

/* syn_generate: test-data synthesis (CUDA-Harness Sec. 4.2.1, "Decoupled Test
 * Data Synthesis": inputs and reference data made by seeded numerical
 * methods, separately from the kernel under test, over broad value ranges).
 *   specs/n_specs   host array of generator specs, run as one batch: no spec
 *                   may read (SV_DOTLIKE factors) what another spec of the
 *                   same call writes, and outputs must not overlap.
 *   d_arena, arena_bytes  device buffer that all offsets refer to.
 *   d_ws, ws_bytes  device workspace, >= sv_generate_workspace_bytes().
 * Errors: SV_EINVAL, SV_EALIGN, SV_ERANGE, SV_EWORKSPACE, SV_ECUDA. */
int syn_generate(const syn_spec* specs, int n_specs, void* d_arena, size_t arena_bytes, void* d_ws,
                 size_t ws_bytes, sv_stream_t stream);

/* A prepared syn_generate, for callers that synthesize the same spec table
 * again and again (every candidate of an evolution round is checked on the
 * same synthesized stages, Sec. 4.2.1/4.2.2): the table is validated,
 * grouped, scheduled and (beyond SV_INLINE_ENTRIES specs) copied into the
 * workspace once, so that each syn_generate_planned call only enqueues its
 * launches.
 *   sv_generate_plan_create: specs as syn_generate, checked against an arena
 *     of arena_bytes; d_ws, ws_bytes >= sv_generate_workspace_bytes() of the
 *     same table (none needed up to SV_INLINE_ENTRIES specs).  Synchronous: it
 *     returns once the table is in the workspace.  *plan receives a host
 *     object owned by the caller.
 *   syn_generate_planned: the bytes syn_generate writes for the plan's specs,
 *     into an arena of at least the size the plan was checked against (the
 *     caller keeps that promise), asynchronous on `stream`.  Nothing else may
 *     use the workspace while the plan lives.  The plan belongs to the device
 *     that was current at its creation.
 *   sv_generate_plan_destroy: frees the host object (NULL: nothing).
 * Errors: as syn_generate (create: also SV_ERANGE when out of host memory);
 * planned: SV_EINVAL (null plan or arena), SV_EALIGN (arena not on 16
 * bytes), SV_ECUDA. */
typedef struct sv_generate_plan sv_generate_plan;
int sv_generate_plan_create(const syn_spec* specs, int n_specs, size_t arena_bytes, void* d_ws, size_t ws_bytes,
                            sv_stream_t stream, sv_generate_plan** plan);
int syn_generate_planned(const sv_generate_plan* plan, void* d_arena, sv_stream_t stream);
void sv_generate_plan_destroy(sv_generate_plan* plan);

/* verify_compare: functional validation, Eq. 1 (CUDA-Harness Sec. 4.2.1),
 * one vc_result per pair.
 *   pairs/n_pairs   host array of segments.
 *   d_cand, cand_bytes / d_ref, ref_bytes  device buffers (may be the same).
 *   d_results       device array of n_pairs vc_result.
 *   d_ws, ws_bytes  device workspace, >= sv_compare_workspace_bytes().
 * Errors: SV_EINVAL, SV_EALIGN, SV_ERANGE, SV_EWORKSPACE, SV_ECUDA. */
int verify_compare(const vc_pair* pairs, int n_pairs, const void* d_cand, size_t cand_bytes,
                   const void* d_ref, size_t ref_bytes, vc_result* d_results, void* d_ws, size_t ws_bytes,
                   sv_stream_t stream);

/* A prepared verify_compare, for callers that compare many candidates on the
 * same segments (every candidate of a round is checked on the same stage
 * layout): the pair table is validated, grouped, scheduled and (beyond
 * SV_INLINE_ENTRIES pairs) copied into the workspace once, so that each
 * verify_compare_planned call only enqueues its launches.
 *   sv_compare_plan_create: pairs as verify_compare, checked against buffers
 *     of cand_bytes / ref_bytes; d_ws, ws_bytes >= sv_compare_workspace_bytes()
 *     of the same table.  Synchronous: it returns once the table is in the
 *     workspace.  *plan receives a host object owned by the caller.
 *   verify_compare_planned: the verdicts of verify_compare with the plan's
 *     pairs, on buffers of at least the sizes the plan was checked against
 *     (the caller keeps that promise; the plan does not see the buffers'
 *     sizes), asynchronous on `stream`.  The plan's workspace holds the table
 *     and the partial records: calls with one plan whose work can overlap on
 *     the GPU race, and nothing else may use the workspace while the plan
 *     lives.  The plan belongs to the device that was current at its creation.
 *   sv_compare_plan_destroy: frees the host object (NULL: nothing); the
 *     workspace stays the caller's.
 * Errors: as verify_compare (create: also SV_ERANGE when out of host memory);
 * planned: SV_EINVAL (null plan or buffers), SV_ECUDA. */
typedef struct sv_compare_plan sv_compare_plan;
int sv_compare_plan_create(const vc_pair* pairs, int n_pairs, size_t cand_bytes, size_t ref_bytes, void* d_ws,
                           size_t ws_bytes, sv_stream_t stream, sv_compare_plan** plan);
int verify_compare_planned(const sv_compare_plan* plan, const void* d_cand, const void* d_ref, vc_result* d_results,
                           sv_stream_t stream);
void sv_compare_plan_destroy(sv_compare_plan* plan);

/* verify_progressive: progressive multi-stage validation (CUDA-Harness
 * Sec. 4.2.2, fail-fast order).  Stages are compared in the given order
 * (size-ascending by convention); once a stage fails, every later stage is
 * skipped on the device (state SV_STAGE_SKIPPED, no data read) without a host
 * round trip.
 *   d_first_failed  device int32: index of the first failing stage, -1 if all
 *                   passed.
 * Other arguments as verify_compare.  Errors as verify_compare. */
int verify_progressive(const vc_pair* stages, int n_stages, const void* d_cand, size_t cand_bytes,
                       const void* d_ref, size_t ref_bytes, vc_result* d_results, int32_t* d_first_failed,
                       void* d_ws, size_t ws_bytes, sv_stream_t stream);

/* verify_compare_tiles: Eq. 1 over a shaped output, one vc_result per tile
 * (d_results: ceil(rows / tile_rows) * ceil(cols / tile_cols) records,
 * row-major over the tile grid).  A tile's statistics are those of
 * verify_compare over its elements in row-major order, except that
 * first_mismatch is the output-wide index row * cols + col.  Bytes between
 * the end of a row and the next row start (the pitch padding) are never read.
 * One CTA reduces a whole tile (no workspace); the GPU fills up with a few
 * hundred tiles or more.  rows or cols 0: nothing to do.
 * Errors: SV_EINVAL (type, flags, tolerance, zero tile extent, pitch < cols,
 * a tile wider or taller than 2^31 - 1), SV_EALIGN, SV_ERANGE (operand beyond
 * its buffer, more than SV_MAX_TILES tiles, a row pitch of 4 GiB or more
 * when tiles span several rows), SV_ECUDA. */
int verify_compare_tiles(const vc_tiles* tiles, const void* d_cand, size_t cand_bytes, const void* d_ref,
                         size_t ref_bytes, vc_result* d_results, sv_stream_t stream);

/* verify_compare_noalloc: the verdicts of verify_compare for callers that
 * cannot allocate device memory, for instance code running inside a host
 * process whose GPU memory is owned and budgeted by another component, or on
 * a latency-critical path that must not pay for an allocation.  Such callers
 * pass only their inputs and outputs; the library keeps the scratch (one
 * 64-byte partial record per CTA and pair) in a fixed array of its own device
 * memory: SV_NOALLOC_SLOTS records, 262,656 bytes, held on every GPU that
 * loads the library until the process exits.  The paper has no counterpart:
 * this is a convenience of the library, not a step of the method.
 *   Arguments and results as verify_compare, without the workspace.
 *   Limits: at most SV_NOALLOC_MAX_PAIRS pairs, and at most SV_NOALLOC_SLOTS
 *   partial records counted as the sum over the call's dtypes of
 *   min(tiles, 4096) + pairs, with tiles = ceil(n * sizeof(dtype) / 16384)
 *   summed over the pairs of that dtype (one large pair of any size fits;
 *   two large pairs of different dtypes do not).  Beyond them: SV_ERANGE,
 *   before anything is enqueued.
 *   The first call on each device looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current) and caches it; make
 *   that first call before any stream capture on the device.  All calls on a
 *   device share the one array: calls whose work can overlap on the GPU race
 *   and must be serialised by the caller.  It allocates nothing (no
 *   cudaMalloc, no cudaFree, no allocating library routine).
 * Errors: as verify_compare, except that SV_EWORKSPACE cannot occur. */
#define SV_NOALLOC_MAX_PAIRS 8
#define SV_NOALLOC_SLOTS 4104
int verify_compare_noalloc(const vc_pair* pairs, int n_pairs, const void* d_cand, size_t cand_bytes,
                           const void* d_ref, size_t ref_bytes, vc_result* d_results, sv_stream_t stream);

/* The Box-Muller step of the normal distribution (Sec. 4.2.1: normal test
 * values over broad ranges) on caller-supplied 32-bit words: pair i,
 * (d_words[2i], d_words[2i+1]) = (wa, wb), gives
 *   d_z[2i]   = r cos(theta),  d_z[2i+1] = r sin(theta),
 *   r = sqrt(-2 ln u1), u1 = ((wa >> 8) + 1) 2^-24,  theta = 2 pi (wb >> 8) 2^-24,
 * in fp32, exactly the values syn_generate makes for N(0, 1) from the same
 * VALUE words (so the transform can be checked alone, on any words).
 * Within 4 ulp of the transform computed in fp64 and rounded once.
 * d_words: n_pairs x 2 uint32 on the device; d_z: n_pairs x 2 float on the
 * device; both 8-byte aligned (SV_EALIGN) and caller-owned.  n_pairs = 0 is a
 * no-op; n_pairs > SV_MAX_LOGICAL_N / 2: SV_ERANGE; null pointers: SV_EINVAL.
 * Asynchronous on `stream`; allocates nothing. */
int syn_box_muller(const uint32_t* d_words, size_t n_pairs, float* d_z, sv_stream_t stream);

/* Static description of a status code. */
const char* sv_strerror(int status);
int sv_abi_version(void);

/* Instrumentation (no counterpart in the paper): the number of CUDA kernels
 * this library has launched in this process, on all devices and streams,
 * since it was loaded.  Read it before and after a piece of work to count that
 * work's launches.  Thread-safe; never fails. */
uint64_t sv_kernel_launches(void);

/* Test hook (no counterpart in the paper): the next n kernel launches of this
 * library, on any device or stream, use an invalid launch configuration, so
 * they fail at launch without running (no device fault; the context stays
 * usable) and the calls that made them return SV_ECUDA.  Lets a caller's
 * error handling be tested without a GPU fault.  n = 0 cancels; n < 0:
 * SV_EINVAL.  Process-wide. */
int sv_debug_fail_launches(int n);

#ifdef __cplusplus
}
#endif
#endif /* SYNVERIFY_H */
