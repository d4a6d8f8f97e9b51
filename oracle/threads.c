/*
 * threads.c -- the oracle's synthesis and verification spread over host
 * threads (POSIX threads), for inputs too large for one core and for the CPU
 * baseline measured on all host cores.
 *
 * TEST INFRASTRUCTURE ONLY, like oracle.c: only the tests, the package's smoke
 * check and the bench's CPU-baseline / reference arm use it.
 *
 * Nothing here computes a value or a verdict.  Every spec and every compare
 * pair is cut into contiguous element chunks, and each chunk goes through
 * the single-threaded functions of oracle.c unchanged:
 *   - a spec chunk is the same spec restricted to elements [i0, i1): its
 *     elem_offset advanced by i0, its logical length stated, its outputs
 *     advanced by i0 elements -- generation is a function of the logical
 *     index (Sec. 4.2.1: seeded, counter-based), so the chunks write exactly
 *     the bytes the whole spec writes;
 *   - a pair chunk is the same pair over elements [i0, i1) (both offsets
 *     advanced), compared by Eq. 1 with or_compare_sums, and the chunks of a
 *     pair are combined in chunk order.
 * Progressive validation (Sec. 4.2.2) runs its stages in order, each stage
 * over all threads, and stops after the first failing stage.
 */
#define _POSIX_C_SOURCE 200809L

#include <pthread.h>
#include <stdatomic.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>
#include <unistd.h>

#include "oracle.h"

int or_threads_default(void) {
  long n = sysconf(_SC_NPROCESSORS_ONLN);
  return n < 1 ? 1 : (n > 1024 ? 1024 : (int)n);
}

static int threads_or_default(int nthreads) { return nthreads > 0 ? nthreads : or_threads_default(); }

/* ------------------------------------------------------------------------ */
/* a minimal job pool: threads take job indices from a shared counter        */
/* ------------------------------------------------------------------------ */
typedef void (*job_fn)(void* ctx, uint64_t job);

typedef struct {
  job_fn fn;
  void* ctx;
  uint64_t n_jobs;
  atomic_ullong next;
} pool_t;

static void* pool_worker(void* arg) {
  pool_t* p = (pool_t*)arg;
  for (;;) {
    uint64_t j = atomic_fetch_add(&p->next, 1);
    if (j >= p->n_jobs) break;
    p->fn(p->ctx, j);
  }
  return NULL;
}

/* runs fn(ctx, j) for every j < n_jobs on up to nthreads threads (the caller
 * is one of them); returns once every job has finished */
static void run_jobs(job_fn fn, void* ctx, uint64_t n_jobs, int nthreads) {
  pool_t p;
  p.fn = fn;
  p.ctx = ctx;
  p.n_jobs = n_jobs;
  atomic_init(&p.next, 0);
  int extra = nthreads - 1;
  if ((uint64_t)extra > n_jobs) extra = n_jobs > 0 ? (int)(n_jobs - 1) : 0;
  pthread_t* th = extra > 0 ? (pthread_t*)malloc(sizeof(pthread_t) * (size_t)extra) : NULL;
  int started = 0;
  for (int i = 0; th && i < extra; ++i)
    if (pthread_create(&th[i], NULL, pool_worker, &p) == 0) ++started;
  pool_worker(&p);
  for (int i = 0; i < started; ++i) pthread_join(th[i], NULL);
  free(th);
}

static uint64_t dtype_bytes(uint32_t dt) { return dt == OR_I64 ? 8 : ((dt == OR_F16 || dt == OR_BF16) ? 2 : 4); }

/* elements per chunk: at least `floor_elems`, and about four chunks per
 * thread for an input of n elements; a multiple of 4 */
static uint64_t chunk_elems(uint64_t n, int nthreads, uint64_t floor_elems) {
  uint64_t c = (n + 4 * (uint64_t)nthreads - 1) / (4 * (uint64_t)nthreads);
  if (c < floor_elems) c = floor_elems;
  return (c + 3) & ~(uint64_t)3;
}

/* ------------------------------------------------------------------------ */
/* synthesis                                                                */
/* ------------------------------------------------------------------------ */
typedef struct {
  const or_spec* spec;  /* the whole spec */
  uint64_t i0, i1;      /* its elements [i0, i1) */
} gen_job;

typedef struct {
  gen_job* jobs;
  uint8_t* arena;
  uint64_t arena_bytes;
} gen_ctx;

static void gen_run(void* ctx, uint64_t j) {
  gen_ctx* c = (gen_ctx*)ctx;
  const gen_job* g = &c->jobs[j];
  or_spec s = *g->spec;
  uint64_t sz = dtype_bytes(s.dtype);
  s.logical_n = g->spec->logical_n ? g->spec->logical_n : g->spec->elem_offset + g->spec->n;
  s.elem_offset += g->i0;
  s.n = g->i1 - g->i0;
  if (s.ref_offset != OR_ABSENT) s.ref_offset += g->i0 * sz;
  if (s.cand_offset != OR_ABSENT) s.cand_offset += g->i0 * sz;
  or_generate(&s, 1, c->arena, c->arena_bytes);
}

int or_generate_mt(const or_spec* specs, int n_specs, uint8_t* arena, uint64_t arena_bytes, int nthreads) {
  nthreads = threads_or_default(nthreads);
  int status = 0;
  uint64_t n_jobs = 0;
  for (int i = 0; i < n_specs; ++i) {
    if (or_check_spec(&specs[i], arena_bytes) != 0) { status = -1; continue; }
    uint64_t ce = chunk_elems(specs[i].n, nthreads, 1 << 16);
    n_jobs += specs[i].n ? (specs[i].n + ce - 1) / ce : 0;
  }
  gen_job* jobs = (gen_job*)malloc(sizeof(gen_job) * (n_jobs ? n_jobs : 1));
  if (!jobs) return -1;
  uint64_t k = 0;
  for (int i = 0; i < n_specs; ++i) {
    if (or_check_spec(&specs[i], arena_bytes) != 0) continue;
    uint64_t n = specs[i].n, ce = chunk_elems(n, nthreads, 1 << 16);
    for (uint64_t a = 0; a < n; a += ce) {
      jobs[k].spec = &specs[i];
      jobs[k].i0 = a;
      jobs[k].i1 = a + ce < n ? a + ce : n;
      ++k;
    }
  }
  gen_ctx c = {jobs, arena, arena_bytes};
  run_jobs(gen_run, &c, n_jobs, nthreads);
  free(jobs);
  return status;
}

/* ------------------------------------------------------------------------ */
/* verification                                                             */
/* ------------------------------------------------------------------------ */
typedef struct {
  const or_pair* pair;
  uint64_t i0, i1;
} cmp_job;

typedef struct {
  cmp_job* jobs;
  or_result* res;
  double* sumsq;
  const uint8_t *cand, *ref;
  uint64_t cand_bytes, ref_bytes;
} cmp_ctx;

static void cmp_run(void* ctx, uint64_t j) {
  cmp_ctx* c = (cmp_ctx*)ctx;
  const cmp_job* g = &c->jobs[j];
  or_pair p = *g->pair;
  uint64_t sz = dtype_bytes(p.dtype);
  p.n = g->i1 - g->i0;
  p.cand_offset += g->i0 * sz;
  p.ref_offset += g->i0 * sz;
  or_compare_sums(&p, 1, c->cand, c->cand_bytes, c->ref, c->ref_bytes, &c->res[j], &c->sumsq[j]);
}

/* the verdict of a whole pair from its chunks' verdicts, in chunk order */
static void combine_chunks(const cmp_job* jobs, const or_result* res, const double* sumsq, uint64_t first_job,
                           uint64_t n_chunks, or_result* out) {
  memset(out, 0, sizeof(*out));
  out->first_mismatch = -1;
  out->state = OR_STAGE_RUN;
  double total = 0.0;
  for (uint64_t c = 0; c < n_chunks; ++c) {
    const or_result* r = &res[first_job + c];
    out->mismatches += r->mismatches;
    out->nan_disagree += r->nan_disagree;
    out->inf_disagree += r->inf_disagree;
    out->n_finite += r->n_finite;
    if (out->first_mismatch < 0 && r->first_mismatch >= 0)
      out->first_mismatch = (int64_t)jobs[first_job + c].i0 + r->first_mismatch;
    if (r->max_abs_u64 > out->max_abs_u64) out->max_abs_u64 = r->max_abs_u64;
    if (r->max_abs > out->max_abs) out->max_abs = r->max_abs;
    if (r->max_rel > out->max_rel) out->max_rel = r->max_rel;
    total += sumsq[first_job + c];
  }
  out->rms = out->n_finite ? sqrt(total / (double)out->n_finite) : 0.0;
  out->pass = out->mismatches == 0;
}

int or_compare_mt(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
                  const uint8_t* ref, uint64_t ref_bytes, or_result* out, int nthreads) {
  for (int i = 0; i < n_pairs; ++i)
    if (or_check_pair(&pairs[i], cand_bytes, ref_bytes) != 0) return -1;
  nthreads = threads_or_default(nthreads);
  uint64_t total = 0;
  for (int i = 0; i < n_pairs; ++i) total += pairs[i].n;
  /* chunks sized for the whole call: a table of many small pairs gives one
   * job per pair, a single large pair about four per thread */
  uint64_t ce = chunk_elems(total, nthreads, 1 << 16);
  uint64_t n_jobs = 0;
  for (int i = 0; i < n_pairs; ++i) n_jobs += pairs[i].n ? (pairs[i].n + ce - 1) / ce : 1;
  cmp_job* jobs = (cmp_job*)malloc(sizeof(cmp_job) * (n_jobs ? n_jobs : 1));
  or_result* res = (or_result*)malloc(sizeof(or_result) * (n_jobs ? n_jobs : 1));
  double* sumsq = (double*)malloc(sizeof(double) * (n_jobs ? n_jobs : 1));
  uint64_t* first = (uint64_t*)malloc(sizeof(uint64_t) * (n_pairs ? (size_t)n_pairs : 1));
  if (!jobs || !res || !sumsq || !first) {
    free(jobs); free(res); free(sumsq); free(first);
    return -1;
  }
  uint64_t k = 0;
  for (int i = 0; i < n_pairs; ++i) {
    first[i] = k;
    uint64_t n = pairs[i].n;
    if (n == 0) {  /* an empty pair: one empty chunk */
      jobs[k].pair = &pairs[i];
      jobs[k].i0 = jobs[k].i1 = 0;
      ++k;
      continue;
    }
    for (uint64_t a = 0; a < n; a += ce) {
      jobs[k].pair = &pairs[i];
      jobs[k].i0 = a;
      jobs[k].i1 = a + ce < n ? a + ce : n;
      ++k;
    }
  }
  cmp_ctx c = {jobs, res, sumsq, cand, ref, cand_bytes, ref_bytes};
  run_jobs(cmp_run, &c, n_jobs, nthreads);
  for (int i = 0; i < n_pairs; ++i) {
    uint64_t end = i + 1 < n_pairs ? first[i + 1] : n_jobs;
    combine_chunks(jobs, res, sumsq, first[i], end - first[i], &out[i]);
  }
  free(jobs); free(res); free(sumsq); free(first);
  return 0;
}

int or_progressive_mt(const or_pair* stages, int n_stages, const uint8_t* cand, uint64_t cand_bytes,
                      const uint8_t* ref, uint64_t ref_bytes, or_result* out, int32_t* first_failed,
                      int nthreads) {
  for (int i = 0; i < n_stages; ++i)
    if (or_check_pair(&stages[i], cand_bytes, ref_bytes) != 0) return -1;
  *first_failed = -1;
  for (int i = 0; i < n_stages; ++i) {
    if (*first_failed >= 0) {
      memset(&out[i], 0, sizeof(out[i]));
      out[i].first_mismatch = -1;
      out[i].state = OR_STAGE_SKIPPED;
      continue;
    }
    if (or_compare_mt(&stages[i], 1, cand, cand_bytes, ref, ref_bytes, &out[i], nthreads) != 0) return -1;
    if (!out[i].pass) *first_failed = i;
  }
  return 0;
}
