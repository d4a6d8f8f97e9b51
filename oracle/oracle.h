/*
 * oracle.h -- plain, slow, single-threaded CPU oracle for the synthesis and
 * verification path of Synthesis-Based Verification (CUDA-Harness, Sec. 4.2).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may include, link or
 * call this code: only the tests, the package's smoke check and the bench's
 * CPU-baseline / reference arm use it.  It shares no code, header, table or
 * constant with the CUDA library; the two agree only through the documented
 * semantics below.
 *
 * Build: C11, -O2 -ffp-contract=off -fno-fast-math (no FMA contraction, no
 * flush-to-zero), so every float operation written here is one IEEE-754
 * round-to-nearest-even operation in the precision of its operands.
 *
 * What is computed (each function below cites the passage it follows):
 *   - test-data synthesis (Sec. 4.2.1, "Decoupled Test Data Synthesis"):
 *     seeded, counter-based generation of inputs with broad value ranges,
 *     special values and candidate perturbations;
 *   - functional validation (Sec. 4.2.1, Eq. 1): |K(x) - y| <= atol + rtol*|y|
 *     element by element, with per-segment statistics;
 *   - progressive validation (Sec. 4.2.2): stages in order, fail fast.
 * Where the paper is silent (generator, value maps, NaN/Inf handling,
 * precision of Eq. 1) the readings are written next to each function.
 */
#ifndef SV_ORACLE_H
#define SV_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* element types */
enum { OR_F32 = 0, OR_F16 = 1, OR_BF16 = 2, OR_I32 = 3, OR_I64 = 4, OR_U32 = 5 };
/* base value distributions */
enum {
  OR_UNIFORM = 0, OR_NORMAL = 1, OR_INT_RANGE = 2, OR_PERMUTATION = 3,
  OR_DOTLIKE = 4, OR_RAW_BITS = 5, OR_CONSTANT = 6, OR_FROM_ARENA = 7
};
/* special-value kinds (bit positions of the mask, drawn in ascending order) */
enum {
  OR_SP_NAN = 1u << 0, OR_SP_PINF = 1u << 1, OR_SP_NINF = 1u << 2,
  OR_SP_DENORM = 1u << 3, OR_SP_ZERO = 1u << 4, OR_SP_IMIN = 1u << 5,
  OR_SP_IMAX = 1u << 6, OR_SP_DUP = 1u << 7
};
/* selection mode bit of the mask: without it each element is special with
 * probability `rate` (Bernoulli); with it exactly round(rate * N) elements of
 * the logical array are, one per stratum (see or_special_index) */
#define OR_SP_EXACT (1u << 31)
#define OR_SP_KINDS 0xFFu
/* candidate perturbations */
enum {
  OR_PERT_NONE = 0, OR_PERT_RATE_ADD_PM = 1, OR_PERT_REL_NOISE = 2,
  OR_PERT_COUNT_SET = 3, OR_PERT_COUNT_ADD = 4, OR_PERT_SWAP_PAIRS = 5
};
/* Philox counter word c3: which quantity a draw is for */
enum {
  OR_P_VALUE = 0, OR_P_SPECIAL_SEL = 1, OR_P_SPECIAL_KIND = 2, OR_P_PERT_SEL = 3,
  OR_P_PERT_VAL = 4, OR_P_INDEX = 5, OR_P_PERM = 6, OR_P_NOISE = 7
};
/* compare flags and stage states */
enum { OR_EQUAL_NAN = 1u };
enum { OR_STAGE_RUN = 1u, OR_STAGE_SKIPPED = 2u };

#define OR_ABSENT UINT64_MAX

typedef struct {
  uint32_t kind;
  uint32_t stream;
  double rate;
  uint64_t count;
  double value;
  int64_t ivalue;
} or_perturb;

typedef struct {
  uint32_t dtype, dist;
  uint64_t n;
  uint64_t seed;
  uint32_t stream;
  uint32_t special_mask;
  double special_rate;
  uint64_t ref_offset;  /* byte offset of the clean output, OR_ABSENT = none */
  uint64_t cand_offset; /* byte offset of the perturbed twin, OR_ABSENT = none */
  uint64_t elem_offset; /* logical index of element 0 of this spec */
  uint64_t logical_n;   /* logical array length (0 -> elem_offset + n) */
  double p0, p1;
  int64_t i0, i1;
  uint64_t rows, cols, dot_k, a_offset, b_offset;
  or_perturb pelem;  /* element-wise kind (RATE_ADD_PM, REL_NOISE) or NONE */
  or_perturb pcount; /* exact-count kind (COUNT_SET, COUNT_ADD, SWAP_PAIRS) or NONE */
} or_spec;

typedef struct {
  uint32_t dtype, flags;
  uint64_t n;
  uint64_t cand_offset, ref_offset;
  double atol, rtol;
} or_pair;

typedef struct {
  uint64_t mismatches, nan_disagree, inf_disagree, n_finite;
  int64_t first_mismatch;
  uint64_t max_abs_u64;
  double max_abs, max_rel, rms;
  uint32_t pass, state;
} or_result;

/* ---- generator primitives (exported so the tests can pin them) ---- */
void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
void or_draw(uint64_t seed, uint32_t stream, uint32_t purpose, uint64_t block, uint32_t out[4]);
uint16_t or_f32_to_bf16(float f);
uint16_t or_f32_to_f16(float f);
float or_bf16_to_f32(uint16_t h);
float or_f16_to_f32(uint16_t h);
float or_uniform_map(float a, float b, uint32_t w);
void or_box_muller(uint32_t wa, uint32_t wb, float* z0, float* z1);
int64_t or_int_range_map32(int64_t lo, uint64_t r, uint32_t w);
uint64_t or_perm_value(uint64_t N, uint64_t seed, uint32_t stream, uint64_t g);
uint64_t or_stratum_index(uint64_t N, uint64_t k, uint64_t seed, uint32_t stream, uint64_t s);
/* exact-count special values: how many (round(rate * N), at most N) and the
 * index drawn in stratum s of [0, N) cut into k strata (SPECIAL_SEL purpose) */
uint64_t or_special_count(double rate, uint64_t N);
uint64_t or_special_index(uint64_t N, uint64_t k, uint64_t seed, uint32_t stream, uint64_t s);
/* the stratum of [0, N) cut into k strata that holds index g */
uint64_t or_stratum_of(uint64_t g, uint64_t k, uint64_t N);

/* bulk maps for exhaustive pins */
void or_map_uniform(float a, float b, const uint32_t* w, uint64_t n, float* out);
void or_map_box_muller(const uint32_t* w, uint64_t n_pairs, float* z);
void or_map_f32_to_bf16(const float* x, uint64_t n, uint16_t* out);
void or_map_f32_to_f16(const float* x, uint64_t n, uint16_t* out);
void or_int_range_histogram(uint64_t r, uint64_t* counts);
void or_map_perm(uint64_t N, uint64_t seed, uint32_t stream, uint64_t g0, uint64_t n, uint64_t* out);

/* ---- synthesis ---- */
/* 0 on success, negative on an invalid spec (nothing written for that spec). */
int or_check_spec(const or_spec* s, uint64_t arena_bytes);
/* value of logical element g: role 0 = clean output, role 1 = perturbed twin.
 * Returned as the element's storage bits, zero-extended to 64 bits. */
uint64_t or_value_at(const or_spec* s, const uint8_t* arena, uint64_t g, int role);
int or_generate(const or_spec* specs, int n_specs, uint8_t* arena, uint64_t arena_bytes);

/* ---- verification ---- */
/* 0 if the pair is valid for buffers of these sizes, else -1 */
int or_check_pair(const or_pair* p, uint64_t cand_bytes, uint64_t ref_bytes);
int or_compare(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
               const uint8_t* ref, uint64_t ref_bytes, or_result* out);
int or_progressive(const or_pair* stages, int n_stages, const uint8_t* cand, uint64_t cand_bytes,
                   const uint8_t* ref, uint64_t ref_bytes, or_result* out, int32_t* first_failed);
/* or_compare that also returns each segment's sum of squared differences
 * (the sum behind rms: rms = sqrt(sumsq / n_finite)), summed in index order */
int or_compare_sums(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
                    const uint8_t* ref, uint64_t ref_bytes, or_result* out, double* sumsq);

/* ---- the same, spread over host threads (threads.c) ----
 * For large inputs and for the CPU baseline measured on all host cores.
 * Each spec or pair is cut into contiguous element chunks; every chunk runs
 * through the single-threaded functions above (a spec chunk as a spec with
 * its elem_offset and logical_n, a pair chunk as a pair at shifted offsets),
 * and a pair's chunk verdicts are combined in chunk order: counts added,
 * the first mismatch taken from the first chunk that has one, maxima
 * maximised, sums of squares added.  Generated bytes and every integer
 * field equal the single-threaded results exactly; rms differs only by the
 * order of its fp64 sum.  nthreads <= 0: one thread per online host core.
 * Returns as the single-threaded function. */
int or_threads_default(void);
int or_generate_mt(const or_spec* specs, int n_specs, uint8_t* arena, uint64_t arena_bytes, int nthreads);
int or_compare_mt(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
                  const uint8_t* ref, uint64_t ref_bytes, or_result* out, int nthreads);
int or_progressive_mt(const or_pair* stages, int n_stages, const uint8_t* cand, uint64_t cand_bytes,
                      const uint8_t* ref, uint64_t ref_bytes, or_result* out, int32_t* first_failed,
                      int nthreads);

/* ---- shaped outputs (Sec. 4.1.1: the manifest gives each output's shape) ----
 * A rows x cols output, row-major, with a row pitch (elements between row
 * starts, >= cols) per operand, cut into tiles of tile_rows x tile_cols (the
 * last tile row / column may be smaller).  out[i * tiles_per_row + j] is the
 * verdict of tile (i, j) by the rule of or_compare over its elements in
 * row-major order; first_mismatch is the output-wide index row * cols + col.
 * Returns -1 (nothing written) for an invalid description. */
typedef struct {
  uint32_t dtype, flags;
  uint64_t rows, cols;
  uint64_t cand_offset, ref_offset;
  uint64_t cand_pitch, ref_pitch;
  uint64_t tile_rows, tile_cols;
  double atol, rtol;
} or_tiles;
int or_compare_tiles(const or_tiles* t, const uint8_t* cand, uint64_t cand_bytes, const uint8_t* ref,
                     uint64_t ref_bytes, or_result* out);

/* ---- value conversion of test data (convert.c) ----
 * The scaffold's helpers read the prepared test inputs and write the
 * outputs (Sec. 4.1.2); loading data of one element type as another (every
 * file read as float) is the loader defect behind 31.4% of the false
 * positives analysed in Sec. 5.2.3.  A dtype-correct load converts VALUES:
 *   - same type: the bytes, unchanged (NaN payloads included);
 *   - integer -> integer: the value; out of the target's range it is clamped
 *     to the nearest limit and counted in *n_bad;
 *   - any -> float: the value rounded once to nearest, ties to even, in the
 *     target format (subnormals kept, no flush to zero); a finite value that
 *     rounds beyond the largest finite value becomes +-Inf and is counted in
 *     *n_bad; +-Inf stay; every NaN becomes the target's canonical quiet NaN
 *     (positive, top fraction bit only); -0 stays -0;
 *   - float -> integer: refused (-1, nothing written): no silent truncation.
 * Element types: the six array types above plus the file-only types below. */
enum { OR_U8 = 6, OR_I8 = 7, OR_I16 = 8, OR_U16 = 9, OR_U64 = 10, OR_F64 = 11 };
int or_dtype_bytes(int dtype); /* 0 for an unknown type */
int or_convert(int src_dtype, const void* src, uint64_t n, int dst_dtype, void* dst, uint64_t* n_bad);

#ifdef __cplusplus
}
#endif
#endif
