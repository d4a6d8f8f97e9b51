/*
 * sv_io.h -- dtype-correct test-data I/O of the GB300 library (part of the
 * same shared library as synverify.h).
 *
 * The scaffold of CUDA-Harness (Sec. 4.1.2) gives every self-contained
 * program two helpers, one that reads the prepared test inputs from files
 * named on the command line and one that writes the kernel's outputs, so a
 * program cannot invent its own inputs.  Sec. 5.2.3 traces 31.4% of the
 * false positives of synthesis-based verification to a template that loaded
 * every test file as float, so uint8 and int32 data arrived as wrong values.
 * These entry points are that pair of helpers made dtype-correct: a file
 * states its element type and shape in a header (or, for a headerless file,
 * the caller states them and the file size must agree), and loading into a
 * buffer of another element type converts VALUES on the GPU instead of
 * reinterpreting bytes.
 *
 * Tensor file layout ("SVT1"), little-endian:
 *   bytes [0, 128)    sv_tensor_header
 *   bytes [128, ...)  n elements of `dtype`, dense, row-major (last extent
 *                     fastest), exactly data_bytes = n * size(dtype) bytes;
 *                     nothing follows.
 * A headerless ("raw") file is the elements alone.
 *
 * Value conversion (file element type S -> buffer element type D):
 *   S == D            the bytes, unchanged.
 *   integer -> integer  the value; outside D's range it is clamped to the
 *                     nearest limit and counted as lost.
 *   any -> float      the value rounded once to nearest, ties to even, in D
 *                     (subnormals kept, no flush to zero); a finite value that
 *                     rounds past D's largest finite value becomes +-Inf and
 *                     is counted as lost; +-Inf stay; every NaN becomes D's
 *                     canonical quiet NaN (positive, top fraction bit only);
 *                     -0 stays -0.
 *   float -> integer  refused: SV_EINVAL, nothing read or written.
 *
 * Threading and memory: every call is synchronous for the host (it returns
 * when its data are in place and its counts are known) and uses `stream` for
 * its copies and kernels; calls of one process are serialised by a lock.  The
 * library keeps SV_IO_SLOTS pinned host buffers of SV_IO_CHUNK_BYTES for file
 * data (allocated on first use, kept for the life of the process) and a pool
 * of host threads that read file stripes in parallel.  It allocates
 * no device memory: a conversion stages file bytes in the caller's workspace.
 */
#ifndef SV_IO_H
#define SV_IO_H

#include "synverify.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Element types of files and buffers: SV_F32 ... SV_U32 (synverify.h) and six more. */
enum { SV_U8 = 6, SV_I8 = 7, SV_I16 = 8, SV_U16 = 9, SV_U64 = 10, SV_F64 = 11 };

/* Further status codes of the I/O entry points. */
enum {
  SV_EIO = -6,      /* a file could not be opened, read, written or sized     */
  SV_EFORMAT = -7,  /* bad header, or the file's type, count or size is not
                       what the caller stated                                  */
  SV_ELOSSY = -8    /* the data are in place, but *n_lost values were clamped
                       or overflowed to infinity by the conversion             */
};

#define SV_TENSOR_MAGIC 0x31545653u /* "SVT1" */
#define SV_TENSOR_HEADER_BYTES 128
#define SV_TENSOR_MAX_DIMS 8
#define SV_IO_CHUNK_BYTES (32u << 20) /* file bytes per pipeline step */
#define SV_IO_SLOTS 4

typedef struct sv_tensor_header {
  uint32_t magic;                      /* SV_TENSOR_MAGIC                      */
  uint32_t header_bytes;               /* SV_TENSOR_HEADER_BYTES               */
  uint32_t dtype;                      /* element type, SV_F32 ... SV_F64      */
  uint32_t ndim;                       /* 0 ... SV_TENSOR_MAX_DIMS             */
  uint64_t shape[SV_TENSOR_MAX_DIMS];  /* extents; entries >= ndim are 0       */
  uint64_t n;                          /* product of the extents (1 if ndim 0) */
  uint64_t data_bytes;                 /* n * element size                     */
  uint64_t reserved[4];                /* 0                                    */
} sv_tensor_header;

/* flags of sv_read_tensor / sv_write_tensor */
enum {
  SV_IO_RAW = 1u,    /* headerless file: the caller states type and count     */
  SV_IO_STRICT = 2u  /* no conversion: the file's type must equal dst_dtype   */
};

/* Bytes of one element of `dtype`, 0 for an unknown type.  Host only. */
int sv_dtype_bytes(int dtype);

/* Reads and checks the header of a tensor file (host only, no CUDA call).
 * Checks: magic, header_bytes, a known dtype, ndim <= SV_TENSOR_MAX_DIMS,
 * n = product of the extents (no overflow), data_bytes = n * size, reserved
 * words zero, and file size = 128 + data_bytes.
 * Errors: SV_EINVAL (null argument), SV_EIO, SV_EFORMAT. */
int sv_tensor_probe(const char* path, sv_tensor_header* out);

/* Device workspace bytes sv_read_tensor needs to load n elements of
 * src_dtype into dst_dtype: 0 when the types are equal, otherwise 256 bytes
 * plus room for two chunks of file data.  0 for unknown types. */
size_t sv_io_workspace_bytes(int src_dtype, int dst_dtype, uint64_t n);

/* sv_read_tensor: loads the test data of a file into device memory, the
 * scaffold's input helper made dtype-correct (Sec. 4.1.2; Sec. 5.2.3).
 *   path        the file.
 *   flags       SV_IO_RAW, SV_IO_STRICT.
 *   file_dtype  the element type the caller expects in the file, or -1 to
 *               take the header's (required, >= 0, for SV_IO_RAW).  A header
 *               with another type: SV_EFORMAT (the file is not what the
 *               caller thinks it is; nothing is loaded).
 *   n_expect    the element count the caller expects, or 0 for whatever the
 *               file holds.  A header with another count: SV_EFORMAT.  With
 *               SV_IO_RAW the file size must be n_expect * size(file_dtype)
 *               exactly (n_expect = 0: any multiple of the element size),
 *               else SV_EFORMAT: a uint8 file of n bytes read as n floats
 *               fails here instead of loading garbage.
 *   dst_dtype   the element type of d_dst; with SV_IO_STRICT it must equal
 *               the file's (else SV_EFORMAT).
 *   d_dst       device buffer, 16-byte aligned, dst_bytes >= n * size(dst).
 *   d_ws        device workspace (256-byte aligned), ws_bytes >=
 *               sv_io_workspace_bytes(file type, dst_dtype, n); may be NULL
 *               when the types are equal.
 *   out_header  optional (NULL): the file's header (for SV_IO_RAW, one made
 *               from the stated type and count, ndim 1).
 *   n_lost      optional (NULL): values clamped or overflowed by the
 *               conversion.
 * Returns 0; SV_ELOSSY when values were lost (data in place, *n_lost set);
 * SV_EINVAL (bad type, float -> integer, null pointer), SV_EALIGN, SV_ERANGE
 * (d_dst too small), SV_EWORKSPACE, SV_EIO, SV_EFORMAT, SV_ECUDA. */
int sv_read_tensor(const char* path, uint32_t flags, int file_dtype, uint64_t n_expect, int dst_dtype,
                   void* d_dst, size_t dst_bytes, void* d_ws, size_t ws_bytes, sv_stream_t stream,
                   sv_tensor_header* out_header, uint64_t* n_lost);

/* sv_write_tensor: writes n = prod(shape) elements of `dtype` from device
 * memory to a file, the scaffold's output helper (Sec. 4.1.2): a header with
 * the type and shape, then the bytes (SV_IO_RAW: the bytes alone).  The file
 * is created or truncated; on an error it may be left partly written.
 *   shape/ndim  host array of extents, ndim <= SV_TENSOR_MAX_DIMS.
 *   d_src       device buffer, 16-byte aligned, src_bytes >= n * size.
 * Work already queued on `stream` is waited for before the bytes are read.
 * Errors: SV_EINVAL, SV_EALIGN, SV_ERANGE, SV_EIO, SV_ECUDA. */
int sv_write_tensor(const char* path, uint32_t flags, int dtype, const uint64_t* shape, int ndim,
                    const void* d_src, size_t src_bytes, sv_stream_t stream);

/* sv_convert: the value conversion alone, device to device, asynchronous on
 * `stream` (no host wait).  n elements of src_dtype at d_src become n
 * elements of dst_dtype at d_dst (both 16-byte aligned, not overlapping).
 * d_lost: optional device uint64 to which the number of clamped or
 * overflowed values is ADDED (the caller zeroes it).  src_dtype ==
 * dst_dtype copies the bytes.
 * Errors: SV_EINVAL (unknown type, float -> integer, null pointer with n > 0),
 * SV_EALIGN, SV_ERANGE (n > 2^40), SV_ECUDA. */
int sv_convert(int src_dtype, const void* d_src, uint64_t n, int dst_dtype, void* d_dst,
               uint64_t* d_lost, sv_stream_t stream);

/* Test hook (no counterpart in the paper): file bytes per pipeline step of
 * later read and write calls, a multiple of 4096 from 4096 to
 * SV_IO_CHUNK_BYTES; 0 restores SV_IO_CHUNK_BYTES; anything else: SV_EINVAL.
 * Lets a test cross many chunk boundaries with small files.  Process-wide. */
int sv_debug_io_chunk_bytes(size_t bytes);

#ifdef __cplusplus
}
#endif
#endif /* SV_IO_H */
