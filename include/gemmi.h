/*
 * gemmi.h -- exact integer GEMM  C += A*B  on NVIDIA GB300 (sm_103a).
 *
 * The operation is the GEMM of Section 4.1 of the paper ("Toward Matrix
 * Multiplication for Deep Learning Inference on the Xilinx Versal"): A is
 * m x k, B is k x n, C is m x n, and C is updated in place, C += A*B.  The
 * paper's micro-kernel takes INT16 operands (Section 6.1) and sums their
 * products in 48-bit accumulators so that nothing overflows (Section 6.2);
 * this library keeps that exactness and widens the result to a 64-bit C.
 *
 * Layout (all entry points): row-major with leading dimensions,
 *     A[i*lda + p],  B[p*ldb + j],  C[i*ldc + j],
 * lda >= max(1,k), ldb >= max(1,n), ldc >= max(1,n).  Entries of C outside the
 * m x n block (the padding of each row) are never read or written.
 *
 * Semantics: bit-exact.  int16 operands accumulate into an int64 C modulo
 * 2^64; int8 operands accumulate into an int32 C modulo 2^32.  Addition modulo
 * 2^w is associative, so the result is unique and independent of the order in
 * which the kernels sum.  m == 0, n == 0 or k == 0 is a no-op returning
 * GEMMI_OK.
 *
 * Errors: every entry point returns a gemmi_status code; the text of the last
 * error of the calling thread is available from gemmi_last_error().  Kernel
 * launches are asynchronous: a device-side failure (a pipeline wait that ran
 * past its time bound) is recorded in a per-device status word that
 * gemmi_device_status() reads (and clears).  No device code traps.
 */
#ifndef GEMMI_H
#define GEMMI_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum gemmi_status {
  GEMMI_OK = 0,
  GEMMI_EINVAL = 1,   /* negative size, ld too small, null pointer with a non-zero size, C overlapping A or B */
  GEMMI_ENOMEM = 2,   /* the device workspace could not be allocated */
  GEMMI_ECUDA = 3,    /* a CUDA runtime/driver call or a kernel launch failed */
  GEMMI_ETIMEOUT = 4, /* a device-side pipeline wait exceeded its bound (reported by gemmi_device_status) */
  GEMMI_EARCH = 5     /* the current device is not an sm_103 (GB300) GPU */
} gemmi_status;

/*
 * gemm_i16 -- C (int64) += A (int16) * B (int16), exactly, modulo 2^64.
 * Section 4.1 (problem statement), Section 6.1 (INT16 operands).
 *
 * A, B, C are DEVICE pointers owned by the caller; A and B are only read,
 * C is read and written.  The call is asynchronous on the library's current
 * stream (gemmi_set_stream; default: the legacy default stream).  The library
 * owns a device workspace for the limb planes of A and B (grown on demand,
 * freed by gemmi_release_workspace) and serialises its use across streams.
 * Returns GEMMI_OK, GEMMI_EINVAL, GEMMI_ENOMEM, GEMMI_ECUDA or GEMMI_EARCH.
 */
int gemm_i16(int64_t m, int64_t n, int64_t k,
             const int16_t* A, int64_t lda,
             const int16_t* B, int64_t ldb,
             int64_t* C, int64_t ldc);

/* gemm_i16 on an explicit stream (a cudaStream_t passed as void*; NULL = legacy default stream). */
int gemm_i16_ex(int64_t m, int64_t n, int64_t k,
                const int16_t* A, int64_t lda,
                const int16_t* B, int64_t ldb,
                int64_t* C, int64_t ldc, void* stream);

/*
 * gemm_i8 -- C (int32) += A (int8) * B (int8), exactly, modulo 2^32.
 * Section 4.1 (problem statement); the INT8 datatype of Section 6.1.
 * Same pointer ownership, layout, stream and error behaviour as gemm_i16.
 */
int gemm_i8(int64_t m, int64_t n, int64_t k,
            const int8_t* A, int64_t lda,
            const int8_t* B, int64_t ldb,
            int32_t* C, int64_t ldc);

int gemm_i8_ex(int64_t m, int64_t n, int64_t k,
               const int8_t* A, int64_t lda,
               const int8_t* B, int64_t ldb,
               int32_t* C, int64_t ldc, void* stream);

/*
 * gemm_i4 -- C (int32) += A (int4) * B (int4), exactly, modulo 2^32.
 * Section 4.1 (problem statement) at a precision below the INT16 / INT8 the paper measures; the
 * paper's datatype discussion (Section 6.1) leaves the lower-precision micro-kernel to future work.
 * Operands are PACKED, two signed 4-bit values to a byte: element (i, p) of A is in byte
 * A[i*lda + p/2], element (p, j) of B in byte B[p*ldb + j/2]; the even index in the low nibble
 * (bits 0-3), the odd one in the high nibble (bits 4-7), two's complement (nibbles 8..15 stand
 * for -8..-1).  lda and ldb count BYTES: lda >= max(1, ceil(k/2)), ldb >= max(1, ceil(n/2));
 * ldc counts int32 elements, ldc >= max(1, n).  The spare high nibble of a row's last byte (odd
 * k for A, odd n for B) and the bytes of the row padding are never read.
 * Same pointer ownership (DEVICE pointers owned by the caller), stream, workspace and error
 * behaviour as gemm_i16.  A C whose base is not 16-byte aligned, or whose ldc is not a multiple
 * of 4, is accumulated through a zeroed scratch array in the workspace and added in one more pass.
 */
int gemm_i4(int64_t m, int64_t n, int64_t k,
            const uint8_t* A, int64_t lda,
            const uint8_t* B, int64_t ldb,
            int32_t* C, int64_t ldc);

int gemm_i4_ex(int64_t m, int64_t n, int64_t k,
               const uint8_t* A, int64_t lda,
               const uint8_t* B, int64_t ldb,
               int32_t* C, int64_t ldc, void* stream);

/*
 * gemm_i16_host / gemm_i8_host -- the same GEMMs on HOST buffers.
 * A, B, C are host pointers (pinned memory gives the fastest copies).  The
 * library copies A, B and C to device buffers it owns, runs the GEMM on its
 * current stream, copies C back and waits for the stream, so C holds the
 * result when the call returns.  With m >= 1024 the copies are pipelined:
 * B goes over once, then row panels of A and C pass through a ring of device
 * slots on separate copy-in and copy-out streams while earlier panels compute.
 * Errors as above; a device-side timeout is returned directly as GEMMI_ETIMEOUT.
 */
int gemm_i16_host(int64_t m, int64_t n, int64_t k,
                  const int16_t* A, int64_t lda,
                  const int16_t* B, int64_t ldb,
                  int64_t* C, int64_t ldc);

int gemm_i8_host(int64_t m, int64_t n, int64_t k,
                 const int8_t* A, int64_t lda,
                 const int8_t* B, int64_t ldb,
                 int32_t* C, int64_t ldc);

/* gemm_i4 on HOST buffers (A and B in gemm_i4's packed format, lda and ldb in bytes); copies,
 * result and errors as gemm_i16_host. */
int gemm_i4_host(int64_t m, int64_t n, int64_t k,
                 const uint8_t* A, int64_t lda,
                 const uint8_t* B, int64_t ldb,
                 int32_t* C, int64_t ldc);

/*
 * gemm_i16_srs -- the output of the paper's AIE micro-kernel (Section 5.2, the
 * simplified micro-kernel listing): the wide accumulator is shifted, rounded and
 * saturated to 16 bits ("srs") and added to an int16 C with a 16-bit addition.
 *
 *   S = A * B (exact), R = S for shift == 0,
 *   R = floor((S + 2^(shift-1)) / 2^shift) for shift >= 1 (round half up),
 *   C[i,j] = (C[i,j] + clamp(R, -32768, 32767)) mod 2^16.
 *
 * The paper leaves the rounding and the kind of addition unstated (its listing
 * shifts by 0); these are this library's readings.  The saturation sees the full
 * reduction (k_c = k).  A, B: int16 device matrices as for gemm_i16; C: int16,
 * row-major with leading dimension ldc, updated in place.  shift in [0, 62].
 * The exact sums pass through a library-owned int64 scratch of m x roundup(n, 8)
 * entries (released by gemmi_release_workspace).  Errors as for gemm_i16.
 */
int gemm_i16_srs(int64_t m, int64_t n, int64_t k,
                 const int16_t* A, int64_t lda,
                 const int16_t* B, int64_t ldb,
                 int16_t* C, int64_t ldc, int shift);
int gemm_i16_srs_ex(int64_t m, int64_t n, int64_t k,
                    const int16_t* A, int64_t lda,
                    const int16_t* B, int64_t ldb,
                    int16_t* C, int64_t ldc, int shift, void* stream);

/*
 * gemmi_conv2d_i16 -- a convolution through the lowered GEMM.  Sections 2 and 3 of
 * the paper cast a convolution as one large GEMM with the IM2COL / IM2ROW transform,
 * and note that the transform may be applied on the fly as part of the packing.
 *
 *   Y[n][ho][wo][co] += sum over r < R, s < S, c < Cin of
 *                       X[n][ho + r - pad_h][wo + s - pad_w][c] * Wt[(r*S + s)*Cin + c][co],
 * stride 1, X read as 0 outside the image, Ho = H + 2*pad_h - R + 1,
 * Wo = W + 2*pad_w - S + 1; exact, modulo 2^64 as gemm_i16.
 *
 * X: int16 NHWC (N x H x W x Cin), dense.  Wt: int16, the lowered weight matrix,
 * R*S*Cin rows in (r, s, c) order by Cout columns, dense.  Y: int64 NHWC
 * (N x Ho x Wo x Cout), dense, updated in place.  All device pointers, owned by
 * the caller; Y may not overlap X or Wt.  When Ho == H, Wo == W (a "same"
 * convolution), Cin % 64 == 0, Cout <= 256 and X is 16-byte aligned, the GEMM
 * reads X directly (no lowered matrix is formed); with Cin == 64 and the further
 * conditions of GEMMI_OPT_CONV_ROWS a direct kernel splits every input pixel once
 * for all taps instead.  Other shapes lower X into library-owned memory first
 * (released by gemmi_release_workspace).  Every path gives the same result.
 * Errors: GEMMI_EINVAL for negative sizes or paddings, R or S below 1, a filter
 * larger than the padded input, null pointers with non-zero sizes, overlapping Y;
 * otherwise as gemm_i16.  Empty outputs return GEMMI_OK.
 */
int gemmi_conv2d_i16(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                     int64_t R, int64_t S, int64_t pad_h, int64_t pad_w,
                     const int16_t* X, const int16_t* Wt, int64_t* Y, void* stream);

/*
 * Weight pre-packing.  Section 5.1 of the paper keeps the weight operand packed,
 * off-line, in fast memory, because a deployed model runs many inputs through
 * the same weights; only the activations are packed at run time.  Here the
 * weights are the B operand: gemmi_pack_b_* converts B (k x n, row-major,
 * DEVICE pointer, only read) once into the library's internal limb planes,
 * held in device memory the handle owns (allocated by this call), on `stream`.
 * gemm_*_packed then computes C += A * B for any A (m x k) with that B,
 * converting only A per call; the result is bit-identical to gemm_i16/gemm_i8/gemm_i4.
 * gemmi_pack_b_i4 takes B in gemm_i4's packed-nibble format (ldb in bytes,
 * >= ceil(n/2)) and gemm_i4_packed an A in that format (lda >= ceil(k/2) bytes).
 * Packed GEMMs always take the tensor-core path (for m <= 16, gemm_i16 on the
 * raw B streams fewer bytes).  The handle belongs to the device that was
 * current when it was made; gemmi_packed_b_free() synchronises that device and
 * frees it.  Errors as for gemm_i16 (a null handle or one of another device:
 * GEMMI_EINVAL).
 */
typedef struct gemmi_packed_b gemmi_packed_b;
int gemmi_pack_b_i16(int64_t k, int64_t n, const int16_t* B, int64_t ldb, void* stream, gemmi_packed_b** out);
int gemmi_pack_b_i8(int64_t k, int64_t n, const int8_t* B, int64_t ldb, void* stream, gemmi_packed_b** out);
int gemm_i16_packed(int64_t m, const int16_t* A, int64_t lda, const gemmi_packed_b* B, int64_t* C, int64_t ldc,
                    void* stream);
int gemm_i8_packed(int64_t m, const int8_t* A, int64_t lda, const gemmi_packed_b* B, int32_t* C, int64_t ldc,
                   void* stream);
int gemmi_pack_b_i4(int64_t k, int64_t n, const uint8_t* B, int64_t ldb, void* stream, gemmi_packed_b** out);
int gemm_i4_packed(int64_t m, const uint8_t* A, int64_t lda, const gemmi_packed_b* B, int32_t* C, int64_t ldc,
                   void* stream);
int gemmi_packed_b_free(gemmi_packed_b* packed);
/* k and n of a packed operand (0 for a null handle). */
int64_t gemmi_packed_b_k(const gemmi_packed_b* packed);
int64_t gemmi_packed_b_n(const gemmi_packed_b* packed);

/* Stream used by gemm_i16 / gemm_i8 / *_host (a cudaStream_t as void*). */
void gemmi_set_stream(void* stream);

/* Text of the calling thread's last error ("" if none).  Owned by the library. */
const char* gemmi_last_error(void);

/*
 * Synchronises the current device and returns, then clears, its device status
 * words: GEMMI_OK, or GEMMI_ETIMEOUT if a kernel gave up a pipeline wait.  Two
 * words are read: the library's own (written by every entry point except
 * gemm_i16_noalloc) and, once gemm_i16_noalloc has run on the device, the word
 * inside that entry point's fixed scratch array.  The first non-zero word
 * decides the result; every non-zero word is cleared.
 * gemmi_device_status_stream(stream) does the same after synchronising only
 * `stream` (a cudaStream_t as void*; NULL = legacy default stream): it sees the
 * failures of the kernels that stream ran, and of any other kernel that had
 * finished by then.  Section 6.2 of the paper makes the accumulators wide so
 * that nothing overflows; a wait that ran out is the one failure left to report.
 * gemmi_device_status_detail() returns the raw word of the last read
 * (low byte: status code; next byte: the wait site; upper half: block index).
 */
int gemmi_device_status(void);
int gemmi_device_status_stream(void* stream);
uint32_t gemmi_device_status_detail(void);

/* Frees the library-owned device workspace of the current device (synchronises it). */
int gemmi_release_workspace(void);

/* Bytes of library-owned device workspace currently held on the current device. */
size_t gemmi_workspace_bytes(void);

/*
 * Tuning and test options (process-wide).
 *   GEMMI_OPT_SKINNY_MAX_M : int16 GEMMs with m <= this value take the
 *                            skinny-M kernel (default 16, maximum 16; 0 disables it).
 *   GEMMI_OPT_WAIT_TIMEOUT_US : bound on every device-side pipeline wait, in
 *                            microseconds (default 4,000,000; 1,000 to 60,000,000).
 *   GEMMI_OPT_SKINNY_KSPLIT : number of CTAs sharing the reduction dimension
 *                            of one skinny column block (0 = automatic).
 *   GEMMI_OPT_TC_CHUNK_SCALE : length of the exact fp32 accumulation runs of the tensor-core
 *                            GEMM: 2 (default) keeps every partial limb sum within 2^24, the limit
 *                            of exact fp32 integer sums; 1 keeps it within 2^23 (twice the drains).
 *                            gemm_i4: 2 drains every 2^18 reduction indices (sums within 2^24),
 *                            1 every 256 (sums within 2^14).
 *   GEMMI_OPT_TC_GROUP_M   : tile raster band height in tile rows; 0 (default) = automatic: 8 for
 *                            the int16 and int8 kernels, 16 for int4.
 *   GEMMI_OPT_TC_L2_HINTS  : L2 eviction policy of the operand tile loads, bits 0-1 for A,
 *                            bits 2-3 for B: 0 normal, 1 evict_last, 2 evict_first (default 0).
 *   GEMMI_OPT_FUSED_MAX_N  : int16 GEMMs with n <= this value (and an A whose base is 16-byte
 *                            aligned with lda % 8 == 0) take the kernel that reads A raw and
 *                            splits it on chip (default 64; 0 disables it; at most 4096).
 *   GEMMI_OPT_TC_PAIR      : 1 (default): tensor-core GEMMs run on pairs of SMs (tcgen05
 *                            cta_group::2, clusters of two CTAs) whenever C is 16-byte aligned
 *                            with ldc * sizeof(element) a multiple of 16; 0: one SM per tile.
 *   GEMMI_OPT_SMALL_MAX_MACS : int16 GEMMs with m <= 256 and m*n*k <= this value (default 2^28)
 *                            run as one launch of the skinny-M kernel, 16 rows of A per grid
 *                            row; 0 disables it (so does GEMMI_OPT_SKINNY_MAX_M = 0).
 *   GEMMI_OPT_KARATSUBA    : 1: int16 GEMMs on the tensor-core path (not skinny, not narrow-n,
 *                            not packed weights) use Karatsuba's three limb products
 *                            HH, LL and (h_a + l_a)(h_b + l_b) instead of four, on one SM per
 *                            tile, with a third plane per operand in the workspace; 0 (default):
 *                            four products.  The tensor work shrinks by a quarter; the measured
 *                            time is longer (shared-memory stages, drains).
 *   GEMMI_OPT_SPLIT_AHEAD  : 1 (default): an int16 GEMM on SM pairs whose A is 16-byte aligned
 *                            with lda % 8 == 0 and k % 8 == 0 splits only the row panels of A
 *                            that the first wave of tiles reads (and B) before the GEMM
 *                            kernel; two warps of every CTA of that kernel split the remaining
 *                            panels while the tensor cores work, and a tile's loads wait until
 *                            its panel is complete; 0: the whole split runs before the GEMM.
 *   GEMMI_OPT_CONV_ROWS    : 1 (default): gemmi_conv2d_i16 runs "same" convolutions with 64 input
 *                            channels, odd R and S with R*S <= 12 and R*S*64 within one exact chunk
 *                            (512 * chunk scale), an even Cout <= 64, W <= 120, W + S - 1 <= 128
 *                            and 16-byte aligned X and Y
 *                            on the direct kernel, which splits every input pixel once per tile of
 *                            output rows (the taps are shifted windows of the split rows); 0:
 *                            such convolutions take the lowered GEMM read tap by tap.
 * Results do not depend on any option; only speed does.  Returns GEMMI_OK or GEMMI_EINVAL.
 */
enum { GEMMI_OPT_SKINNY_MAX_M = 1, GEMMI_OPT_WAIT_TIMEOUT_US = 2, GEMMI_OPT_SKINNY_KSPLIT = 3,
       GEMMI_OPT_TC_CHUNK_SCALE = 4, GEMMI_OPT_TC_GROUP_M = 5, GEMMI_OPT_TC_L2_HINTS = 6,
       GEMMI_OPT_FUSED_MAX_N = 7, GEMMI_OPT_TC_PAIR = 8, GEMMI_OPT_SMALL_MAX_MACS = 9,
       GEMMI_OPT_KARATSUBA = 10, GEMMI_OPT_SPLIT_AHEAD = 11, GEMMI_OPT_CONV_ROWS = 12 };
int gemmi_set_option(int option, int64_t value);
int64_t gemmi_get_option(int option);

/*
 * Failure-detection self-test: launches one tiny kernel whose single thread
 * waits, with a bound of `timeout_us` microseconds, on a shared-memory barrier
 * that nothing ever completes.  The wait gives up, the kernel records
 * GEMMI_ETIMEOUT in the device status word and returns normally; the context
 * stays usable.  Returns the status word's code read back by
 * gemmi_device_status() (GEMMI_ETIMEOUT when detection works).
 */
int gemmi_selftest_wait_timeout(int64_t timeout_us);

/*
 * Per-kernel timing for benchmarks.  While enabled, the library records a CUDA
 * event pair on the launching stream around each launch of the kernels below;
 * gemmi_kernel_time() waits for the recorded events and returns the summed
 * device time (milliseconds) and the number of timed launches of one kernel.
 * gemmi_kernel_timing(0|1) switches recording and resets the sums.
 *   GEMMI_KERNEL_SPLIT   : the limb split / conversion of A and B (one launch per call)
 *   GEMMI_KERNEL_TC_I16  : the tcgen05 int16 GEMM kernel
 *   GEMMI_KERNEL_TC_I8   : the tcgen05 int8 GEMM kernel
 *   GEMMI_KERNEL_SKINNY  : the skinny-M int16 kernel
 *   GEMMI_KERNEL_FUSED_I16 : the narrow-n int16 kernel that splits A on chip
 *   GEMMI_KERNEL_SRS     : the requantising pass of gemm_i16_srs
 *   GEMMI_KERNEL_TC_PAIR_I16 : the tcgen05 int16 GEMM kernel on SM pairs
 *   GEMMI_KERNEL_TC_PAIR_I8  : the tcgen05 int8 GEMM kernel on SM pairs
 *   GEMMI_KERNEL_TC_PAIR_I4  : the tcgen05 int4 GEMM kernel on SM pairs (E4M3 operands)
 *   GEMMI_KERNEL_ADD_I32     : gemm_i4's add of its scratch result into a C that the pair
 *                              kernel cannot reduce into directly
 *   GEMMI_KERNEL_CONVERT_I4  : gemm_i4's conversion of the packed operands to E4M3 planes
 *   GEMMI_KERNEL_TC_KARATSUBA : the three-product int16 kernel (GEMMI_OPT_KARATSUBA; its limb-sum
 *                              planes are timed with GEMMI_KERNEL_SPLIT)
 *   GEMMI_KERNEL_TC_PAIR_I16_AHEAD : the int16 GEMM kernel on SM pairs when its own warps split
 *                              the later row panels of A (GEMMI_OPT_SPLIT_AHEAD); such a call
 *                              counts here instead of GEMMI_KERNEL_TC_PAIR_I16
 *   GEMMI_KERNEL_CONV_ROWS   : gemmi_conv2d_i16's direct convolution kernel (GEMMI_OPT_CONV_ROWS;
 *                              the split of its weights is timed with GEMMI_KERNEL_SPLIT)
 */
enum { GEMMI_KERNEL_SPLIT = 0, GEMMI_KERNEL_TC_I16 = 1, GEMMI_KERNEL_TC_I8 = 2, GEMMI_KERNEL_SKINNY = 3,
       GEMMI_KERNEL_FUSED_I16 = 4, GEMMI_KERNEL_SRS = 5, GEMMI_KERNEL_TC_PAIR_I16 = 6, GEMMI_KERNEL_TC_PAIR_I8 = 7,
       GEMMI_KERNEL_TC_PAIR_I4 = 8, GEMMI_KERNEL_ADD_I32 = 9, GEMMI_KERNEL_CONVERT_I4 = 10,
       GEMMI_KERNEL_TC_KARATSUBA = 11, GEMMI_KERNEL_TC_PAIR_I16_AHEAD = 12, GEMMI_KERNEL_CONV_ROWS = 13,
       GEMMI_KERNEL_COUNT = 14 };
int gemmi_kernel_timing(int enable);
int gemmi_kernel_time(int kernel, double* total_ms, int64_t* launches);

/*
 * gemm_i16_noalloc -- gemm_i16 for callers that must not allocate device memory.
 * The paper has no counterpart; this entry point exists for deployment.  Some
 * callers cannot allocate at call time: an inference server that has given all
 * free device memory to its own pool at start-up (a cudaMalloc would fail), or a
 * latency-critical loop that cannot absorb the device-wide synchronisation of
 * growing or freeing a buffer.  This call allocates nothing: no cudaMalloc,
 * cudaFree or allocating library routine.  Its scratch (the fp16 limb planes of
 * A and B and a status word) is one fixed, file-scope device array of
 * GEMMI_NOALLOC_SCRATCH_BYTES that every GPU loading the library holds until the
 * process exits.
 *
 * Same operation, layout, pointer ownership (DEVICE pointers owned by the
 * caller) and bit-exact result as gemm_i16, always on the tensor-core path
 * (the limb split, then the one-SM-per-tile tcgen05 kernel, whose 128x128 tiles
 * cover problems of this size), asynchronous on `stream` (a cudaStream_t as
 * void*; NULL = legacy default stream).
 * Limit: 4*(m+n)*roundup(k,8) + 256 <= GEMMI_NOALLOC_SCRATCH_BYTES (for m = n = k,
 * up to about 2000); larger problems return GEMMI_EINVAL with a message saying so.
 * The first call on a device looks up the array's device address (with that
 * device current) and caches it; make that first call before any stream capture.
 * Every call shares the one array: calls that overlap on the GPU (on different
 * streams, or from several threads) race on it and must be serialised by the caller.
 * Every plane byte a call reads is written by that call first, so what an
 * earlier call left in the array never reaches C.
 * Device-side failures: both kernels bound their pipeline waits by
 * GEMMI_OPT_WAIT_TIMEOUT_US and record a wait that ran out in a status word at
 * the start of the array (sticky until read); gemmi_device_status() and
 * gemmi_device_status_stream() read and clear it.
 * Returns GEMMI_OK, GEMMI_EINVAL, GEMMI_ECUDA or GEMMI_EARCH.
 */
#define GEMMI_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)
int gemm_i16_noalloc(int64_t m, int64_t n, int64_t k,
                     const int16_t* A, int64_t lda,
                     const int16_t* B, int64_t ldb,
                     int64_t* C, int64_t ldc, void* stream);

/*
 * Failure-detection self-test of gemm_i16_noalloc's status word (no paper
 * counterpart, like the entry point itself): launches, on `stream`, the probe of
 * gemmi_selftest_wait_timeout with the word inside the fixed scratch array as
 * its status word (setting up the array's address on first use, as the entry
 * point does).  Allocates nothing.  Returns GEMMI_OK once launched; a following
 * gemmi_device_status_stream(stream) then returns GEMMI_ETIMEOUT.
 */
int gemmi_noalloc_selftest_wait_timeout(int64_t timeout_us, void* stream);

/*
 * Measurement aid (no counterpart in the paper): the read floor of the skinny-M
 * path.  Reads the k x n int16 matrix B (a DEVICE pointer, 16-byte aligned,
 * ldb % 8 == 0) exactly as the m <= 16 kernel streams its B -- the same grid,
 * TMA boxes, four-stage ring and programmatic dependent launch -- and discards
 * it.  Asynchronous on `stream`; a wait that runs out is reported by
 * gemmi_device_status().  Returns GEMMI_OK, GEMMI_EINVAL, GEMMI_ECUDA or
 * GEMMI_EARCH.
 */
int gemmi_stream_read_probe(int64_t k, int64_t n, const int16_t* B, int64_t ldb, void* stream);

/* Library version string. */
const char* gemmi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GEMMI_H */
