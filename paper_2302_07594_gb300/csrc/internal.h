// internal.h -- host-side interfaces between the C ABI (api.cu) and the kernels.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace gemmi {

// Limb planes of one operand: NL fp16 planes of `rows` x `pitch` elements (K-major:
// element (r, p) of plane l at planes[l][r * pitch + p]).  pitch is a multiple of 8.  The third
// plane (s = h + l) is used by the Karatsuba variant only.
struct LimbPlanes {
  void* plane[3];
  int64_t rows;
  int64_t pitch;
};

// ---- split.cu: operands -> fp16 limb planes (K-major).
// int16: two centred 8-bit limbs, a = 256*h + l, h in [-128,128], l in [-128,127].
// int8: one plane holding the value itself.
// One launch converts both operands: A (m x k, lda) -> pa (rows m), B (k x n, ldb) -> pb (rows n).
// A null A (or B) skips that operand.
// Operands whose base is 16-byte aligned with a row stride that is a multiple of 16 bytes are
// streamed through shared memory by TMA (every wait bounded by timeout_ns; a timeout is recorded
// in *status when status is not null); others take a plain-load kernel.
cudaError_t split_i16(const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                      LimbPlanes pa, LimbPlanes pb, cudaStream_t s, uint32_t* status = nullptr,
                      uint64_t timeout_ns = 4000000000ull);
cudaError_t convert_i8(const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                       LimbPlanes pa, LimbPlanes pb, cudaStream_t s, uint32_t* status = nullptr,
                       uint64_t timeout_ns = 4000000000ull);
// The Karatsuba variant's third plane of each operand: plane[2] = plane[0] + plane[1] (h + l,
// exact in fp16), for the `rows` x `pitch` planes of pa and pb (an operand with null plane[2] is
// skipped).
cudaError_t limb_sum_planes(LimbPlanes pa, LimbPlanes pb, int num_sms, cudaStream_t s);

// ---- gemm_tc.cu: tcgen05 GEMM on limb planes, C (int64 for NL=2, int32 for NL=1) += combine(limb products).
struct TcGemmArgs {
  int64_t m, n, k;
  LimbPlanes a;  // rows = m
  LimbPlanes b;  // rows = n (B transposed to K-major)
  void* C;
  int64_t ldc;
  uint32_t* status;
  uint64_t timeout_ns;
  int num_sms;
  int chunk_scale;  // 1: exact-sum chunks keep partial sums within 2^23; 2: within 2^24 (half the drains)
  int group_m;   // tile raster band height (row tiles), 0 = default
  int hint_a;    // L2 policy for A / B tile loads: 0 normal, 1 evict_last, 2 evict_first
  int hint_b;
  // Overlapped A split (tc_pair_gemm_i16 only).  When a_raw is not null, the caller has split
  // only A's row panels (128 rows each) below ahead_first into args.a; two extra warps per CTA
  // split the remaining panels from a_raw (16-byte aligned, lda % 8 == 0, k % 8 == 0, planes of
  // pitch k) while the tensor cores work on the earlier ones, and each tile's loads wait until
  // its panel is complete.  ahead: 2 + (number of row panels) words, zeroed by the caller before
  // the launch.
  const int16_t* a_raw = nullptr;
  int64_t lda = 0;
  uint32_t* ahead = nullptr;
  int ahead_first = 0;
};
cudaError_t tc_gemm_i16(const TcGemmArgs& args, cudaStream_t s, const char** why);
cudaError_t tc_gemm_i8(const TcGemmArgs& args, cudaStream_t s, const char** why);
// int16 by Karatsuba's three products: args.a / args.b hold three planes each (h, l, h + l).
cudaError_t tc_gemm_i16_karatsuba(const TcGemmArgs& args, cudaStream_t s, const char** why);

// ---- gemm_pair.cu: the same GEMM on SM pairs (tcgen05 cta_group::2).  The kernel adds into C with
// bulk reductions: C 16-byte aligned and ldc * sizeof(C element) a multiple of 16.
cudaError_t tc_pair_gemm_i16(const TcGemmArgs& args, cudaStream_t s, const char** why);
// Row panels of A (128 rows each) that the first wave of pair-kernel tiles reads, for an int16
// GEMM of m x n outputs with raster band group_m (0 = the default) on num_sms SMs: the panels the
// caller splits before an overlapped-split launch.
int pair_first_wave_panels(int64_t m, int64_t n, int group_m, int num_sms);
cudaError_t tc_pair_gemm_i8(const TcGemmArgs& args, cudaStream_t s, const char** why);
// int4: args.a / args.b hold one E4M3 plane each (int4.cu), pitch in bytes; C is int32.
cudaError_t tc_pair_gemm_i4(const TcGemmArgs& args, cudaStream_t s, const char** why);

// ---- int4.cu: packed int4 operands -> K-major E4M3 planes (pitch in bytes, a multiple of 16).
// A: m x k values, two per byte along the row (even index in the low nibble), row pitch lda bytes;
// B: k x n values packed along its rows (pitch ldb bytes), written transposed (rows = n).
// A null A (or B) skips that operand.
cudaError_t convert_i4(const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                       LimbPlanes pa, LimbPlanes pb, int num_sms, cudaStream_t s);
// C (m x n, pitch ldc) += T (pitch ldt), int32 modulo 2^32.
cudaError_t add_into_i32(int32_t* C, int64_t ldc, const int32_t* T, int64_t ldt, int64_t m, int64_t n, int num_sms,
                         cudaStream_t s);

// ---- gemm_fused.cu: int16 GEMM, n <= 64 per tile column, A read raw (int16) and split on chip.
struct FusedArgs {
  int64_t m, n, k;
  const int16_t* A;  // m x k row-major; base 16-byte aligned and lda % 8 == 0 (TMA)
  int64_t lda;
  LimbPlanes b;      // B's two limb planes (rows = n)
  int64_t* C;
  int64_t ldc;
  uint32_t* status;
  uint64_t timeout_ns;
  int num_sms;
  int chunk_scale;
  int group_m;
  // Implicit IM2COL (conv != 0): A is not a matrix but an NHWC tensor of conv_pixels pixels of
  // conv_cin channels (base 16-byte aligned, conv_cin % 64 == 0); row m of the lowered matrix is
  // output pixel m of a stride-1 convolution with Ho == H and Wo == W, and its K block kb is the
  // 64 channels cb = kb % (cin / 64) of filter tap (r, s) = (tap / S, tap % S), tap = kb / (cin / 64).
  int conv = 0;
  int64_t conv_pixels = 0;
  int conv_cin = 0, conv_h = 0, conv_w = 0, conv_s = 0, conv_ph = 0, conv_pw = 0;
};
cudaError_t tc_gemm_fused_i16(const FusedArgs& args, cudaStream_t s, const char** why);

// ---- conv_rows.cu: "same" stride-1 int16 convolution with 64 input channels, at most 64 output
// channels, odd R and S; each input pixel split once per tile (the filter taps are shifted windows
// of the split rows).
struct ConvRowsArgs {
  const int16_t* X;  // N x H x W x 64 (NHWC), 16-byte aligned
  int64_t N, H, W, R, S, cout;
  LimbPlanes b;      // the lowered weights' limb planes (rows = cout, K = R*S*64)
  int64_t* Y;        // N x H x W x cout (NHWC), 16-byte aligned, cout even
  uint32_t* status;
  uint64_t timeout_ns;
  int num_sms;
  int chunk_scale;
};
// The tile geometry of the direct convolution for image width W and an R x S filter, or false when
// the kernel does not cover the shape (even R or S, R*S above 12, R*S*64 above one exact chunk of
// 512*chunk_scale, padded rows wider than 128 pixels or a shifted window beyond its buffer).
bool conv_rows_geometry(int64_t W, int64_t R, int64_t S, int chunk_scale, int* Wp, int* T, int* PB, int* wpad);
cudaError_t conv_rows_i16(const ConvRowsArgs& args, cudaStream_t s, const char** why);
// ---- skinny.cu: m <= 16 int16 GEMM streaming B once.
struct SkinnyArgs {
  int64_t m, n, k;
  const int16_t* A;  // m x k, row-major (any alignment)
  int64_t lda;
  const int16_t* B;  // k x n, row-major, 16-byte aligned base, ldb % 8 == 0
  int64_t ldb;
  int64_t* C;
  int64_t ldc;
  uint32_t* status;
  uint64_t timeout_ns;
  int num_sms;
  int ksplit;  // 0 = automatic
};
cudaError_t skinny_gemm_i16(const SkinnyArgs& args, cudaStream_t s, const char** why);

// ---- probe.cu: reads a k x n int16 matrix (16-byte aligned, ldb % 8 == 0) the way skinny.cu
// streams B, and discards it (the skinny GEMM's read floor).
cudaError_t stream_read_probe(const int16_t* B, int64_t k, int64_t n, int64_t ldb, int num_sms, uint32_t* status,
                              uint64_t timeout_ns, cudaStream_t s, const char** why);

// ---- error text of the calling thread, as returned by gemmi_last_error().
void record_error(const char* msg);

// ---- requant.cu: C16 += srs(S, shift), S an int64 m x n matrix with row pitch lds (a multiple of 8).
cudaError_t srs_add_i16(const int64_t* S, int64_t lds, int16_t* C, int64_t ldc, int64_t m, int64_t n, int shift,
                        cudaStream_t s);

// ---- im2col.cu: the explicit IM2COL lowering of a stride-1 convolution (lda % 8 == 0, Aout 16-byte aligned).
cudaError_t im2col_i16(const int16_t* X, int16_t* Aout, int64_t lda, int64_t N, int64_t H, int64_t W, int64_t Cin,
                       int64_t R, int64_t S, int64_t ph, int64_t pw, cudaStream_t s);

// ---- noalloc.cu: device address of the allocation-free entry point's status word on device `dev`
// (inside its static scratch array), or null when that entry point has not run there.
uint32_t* noalloc_status_word(int dev);

// ---- selftest of the bounded wait.
cudaError_t launch_wait_timeout_probe(uint32_t* status, uint64_t timeout_ns, cudaStream_t s);

// Tensor-map encoder from the driver (resolved once through the runtime).  dtype: 0 = 16-bit
// integer, 1 = fp16, 2 = 8-bit integer, 3 = 64-bit integer, 4 = 32-bit integer (unsigned types:
// reductions through them add modulo 2^64 / 2^32).  row_bytes is the byte stride between rows.
bool encode_tensor_map_2d(void* map, int dtype, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle_bytes,
                          const char** why);

}  // namespace gemmi
