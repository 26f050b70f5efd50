// requant.cu -- the paper's micro-kernel output: C16 += srs(S, shift).
//
// The AIE micro-kernel (Section 5.2) ends by shifting, rounding and saturating
// its wide accumulator to 16 bits ("srs") and adding the result to the int16 C
// block with a plain 16-bit vector addition.  gemm_i16_srs computes the exact
// product S = A*B into an int64 scratch matrix with the regular GEMM paths and
// then runs this kernel, which applies, per entry,
//     R = S                                  for shift == 0,
//     R = floor((S + 2^(shift-1)) / 2^shift)  otherwise (round half up),
//     C16 = (C16 + clamp(R, -32768, 32767)) mod 2^16.
// The saturation needs the whole sum, so it cannot run inside the kernels that
// split a reduction across CTAs; this pass reads S once (8 bytes) and C once
// (2 bytes) and writes C (2 bytes) per entry: HBM-bound.
#include <cuda_runtime.h>

#include "internal.h"

namespace gemmi {
namespace {

constexpr int THREADS = 256;

__device__ __forceinline__ uint16_t srs_add(int64_t s, uint16_t c, int shift) {
  // arithmetic right shift of a signed value: floor division by 2^shift
  int64_t r = shift == 0 ? s : (s + (static_cast<int64_t>(1) << (shift - 1))) >> shift;
  r = r > 32767 ? 32767 : r < -32768 ? -32768 : r;
  return static_cast<uint16_t>(c + static_cast<uint16_t>(r));
}

// Four consecutive columns per thread; S rows are padded to a multiple of 8 entries by the caller
// (16-byte aligned vector loads), C takes an 8-byte vector access when vec_c is set.
__global__ void __launch_bounds__(THREADS)
srs_add_kernel(const int64_t* __restrict__ S, int64_t lds, int16_t* __restrict__ C, int64_t ldc, int64_t m,
               int64_t n, int shift, int vec_c) {
  const int64_t groups = (n + 3) / 4;
  const int64_t total = m * groups;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(THREADS) + threadIdx.x; g < total;
       g += static_cast<int64_t>(gridDim.x) * THREADS) {
    const int64_t i = g / groups;
    const int64_t j = (g - i * groups) * 4;
    const int64_t* srow = S + i * lds + j;
    const longlong2 s01 = *reinterpret_cast<const longlong2*>(srow);
    const longlong2 s23 = *reinterpret_cast<const longlong2*>(srow + 2);
    const int64_t sv[4] = {s01.x, s01.y, s23.x, s23.y};
    int16_t* crow = C + i * ldc + j;
    if (vec_c && j + 4 <= n) {
      uint2 cv = *reinterpret_cast<const uint2*>(crow);
      const uint16_t r0 = srs_add(sv[0], static_cast<uint16_t>(cv.x & 0xFFFFu), shift);
      const uint16_t r1 = srs_add(sv[1], static_cast<uint16_t>(cv.x >> 16), shift);
      const uint16_t r2 = srs_add(sv[2], static_cast<uint16_t>(cv.y & 0xFFFFu), shift);
      const uint16_t r3 = srs_add(sv[3], static_cast<uint16_t>(cv.y >> 16), shift);
      cv.x = static_cast<uint32_t>(r0) | (static_cast<uint32_t>(r1) << 16);
      cv.y = static_cast<uint32_t>(r2) | (static_cast<uint32_t>(r3) << 16);
      *reinterpret_cast<uint2*>(crow) = cv;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (j + q < n)
          crow[q] = static_cast<int16_t>(srs_add(sv[q], static_cast<uint16_t>(crow[q]), shift));
    }
  }
}

}  // namespace

cudaError_t srs_add_i16(const int64_t* S, int64_t lds, int16_t* C, int64_t ldc, int64_t m, int64_t n, int shift,
                        cudaStream_t s) {
  const int64_t total = m * ((n + 3) / 4);
  if (total <= 0) return cudaSuccess;
  int64_t blocks = (total + THREADS - 1) / THREADS;
  if (blocks > 152 * 16) blocks = 152 * 16;
  const int vec_c = (reinterpret_cast<uintptr_t>(C) % 8 == 0) && (ldc % 4 == 0);
  srs_add_kernel<<<static_cast<unsigned>(blocks), THREADS, 0, s>>>(S, lds, C, ldc, m, n, shift, vec_c);
  return cudaGetLastError();
}

}  // namespace gemmi
