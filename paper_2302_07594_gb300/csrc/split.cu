// split.cu -- operand packing: integer operands -> fp16 limb planes in K-major order.
//
// This is the packing step of the paper's blocked GEMM (Section 4.1, the
// routines that copy A and B into the buffers A_c and B_c, and Section 5.1,
// where the activation operand is packed at run time), re-targeted: instead of
// re-ordering into micro-panels, each int16 value a is written as two exact
// fp16 "limbs" so the tensor cores can multiply them:
//     h = floor((a + 128) / 256)  in [-128, 128],   l = a - 256*h  in [-128, 127],
// so a = 256*h + l and every limb product is at most 2^14 in magnitude.
// int8 values are exact in fp16 and are written unchanged (one plane).
//
// Both operands end up K-major (the reduction index is contiguous): A keeps
// its row-major layout; B (k x n, row-major) is transposed to n x k.  Plane
// rows have a pitch that is a multiple of 8 elements (16 bytes), which the TMA
// tensor maps require.  Pitch columns at and beyond k are written as zero.
#include <cuda_fp16.h>

#include "internal.h"

namespace gemmi {
namespace {

// Every integer of magnitude <= 2048 is exactly representable in fp16 (11-bit significand).
__device__ __forceinline__ __half to_half_exact(int v) { return __int2half_rn(v); }

__device__ __forceinline__ void limbs16(int a, __half& h, __half& l) {
  const int hi = (a + 128) >> 8;  // arithmetic shift = floor division by 256
  const int lo = a - (hi << 8);
  h = to_half_exact(hi);
  l = to_half_exact(lo);
}

// A: m x k (lda) -> planes m x pitch.  One thread per 8 consecutive elements of a row.
template <typename T, int NL>
__global__ void split_rows_kernel(const T* __restrict__ A, int64_t lda, int64_t m, int64_t k,
                                  __half* __restrict__ P0, __half* __restrict__ P1, int64_t pitch, bool vec) {
  const int64_t groups_per_row = pitch / 8;
  const int64_t total = m * groups_per_row;
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = g / groups_per_row;
    const int64_t p0 = (g - r * groups_per_row) * 8;
    const T* src = A + r * lda + p0;
    int v[8];
    if (vec && p0 + 8 <= k) {
      if constexpr (sizeof(T) == 2) {
        const uint4 u = *reinterpret_cast<const uint4*>(src);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          v[2 * i] = static_cast<int16_t>(w[i] & 0xFFFFu);
          v[2 * i + 1] = static_cast<int16_t>(w[i] >> 16);
        }
      } else {
        const uint2 u = *reinterpret_cast<const uint2*>(src);
        const uint32_t w[2] = {u.x, u.y};
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = static_cast<int8_t>((w[i / 4] >> (8 * (i % 4))) & 0xFFu);
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = (p0 + i < k) ? static_cast<int>(src[i]) : 0;
    }
    __align__(16) __half h[8];
    __align__(16) __half l[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if constexpr (NL == 2) {
        limbs16(v[i], h[i], l[i]);
      } else {
        h[i] = to_half_exact(v[i]);
      }
    }
    *reinterpret_cast<uint4*>(P0 + r * pitch + p0) = *reinterpret_cast<const uint4*>(h);
    if constexpr (NL == 2) *reinterpret_cast<uint4*>(P1 + r * pitch + p0) = *reinterpret_cast<const uint4*>(l);
  }
}

// B: k x n (ldb) -> planes n x pitch (transposed).  64 x 64 tiles through shared memory.
constexpr int TT = 64;

template <typename T, int NL>
__global__ void split_cols_kernel(const T* __restrict__ B, int64_t ldb, int64_t k, int64_t n,
                                  __half* __restrict__ P0, __half* __restrict__ P1, int64_t pitch) {
  __shared__ int16_t tile[TT][TT + 2];
  const int64_t p_base = static_cast<int64_t>(blockIdx.x) * TT;  // reduction index (rows of B)
  const int64_t j_base = static_cast<int64_t>(blockIdx.y) * TT;  // column of B
  const int tx = threadIdx.x % TT;
  const int ty = threadIdx.x / TT;  // 0..3
  for (int r = ty; r < TT; r += 4) {
    const int64_t p = p_base + r, j = j_base + tx;
    tile[r][tx] = (p < k && j < n) ? static_cast<int16_t>(B[p * ldb + j]) : static_cast<int16_t>(0);
  }
  __syncthreads();
  // write: row j of the planes, columns p (zero beyond k up to the pitch)
  for (int r = ty; r < TT; r += 4) {
    const int64_t j = j_base + r, p = p_base + tx;
    if (j < n && p < pitch) {
      const int v = tile[tx][r];
      if constexpr (NL == 2) {
        __half h, l;
        limbs16(v, h, l);
        P0[j * pitch + p] = h;
        P1[j * pitch + p] = l;
      } else {
        P0[j * pitch + p] = to_half_exact(v);
      }
    }
  }
}

int grid_for(int64_t work, int threads) {
  int64_t b = (work + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 152 * 32) b = 152 * 32;
  return static_cast<int>(b);
}

template <typename T, int NL>
cudaError_t rows_impl(const T* A, int64_t lda, int64_t m, int64_t k, LimbPlanes out, cudaStream_t s) {
  const bool vec = (reinterpret_cast<uintptr_t>(A) % 16 == 0) && ((lda * static_cast<int64_t>(sizeof(T))) % 16 == 0);
  const int64_t work = m * (out.pitch / 8);
  split_rows_kernel<T, NL><<<grid_for(work, 256), 256, 0, s>>>(A, lda, m, k, static_cast<__half*>(out.plane[0]),
                                                               static_cast<__half*>(out.plane[1]), out.pitch, vec);
  return cudaGetLastError();
}

template <typename T, int NL>
cudaError_t cols_impl(const T* B, int64_t ldb, int64_t k, int64_t n, LimbPlanes out, cudaStream_t s) {
  const int64_t gp = (out.pitch + TT - 1) / TT;  // cover the zero padding up to the pitch too
  const int64_t gj = (n + TT - 1) / TT;
  if (gp > 0x7FFFFFFF || gj > 65535) return cudaErrorInvalidValue;
  dim3 grid(static_cast<unsigned>(gp), static_cast<unsigned>(gj));
  split_cols_kernel<T, NL><<<grid, 256, 0, s>>>(B, ldb, k, n, static_cast<__half*>(out.plane[0]),
                                                static_cast<__half*>(out.plane[1]), out.pitch);
  return cudaGetLastError();
}

}  // namespace

cudaError_t split_rows_i16(const int16_t* A, int64_t lda, int64_t m, int64_t k, LimbPlanes out, cudaStream_t s) {
  return rows_impl<int16_t, 2>(A, lda, m, k, out, s);
}
cudaError_t split_cols_i16(const int16_t* B, int64_t ldb, int64_t k, int64_t n, LimbPlanes out, cudaStream_t s) {
  return cols_impl<int16_t, 2>(B, ldb, k, n, out, s);
}
cudaError_t convert_rows_i8(const int8_t* A, int64_t lda, int64_t m, int64_t k, LimbPlanes out, cudaStream_t s) {
  return rows_impl<int8_t, 1>(A, lda, m, k, out, s);
}
cudaError_t convert_cols_i8(const int8_t* B, int64_t ldb, int64_t k, int64_t n, LimbPlanes out, cudaStream_t s) {
  return cols_impl<int8_t, 1>(B, ldb, k, n, out, s);
}

}  // namespace gemmi
