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
//
// One launch converts both operands (or just one: a null operand is skipped): the first blocks of the grid stream A
// (16-byte loads, 2 x 16-byte stores per 8 elements), the rest transpose B in
// 64 x 64 tiles through shared memory (16-byte loads and stores on both sides).
// The kernel is bound by HBM: per int16 element 2 bytes are read and 4 written.
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

template <typename T>
struct Part {
  const T* src;
  int64_t ld;
  int64_t rows;   // A: m;  B: k (rows of B)
  int64_t cols;   // A: k;  B: n
  __half* p0;
  __half* p1;
  int64_t pitch;  // plane row pitch (elements)
  bool vec;       // 16-byte (int16) / 8-byte (int8) loads of 8 elements are aligned
};

template <typename T>
__device__ __forceinline__ void load8(const T* src, bool vec, int64_t valid, int (&v)[8]) {
  if (vec && valid >= 8) {
    if constexpr (sizeof(T) == 2) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(src));
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[2 * i] = static_cast<int16_t>(w[i] & 0xFFFFu);
        v[2 * i + 1] = static_cast<int16_t>(w[i] >> 16);
      }
    } else {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(src));
      const uint32_t w[2] = {u.x, u.y};
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = static_cast<int8_t>((w[i / 4] >> (8 * (i % 4))) & 0xFFu);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = (i < valid) ? static_cast<int>(src[i]) : 0;
  }
}

template <int NL>
__device__ __forceinline__ void store8(__half* p0, __half* p1, const int (&v)[8]) {
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
  *reinterpret_cast<uint4*>(p0) = *reinterpret_cast<const uint4*>(h);
  if constexpr (NL == 2) *reinterpret_cast<uint4*>(p1) = *reinterpret_cast<const uint4*>(l);
}

constexpr int TT = 64;      // transpose tile edge
constexpr int THREADS = 256;

template <typename T, int NL>
__global__ void __launch_bounds__(THREADS)
split_kernel(Part<T> a, Part<T> b, int a_blocks, int64_t b_tiles_j, int64_t b_tiles) {
  __shared__ int16_t tile[TT][TT + 8];
  if (static_cast<int>(blockIdx.x) < a_blocks) {
    // ---- A: m x k (lda) -> planes m x pitch, 8 consecutive elements per thread
    const int64_t groups_per_row = a.pitch / 8;
    const int64_t total = a.rows * groups_per_row;
    for (int64_t g = blockIdx.x * static_cast<int64_t>(THREADS) + threadIdx.x; g < total;
         g += static_cast<int64_t>(a_blocks) * THREADS) {
      const int64_t r = g / groups_per_row;
      const int64_t p0 = (g - r * groups_per_row) * 8;
      int v[8];
      load8(a.src + r * a.ld + p0, a.vec, a.cols - p0, v);
      store8<NL>(a.p0 + r * a.pitch + p0, a.p1 + r * a.pitch + p0, v);
    }
    return;
  }
  // ---- B: k x n (ldb) -> planes n x pitch (transposed), 64 x 64 tiles
  const int64_t nblk = gridDim.x - a_blocks;
  for (int64_t t = blockIdx.x - a_blocks; t < b_tiles; t += nblk) {
    const int64_t p_base = (t / b_tiles_j) * TT;  // reduction index = row of B
    const int64_t j_base = (t % b_tiles_j) * TT;  // column of B
#pragma unroll
    for (int q = threadIdx.x; q < TT * TT / 8; q += THREADS) {
      const int r = q >> 3;
      const int c8 = (q & 7) * 8;
      const int64_t p = p_base + r, j = j_base + c8;
      int v[8];
      if (p < b.rows) {
        load8(b.src + p * b.ld + j, b.vec, b.cols - j, v);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = 0;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) tile[r][c8 + i] = static_cast<int16_t>(v[i]);
    }
    __syncthreads();
#pragma unroll
    for (int q = threadIdx.x; q < TT * TT / 8; q += THREADS) {
      const int jj = q >> 3;
      const int pc = (q & 7) * 8;
      const int64_t j = j_base + jj, p = p_base + pc;
      if (j < b.cols && p < b.pitch) {
        int v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = tile[pc + i][jj];
        store8<NL>(b.p0 + j * b.pitch + p, b.p1 + j * b.pitch + p, v);
      }
    }
    __syncthreads();
  }
}

template <typename T, int NL>
cudaError_t launch(const T* A, int64_t lda, const T* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                   LimbPlanes pa, LimbPlanes pb, cudaStream_t s) {
  constexpr int64_t esz = sizeof(T);
  Part<T> a{A, lda, m, k, static_cast<__half*>(pa.plane[0]), static_cast<__half*>(pa.plane[NL - 1]), pa.pitch,
            reinterpret_cast<uintptr_t>(A) % (8 * esz) == 0 && (lda * esz) % (8 * esz) == 0};
  Part<T> b{B, ldb, k, n, static_cast<__half*>(pb.plane[0]), static_cast<__half*>(pb.plane[NL - 1]), pb.pitch,
            reinterpret_cast<uintptr_t>(B) % (8 * esz) == 0 && (ldb * esz) % (8 * esz) == 0};
  // A: about 8 elements per thread per grid-stride step; B: one 64 x 64 tile per block step.
  // A null operand is skipped (packing only the weights, or only the activations).
  const int64_t a_work = A != nullptr ? m * (pa.pitch / 8) : 0;
  int64_t a_blocks = (a_work + THREADS - 1) / THREADS;
  if (a_blocks > 152 * 8) a_blocks = 152 * 8;
  const int64_t tiles_p = (pb.pitch + TT - 1) / TT;  // cover the zero padding up to the pitch too
  const int64_t tiles_j = B != nullptr ? (n + TT - 1) / TT : 0;
  const int64_t b_tiles = tiles_p * tiles_j;
  int64_t b_blocks = b_tiles < 152 * 8 ? b_tiles : 152 * 8;
  if (a_blocks + b_blocks < 1) return cudaSuccess;
  split_kernel<T, NL><<<static_cast<unsigned>(a_blocks + b_blocks), THREADS, 0, s>>>(
      a, b, static_cast<int>(a_blocks), tiles_j, b_tiles);
  return cudaGetLastError();
}

}  // namespace

cudaError_t split_i16(const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                      LimbPlanes pa, LimbPlanes pb, cudaStream_t s) {
  return launch<int16_t, 2>(A, lda, B, ldb, m, n, k, pa, pb, s);
}

cudaError_t convert_i8(const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                       LimbPlanes pa, LimbPlanes pb, cudaStream_t s) {
  return launch<int8_t, 1>(A, lda, B, ldb, m, n, k, pa, pb, s);
}

}  // namespace gemmi
