// int4.cu -- operand conversion for the int4 GEMM, and the add of a scratch result into C.
//
// The int4 GEMM (the lower-precision point of Section 5.1: the paper carries its INT16 design to
// narrower types) runs on the fp8 tensor-core path, tcgen05.mma kind::f8f6f4 with E4M3 operands:
// every integer in [-8, 8] is an E4M3 value exactly (at most three significant bits), so the
// products, at most 64 in magnitude, are exact and so are fp32 sums of up to 2^18 of them.
//
// Operands arrive packed two to a byte (element with even index in the low nibble, odd index in
// the high nibble, two's complement).  The planes the GEMM reads are K-major E4M3 bytes: plane A
// holds row i of A at a.plane[0] + i * pitch, plane B holds column j of B (transposed) at
// b.plane[0] + j * pitch; pitch (bytes) is a multiple of 16, bytes past k are not read.
#include <cstdint>

#include "internal.h"

namespace gemmi {
namespace {

// The E4M3 encoding of an integer v in [-8, 8], from the format's definition: sign bit, 4-bit
// exponent with bias 7, 3-bit fraction; |v| = 2^e * (1 + f/8) with e = floor(log2 |v|).
__device__ __forceinline__ uint32_t e4m3_of_int(int v) {
  if (v == 0) return 0u;
  const uint32_t sign = v < 0 ? 0x80u : 0u;
  const int a = v < 0 ? -v : v;
  const int e = 31 - __clz(a);
  const int f = ((a << 3) >> e) - 8;
  return sign | (static_cast<uint32_t>(e + 7) << 3) | static_cast<uint32_t>(f);
}

__device__ __forceinline__ int nibble_value(uint32_t nib) { return nib >= 8u ? static_cast<int>(nib) - 16 : static_cast<int>(nib); }

// Shared table: packed byte -> its two E4M3 bytes (low nibble's code in the low byte).
__device__ __forceinline__ void fill_pair_table(uint16_t* lut) {
  for (int b = threadIdx.x; b < 256; b += blockDim.x)
    lut[b] = static_cast<uint16_t>(e4m3_of_int(nibble_value(b & 15u)) | (e4m3_of_int(nibble_value(b >> 4)) << 8));
}

__device__ __forceinline__ uint32_t pairs_of4(const uint16_t* lut, uint32_t w, int half) {
  // two packed bytes of w (half 0: bytes 0-1, 1: bytes 2-3) -> four E4M3 bytes
  const uint32_t b0 = (w >> (16 * half)) & 0xFFu, b1 = (w >> (16 * half + 8)) & 0xFFu;
  return static_cast<uint32_t>(lut[b0]) | (static_cast<uint32_t>(lut[b1]) << 16);
}

// A (m rows of wb = ceil(k/2) packed bytes, row pitch lda bytes) -> plane rows of k E4M3 bytes.
// Thread t converts packed bytes 16c .. 16c+15 of row i (t = i * cpr + c) into 32 plane bytes.
template <bool VEC>
__global__ void __launch_bounds__(256) convert_rows_i4(const uint8_t* __restrict__ A, int64_t lda, int64_t m,
                                                       int64_t k, uint8_t* __restrict__ plane, int64_t pitch) {
  __shared__ uint16_t lut[256];
  fill_pair_table(lut);
  __syncthreads();
  const int64_t wb = (k + 1) / 2;
  const int64_t cpr = (wb + 15) / 16;
  const int64_t total = m * cpr;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t i = t / cpr;
    const int64_t c = t - i * cpr;
    const uint8_t* src = A + i * lda + 16 * c;
    uint8_t* dst = plane + i * pitch + 32 * c;
    if (VEC && 16 * c + 16 <= wb && (k % 2 == 0 || 16 * c + 16 < wb)) {
      const uint4 w = __ldg(reinterpret_cast<const uint4*>(src));
      uint4 lo, hi;
      lo.x = pairs_of4(lut, w.x, 0);
      lo.y = pairs_of4(lut, w.x, 1);
      lo.z = pairs_of4(lut, w.y, 0);
      lo.w = pairs_of4(lut, w.y, 1);
      hi.x = pairs_of4(lut, w.z, 0);
      hi.y = pairs_of4(lut, w.z, 1);
      hi.z = pairs_of4(lut, w.w, 0);
      hi.w = pairs_of4(lut, w.w, 1);
      reinterpret_cast<uint4*>(dst)[0] = lo;
      reinterpret_cast<uint4*>(dst)[1] = hi;
    } else {
      // a row's tail (or an unaligned operand): byte by byte; the spare high nibble of an odd
      // k's last byte becomes a zero (the GEMM never reads it)
      const int64_t end = (16 * c + 16 < wb) ? 16 * c + 16 : wb;
      for (int64_t b = 16 * c; b < end; ++b) {
        const uint32_t byte = src[b - 16 * c];
        dst[2 * (b - 16 * c)] = static_cast<uint8_t>(e4m3_of_int(nibble_value(byte & 15u)));
        dst[2 * (b - 16 * c) + 1] =
            2 * b + 1 < k ? static_cast<uint8_t>(e4m3_of_int(nibble_value(byte >> 4))) : static_cast<uint8_t>(0);
      }
    }
  }
}

// B (k rows of wbn = ceil(n/2) packed bytes, pitch ldb) -> plane rows j (one per column of B) of k
// E4M3 bytes.  A block transposes tiles of 64 rows p x 64 packed bytes (128 columns j), tile
// t = pt * ntj + jt for t = blockIdx.x, blockIdx.x + gridDim.x, ...
constexpr int TP = 64, TJB = 64;
template <bool VEC>
__global__ void __launch_bounds__(256) convert_cols_i4(const uint8_t* __restrict__ B, int64_t ldb, int64_t k,
                                                       int64_t n, uint8_t* __restrict__ plane, int64_t pitch) {
  __shared__ uint8_t lut8[16];
  __shared__ __align__(16) uint8_t tile[TP][TJB + 16];
  if (threadIdx.x < 16) lut8[threadIdx.x] = static_cast<uint8_t>(e4m3_of_int(nibble_value(threadIdx.x)));
  const int64_t wbn = (n + 1) / 2;
  const int64_t ntj = (wbn + TJB - 1) / TJB, ntp = (k + TP - 1) / TP;
  for (int64_t t = blockIdx.x; t < ntj * ntp; t += gridDim.x) {
    const int64_t jb0 = (t % ntj) * TJB;  // first packed byte (column j0 = 2 * jb0)
    const int64_t p0 = (t / ntj) * TP;
    __syncthreads();  // the previous tile has been read
    {
      const int r = threadIdx.x / 4, q = threadIdx.x % 4;  // row r of the tile, 16-byte segment q
      const int64_t p = p0 + r;
      const int64_t b = jb0 + 16 * q;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (p < k) {
        const uint8_t* src = B + p * ldb + b;
        if (VEC && b + 16 <= wbn) {
          v = __ldg(reinterpret_cast<const uint4*>(src));
        } else {
          uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
          for (int e = 0; e < 16; ++e)
            if (b + e < wbn) w[e / 4] |= static_cast<uint32_t>(src[e]) << (8 * (e % 4));
          v = make_uint4(w[0], w[1], w[2], w[3]);
        }
      }
      *reinterpret_cast<uint4*>(&tile[r][16 * q]) = v;
    }
    __syncthreads();
    // thread t writes plane row j = 2 * jb0 + t / 2, bytes p0 + 32 * (t % 2) .. +31
    const int jl = threadIdx.x / 2, h = threadIdx.x % 2;
    const int64_t j = 2 * jb0 + jl;
    if (j >= n) continue;
    uint8_t* dst = plane + j * pitch + p0 + 32 * h;
    const int shift = 4 * (jl & 1);
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      if (p0 + 32 * h + 16 * s >= pitch) break;  // pitch is a multiple of 16: whole 16-byte units
      uint32_t w[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        uint32_t word = 0;
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) {
          const int r = 32 * h + 16 * s + 4 * e + bb;
          const uint32_t nib = (tile[r][jl / 2] >> shift) & 15u;
          word |= static_cast<uint32_t>(lut8[nib]) << (8 * bb);
        }
        w[e] = word;
      }
      reinterpret_cast<uint4*>(dst)[s] = make_uint4(w[0], w[1], w[2], w[3]);
    }
  }
}

__global__ void __launch_bounds__(256) add_i32(int32_t* __restrict__ C, int64_t ldc, const int32_t* __restrict__ T,
                                               int64_t ldt, int64_t m, int64_t n) {
  const int64_t total = m * n;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t i = t / n, j = t - i * n;
    // two's-complement wrap, as the GEMM's sums: add in unsigned arithmetic
    C[i * ldc + j] = static_cast<int32_t>(static_cast<uint32_t>(C[i * ldc + j]) + static_cast<uint32_t>(T[i * ldt + j]));
  }
}

unsigned grid_for(int64_t work, int num_sms) {
  const int64_t blocks = (work + 255) / 256;
  const int64_t cap = static_cast<int64_t>(num_sms > 0 ? num_sms : 148) * 8;
  return static_cast<unsigned>(blocks < 1 ? 1 : (blocks < cap ? blocks : cap));
}

}  // namespace

cudaError_t convert_i4(const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                       LimbPlanes pa, LimbPlanes pb, int num_sms, cudaStream_t s) {
  if (k <= 0) return cudaSuccess;
  if (A != nullptr && m > 0) {
    const bool vec = reinterpret_cast<uintptr_t>(A) % 16 == 0 && lda % 16 == 0;
    const int64_t work = m * (((k + 1) / 2 + 15) / 16);
    const unsigned g = grid_for(work, num_sms);
    if (vec) convert_rows_i4<true><<<g, 256, 0, s>>>(A, lda, m, k, static_cast<uint8_t*>(pa.plane[0]), pa.pitch);
    else convert_rows_i4<false><<<g, 256, 0, s>>>(A, lda, m, k, static_cast<uint8_t*>(pa.plane[0]), pa.pitch);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (B != nullptr && n > 0) {
    const bool vec = reinterpret_cast<uintptr_t>(B) % 16 == 0 && ldb % 16 == 0;
    const int64_t tiles = (((n + 1) / 2 + TJB - 1) / TJB) * ((k + TP - 1) / TP);
    const int64_t cap = static_cast<int64_t>(num_sms > 0 ? num_sms : 148) * 8;
    const unsigned g = static_cast<unsigned>(tiles < cap ? tiles : cap);
    if (vec) convert_cols_i4<true><<<g, 256, 0, s>>>(B, ldb, k, n, static_cast<uint8_t*>(pb.plane[0]), pb.pitch);
    else convert_cols_i4<false><<<g, 256, 0, s>>>(B, ldb, k, n, static_cast<uint8_t*>(pb.plane[0]), pb.pitch);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

cudaError_t add_into_i32(int32_t* C, int64_t ldc, const int32_t* T, int64_t ldt, int64_t m, int64_t n, int num_sms,
                         cudaStream_t s) {
  if (m <= 0 || n <= 0) return cudaSuccess;
  add_i32<<<grid_for(m * n, num_sms), 256, 0, s>>>(C, ldc, T, ldt, m, n);
  return cudaGetLastError();
}

}  // namespace gemmi
