// int4.cu -- operand conversion for the int4 GEMM, and the add of a scratch result into C.
//
// The int4 GEMM (a lower-precision point: Section 6.1 leaves the adaptation of the paper's INT16
// design to narrower types to future work) runs on the fp8 tensor-core path, tcgen05.mma kind::f8f6f4 with E4M3 operands:
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

// E4M3 codes of the 4-bit values, from the format's definition (sign bit, 4-bit exponent with
// bias 7, 3-bit fraction: |v| = 2^e * (1 + f/8)), four to a word, indexed by the low three bits of
// the nibble: kPos for nibbles 0..7 (values 0..7), kNeg for nibbles 8..15 (values -8..-1).
//   0 -> 0x00, 1 -> 0x38, 2 -> 0x40, 3 -> 0x44, 4 -> 0x48, 5 -> 0x4A, 6 -> 0x4C, 7 -> 0x4E,
//  -8 -> 0xD0, -7 -> 0xCE, -6 -> 0xCC, -5 -> 0xCA, -4 -> 0xC8, -3 -> 0xC4, -2 -> 0xC0, -1 -> 0xB8.
constexpr uint32_t kPos0 = 0x44403800u, kPos1 = 0x4E4C4A48u;
constexpr uint32_t kNeg0 = 0xCACCCED0u, kNeg1 = 0xB8C0C4C8u;

// Four nibbles, as 4-bit fields in bits 0-15 of `sel`, -> their four E4M3 bytes: two byte
// permutes look up the non-negative and the negative code of each, a third keeps one per byte
// by the nibble's top bit (byte selector i or i + 4).
__device__ __forceinline__ uint32_t e4m3x4(uint32_t sel) {
  const uint32_t idx = sel & 0x7777u;
  const uint32_t pos = __byte_perm(kPos0, kPos1, idx);
  const uint32_t neg = __byte_perm(kNeg0, kNeg1, idx);
  return __byte_perm(pos, neg, 0x3210u | ((sel >> 1) & 0x4444u));
}

// A word of eight packed nibbles (elements 8q .. 8q+7 of a row, in order) -> eight E4M3 bytes.
__device__ __forceinline__ uint2 e4m3x8_row(uint32_t w) { return make_uint2(e4m3x4(w & 0xFFFFu), e4m3x4(w >> 16)); }

// Four packed bytes of four consecutive rows (byte i from row p+i) -> the E4M3 bytes of the four
// low nibbles (column 2c) and of the four high nibbles (column 2c+1), each in row order.
__device__ __forceinline__ uint2 e4m3x4_cols(uint32_t w) {
  const uint32_t lo = w & 0x0F0F0F0Fu, hi = (w >> 4) & 0x0F0F0F0Fu;
  // gather the nibbles of bytes 0..3 into 4-bit fields 0..3
  const uint32_t sl = __byte_perm(lo | (lo >> 4), 0u, 0x4420u);
  const uint32_t sh = __byte_perm(hi | (hi >> 4), 0u, 0x4420u);
  return make_uint2(e4m3x4(sl), e4m3x4(sh));
}

// One launch converts both operands.  Blocks [0, a_blocks) convert A: block b takes the 512
// 16-byte units b*512 + tid and b*512 + 256 + tid of A's rows (unit u = row i, bytes 16c .. 16c+15
// with u = i * upr + c), each into 32 plane bytes.  The other blocks transpose B: block
// a_blocks + t takes tile t of 128 rows p x 64 packed bytes (128 columns j) into 128 plane rows
// of 128 bytes.
struct ConvertI4Params {
  const uint8_t* A;
  int64_t lda, m;
  uint8_t* pa;
  const uint8_t* B;
  int64_t ldb, n;
  uint8_t* pb;
  int64_t k, pitch;
  int64_t a_blocks, b_tiles_j;
  int a_vec, b_vec;
};
constexpr int TP = 128, TJB = 64;

__device__ __forceinline__ void convert_a_unit(const ConvertI4Params& P, int64_t i, int64_t c, uint4 w, bool have) {
  const int64_t wb = (P.k + 1) / 2;
  uint8_t* dst = P.pa + i * P.pitch + 32 * c;
  if (have) {
    const uint2 a = e4m3x8_row(w.x), b = e4m3x8_row(w.y), d = e4m3x8_row(w.z), e = e4m3x8_row(w.w);
    reinterpret_cast<uint4*>(dst)[0] = make_uint4(a.x, a.y, b.x, b.y);
    reinterpret_cast<uint4*>(dst)[1] = make_uint4(d.x, d.y, e.x, e.y);
    return;
  }
  // a row's last unit when it is partial or holds an odd k's spare nibble, or an operand whose
  // rows are not 16-byte aligned: byte by byte (the spare nibble becomes a zero, never read)
  const uint8_t* src = P.A + i * P.lda + 16 * c;
  const int64_t nb = (16 * c + 16 < wb) ? 16 : wb - 16 * c;
  for (int64_t b = 0; b < nb; ++b) {
    const uint32_t codes = e4m3x4(static_cast<uint32_t>(src[b]));
    dst[2 * b] = static_cast<uint8_t>(codes & 0xFFu);
    dst[2 * b + 1] = 2 * (16 * c + b) + 1 < P.k ? static_cast<uint8_t>((codes >> 8) & 0xFFu) : static_cast<uint8_t>(0);
  }
}

__global__ void __launch_bounds__(256) convert_i4_kernel(const ConvertI4Params P) {
  __shared__ __align__(16) uint8_t tile[TP][TJB];
  if (blockIdx.x < P.a_blocks) {
    // ---- A: two units per thread, both loads issued before either is converted
    const int64_t wb = (P.k + 1) / 2;
    const int64_t upr = (wb + 15) / 16;
    const int64_t units = P.m * upr;
    int64_t row[2], col[2];
    uint4 w[2];
    bool full[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t u = static_cast<int64_t>(blockIdx.x) * 512 + 256 * h + threadIdx.x;
      full[h] = false;
      w[h] = make_uint4(0u, 0u, 0u, 0u);
      row[h] = -1;
      if (u < units) {
        // unit -> (row, unit in row): 32-bit division when the unit count allows (the usual case)
        if (units <= 0xFFFFFFFFll) {
          const uint32_t q = static_cast<uint32_t>(u) / static_cast<uint32_t>(upr);
          row[h] = q;
          col[h] = static_cast<int64_t>(static_cast<uint32_t>(u) - q * static_cast<uint32_t>(upr));
        } else {
          row[h] = u / upr;
          col[h] = u - row[h] * upr;
        }
        // whole 16-byte units only, and not the one that holds an odd k's spare nibble
        const int64_t c = col[h];
        full[h] = P.a_vec && (16 * c + 16 < wb || (16 * c + 16 == wb && P.k % 2 == 0));
        if (full[h]) w[h] = __ldg(reinterpret_cast<const uint4*>(P.A + row[h] * P.lda + 16 * c));
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h)
      if (row[h] >= 0) convert_a_unit(P, row[h], col[h], w[h], full[h]);
    return;
  }
  // ---- B: one tile of 128 rows p x 64 packed bytes
  const int64_t t = static_cast<int64_t>(blockIdx.x) - P.a_blocks;
  const int64_t wbn = (P.n + 1) / 2;
  const int64_t jb0 = (t % P.b_tiles_j) * TJB;  // first packed byte of the tile (column 2 * jb0)
  const int64_t p0 = (t / P.b_tiles_j) * TP;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int r = (threadIdx.x >> 2) + 64 * h, q = threadIdx.x & 3;  // tile row r, 16-byte segment q
    const int64_t p = p0 + r;
    const int64_t b = jb0 + 16 * q;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (p < P.k) {
      const uint8_t* src = P.B + p * P.ldb + b;
      if (P.b_vec && b + 16 <= wbn) {
        v = __ldg(reinterpret_cast<const uint4*>(src));
      } else {
        uint32_t x[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int e = 0; e < 16; ++e)
          if (b + e < wbn) x[e / 4] |= static_cast<uint32_t>(src[e]) << (8 * (e % 4));
        v = make_uint4(x[0], x[1], x[2], x[3]);
      }
    }
    *reinterpret_cast<uint4*>(&tile[r][16 * q]) = v;
  }
  __syncthreads();
  // thread (jb, pq): packed byte column jb of tile rows 32pq .. 32pq+31 -> 32 plane bytes of
  // column 2*(jb0+jb) (low nibbles) and 32 of column 2*(jb0+jb)+1 (high nibbles)
  const int jb = threadIdx.x & 63, pq = threadIdx.x >> 6;
  const int64_t j = 2 * (jb0 + jb);
  const int64_t pstart = p0 + 32 * pq;
  if (j >= P.n || pstart >= P.pitch) return;
  uint32_t lo[8], hi[8];
#pragma unroll
  for (int g = 0; g < 8; ++g) {
    const int r = 32 * pq + 4 * g;
    const uint32_t word = __byte_perm(__byte_perm(tile[r][jb], tile[r + 1][jb], 0x0040u),
                                      __byte_perm(tile[r + 2][jb], tile[r + 3][jb], 0x0040u), 0x5410u);
    const uint2 c = e4m3x4_cols(word);
    lo[g] = c.x;
    hi[g] = c.y;
  }
  // the plane rows end at pitch, a multiple of 16: whole 16-byte units
  const bool second = pstart + 16 < P.pitch;
  uint4* d0 = reinterpret_cast<uint4*>(P.pb + j * P.pitch + pstart);
  d0[0] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
  if (second) d0[1] = make_uint4(lo[4], lo[5], lo[6], lo[7]);
  if (j + 1 < P.n) {
    uint4* d1 = reinterpret_cast<uint4*>(P.pb + (j + 1) * P.pitch + pstart);
    d1[0] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    if (second) d1[1] = make_uint4(hi[4], hi[5], hi[6], hi[7]);
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
  (void)num_sms;
  if (k <= 0) return cudaSuccess;
  ConvertI4Params P{};
  P.A = A;
  P.lda = lda;
  P.m = A != nullptr ? m : 0;
  P.pa = static_cast<uint8_t*>(pa.plane[0]);
  P.B = B;
  P.ldb = ldb;
  P.n = B != nullptr ? n : 0;
  P.pb = static_cast<uint8_t*>(pb.plane[0]);
  P.k = k;
  P.pitch = A != nullptr ? pa.pitch : pb.pitch;
  if (A != nullptr && B != nullptr && pa.pitch != pb.pitch) return cudaErrorInvalidValue;
  const int64_t a_units = P.m * (((k + 1) / 2 + 15) / 16);
  P.a_blocks = (a_units + 511) / 512;
  P.b_tiles_j = ((P.n + 1) / 2 + TJB - 1) / TJB;
  const int64_t b_tiles = P.n > 0 ? P.b_tiles_j * ((k + TP - 1) / TP) : 0;
  P.a_vec = A != nullptr && reinterpret_cast<uintptr_t>(A) % 16 == 0 && lda % 16 == 0;
  P.b_vec = B != nullptr && reinterpret_cast<uintptr_t>(B) % 16 == 0 && ldb % 16 == 0;
  const int64_t blocks = P.a_blocks + b_tiles;
  if (blocks == 0) return cudaSuccess;
  if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
  convert_i4_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(P);
  return cudaGetLastError();
}

cudaError_t add_into_i32(int32_t* C, int64_t ldc, const int32_t* T, int64_t ldt, int64_t m, int64_t n, int num_sms,
                         cudaStream_t s) {
  if (m <= 0 || n <= 0) return cudaSuccess;
  add_i32<<<grid_for(m * n, num_sms), 256, 0, s>>>(C, ldc, T, ldt, m, n);
  return cudaGetLastError();
}

}  // namespace gemmi
