// skinny.cu -- exact int16 GEMM C (int64) += A*B for a small number of rows m <= 16.
//
// With m <= 16 (a batch of a few samples through a fully-connected layer) the
// GEMM of Section 4.1 is bound by streaming B (k x n) once from HBM: every B
// element is used m times only.  The paper notes that DL GEMMs often have one
// large and two small dimensions (Section 2, IM2COL lowering).  This kernel is
// built around the stream of B:
//
//   * B is cut into column blocks of 32 (64 bytes of int16 per row); each CTA
//     owns one column block and a range of the reduction dimension, and a
//     producer warp streams 128-row x 32-column tiles of it into a ring of
//     shared-memory stages with 2-D TMA loads (64-byte swizzle);
//   * eight consumer warps each take a 16-row slab of every stage, read it
//     transposed with ldmatrix (so that it is the "A" operand of
//     C^T = B^T A^T), split each int16 into 8-bit limbs
//         b = 256*hi + lo,  hi = b >> 8 in [-128,127],  lo = b & 255 in [0,255],
//     exactly representable in fp16, and multiply on the tensor cores with
//     mma.sync m16n8k16 (fp16 in, fp32 accumulate) against the limbs of A;
//   * three fp32 accumulator sets HH, X, LL hold exact integer sums while every
//     partial sum stays below 2^23 (a warp's run of 128 reduction indices:
//     128 * 255 * 255 < 2^23), then are drained into int64 registers as
//     HH*2^16 + X*2^8 + LL;
//   * the eight warps' int64 partials are summed in shared memory and added
//     into C (plain read-modify-write when one CTA owns the whole reduction,
//     64-bit atomic adds -- exact and order-independent modulo 2^64 -- when the
//     reduction dimension is split across CTAs).
#include <cuda.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"

namespace gemmi {
namespace {

constexpr int JB = 32;          // columns of B per CTA
constexpr int KS = 128;         // rows of B per stage
constexpr int STAGES = 8;
constexpr int STAGE_BYTES = KS * JB * 2;  // 8 KB
constexpr int NCONS = 8;        // consumer warps, one 16-row slab of a stage each
constexpr int THREADS = (NCONS + 1) * 32;
constexpr int DRAIN_EVERY = 8;  // stages per drain: 8 k-steps of 16 = 128 reduction indices per warp
constexpr uint32_t STATUS_TIMEOUT = 4;

struct SkParams {
  int64_t m, n, k;
  const int16_t* A;
  int64_t lda;
  int64_t* C;
  int64_t ldc;
  int64_t stages_per_cta;   // K range of one CTA, in stages
  int64_t total_stages;
  int atomic_out;
  int a_vec;                // A rows 4-byte aligned: 32-bit fragment loads
  uint64_t timeout_ns;
  uint32_t* status;
};

template <int NT>
constexpr size_t sk_smem() {
  return 1024 + STAGES * STAGE_BYTES + static_cast<size_t>(NCONS) * (2 * NT * 4 * 32) * 8 + 8 * (2 * STAGES) + 16;
}

// int16 pair -> fp16 pairs of its high (signed) and low (unsigned) bytes, exactly.
// 0x64xx as fp16 is 1024 + xx, so the byte is recovered by one subtraction.
__device__ __forceinline__ void split_pair(uint32_t x, uint32_t& hi, uint32_t& lo) {
  const uint32_t lo_bits = (x & 0x00FF00FFu) | 0x64006400u;                // 1024 + lo
  const uint32_t hi_bits = ((x >> 8) & 0x00FF00FFu) ^ 0x64806480u;         // 1024 + (hi + 128)
  const __half2 l = __hsub2(*reinterpret_cast<const __half2*>(&lo_bits), __half2half2(__ushort_as_half(0x6400)));
  const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&hi_bits), __half2half2(__ushort_as_half(0x6480)));
  lo = *reinterpret_cast<const uint32_t*>(&l);
  hi = *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// Two consecutive reduction indices p, p+1 of row i of A as a packed int16 pair (zero outside).
__device__ __forceinline__ uint32_t load_a_pair(const SkParams& P, int64_t i, int64_t p) {
  if (i >= P.m || p >= P.k) return 0u;
  const int16_t* row = P.A + i * P.lda;
  if (P.a_vec && p + 1 < P.k) return __ldg(reinterpret_cast<const uint32_t*>(row + p));
  const uint32_t v0 = static_cast<uint16_t>(__ldg(row + p));
  const uint32_t v1 = (p + 1 < P.k) ? static_cast<uint16_t>(__ldg(row + p + 1)) : 0u;
  return v0 | (v1 << 16);
}

__device__ __forceinline__ int32_t f2i(float f) {
  int32_t v;
  asm("cvt.rni.s32.f32 %0, %1;" : "=r"(v) : "f"(f));
  return v;
}

template <int NT>
__global__ void __launch_bounds__(THREADS, 1)
skinny_kernel(const __grid_constant__ CUtensorMap mapB, SkParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* red = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  constexpr int RED_PER_WARP = 2 * NT * 4 * 32;
  uint64_t* bars = red + NCONS * RED_PER_WARP;
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int64_t j_base = static_cast<int64_t>(blockIdx.x) * JB;
  const int64_t st_begin = static_cast<int64_t>(blockIdx.y) * P.stages_per_cta;
  int64_t st_end = st_begin + P.stages_per_cta;
  if (st_end > P.total_stages) st_end = P.total_stages;
  const int64_t nst = st_end > st_begin ? st_end - st_begin : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, NCONS);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == NCONS) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&mapB);
      int64_t issued = 0;
      for (int64_t i = 0; i < nst; ++i) {
        const int s = static_cast<int>(i % STAGES);
        const uint32_t par = static_cast<uint32_t>((i / STAGES) & 1);
        if (!bounded_wait(empty0 + 8 * s, par ^ 1u, P.timeout_ns)) {
          report_status(P.status, STATUS_TIMEOUT, 11);
          break;
        }
        mbar_arrive_expect_tx(full0 + 8 * s, STAGE_BYTES);
        tma_load_2d(smem_u32(smem + s * STAGE_BYTES), &mapB, full0 + 8 * s, static_cast<int32_t>(j_base),
                    static_cast<int32_t>((st_begin + i) * KS));
        ++issued;
      }
      const int64_t first = issued > STAGES ? issued - STAGES : 0;
      for (int64_t i = first; i < issued; ++i)
        bounded_wait(full0 + 8 * static_cast<int>(i % STAGES), static_cast<uint32_t>((i / STAGES) & 1), P.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int g = lane >> 2;
    const int t = lane & 3;
    float hh[2][NT][4], xx[2][NT][4], ll[2][NT][4];
    uint64_t acc[2][NT][4];
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          hh[mt][nt][c] = xx[mt][nt][c] = ll[mt][nt][c] = 0.f;
          acc[mt][nt][c] = 0;
        }
    // ldmatrix row address pieces: lanes 0-7 matrix 0 (k 0-7, j 0-7), 8-15 matrix 1 (k 0-7, j 8-15),
    // 16-23 matrix 2 (k 8-15, j 0-7), 24-31 matrix 3 (k 8-15, j 8-15)
    const int mrow = warp * 16 + (lane & 7) + ((lane >> 4) << 3);  // row of the stage tile (k)
    const int mchunk = (lane >> 3) & 1;                             // +8 columns (j)
    bool ok = true;
    for (int64_t i = 0; i < nst; ++i) {
      const int s = static_cast<int>(i % STAGES);
      const uint32_t par = static_cast<uint32_t>((i / STAGES) & 1);
      const bool got = bounded_wait(full0 + 8 * s, par, P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, got)) {
        if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 12);
        ok = false;
        break;
      }
      const uint32_t tile = smem_u32(smem + s * STAGE_BYTES);
      const int64_t k0 = (st_begin + i) * KS + warp * 16;  // first reduction index of this warp's slab
      // A fragments (the mma's B operand: 16 reduction indices x 8 rows of A)
      uint32_t ahi[NT][2], alo[NT][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int64_t row = nt * 8 + g;
        split_pair(load_a_pair(P, row, k0 + 2 * t), ahi[nt][0], alo[nt][0]);
        split_pair(load_a_pair(P, row, k0 + 2 * t + 8), ahi[nt][1], alo[nt][1]);
      }
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        // 64-byte swizzle: 16-byte chunk c of row r sits at chunk c ^ ((r >> 1) & 3)
        const int chunk = mt * 2 + mchunk;
        const uint32_t addr = tile + mrow * 64 + ((chunk ^ ((mrow >> 1) & 3)) << 4);
        uint32_t b[4], bhi[4], blo[4];
        ldsm_x4_trans(addr, b);
#pragma unroll
        for (int q = 0; q < 4; ++q) split_pair(b[q], bhi[q], blo[q]);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          mma16816(hh[mt][nt], bhi, ahi[nt][0], ahi[nt][1]);
          mma16816(xx[mt][nt], bhi, alo[nt][0], alo[nt][1]);
          mma16816(xx[mt][nt], blo, ahi[nt][0], ahi[nt][1]);
          mma16816(ll[mt][nt], blo, alo[nt][0], alo[nt][1]);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * s);
      if ((i + 1) % DRAIN_EVERY == 0 || i + 1 == nst) {
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              acc[mt][nt][c] += (static_cast<uint64_t>(static_cast<int64_t>(f2i(hh[mt][nt][c]))) << 16) +
                                (static_cast<uint64_t>(static_cast<int64_t>(f2i(xx[mt][nt][c]))) << 8) +
                                static_cast<uint64_t>(static_cast<int64_t>(f2i(ll[mt][nt][c])));
              hh[mt][nt][c] = xx[mt][nt][c] = ll[mt][nt][c] = 0.f;
            }
      }
    }
    if (!__all_sync(0xFFFFFFFFu, ok)) ok = false;
    // partials to shared memory: red[warp][((mt*NT + nt)*4 + c)*32 + lane]
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int c = 0; c < 4; ++c) red[warp * RED_PER_WARP + ((mt * NT + nt) * 4 + c) * 32 + lane] = acc[mt][nt][c];
  }
  __syncthreads();
  // ------------------------------------------------------------ reduce the warps and update C
  if (warp < NCONS) {
    for (int idx = threadIdx.x; idx < RED_PER_WARP; idx += NCONS * 32) {
      uint64_t sum = 0;
#pragma unroll
      for (int w = 0; w < NCONS; ++w) sum += red[w * RED_PER_WARP + idx];
      const int ln = idx & 31;
      const int c = (idx >> 5) & 3;
      const int mn = idx >> 7;  // mt * NT + nt
      const int mt = mn / NT, nt = mn % NT;
      const int gg = ln >> 2, tt = ln & 3;
      const int64_t i = nt * 8 + 2 * tt + (c & 1);             // row of C (n side of the mma)
      const int64_t j = j_base + mt * 16 + gg + 8 * (c >> 1);  // column of C (m side of the mma)
      if (i < P.m && j < P.n && nst > 0) {
        unsigned long long* dst = reinterpret_cast<unsigned long long*>(P.C + i * P.ldc + j);
        if (P.atomic_out) atomicAdd(dst, static_cast<unsigned long long>(sum));
        else *dst = *dst + static_cast<unsigned long long>(sum);
      }
    }
  }
}

template <int NT>
cudaError_t launch(const SkinnyArgs& a, cudaStream_t s, const char** why) {
  CUtensorMap map;
  if (!encode_tensor_map_2d(&map, 0, a.B, static_cast<uint64_t>(a.n), static_cast<uint64_t>(a.k),
                            static_cast<uint64_t>(a.ldb) * 2, JB, KS, 64, why))
    return cudaErrorInvalidValue;
  const int64_t nj = (a.n + JB - 1) / JB;
  const int64_t total_stages = (a.k + KS - 1) / KS;
  int64_t ksplit = a.ksplit;
  if (ksplit <= 0) {
    // one CTA per column block when that already fills most SMs; else split the reduction
    ksplit = nj * 4 >= static_cast<int64_t>(a.num_sms) * 3 ? 1 : (a.num_sms + nj - 1) / nj;
  }
  if (ksplit > total_stages) ksplit = total_stages;
  if (ksplit < 1) ksplit = 1;
  const int64_t per = (total_stages + ksplit - 1) / ksplit;
  ksplit = (total_stages + per - 1) / per;
  if (nj > 0x7FFFFFFF || ksplit > 65535) {
    *why = "skinny GEMM grid too large";
    return cudaErrorInvalidValue;
  }
  SkParams P;
  P.m = a.m;
  P.n = a.n;
  P.k = a.k;
  P.A = a.A;
  P.lda = a.lda;
  P.C = a.C;
  P.ldc = a.ldc;
  P.stages_per_cta = per;
  P.total_stages = total_stages;
  P.atomic_out = ksplit > 1 ? 1 : 0;
  P.a_vec = (reinterpret_cast<uintptr_t>(a.A) % 4 == 0) && (a.lda % 2 == 0);
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  constexpr size_t smem = sk_smem<NT>();
  cudaError_t e = cudaFuncSetAttribute(skinny_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(static_cast<unsigned>(nj), static_cast<unsigned>(ksplit));
  skinny_kernel<NT><<<grid, THREADS, smem, s>>>(map, P);
  return cudaGetLastError();
}

}  // namespace

cudaError_t skinny_gemm_i16(const SkinnyArgs& args, cudaStream_t s, const char** why) {
  return args.m <= 8 ? launch<1>(args, s, why) : launch<2>(args, s, why);
}

}  // namespace gemmi
