// gemm_fused.cu -- int16 GEMM for narrow outputs (n <= 64) that converts A inside the kernel.
//
// Convolutions lowered with IM2COL/IM2ROW give GEMMs with one very large and
// two small dimensions (Section 2 of the paper): m = batch*H*W rows of
// activations, n = output channels, k = C_in*3*3.  Such a GEMM is bound by
// reading A once from HBM; a separate limb-split pass (split.cu) would read A,
// write its two fp16 limb planes (twice A's bytes) and read them again.  Here
// A is streamed raw (int16) and split on chip, the way the paper packs the
// activation operand at run time while the weights stay packed (Section 5.1):
//
//   warp 8      TMA producer of raw A tiles (128 rows x 64 reduction indices of
//               int16, 128-byte swizzle) into a ring of RAW_STAGES smem slots;
//   warp 9      TMA producer of B's limb tiles (64 x 64 fp16, from the split or
//               packed planes) into the limb stages;
//   warps 10-11 MMA issuers, as in gemm_tc.cu: tcgen05.mma kind::f16, M=128,
//               N=64, issuer 0 owns HH and LL, issuer 1 owns X;
//   warps 0-7   epilogue: they split each raw A tile into the fp16 limb tiles
//               AH, AL of a limb stage -- the raw and the limb tiles share one
//               swizzled layout, so every 16-byte chunk converts in place --
//               running LOOKAHEAD K blocks ahead of their main job, which is to
//               drain the accumulators (staggered exact chunks, as in gemm_tc.cu)
//               into int64 registers and read-modify-write C once per tile.
//
// Limb split of a packed int16 pair x = (a1 << 16) | a0 with centred limbs
// h = floor((a + 128) / 256), l = a - 256 h, done on both halves at once:
//   l + 128 = lo_byte ^ 0x80,   h + 128 = (hi_byte ^ 0x80) + (lo_byte >> 7),
// each placed under the fp16 exponent of 1024 (bits 0x6400) and recovered
// exactly by one fp16 subtraction of 1152.
//
// TMEM: eight 64-column accumulator slots (three live, five spare).  Every
// mbarrier wait is bounded; a wait that runs out records GEMMI_ETIMEOUT.
#include <cuda.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

using namespace tc;
using S = Scheme<2>;

constexpr int BN = 64;
constexpr int NUM_EPI_WARPS = 8;
constexpr int A_PRODUCER_WARP = 8;
constexpr int B_PRODUCER_WARP = 9;
constexpr int MMA_WARP0 = 10;
constexpr int NISSUE = 2;
constexpr int NUM_THREADS = (NUM_EPI_WARPS + 2 + NISSUE) * 32;
constexpr int NSLOT = 8;
constexpr int SLOT_COLS = 64;
constexpr int TMEM_COLS = NSLOT * SLOT_COLS;  // 512
constexpr int STAGES = 3;                     // limb stages
constexpr int RAW_STAGES = 4;                 // raw A stages
constexpr int TILE_A = BM * BK * 2;           // 16 KB: a raw int16 A tile, and each A limb tile
constexpr int TILE_B = BN * BK * 2;           // 8 KB: each B limb tile
constexpr int SB = 2 * TILE_A + 2 * TILE_B;   // limb stage: AH, AL, BH, BL
constexpr int LOOKAHEAD = 2;                  // conversions run ahead of drains (< STAGES)
constexpr int COLS = 32;                      // C columns per epilogue thread
constexpr int CHUNKS_PER_WARP = TILE_A / 16 / NUM_EPI_WARPS;  // 16-byte chunks converted per warp
constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * SB + static_cast<size_t>(RAW_STAGES) * TILE_A +
                        8 * (2 * STAGES + 2 * RAW_STAGES + 2 * NSLOT + 1) + 16;
static_assert(SMEM <= 227 * 1024, "shared memory budget");
static_assert(LOOKAHEAD < STAGES, "conversions may not wait on MMAs that wait on later drains");

struct FusedParams {
  int64_t m, n, k;
  int64_t* C;
  int64_t ldc;
  int num_m_tiles, num_n_tiles, num_k_blocks;
  int c_vec;
  int group_m;
  uint64_t timeout_ns;
  uint32_t* status;
};

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// centred limbs of both int16 halves of x, as fp16 pairs (exact)
__device__ __forceinline__ void split_centred(uint32_t x, uint32_t& hi, uint32_t& lo) {
  const uint32_t l_bits = (x & 0x00FF00FFu) ^ 0x64806480u;                                 // 1024 + (l + 128)
  const uint32_t h_bits = (((x >> 8) & 0x00FF00FFu) ^ 0x64806480u) + ((x >> 7) & 0x00010001u);  // 1024 + (h + 128)
  const __half2 bias = __half2half2(__ushort_as_half(0x6480));  // 1152
  const __half2 l = __hsub2(*reinterpret_cast<const __half2*>(&l_bits), bias);
  const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&h_bits), bias);
  lo = *reinterpret_cast<const uint32_t*>(&l);
  hi = *reinterpret_cast<const uint32_t*>(&h);
}

template <int CS>
__global__ void __launch_bounds__(NUM_THREADS, 1)
fused_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapBH,
             const __grid_constant__ CUtensorMap mapBL, FusedParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* raw = smem + STAGES * SB;
  uint64_t* bars = reinterpret_cast<uint64_t*>(raw + RAW_STAGES * TILE_A);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t rfull0 = empty0 + 8 * STAGES;
  const uint32_t rempty0 = rfull0 + 8 * RAW_STAGES;
  const uint32_t sfull0 = rempty0 + 8 * RAW_STAGES;
  const uint32_t sempty0 = sfull0 + 8 * NSLOT;
  const uint32_t final_bar = sempty0 + 8 * NSLOT;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2 * RAW_STAGES + 2 * NSLOT + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1 + NUM_EPI_WARPS);  // B producer's expect_tx arrival + 8 converter warps
      mbar_init(empty0 + 8 * s, NISSUE);
    }
    for (int s = 0; s < RAW_STAGES; ++s) {
      mbar_init(rfull0 + 8 * s, 1);
      mbar_init(rempty0 + 8 * s, NUM_EPI_WARPS);
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(sfull0 + 8 * s, 1);
      mbar_init(sempty0 + 8 * s, NUM_EPI_WARPS);
    }
    mbar_init(final_bar, NISSUE);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == MMA_WARP0) {
    tmem_alloc(smem_u32(tmem_holder), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  const int total_tiles = P.num_m_tiles * P.num_n_tiles;
  const int nkb = P.num_k_blocks;
  const int my_tiles = total_tiles > static_cast<int>(blockIdx.x)
                           ? (total_tiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                                 static_cast<int>(gridDim.x)
                           : 0;
  const int64_t total_q = static_cast<int64_t>(my_tiles) * nkb;  // this CTA's K blocks, over its tiles

  if (warp == A_PRODUCER_WARP) {
    // ------------------------------------------------------------ raw A tiles
    if (lane == 0) {
      tma_prefetch_desc(&mapA);
      int64_t issued = 0;
      for (int64_t q = 0; q < total_q; ++q) {
        const int i = static_cast<int>(q / nkb), kb = static_cast<int>(q % nkb);
        int mt, nt;
        tile_coords(static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x), P.num_m_tiles, P.num_n_tiles,
                    P.group_m, mt, nt);
        const int r = static_cast<int>(q % RAW_STAGES);
        const uint32_t par = static_cast<uint32_t>((q / RAW_STAGES) & 1);
        if (!bounded_wait(rempty0 + 8 * r, par ^ 1u, P.timeout_ns) || *abort_flag) {
          report_status(P.status, STATUS_TIMEOUT, 21);
          *abort_flag = 1;
          break;
        }
        mbar_arrive_expect_tx(rfull0 + 8 * r, TILE_A);
        tma_load_2d(smem_u32(raw + r * TILE_A), &mapA, rfull0 + 8 * r, kb * BK, mt * BM);
        ++issued;
      }
      for (int64_t q = issued > RAW_STAGES ? issued - RAW_STAGES : 0; q < issued; ++q)
        bounded_wait(rfull0 + 8 * static_cast<int>(q % RAW_STAGES), static_cast<uint32_t>((q / RAW_STAGES) & 1),
                     P.timeout_ns);
    }
  } else if (warp == B_PRODUCER_WARP) {
    // ------------------------------------------------------------ B limb tiles
    if (lane == 0) {
      tma_prefetch_desc(&mapBH);
      tma_prefetch_desc(&mapBL);
      int64_t issued = 0;
      for (int64_t q = 0; q < total_q; ++q) {
        const int i = static_cast<int>(q / nkb), kb = static_cast<int>(q % nkb);
        int mt, nt;
        tile_coords(static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x), P.num_m_tiles, P.num_n_tiles,
                    P.group_m, mt, nt);
        const int s = static_cast<int>(q % STAGES);
        const uint32_t par = static_cast<uint32_t>((q / STAGES) & 1);
        if (!bounded_wait(empty0 + 8 * s, par ^ 1u, P.timeout_ns) || *abort_flag) {
          report_status(P.status, STATUS_TIMEOUT, 22);
          *abort_flag = 1;
          break;
        }
        const uint32_t fb = full0 + 8 * s;
        const uint32_t base = smem_u32(smem + s * SB);
        mbar_arrive_expect_tx(fb, 2 * TILE_B);
        tma_load_2d(base + 2 * TILE_A, &mapBH, fb, kb * BK, nt * BN);
        tma_load_2d(base + 2 * TILE_A + TILE_B, &mapBL, fb, kb * BK, nt * BN);
        ++issued;
      }
      for (int64_t q = issued > STAGES ? issued - STAGES : 0; q < issued; ++q)
        bounded_wait(full0 + 8 * static_cast<int>(q % STAGES), static_cast<uint32_t>((q / STAGES) & 1), P.timeout_ns);
    }
  } else if (warp >= MMA_WARP0) {
    // ------------------------------------------------------------ MMA issuers
    const int me = warp - MMA_WARP0;
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN);
      SlotRing<S::NACC, NSLOT> ring;
      ring.init();
      uint32_t wait_par[S::NACC];
      bool need_acquire[S::NACC], fresh[S::NACC];
#pragma unroll
      for (int a = 0; a < S::NACC; ++a) {
        wait_par[a] = 1u;
        need_acquire[a] = true;
        fresh[a] = true;
      }
      bool ok = true;
      for (int64_t q = 0; q < total_q && ok; ++q) {
        const int kb = static_cast<int>(q % nkb);
        const int s = static_cast<int>(q % STAGES);
        if (!bounded_wait(full0 + 8 * s, static_cast<uint32_t>((q / STAGES) & 1), P.timeout_ns)) {
          report_status(P.status, STATUS_TIMEOUT, 23);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t base = smem_u32(smem + s * SB);
#pragma unroll
        for (int p = 0; p < S::NPROD; ++p) {
          if (S::issuer(p, kb) != me) continue;
          const int a = S::acc(p, kb);
          if (need_acquire[a]) {
            if (!bounded_wait(sempty0 + 8 * ring.slot_of[a], wait_par[a], P.timeout_ns)) {
              report_status(P.status, STATUS_TIMEOUT, 24);
              *abort_flag = 1;
              ok = false;
              break;
            }
            need_acquire[a] = false;
            tc_fence_after();
          }
          const uint32_t d = tmem_base + static_cast<uint32_t>(ring.slot_of[a] * SLOT_COLS);
          const uint64_t adesc = smem_desc_kmajor<128>(base + S::a_limb(p) * TILE_A);
          const uint64_t bdesc = smem_desc_kmajor<128>(base + 2 * TILE_A + S::b_limb(p) * TILE_B);
#pragma unroll
          for (int kk = 0; kk < BK / UMMA_K; ++kk)
            tc_mma_f16(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, (fresh[a] && kk == 0) ? 0u : 1u);
          fresh[a] = false;
        }
        if (!ok) break;
        tc_commit(empty0 + 8 * s);
#pragma unroll
        for (int a = 0; a < S::NACC; ++a) {
          if (!S::template chunk_ends<CS>(a, kb, nkb)) continue;
          if (S::owner(a) == me) tc_commit(sfull0 + 8 * ring.slot_of[a]);
          const uint32_t par = ring.rotate(a);
          if (S::owner(a) == me) {
            wait_par[a] = par;
            need_acquire[a] = true;
            fresh[a] = true;
          }
        }
      }
      tc_commit(final_bar);
      bounded_wait(final_bar, 0, P.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue: convert A, drain, C
    const int quad = warp & 3;
    const int half = warp >> 2;
    SlotRing<S::NACC, NSLOT> ring;
    ring.init();
    uint32_t drain_parity = 0;
    bool ok = true;
    int64_t cq = 0;  // next K block (over this CTA's tiles) whose A tile this warp converts

    // Converts this warp's share of raw A tile qq into the A limb tiles of its limb stage.
    auto convert = [&](int64_t qq) -> bool {
      const int r = static_cast<int>(qq % RAW_STAGES);
      const int s = static_cast<int>(qq % STAGES);
      const bool got_raw = bounded_wait(rfull0 + 8 * r, static_cast<uint32_t>((qq / RAW_STAGES) & 1), P.timeout_ns);
      const bool got_stage =
          got_raw && bounded_wait(empty0 + 8 * s, static_cast<uint32_t>(((qq / STAGES) & 1) ^ 1), P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, got_stage)) {
        if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 25);
        *abort_flag = 1;
        return false;
      }
      const uint32_t src = smem_u32(raw + r * TILE_A);
      const uint32_t dst_h = smem_u32(smem + s * SB);
      const uint32_t dst_l = dst_h + TILE_A;
#pragma unroll
      for (int c = 0; c < CHUNKS_PER_WARP / 32; ++c) {
        const uint32_t off = static_cast<uint32_t>((warp * CHUNKS_PER_WARP + c * 32 + lane) * 16);
        const uint4 x = lds128(src + off);
        uint4 h, l;
        split_centred(x.x, h.x, l.x);
        split_centred(x.y, h.y, l.y);
        split_centred(x.z, h.z, l.z);
        split_centred(x.w, h.w, l.w);
        sts128(dst_h + off, h);
        sts128(dst_l + off, l);
      }
      fence_proxy_async_smem();  // the tensor core reads these tiles through the async proxy
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(full0 + 8 * s);
        mbar_arrive(rempty0 + 8 * r);
      }
      return true;
    };

    int64_t q = 0;
    for (int i = 0; i < my_tiles && ok; ++i) {
      int mt, nt;
      tile_coords(static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x), P.num_m_tiles, P.num_n_tiles,
                  P.group_m, mt, nt);
      const int64_t row = static_cast<int64_t>(mt) * BM + quad * 32 + lane;
      const int64_t col0 = static_cast<int64_t>(nt) * BN + half * COLS;
      int64_t* crow = P.C + row * P.ldc + col0;
      const bool row_ok = row < P.m;
      const bool full_cols = col0 + COLS <= P.n;
      uint64_t acc[COLS];
      if (row_ok && full_cols && P.c_vec) {
#pragma unroll
        for (int c = 0; c < COLS; c += 2) {
          const longlong2 v = *reinterpret_cast<const longlong2*>(crow + c);
          acc[c] = static_cast<uint64_t>(v.x);
          acc[c + 1] = static_cast<uint64_t>(v.y);
        }
      } else {
#pragma unroll
        for (int c = 0; c < COLS; ++c) acc[c] = (row_ok && col0 + c < P.n) ? static_cast<uint64_t>(crow[c]) : 0ull;
      }
      for (int kb = 0; kb < nkb && ok; ++kb, ++q) {
        while (ok && cq <= q + LOOKAHEAD && cq < total_q) ok = convert(cq++);
        if (!ok) break;
#pragma unroll
        for (int a = 0; a < S::NACC; ++a) {
          if (!S::template chunk_ends<CS>(a, kb, nkb)) continue;
          const int s = ring.slot_of[a];
          const bool got = bounded_wait(sfull0 + 8 * s, (drain_parity >> s) & 1u, P.timeout_ns);
          if (!__all_sync(0xFFFFFFFFu, got)) {
            if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 26);
            *abort_flag = 1;
            ok = false;
            break;
          }
          drain_parity ^= 1u << s;
          tc_fence_after();
          const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                 static_cast<uint32_t>(s * SLOT_COLS + half * COLS);
          uint32_t r0[16], r1[16];
          tc_ld_32x32b_x16(taddr, r0);
          tc_ld_32x32b_x16(taddr + 16, r1);
          tc_wait_ld();
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            acc[j] += static_cast<uint64_t>(static_cast<int64_t>(f32_to_i32(r0[j]))) << S::shift(a);
            acc[16 + j] += static_cast<uint64_t>(static_cast<int64_t>(f32_to_i32(r1[j]))) << S::shift(a);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sempty0 + 8 * s);
          ring.rotate(a);
        }
      }
      if (!ok) break;
      if (row_ok && full_cols && P.c_vec) {
#pragma unroll
        for (int c = 0; c < COLS; c += 2)
          *reinterpret_cast<longlong2*>(crow + c) =
              make_longlong2(static_cast<long long>(acc[c]), static_cast<long long>(acc[c + 1]));
      } else if (row_ok) {
#pragma unroll
        for (int c = 0; c < COLS; ++c)
          if (col0 + c < P.n) crow[c] = static_cast<int64_t>(acc[c]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == MMA_WARP0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

template <int CS>
cudaError_t launch(const FusedArgs& a, cudaStream_t s, const char** why) {
  CUtensorMap mapA, mapBH, mapBL;
  if (!encode_tensor_map_2d(&mapA, 0, a.A, static_cast<uint64_t>(a.k), static_cast<uint64_t>(a.m),
                            static_cast<uint64_t>(a.lda) * 2, BK, BM, 128, why) ||
      !encode_tensor_map_2d(&mapBH, 1, a.b.plane[0], static_cast<uint64_t>(a.k), static_cast<uint64_t>(a.b.rows),
                            static_cast<uint64_t>(a.b.pitch) * 2, BK, BN, 128, why) ||
      !encode_tensor_map_2d(&mapBL, 1, a.b.plane[1], static_cast<uint64_t>(a.k), static_cast<uint64_t>(a.b.rows),
                            static_cast<uint64_t>(a.b.pitch) * 2, BK, BN, 128, why))
    return cudaErrorInvalidValue;
  FusedParams P;
  P.m = a.m;
  P.n = a.n;
  P.k = a.k;
  P.C = a.C;
  P.ldc = a.ldc;
  P.num_m_tiles = static_cast<int>((a.m + BM - 1) / BM);
  P.num_n_tiles = static_cast<int>((a.n + BN - 1) / BN);
  P.num_k_blocks = static_cast<int>((a.k + BK - 1) / BK);
  P.c_vec = (reinterpret_cast<uintptr_t>(a.C) % 16 == 0) && (a.ldc % 2 == 0);
  P.group_m = a.group_m > 0 ? a.group_m : 16;
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  const int64_t tiles = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles;
  const int grid = static_cast<int>(tiles < a.num_sms ? tiles : a.num_sms);
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t attr = cudaFuncSetAttribute(fused_kernel<CS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  static_cast<int>(SMEM));
    if (attr != cudaSuccess) return attr;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  fused_kernel<CS><<<grid, NUM_THREADS, SMEM, s>>>(mapA, mapBH, mapBL, P);
  return cudaGetLastError();
}

}  // namespace

cudaError_t tc_gemm_fused_i16(const FusedArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch<2>(args, s, why) : launch<1>(args, s, why);
}

}  // namespace gemmi
