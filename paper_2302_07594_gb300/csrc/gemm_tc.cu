// gemm_tc.cu -- exact integer GEMM on the 5th-generation tensor cores (tcgen05, sm_103a).
//
// What it computes: C += A*B (Section 4.1 of the paper) for int16 operands and
// an int64 C, or int8 operands and an int32 C, bit-exactly.
//
// How.  The operands arrive as fp16 limb planes (split.cu): a = 256*h + l with
// |h|, |l| <= 128, so for one reduction index
//     a*b = 2^16 * (h_a h_b) + 2^8 * (h_a l_b + l_a h_b) + (l_a l_b).
// B's two limb tiles sit one above the other in shared memory, so one
// tcgen05.mma of N = 256 multiplies an A limb by both B limbs at once: the
// accumulator of A_high holds HH | HL, the accumulator of A_low holds LH | LL
// (column halves).  Each limb product is an integer of magnitude <= 2^14 that
// fp16 x fp16 forms exactly, and an fp32 accumulator sums integers exactly
// while every partial sum stays below 2^24.  So an accumulator is only allowed
// a bounded run of the reduction dimension (a "chunk": by default 1024
// indices), after which it is drained: converted to an integer and added,
// shifted by its weight (16, 8 or 0 bits), into a 64-bit running sum held in
// registers.  This plays the role of the AIE's 48-bit accumulators (Section
// 6.2): wide accumulation so nothing overflows, here built from exact fp32
// chunks and int64 registers.  The int8 path multiplies the values themselves
// (one plane) into one accumulator per 128-column half of a 128 x 256 tile.
//
// Structure (one persistent CTA per SM, 352 threads, 128x128 output tiles for
// int16):
//   warp 8      TMA producer: 2-D tiled bulk-tensor loads of 64-wide K blocks of
//               the limb planes (128-byte swizzle) into a ring of smem stages;
//   warps 9-10  MMA issuers: tcgen05.mma kind::f16 (M=128, K=16, N=256 for
//               int16, N=128 for int8) from smem descriptors into fp32
//               accumulators in tensor memory (TMEM).  A single issuing thread
//               leaves the tensor pipe idle for every cycle it spends waiting or
//               book-keeping (the pipe buffers almost no instructions), so two
//               warps issue concurrently, each owning its own accumulator;
//   warps 0-7   epilogue: drain accumulators (tcgen05.ld) into int64 registers,
//               and read-modify-write C once per tile.
// TMEM holds the accumulators: two 256-column slots for int16 (chunk ends
// staggered by half a chunk, so while one issuer waits for the drain of its
// slot the other keeps the tensor pipe busy), four 128-column slots for int8
// (two live, two spare: at a chunk end the owning issuer moves its accumulator
// into the oldest spare and keeps issuing).  Every role replays the same
// deterministic chunk schedule, so slot assignments need no communication
// beyond the full/empty barriers of each slot.  This takes the place of the
// paper's loop L6 / micro-kernel (Figure 1, Section 5.2); the smem stage ring
// takes the place of the B_r copies into local memory (Section 5.1).
//
// Every mbarrier wait is bounded (ptx.cuh); a wait that runs out records
// GEMMI_ETIMEOUT in the device status word and the CTA winds down cleanly.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

using namespace tc;
constexpr int NUM_EPI_WARPS = 8;
constexpr int PRODUCER_WARP = 8;
constexpr int MMA_WARP0 = 9;                  // issuer warps 9 and 10; warp 9 also owns the TMEM allocation
constexpr int NISSUE = 2;
constexpr int NUM_THREADS = (NUM_EPI_WARPS + 1 + NISSUE) * 32;
constexpr int TMEM_COLS = 512;

// Tile geometry: K blocks of 64 fp16 (128-byte rows, the 128-byte swizzle span).
template <int NL>
struct Geom {
  static constexpr int BN = Scheme<NL>::BN;
  static constexpr int TILE_A = BM * BK * 2;              // one limb tile of A
  static constexpr int TILE_B = BN * BK * 2;              // one limb tile of B
  static constexpr int SB = NL * (TILE_A + TILE_B);       // one stage: NL tiles of A, then NL of B
  static constexpr int STAGES = (192 * 1024) / SB;        // 192 KB of stages
  static constexpr int SWIZZLE = BK * 2;                  // bytes per swizzled row
  static constexpr int NSLOT = Scheme<NL>::NSLOT;
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * SB + 8 * (2 * STAGES + 2 * NSLOT + 1) + 16;
  static_assert(NSLOT * Scheme<NL>::SLOT_COLS <= TMEM_COLS, "tensor memory budget");
  static_assert(SMEM <= 227 * 1024, "shared memory budget");
};

struct TcParams {
  int64_t m, n, k;
  void* C;
  int64_t ldc;
  int num_m_tiles, num_n_tiles, num_k_blocks;
  int c_vec;
  int group_m;        // tile raster: bands of group_m row tiles, column-major inside a band
  int hint_a;         // L2 policy of A loads: 0 normal, 1 evict_last, 2 evict_first
  int hint_b;         // same for B
  uint64_t timeout_ns;
  uint32_t* status;
};

template <int NL, int CS>
__global__ void __launch_bounds__(NUM_THREADS, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap mapA0, const __grid_constant__ CUtensorMap mapA1,
               const __grid_constant__ CUtensorMap mapA2, const __grid_constant__ CUtensorMap mapB0,
               const __grid_constant__ CUtensorMap mapB1, const __grid_constant__ CUtensorMap mapB2, TcParams P) {
  using S = Scheme<NL>;
  using G = Geom<NL>;
  constexpr int STAGES = G::STAGES;
  constexpr int SB = G::SB;
  constexpr int TILE_A = G::TILE_A;
  constexpr int TILE_B = G::TILE_B;
  constexpr int BN = S::BN;
  constexpr int COLS = S::COLS;
  constexpr int NSLOT = S::NSLOT;
  constexpr int SLOT_COLS = S::SLOT_COLS;
  constexpr int UMMA_N = S::UMMA_N;
  // C element type and the unsigned type of the running sum (wrap-around is modular, never UB)
  using CT = typename std::conditional<NL >= 2, int64_t, int32_t>::type;
  using UT = typename std::conditional<NL >= 2, uint64_t, uint32_t>::type;
  const CUtensorMap* const amap[3] = {&mapA0, &mapA1, &mapA2};
  const CUtensorMap* const bmap[3] = {&mapB0, &mapB1, &mapB2};

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * SB);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t sfull0 = empty0 + 8 * STAGES;
  const uint32_t sempty0 = sfull0 + 8 * NSLOT;
  const uint32_t final_bar = sempty0 + 8 * NSLOT;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2 * NSLOT + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, S::EMPTY_COUNT);
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(sfull0 + 8 * s, 1);
      mbar_init(sempty0 + 8 * s, S::DRAIN_WARPS);
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

  if (warp == PRODUCER_WARP) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
#pragma unroll
      for (int l = 0; l < NL; ++l) {
        tma_prefetch_desc(amap[l]);
        tma_prefetch_desc(bmap[l]);
      }
      const uint64_t pol_a = l2_policy(P.hint_a);
      const uint64_t pol_b = l2_policy(P.hint_b);
      int stage = 0;
      uint32_t phase = 0;
      int64_t issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total_tiles && ok; t += gridDim.x) {
        int mt, nt;
        tile_coords(t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!bounded_wait(empty0 + 8 * stage, phase ^ 1u, P.timeout_ns)) {
            report_status(P.status, STATUS_TIMEOUT, 1);
            *abort_flag = 1;
            ok = false;
            break;
          }
          if (*abort_flag) { ok = false; break; }
          const uint32_t fb = full0 + 8 * stage;
          mbar_arrive_expect_tx(fb, SB);
          const uint32_t base = smem_u32(smem + stage * SB);
#pragma unroll
          for (int l = 0; l < NL; ++l)
            tma_load_2d_hint(base + l * TILE_A, amap[l], fb, kb * BK, mt * BM, P.hint_a, pol_a);
#pragma unroll
          for (int l = 0; l < NL; ++l)
            tma_load_2d_hint(base + NL * TILE_A + l * TILE_B, bmap[l], fb, kb * BK, nt * BN, P.hint_b, pol_b);
          ++issued;
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      // Make sure no bulk copy is still landing in shared memory when the CTA exits.
      const int64_t first = issued > STAGES ? issued - STAGES : 0;
      for (int64_t i = first; i < issued; ++i) {
        const int s = static_cast<int>(i % STAGES);
        const uint32_t par = static_cast<uint32_t>((i / STAGES) & 1);
        bounded_wait(full0 + 8 * s, par, P.timeout_ns);
      }
    }
  } else if (warp >= MMA_WARP0) {
    // ------------------------------------------------------------ MMA issuers (one thread each)
    const int me = warp - MMA_WARP0;
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, UMMA_N);
      int stage = 0;
      uint32_t phase = 0;
      SlotRing<S::NACC, NSLOT> ring;
      ring.init();
      uint32_t wait_par[S::NACC];
      bool need_acquire[S::NACC], fresh[S::NACC];
#pragma unroll
      for (int a = 0; a < S::NACC; ++a) {
        wait_par[a] = 1u;  // first use of the initial slots: nothing to wait for
        need_acquire[a] = true;
        fresh[a] = true;
      }
      bool ok = true;
      for (int t = blockIdx.x; t < total_tiles && ok; t += gridDim.x) {
        for (int kb = 0; kb < nkb && ok; ++kb) {
          bool mine = false;
#pragma unroll
          for (int p = 0; p < S::NPROD; ++p) mine |= S::issuer(p, kb) == me;
          if (mine) {
            if (!bounded_wait(full0 + 8 * stage, phase, P.timeout_ns)) {
              report_status(P.status, STATUS_TIMEOUT, 2);
              *abort_flag = 1;
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t base = smem_u32(smem + stage * SB);
#pragma unroll
            for (int p = 0; p < S::NPROD; ++p) {
              if (S::issuer(p, kb) != me) continue;
              const int a = S::acc(p, kb);
              if (need_acquire[a]) {
                // the slot's previous chunk (any accumulator's) must have been drained
                if (!bounded_wait(sempty0 + 8 * ring.slot_of[a], wait_par[a], P.timeout_ns)) {
                  report_status(P.status, STATUS_TIMEOUT, 3);
                  *abort_flag = 1;
                  ok = false;
                  break;
                }
                need_acquire[a] = false;
                tc_fence_after();
              }
              const uint32_t d = tmem_base + static_cast<uint32_t>(ring.slot_of[a] * SLOT_COLS);
              const uint64_t adesc = smem_desc_kmajor<G::SWIZZLE>(base + S::a_limb(p) * TILE_A);
              const uint64_t bdesc = smem_desc_kmajor<G::SWIZZLE>(base + NL * TILE_A + S::b_limb(p) * TILE_B +
                                                                  S::b_row0(p) * (BK * 2));
#pragma unroll
              for (int kk = 0; kk < BK / UMMA_K; ++kk) {
                // advancing the start address by 32 bytes (16 fp16) steps K inside the swizzled row
                const uint32_t acc_flag = (fresh[a] && kk == 0) ? 0u : 1u;
                tc_mma_f16(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, acc_flag);
              }
              fresh[a] = false;
            }
            if (!ok) break;
            tc_commit(empty0 + 8 * stage);  // this issuer has finished reading the stage once its MMAs complete
          }
          // replay every chunk end (own and the other issuer's) to keep the slot ring in step
#pragma unroll
          for (int a = 0; a < S::NACC; ++a) {
            if (!S::template chunk_ends<CS>(a, kb, nkb)) continue;
            if (S::owner(a) == me) tc_commit(sfull0 + 8 * ring.slot_of[a]);  // chunk ready to drain
            const uint32_t par = ring.rotate(a);
            if (S::owner(a) == me) {
              wait_par[a] = par;
              need_acquire[a] = true;
              fresh[a] = true;
            }
          }
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      // all MMAs issued by both threads must be complete before TMEM is released
      tc_commit(final_bar);
      bounded_wait(final_bar, 0, P.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 0..7)
    const int quad = warp & 3;       // TMEM lanes 32*quad .. 32*quad+31 (hardware lane quadrant)
    const int half = warp >> 2;      // column half of the tile: columns half*COLS .. +COLS-1
    SlotRing<S::NACC, NSLOT> ring;
    ring.init();
    uint32_t drain_parity = 0;  // bit s: parity of the number of drains of slot s
    bool ok = true;
    UT acc[COLS];
    for (int t = blockIdx.x; t < total_tiles && ok; t += gridDim.x) {
      int mt, nt;
      tile_coords(t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
      const int64_t row = static_cast<int64_t>(mt) * BM + quad * 32 + lane;
      const int64_t col0 = static_cast<int64_t>(nt) * BN + half * COLS;
      CT* crow = static_cast<CT*>(P.C) + row * P.ldc + col0;
      const bool row_ok = row < P.m;
      const bool full_cols = col0 + COLS <= P.n;
      // running sum starts from C itself, so the tile ends with a plain store
      if (row_ok && full_cols && P.c_vec) {
        if constexpr (NL >= 2) {
#pragma unroll
          for (int c = 0; c < COLS; c += 2) {
            const longlong2 v = *reinterpret_cast<const longlong2*>(crow + c);
            acc[c] = static_cast<UT>(v.x);
            acc[c + 1] = static_cast<UT>(v.y);
          }
        } else {
#pragma unroll
          for (int c = 0; c < COLS; c += 4) {
            const int4 v = *reinterpret_cast<const int4*>(crow + c);
            acc[c] = static_cast<UT>(v.x);
            acc[c + 1] = static_cast<UT>(v.y);
            acc[c + 2] = static_cast<UT>(v.z);
            acc[c + 3] = static_cast<UT>(v.w);
          }
        }
      } else {
#pragma unroll
        for (int c = 0; c < COLS; ++c) acc[c] = (row_ok && col0 + c < P.n) ? static_cast<UT>(crow[c]) : UT(0);
      }
      {
        // warm L2 with this thread's C row segment of the next tile it will process
        const int tn = t + gridDim.x;
        if (tn < total_tiles) {
          int mn, nn;
          tile_coords(tn, P.num_m_tiles, P.num_n_tiles, P.group_m, mn, nn);
          const int64_t prow = static_cast<int64_t>(mn) * BM + quad * 32 + lane;
          const int64_t pcol = static_cast<int64_t>(nn) * BN + half * COLS;
          if (prow < P.m && pcol < P.n) {
            const CT* pc = static_cast<const CT*>(P.C) + prow * P.ldc + pcol;
            const int64_t cols = min(static_cast<int64_t>(COLS), P.n - pcol);
            for (int64_t c = 0; c < cols; c += 128 / static_cast<int64_t>(sizeof(CT)))
              asm volatile("prefetch.global.L2 [%0];" ::"l"(pc + c));
          }
        }
      }
      for (int kb = 0; kb < nkb && ok; ++kb) {
#pragma unroll
        for (int a = 0; a < S::NACC; ++a) {
          if (!S::template chunk_ends<CS>(a, kb, nkb)) continue;
          if (!S::drains(half, a)) {
            // another half's accumulator: its chunk still completes one phase of this slot's full
            // barrier (slots pass between accumulators), so keep that parity and the ring in step
            drain_parity ^= 1u << ring.slot_of[a];
            ring.rotate(a);
            continue;
          }
          const int s = ring.slot_of[a];
          // every lane waits; the warp then decides together (tcgen05.ld needs a converged warp)
          const bool got = bounded_wait(sfull0 + 8 * s, (drain_parity >> s) & 1u, P.timeout_ns);
          if (!__all_sync(0xFFFFFFFFu, got)) {
            if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 4);
            *abort_flag = 1;
            ok = false;
            break;
          }
          drain_parity ^= 1u << s;
          tc_fence_after();
          // this warp's columns of the accumulator: all 128 (int8, one accumulator per half)
          // or its 64-column half (int16)
          if constexpr (NL == 3) {
            // Karatsuba: this warp's 64 columns of the 128-column accumulator, times its weight
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(s * SLOT_COLS + half * COLS);
            const UT w = S::weight(a);
#pragma unroll
            for (int c = 0; c < COLS; c += 32) {
              uint32_t r0[16], r1[16];
              tc_ld_32x32b_x16(taddr + c, r0);
              tc_ld_32x32b_x16(taddr + c + 16, r1);
              tc_wait_ld();
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                acc[c + i] += w * static_cast<UT>(static_cast<CT>(f32_to_i32(r0[i])));
                acc[c + 16 + i] += w * static_cast<UT>(static_cast<CT>(f32_to_i32(r1[i])));
              }
            }
          } else if constexpr (NL == 2) {
            // this warp's 64 output columns: the B-high part (accumulator columns 0-127) and the
            // B-low part (columns 128-255) of each, 16 columns at a time
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(s * SLOT_COLS + half * COLS);
#pragma unroll
            for (int c = 0; c < COLS; c += 16) {
              uint32_t rh[16], rl[16];
              tc_ld_32x32b_x16(taddr + c, rh);
              tc_ld_32x32b_x16(taddr + BN + c, rl);
              tc_wait_ld();
#pragma unroll
              for (int i = 0; i < 16; ++i)
                acc[c + i] += (static_cast<UT>(static_cast<CT>(f32_to_i32(rh[i]))) << S::shift(a)) +
                              (static_cast<UT>(static_cast<CT>(f32_to_i32(rl[i]))) << S::shift_low(a));
            }
          } else {
            // this warp's 128 columns: the accumulator of its half
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(s * SLOT_COLS);
#pragma unroll
            for (int c = 0; c < COLS; c += 32) {
              uint32_t r0[16], r1[16];
              tc_ld_32x32b_x16(taddr + c, r0);
              tc_ld_32x32b_x16(taddr + c + 16, r1);
              tc_wait_ld();
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                // sign-extend to the unsigned running-sum type (modular)
                acc[c + i] += static_cast<UT>(static_cast<CT>(f32_to_i32(r0[i])));
                acc[c + 16 + i] += static_cast<UT>(static_cast<CT>(f32_to_i32(r1[i])));
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sempty0 + 8 * s);
          ring.rotate(a);
        }
      }
      if (!ok) break;
      if (row_ok && full_cols && P.c_vec) {
        if constexpr (NL >= 2) {
#pragma unroll
          for (int c = 0; c < COLS; c += 2)
            *reinterpret_cast<longlong2*>(crow + c) =
                make_longlong2(static_cast<long long>(acc[c]), static_cast<long long>(acc[c + 1]));
        } else {
#pragma unroll
          for (int c = 0; c < COLS; c += 4)
            *reinterpret_cast<int4*>(crow + c) =
                make_int4(static_cast<int>(acc[c]), static_cast<int>(acc[c + 1]), static_cast<int>(acc[c + 2]),
                          static_cast<int>(acc[c + 3]));
        }
      } else if (row_ok) {
#pragma unroll
        for (int c = 0; c < COLS; ++c)
          if (col0 + c < P.n) crow[c] = static_cast<CT>(acc[c]);
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

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

template <int NL, int CS>
cudaError_t launch(const TcGemmArgs& a, cudaStream_t s, const char** why) {
  using G = Geom<NL>;
  CUtensorMap maps[6];
  const LimbPlanes* ops[2] = {&a.a, &a.b};
  for (int o = 0; o < 2; ++o) {
    for (int l = 0; l < 3; ++l) {
      const void* base = ops[o]->plane[l < NL ? l : 0];
      if (!encode_tensor_map_2d(&maps[3 * o + l], 1, base, static_cast<uint64_t>(a.k),
                                static_cast<uint64_t>(ops[o]->rows), static_cast<uint64_t>(ops[o]->pitch) * 2, BK,
                                o == 0 ? BM : G::BN, G::SWIZZLE, why))
        return cudaErrorInvalidValue;
    }
  }
  TcParams P;
  P.m = a.m;
  P.n = a.n;
  P.k = a.k;
  P.C = a.C;
  P.ldc = a.ldc;
  P.num_m_tiles = static_cast<int>((a.m + BM - 1) / BM);
  P.num_n_tiles = static_cast<int>((a.n + G::BN - 1) / G::BN);
  P.num_k_blocks = static_cast<int>((a.k + BK - 1) / BK);
  const size_t esz = NL >= 2 ? 8 : 4;
  P.c_vec = (reinterpret_cast<uintptr_t>(a.C) % 16 == 0) && ((a.ldc * esz) % 16 == 0);
  P.group_m = a.group_m > 0 ? a.group_m : 16;
  P.hint_a = a.hint_a;
  P.hint_b = a.hint_b;
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  const int64_t tiles = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles;
  const int grid = static_cast<int>(tiles < a.num_sms ? tiles : a.num_sms);
  constexpr size_t smem = G::SMEM;
  // the shared-memory opt-in is set once per device for this kernel
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t attr = cudaFuncSetAttribute(tc_gemm_kernel<NL, CS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  static_cast<int>(smem));
    if (attr != cudaSuccess) return attr;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  tc_gemm_kernel<NL, CS><<<grid, NUM_THREADS, smem, s>>>(maps[0], maps[1], maps[2], maps[3], maps[4], maps[5], P);
  return cudaGetLastError();
}

}  // namespace

bool encode_tensor_map_2d(void* map, int dtype, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle_bytes,
                          const char** why) {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (g_encode == nullptr) {
    *why = "cuTensorMapEncodeTiled is not available from the driver";
    return false;
  }
  const CUtensorMapDataType dt = dtype == 1   ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                 : dtype == 2 ? CU_TENSOR_MAP_DATA_TYPE_UINT8
                                 : dtype == 3 ? CU_TENSOR_MAP_DATA_TYPE_UINT64
                                 : dtype == 4 ? CU_TENSOR_MAP_DATA_TYPE_UINT32
                                              : CU_TENSOR_MAP_DATA_TYPE_UINT16;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                : swizzle_bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                                                      : CU_TENSOR_MAP_SWIZZLE_NONE;
  const CUresult r = g_encode(static_cast<CUtensorMap*>(map), dt, 2, const_cast<void*>(base), dims, strides, box,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected the operand layout";
    return false;
  }
  return true;
}

cudaError_t tc_gemm_i16(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch<2, 2>(args, s, why) : launch<2, 1>(args, s, why);
}
cudaError_t tc_gemm_i8(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch<1, 2>(args, s, why) : launch<1, 1>(args, s, why);
}
cudaError_t tc_gemm_i16_karatsuba(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch<3, 2>(args, s, why) : launch<3, 1>(args, s, why);
}

}  // namespace gemmi
