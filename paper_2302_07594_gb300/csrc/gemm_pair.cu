// gemm_pair.cu -- exact integer GEMM on SM pairs: tcgen05.mma with cta_group::2 (sm_103a).
//
// What it computes: C += A*B (Section 4.1 of the paper) for int16 operands and an int64 C, or int8
// operands and an int32 C, bit-exactly -- the same operation as gemm_tc.cu, from the same fp16
// limb planes (split.cu), with the same exact-chunk accumulation (fp32 sums of at most 512 * CS
// limb products of magnitude <= 2^14, drained into 64-bit registers; the role of the AIE's wide
// accumulators, Section 6.2).
//
// How it differs.  Two CTAs of a cluster, on two SMs, form a pair.  One thread of the even CTA
// issues tcgen05.mma.cta_group::2 of M = 256, N = 256, K = 16: rows 0-127 of the A operand and
// of the accumulator live in the even CTA, rows 128-255 in the odd one, and each CTA holds half
// of the (K-major) B operand.  The pair gives every SM a single 256-column accumulator, so the
// other 256 TMEM columns are a spare slot: at a chunk end the MMAs move on into the spare while
// the epilogue drains the full slot, and the tensor pipe does not wait for drains.
//   int16: the even CTA holds the high limb of A's 128 rows, the odd CTA the low limb of the same
//          rows; B's high limb tile is the even CTA's half of B, the low limb tile the odd CTA's.
//          So the even SM accumulates A_high * [B_high | B_low] (weights 2^16 | 2^8) and the odd
//          SM A_low * [B_high | B_low] (weights 2^8 | 1) for one 128 x 128 output tile.
//   int8:  a 256 x 256 output tile; each SM holds 128 rows of A and 128 rows (output columns)
//          of B, and accumulates its 128 rows x all 256 columns.
//   int4:  the int8 geometry on E4M3 planes (int4.cu) with tcgen05.mma kind::f8f6f4, K = 32 per
//          instruction: a K block is 128 one-byte elements, the same 128 bytes per operand row,
//          so tiles, stages and descriptors are those of the fp16 planes, at twice the MMA rate.
// Per K block of 64 each SM loads 32 KB (its A tile and its B tile) for 512 tensor cycles: 64 B
// per cycle from L2, where a single-SM 128 x 256 int8 tile needs 96.
//
// The running int64 (int32) sums of a tile are added into C with 2-D tensor reductions
// (cp.reduce.async.bulk.tensor .add, one 32-row x 128-byte box per warp and round, through an
// unsigned tensor map so the adds wrap modulo 2^64 / 2^32), so the two SMs of an int16 tile add
// their weighted halves into C independently, C is never read by the SMs, and TMA clips the
// ragged edges.  Few large reductions matter: the cost of a bulk operation is mostly per
// operation, and 128-byte ones made the tile ends several times slower.
//
// Structure (one CTA per SM, clusters of two, 320 threads per CTA):
//   warp 8   TMA producer: both CTAs load their halves; every load completes on the full
//            barrier of the even CTA, which expects the bytes of both;
//   warp 9   TMEM allocation (both CTAs) and, in the even CTA, the single MMA-issuing thread;
//            its commits arrive on the barriers of both CTAs (multicast);
//   warps 0-7 epilogue: drain this SM's accumulator (tcgen05.ld), release the slot on the even
//            CTA's barrier (a remote arrival from the odd CTA), and reduce finished tiles into C;
//   warps 10-11 (int16 with the overlapped A split only): convert A's row panels past the first
//            wave of tiles into the limb planes while the tensor cores work on the first ones; a
//            producer loads a tile only once its panel's counter in global memory is complete.
//            Measured at 8192^3: the kernel runs about 30 us longer, the split launch before it
//            58 us shorter.
// Every wait is bounded (a timeout records GEMMI_ETIMEOUT in the status word); a final handshake
// between the two CTAs keeps each alive until its peer no longer signals it.
#include <cuda.h>
#include <cuda_fp16.h>

#include <type_traits>

#include "internal.h"
#include "ptx.cuh"
#include "ptx_pair.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

using tc::BK;
using tc::UMMA_K;

constexpr int NUM_EPI_WARPS = 8;
constexpr int PRODUCER_WARP = 8;
constexpr int MMA_WARP = 9;
constexpr int NUM_THREADS = 10 * 32;
constexpr int TMEM_COLS = 512;
constexpr int NSLOT = 2;                      // accumulator slots of 256 columns
constexpr int SLOT_COLS = 256;
constexpr int UMMA_M = 256;
constexpr int UMMA_N = 256;
constexpr int HALF = 128;                     // rows of A, and of K-major B, per CTA and stage
constexpr int TILE_A = HALF * BK * 2;         // 16 KB
constexpr int TILE_B = HALF * BK * 2;         // 16 KB
constexpr int SBK = TILE_A + TILE_B;          // one CTA's tiles of one K block
// Two K blocks per pipeline stage: the single MMA thread waits on a stage barrier and commits once
// per eight MMAs instead of four.  That per-stage work does not overlap the tensor pipe (the
// thread cannot run far ahead of the MMAs it issues), so halving it raises the pipe's busy time.
constexpr int KPS = 2;
constexpr int SB = KPS * SBK;                 // one CTA's part of a stage
constexpr int STAGES = 3;
constexpr int SWIZZLE = BK * 2;               // 128-byte rows
constexpr int RED_BYTES = 128;                // bytes of C per row of one reduction box
constexpr int STG_WARP = 32 * RED_BYTES;      // one warp's box: 32 rows x 128 bytes, 128-byte swizzle
constexpr int STG_BYTES = NUM_EPI_WARPS * STG_WARP;
constexpr int NBAR = 2 * STAGES + 2 * NSLOT + 2;  // full, empty, slot full, slot empty, final, bye
constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * SB + STG_BYTES + 8 * NBAR + 16;
static_assert(SMEM <= 227 * 1024, "shared memory budget");
static_assert((8 % KPS) == 0, "exact chunks (multiples of 8 K blocks) must end on stage boundaries");
static_assert(NSLOT * SLOT_COLS <= TMEM_COLS, "tensor memory budget");
// Overlapped A split: two more warps per CTA (warps 10-11) convert A's later row panels into the
// limb planes while the tensor cores work on the first ones.  A work item is one row panel
// (128 rows) x AHEAD_KQ reduction indices: each lane owns 8 columns (16 bytes) of every row.
constexpr int AHEAD_WARPS = 2;
constexpr int AHEAD_WARP0 = 10;
constexpr int AHEAD_KQ = 256;
constexpr int AHEAD_ROWS_IN_FLIGHT = 8;     // 16-byte loads in flight per lane
constexpr uint32_t SITE_AHEAD_WAIT = 26;

// Output tile of one pair and where each CTA's operand rows start inside it.
template <int NL>
struct PairGeom;
template <>
struct PairGeom<2> {
  static constexpr int TM = 128, TN = 128;           // output tile
  static constexpr int A_STEP = 0, B_STEP = 0;       // both CTAs read the same rows (other limb)
  static constexpr int COLS = 64;                    // output columns per epilogue thread
};
template <>
struct PairGeom<1> {
  static constexpr int TM = 256, TN = 256;
  static constexpr int A_STEP = 128, B_STEP = 128;   // the odd CTA's rows / columns
  static constexpr int COLS = 128;
};

struct PairParams {
  int64_t m, n, k;
  void* C;
  int64_t ldc;
  int num_m_tiles, num_n_tiles, num_k_blocks;
  int group_m;
  int hint_a, hint_b;
  uint64_t timeout_ns;
  uint32_t* status;
};

// The overlapped A split's parameters (AHEAD kernels only).
struct AheadParams {
  int64_t m, k;
  const int16_t* a_raw;
  int64_t lda;
  __half* a_p0;          // A's limb planes (pitch k)
  __half* a_p1;
  uint32_t* ahead;       // [0] claimed items, [1] finished items, [2 + p] finished items of row panel p
  int ahead_first;       // first row panel the kernel splits
  int ahead_nq;          // items per row panel
  uint32_t ahead_items;  // items in all
};

__device__ __forceinline__ void load_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y, int hint,
                                          uint64_t policy) {
  if (hint == 0) tma_load_2d_pair(dst, map, bar, x, y);
  else tma_load_2d_pair_hint(dst, map, bar, x, y, policy);
}

// The work of one pair.  While a full wave of tiles remains, whole tiles round-robin
// (t = pair, pair + npairs, ...), so the pairs running at one time share operand rows and
// columns in L2.  The last, partial wave is split along K ("stream-K"): its K blocks are dealt
// out evenly to up to npairs pairs, in shares of at least MIN_SHARE K blocks, and a share may
// start or end inside a tile.  Every segment's sums reach C through the same reductions, so the
// pieces of a tile need no further combining.  Every role replays the same schedule.
constexpr int MIN_SHARE = 4;
struct PairSched {
  int64_t nkb, full_tiles, next_tile, u, uend;
  int npairs;
  __device__ __forceinline__ void init(int pair, int npairs_, int64_t tiles, int64_t nkb_) {
    nkb = nkb_;
    npairs = npairs_;
    full_tiles = (tiles / npairs) * npairs;
    next_tile = pair;
    const int64_t tail_units = (tiles - full_tiles) * nkb;
    const int64_t max_split = nkb / MIN_SHARE > 1 ? nkb / MIN_SHARE : 1;
    const int64_t sharers = min(static_cast<int64_t>(npairs), (tiles - full_tiles) * max_split);
    const int64_t base = full_tiles * nkb;
    u = uend = base;
    if (pair < sharers) {
      u = base + tail_units * pair / sharers;
      uend = base + tail_units * (pair + 1) / sharers;
    }
  }
  // The next segment: a tile and its K blocks [kb0, kb1).  False when the pair's work is done.
  __device__ __forceinline__ bool next(int& tile, int& kb0, int& kb1) {
    if (next_tile < full_tiles) {
      tile = static_cast<int>(next_tile);
      kb0 = 0;
      kb1 = static_cast<int>(nkb);
      next_tile += npairs;
      return true;
    }
    if (u < uend) {
      const int64_t t = u / nkb;
      const int64_t k0 = u - t * nkb;
      const int64_t k1 = min(nkb, k0 + (uend - u));
      tile = static_cast<int>(t);
      kb0 = static_cast<int>(k0);
      kb1 = static_cast<int>(k1);
      u += k1 - k0;
      return true;
    }
    return false;
  }
};

// The epilogue of one CTA.  For int16 the weights of accumulator columns 0-127 and 128-255 depend
// on the CTA's A limb: 2^16 | 2^8 in the even CTA, 2^8 | 1 in the odd one.  Both CTAs drain
// with the odd CTA's weights (one code path, constant shifts) and the even CTA scales its tile's
// sums by 2^8 when it adds them into C: shifting commutes with addition modulo 2^64.
template <int NL, int KPC>
__device__ __forceinline__ void epilogue(const PairParams& P, const CUtensorMap* cmap, uint32_t rank,
                                         uint32_t tmem_base, uint32_t sfull0, uint32_t sempty_leader0, uint8_t* stg,
                                         int pair, int npairs) {
  const uint32_t tile_shift = (NL == 2 && rank == 0) ? 8u : 0u;
  using G = PairGeom<NL>;
  using CT = typename std::conditional<NL == 2, int64_t, int32_t>::type;
  using UT = typename std::conditional<NL == 2, uint64_t, uint32_t>::type;
  constexpr int COLS = G::COLS;
  constexpr int EPR = RED_BYTES / static_cast<int>(sizeof(CT));  // elements per reduction
  constexpr int ROUNDS = COLS / EPR;
  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int quad = warp & 3;   // TMEM lanes 32*quad .. +31 (the warp's hardware lane quadrant)
  const int half = warp >> 2;  // output columns half*COLS .. +COLS-1 of the tile
  uint8_t* wstg = stg + warp * STG_WARP;
  const uint32_t wstg_s = smem_u32(wstg);
  PairSched sched;
  sched.init(pair, npairs, static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles, P.num_k_blocks);
  int chunk = 0;
  bool ok = true;
  UT acc[COLS];
  int t, kb0, kb1;
  while (ok && sched.next(t, kb0, kb1)) {
    int mt, nt;
    tc::tile_coords(t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
    const int nchunks = (kb1 - kb0 + KPC - 1) / KPC;
    const int64_t row0 = static_cast<int64_t>(mt) * G::TM + rank * G::A_STEP + quad * 32;  // the warp's rows
    const int64_t col0 = static_cast<int64_t>(nt) * G::TN + half * COLS;
#pragma unroll
    for (int c = 0; c < COLS; ++c) acc[c] = 0;
    for (int ch = 0; ch < nchunks; ++ch, ++chunk) {
      const int slot = chunk & 1;
      const uint32_t use = static_cast<uint32_t>(chunk >> 1);
      // every lane waits; the warp then decides together (tcgen05.ld needs a converged warp)
      const bool got = bounded_wait(sfull0 + 8 * slot, use & 1u, P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, got)) {
        if (lane == 0) report_status(P.status, tc::STATUS_TIMEOUT, 24);
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                             static_cast<uint32_t>(slot * SLOT_COLS + half * COLS);
      if constexpr (NL == 2) {
        // this thread's 64 output columns: weight 2^8 from accumulator columns 0-127 (B high
        // limb), 1 from columns 128-255 (B low limb), before the tile shift
#pragma unroll
        for (int c = 0; c < COLS; c += 8) {
          uint32_t rh[8], rl[8];  // eight columns at a time: the 64 running sums take 128 registers
          tc_ld_32x32b_x8(taddr + c, rh);
          tc_ld_32x32b_x8(taddr + 128 + c, rl);
          tc_wait_ld();
#pragma unroll
          for (int i = 0; i < 8; ++i)
            acc[c + i] += (static_cast<UT>(static_cast<CT>(tc::f32_to_i32(rh[i]))) << 8) +
                          static_cast<UT>(static_cast<CT>(tc::f32_to_i32(rl[i])));
        }
      } else {
#pragma unroll
        for (int c = 0; c < COLS; c += 32) {
          uint32_t r0[16], r1[16];
          tc_ld_32x32b_x16(taddr + c, r0);
          tc_ld_32x32b_x16(taddr + c + 16, r1);
          tc_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            acc[c + i] += static_cast<UT>(tc::f32_to_i32(r0[i]));
            acc[c + 16 + i] += static_cast<UT>(tc::f32_to_i32(r1[i]));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(sempty_leader0 + 8 * slot);
    }
    if (!ok) break;
    // add the segment's running sums into C: per round, one 32-row x 128-byte box per warp,
    // written to the staging area in the box's 128-byte-swizzled layout (row r, 16-byte chunk c
    // at r * 128 + (c ^ (r % 8)) * 16: the eight chunk stores of a warp hit distinct banks)
    if (row0 < P.m) {
#pragma unroll
      for (int j = 0; j < ROUNDS; ++j) {
        const int64_t x = col0 + j * EPR;
        if (x >= P.n) break;
        if (lane == 0) bulk_wait_read_all();  // the previous box has left the staging area
        __syncwarp();
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          uint8_t* dst = wstg + lane * RED_BYTES + ((q ^ (lane & 7)) << 4);
          if constexpr (NL == 2) {
            *reinterpret_cast<ulonglong2*>(dst) =
                make_ulonglong2(acc[j * EPR + 2 * q] << tile_shift, acc[j * EPR + 2 * q + 1] << tile_shift);
          } else {
            *reinterpret_cast<uint4*>(dst) = make_uint4(acc[j * EPR + 4 * q], acc[j * EPR + 4 * q + 1],
                                                        acc[j * EPR + 4 * q + 2], acc[j * EPR + 4 * q + 3]);
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_reduce_add_2d(cmap, wstg_s, static_cast<int32_t>(x), static_cast<int32_t>(row0));
          bulk_commit();
        }
      }
    }
  }
  if (lane == 0) bulk_wait_all();
}

// The splitter warps of the overlapped A split.  Items (row panel p, reduction range q) are
// claimed in order, panel by panel, so the panels the raster reaches first are finished first.
// A warp converts its item (up to 128 rows x 256 columns of raw A: 512 bytes of each row per
// warp-wide load) into both limb planes, then publishes it: every lane orders its stores for the
// async proxy (the TMA loads that will read them) and for the GPU, and one lane adds the item to
// its panel's count and to the total with release semantics.  The splitters wait for nothing, so
// every claimed item is finished.
__device__ __forceinline__ void split_ahead(const AheadParams& P) {
  constexpr int U = AHEAD_ROWS_IN_FLIGHT;
  const int lane = threadIdx.x % 32;
  while (true) {
    uint32_t item = 0;
    if (lane == 0) item = atomicAdd(P.ahead, 1u);
    item = __shfl_sync(0xFFFFFFFFu, item, 0);
    if (item >= P.ahead_items) break;
    const int p = P.ahead_first + static_cast<int>(item / static_cast<uint32_t>(P.ahead_nq));
    const int q = static_cast<int>(item % static_cast<uint32_t>(P.ahead_nq));
    const int64_t r0 = static_cast<int64_t>(p) * PairGeom<2>::TM;
    const int rows = static_cast<int>(min(static_cast<int64_t>(PairGeom<2>::TM), P.m - r0));
    const int64_t c0 = static_cast<int64_t>(q) * AHEAD_KQ + lane * 8;
    if (c0 < P.k) {  // k % 8 == 0: the lane's 8 columns are all inside the row
      const int16_t* src = P.a_raw + r0 * P.lda + c0;
      __half* d0 = P.a_p0 + r0 * P.k + c0;
      __half* d1 = P.a_p1 + r0 * P.k + c0;
      for (int r = 0; r < rows; r += U) {
        uint4 v[U];
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (r + u < rows) v[u] = ld_nc_v4(src + static_cast<int64_t>(r + u) * P.lda);
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (r + u < rows) {
            uint4 h, l;
            tc::limbs16x2(v[u].x, h.x, l.x);
            tc::limbs16x2(v[u].y, h.y, l.y);
            tc::limbs16x2(v[u].z, h.z, l.z);
            tc::limbs16x2(v[u].w, h.w, l.w);
            *reinterpret_cast<uint4*>(d0 + static_cast<int64_t>(r + u) * P.k) = h;
            *reinterpret_cast<uint4*>(d1 + static_cast<int64_t>(r + u) * P.k) = l;
          }
        }
      }
    }
    fence_proxy_async_global();
    __threadfence();
    __syncwarp();
    if (lane == 0) {
      red_release_gpu_add(P.ahead + 2 + p, 1u);
      red_release_gpu_add(P.ahead + 1, 1u);
    }
  }
}

// K blocks per exact chunk.  fp16 limbs: a K block is 64 indices of products of magnitude <= 2^14,
// so 8 * CS blocks keep every fp32 partial sum within 2^(23 + CS - 1).  E4M3 int4 values: a K block
// is 128 indices of products <= 2^6; CS = 2 gives 2048 blocks (2^18 indices, sums <= 2^24), CS = 1
// two blocks (256 indices, sums <= 2^14).  Every length is a multiple of KPS.
template <int CS, bool F8>
__host__ __device__ constexpr int chunk_kblocks() {
  return F8 ? (CS == 2 ? 2048 : 2) : 8 * CS;
}

template <int NL, int CS, bool F8, bool AHEAD>
__global__ void __launch_bounds__(AHEAD ? NUM_THREADS + 32 * AHEAD_WARPS : NUM_THREADS, 1)
tc_pair_kernel(const __grid_constant__ CUtensorMap mapA0, const __grid_constant__ CUtensorMap mapA1,
               const __grid_constant__ CUtensorMap mapB0, const __grid_constant__ CUtensorMap mapB1,
               const __grid_constant__ CUtensorMap mapC, PairParams P, AheadParams H) {
  using G = PairGeom<NL>;
  static_assert(!F8 || NL == 1, "the E4M3 path has one plane per operand");
  static_assert(!AHEAD || (NL == 2 && !F8), "the overlapped split is the int16 path's");
  constexpr int KPC = chunk_kblocks<CS, F8>();
  static_assert(KPC % KPS == 0, "chunks end on stage boundaries");
  constexpr int BKE = F8 ? 2 * BK : BK;  // elements per K block: 128 bytes of a row either way

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* stg = smem + STAGES * SB;
  uint64_t* bars = reinterpret_cast<uint64_t*>(stg + STG_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t sfull0 = empty0 + 8 * STAGES;
  const uint32_t sempty0 = sfull0 + 8 * NSLOT;
  const uint32_t final_bar = sempty0 + 8 * NSLOT;
  const uint32_t bye_bar = final_bar + 8;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + NBAR);

  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);   // the even CTA's producer arrives (with both CTAs' bytes)
      mbar_init(empty0 + 8 * s, 1);  // one commit of the MMA thread
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(sfull0 + 8 * s, 1);
      mbar_init(sempty0 + 8 * s, 2 * NUM_EPI_WARPS);  // every epilogue warp of both CTAs
    }
    mbar_init(final_bar, 1);
    mbar_init(bye_bar, 1);
    fence_mbar_init();
  }
  if (warp == MMA_WARP) {
    tmem_alloc_pair(smem_u32(tmem_holder), TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // Launched with programmatic stream serialization: the setup above may overlap the end of the
  // previous kernel (the operand split); every global access comes after this wait.  The next
  // kernel may be scheduled as this grid's CTAs retire.
  pdl_wait();
  pdl_launch_dependents();

  const int pair = static_cast<int>(cluster_id_x());
  const int npairs = static_cast<int>(cluster_count_x());
  const int64_t total_tiles = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles;
  PairSched sched;
  sched.init(pair, npairs, total_tiles, P.num_k_blocks);

  if (warp == PRODUCER_WARP) {
    // ------------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      const CUtensorMap* ma = (NL == 2 && rank == 1) ? &mapA1 : &mapA0;
      const CUtensorMap* mb = (NL == 2 && rank == 1) ? &mapB1 : &mapB0;
      tma_prefetch_desc(ma);
      tma_prefetch_desc(mb);
      const uint64_t pol_a = tc::l2_policy(P.hint_a);
      const uint64_t pol_b = tc::l2_policy(P.hint_b);
      const uint32_t full_leader0 = map_to_rank(full0, 0);
      tc::RingPos st;
      int64_t issued = 0;
      bool ok = true;
      int t, kb0, kb1;
      bool all_split = !AHEAD;  // overlapped split: every panel finished (then no more checks)
      int ready_mt = -1;        // the last panel found finished
      while (ok && sched.next(t, kb0, kb1)) {
        int mt, nt;
        tc::tile_coords(t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
        if constexpr (AHEAD) {
          // the tile's A panel must be in the limb planes before its first load
          if (!all_split && mt >= H.ahead_first && mt != ready_mt) {
            if (ld_acquire_gpu(H.ahead + 1) >= H.ahead_items) {
              all_split = true;
            } else if (!bounded_wait_counter(H.ahead + 2 + mt, static_cast<uint32_t>(H.ahead_nq), P.timeout_ns)) {
              report_status(P.status, tc::STATUS_TIMEOUT, SITE_AHEAD_WAIT);
              ok = false;
              break;
            }
            fence_proxy_async_global();
            ready_mt = mt;
          }
        }
        const int arow = mt * G::TM + static_cast<int>(rank) * G::A_STEP;
        const int brow = nt * G::TN + static_cast<int>(rank) * G::B_STEP;
        // stages hold KPS consecutive K blocks of a segment (its last stage possibly fewer)
        for (int kb = kb0; kb < kb1; kb += KPS) {
          const int nsub = min(KPS, kb1 - kb);
          if (!spin_wait(empty0 + 8 * st.slot, st.phase ^ 1u, P.timeout_ns)) {
            report_status(P.status, tc::STATUS_TIMEOUT, 21);
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full0 + 8 * st.slot, 2 * nsub * SBK);
          const uint32_t fb = full_leader0 + 8 * st.slot;
#pragma unroll
          for (int j = 0; j < KPS; ++j) {
            if (j >= nsub) break;
            const uint32_t base = smem_u32(smem + st.slot * SB + j * SBK);
            load_pair(base, ma, fb, (kb + j) * BKE, arow, P.hint_a, pol_a);
            load_pair(base + TILE_A, mb, fb, (kb + j) * BKE, brow, P.hint_b, pol_b);
          }
          ++issued;
          st.advance(STAGES);
        }
      }
      // no copy of this CTA may still be landing when it exits: the last stages must have been
      // consumed by the MMAs (which waited for every byte of them)
      const int64_t first = issued > STAGES ? issued - STAGES : 0;
      for (int64_t i = first; i < issued; ++i)
        bounded_wait(empty0 + 8 * static_cast<int>(i % STAGES), static_cast<uint32_t>((i / STAGES) & 1), P.timeout_ns);
    }
  } else if (warp == MMA_WARP) {
    // ------------------------------------------------------------ MMA issue (even CTA, one thread)
    if (lane == 0) {
      if (leader) {
        constexpr uint32_t idesc = F8 ? idesc_e4m3_f32(UMMA_M, UMMA_N) : idesc_f16_f32(UMMA_M, UMMA_N);
        tc::RingPos st;
        int chunk = 0;
        bool ok = true;
        int t, kb0, kb1;
        while (ok && sched.next(t, kb0, kb1)) {
          const int nchunks = (kb1 - kb0 + KPC - 1) / KPC;
          for (int ch = 0; ch < nchunks; ++ch, ++chunk) {
            const int slot = chunk & 1;
            const uint32_t use = static_cast<uint32_t>(chunk >> 1);
            // the slot's previous chunk must have been drained by both CTAs
            if (!bounded_wait_cluster(sempty0 + 8 * slot, (use & 1u) ^ 1u, P.timeout_ns)) {
              report_status(P.status, tc::STATUS_TIMEOUT, 22);
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t d = tmem_base + static_cast<uint32_t>(slot * SLOT_COLS);
            const int cb0 = kb0 + ch * KPC;
            const int cb1 = min(kb1, cb0 + KPC);
            // chunk lengths are multiples of KPS, so chunks and stages share boundaries
            for (int kb = cb0; kb < cb1; kb += KPS) {
              const int nsub = min(KPS, cb1 - kb);
              if (!spin_wait(full0 + 8 * st.slot, st.phase, P.timeout_ns)) {
                report_status(P.status, tc::STATUS_TIMEOUT, 23);
                ok = false;
                break;
              }
              tc_fence_after();
#pragma unroll
              for (int j = 0; j < KPS; ++j) {
                if (j >= nsub) break;
                const uint32_t base = smem_u32(smem + st.slot * SB + j * SBK);
                const uint64_t adesc = smem_desc_kmajor<SWIZZLE>(base);
                const uint64_t bdesc = smem_desc_kmajor<SWIZZLE>(base + TILE_A);
#pragma unroll
                for (int kk = 0; kk < BK / UMMA_K; ++kk) {
                  // advancing the start address by 32 bytes (16 fp16 or 32 E4M3) steps K inside the
                  // swizzled row
                  const uint32_t acc = (kb + j == cb0 && kk == 0) ? 0u : 1u;
                  if constexpr (F8) tc_mma_f8_pair(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, acc);
                  else tc_mma_f16_pair(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, acc);
                }
              }
              tc_commit_pair(empty0 + 8 * st.slot, 0x3);  // stage free in both CTAs once read
              st.advance(STAGES);
            }
            if (!ok) break;
            tc_commit_pair(sfull0 + 8 * slot, 0x3);  // chunk ready to drain in both CTAs
          }
        }
        tc_commit_pair(final_bar, 0x3);
      }
      // both CTAs: every MMA of the pair, and every commit arrival, has landed
      bounded_wait(final_bar, 0, P.timeout_ns);
    }
  } else if (AHEAD && warp >= AHEAD_WARP0) {
    // ------------------------------------------------------------ overlapped A split (warps 10-11)
    if constexpr (AHEAD) split_ahead(H);
  } else {
    // ------------------------------------------------------------ epilogue (warps 0..7)
    const uint32_t sempty_leader0 = map_to_rank(sempty0, 0);
    epilogue<NL, KPC>(P, &mapC, rank, tmem_base, sfull0, sempty_leader0, stg, pair, npairs);
  }

  // Pair handshake: neither CTA exits (or frees tensor memory) while its peer may still signal it.
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    mbar_arrive_cluster(map_to_rank(bye_bar, rank ^ 1u));
    if (!bounded_wait_cluster(bye_bar, 0, P.timeout_ns)) report_status(P.status, tc::STATUS_TIMEOUT, 25);
  }
  __syncthreads();
  if (warp == MMA_WARP) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------- host side
template <int NL, int CS, bool F8, bool AHEAD = false>
cudaError_t launch_pair(const TcGemmArgs& a, cudaStream_t s, const char** why) {
  using G = PairGeom<NL>;
  constexpr int BKE = F8 ? 2 * BK : BK;
  constexpr int OPSZ = F8 ? 1 : 2;  // bytes per plane element
  CUtensorMap maps[4];
  const LimbPlanes* ops[2] = {&a.a, &a.b};
  for (int o = 0; o < 2; ++o) {
    for (int l = 0; l < 2; ++l) {
      const void* base = ops[o]->plane[l < NL ? l : 0];
      if (!encode_tensor_map_2d(&maps[2 * o + l], F8 ? 2 : 1, base, static_cast<uint64_t>(a.k),
                                static_cast<uint64_t>(ops[o]->rows), static_cast<uint64_t>(ops[o]->pitch) * OPSZ,
                                BKE, HALF, SWIZZLE, why))
        return cudaErrorInvalidValue;
    }
  }
  // C as the target of the tile reductions: an unsigned integer tensor of its element width
  CUtensorMap mapC;
  constexpr int ESZ = NL == 2 ? 8 : 4;
  if (!encode_tensor_map_2d(&mapC, NL == 2 ? 3 : 4, a.C, static_cast<uint64_t>(a.n), static_cast<uint64_t>(a.m),
                            static_cast<uint64_t>(a.ldc) * ESZ, RED_BYTES / ESZ, 32, 128, why))
    return cudaErrorInvalidValue;
  PairParams P;
  P.m = a.m;
  P.n = a.n;
  P.k = a.k;
  P.C = a.C;
  P.ldc = a.ldc;
  P.num_m_tiles = static_cast<int>((a.m + G::TM - 1) / G::TM);
  P.num_n_tiles = static_cast<int>((a.n + G::TN - 1) / G::TN);
  P.num_k_blocks = static_cast<int>((a.k + BKE - 1) / BKE);
  P.group_m = a.group_m > 0 ? a.group_m : 16;
  P.hint_a = a.hint_a;
  P.hint_b = a.hint_b;
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  AheadParams H = {};
  if constexpr (AHEAD) {
    if (a.a_raw == nullptr || a.ahead == nullptr || a.k % 8 != 0 || a.lda % 8 != 0 || a.a.pitch != a.k ||
        reinterpret_cast<uintptr_t>(a.a_raw) % 16 != 0 || a.ahead_first < 0 || a.ahead_first >= P.num_m_tiles) {
      *why = "overlapped A split: unsupported operand layout";
      return cudaErrorInvalidValue;
    }
    H.m = a.m;
    H.k = a.k;
    H.a_raw = a.a_raw;
    H.lda = a.lda;
    H.a_p0 = static_cast<__half*>(a.a.plane[0]);
    H.a_p1 = static_cast<__half*>(a.a.plane[1]);
    H.ahead = a.ahead;
    H.ahead_first = a.ahead_first;
    H.ahead_nq = static_cast<int>((a.k + AHEAD_KQ - 1) / AHEAD_KQ);
    H.ahead_items = static_cast<uint32_t>(static_cast<int64_t>(P.num_m_tiles - a.ahead_first) * H.ahead_nq);
  }
  const int64_t tiles = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles;

  auto kernel = tc_pair_kernel<NL, CS, F8, AHEAD>;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(AHEAD ? NUM_THREADS + 32 * AHEAD_WARPS : NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;  // the occupancy query sees the cluster shape only
  // the shared-memory opt-in and the number of co-resident pairs, once per device
  static int max_pairs[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  int pairs_here = (dev >= 0 && dev < 64) ? max_pairs[dev] : 0;
  if (pairs_here == 0) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(SMEM));
    if (e != cudaSuccess) return e;
    cfg.gridDim = dim3(2 * static_cast<unsigned>(a.num_sms / 2), 1, 1);
    e = cudaOccupancyMaxActiveClusters(&pairs_here, kernel, &cfg);
    if (e != cudaSuccess) return e;
    if (pairs_here <= 0) {
      *why = "no two SMs can host a CTA pair of the tcgen05 pair GEMM";
      return cudaErrorInvalidConfiguration;
    }
    if (dev >= 0 && dev < 64) max_pairs[dev] = pairs_here;
  }
  // enough pairs for every tile, or for every stream-K share when there are fewer tiles than pairs
  const int64_t max_split = P.num_k_blocks / MIN_SHARE > 1 ? P.num_k_blocks / MIN_SHARE : 1;
  const int64_t useful = tiles * max_split;
  const int npairs = static_cast<int>(useful < pairs_here ? useful : pairs_here);
  cfg.gridDim = dim3(2 * static_cast<unsigned>(npairs), 1, 1);
  *why = "tcgen05 pair GEMM launch";
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, maps[0], maps[1], maps[2], maps[3], mapC, P, H);
}

}  // namespace

cudaError_t tc_pair_gemm_i16(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  if (args.a_raw != nullptr)
    return args.chunk_scale == 2 ? launch_pair<2, 2, false, true>(args, s, why)
                                 : launch_pair<2, 1, false, true>(args, s, why);
  return args.chunk_scale == 2 ? launch_pair<2, 2, false>(args, s, why) : launch_pair<2, 1, false>(args, s, why);
}

int pair_first_wave_panels(int64_t m, int64_t n, int group_m, int num_sms) {
  const int num_m = static_cast<int>((m + PairGeom<2>::TM - 1) / PairGeom<2>::TM);
  const int num_n = static_cast<int>((n + PairGeom<2>::TN - 1) / PairGeom<2>::TN);
  const int gm = group_m > 0 ? group_m : 16;
  const int64_t tiles = static_cast<int64_t>(num_m) * num_n;
  const int first_wave = static_cast<int>(tiles < num_sms / 2 ? tiles : num_sms / 2);
  int panels = 0;
  for (int t = 0; t < first_wave; ++t) {
    int mt, nt;
    tc::tile_coords(t, num_m, num_n, gm, mt, nt);
    if (mt + 1 > panels) panels = mt + 1;
  }
  return panels;
}
cudaError_t tc_pair_gemm_i8(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch_pair<1, 2, false>(args, s, why) : launch_pair<1, 1, false>(args, s, why);
}
cudaError_t tc_pair_gemm_i4(const TcGemmArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch_pair<1, 2, true>(args, s, why) : launch_pair<1, 1, true>(args, s, why);
}

}  // namespace gemmi
