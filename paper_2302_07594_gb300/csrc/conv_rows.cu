// conv_rows.cu -- exact int16 "same" convolution (stride 1) that splits every input pixel once.
//
// What it computes: the convolution of gemmi_conv2d_i16,
//   Y[n][h][w][co] += sum over r < R, s < S, c < 64 of
//                     X[n][h + r - ph][w + s - pw][c] * Wt[(r*S + s)*64 + c][co],
// X read as 0 outside the image, bit-exactly modulo 2^64, for 64 input channels, at most 64 output
// channels and odd R, S (R*S <= 12) with ph = (R - 1) / 2, pw = (S - 1) / 2 (the output has the
// input's size).  Sections 2 and 3 of the paper lower a convolution to one GEMM (IM2COL) and note
// that the lowering can be done on the fly while the activations are packed; this kernel packs
// each activation once for all filter taps.
//
// Why a kernel of its own.  The lowered matrix holds every input pixel R*S times.  The narrow-n
// fused kernel (gemm_fused.cu) reads it tap by tap and splits every copy into limbs, so its
// converters do R*S times the work of the input.  Here a CTA splits the input rows that a tile
// needs once, into shared memory, in a layout in which every filter tap is a shifted window.
//
// Geometry.  Wp = W + 2*pw is a padded image row.  A tile is T consecutive output rows of one
// image (T * Wp <= 128).  MMA row p (0..127) is output pixel (h0 + p / Wp, p % Wp); it is stored
// when p / Wp < T, h0 + p / Wp < H and p % Wp < W (the other rows are computed and dropped).
// Buffer position q holds input pixel (h0 - ph + q / Wp, q % Wp - pw), zero outside the image, so
// tap (r, s) of MMA row p is buffer position p + r*Wp + s: the A operand of tap (r, s) is the 128
// positions from r*Wp + s on (an output pixel's taps never leave its padded row).
//
// Shared-memory layout of a limb plane: K-major with the 128-byte swizzle, one 128-byte row per
// position (64 channels), the 16-byte chunk of channel octet c of position q at chunk c ^ (q % 8).
// The window from position q0 on is the matrix descriptor with start address + 128*q0 (the
// swizzle follows the address bits, so the matrix base offset stays 0 at any start row); the
// eight threads that store one position's eight chunks hit distinct bank groups.
//
// Arithmetic.  Every buffered int16 is split into its centred limbs a = 256h + l (h in [-128,128],
// l in [-128,127], exact in fp16; the split of split.cu).  Per tap, limb e of the window times
// the stacked limb tiles of B (the weights, split once per call: B_high in columns 0-63, B_low in
// columns 64-127) accumulates into accumulator e (N = 128) in TMEM.  Each column sums R*S*64 <= 512*CS products of magnitude <= 2^14, exactly in fp32.  The
// epilogue weights the four quarters by 2^16, 2^8, 2^8 and 1 into int64 and adds each valid image
// row of the tile into Y with 2-D tensor reductions (16 channels x W pixels each) through an
// unsigned 64-bit tensor map, so the adds wrap modulo 2^64 and Y is never read by the SMs.
//
// SM pairs.  Two CTAs of a cluster, on two SMs, take two consecutive tiles, and one thread of the
// even CTA issues tcgen05.mma.cta_group::2 of M = 256: MMA rows 0-127 are the even CTA's window,
// rows 128-255 the odd CTA's (each CTA's limb planes at the same shared-memory offsets), and the
// stacked weights are split between them (B_high rows in the even CTA, B_low rows in the odd
// one).  Each SM so reads 4 KB of pixels and 2 KB of weights per MMA step instead of 4 + 4.  Each
// CTA loads its half of the weights' limb tiles for every tap once, when it starts, and keeps them:
// the MMA threads then wait and commit once per tile, not once per tap (the per-tap stage
// handshakes drained the tensor pipe at every tap boundary).
//
// Roles (one CTA per SM, clusters of two, 608 threads per CTA):
//   warps 0-7   epilogue: warp w drains TMEM lanes 32*(w % 4) .. +31 (MMA rows) for output
//               channels 32*(w / 4) .. +31, into a 128-byte-swizzled staging area;
//               lane 0 of warp 0 issues the tile's reductions;
//   warps 8-15  converters: load the next tile's pixels into registers while the tensor cores
//               work on the current one, then split them into the limb planes once those MMAs
//               are done;
//   warp 16     TMEM allocation (both CTAs); lane 0 loads this CTA's half of B's stacked limb
//               tiles (one per tap) by TMA, every load completing on the even CTA's barrier;
//   warps 17-18 lane 0 of the even CTA: the MMA issuer of A limb 0 (high) and of A limb 1 (low);
//               their commits arrive on the barriers of both CTAs.
// Every wait is bounded by the global timer; one that runs out records GEMMI_ETIMEOUT in the
// status word and the CTA winds down.  Before either CTA of a pair frees tensor memory or exits,
// the two exchange one arrival, so neither outlives signals aimed at it.
#include <cuda.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"
#include "ptx_pair.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

using tc::STATUS_TIMEOUT;

constexpr int BM = 128;                      // MMA rows (buffer window) per CTA and tile
constexpr int BN = 64;                       // output channels per block
constexpr int CIN = 64;                      // input channels
constexpr int UMMA_M = 2 * BM;               // both CTAs' windows
constexpr int UMMA_N = 2 * BN;               // B's two limb tiles stacked
constexpr int UMMA_K = 16;
constexpr int NUM_EPI_WARPS = 8;
constexpr int CONV_WARP0 = 8;
constexpr int NUM_CONV_WARPS = 8;
constexpr int NUM_CONV_THREADS = NUM_CONV_WARPS * 32;
constexpr int B_WARP = 16;
constexpr int ISSUE_WARP0 = 17;
constexpr int NUM_THREADS = 19 * 32;
constexpr int PB_MAX = 256;                  // buffered positions
constexpr int ITEMS_PER_THREAD = PB_MAX * 8 / NUM_CONV_THREADS;  // 16-byte cells per converter thread
constexpr int LIMB_BYTES = PB_MAX * 128;     // one limb plane: a 128-byte row per position
constexpr int MAX_TAPS = 12;                 // R * S: this CTA's weight halves stay resident
constexpr int TILE_BH = BN * CIN * 2;        // 8 KB: this CTA's half of a stacked limb tile
constexpr int STG_ROWS = 120;                // staged output pixels per tile: T * round_up(W, 8)
constexpr int STG_G = STG_ROWS * 128;        // one group of 16 output channels (int64)
constexpr int OFF_LIMB = 0;
constexpr int OFF_B = 2 * LIMB_BYTES;
constexpr int OFF_STG = OFF_B + MAX_TAPS * TILE_BH;
constexpr int OFF_BAR = OFF_STG + 4 * STG_G;
// limbs full / empty, B full, accumulator full / empty (two slots), staging full / free, final, bye
constexpr int NBAR = 2 + 1 + 4 + 2 + 2;
constexpr size_t SMEM = 1024 + static_cast<size_t>(OFF_BAR) + 8 * NBAR + 16;
static_assert(SMEM <= 227 * 1024, "shared memory budget");
static_assert(OFF_B % 1024 == 0 && OFF_STG % 1024 == 0 && STG_G % 1024 == 0 && TILE_BH % 1024 == 0,
              "1024-byte aligned TMA areas");
constexpr int TMEM_COLS = 512;
constexpr int SLOT_COLS = 2 * UMMA_N;        // both accumulators of one (tile, channel block)

struct ConvParams {
  const int16_t* X;
  int H, W, R, S, ph, pw;
  int Wp, T, PB, wpad;
  int tiles_per_image, num_tiles, num_pair_tiles, cout;
  uint64_t timeout_ns;
  uint32_t* status;
};

// Shared-memory descriptor of a K-major operand with 128-byte rows in the 128-byte swizzle whose
// start need not be 1024-byte aligned: groups of 8 rows 1024 bytes apart (stride byte offset).  The
// swizzle follows the address bits, so a window that starts r rows into the plane reads the rows
// the converters stored there (the matrix base offset stays 0; measured exact on every start row).
__device__ __forceinline__ uint64_t smem_desc_kmajor_sw128_at(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1u) << 16;                        // leading byte offset (unused)
  d |= static_cast<uint64_t>((1024u >> 4) & 0x3FFFu) << 32;    // stride byte offset
  d |= static_cast<uint64_t>(1u) << 46;                        // descriptor version for tcgen05
  d |= static_cast<uint64_t>(2u) << 61;                        // 128-byte swizzle
  return d;
}

__device__ __forceinline__ void tc_ld_x8(uint32_t taddr, uint32_t (&r)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "r"(taddr));
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ uint64_t widen(uint32_t f32_bits) {
  return static_cast<uint64_t>(static_cast<int64_t>(tc::f32_to_i32(f32_bits)));
}

// Polls (no suspend hint) a barrier that the peer CTA arrives on, with cluster-scope acquire.
__device__ __forceinline__ bool spin_wait_cluster(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_wait_cluster(bar, parity, 0u)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    for (int i = 0; i < 256; ++i)
      if (mbar_try_wait_cluster(bar, parity, 0u)) return true;
    if (global_timer_ns() - t0 > timeout_ns) return false;
  }
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
conv_rows_kernel(const __grid_constant__ CUtensorMap mapBH, const __grid_constant__ CUtensorMap mapBL,
                 const __grid_constant__ CUtensorMap mapY, ConvParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  const uint32_t limbs_full = smem_u32(bars);           // both CTAs' converters stored (even CTA's)
  const uint32_t limbs_empty = limbs_full + 8;          // the tile's MMAs are done with the planes
  const uint32_t b_full = limbs_empty + 8;              // every tap's halves landed (even CTA's)
  const uint32_t acc_full0 = b_full + 8;
  const uint32_t acc_empty0 = acc_full0 + 16;           // both CTAs' epilogue warps drained (even CTA's)
  const uint32_t stg_full = acc_empty0 + 16;            // this CTA's epilogue warps staged the unit
  const uint32_t stg_free = stg_full + 8;               // the unit's reductions have read the staging
  const uint32_t final_bar = stg_free + 8;
  const uint32_t bye_bar = final_bar + 8;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  if (threadIdx.x == 0) {
    mbar_init(limbs_full, 2 * NUM_CONV_WARPS);
    mbar_init(limbs_empty, 2);
    mbar_init(b_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(acc_full0 + 8 * s, 2);
      mbar_init(acc_empty0 + 8 * s, 2 * NUM_EPI_WARPS);
    }
    mbar_init(stg_full, NUM_EPI_WARPS);
    mbar_init(stg_free, 1);
    mbar_init(final_bar, 2);
    mbar_init(bye_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == B_WARP) {
    tmem_alloc_pair(smem_u32(tmem_holder), TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // Launched with programmatic stream serialization: the set-up above may overlap the previous
  // kernel (the weights' split); every global access comes after this wait.
  pdl_wait();
  pdl_launch_dependents();

  // pair tiles pair, pair + npairs, ...: this CTA's tile is 2 * (pair tile) + rank (none past the end)
  const int pair = static_cast<int>(cluster_id_x());
  const int npairs = static_cast<int>(cluster_count_x());
  const int ntiles = (P.num_pair_tiles - pair + npairs - 1) / npairs;
  const int taps = P.R * P.S;
  auto tile_of = [&](int i) { return 2 * (pair + i * npairs) + static_cast<int>(rank); };

  if (warp >= CONV_WARP0 && warp < CONV_WARP0 + NUM_CONV_WARPS) {
    // ------------------------------------------------------------ converters
    // Thread tid holds cells i = tid + 256 j of the buffer: position q = i / 8, channel octet
    // c = i % 8 (eight consecutive threads load one pixel's 128 bytes).  Positions do not depend
    // on the tile, so their rows and columns are computed once.
    const int tid = threadIdx.x - CONV_WARP0 * 32;
    const int c = tid & 7;
    const int items = P.PB * 8;
    int rb[ITEMS_PER_THREAD], cb[ITEMS_PER_THREAD];
#pragma unroll
    for (int j = 0; j < ITEMS_PER_THREAD; ++j) {
      const int q = (tid >> 3) + 32 * j;
      rb[j] = q / P.Wp;
      cb[j] = q - rb[j] * P.Wp - P.pw;
    }
    uint4 x[ITEMS_PER_THREAD];
    auto fetch = [&](int t) {
      const bool real = t < P.num_tiles;  // the odd CTA of the last pair may have no tile
      const int n = real ? t / P.tiles_per_image : 0;
      const int h0 = real ? (t - n * P.tiles_per_image) * P.T : 0;
#pragma unroll
      for (int j = 0; j < ITEMS_PER_THREAD; ++j) {
        x[j] = make_uint4(0u, 0u, 0u, 0u);
        const int h = h0 - P.ph + rb[j];
        if (real && tid + NUM_CONV_THREADS * j < items && h >= 0 && h < P.H && cb[j] >= 0 && cb[j] < P.W)
          x[j] = ld_nc_v4(P.X + ((static_cast<int64_t>(n) * P.H + h) * P.W + cb[j]) * CIN + c * 8);
      }
    };
    const uint32_t full_leader = map_to_rank(limbs_full, 0);
    const uint32_t l0 = smem_u32(smem + OFF_LIMB);
    const uint32_t l1 = l0 + LIMB_BYTES;
    if (ntiles > 0) fetch(tile_of(0));
    for (int i = 0; i < ntiles; ++i) {
      // the previous tile's MMAs must be done with the planes
      const bool got = bounded_wait(limbs_empty, (static_cast<uint32_t>(i) & 1u) ^ 1u, P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, got && !*abort_flag)) {  // the warp decides together
        if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 41);
        *abort_flag = 1;
        break;
      }
#pragma unroll
      for (int j = 0; j < ITEMS_PER_THREAD; ++j) {
        if (tid + NUM_CONV_THREADS * j < items) {
          uint32_t h[4], l[4];
          tc::limbs16x2(x[j].x, h[0], l[0]);
          tc::limbs16x2(x[j].y, h[1], l[1]);
          tc::limbs16x2(x[j].z, h[2], l[2]);
          tc::limbs16x2(x[j].w, h[3], l[3]);
          const uint32_t q = static_cast<uint32_t>((tid >> 3) + 32 * j);
          const uint32_t off = q * 128u + ((static_cast<uint32_t>(c) ^ (q & 7u)) << 4);
          sts128(l0 + off, h[0], h[1], h[2], h[3]);
          sts128(l1 + off, l[0], l[1], l[2], l[3]);
        }
      }
      fence_proxy_async_smem();  // the tensor cores read the planes through the async proxy
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(full_leader);
      if (i + 1 < ntiles) fetch(tile_of(i + 1));
    }
  } else if (warp == B_WARP) {
    // ------------------------------------------------------------ weights (both CTAs), once
    if (lane == 0 && ntiles > 0) {
      const CUtensorMap* mb = leader ? &mapBH : &mapBL;
      tma_prefetch_desc(mb);
      if (leader) mbar_arrive_expect_tx(b_full, static_cast<uint32_t>(2 * taps * TILE_BH));
      const uint32_t full_leader = map_to_rank(b_full, 0);
      for (int tap = 0; tap < taps; ++tap)
        tma_load_2d_pair(smem_u32(smem + OFF_B + tap * TILE_BH), mb, full_leader, tap * CIN, 0);
      // no copy of this CTA may still be landing when it exits: every MMA of the pair has waited
      // for all of them, and this warp's lane 0 waits for the MMAs to be done (final barrier)
      bounded_wait(final_bar, 0, P.timeout_ns);
    }
  } else if (warp == ISSUE_WARP0 || warp == ISSUE_WARP0 + 1) {
    // ------------------------------------------------------------ MMA issuers (even CTA; issuer e: A limb e)
    if (lane == 0) {
      if (leader) {
        const int me = warp - ISSUE_WARP0;
        constexpr uint32_t idesc = idesc_f16_f32(UMMA_M, UMMA_N);
        bool ok = ntiles == 0 || spin_wait(b_full, 0, P.timeout_ns);
        if (!ok) {
          report_status(P.status, STATUS_TIMEOUT, 45);
          *abort_flag = 1;
        }
        const uint32_t bbase = smem_u32(smem + OFF_B);
        for (int i = 0; i < ntiles && ok; ++i) {
          const int slot = i & 1;
          const uint32_t use = static_cast<uint32_t>(i >> 1);
          if (!spin_wait_cluster(limbs_full, static_cast<uint32_t>(i) & 1u, P.timeout_ns) ||
              !spin_wait_cluster(acc_empty0 + 8 * slot, (use & 1u) ^ 1u, P.timeout_ns) || *abort_flag) {
            report_status(P.status, STATUS_TIMEOUT, 43);
            *abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint32_t limb = smem_u32(smem + OFF_LIMB + me * LIMB_BYTES);
          const uint32_t d = tmem_base + static_cast<uint32_t>(slot * SLOT_COLS + me * UMMA_N);
          for (int tap = 0; tap < taps; ++tap) {
            const int r = tap / P.S;
            const int s = tap - r * P.S;
            const uint32_t a0 = limb + static_cast<uint32_t>((r * P.Wp + s) * 128);
            const uint64_t bdesc = smem_desc_kmajor<128>(bbase + static_cast<uint32_t>(tap * TILE_BH));
#pragma unroll
            for (int kk = 0; kk < CIN / UMMA_K; ++kk) {
              // K step kk: 16 channels, 32 bytes into the swizzled rows of both operands
              const uint64_t adesc = smem_desc_kmajor_sw128_at(a0 + static_cast<uint32_t>(32 * kk));
              tc_mma_f16_pair(d, adesc, bdesc + 2 * kk, idesc, (tap == 0 && kk == 0) ? 0u : 1u);
            }
          }
          tc_commit_pair(acc_full0 + 8 * slot, 0x3);
          tc_commit_pair(limbs_empty, 0x3);
        }
        tc_commit_pair(final_bar, 0x3);
      }
      // both CTAs: every MMA of the pair, and every commit arrival, has landed
      bounded_wait(final_bar, 0, P.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 0-7)
    const int quad = warp & 3;
    const int half = warp >> 2;
    const int p = quad * 32 + lane;  // this thread's MMA row within this CTA's window
    const int hr = p / P.Wp;
    const int wq = p - hr * P.Wp;
    const uint32_t lane_field = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t stg = smem_u32(smem + OFF_STG);
    const uint32_t rowi = static_cast<uint32_t>(hr * P.wpad + wq);
    const uint32_t empty_leader0 = map_to_rank(acc_empty0, 0);
    const bool reducer = warp == 0 && lane == 0;
    int unit = 0;
    bool ok = true;
    for (int i = 0; i < ntiles && ok; ++i) {
      const int t = tile_of(i);
      const bool real = t < P.num_tiles;
      const int n = real ? t / P.tiles_per_image : 0;
      const int h0 = real ? (t - n * P.tiles_per_image) * P.T : 0;
      const bool valid = real && hr < P.T && h0 + hr < P.H && wq < P.W;
      {
        const int slot = unit & 1;
        const uint32_t suse = static_cast<uint32_t>(unit >> 1);
        const uint32_t upar = static_cast<uint32_t>(unit) & 1u;
        // the staging area is free once the previous unit's reductions have read it
        bool got = bounded_wait(stg_free, upar ^ 1u, P.timeout_ns);
        got = got && bounded_wait(acc_full0 + 8 * slot, suse & 1u, P.timeout_ns);
        if (!__all_sync(0xFFFFFFFFu, got && !*abort_flag)) {  // the warp decides together
          if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 46);
          *abort_flag = 1;
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem_base + lane_field + static_cast<uint32_t>(slot * SLOT_COLS + 32 * half);
#pragma unroll
        for (int j = 0; j < 4; ++j) {  // eight output channels at a time
          uint32_t hh[8], hl[8], lh[8], ll[8];
          tc_ld_x8(acc + 8 * j, hh);                        // A high x B high: 2^16
          tc_ld_x8(acc + BN + 8 * j, hl);                   // A high x B low:  2^8
          tc_ld_x8(acc + UMMA_N + 8 * j, lh);               // A low  x B high: 2^8
          tc_ld_x8(acc + UMMA_N + BN + 8 * j, ll);          // A low  x B low:  1
          tc_wait_ld();
          if (valid) {
            uint64_t v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
              v[e] = (widen(hh[e]) << 16) + ((widen(hl[e]) + widen(lh[e])) << 8) + widen(ll[e]);
            // channels 32 half + 8 j .. +7: group 2 half + j / 2, 16-byte chunks 4 (j % 2) .. +3 of
            // the staged row, stored at chunk ^ (row % 8) (the reductions' 128-byte swizzle)
            const uint32_t gbase = stg + static_cast<uint32_t>((2 * half + (j >> 1)) * STG_G) + rowi * 128u;
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
              const uint32_t chunk = static_cast<uint32_t>(4 * (j & 1) + cc) ^ (rowi & 7u);
              sts128(gbase + (chunk << 4), static_cast<uint32_t>(v[2 * cc]), static_cast<uint32_t>(v[2 * cc] >> 32),
                     static_cast<uint32_t>(v[2 * cc + 1]), static_cast<uint32_t>(v[2 * cc + 1] >> 32));
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(empty_leader0 + 8 * slot);
        fence_proxy_async_smem();  // the reductions read the staging area through the async proxy
        __syncwarp();
        if (lane == 0) mbar_arrive(stg_full);
        if (reducer) {
          if (!bounded_wait(stg_full, upar, P.timeout_ns)) {
            report_status(P.status, STATUS_TIMEOUT, 47);
            *abort_flag = 1;
          } else if (real) {
            for (int r2 = 0; r2 < P.T; ++r2) {
              if (h0 + r2 >= P.H) break;
              const int32_t y = (n * P.H + h0 + r2) * P.W;
#pragma unroll
              for (int g = 0; g < 4; ++g) {
                const int x0 = g * 16;
                if (x0 < P.cout)
                  tma_reduce_add_2d(&mapY, stg + static_cast<uint32_t>(g * STG_G + r2 * P.wpad * 128), x0, y);
              }
            }
            bulk_commit();
          }
          bulk_wait_read_all();
          mbar_arrive(stg_free);
        }
        ++unit;
      }
    }
    if (reducer) bulk_wait_all();
  }

  // Pair handshake: neither CTA exits (or frees tensor memory) while its peer may still signal it.
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    mbar_arrive_cluster(map_to_rank(bye_bar, rank ^ 1u));
    if (!bounded_wait_cluster(bye_bar, 0, P.timeout_ns)) report_status(P.status, STATUS_TIMEOUT, 48);
  }
  __syncthreads();
  if (warp == B_WARP) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

}  // namespace

bool conv_rows_geometry(int64_t W, int64_t R, int64_t S, int chunk_scale, int* Wp, int* T, int* PB, int* wpad) {
  if (W < 1 || R < 1 || S < 1 || (R % 2) == 0 || (S % 2) == 0) return false;
  if (R * S * CIN > 512 * chunk_scale || R * S > MAX_TAPS) return false;  // one exact chunk per tile
  const int64_t wp = W + S - 1;
  if (wp > BM) return false;
  const int64_t wpd = (W + 7) / 8 * 8;
  int64_t t = BM / wp;
  if (t > STG_ROWS / wpd) t = STG_ROWS / wpd;
  if (t < 1) return false;
  const int64_t pb = (BM + (R - 1) * wp + (S - 1) + 7) / 8 * 8;
  if (pb > PB_MAX) return false;
  *Wp = static_cast<int>(wp);
  *T = static_cast<int>(t);
  *PB = static_cast<int>(pb);
  *wpad = static_cast<int>(wpd);
  return true;
}

cudaError_t conv_rows_i16(const ConvRowsArgs& a, cudaStream_t s, const char** why) {
  ConvParams P;
  if (!conv_rows_geometry(a.W, a.R, a.S, a.chunk_scale, &P.Wp, &P.T, &P.PB, &P.wpad) || a.cout < 1 ||
      a.cout % 2 != 0 || a.cout > BN || a.N * a.H * a.W >= (int64_t(1) << 31) || reinterpret_cast<uintptr_t>(a.X) % 16 != 0 ||
      reinterpret_cast<uintptr_t>(a.Y) % 16 != 0 || a.num_sms < 2) {
    *why = "direct convolution: unsupported shape";
    return cudaErrorInvalidValue;
  }
  const int64_t k = a.R * a.S * CIN;
  CUtensorMap mapBH, mapBL, mapY;
  if (!encode_tensor_map_2d(&mapBH, 1, a.b.plane[0], static_cast<uint64_t>(k), static_cast<uint64_t>(a.b.rows),
                            static_cast<uint64_t>(a.b.pitch) * 2, CIN, BN, 128, why) ||
      !encode_tensor_map_2d(&mapBL, 1, a.b.plane[1], static_cast<uint64_t>(k), static_cast<uint64_t>(a.b.rows),
                            static_cast<uint64_t>(a.b.pitch) * 2, CIN, BN, 128, why) ||
      !encode_tensor_map_2d(&mapY, 3, a.Y, static_cast<uint64_t>(a.cout), static_cast<uint64_t>(a.N * a.H * a.W),
                            static_cast<uint64_t>(a.cout) * 8, 16, static_cast<uint32_t>(a.W), 128, why))
    return cudaErrorInvalidValue;
  P.X = a.X;
  P.H = static_cast<int>(a.H);
  P.W = static_cast<int>(a.W);
  P.R = static_cast<int>(a.R);
  P.S = static_cast<int>(a.S);
  P.ph = static_cast<int>((a.R - 1) / 2);
  P.pw = static_cast<int>((a.S - 1) / 2);
  P.tiles_per_image = static_cast<int>((a.H + P.T - 1) / P.T);
  P.num_tiles = static_cast<int>(a.N * P.tiles_per_image);
  P.num_pair_tiles = (P.num_tiles + 1) / 2;
  P.cout = static_cast<int>(a.cout);
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t e = cudaFuncSetAttribute(conv_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(SMEM));
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  const int max_pairs = a.num_sms / 2;
  const int npairs = P.num_pair_tiles < max_pairs ? P.num_pair_tiles : max_pairs;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * static_cast<unsigned>(npairs), 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  *why = "direct convolution launch";
  return cudaLaunchKernelEx(&cfg, conv_rows_kernel, mapBH, mapBL, mapY, P);
}

}  // namespace gemmi
