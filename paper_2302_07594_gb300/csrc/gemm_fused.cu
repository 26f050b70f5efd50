// gemm_fused.cu -- int16 GEMM for narrow outputs (n <= 64) that converts A inside the kernel.
//
// Convolutions lowered with IM2COL/IM2ROW give GEMMs with one very large and
// two small dimensions (Section 2 of the paper): m = batch*H*W rows of
// activations, n = output channels, k = C_in*3*3.  Such a GEMM is bound by
// reading A once and C twice from HBM.  A separate limb-split pass (split.cu)
// would read A, write its two fp16 limb planes (twice A's bytes) and read them
// again; here A is streamed raw (int16) and split on chip, the way the paper
// packs the activation operand at run time while the weights stay packed
// (Section 5.1).  C is never loaded into the SM: each tile's A*B is added into
// C by bulk reductions that L2 carries out.
//
// Roles (one CTA per SM, 128 x 64 output tiles, K blocks of 64):
//   warp 8      TMA producer of raw A tiles (128 rows x 64 reduction indices of
//               int16, 128-byte swizzle) into a ring of RAW_STAGES slots.  A slot
//               is free again as soon as the converters have read it, so the HBM
//               stream never waits for the tensor cores; the ring is deep
//               because nothing else of A lives in shared memory.
//   warp 9      TMA producer of B's two limb tiles (64 x 64 fp16 each, stacked
//               into one 128-row tile) into a ring of B_STAGES slots.
//   warps 10-11 MMA issuers.  Issuer p multiplies A limb p (0 high, 1 low),
//               which sits in tensor memory, by the stacked B tile with one
//               tcgen05.mma of N = 128: columns 0-63 of its accumulator get
//               A_p * B_high, columns 64-127 get A_p * B_low.
//   warps 12-19 converters, two warpgroups.  Thread (warp 12 + 4h + j, lane t)
//               splits half h (32 reduction indices) of row 32j + t of each raw
//               tile into the two fp16 limbs and stores them in its TMEM lane of
//               the A limb stage (tcgen05.st).  A warp's chain of shared-memory
//               loads, byte logic and TMEM stores is latency-bound, so two warps
//               per scheduler convert each K block.
//   warps 0-7   epilogue.  Warp (quadrant q = w % 4, half h = w / 4), lane t,
//               drains row 32q + t, output columns 32h .. 32h + 31, of the
//               accumulators (staggered exact chunks) into int64 registers.  At
//               the end of a tile the two warps of a quadrant write their 32 rows
//               into a dense staging block that goes out as one bulk reduction
//               (cp.reduce.async.bulk .add.u64) when C's rows are 64 wide and
//               contiguous, or as one reduction per row otherwise.
//
// Limb split of a packed int16 pair x = (a1 << 16) | a0 with centred limbs
// h = floor((a + 128) / 256), l = a - 256 h, done on both halves at once:
//   l + 128 = lo_byte ^ 0x80,   h + 128 = (hi_byte ^ 0x80) + (lo_byte >> 7),
// each placed under the fp16 exponent of 1024 (bits 0x6400) and recovered
// exactly by one fp16 subtraction of 1152.  Every limb product is at most 2^14
// in magnitude, so a chunk of 512 * CS reduction indices sums exactly in fp32.
//
// TMEM (512 columns): two A limb stages of 64 columns (high limb 0-31, low
// 32-63; K packed two fp16 per column) and three 128-column accumulator slots
// (two live, one spare).  Registers: 640 threads are launched with 96 each;
// the warpgroups then re-split them with setmaxnreg (epilogue 136, producers
// and issuers 56, converters 72), within the launch allocation, which the host
// checks against the compiled kernel before every launch.  Every mbarrier wait
// is bounded; a wait that runs out records GEMMI_ETIMEOUT.
//
// Implicit IM2COL (FusedArgs::conv): for a "same" stride-1 convolution with
// Cin % 64 == 0, K block kb is filter tap (r, s) of 64 channels, and its A tile
// is the box of 128 input pixels starting (r - pad_h) * W + (s - pad_w) pixels
// from the tile's first output pixel; the converters zero the taps that fall
// outside the image.
#include <cuda.h>
#include <cuda_fp16.h>

#include <type_traits>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

using namespace tc;

constexpr int BN = 64;                        // output tile width
constexpr int UMMA_N = 2 * BN;                // B's two limbs stacked
constexpr int NUM_EPI_WARPS = 8;
constexpr int A_PRODUCER_WARP = 8;
constexpr int B_PRODUCER_WARP = 9;
constexpr int MMA_WARP0 = 10;
constexpr int NISSUE = 2;
constexpr int CONV_WARP0 = 12;                // converter warpgroups: warp 12 + 4h + j serves TMEM lanes 32j .. 32j + 31
constexpr int NUM_CONV_WARPS = 8;            // two warpgroups: warp 12 + 4h + j converts K-block half h of quadrant j
// per-role register budgets (setmaxnreg), per thread: epilogue, producers and issuers, converters
constexpr int EPI_REGS = 136, CTRL_REGS = 56, CONV_REGS = 72;

constexpr int NUM_THREADS = (CONV_WARP0 + NUM_CONV_WARPS) * 32;
static_assert(CONV_WARP0 % 4 == 0, "a warp reaches the TMEM lane quadrant of its warp index modulo 4");
static_assert((2 * EPI_REGS + CTRL_REGS + 2 * CONV_REGS) * 128 <= NUM_THREADS * 96,
              "the split must fit what 640 threads are launched with (96 registers each)");
static_assert((2 * EPI_REGS + CTRL_REGS + 2 * CONV_REGS) * 32 <= 16384,
              "each scheduler holds one warp of every warpgroup: its quarter of the register file");
constexpr int NACC = 2;                       // accumulator p: A limb p times both B limbs
constexpr int NSLOT = 3;
constexpr int SLOT_COLS = UMMA_N;             // 128
constexpr int A_STAGES = 2;                   // A limb stages in TMEM
constexpr int A_STAGE_COLS = BK;              // 2 limbs x 64 fp16 / 2 per column
constexpr int ACC_COL0 = A_STAGES * A_STAGE_COLS;
constexpr int TMEM_COLS = 512;
static_assert(ACC_COL0 + NSLOT * SLOT_COLS <= TMEM_COLS, "tensor memory budget");
constexpr int TILE_RAW = BM * BK * 2;         // 16 KB: a raw int16 A tile
constexpr int TILE_B = UMMA_N * BK * 2;       // 16 KB: the stacked B limb tiles
constexpr int RAW_STAGES = 7;
constexpr int B_STAGES = 3;
constexpr int COLS = 32;                      // C columns per epilogue thread
constexpr int STG_ROW = BN * 8;               // staging: dense int64 rows of the C tile
constexpr int STG_QUAD = 32 * STG_ROW;        // the 32 rows of one TMEM lane quadrant (16 KB)
constexpr int OFF_B = RAW_STAGES * TILE_RAW;
constexpr int OFF_STG = OFF_B + B_STAGES * TILE_B;
constexpr int OFF_BAR = OFF_STG + 4 * STG_QUAD;
constexpr int NBAR = 2 * RAW_STAGES + 2 * A_STAGES + 2 * B_STAGES + 2 * NSLOT + 1 + 2 * 4;
constexpr size_t SMEM = 1024 + static_cast<size_t>(OFF_BAR) + 8 * NBAR + 16;
static_assert(SMEM <= 227 * 1024, "shared memory budget");
static_assert(OFF_B % 1024 == 0 && OFF_STG % 1024 == 0, "swizzled tiles start on 1024-byte boundaries");

// The two accumulators' exact chunks: at most 512 * CS reduction indices, staggered by half a
// chunk so that their drains alternate.  When a whole tile fits in one chunk (k <= 512 * CS) there
// is no chunk end inside a tile: both accumulators are drained once, where the tile (or this CTA's
// part of it) ends.
template <int CS>
__device__ __forceinline__ bool chunk_ends(int a, int kb, int nkb) {
  if (nkb * BK <= 512 * CS) return kb == nkb - 1;
  return kb == nkb - 1 || (((kb + 1) * BK + a * 256 * CS) % (512 * CS)) == 0;
}
// weights of accumulator a's two column halves: A limb a times B limb 0 (high) and 1 (low)
__device__ __forceinline__ int shift_left_half(int a) { return a == 0 ? 16 : 8; }
__device__ __forceinline__ int shift_right_half(int a) { return a == 0 ? 8 : 0; }

struct FusedParams {
  int64_t m, n, k;
  int64_t* C;
  int64_t ldc;
  int num_m_tiles, num_n_tiles, num_k_blocks;
  int c_bulk;   // C base 16-byte aligned and ldc even: the tile goes out as bulk reductions
  int c_dense;  // also n == ldc == 64: the 32 rows of a lane quadrant are one 16 KB block of C
  int group_m;
  uint64_t timeout_ns;
  uint32_t* status;
  // implicit IM2COL (see FusedArgs): image height and width, filter width, paddings, channel blocks
  int conv, conv_h, conv_w, conv_s, conv_ph, conv_pw, conv_cb;
};

// The filter tap (r, s) and channel block cb of K block kb of an implicit-IM2COL GEMM, advanced
// one K block at a time (the division happens once, where a CTA's part of a tile starts).
struct TapPos {
  int cb, s, r;
  __device__ __forceinline__ void set(int kb, const FusedParams& P) {
    const int tap = kb / P.conv_cb;
    cb = kb - tap * P.conv_cb;
    r = tap / P.conv_s;
    s = tap - r * P.conv_s;
  }
  __device__ __forceinline__ void advance(const FusedParams& P) {
    if (++cb == P.conv_cb) {
      cb = 0;
      if (++s == P.conv_s) {
        s = 0;
        ++r;
      }
    }
  }
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

// Writes this thread's 32 accumulated values (one C row segment) into its row of the dense
// staging block.  Row segments of consecutive lanes are 512 bytes apart, so storing the same
// 16-byte chunk on every lane would hit one bank group eight times per quarter warp; instead
// step c stores chunk c ^ (lane % 8), and the values are first permuted to match by three
// conditional swaps of register pairs (static indexing keeps them in registers).
__device__ __forceinline__ void stage_row(uint32_t row_addr, uint64_t (&acc)[COLS], uint32_t lane) {
  const uint32_t x = lane & 7u;
#pragma unroll
  for (int b = 0; b < 3; ++b) {
    const bool sw = (x >> b) & 1u;
#pragma unroll
    for (int j = 0; j < COLS / 2; ++j) {
      if (j & (1 << b)) continue;
      const int j2 = j | (1 << b);
      const uint64_t a0 = acc[2 * j], a1 = acc[2 * j + 1], b0 = acc[2 * j2], b1 = acc[2 * j2 + 1];
      acc[2 * j] = sw ? b0 : a0;
      acc[2 * j + 1] = sw ? b1 : a1;
      acc[2 * j2] = sw ? a0 : b0;
      acc[2 * j2 + 1] = sw ? a1 : b1;
    }
  }
#pragma unroll
  for (int c = 0; c < COLS / 2; ++c) {
    uint4 v;
    v.x = static_cast<uint32_t>(acc[2 * c]);
    v.y = static_cast<uint32_t>(acc[2 * c] >> 32);
    v.z = static_cast<uint32_t>(acc[2 * c + 1]);
    v.w = static_cast<uint32_t>(acc[2 * c + 1] >> 32);
    sts128(row_addr + ((static_cast<uint32_t>(c) ^ x) << 4), v);
  }
}

// Adds `count` staged columns of one row into C: the even part as one bulk reduction, an odd
// last column by an atomic add read back from the staging row.
__device__ __forceinline__ void reduce_row(int64_t* dst, uint32_t stage_row, int count) {
  const int even = count & ~1;
  if (even > 0) bulk_reduce_add_u64(dst, stage_row, static_cast<uint32_t>(even * 8));
  if (count & 1) {
    unsigned long long last;
    asm volatile("ld.shared.u64 %0, [%1];" : "=l"(last) : "r"(stage_row + (count - 1) * 8));
    atomicAdd(reinterpret_cast<unsigned long long*>(dst + count - 1), last);
  }
}

// This CTA's share of the work: the K-block units (tile t, K block kb), numbered t * nkb + kb with
// the tiles in raster order, split into gridDim.x contiguous ranges of equal length (within one).
// A tile whose K blocks straddle two ranges is computed in two parts that are both added into C,
// which the bulk reductions do anyway; so every CTA finishes at the same time however the tile
// count divides by the SM count.
struct Span {
  int64_t u, first, end;  // current unit, this CTA's first unit, one past its last
  int t, kb, nkb;         // current tile and K block
  __device__ __forceinline__ void init(int64_t total_units, int nkb_) {
    nkb = nkb_;
    first = static_cast<int64_t>(blockIdx.x) * total_units / gridDim.x;
    end = (static_cast<int64_t>(blockIdx.x) + 1) * total_units / gridDim.x;
    u = first;
    t = static_cast<int>(u / nkb);
    kb = static_cast<int>(u - static_cast<int64_t>(t) * nkb);
  }
  __device__ __forceinline__ bool done() const { return u >= end; }
  __device__ __forceinline__ bool part_first() const { return kb == 0 || u == first; }
  __device__ __forceinline__ bool part_last() const { return kb == nkb - 1 || u + 1 == end; }
  __device__ __forceinline__ void next() {
    ++u;
    if (++kb == nkb) {
      kb = 0;
      ++t;
    }
  }
};

template <int CS>
__global__ void __launch_bounds__(NUM_THREADS, 1)
fused_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapBH,
             const __grid_constant__ CUtensorMap mapBL, FusedParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  const uint32_t raw_full0 = smem_u32(bars);                 // raw A tile landed
  const uint32_t raw_empty0 = raw_full0 + 8 * RAW_STAGES;    // raw A tile read by the 4 converter warps
  const uint32_t a_ready0 = raw_empty0 + 8 * RAW_STAGES;     // A limbs stored in TMEM by the 4 converter warps
  const uint32_t a_empty0 = a_ready0 + 8 * A_STAGES;         // both issuers' MMAs on the A limb stage completed
  const uint32_t b_full0 = a_empty0 + 8 * A_STAGES;          // B limb tiles landed
  const uint32_t b_empty0 = b_full0 + 8 * B_STAGES;          // both issuers' MMAs on the B limbs completed
  const uint32_t sfull0 = b_empty0 + 8 * B_STAGES;
  const uint32_t sempty0 = sfull0 + 8 * NSLOT;
  const uint32_t final_bar = sempty0 + 8 * NSLOT;
  const uint32_t stg_free0 = final_bar + 8;        // per quadrant: its staging block has been read
  const uint32_t stg_full0 = stg_free0 + 8 * 4;    // per quadrant: both warps have staged their rows
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < RAW_STAGES; ++s) {
      mbar_init(raw_full0 + 8 * s, 1);
      mbar_init(raw_empty0 + 8 * s, NUM_CONV_WARPS);
    }
    for (int s = 0; s < A_STAGES; ++s) {
      mbar_init(a_ready0 + 8 * s, NUM_CONV_WARPS);
      mbar_init(a_empty0 + 8 * s, NISSUE);
    }
    for (int s = 0; s < B_STAGES; ++s) {
      mbar_init(b_full0 + 8 * s, 1);
      mbar_init(b_empty0 + 8 * s, NISSUE);
    }
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(sfull0 + 8 * s, 1);
      mbar_init(sempty0 + 8 * s, NUM_EPI_WARPS);
    }
    mbar_init(final_bar, NISSUE);
    for (int qd = 0; qd < 4; ++qd) {
      mbar_init(stg_free0 + 8 * qd, 1);
      mbar_init(stg_full0 + 8 * qd, 2);
    }
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
  // Launched with programmatic stream serialization: the setup above may overlap the end of the
  // previous kernel (B's limb split, or the previous GEMM); every global access comes after this
  // wait.  The next kernel may be scheduled as this grid's CTAs retire.
  pdl_wait();
  pdl_launch_dependents();

  const int nkb = P.num_k_blocks;
  const int64_t total_units = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles * nkb;
  Span span;
  span.init(total_units, nkb);

  if (warp >= CONV_WARP0) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(CONV_REGS) : "memory");
    // ------------------------------------------------------------ converters: raw A -> limbs in TMEM
    // Thread (warp 12 + 4h + j, lane t) converts half h of row 32j + t of every raw tile: it loads
    // the half's four 16-byte chunks (128-byte swizzle: chunk c sits at c ^ (row % 8)), hands the
    // raw slot back at once, splits the 32 values into their two limbs and stores them in its TMEM
    // lane.
    const int quad = (warp - CONV_WARP0) & 3;
    const int khalf = (warp - CONV_WARP0) >> 2;  // reduction indices 32*khalf .. +31 of each K block
    const uint32_t row = static_cast<uint32_t>(quad * 32 + lane);
    const uint32_t lane_field = static_cast<uint32_t>(quad * 32) << 16;
    RingPos craw, cstage;
    bool ok = true;
    TapPos tap;
    int ho = 0, wo = 0;  // implicit IM2COL: this row's output pixel
    for (Span sp = span; !sp.done() && ok; sp.next()) {
      if (P.conv && sp.part_first()) {
        int mt, nt;
        tile_coords(sp.t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
        const int64_t m = static_cast<int64_t>(mt) * BM + row;
        const int64_t img_row = m / P.conv_w;
        wo = static_cast<int>(m - img_row * P.conv_w);
        ho = static_cast<int>(img_row % P.conv_h);
        tap.set(sp.kb, P);
      }
      const bool got = bounded_wait(raw_full0 + 8 * craw.slot, craw.phase, P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, got)) {
        if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 25);
        *abort_flag = 1;
        break;
      }
      const uint32_t src = smem_u32(smem + craw.slot * TILE_RAW) + row * 128;
      uint4 x[4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
        x[c] = lds128(src + ((static_cast<uint32_t>(4 * khalf + c) ^ (row & 7u)) << 4));
      __syncwarp();
      if (lane == 0) mbar_arrive(raw_empty0 + 8 * craw.slot);
      craw.advance(RAW_STAGES);
      if (P.conv) {
        // zero padding: the tap reads outside the image for this output pixel
        const int h = ho + tap.r - P.conv_ph, w = wo + tap.s - P.conv_pw;
        if (h < 0 || h >= P.conv_h || w < 0 || w >= P.conv_w) {
#pragma unroll
          for (int c = 0; c < 4; ++c) x[c] = make_uint4(0u, 0u, 0u, 0u);
        }
        tap.advance(P);
      }
      const bool free_stage = bounded_wait(a_empty0 + 8 * cstage.slot, cstage.phase ^ 1u, P.timeout_ns);
      if (!__all_sync(0xFFFFFFFFu, free_stage)) {
        if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 29);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t t = tmem_base + lane_field + static_cast<uint32_t>(cstage.slot * A_STAGE_COLS);
      {  // 32 reduction indices: one TMEM store of 16 columns per limb
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          split_centred(x[i].x, hi[4 * i + 0], lo[4 * i + 0]);
          split_centred(x[i].y, hi[4 * i + 1], lo[4 * i + 1]);
          split_centred(x[i].z, hi[4 * i + 2], lo[4 * i + 2]);
          split_centred(x[i].w, hi[4 * i + 3], lo[4 * i + 3]);
        }
        tc_st_32x32b_x16(t + khalf * 16, hi);
        tc_st_32x32b_x16(t + BK / 2 + khalf * 16, lo);
      }
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(a_ready0 + 8 * cstage.slot);
      cstage.advance(A_STAGES);
    }
    (void)ok;
  } else if (warp >= NUM_EPI_WARPS) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(CTRL_REGS) : "memory");
    if (warp == A_PRODUCER_WARP || warp == B_PRODUCER_WARP) {
    // ------------------------------------------------------------ TMA producers
    const bool is_a = warp == A_PRODUCER_WARP;
    const int nst = is_a ? RAW_STAGES : B_STAGES;
    const uint32_t full0 = is_a ? raw_full0 : b_full0;
    const uint32_t empty0 = is_a ? raw_empty0 : b_empty0;
    if (lane == 0) {
      if (is_a) {
        tma_prefetch_desc(&mapA);
      } else {
        tma_prefetch_desc(&mapBH);
        tma_prefetch_desc(&mapBL);
      }
      RingPos pos;
      int64_t issued = 0;
      bool stop = false;
      int mt = 0, nt = 0;
      TapPos tap;
      for (Span sp = span; !sp.done() && !stop; sp.next()) {
        const int kb = sp.kb;
        if (sp.part_first()) {
          tile_coords(sp.t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
          if (P.conv) tap.set(kb, P);
        }
        {
          if (!bounded_wait(empty0 + 8 * pos.slot, pos.phase ^ 1u, P.timeout_ns) || *abort_flag) {
            report_status(P.status, STATUS_TIMEOUT, is_a ? 21 : 22);
            *abort_flag = 1;
            stop = true;
            break;
          }
          const uint32_t fb = full0 + 8 * pos.slot;
          if (is_a) {
            // implicit IM2COL: the tap's 128 input pixels start (r - pad_h) rows and (s - pad_w)
            // columns away from the tile's first output pixel (pixels outside the tensor read as 0;
            // the converters zero those that fall outside the image)
            int32_t x = kb * BK, y = mt * BM;
            if (P.conv) {
              x = tap.cb * BK;
              y += (tap.r - P.conv_ph) * P.conv_w + (tap.s - P.conv_pw);
              tap.advance(P);
            }
            mbar_arrive_expect_tx(fb, TILE_RAW);
            tma_load_2d(smem_u32(smem + pos.slot * TILE_RAW), &mapA, fb, x, y);
          } else {
            const uint32_t base = smem_u32(smem + OFF_B + pos.slot * TILE_B);
            mbar_arrive_expect_tx(fb, TILE_B);
            tma_load_2d(base, &mapBH, fb, kb * BK, nt * BN);
            tma_load_2d(base + TILE_B / 2, &mapBL, fb, kb * BK, nt * BN);
          }
          pos.advance(nst);
          ++issued;
        }
      }
      // the copies still in flight: slots below pos.slot in this round, the others in the last one
      for (int x = 0; x < nst; ++x) {
        if (x < pos.slot)
          bounded_wait(full0 + 8 * x, pos.phase, P.timeout_ns);
        else if (issued >= nst)
          bounded_wait(full0 + 8 * x, pos.phase ^ 1u, P.timeout_ns);
      }
    }
    } else {
    // ------------------------------------------------------------ MMA issuers (issuer me owns accumulator me)
    // `me` is a compile-time constant in each issuer's copy of the loop: indexed at run time, the
    // slot ring's arrays lived in local memory, and every unit's few book-keeping steps waited on
    // it behind the converters' shared-memory traffic (about 0.25 us per unit, with the tensor
    // pipe idle meanwhile)
    auto issuer = [&](auto me_c) {
      constexpr int me = decltype(me_c)::value;
      constexpr uint32_t idesc = idesc_f16_f32(BM, UMMA_N);
      SlotRing<NACC, NSLOT> ring;
      ring.init();
      uint32_t wait_par = 1u;
      bool need_acquire = true, fresh = true;
      bool ok = true;
      RingPos pa, pb;
      for (Span sp = span; !sp.done() && ok; sp.next()) {
        const int kb = sp.kb;
        {
          if (!bounded_wait(a_ready0 + 8 * pa.slot, pa.phase, P.timeout_ns) ||
              !bounded_wait(b_full0 + 8 * pb.slot, pb.phase, P.timeout_ns)) {
            report_status(P.status, STATUS_TIMEOUT, 23);
            *abort_flag = 1;
            ok = false;
            break;
          }
          if (need_acquire) {
            if (!bounded_wait(sempty0 + 8 * ring.slot_of[me], wait_par, P.timeout_ns)) {
              report_status(P.status, STATUS_TIMEOUT, 24);
              *abort_flag = 1;
              ok = false;
              break;
            }
            need_acquire = false;
          }
          tc_fence_after();
          const uint32_t d = tmem_base + static_cast<uint32_t>(ACC_COL0 + ring.slot_of[me] * SLOT_COLS);
          const uint32_t a_tmem = tmem_base + static_cast<uint32_t>(pa.slot * A_STAGE_COLS + me * (BK / 2));
          const uint64_t bdesc = smem_desc_kmajor<128>(smem_u32(smem + OFF_B + pb.slot * TILE_B));
#pragma unroll
          for (int kk = 0; kk < BK / UMMA_K; ++kk)
            tc_mma_f16_ts(d, a_tmem + kk * (UMMA_K / 2), bdesc + 2 * kk, idesc, (fresh && kk == 0) ? 0u : 1u);
          fresh = false;
          tc_commit(a_empty0 + 8 * pa.slot);
          tc_commit(b_empty0 + 8 * pb.slot);
          pa.advance(A_STAGES);
          pb.advance(B_STAGES);
          const bool part_last = sp.part_last();
#pragma unroll
          for (int a = 0; a < NACC; ++a) {
            if (!part_last && !chunk_ends<CS>(a, kb, nkb)) continue;
            if (a == me) tc_commit(sfull0 + 8 * ring.slot_of[a]);
            const uint32_t par = ring.rotate(a);
            if (a == me) {
              wait_par = par;
              need_acquire = true;
              fresh = true;
            }
          }
        }
      }
      tc_commit(final_bar);
      bounded_wait(final_bar, 0, P.timeout_ns);
    };
    if (lane == 0) {
      if (warp == MMA_WARP0) issuer(std::integral_constant<int, 0>{});
      else issuer(std::integral_constant<int, 1>{});
    }
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(EPI_REGS) : "memory");
    // ------------------------------------------------------------ epilogue: drain, reduce into C
    const int quad = warp & 3;
    const int half = warp >> 2;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;  // TMEM lane field of this quadrant
    SlotRing<NACC, NSLOT> ring;
    ring.init();
    uint32_t drain_parity = 0;
    bool ok = true;
    uint64_t acc[COLS];
    const uint32_t quad_stage = smem_u32(smem + OFF_STG + quad * STG_QUAD);
    uint32_t tile_ends = 0;  // staged tile ends so far (the quadrant barriers' phase)

    int mt = 0, nt = 0;
    for (Span sp = span; !sp.done() && ok; sp.next()) {
      const int kb = sp.kb;
      const bool part_last = sp.part_last();
      if (sp.part_first()) {
        tile_coords(sp.t, P.num_m_tiles, P.num_n_tiles, P.group_m, mt, nt);
#pragma unroll
        for (int c = 0; c < COLS; ++c) acc[c] = 0;
      }
      {
#pragma unroll
        for (int a = 0; a < NACC; ++a) {
          if (!part_last && !chunk_ends<CS>(a, kb, nkb)) continue;
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
          const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(ACC_COL0 + s * SLOT_COLS + half * COLS);
          const int sl = shift_left_half(a), sr = shift_right_half(a);
#pragma unroll
          for (int g = 0; g < 2; ++g) {  // 16 output columns at a time: B high limb part, B low limb part
            uint32_t lv[16], rv[16];
            tc_ld_32x32b_x16(taddr + g * 16, lv);
            tc_ld_32x32b_x16(taddr + BN + g * 16, rv);
            tc_wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j)
              acc[16 * g + j] += (static_cast<uint64_t>(static_cast<int64_t>(f32_to_i32(lv[j]))) << sl) +
                                 (static_cast<uint64_t>(static_cast<int64_t>(f32_to_i32(rv[j]))) << sr);
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sempty0 + 8 * s);
          ring.rotate(a);
        }
      }
      if (!ok) break;
      if (!part_last) continue;
      // ---- C tile += acc (this CTA's part of the tile's K blocks), through the staging block and
      //      bulk reductions
      const int64_t row0 = static_cast<int64_t>(mt) * BM + quad * 32;
      const int64_t row = row0 + lane;
      const int64_t tcol0 = static_cast<int64_t>(nt) * BN;
      const int64_t left = P.n - tcol0;
      const int tile_cols = left >= BN ? BN : static_cast<int>(left);
      if (P.c_bulk) {
        const uint32_t par = tile_ends & 1u;
        if (half == 0) {  // this warp issues the quadrant's reductions: they must have read the block
          bulk_wait_read_all();
          __syncwarp();
          if (lane == 0) mbar_arrive(stg_free0 + 8 * quad);
        } else if (!__all_sync(0xFFFFFFFFu, bounded_wait(stg_free0 + 8 * quad, par, P.timeout_ns))) {
          if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 27);
          *abort_flag = 1;
          ok = false;
          break;
        }
        const uint32_t my_row = quad_stage + static_cast<uint32_t>(lane * STG_ROW + half * COLS * 8);
        stage_row(my_row, acc, lane);
        fence_proxy_async_smem();  // the bulk reductions read the block through the async proxy
        __syncwarp();
        if (lane == 0) mbar_arrive(stg_full0 + 8 * quad);
        if (half == 0) {
          if (!__all_sync(0xFFFFFFFFu, bounded_wait(stg_full0 + 8 * quad, par, P.timeout_ns))) {
            if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 28);
            *abort_flag = 1;
            ok = false;
            break;
          }
          if (P.c_dense) {
            const int64_t rows = P.m - row0 < 32 ? P.m - row0 : 32;
            if (lane == 0 && rows > 0) {
              bulk_reduce_add_u64(P.C + row0 * BN, quad_stage, static_cast<uint32_t>(rows * STG_ROW));
              bulk_commit();
            }
          } else if (row < P.m) {
            reduce_row(P.C + row * P.ldc + tcol0, quad_stage + static_cast<uint32_t>(lane * STG_ROW), tile_cols);
            bulk_commit();
          }
        }
        ++tile_ends;
      } else if (row < P.m) {
        int64_t* crow = P.C + row * P.ldc + tcol0 + half * COLS;
        const int valid = tile_cols - half * COLS;
#pragma unroll
        for (int c = 0; c < COLS; ++c)
          if (c < valid)
            atomicAdd(reinterpret_cast<unsigned long long*>(crow + c), static_cast<unsigned long long>(acc[c]));
      }
    }
    bulk_wait_all();
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
  // A: the lowered matrix, or for an implicit IM2COL the NHWC tensor as (pixels x channels)
  const uint64_t a_inner = a.conv ? static_cast<uint64_t>(a.conv_cin) : static_cast<uint64_t>(a.k);
  const uint64_t a_outer = a.conv ? static_cast<uint64_t>(a.conv_pixels) : static_cast<uint64_t>(a.m);
  const uint64_t a_row_bytes = a.conv ? static_cast<uint64_t>(a.conv_cin) * 2 : static_cast<uint64_t>(a.lda) * 2;
  if (!encode_tensor_map_2d(&mapA, 0, a.A, a_inner, a_outer, a_row_bytes, BK, BM, 128, why) ||
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
  P.c_bulk = (reinterpret_cast<uintptr_t>(a.C) % 16 == 0) && (a.ldc % 2 == 0);
  P.c_dense = P.c_bulk && a.n == BN && a.ldc == BN;
  P.group_m = a.group_m > 0 ? a.group_m : 16;
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  P.conv = a.conv;
  P.conv_h = a.conv_h;
  P.conv_w = a.conv_w;
  P.conv_s = a.conv_s;
  P.conv_ph = a.conv_ph;
  P.conv_pw = a.conv_pw;
  P.conv_cb = a.conv ? a.conv_cin / BK : 1;
  const int64_t units = static_cast<int64_t>(P.num_m_tiles) * P.num_n_tiles * P.num_k_blocks;
  const int grid = static_cast<int>(units < a.num_sms ? units : a.num_sms);
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t attr = cudaFuncSetAttribute(fused_kernel<CS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  static_cast<int>(SMEM));
    if (attr != cudaSuccess) return attr;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  // setmaxnreg.inc waits for registers the CTA was launched with: never launch a split that the
  // launch allocation cannot cover (it would wait forever)
  {
    cudaFuncAttributes fattr;
    const cudaError_t ae = cudaFuncGetAttributes(&fattr, fused_kernel<CS>);
    if (ae != cudaSuccess) return ae;
    constexpr int need = (2 * EPI_REGS + CTRL_REGS + 2 * CONV_REGS) * 128;
    if (fattr.numRegs * NUM_THREADS < need) {
      *why = "fused kernel: per-role register split exceeds the launch allocation";
      return cudaErrorInvalidConfiguration;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fused_kernel<CS>, mapA, mapBH, mapBL, P);
}

}  // namespace

cudaError_t tc_gemm_fused_i16(const FusedArgs& args, cudaStream_t s, const char** why) {
  return args.chunk_scale == 2 ? launch<2>(args, s, why) : launch<1>(args, s, why);
}

}  // namespace gemmi
