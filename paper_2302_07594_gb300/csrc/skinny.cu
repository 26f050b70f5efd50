// skinny.cu -- exact int16 GEMM C (int64) += A*B for a small number of rows m <= 16, and for
// small problems (up to 256 rows) as groups of 16 rows along the grid's z dimension: one launch,
// no separate operand split, where the tensor-core path pays two launches and their latency.
//
// With m <= 16 (a batch of a few samples through a fully-connected layer) the
// GEMM of Section 4.1 is bound by streaming B (k x n) once from HBM: every B
// element is used m times only.  The paper notes that DL GEMMs often have one
// large and two small dimensions (Section 2, IM2COL lowering).  This kernel is
// built around the stream of B:
//
//   * the CTA's slice of A is fetched by bulk copies (one per row) issued right after the first B
//     stage and split into limbs once, so B starts streaming at once (with plain loads issued
//     by the consumers, the first B stage waited about 3 us for them).  The limbs are stored in
//     the order of the mma fragments: per row and 16 reduction indices (8 index pairs p), lane
//     quad t holds [hi p=t, hi p=t+4, lo p=t, lo p=t+4] in one 16-byte word, so a lane takes
//     its A fragments of a k-step with one shared-memory load instead of four (8.62 against
//     8.73 us for 8 x 4096 x 4096, 7.58 against 7.82 us for 256^3);
//   * B is cut into column blocks of 512 (1 KB contiguous of every row, which
//     DRAM streams markedly better than 512-byte runs) and the reduction
//     dimension into ranges, one (column block, range) per CTA, about one CTA
//     per SM; a producer warp streams 32-row x 512-column stages of B (eight
//     2-D TMA boxes, 128-byte swizzle) into a ring of shared-memory stages: as many 32 KB
//     stages (3 or 4) as fit beside the A limbs, which are sized for the CTA's own reduction
//     range.  Under load a stage takes 2-3 us from request to landing, so the bytes in flight
//     per SM, not the arithmetic, set the pace; the CTA's slice of A (m <= 16 rows, at most
//     1024 reduction indices) is split into fp16 limbs once, into shared memory, when the CTA
//     starts, so the inner loop converts only B;
//   * sixteen consumer warps each own 32 columns of the block, two m16 tiles
//     (four warps per scheduler, so the latencies of one warp's dependent
//     ldmatrix / mma chains are covered by the others).  A warp first reads its whole
//     share of a stage (32 reduction indices x 32 columns) into registers, transposed with
//     ldmatrix (the "A" operand of C^T = B^T A^T), and releases the stage at once, so the
//     producer refills it while the warp computes (holding the stage through the arithmetic
//     stretched every refill by about half a microsecond).  For m <= 8 it then takes the two bytes of
//         u = b + 32768 = 256*H + L,  H = (b >> 8) + 128 and L = b & 255, both in [0,255],
//     as fp16 subnormals (bit pattern 0x00XX is the value XX * 2^-24, exactly), one mask for L
//     and a shift and a mask for H, and multiplies them on the tensor cores with mma.sync
//     m16n8k16 (fp16 in, fp32 accumulate) against the centred limbs of A (a = 256*h + l,
//     |h|, |l| <= 128, split once per CTA).  Since u = b + 32768, the sums over the CTA's
//     reduction range are sum(a*b) + 32768 * sum(a); the row sums of the CTA's slice of A,
//     formed once, take the second term back off where the partial sums go into C.  (The 16-row
//     instantiation splits B into its signed high and unsigned low byte as fp16 values 1024 + x
//     less 1024, two more operations per pair; it measured faster there, its A limbs being
//     non-centred: hi = a >> 8, lo = a & 255.)
//   * three fp32 accumulator sets HH, X, LL hold exact sums, in units of 2^-24, while every
//     partial sum stays within 2^24 units (a run of 256 reduction indices of products of at
//     most 255 * 128: 256 * 2 * 32640 = 16,711,680 < 2^24 for the cross terms), then are
//     scaled by 2^24, converted and drained into int64 registers as HH*2^16 + X*2^8 + LL;
//   * each warp adds its partial sums into C: 64-bit atomic adds (exact and order-independent
//     modulo 2^64) when the reduction range is split, a plain read-modify-write otherwise.
#include <cuda.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

constexpr int JB = 512;                 // columns of B per CTA (1 KB of every row: long DRAM runs)
constexpr int BOX_J = 64;               // columns per TMA box (128 bytes, the swizzle span)
constexpr int NBOX = JB / BOX_J;        // 8 boxes per stage
constexpr int KS = 32;                  // rows of B per stage (two 16-row mma steps)
constexpr int MIN_STAGES = 3;
constexpr int MAX_STAGES = 4;           // more stages in flight measured slower (burstier arrival)
constexpr int STAGE_BYTES = KS * JB * 2;         // 32 KB of B per stage
constexpr int A_ROWS = 16;
constexpr int KMAX_CTA = 1024;                   // reduction indices per CTA (bounds the A limbs in smem)
constexpr size_t SMEM_MAX = 227 * 1024;
constexpr int NCONS = 16;               // consumer warps
constexpr int MT = JB / (16 * NCONS);   // m16 tiles (of 16 columns) per consumer warp
static_assert(MT * 16 * NCONS == JB, "the consumer warps cover the column block");
constexpr int THREADS = (NCONS + 1) * 32;
constexpr int DRAIN_EVERY = 8;          // stages per drain: 8 x 32 = 256 reduction indices
constexpr uint32_t STATUS_TIMEOUT = 4;

struct SkParams {
  int64_t m, n, k;
  const int16_t* A;
  int64_t lda;
  int64_t* C;
  int64_t ldc;
  int64_t stages_per_cta;   // reduction range of one CTA, in stages
  int64_t total_stages;
  int atomic_out;
  int a_bulk;               // A's slices can be bulk-copied: 16-byte aligned rows, k % 8 == 0
  int stages;               // B stages in the ring, MIN_STAGES .. MAX_STAGES
  int a_stride;             // 32-bit words per interleaved A limb row (16 mod 32, at least 2 * pairs)
  uint64_t timeout_ns;
  uint32_t* status;
};

// Bulk copy global -> this CTA's shared memory, completion (bytes) counted on `bar`.  Both
// addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

// Dynamic shared memory: alignment slack, the B ring, the interleaved A limbs (16 rows of a_stride
// words), the raw A slice as it lands (16 rows of `pairs` words: two int16 per word), the barriers,
// the row sums of the A slice (16 int32).
constexpr size_t sk_smem(int stages, int a_stride, int pairs) {
  return 1024 + static_cast<size_t>(stages) * STAGE_BYTES + static_cast<size_t>(A_ROWS) * a_stride * 4 +
         static_cast<size_t>(A_ROWS) * pairs * 4 + 8 * (2 * stages + 1) + 4 * A_ROWS + 16;
}
static_assert(sk_smem(4, KMAX_CTA + 16, KMAX_CTA / 2) <= SMEM_MAX, "four stages fit beside the largest A slice");

// int16 pair -> fp16 subnormal pairs of the bytes of u = b + 32768: L = b & 255 and H = (b >> 8) + 128
// (the high byte with its sign bit flipped), each the value byte * 2^-24 exactly.
__device__ __forceinline__ void split_pair_u(uint32_t x, uint32_t& hi, uint32_t& lo) {
  lo = x & 0x00FF00FFu;
  hi = ((x >> 8) & 0x00FF00FFu) ^ 0x00800080u;
}

// int16 pair -> fp16 pairs of its high (signed) and low (unsigned) bytes, exactly (the 16-row
// instantiation's B split, and its A split).  0x64xx as fp16 is 1024 + xx, so each byte is
// recovered by one subtraction.
__device__ __forceinline__ void split_pair(uint32_t x, uint32_t& hi, uint32_t& lo) {
  const uint32_t lo_bits = (x & 0x00FF00FFu) | 0x64006400u;         // 1024 + lo
  const uint32_t hi_bits = ((x >> 8) & 0x00FF00FFu) ^ 0x64806480u;  // 1024 + (hi + 128)
  const __half2 l = __hsub2(*reinterpret_cast<const __half2*>(&lo_bits), __half2half2(__ushort_as_half(0x6400)));
  const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&hi_bits), __half2half2(__ushort_as_half(0x6480)));
  lo = *reinterpret_cast<const uint32_t*>(&l);
  hi = *reinterpret_cast<const uint32_t*>(&h);
}

// Not volatile: a register-only operation, which the compiler may then schedule among the limb
// splits (measured 8.70 against 8.75 us for 8 x 4096 x 4096).
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

__device__ __forceinline__ int32_t f2i(float f) {
  int32_t v;
  asm("cvt.rni.s32.f32 %0, %1;" : "=r"(v) : "f"(f));
  return v;
}

// 17 warps: one of the four schedulers hosts five of them, and its quarter of the register file
// (16,384) caps every thread at 96 registers.
template <int NT>
__global__ void __launch_bounds__(THREADS, 1)
skinny_kernel(const __grid_constant__ CUtensorMap mapB, SkParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int stages = P.stages;
  const int a_stride = P.a_stride;
  const int cta_pairs = static_cast<int>(P.stages_per_cta * (KS / 2));  // index pairs of a CTA's range
  uint32_t* a_limb = reinterpret_cast<uint32_t*>(smem + static_cast<size_t>(stages) * STAGE_BYTES);  // [16][a_stride]
  uint32_t* a_raw = a_limb + A_ROWS * a_stride;                                                      // [16][cta_pairs]
  uint64_t* bars = reinterpret_cast<uint64_t*>(a_raw + A_ROWS * cta_pairs);
  int32_t* row_sum = reinterpret_cast<int32_t*>(bars + 2 * stages + 1);  // [16]: the A slice's row sums
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * stages;
  const uint32_t abar = empty0 + 8 * stages;  // the CTA's A slice has landed

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int64_t j_base = static_cast<int64_t>(blockIdx.x) * JB;
  const int64_t st_begin = static_cast<int64_t>(blockIdx.y) * P.stages_per_cta;
  // grid z: groups of 16 rows of A and C (one group when m <= 16)
  const int64_t row0 = static_cast<int64_t>(blockIdx.z) * A_ROWS;
  const int64_t mrows = P.m - row0 < A_ROWS ? P.m - row0 : A_ROWS;
  const int16_t* Ag = P.A + row0 * P.lda;
  int64_t* Cg = P.C + row0 * P.ldc;
  int64_t st_end = st_begin + P.stages_per_cta;
  if (st_end > P.total_stages) st_end = P.total_stages;
  const int nst = st_end > st_begin ? static_cast<int>(st_end - st_begin) : 0;

  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, NCONS);
    }
    mbar_init(abar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();  // A, B and C may come from the previous kernel in the stream

  if (warp == NCONS) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&mapB);
      // rows 0..m-1 of A, reduction indices k0 .. k0 + kv, land in the raw area (row r at
      // r * cta_pairs words), from where the consumers split them.  They are needed with the
      // first B stage: for up to 8 rows they go out right behind it (9.08 against 9.47 us for
      // 8 x 4096 x 4096 with A first), for 16-row groups first (7.9 against 8.2 us for the 256^3
      // problem); behind the first ring of B stages the consumers waited for them (1.35 us longer).
      auto load_a = [&]() {
        const int64_t k0 = st_begin * KS;
        const int64_t kv = min(static_cast<int64_t>(nst) * KS, P.k - k0);
        const uint32_t row_bytes = static_cast<uint32_t>(kv * 2);
        const int rows = static_cast<int>(mrows);
        mbar_arrive_expect_tx(abar, static_cast<uint32_t>(rows) * row_bytes);
        for (int r = 0; r < rows; ++r)
          bulk_load(smem_u32(a_raw + r * cta_pairs), Ag + r * P.lda + k0, row_bytes, abar);
      };
      if (NT == 2 && P.a_bulk && nst > 0) load_a();
      int s = 0;
      uint32_t par = 0;
      int issued = 0;
      for (int i = 0; i < nst; ++i) {
        if (!bounded_wait(empty0 + 8 * s, par ^ 1u, P.timeout_ns)) {
          report_status(P.status, STATUS_TIMEOUT, 11);
          break;
        }
        const uint32_t fb = full0 + 8 * s;
        const uint32_t dst = smem_u32(smem + static_cast<size_t>(s) * STAGE_BYTES);
        const int32_t krow = static_cast<int32_t>((st_begin + i) * KS);
        mbar_arrive_expect_tx(fb, STAGE_BYTES);
#pragma unroll
        for (int b = 0; b < NBOX; ++b)
          tma_load_2d(dst + b * (KS * BOX_J * 2), &mapB, fb, static_cast<int32_t>(j_base + b * BOX_J), krow);
        ++issued;
        if (NT == 1 && i == 0 && P.a_bulk) load_a();
        if (++s == stages) {
          s = 0;
          par ^= 1u;
        }
      }
      // wait for the copies in flight before the CTA may exit
      const int first = issued > stages ? issued - stages : 0;
      for (int i = first; i < issued; ++i)
        bounded_wait(full0 + 8 * (i % stages), static_cast<uint32_t>((i / stages) & 1), P.timeout_ns);
    }
    return;
  }

  // ------------------------------------------------------------ consumers
  // A consumer warp that gives up a wait records it and skips the rest of its stages, but still
  // reaches every named barrier of the other consumer warps (whose own waits are bounded too).
  bool ok = true;
  // Split this CTA's slice of A once: rows 0..15 (zero beyond m), reduction indices
  // k0 .. k0 + KS*nst (zero beyond k), as packed fp16 pairs of the high and low limbs, stored
  // in fragment order: index pair kp of a row goes to k-step kp / 8, lane quad kp % 4, high limb
  // at word (kp / 4) % 2 and low limb two words further.
  auto store_limbs = [&](int row, int kp, uint32_t x) {
    uint32_t hi, lo;
    if constexpr (NT == 1) tc::limbs16x2(x, hi, lo);  // centred limbs: |h|, |l| <= 128
    else split_pair(x, hi, lo);
    const int w = row * a_stride + (kp >> 3) * 16 + (kp & 3) * 4 + ((kp >> 2) & 1);
    a_limb[w] = hi;
    a_limb[w + 2] = lo;
  };
  if (P.a_bulk) {
    bool landed = true;
    if (nst > 0) {
      landed = __all_sync(0xFFFFFFFFu, bounded_wait(abar, 0, P.timeout_ns));
      if (!landed && lane == 0) report_status(P.status, STATUS_TIMEOUT, 13);
    }
    const int64_t k0 = st_begin * KS;
    const int64_t kv = nst > 0 ? min(static_cast<int64_t>(nst) * KS, P.k - k0) : 0;
    const int pairs = landed ? nst * KS / 2 : 0;
    for (int idx = threadIdx.x; idx < A_ROWS * pairs; idx += NCONS * 32) {
      const int row = idx / pairs;
      const int kp = idx - row * pairs;
      store_limbs(row, kp, (row < mrows && 2 * kp < kv) ? a_raw[row * cta_pairs + kp] : 0u);
    }
    if constexpr (NT == 1) {
      // warp w sums row w of the slice (two int16 per word): the correction of B's offset
      int32_t rs = 0;
      if (warp < mrows)
        for (int kp = lane; kp < pairs && 2 * kp < kv; kp += 32) {
          const uint32_t x = a_raw[warp * cta_pairs + kp];
          rs += static_cast<int32_t>(static_cast<int16_t>(x & 0xFFFFu)) +
                static_cast<int32_t>(static_cast<int16_t>(x >> 16));
        }
      for (int o = 16; o > 0; o >>= 1) rs += __shfl_xor_sync(0xFFFFFFFFu, rs, o);
      if (lane == 0 && warp < A_ROWS) row_sum[warp] = rs;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(NCONS * 32) : "memory");  // every consumer warp arrives
    ok = landed;
  } else {
    const int64_t k0 = st_begin * KS;
    const int pairs = nst * KS / 2;
    for (int idx = threadIdx.x; idx < A_ROWS * pairs; idx += NCONS * 32) {
      const int row = idx / pairs;
      const int kp = idx - row * pairs;
      const int64_t k = k0 + 2 * kp;
      uint32_t x = 0;
      if (row < mrows) {
        const int16_t* src = Ag + row * P.lda + k;
        const uint32_t v0 = k < P.k ? static_cast<uint16_t>(src[0]) : 0u;
        const uint32_t v1 = k + 1 < P.k ? static_cast<uint16_t>(src[1]) : 0u;
        x = v0 | (v1 << 16);
      }
      store_limbs(row, kp, x);
    }
    if constexpr (NT == 1) {
      // warp w sums row w of the slice: the correction of B's offset
      int32_t rs = 0;
      if (warp < mrows) {
        const int64_t kend = min(k0 + static_cast<int64_t>(nst) * KS, P.k);
        for (int64_t k = k0 + lane; k < kend; k += 32) rs += Ag[warp * P.lda + k];
      }
      for (int o = 16; o > 0; o >>= 1) rs += __shfl_xor_sync(0xFFFFFFFFu, rs, o);
      if (lane == 0 && warp < A_ROWS) row_sum[warp] = rs;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(NCONS * 32) : "memory");  // consumer warps only
  }
  const int g = lane >> 2;
  const int t = lane & 3;
  float hh[MT][NT][4], xx[MT][NT][4], ll[MT][NT][4];
  uint64_t acc[MT][NT][4];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        hh[mt][nt][c] = xx[mt][nt][c] = ll[mt][nt][c] = 0.f;
        acc[mt][nt][c] = 0;
      }
  // this warp's 16*MT columns start in box (warp*16*MT)/64, at 16-byte chunk ((warp*16*MT)%64)/8
  // of each 128-byte row (two chunks per m16 tile)
  const int box = (warp * 16 * MT) / BOX_J;
  const int chunk_base = ((warp * 16 * MT) % BOX_J) / 8;
  // ldmatrix lanes: 0-7 rows 0-7 / cols 0-7, 8-15 rows 0-7 / cols 8-15, 16-23 rows 8-15 / cols 0-7,
  // 24-31 rows 8-15 / cols 8-15 of a 16x16 (reduction x column) slab
  const int lrow = (lane & 7) + ((lane >> 4) << 3);
  const int lchunk = (lane >> 3) & 1;
  // 128-byte swizzle: 16-byte chunk c of row r is stored at chunk c ^ (r & 7); the rows a lane
  // addresses differ by multiples of 16, so its swizzled offset inside a row never changes
  uint32_t lane_off[MT];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
    lane_off[mt] = box * (KS * BOX_J * 2) + lrow * 128 + (((chunk_base + mt * 2 + lchunk) ^ (lrow & 7)) << 4);
  // this lane's A fragments: row g (+ 8 nt), lane quad t, of each k-step
  const uint32_t a_lane = smem_u32(a_limb) + static_cast<uint32_t>((g * a_stride + t * 4) * 4);
  int s = 0;
  uint32_t par = 0;
  // this warp's share of a stage (32 reduction indices x 16*MT columns) in registers
  auto load_stage = [&](uint32_t (&dst)[KS / 16][MT][4], int st) {
    const uint32_t sbase = smem_u32(smem + static_cast<size_t>(st) * STAGE_BYTES);
#pragma unroll
    for (int ks = 0; ks < KS / 16; ++ks)
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) ldsm_x4_trans(sbase + ks * (16 * 128) + lane_off[mt], dst[ks][mt]);
  };
  auto compute_half = [&](const uint32_t (&bk)[MT][4], int i, int ks) {
    // A fragments (the mma's B operand: 16 reduction indices x 8 rows of A), already split:
    // index pairs t and t + 4 of k-step 2i + ks, high and low limb, in one 16-byte load
    uint32_t ahi[NT][2], alo[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const uint4 v = lds128(a_lane + static_cast<uint32_t>((nt * 8 * a_stride + (i * 2 + ks) * 16) * 4));
      ahi[nt][0] = v.x;
      ahi[nt][1] = v.y;
      alo[nt][0] = v.z;
      alo[nt][1] = v.w;
    }
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      uint32_t bhi[4], blo[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if constexpr (NT == 1) split_pair_u(bk[mt][q], bhi[q], blo[q]);
        else split_pair(bk[mt][q], bhi[q], blo[q]);
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        mma16816(hh[mt][nt], bhi, ahi[nt][0], ahi[nt][1]);
        mma16816(xx[mt][nt], bhi, alo[nt][0], alo[nt][1]);
        mma16816(xx[mt][nt], blo, ahi[nt][0], ahi[nt][1]);
        mma16816(ll[mt][nt], blo, alo[nt][0], alo[nt][1]);
      }
    }
  };
  uint32_t b[KS / 16][MT][4];
  for (int i = 0; ok && i < nst; ++i) {
    const bool got = bounded_wait(full0 + 8 * s, par, P.timeout_ns);
    if (!__all_sync(0xFFFFFFFFu, got)) {
      if (lane == 0) report_status(P.status, STATUS_TIMEOUT, 12);
      ok = false;
      break;
    }
    if constexpr (NT == 1) {
      load_stage(b, s);
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * s);  // the producer may refill it while this warp computes
      compute_half(b[0], i, 0);
      compute_half(b[1], i, 1);
    } else {
      // two groups of 8 rows hold twice the accumulators: a whole stage's fragments at once would
      // spill, so each half stage is loaded just before its products and the stage is handed back
      // after both (loading both first measured 7.8 -> 8.7 us for the 256^3 problem)
      const uint32_t sbase = smem_u32(smem + static_cast<size_t>(s) * STAGE_BYTES);
#pragma unroll
      for (int ks = 0; ks < KS / 16; ++ks) {
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) ldsm_x4_trans(sbase + ks * (16 * 128) + lane_off[mt], b[ks][mt]);
        compute_half(b[ks], i, ks);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * s);
    }
    if (++s == stages) {
      s = 0;
      par ^= 1u;
    }
    if ((i + 1) % DRAIN_EVERY == 0 || i + 1 == nst) {
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            // m <= 8: the sums are in units of 2^-24 (the subnormal bytes of B); scaling is exact
            constexpr float unit = NT == 1 ? 16777216.0f : 1.0f;
            acc[mt][nt][c] += (static_cast<uint64_t>(static_cast<int64_t>(f2i(hh[mt][nt][c] * unit))) << 16) +
                              (static_cast<uint64_t>(static_cast<int64_t>(f2i(xx[mt][nt][c] * unit))) << 8) +
                              static_cast<uint64_t>(static_cast<int64_t>(f2i(ll[mt][nt][c] * unit)));
            hh[mt][nt][c] = xx[mt][nt][c] = ll[mt][nt][c] = 0.f;
          }
    }
  }
  if (nst == 0) return;  // the same for every warp of the CTA
  // C fragment (m16n8): c0 (row g, col 2t), c1 (g, 2t+1), c2 (g+8, 2t), c3 (g+8, 2t+1);
  // the mma's rows are columns j of C, its columns are rows i of C.
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int64_t i = nt * 8 + 2 * t + (c & 1);
        const int64_t j = j_base + warp * (16 * MT) + mt * 16 + g + 8 * (c >> 1);
        if (i < mrows && j < P.n) {
          unsigned long long* dst = reinterpret_cast<unsigned long long*>(Cg + i * P.ldc + j);
          // m <= 8: B entered as u = b + 32768, so 32768 times the row's sum of A comes back off
          unsigned long long v = static_cast<unsigned long long>(acc[mt][nt][c]);
          if constexpr (NT == 1) v -= static_cast<unsigned long long>(static_cast<int64_t>(row_sum[i])) << 15;
          if (P.atomic_out) atomicAdd(dst, v);
          else *dst = *dst + v;
        }
      }
}

template <int NT>
cudaError_t launch(const SkinnyArgs& a, cudaStream_t s, const char** why) {
  CUtensorMap mapB;
  if (!encode_tensor_map_2d(&mapB, 0, a.B, static_cast<uint64_t>(a.n), static_cast<uint64_t>(a.k),
                            static_cast<uint64_t>(a.ldb) * 2, BOX_J, KS, 128, why))
    return cudaErrorInvalidValue;
  const int64_t nj = (a.n + JB - 1) / JB;
  const int64_t total_stages = (a.k + KS - 1) / KS;
  int64_t ksplit = a.ksplit;
  const int64_t groups = (a.m + A_ROWS - 1) / A_ROWS;
  if (ksplit <= 0) {
    // about one CTA per SM: the reduction range is split across the CTAs of a column block, down
    // to a single stage per CTA (below) when the problem is small.  A floor of four stages per CTA
    // measured slower on every small shape tried: 7.6 against 4.9 us for 256^3, 8.6 against 6.5 us
    // for 16 x 2048 x 1024; latency, not the ring, bounds such calls
    ksplit = a.num_sms / (nj * groups);
    if (ksplit < 1) ksplit = 1;
  }
  // at most KMAX_CTA reduction indices per CTA: its A limbs must fit in shared memory
  const int64_t min_split = (total_stages + (KMAX_CTA / KS) - 1) / (KMAX_CTA / KS);
  if (ksplit < min_split) ksplit = min_split;
  if (ksplit > total_stages) ksplit = total_stages;
  if (ksplit < 1) ksplit = 1;
  const int64_t per = (total_stages + ksplit - 1) / ksplit;
  ksplit = (total_stages + per - 1) / per;
  if (nj > 0x7FFFFFFF || ksplit > 65535 || groups > 65535) {
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
  P.a_bulk = reinterpret_cast<uintptr_t>(a.A) % 16 == 0 && (a.lda * 2) % 16 == 0 && a.k % 8 == 0;
  P.timeout_ns = a.timeout_ns;
  P.status = a.status;
  // the A limbs hold the CTA's reduction range (pairs of indices, two limb words each); a row
  // stride of 16 words modulo 32 puts the two rows that a quarter warp's 16-byte fragment loads
  // touch in different halves of the banks.  The rest of the shared memory goes to B stages.
  const int64_t pairs = per * KS / 2;
  P.a_stride = static_cast<int>((2 * pairs + 15) / 32 * 32 + 16);
  P.stages = MAX_STAGES;
  while (P.stages > MIN_STAGES && sk_smem(P.stages, P.a_stride, static_cast<int>(pairs)) > SMEM_MAX) --P.stages;
  const size_t smem = sk_smem(P.stages, P.a_stride, static_cast<int>(pairs));
  if (smem > SMEM_MAX) {
    *why = "skinny GEMM shared-memory layout does not fit";
    return cudaErrorInvalidValue;
  }
  // the shared-memory opt-in (the largest layout) is set once per device for this kernel
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t attr = cudaFuncSetAttribute(skinny_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  static_cast<int>(SMEM_MAX));
    if (attr != cudaSuccess) return attr;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  // programmatic stream serialization: the kernel may be scheduled while the previous kernel in
  // the stream drains; it waits (griddepcontrol.wait) before its first global memory access
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(nj), static_cast<unsigned>(ksplit), static_cast<unsigned>(groups));
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, skinny_kernel<NT>, mapB, P);
}

}  // namespace

cudaError_t skinny_gemm_i16(const SkinnyArgs& args, cudaStream_t s, const char** why) {
  return args.m <= 8 ? launch<1>(args, s, why) : launch<2>(args, s, why);
}

}  // namespace gemmi
