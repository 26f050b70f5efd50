// tc_common.cuh -- pieces shared by the tcgen05 GEMM kernels (gemm_tc.cu, gemm_fused.cu):
// the limb-product / accumulator schemes with their exact-chunk schedules, the TMEM slot ring,
// the tile raster and small device helpers.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

#include "ptx.cuh"

namespace gemmi {
namespace tc {

constexpr int BM = 128;                      // output tile rows (= TMEM lanes)
constexpr int BK = 64;                       // K block: 64 fp16 = 128 bytes = one swizzle row
constexpr int UMMA_K = 16;                   // K of one tcgen05.mma kind::f16
constexpr uint32_t STATUS_TIMEOUT = 4;

template <int NL>
struct Scheme;

// int16: two limbs per operand.  B's two limb tiles are stacked into one 256-row tile, so one
// tcgen05.mma of N = 256 multiplies an A limb by both B limbs: accumulator p (owned by issuer p)
// holds A_p * B_high in its columns 0-127 and A_p * B_low in columns 128-255 (limb 0 = high,
// 1 = low), weights 2^16 | 2^8 for p = 0 and 2^8 | 1 for p = 1.  Compared with four N = 128
// products this halves the MMA count and the times each A tile is read from shared memory.
// The two accumulators fill TMEM (two 256-column slots, no spare): at a chunk end the owning
// issuer waits for the drain of its slot, while the other issuer -- whose chunk ends half a
// chunk later -- keeps the tensor pipe busy.
template <>
struct Scheme<2> {
  static constexpr int BN = 128;          // output tile width
  static constexpr int UMMA_N = 256;      // B's two limbs stacked
  static constexpr int NACC = 2;
  static constexpr int NPROD = 2;         // product p: A limb p times the stacked B
  static constexpr int NSLOT = 2;
  static constexpr int SLOT_COLS = 256;
  static constexpr int EMPTY_COUNT = 2;   // both issuers read every stage
  static constexpr int COLS = 64;         // C columns per epilogue thread (two warps per lane quadrant)
  static constexpr int DRAIN_WARPS = 8;   // every epilogue warp drains every accumulator (its 64 columns)
  __device__ static constexpr bool drains(int, int) { return true; }
  __device__ static constexpr int a_limb(int p) { return p; }
  __device__ static constexpr int b_limb(int) { return 0; }  // the stacked B starts at the high limb
  __device__ static constexpr int b_row0(int) { return 0; }
  __device__ static constexpr int acc(int p, int) { return p; }
  __device__ static constexpr int issuer(int p, int) { return p; }
  __device__ static constexpr int owner(int a) { return a; }
  __device__ static constexpr int shift(int a) { return a == 0 ? 16 : 8; }       // columns 0-127
  __device__ static constexpr int shift_low(int a) { return a == 0 ? 8 : 0; }    // columns 128-255
  // Chunks of 512 * CS reduction indices, |sum| <= 512 * CS * 2^14 (within 2^23 for CS = 1,
  // 2^24 for CS = 2, the limit of exact fp32 integer sums); the two accumulators' chunk ends
  // are staggered by half a chunk.
  template <int CS>
  __device__ static bool chunk_ends(int a, int kb, int nkb) {
    return kb == nkb - 1 || (((kb + 1) * 64 + a * 256 * CS) % (512 * CS)) == 0;
  }
};

// int8: the value itself in one fp16 plane, one product per K block and output column half.
// The tile is 128 x 256: each issuer owns one 128-column half (its own accumulator), so both
// halves reuse the same A tile.  Chunks of 512*CS reduction indices, |sum| <= 512*CS * 2^14;
// the two accumulators' chunk ends are staggered by half a chunk.
template <>
struct Scheme<1> {
  static constexpr int BN = 256;
  static constexpr int UMMA_N = 128;      // one column half per MMA
  static constexpr int NSLOT = 4;
  static constexpr int SLOT_COLS = 128;
  static constexpr int NACC = 2;
  static constexpr int NPROD = 2;         // product p: column half p
  static constexpr int EMPTY_COUNT = 2;   // both issuers read every stage
  static constexpr int COLS = 128;        // C columns per epilogue thread: warp (quad, half) owns half h
  static constexpr int DRAIN_WARPS = 4;   // an accumulator is drained by the four warps of its half
  __device__ static constexpr bool drains(int half, int a) { return half == a; }
  __device__ static constexpr int a_limb(int) { return 0; }
  __device__ static constexpr int b_limb(int) { return 0; }
  __device__ static constexpr int b_row0(int p) { return p * 128; }
  __device__ static constexpr int acc(int p, int) { return p; }
  __device__ static constexpr int issuer(int p, int) { return p; }
  __device__ static constexpr int owner(int a) { return a; }
  __device__ static constexpr int shift(int) { return 0; }
  template <int CS>
  __device__ static bool chunk_ends(int a, int kb, int nkb) {
    return kb == nkb - 1 || (((kb + 1) * 64 + a * 256 * CS) % (512 * CS)) == 0;
  }
};

// int16 by Karatsuba's three products (an option, GEMMI_OPT_KARATSUBA): besides the limbs h and l
// every operand has a third plane s = h + l (|s| <= 255, exact in fp16), and
//     a*b = 2^16 h_a h_b + 2^8 (s_a s_b - h_a h_b - l_a l_b) + l_a l_b
//         = (2^16 - 2^8) HH + 2^8 SS + (1 - 2^8) LL,
// three products of N = 128 per K block (HH = h_a h_b, LL = l_a l_b, SS = s_a s_b) instead of the
// four limb products (two of N = 256).  Issuer 0 owns HH and LL, issuer 1 owns SS.  HH and LL
// products are at most 2^14 in magnitude (chunks of 512 * CS indices, staggered by half a chunk),
// SS products up to 255^2 < 2^16: its chunks are 128 * CS indices (sums within 2^23 for CS = 1,
// 2^24 for CS = 2).  Three accumulators live in four 128-column slots: one spare, into which the
// owner moves an accumulator at its chunk end while the old slot is drained.
template <>
struct Scheme<3> {
  static constexpr int BN = 128;
  static constexpr int UMMA_N = 128;
  static constexpr int NACC = 3;
  static constexpr int NPROD = 3;         // product p: plane p of A times plane p of B
  static constexpr int NSLOT = 4;
  static constexpr int SLOT_COLS = 128;
  static constexpr int EMPTY_COUNT = 2;   // both issuers read every stage
  static constexpr int COLS = 64;         // C columns per epilogue thread (two warps per lane quadrant)
  static constexpr int DRAIN_WARPS = 8;   // every epilogue warp drains every accumulator (its 64 columns)
  __device__ static constexpr bool drains(int, int) { return true; }
  __device__ static constexpr int a_limb(int p) { return p; }
  __device__ static constexpr int b_limb(int p) { return p; }
  __device__ static constexpr int b_row0(int) { return 0; }
  __device__ static constexpr int acc(int p, int) { return p; }
  __device__ static constexpr int issuer(int p, int) { return p == 2 ? 1 : 0; }
  __device__ static constexpr int owner(int a) { return a == 2 ? 1 : 0; }
  // weight of accumulator a (0: HH, 1: LL, 2: SS), modulo 2^64
  __device__ static constexpr uint64_t weight(int a) {
    return a == 0 ? uint64_t{65280} : a == 1 ? ~uint64_t{254} : uint64_t{256};  // 2^16 - 2^8, 1 - 2^8, 2^8
  }
  template <int CS>
  __device__ static bool chunk_ends(int a, int kb, int nkb) {
    if (kb == nkb - 1) return true;
    if (a == 2) return (((kb + 1) * 64) % (128 * CS)) == 0;
    return (((kb + 1) * 64 + a * 256 * CS) % (512 * CS)) == 0;
  }
};

// Assignment of accumulators to the four TMEM slots, replayed identically by every role.
// Spare slots form a FIFO: a chunk end moves the accumulator into the oldest spare and queues
// its old slot.  rotate() returns the parity to wait on (the slot's empty barrier) before the
// new slot may be written: the n-th assignment of a slot waits for its (n-1)-th drain.
template <int NACC, int NSLOT>
struct SlotRing {
  int slot_of[NACC];
  int spares[NSLOT - NACC];
  uint32_t assign_parity;  // bit s: parity of the number of assignments of slot s so far

  __device__ __forceinline__ void init() {
    assign_parity = 0;
#pragma unroll
    for (int a = 0; a < NACC; ++a) {
      slot_of[a] = a;
      assign_parity ^= 1u << a;
    }
#pragma unroll
    for (int i = 0; i < NSLOT - NACC; ++i) spares[i] = NACC + i;
  }
  __device__ __forceinline__ uint32_t rotate(int a) {
    const int old = slot_of[a];
    const int fresh = spares[0];
#pragma unroll
    for (int i = 0; i + 1 < NSLOT - NACC; ++i) spares[i] = spares[i + 1];
    spares[NSLOT - NACC - 1] = old;
    slot_of[a] = fresh;
    const uint32_t par = ((assign_parity >> fresh) & 1u) ^ 1u;
    assign_parity ^= 1u << fresh;
    return par;
  }
};

// No spare slots: accumulator a keeps slot a, and each new chunk waits for the previous chunk's
// drain of that slot.
template <int NACC>
struct SlotRing<NACC, NACC> {
  int slot_of[NACC];
  uint32_t assign_parity;

  __device__ __forceinline__ void init() {
    assign_parity = 0;
#pragma unroll
    for (int a = 0; a < NACC; ++a) {
      slot_of[a] = a;
      assign_parity ^= 1u << a;
    }
  }
  __device__ __forceinline__ uint32_t rotate(int a) {
    const int slot = slot_of[a];
    const uint32_t par = ((assign_parity >> slot) & 1u) ^ 1u;
    assign_parity ^= 1u << slot;
    return par;
  }
};

// Centred limbs of both int16 halves of x as fp16 pairs, exactly: h = floor((a + 128) / 256) and
// l = a - 256 h, computed with byte logic as
//   l + 128 = lo_byte ^ 0x80,   h + 128 = (hi_byte ^ 0x80) + (lo_byte >> 7),
// each placed under the fp16 bit pattern 0x6400 (1024 + v, v <= 256) and recovered by one fp16
// subtraction of 1152 = 0x6480.
__device__ __forceinline__ void limbs16x2(uint32_t x, uint32_t& hi, uint32_t& lo) {
  const uint32_t l_bits = (x & 0x00FF00FFu) ^ 0x64806480u;
  const uint32_t h_bits = (((x >> 8) & 0x00FF00FFu) ^ 0x64806480u) + ((x >> 7) & 0x00010001u);
  const __half2 k = __half2half2(__ushort_as_half(0x6480));
  const __half2 l = __hsub2(*reinterpret_cast<const __half2*>(&l_bits), k);
  const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&h_bits), k);
  lo = *reinterpret_cast<const uint32_t*>(&l);
  hi = *reinterpret_cast<const uint32_t*>(&h);
}

// Position in a ring of n slots: the slot and the parity of its current use.  Pipeline loops
// advance it by one per K block instead of dividing a running counter (64-bit division is a
// long software routine on the GPU, and it sat on every producer's critical path).
struct RingPos {
  int slot = 0;
  uint32_t phase = 0;
  __device__ __forceinline__ void advance(int n) {
    if (++slot == n) {
      slot = 0;
      phase ^= 1u;
    }
  }
};

__host__ __device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int group_m, int& mt, int& nt) {
  const int per_group = group_m * num_n;
  const int group = t / per_group;
  const int first_m = group * group_m;
  const int rows_here = group_m < num_m - first_m ? group_m : num_m - first_m;
  const int in_group = t - group * per_group;
  mt = first_m + in_group % rows_here;
  nt = in_group / rows_here;
}

__device__ __forceinline__ uint64_t l2_policy(int hint) {
  uint64_t p = 0;
  if (hint == 1) asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  else if (hint == 2) asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const void* map, uint32_t bar, int32_t x, int32_t y,
                                                 int hint, uint64_t policy) {
  if (hint == 0) {
    tma_load_2d(dst, map, bar, x, y);
  } else {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%3, %4}], [%2], %5;"
        ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "l"(policy)
        : "memory");
  }
}

__device__ __forceinline__ int32_t f32_to_i32(uint32_t bits) {
  int32_t v;
  asm("cvt.rni.s32.f32 %0, %1;" : "=r"(v) : "f"(__uint_as_float(bits)));
  return v;
}

}  // namespace tc
}  // namespace gemmi
