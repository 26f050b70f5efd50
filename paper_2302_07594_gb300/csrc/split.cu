// split.cu -- operand packing: integer operands -> fp16 limb planes in K-major order.
//
// This is the packing step of the paper's blocked GEMM (Section 4.1, the
// routines that copy A and B into the buffers A_c and B_c, and Section 5.1,
// where the activation operand is packed at run time), re-targeted: instead of
// re-ordering into micro-panels, each int16 value a is written as two exact
// fp16 "limbs" so the tensor cores can multiply them:
//     h = floor((a + 128) / 256)  in [-128, 128],   l = a - 256*h  in [-128, 127],
// so a = 256*h + l and every limb product is at most 2^14 in magnitude.
// int8 values are exact in fp16 and are written unchanged (one plane).
//
// Both operands end up K-major (the reduction index is contiguous): A keeps
// its row-major layout; B (k x n, row-major) is transposed to n x k.  Plane
// rows have a pitch that is a multiple of 8 elements (16 bytes), which the TMA
// tensor maps require.  Pitch columns at and beyond k are written as zero.
//
// One launch converts both operands (or just one: a null operand is skipped): the first blocks
// of the grid stream A, one warp per row (16-byte loads, 16-byte stores per plane and 8
// elements), the rest transpose B in 64 x 64 tiles through shared memory (16-byte accesses on
// both sides, swizzled so neither side has bank conflicts).  The kernel is bound by HBM: per
// int16 element 2 bytes are read and 4 written; per int8 element 1 and 2.
#include <cuda.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace gemmi {
namespace {

// Every integer of magnitude <= 2048 is exactly representable in fp16 (11-bit significand).
__device__ __forceinline__ __half to_half_exact(int v) { return __int2half_rn(v); }

__device__ __forceinline__ void limbs16(int a, __half& h, __half& l) {
  const int hi = (a + 128) >> 8;  // arithmetic shift = floor division by 256
  const int lo = a - (hi << 8);
  h = to_half_exact(hi);
  l = to_half_exact(lo);
}

template <typename T>
struct Part {
  const T* src;
  int64_t ld;
  int64_t rows;   // A: m;  B: k (rows of B)
  int64_t cols;   // A: k;  B: n
  __half* p0;
  __half* p1;
  int64_t pitch;  // plane row pitch (elements)
  bool vec;       // 16-byte (int16) / 8-byte (int8) loads of 8 elements are aligned
};

template <typename T>
__device__ __forceinline__ void load8(const T* src, bool vec, int64_t valid, int (&v)[8]) {
  if (vec && valid >= 8) {
    if constexpr (sizeof(T) == 2) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(src));
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[2 * i] = static_cast<int16_t>(w[i] & 0xFFFFu);
        v[2 * i + 1] = static_cast<int16_t>(w[i] >> 16);
      }
    } else {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(src));
      const uint32_t w[2] = {u.x, u.y};
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = static_cast<int8_t>((w[i / 4] >> (8 * (i % 4))) & 0xFFu);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = (i < valid) ? static_cast<int>(src[i]) : 0;
  }
}

template <int NL>
__device__ __forceinline__ void store8(__half* p0, __half* p1, const int (&v)[8]) {
  __align__(16) __half h[8];
  __align__(16) __half l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if constexpr (NL == 2) {
      limbs16(v[i], h[i], l[i]);
    } else {
      h[i] = to_half_exact(v[i]);
    }
  }
  *reinterpret_cast<uint4*>(p0) = *reinterpret_cast<const uint4*>(h);
  if constexpr (NL == 2) *reinterpret_cast<uint4*>(p1) = *reinterpret_cast<const uint4*>(l);
}

constexpr int TT = 64;      // transpose tile edge: 64 reduction indices x 64 columns of B
constexpr int THREADS = 256;
constexpr int WARPS = THREADS / 32;

// A: m x k (lda) -> planes m x pitch.  One warp per row at a time; each lane converts U groups of
// 8 elements per step, all loads issued before the stores (U * 16 bytes of int16 in flight).
template <typename T, int NL>
__device__ __forceinline__ void split_rows(const Part<T>& a, int a_blocks) {
  constexpr int U = sizeof(T) == 2 ? 2 : 4;
  const int lane = threadIdx.x % 32;
  const int64_t groups = a.pitch / 8;
  const int64_t nwarps = static_cast<int64_t>(a_blocks) * WARPS;
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * WARPS + threadIdx.x / 32; r < a.rows; r += nwarps) {
    const T* src = a.src + r * a.ld;
    __half* d0 = a.p0 + r * a.pitch;
    __half* d1 = a.p1 + r * a.pitch;
    for (int64_t g0 = lane; g0 < groups; g0 += 32 * U) {
      int v[U][8];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t p = (g0 + 32 * u) * 8;
        if (p < a.pitch) load8(src + p, a.vec, a.cols - p, v[u]);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t p = (g0 + 32 * u) * 8;
        if (p < a.pitch) store8<NL>(d0 + p, d1 + p, v[u]);
      }
    }
  }
}

// B: k x n (ldb) -> planes n x pitch (transposed), one 64 x 64 tile per step.  The tile passes
// through shared memory already converted to fp16, stored untransposed (row = reduction index p,
// 128 bytes = 64 columns j) with its 16-byte chunks XOR-swizzled by bits 3-5 of p.  Rows are
// written a 16-byte chunk per thread; the transposed read gathers column j of 8 consecutive rows
// p, and the swizzle puts the 8 row groups of one read in 8 different bank groups.
template <typename T, int NL>
__device__ __forceinline__ void split_cols(const Part<T>& b, int a_blocks, int64_t b_tiles_j, int64_t b_tiles,
                                           __half (*sm)[TT * TT]) {
  const int64_t nblk = gridDim.x - a_blocks;
  for (int64_t t = blockIdx.x - a_blocks; t < b_tiles; t += nblk) {
    const int64_t p_base = (t / b_tiles_j) * TT;  // reduction index = row of B
    const int64_t j_base = (t % b_tiles_j) * TT;  // column of B
    // load: 64 rows x 8 groups of 8 columns
#pragma unroll
    for (int q = threadIdx.x; q < TT * TT / 8; q += THREADS) {
      const int r = q >> 3;       // p - p_base
      const int c = q & 7;        // 16-byte chunk = columns 8c .. 8c+7
      const int64_t p = p_base + r, j = j_base + 8 * c;
      int v[8];
      if (p < b.rows) {
        load8(b.src + p * b.ld + j, b.vec, b.cols - j, v);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = 0;
      }
      const int off = r * TT + ((c ^ ((r >> 3) & 7)) * 8);
      store8<NL>(&sm[0][off], &sm[NL - 1][off], v);
    }
    __syncthreads();
    // store: 64 plane rows j x 8 chunks of 8 reduction indices; 8 lanes write one 128-byte row
#pragma unroll
    for (int q = threadIdx.x; q < TT * TT / 8; q += THREADS) {
      const int jj = q >> 3;      // j - j_base
      const int g = q & 7;        // reduction indices p_base + 8g .. +7
      const int64_t j = j_base + jj, p = p_base + 8 * g;
      if (j < b.cols && p < b.pitch) {
        const int col = ((jj >> 3) ^ g) * 8 + (jj & 7);  // rows 8g..8g+7 all have swizzle g
#pragma unroll
        for (int l = 0; l < NL; ++l) {
          __align__(16) __half h[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) h[i] = sm[l][(8 * g + i) * TT + col];
          __half* dst = (l == 0 ? b.p0 : b.p1) + j * b.pitch + p;
          *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(h);
        }
      }
    }
    __syncthreads();
  }
}

template <typename T, int NL>
__global__ void __launch_bounds__(THREADS)
split_kernel(Part<T> a, Part<T> b, int a_blocks, int64_t b_tiles_j, int64_t b_tiles) {
  __shared__ __align__(16) __half sm[NL][TT * TT];
  pdl_launch_dependents();
  if (static_cast<int>(blockIdx.x) < a_blocks) split_rows<T, NL>(a, a_blocks);
  else split_cols<T, NL>(b, a_blocks, b_tiles_j, b_tiles, sm);
}

// ---------------------------------------------------------------- TMA-fed variant
// For operands whose rows TMA can address (16-byte aligned base and row stride), raw tiles of
// 8 KB stream into a 4-stage shared-memory ring (one producer thread, mbarriers), so each SM
// keeps about 100 KB of loads in flight; eight consumer warps convert them.
//   A item: 32 rows x 256 bytes of raw A -> fp16 planes with coalesced 16-byte stores.
//   B item: 64 reduction indices x 128 bytes of raw B (64 int16 or 128 int8 columns), loaded
//           with the 128-byte swizzle.  A warp converts 8 rows x 32 columns at a time: each lane
//           reads the 2 columns of one row that an 8 x 8 matrix fragment holds (32-bit loads, no
//           bank conflicts), converts them to an fp16 pair, and stmatrix.trans writes the four
//           8 x 8 blocks transposed into a staging tile in the same swizzled layout (row j = 64
//           reduction indices), which goes out by a TMA store.
// Every wait is bounded; there is no hardware barrier after the start, so a timeout in one warp
// can only make the others time out too.
namespace tsplit {
constexpr int CONSUMERS = 256;
constexpr int THREADS = CONSUMERS + 32;
constexpr int RAW = 8192;
constexpr int STAGES = 4;
constexpr int A_ROWS = 32;
constexpr int B_P = 64;
constexpr int STG = 16384;
constexpr int NBAR = 2 * STAGES + 4;  // full, empty, staging full x2, staging free x2
constexpr size_t SMEM = 1024 + STAGES * RAW + 2 * STG + 8 * NBAR;
static_assert((RAW / 16) % CONSUMERS == 0, "whole raw chunks per consumer thread");
constexpr int CTAS_PER_SM = 3;  // 65 KB of shared memory each: three fit in an SM's 228 KB
static_assert(CTAS_PER_SM * SMEM <= 228 * 1024, "resident CTAs per SM");
}  // namespace tsplit

struct TmaSplitParams {
  int64_t m, a_pitch;
  __half* a_p0;
  __half* a_p1;
  int64_t a_tiles_k, a_items;
  int64_t b_tiles_j, b_items;
  uint32_t* status;
  uint64_t timeout_ns;
};

// Four int8 values packed in a word -> two fp16 pairs, exactly: u = w ^ 0x80808080 holds v + 128
// in each byte; a byte permute puts each byte under the fp16 bit pattern 0x64xx = 1024 + xx, and
// one fp16 subtraction of 1152 = 0x6480 per pair leaves v (every integer up to 2048 is exact).
__device__ __forceinline__ void i8x4_to_half2x2(uint32_t w, uint32_t& h01, uint32_t& h23) {
  const uint32_t u = w ^ 0x80808080u;
  const uint32_t a = __byte_perm(u, 0x64646464u, 0x5140);
  const uint32_t b = __byte_perm(u, 0x64646464u, 0x7362);
  const __half2 k = __half2half2(__ushort_as_half(0x6480));
  const __half2 ha = __hsub2(*reinterpret_cast<const __half2*>(&a), k);
  const __half2 hb = __hsub2(*reinterpret_cast<const __half2*>(&b), k);
  h01 = *reinterpret_cast<const uint32_t*>(&ha);
  h23 = *reinterpret_cast<const uint32_t*>(&hb);
}

using tc::limbs16x2;

// Bytes s and s + 1 (s = 0 or 2) of a word of four int8 values -> one fp16 pair, exactly.
__device__ __forceinline__ uint32_t i8x2_to_half2(uint32_t w, uint32_t s) {
  const uint32_t b = __byte_perm(w ^ 0x80808080u, 0x64646464u, 0x4040u + s + (s << 8) + 0x0100u);
  const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&b), __half2half2(__ushort_as_half(0x6480)));
  return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}

// Four 8 x 8 b16 matrices, stored transposed: lane l holds (row l / 4, columns 2(l % 4), +1) of
// matrix i in r[i]; lane 8i + t gives the address of the 16-byte row t of stored matrix i, which
// receives column t of matrix i.
__device__ __forceinline__ void stsm_x4_trans(uint32_t addr, const uint32_t (&r)[4]) {
  asm volatile("stmatrix.sync.aligned.m8n8.x4.trans.shared.b16 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(r[0]),
               "r"(r[1]), "r"(r[2]), "r"(r[3])
               : "memory");
}

// q = a / b, r = a - q * b, in 32-bit arithmetic when both fit (a 64-bit division is a long
// software routine, and it sat on every item of the split kernel).
__device__ __forceinline__ void divmod(int64_t a, int64_t b, int64_t& q, int64_t& r) {
  if (((static_cast<uint64_t>(a) | static_cast<uint64_t>(b)) >> 31) == 0)
    q = static_cast<int64_t>(static_cast<uint32_t>(a) / static_cast<uint32_t>(b));
  else
    q = a / b;
  r = a - q * b;
}

__device__ __forceinline__ void tma_store_2d(const void* map, uint32_t src, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }

template <typename T, int NL>
__global__ void __launch_bounds__(tsplit::THREADS)
split_tma_kernel(const __grid_constant__ CUtensorMap rawA, const __grid_constant__ CUtensorMap rawB,
                 const __grid_constant__ CUtensorMap outB0, const __grid_constant__ CUtensorMap outB1,
                 TmaSplitParams P) {
  using namespace tsplit;
  constexpr int A_COLS = 256 / static_cast<int>(sizeof(T));  // raw A tile: 128 int16 / 256 int8
  constexpr int JB = 128 / static_cast<int>(sizeof(T));      // raw B tile columns: 64 int16 / 128 int8
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* stg = smem + STAGES * RAW;
  uint64_t* bars = reinterpret_cast<uint64_t*>(stg + 2 * STG);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t sfull0 = empty0 + 8 * STAGES;  // staging buffer b written by all consumers
  const uint32_t sfree0 = sfull0 + 16;          // staging buffer b read by its TMA store
  const int64_t items = P.a_items + P.b_items;
  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  // a GEMM launched after this split with programmatic stream serialization may set itself up
  // meanwhile; it waits for this grid's completion before it reads the planes
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, CONSUMERS / 32);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(sfull0 + 8 * b, CONSUMERS);
      mbar_init(sfree0 + 8 * b, 1);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == CONSUMERS / 32) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      if (P.a_items) tma_prefetch_desc(&rawA);
      if (P.b_items) tma_prefetch_desc(&rawB);
      tc::RingPos st;
      int64_t issued = 0;
      for (int64_t it = blockIdx.x; it < items; it += gridDim.x) {
        if (!bounded_wait(empty0 + 8 * st.slot, st.phase ^ 1u, P.timeout_ns)) {
          report_status(P.status, tc::STATUS_TIMEOUT, 31);
          break;
        }
        const uint32_t fb = full0 + 8 * st.slot;
        mbar_arrive_expect_tx(fb, RAW);
        const uint32_t dst = smem_u32(smem + st.slot * RAW);
        if (it < P.a_items) {
          int64_t rt, kt;
          divmod(it, P.a_tiles_k, rt, kt);
          tma_load_2d(dst, &rawA, fb, static_cast<int32_t>(kt * A_COLS), static_cast<int32_t>(rt * A_ROWS));
        } else {
          int64_t pt, jt;
          divmod(it - P.a_items, P.b_tiles_j, pt, jt);
          tma_load_2d(dst, &rawB, fb, static_cast<int32_t>(jt * JB), static_cast<int32_t>(pt * B_P));
        }
        ++issued;
        st.advance(STAGES);
      }
      // stay until the last copies have landed: if the consumers gave up, the CTA must not exit
      // with copies still writing its shared memory
      const int64_t first = issued > STAGES ? issued - STAGES : 0;
      for (int64_t i = first; i < issued; ++i)
        bounded_wait(full0 + 8 * static_cast<int>(i % STAGES), static_cast<uint32_t>((i / STAGES) & 1), P.timeout_ns);
    }
    return;
  }

  // -------------------------------------------------------------------- consumers (warps 0-7)
  const int tid = threadIdx.x;
  tc::RingPos st;
  int nb = 0;  // B items processed so far (staging buffer = nb & 1, its use = nb >> 1)
  for (int64_t it = blockIdx.x; it < items; it += gridDim.x) {
    const bool got = bounded_wait(full0 + 8 * st.slot, st.phase, P.timeout_ns);
    if (!__all_sync(0xFFFFFFFFu, got)) {
      if (lane == 0) report_status(P.status, tc::STATUS_TIMEOUT, 32);
      break;
    }
    const uint8_t* rawt = smem + st.slot * RAW;
    if (it < P.a_items) {
      int64_t rt, kt;
      divmod(it, P.a_tiles_k, rt, kt);
      if constexpr (sizeof(T) == 2) {
        // ---- A (int16): row = q / 16, 16-byte chunk c = q % 16 of the 256-byte raw row; the 16
        //      lanes of a row store 256 contiguous bytes of each plane row
        constexpr int ACH = RAW / 16 / CONSUMERS;  // 16-byte raw chunks per thread
        uint4 w[ACH];
#pragma unroll
        for (int u = 0; u < ACH; ++u) w[u] = *reinterpret_cast<const uint4*>(rawt + (tid + CONSUMERS * u) * 16);
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * st.slot);
#pragma unroll
        for (int u = 0; u < ACH; ++u) {
          const int q = tid + CONSUMERS * u;
          const int64_t row = rt * A_ROWS + (q >> 4);
          const int64_t col = kt * A_COLS + (q & 15) * 8;
          if (row >= P.m || col >= P.a_pitch) continue;
          uint4 h, l;
          limbs16x2(w[u].x, h.x, l.x);
          limbs16x2(w[u].y, h.y, l.y);
          limbs16x2(w[u].z, h.z, l.z);
          limbs16x2(w[u].w, h.w, l.w);
          *reinterpret_cast<uint4*>(P.a_p0 + row * P.a_pitch + col) = h;
          *reinterpret_cast<uint4*>(P.a_p1 + row * P.a_pitch + col) = l;
        }
      } else {
        // ---- A (int8): 8-byte pieces; lane c of a warp takes piece c of one 256-byte raw row, so
        //      each 16-byte store instruction writes 512 contiguous bytes of the plane row (with
        //      16-byte pieces every store left half of each 32-byte sector to the next one)
        constexpr int PIECES = RAW / 8 / CONSUMERS;
        uint2 w[PIECES];
#pragma unroll
        for (int u = 0; u < PIECES; ++u) w[u] = *reinterpret_cast<const uint2*>(rawt + (tid + CONSUMERS * u) * 8);
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * st.slot);
#pragma unroll
        for (int u = 0; u < PIECES; ++u) {
          const int q = tid + CONSUMERS * u;
          const int64_t row = rt * A_ROWS + (q >> 5);
          const int64_t col = kt * A_COLS + (q & 31) * 8;
          if (row >= P.m || col >= P.a_pitch) continue;
          uint4 o;
          i8x4_to_half2x2(w[u].x, o.x, o.y);
          i8x4_to_half2x2(w[u].y, o.z, o.w);
          *reinterpret_cast<uint4*>(P.a_p0 + row * P.a_pitch + col) = o;
        }
      }
    } else {
      // ---- B: 8 x 32 blocks (rows 8g .., columns 32jq ..) converted in fragments and written
      //      transposed to the staging tile by stmatrix
      int64_t pt, jt;
      divmod(it - P.a_items, P.b_tiles_j, pt, jt);
      const int buf = nb & 1;
      const uint32_t use = static_cast<uint32_t>(nb >> 1);
      if (use > 0) {
        const bool freed = bounded_wait(sfree0 + 8 * buf, (use - 1) & 1u, P.timeout_ns);
        if (!__all_sync(0xFFFFFFFFu, freed)) {
          if (lane == 0) report_status(P.status, tc::STATUS_TIMEOUT, 33);
          break;
        }
      }
      uint8_t* sbuf = stg + buf * STG;
      // warp w takes the units (p-block g, 32-column group jq) w, w + 8, ...; lane (r, q) =
      // (l / 4, l % 4) reads columns 32jq + 8i + 2q, +1 (i = 0..3) of row 8g + r, the fragment
      // of the 8 x 8 block i.  Eight rows meet eight different 16-byte chunk positions under the
      // swizzle, so the 32 lanes' loads hit 32 banks (int8: lanes 2s and 2s + 1 share a word).
      constexpr int JQ = JB / 32;                 // 32-column groups per raw tile: 2 (int16) / 4 (int8)
      constexpr int UNITS = 8 * JQ / (CONSUMERS / 32);  // per warp
      const int r = lane >> 2, q = lane & 3;
      uint32_t raw[UNITS][4];
#pragma unroll
      for (int u = 0; u < UNITS; ++u) {
        const int un = warp + (CONSUMERS / 32) * u;
        const int g = un / JQ, jq = un % JQ;
        const int p = 8 * g + r;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int x = static_cast<int>(sizeof(T)) * (32 * jq + 8 * i + 2 * q);  // byte offset in row p
          raw[u][i] = lds32(smem_u32(rawt) + p * 128 + (((x >> 4) ^ (p & 7)) << 4) + (x & 12));
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * st.slot);
      // lane 8i + t addresses staging row j = 32jq + 8i + t (block i's column t), chunk g
      const int mi = lane >> 3, t = lane & 7;
#pragma unroll
      for (int u = 0; u < UNITS; ++u) {
        const int un = warp + (CONSUMERS / 32) * u;
        const int g = un / JQ, jq = un % JQ;
        const uint32_t row_addr = smem_u32(sbuf) + (32 * jq + 8 * mi + t) * 128 + ((g ^ t) << 4);
        if constexpr (sizeof(T) == 2) {
          uint32_t h[4], l[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) limbs16x2(raw[u][i], h[i], l[i]);
          stsm_x4_trans(row_addr, h);
          stsm_x4_trans(row_addr + 8192, l);
        } else {
          uint32_t h[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) h[i] = i8x2_to_half2(raw[u][i], static_cast<uint32_t>((2 * q) & 2));
          stsm_x4_trans(row_addr, h);
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(sfull0 + 8 * buf);
      if (tid == 0) {
        // all consumers have written the staging tile: store it, then release the other buffer
        // once its store (issued for the previous B item) has finished reading
        if (!bounded_wait(sfull0 + 8 * buf, use & 1u, P.timeout_ns)) {
          report_status(P.status, tc::STATUS_TIMEOUT, 34);
        } else {
          const int32_t x = static_cast<int32_t>(pt * B_P), y = static_cast<int32_t>(jt * JB);
          tma_store_2d(&outB0, smem_u32(sbuf), x, y);
          if constexpr (NL == 2) tma_store_2d(&outB1, smem_u32(sbuf + 8192), x, y);
          bulk_commit();
          if (nb > 0) {
            bulk_wait_read_1();
            mbar_arrive(sfree0 + 8 * (buf ^ 1));
          }
        }
      }
      ++nb;
    }
    st.advance(STAGES);
  }
  if (tid == 0) bulk_wait_all();
}

// Streaming multiprocessors of the current device (queried once per device).
int device_sms() {
  static int sms[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return 148;
  if (sms[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) {
      cudaGetLastError();
      v = 148;
    }
    sms[dev] = v;
  }
  return sms[dev];
}

template <typename T, int NL>
bool launch_tma(const T* A, int64_t lda, const T* B, int64_t ldb, int64_t m, int64_t n, int64_t k, LimbPlanes pa,
                LimbPlanes pb, cudaStream_t s, uint32_t* status, uint64_t timeout_ns, cudaError_t* err) {
  constexpr int64_t esz = sizeof(T);
  constexpr int A_COLS = 256 / static_cast<int>(esz);
  constexpr int JB = 128 / static_cast<int>(esz);
  const int dt = esz == 2 ? 0 : 2;
  auto aligned = [](const void* p, int64_t ld_bytes) {
    return p == nullptr || (reinterpret_cast<uintptr_t>(p) % 16 == 0 && ld_bytes % 16 == 0);
  };
  if (!aligned(A, lda * esz) || !aligned(B, ldb * esz)) return false;
  CUtensorMap maps[4] = {};
  const char* why = nullptr;
  TmaSplitParams P = {};
  P.status = status;
  P.timeout_ns = timeout_ns;
  if (A != nullptr) {
    if (!encode_tensor_map_2d(&maps[0], dt, A, static_cast<uint64_t>(k), static_cast<uint64_t>(m),
                              static_cast<uint64_t>(lda * esz), A_COLS, tsplit::A_ROWS, 0, &why))
      return false;
    P.m = m;
    P.a_pitch = pa.pitch;
    P.a_p0 = static_cast<__half*>(pa.plane[0]);
    P.a_p1 = static_cast<__half*>(pa.plane[NL - 1]);
    P.a_tiles_k = (pa.pitch + A_COLS - 1) / A_COLS;
    P.a_items = ((m + tsplit::A_ROWS - 1) / tsplit::A_ROWS) * P.a_tiles_k;
  }
  if (B != nullptr) {
    if (!encode_tensor_map_2d(&maps[1], dt, B, static_cast<uint64_t>(n), static_cast<uint64_t>(k),
                              static_cast<uint64_t>(ldb * esz), JB, tsplit::B_P, 128, &why))
      return false;
    for (int l = 0; l < NL; ++l)
      if (!encode_tensor_map_2d(&maps[2 + l], 1, pb.plane[l], static_cast<uint64_t>(pb.pitch),
                                static_cast<uint64_t>(n), static_cast<uint64_t>(pb.pitch * 2), 64, JB, 128, &why))
        return false;
    if (NL == 1) maps[3] = maps[2];
    P.b_tiles_j = (n + JB - 1) / JB;
    P.b_items = ((pb.pitch + tsplit::B_P - 1) / tsplit::B_P) * P.b_tiles_j;
  }
  const int64_t items = P.a_items + P.b_items;
  if (items == 0) {
    *err = cudaSuccess;
    return true;
  }
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t e = cudaFuncSetAttribute(split_tma_kernel<T, NL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(tsplit::SMEM));
    if (e != cudaSuccess) {
      *err = e;
      return true;
    }
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  const int64_t resident = static_cast<int64_t>(device_sms()) * tsplit::CTAS_PER_SM;
  const int64_t grid = items < resident ? items : resident;
  split_tma_kernel<T, NL><<<static_cast<unsigned>(grid), tsplit::THREADS, tsplit::SMEM, s>>>(maps[0], maps[1], maps[2],
                                                                                            maps[3], P);
  *err = cudaGetLastError();
  return true;
}

template <typename T, int NL>
cudaError_t launch(const T* A, int64_t lda, const T* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                   LimbPlanes pa, LimbPlanes pb, cudaStream_t s, uint32_t* status, uint64_t timeout_ns) {
  constexpr int64_t esz = sizeof(T);
  cudaError_t err = cudaSuccess;
  if (launch_tma<T, NL>(A, lda, B, ldb, m, n, k, pa, pb, s, status, timeout_ns, &err)) return err;
  Part<T> a{A, lda, m, k, static_cast<__half*>(pa.plane[0]), static_cast<__half*>(pa.plane[NL - 1]), pa.pitch,
            reinterpret_cast<uintptr_t>(A) % (8 * esz) == 0 && (lda * esz) % (8 * esz) == 0};
  Part<T> b{B, ldb, k, n, static_cast<__half*>(pb.plane[0]), static_cast<__half*>(pb.plane[NL - 1]), pb.pitch,
            reinterpret_cast<uintptr_t>(B) % (8 * esz) == 0 && (ldb * esz) % (8 * esz) == 0};
  // A: one warp per row per step; B: one 64 x 64 tile per block step.
  // A null operand is skipped (packing only the weights, or only the activations).
  const int64_t a_rows = A != nullptr ? m : 0;
  int64_t a_blocks = (a_rows + WARPS - 1) / WARPS;
  const int64_t cap = static_cast<int64_t>(device_sms()) * 8;
  if (a_blocks > cap) a_blocks = cap;
  const int64_t tiles_p = (pb.pitch + TT - 1) / TT;  // cover the zero padding up to the pitch too
  const int64_t tiles_j = B != nullptr ? (n + TT - 1) / TT : 0;
  const int64_t b_tiles = tiles_p * tiles_j;
  int64_t b_blocks = b_tiles < cap ? b_tiles : cap;
  if (a_blocks + b_blocks < 1) return cudaSuccess;
  split_kernel<T, NL><<<static_cast<unsigned>(a_blocks + b_blocks), THREADS, 0, s>>>(
      a, b, static_cast<int>(a_blocks), tiles_j, b_tiles);
  return cudaGetLastError();
}

// The Karatsuba variant's third plane: s = h + l, eight fp16 values per 16-byte access.  Both
// limbs are integers of magnitude <= 128 and their sum (|s| <= 255) is exact in fp16.
__global__ void __launch_bounds__(256) limb_sum_kernel(const uint4* __restrict__ h, const uint4* __restrict__ l,
                                                       uint4* __restrict__ out, int64_t n_vec) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n_vec;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const uint4 a = __ldg(h + i), b = __ldg(l + i);
    uint4 r;
    const uint32_t* pa = &a.x;
    const uint32_t* pb = &b.x;
    uint32_t* pr = &r.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const __half2 sum = __hadd2(*reinterpret_cast<const __half2*>(pa + q), *reinterpret_cast<const __half2*>(pb + q));
      pr[q] = *reinterpret_cast<const uint32_t*>(&sum);
    }
    out[i] = r;
  }
}

}  // namespace

cudaError_t split_i16(const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                      LimbPlanes pa, LimbPlanes pb, cudaStream_t s, uint32_t* status, uint64_t timeout_ns) {
  return launch<int16_t, 2>(A, lda, B, ldb, m, n, k, pa, pb, s, status, timeout_ns);
}

cudaError_t convert_i8(const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb, int64_t m, int64_t n, int64_t k,
                       LimbPlanes pa, LimbPlanes pb, cudaStream_t s, uint32_t* status, uint64_t timeout_ns) {
  return launch<int8_t, 1>(A, lda, B, ldb, m, n, k, pa, pb, s, status, timeout_ns);
}

}  // namespace gemmi

namespace gemmi {
cudaError_t limb_sum_planes(LimbPlanes pa, LimbPlanes pb, int num_sms, cudaStream_t s) {
  const LimbPlanes* ops[2] = {&pa, &pb};
  for (const LimbPlanes* p : ops) {
    if (p->plane[2] == nullptr || p->rows == 0) continue;
    // rows x pitch fp16 values, pitch a multiple of 8: whole 16-byte vectors
    const int64_t n_vec = p->rows * p->pitch / 8;
    const int64_t blocks = (n_vec + 255) / 256;
    const int grid = static_cast<int>(blocks < 8 * static_cast<int64_t>(num_sms) ? blocks : 8 * static_cast<int64_t>(num_sms));
    limb_sum_kernel<<<grid, 256, 0, s>>>(static_cast<const uint4*>(p->plane[0]), static_cast<const uint4*>(p->plane[1]),
                                         static_cast<uint4*>(p->plane[2]), n_vec);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}
}  // namespace gemmi
