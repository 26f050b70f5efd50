/*
 * gemm_oracle.c -- the CPU oracle for the exact integer GEMM  C += A*B.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file or the library built from it; only the test-suite, the smoke
 * check and the timed CPU baseline of the benchmark use it.  It shares no code,
 * header, table or helper with the CUDA library.
 *
 * What it computes (paper, Section 4.1, the GEMM definition): A is m x k,
 * B is k x n, C is m x n, and C is updated in place by the product A*B.  The
 * paper's micro-kernel (Section 4.1, loop L6 of Figure 1) builds that update as
 * a sequence of rank-1 updates, one per index p of the reduction dimension,
 * and its AIE accumulators are wide (48-bit) precisely so that the 16-bit
 * products are summed without overflow (Section 6.2, closing remarks).
 *
 * The oracle is that definition written out: for every row i, every p and
 * every column j, C[i][j] += A[i][p] * B[p][j], each product formed exactly
 * (a 16x16-bit product needs at most 31 bits) and summed in 64-bit unsigned
 * arithmetic, i.e. modulo 2^64.  Because addition modulo 2^64 is associative
 * and commutative, the final C is unique whatever order a fast implementation
 * sums in, so the comparison against a GPU result is bit-exact.  The int8
 * variant is the same update with int8 operands and an int32 C, taken modulo
 * 2^32 (each product is exact in 32 bits; the sums run in unsigned 32-bit
 * arithmetic, the same rank-1 order as the int16 loop).  Further
 * down: the int4 variant (operands packed two to a byte), the paper's
 * micro-kernel output (shift, round, saturate to int16) and the convolution
 * written out from its definition; each states its own layout.
 *
 * Storage is row-major with leading dimensions: A[i*lda+p], B[p*ldb+j],
 * C[i*ldc+j]; entries of C outside the m x n block are never read or written.
 * All pointers are HOST pointers.  nthreads > 1 splits the rows i across
 * OpenMP threads (each thread owns whole rows of C, so the sum for each entry
 * is still the plain sequential loop over p); it exists only so that large
 * cases finish in reasonable time on many cores.
 *
 * Return value: 0 on success, 1 on an invalid argument (negative size, ld too
 * small, null pointer with a non-zero size).
 */
#include <stdint.h>
#include <stddef.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static int oracle_check(int64_t m, int64_t n, int64_t k, const void* A, int64_t lda,
                        const void* B, int64_t ldb, const void* C, int64_t ldc) {
  if (m < 0 || n < 0 || k < 0) return 1;
  if (m == 0 || n == 0) return 0;
  if (ldc < n) return 1;
  if (C == NULL) return 1;
  if (k == 0) return 0;
  if (lda < k || ldb < n) return 1;
  if (A == NULL || B == NULL) return 1;
  return 0;
}

/* C (int64, m x n) += A (int16, m x k) * B (int16, k x n), modulo 2^64. */
int gemm_oracle_i16(int64_t m, int64_t n, int64_t k,
                    const int16_t* A, int64_t lda,
                    const int16_t* B, int64_t ldb,
                    int64_t* C, int64_t ldc, int nthreads) {
  if (oracle_check(m, n, k, A, lda, B, ldb, C, ldc)) return 1;
  if (m == 0 || n == 0 || k == 0) return 0;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
#else
  (void)nthreads;
#endif
  for (int64_t i = 0; i < m; ++i) {
    uint64_t* c = (uint64_t*)(C + i * ldc);
    for (int64_t p = 0; p < k; ++p) {
      /* one rank-1 term: row i of C gains A[i][p] times row p of B */
      const int64_t a = (int64_t)A[i * lda + p];
      const int16_t* b = B + p * ldb;
      for (int64_t j = 0; j < n; ++j)
        c[j] += (uint64_t)(a * (int64_t)b[j]);
    }
  }
  return 0;
}

/* C (int32, m x n) += A (int8, m x k) * B (int8, k x n), modulo 2^32. */
int gemm_oracle_i8(int64_t m, int64_t n, int64_t k,
                   const int8_t* A, int64_t lda,
                   const int8_t* B, int64_t ldb,
                   int32_t* C, int64_t ldc, int nthreads) {
  if (oracle_check(m, n, k, A, lda, B, ldb, C, ldc)) return 1;
  if (m == 0 || n == 0 || k == 0) return 0;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
#else
  (void)nthreads;
#endif
  for (int64_t i = 0; i < m; ++i) {
    /* unsigned 32-bit arithmetic: every addition is taken modulo 2^32 */
    uint32_t* c = (uint32_t*)(C + i * ldc);
    for (int64_t p = 0; p < k; ++p) {
      /* one rank-1 term, as in the int16 loop: row i of C gains A[i][p] times row p of B */
      const int32_t a = (int32_t)A[i * lda + p];
      const int8_t* b8 = B + p * ldb;
      for (int64_t j = 0; j < n; ++j)
        c[j] += (uint32_t)(a * (int32_t)b8[j]);
    }
  }
  return 0;
}

/*
 * Lower precision (Section 6.1, the datatype discussion: the INT16 micro-kernel is the paper's
 * baseline and its design is to be carried to lower precision).  The int4 variant is the same
 * update with signed 4-bit operands and an int32 C, modulo 2^32.  Two operands share a byte: the
 * element with even index sits in the low nibble (bits 0-3), the one with odd index in the high
 * nibble (bits 4-7), each in two's complement (nibble values 8..15 stand for -8..-1).  A packs
 * along its rows (element (i, p) in byte A[i*lda + p/2]), B along its rows too (element (p, j) in
 * byte B[p*ldb + j/2]); lda and ldb count BYTES and must be at least ceil(k/2) and ceil(n/2).  The
 * unused high nibble of a row's last byte (odd k for A, odd n for B) is never read.
 */
static int64_t oracle_nibble(const uint8_t* row, int64_t idx) {
  const unsigned byte = row[idx / 2];
  const unsigned v = (idx % 2 == 0) ? (byte & 15u) : (byte >> 4);
  return v >= 8 ? (int64_t)v - 16 : (int64_t)v;
}

int gemm_oracle_i4(int64_t m, int64_t n, int64_t k,
                   const uint8_t* A, int64_t lda,
                   const uint8_t* B, int64_t ldb,
                   int32_t* C, int64_t ldc, int nthreads) {
  if (m < 0 || n < 0 || k < 0) return 1;
  if (m == 0 || n == 0) return 0;
  if (ldc < n || C == NULL) return 1;
  if (k == 0) return 0;
  if (lda < (k + 1) / 2 || ldb < (n + 1) / 2) return 1;
  if (A == NULL || B == NULL) return 1;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
#else
  (void)nthreads;
#endif
  for (int64_t i = 0; i < m; ++i) {
    int32_t* c = C + i * ldc;
    for (int64_t j = 0; j < n; ++j) {
      uint64_t s = (uint64_t)(int64_t)c[j];
      for (int64_t p = 0; p < k; ++p)
        s += (uint64_t)(oracle_nibble(A + i * lda, p) * oracle_nibble(B + p * ldb, j));
      c[j] = (int32_t)(uint32_t)s; /* keep the low 32 bits: modulo 2^32 */
    }
  }
  return 0;
}

/*
 * The paper's micro-kernel output (Section 5.2, the simplified AIE micro-kernel listing): the
 * wide accumulator is shifted, rounded and saturated to 16 bits ("srs") and added to the int16
 * C block with a plain 16-bit vector addition.  The paper is silent on the rounding of the shift
 * (its listing uses shift 0, where there is none), on how wide the accumulated reduction is when
 * k_c < k, and on whether the addition saturates.  The readings taken here:
 *   - the accumulator holds the full reduction, S = sum_p A[i][p] * B[p][j] (k_c = k, the
 *     configuration of the paper's best result);
 *   - the shift rounds half up: R = floor((S + 2^(shift-1)) / 2^shift) for shift >= 1, R = S
 *     for shift 0;
 *   - saturation clamps R to [-32768, 32767];
 *   - the addition wraps modulo 2^16.
 * S is formed exactly: |S| <= k * 2^30 < 2^62 for every k below 2^31, so no step wraps.
 */
static int64_t oracle_floor_div_pow2(int64_t v, int shift) {
  /* floor(v / 2^shift) written with non-negative operands only */
  const int64_t d = (int64_t)1 << shift;
  if (v >= 0) return v / d;
  return -((-v + d - 1) / d);
}

int gemm_oracle_i16_srs(int64_t m, int64_t n, int64_t k,
                        const int16_t* A, int64_t lda,
                        const int16_t* B, int64_t ldb,
                        int16_t* C, int64_t ldc, int shift, int nthreads) {
  if (oracle_check(m, n, k, A, lda, B, ldb, C, ldc)) return 1;
  if (shift < 0 || shift > 62) return 1;
  if (m == 0 || n == 0) return 0;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
#else
  (void)nthreads;
#endif
  for (int64_t i = 0; i < m; ++i) {
    for (int64_t j = 0; j < n; ++j) {
      int64_t s = 0;
      for (int64_t p = 0; p < k; ++p) s += (int64_t)A[i * lda + p] * (int64_t)B[p * ldb + j];
      int64_t r = shift == 0 ? s : oracle_floor_div_pow2(s + ((int64_t)1 << (shift - 1)), shift);
      if (r > 32767) r = 32767;
      if (r < -32768) r = -32768;
      const uint16_t sum = (uint16_t)((uint16_t)C[i * ldc + j] + (uint16_t)r);
      C[i * ldc + j] = (int16_t)sum;
    }
  }
  return 0;
}

/*
 * A convolution lowered to the GEMM (Sections 2 and 3 of the paper: the IM2COL / IM2ROW
 * transform turns the convolution operator into one large GEMM, and the transform can be applied
 * on the fly as part of the packing).  The oracle is the convolution itself, written out from its
 * definition rather than through a lowered matrix:
 *   Y[n][ho][wo][co] += sum over r < R, s < S, c < Cin of
 *                       X[n][ho + r - pad_h][wo + s - pad_w][c] * Wt[(r*S + s)*Cin + c][co],
 * with X taken as 0 outside 0 <= h < H, 0 <= w < W (zero padding), stride 1, and
 * Ho = H + 2*pad_h - R + 1, Wo = W + 2*pad_w - S + 1.  X is NHWC (N x H x W x Cin), Wt is the
 * weight matrix of the lowered GEMM (R*S*Cin rows in (r, s, c) order, Cout columns), Y is NHWC
 * (N x Ho x Wo x Cout); all dense, all HOST pointers.  Sums modulo 2^64 as in the GEMM.
 * Returns 0, or 1 on an invalid argument.
 */
int gemm_oracle_conv2d_i16(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                           int64_t R, int64_t S, int64_t pad_h, int64_t pad_w,
                           const int16_t* X, const int16_t* Wt, int64_t* Y, int nthreads) {
  if (N < 0 || H < 0 || W < 0 || Cin < 0 || Cout < 0 || R < 1 || S < 1 || pad_h < 0 || pad_w < 0) return 1;
  const int64_t Ho = H + 2 * pad_h - R + 1, Wo = W + 2 * pad_w - S + 1;
  if (Ho < 0 || Wo < 0) return 1;
  if (N == 0 || Ho == 0 || Wo == 0 || Cout == 0) return 0;
  if (Y == NULL) return 1;
  if (Cin == 0) return 0;
  if (X == NULL || Wt == NULL) return 1;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
#else
  (void)nthreads;
#endif
  for (int64_t row = 0; row < N * Ho; ++row) {
    const int64_t n = row / Ho, ho = row % Ho;
    for (int64_t wo = 0; wo < Wo; ++wo) {
      uint64_t* y = (uint64_t*)(Y + ((n * Ho + ho) * Wo + wo) * Cout);
      for (int64_t r = 0; r < R; ++r) {
        const int64_t h = ho + r - pad_h;
        if (h < 0 || h >= H) continue;
        for (int64_t s = 0; s < S; ++s) {
          const int64_t w = wo + s - pad_w;
          if (w < 0 || w >= W) continue;
          const int16_t* x = X + ((n * H + h) * W + w) * Cin;
          for (int64_t c = 0; c < Cin; ++c) {
            const int64_t a = (int64_t)x[c];
            const int16_t* wt = Wt + ((r * S + s) * Cin + c) * Cout;
            for (int64_t co = 0; co < Cout; ++co) y[co] += (uint64_t)(a * (int64_t)wt[co]);
          }
        }
      }
    }
  }
  return 0;
}

/*
 * The same two functions under the names of the library's oracle interface (gemmi_oracle_*):
 * identical arguments, host pointers, the int nthreads of the loops above.
 */
int gemmi_oracle_i16(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda,
                     const int16_t* B, int64_t ldb, int64_t* C, int64_t ldc, int nthreads) {
  return gemm_oracle_i16(m, n, k, A, lda, B, ldb, C, ldc, nthreads);
}

int gemmi_oracle_i8(int64_t m, int64_t n, int64_t k, const int8_t* A, int64_t lda,
                    const int8_t* B, int64_t ldb, int32_t* C, int64_t ldc, int nthreads) {
  return gemm_oracle_i8(m, n, k, A, lda, B, ldb, C, ldc, nthreads);
}

/* Threads the library was built to use (1 without OpenMP). */
int gemm_oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
