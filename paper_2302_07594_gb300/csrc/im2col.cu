// im2col.cu -- the IM2COL transform (Sections 2 and 3 of the paper), written out.
//
// Lowers a stride-1, zero-padded convolution of an NHWC int16 tensor X into the
// GEMM operand A: row m = (n, ho, wo) of the output, column kk = (r, s, c) of
// the filter, A[m][kk] = X[n][ho + r - pad_h][wo + s - pad_w][c], or 0 where
// that pixel lies outside the image; columns K .. lda - 1 are written as 0.
// gemmi_conv2d_i16 uses this only for shapes its implicit path (the fused
// kernel reading X directly) does not cover.  HBM-bound: it reads X about R*S
// times (mostly from L2) and writes the lowered matrix once.
#include <cuda_runtime.h>

#include "internal.h"

namespace gemmi {
namespace {

constexpr int THREADS = 256;

__global__ void __launch_bounds__(THREADS)
im2col_kernel(const int16_t* __restrict__ X, int16_t* __restrict__ Aout, int64_t lda, int64_t M, int64_t K,
              int H, int W, int Cin, int Ho, int Wo, int S, int ph, int pw) {
  const int64_t groups = lda / 8;
  const int64_t total = M * groups;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(THREADS) + threadIdx.x; g < total;
       g += static_cast<int64_t>(gridDim.x) * THREADS) {
    const int64_t m = g / groups;
    const int64_t k0 = (g - m * groups) * 8;
    const int64_t pix = m / Wo;
    const int wo = static_cast<int>(m - pix * Wo);
    const int ho = static_cast<int>(pix % Ho);
    const int64_t n = pix / Ho;
    __align__(16) int16_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int64_t kk = k0 + i;
      int16_t x = 0;
      if (kk < K) {
        const int64_t tap = kk / Cin;
        const int c = static_cast<int>(kk - tap * Cin);
        const int r = static_cast<int>(tap / S), s = static_cast<int>(tap % S);
        const int h = ho + r - ph, w = wo + s - pw;
        if (h >= 0 && h < H && w >= 0 && w < W) x = X[((n * H + h) * W + w) * Cin + c];
      }
      v[i] = x;
    }
    *reinterpret_cast<uint4*>(Aout + m * lda + k0) = *reinterpret_cast<const uint4*>(v);
  }
}

}  // namespace

cudaError_t im2col_i16(const int16_t* X, int16_t* Aout, int64_t lda, int64_t N, int64_t H, int64_t W, int64_t Cin,
                       int64_t R, int64_t S, int64_t ph, int64_t pw, cudaStream_t s) {
  const int64_t Ho = H + 2 * ph - R + 1, Wo = W + 2 * pw - S + 1;
  const int64_t M = N * Ho * Wo, K = R * S * Cin;
  const int64_t total = M * (lda / 8);
  if (total <= 0) return cudaSuccess;
  int64_t blocks = (total + THREADS - 1) / THREADS;
  if (blocks > 152 * 16) blocks = 152 * 16;
  im2col_kernel<<<static_cast<unsigned>(blocks), THREADS, 0, s>>>(
      X, Aout, lda, M, K, static_cast<int>(H), static_cast<int>(W), static_cast<int>(Cin), static_cast<int>(Ho),
      static_cast<int>(Wo), static_cast<int>(S), static_cast<int>(ph), static_cast<int>(pw));
  return cudaGetLastError();
}

}  // namespace gemmi
