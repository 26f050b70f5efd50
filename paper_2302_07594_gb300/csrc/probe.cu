// probe.cu -- gemmi_stream_read_probe: the read-bandwidth floor of the skinny-M GEMM.
//
// A measurement aid with no counterpart in the paper.  It reads a k x n int16 matrix exactly the
// way the skinny kernel (skinny.cu) streams B -- the same grid of 512-column blocks by reduction
// ranges, the same 32-row x 64-column TMA boxes with the 128-byte swizzle, the same ring of four
// 32 KB stages per CTA and programmatic dependent launch -- and does nothing with the data: one
// thread per CTA waits for each stage and hands it straight back.  Timed like the skinny GEMM, it
// is the time one such launch needs to move B from HBM into shared memory, the floor that any
// kernel streaming B this way sits on.  Every wait is bounded; a wait that runs out is recorded in
// the status word.
#include <cuda.h>

#include "internal.h"
#include "ptx.cuh"

namespace gemmi {
namespace {

constexpr int JB = 512;
constexpr int BOX_J = 64;
constexpr int NBOX = JB / BOX_J;
constexpr int KS = 32;
constexpr int STAGES = 4;
constexpr int STAGE_BYTES = KS * JB * 2;
constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES;

__global__ void __launch_bounds__(64, 1)
stream_probe_kernel(const __grid_constant__ CUtensorMap map, int per, int total, uint64_t timeout_ns, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t bars[2 * STAGES];
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * STAGES;
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  const int st0 = blockIdx.y * per;
  const int st1 = st0 + per < total ? st0 + per : total;
  const int nst = st1 > st0 ? st1 - st0 : 0;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (lane != 0) return;
  if (warp == 0) {
    tma_prefetch_desc(&map);
    for (int i = 0; i < nst; ++i) {
      const int s = i % STAGES;
      const uint32_t par = (i / STAGES) & 1;
      if (!bounded_wait(empty0 + 8 * s, par ^ 1u, timeout_ns)) {
        report_status(status, 4, 31);
        return;
      }
      mbar_arrive_expect_tx(full0 + 8 * s, STAGE_BYTES);
      for (int b = 0; b < NBOX; ++b)
        tma_load_2d(smem_u32(smem + s * STAGE_BYTES + b * (KS * BOX_J * 2)), &map, full0 + 8 * s,
                    static_cast<int32_t>(blockIdx.x * JB + b * BOX_J), (st0 + i) * KS);
    }
  } else {
    // the consumer thread returns only once every stage has landed, so the CTA never exits with a
    // copy in flight
    for (int i = 0; i < nst; ++i) {
      const int s = i % STAGES;
      const uint32_t par = (i / STAGES) & 1;
      if (!bounded_wait(full0 + 8 * s, par, timeout_ns)) {
        report_status(status, 4, 32);
        return;
      }
      mbar_arrive(empty0 + 8 * s);
    }
  }
}

}  // namespace

cudaError_t stream_read_probe(const int16_t* B, int64_t k, int64_t n, int64_t ldb, int num_sms, uint32_t* status,
                              uint64_t timeout_ns, cudaStream_t s, const char** why) {
  CUtensorMap map;
  if (!encode_tensor_map_2d(&map, 0, B, static_cast<uint64_t>(n), static_cast<uint64_t>(k),
                            static_cast<uint64_t>(ldb) * 2, BOX_J, KS, 128, why))
    return cudaErrorInvalidValue;
  // the skinny kernel's grid for m <= 16: about one CTA per SM, at least 4 stages per CTA
  const int64_t nj = (n + JB - 1) / JB;
  const int64_t total = (k + KS - 1) / KS;
  int64_t ksplit = num_sms / nj;
  if (ksplit < 1) ksplit = 1;
  const int64_t cap = total / 4 > 0 ? total / 4 : 1;
  if (ksplit > cap) ksplit = cap;
  const int64_t min_split = (total + 31) / 32;
  if (ksplit < min_split) ksplit = min_split;
  if (ksplit > total) ksplit = total;
  const int64_t per = (total + ksplit - 1) / ksplit;
  ksplit = (total + per - 1) / per;
  if (nj > 0x7FFFFFFF || ksplit > 65535 || total > 0x7FFFFFFF) {
    *why = "read probe grid too large";
    return cudaErrorInvalidValue;
  }
  static bool attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_done[dev]) {
    const cudaError_t e =
        cudaFuncSetAttribute(stream_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(SMEM));
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) attr_done[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(nj), static_cast<unsigned>(ksplit), 1);
  cfg.blockDim = dim3(64);
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stream_probe_kernel, map, static_cast<int>(per), static_cast<int>(total), timeout_ns,
                            status);
}

}  // namespace gemmi
