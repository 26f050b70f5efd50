// noalloc.cu -- gemm_i16_noalloc: the int16 tensor-core GEMM without any device allocation.
//
// Who needs this: some callers cannot allocate device memory at the moment they run a GEMM.
// An inference server may have handed all free device memory to its own pool at start-up, so
// a cudaMalloc inside the library would fail; a latency-critical loop may not tolerate the
// device-wide synchronisation that growing or freeing a buffer (cudaFree) implies.  The
// regular entry points grow a library-owned workspace on demand; this one does not.
//
// How: the scratch that the int16 path needs (the fp16 limb planes of A and B, plus a device
// status word) lives in one file-scope static __device__ array of fixed size,
// GEMMI_NOALLOC_SCRATCH_BYTES.  Every GPU that loads the library holds that array until the
// process exits.  Host code cannot hand the array's name to a kernel (in host code it is only a
// stand-in, not a device address), so the first call on each device, with that device current,
// looks up its device address once with cudaGetSymbolAddress, clears the status word and caches
// the address; that first call should therefore come before any stream capture.  Nothing here
// calls cudaMalloc, cudaFree or an allocating library routine.
//
// Failure reporting: both kernels of a call (the limb split and the GEMM) bound every pipeline
// wait by GEMMI_OPT_WAIT_TIMEOUT_US and record the first wait that runs out in the status word at
// the start of the array.  The word is sticky: calls do not clear it.  gemmi_device_status() and
// gemmi_device_status_stream() read it beside the library's own status word and clear it.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "gemmi.h"
#include "internal.h"

namespace {

constexpr size_t kScratchBytes = GEMMI_NOALLOC_SCRATCH_BYTES;
constexpr size_t kStatusBytes = 256;  // the device status word, padded to keep the planes 256-byte aligned
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_noalloc_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

int fail(int code, const std::string& msg) {
  gemmi::record_error(msg.c_str());
  return code;
}

bool overlaps(const void* a, size_t abytes, const void* b, size_t bbytes) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
  return a0 < b0 + bbytes && b0 < a0 + abytes;
}

// Bytes spanned by `rows` rows of `cols` elements at pitch `ld` elements, or false on overflow.
bool span_bytes(int64_t rows, int64_t ld, int64_t cols, size_t esize, size_t* out) {
  uint64_t a = 0, b = 0, c = 0;
  if (__builtin_mul_overflow(static_cast<uint64_t>(rows - 1), static_cast<uint64_t>(ld), &a)) return false;
  if (__builtin_add_overflow(a, static_cast<uint64_t>(cols), &b)) return false;
  if (__builtin_mul_overflow(b, static_cast<uint64_t>(esize), &c)) return false;
  *out = static_cast<size_t>(c);
  return true;
}

// The current device (checked to be an sm_103 GPU), its SM count, and the device address of the
// static scratch array there.  The first use on a device looks the address up with that device
// current and clears the status word on `s`.
int scratch_of_current_device(cudaStream_t s, char** scratch, int* sms_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GEMMI_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(GEMMI_EINVAL, "device ordinal out of range");
  int major = 0, minor = 0, sms = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (major != 10 || minor != 3)
    return fail(GEMMI_EARCH, "the current device is not an sm_103 (GB300) GPU; this library has no other path");
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr)
      return fail(GEMMI_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
    // the status word starts at zero (a kernel records only the first failure into a zero word)
    e = cudaMemsetAsync(ptr, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess) return fail(GEMMI_ECUDA, std::string("cudaMemsetAsync(status): ") + cudaGetErrorString(e));
    g_scratch_ptr[dev] = ptr;
  }
  *scratch = static_cast<char*>(g_scratch_ptr[dev]);
  *sms_out = sms;
  return GEMMI_OK;
}

}  // namespace

namespace gemmi {
uint32_t* noalloc_status_word(int dev) {
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  return static_cast<uint32_t*>(g_scratch_ptr[dev]);
}
}  // namespace gemmi

extern "C" int gemm_i16_noalloc(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
                                int64_t ldb, int64_t* C, int64_t ldc, void* stream) {
  // same argument rules as gemm_i16
  if (m < 0 || n < 0 || k < 0) return fail(GEMMI_EINVAL, "negative matrix dimension");
  if (ldc < (n > 1 ? n : 1)) return fail(GEMMI_EINVAL, "ldc < max(1, n)");
  if (lda < (k > 1 ? k : 1)) return fail(GEMMI_EINVAL, "lda < max(1, k)");
  if (ldb < (n > 1 ? n : 1)) return fail(GEMMI_EINVAL, "ldb < max(1, n)");
  if (m == 0 || n == 0) return GEMMI_OK;
  if (C == nullptr) return fail(GEMMI_EINVAL, "C is null");
  if (k == 0) return GEMMI_OK;
  if (A == nullptr || B == nullptr) return fail(GEMMI_EINVAL, "A or B is null");
  if (m > (int64_t(1) << 31) || n > (int64_t(1) << 31) || k > (int64_t(1) << 31))
    return fail(GEMMI_EINVAL, "matrix dimension too large");
  size_t a_bytes = 0, b_bytes = 0, c_bytes = 0;
  if (!span_bytes(m, lda, k, 2, &a_bytes) || !span_bytes(k, ldb, n, 2, &b_bytes) ||
      !span_bytes(m, ldc, n, 8, &c_bytes))
    return fail(GEMMI_EINVAL, "leading dimension too large: the operand's extent overflows 64 bits");
  if (overlaps(C, c_bytes, A, a_bytes) || overlaps(C, c_bytes, B, b_bytes))
    return fail(GEMMI_EINVAL, "C overlaps A or B");

  // the four limb planes must fit in the fixed scratch array
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  const size_t a_plane = round_up(static_cast<size_t>(m) * pitch * 2, 256);
  const size_t b_plane = round_up(static_cast<size_t>(n) * pitch * 2, 256);
  const size_t need = kStatusBytes + 2 * a_plane + 2 * b_plane;
  if (need > kScratchBytes)
    return fail(GEMMI_EINVAL, "gemm_i16_noalloc: this problem needs " + std::to_string(need) +
                                  " bytes of scratch, more than the fixed " + std::to_string(kScratchBytes) +
                                  " (4*(m+n)*roundup(k,8) bytes of limb planes plus 256)");

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* scratch = nullptr;
  int sms = 0;
  int rc = scratch_of_current_device(s, &scratch, &sms);
  if (rc != GEMMI_OK) return rc;
  uint32_t* status = reinterpret_cast<uint32_t*>(scratch);
  const uint64_t timeout_ns = static_cast<uint64_t>(gemmi_get_option(GEMMI_OPT_WAIT_TIMEOUT_US)) * 1000u;
  char* planes = scratch + kStatusBytes;
  gemmi::LimbPlanes pa{{planes, planes + a_plane}, m, pitch};
  gemmi::LimbPlanes pb{{planes + 2 * a_plane, planes + 2 * a_plane + b_plane}, n, pitch};
  // every plane byte the GEMM reads is written here first (pitch padding included), so nothing
  // left over from an earlier call is ever read
  cudaError_t e = gemmi::split_i16(A, lda, B, ldb, m, n, k, pa, pb, s, status, timeout_ns);
  if (e != cudaSuccess) return fail(GEMMI_ECUDA, std::string("limb split launch: ") + cudaGetErrorString(e));
  gemmi::TcGemmArgs ta;
  ta.m = m;
  ta.n = n;
  ta.k = k;
  ta.a = pa;
  ta.b = pb;
  ta.C = C;
  ta.ldc = ldc;
  ta.status = status;
  ta.timeout_ns = timeout_ns;
  ta.num_sms = sms;
  ta.chunk_scale = static_cast<int>(gemmi_get_option(GEMMI_OPT_TC_CHUNK_SCALE));
  ta.group_m = static_cast<int>(gemmi_get_option(GEMMI_OPT_TC_GROUP_M));
  const int64_t hints = gemmi_get_option(GEMMI_OPT_TC_L2_HINTS);
  ta.hint_a = static_cast<int>(hints & 3);
  ta.hint_b = static_cast<int>((hints >> 2) & 3);
  const char* why = "tcgen05 GEMM launch";
  e = gemmi::tc_gemm_i16(ta, s, &why);
  if (e != cudaSuccess) return fail(GEMMI_ECUDA, std::string(why) + ": " + cudaGetErrorString(e));
  return GEMMI_OK;
}

extern "C" int gemmi_noalloc_selftest_wait_timeout(int64_t timeout_us, void* stream) {
  if (timeout_us < 1 || timeout_us > 10000000) return fail(GEMMI_EINVAL, "timeout must be in [1 us, 10 s]");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* scratch = nullptr;
  int sms = 0;
  int rc = scratch_of_current_device(s, &scratch, &sms);
  if (rc != GEMMI_OK) return rc;
  cudaError_t e = gemmi::launch_wait_timeout_probe(reinterpret_cast<uint32_t*>(scratch),
                                                   static_cast<uint64_t>(timeout_us) * 1000u, s);
  if (e != cudaSuccess) return fail(GEMMI_ECUDA, std::string("wait probe launch: ") + cudaGetErrorString(e));
  return GEMMI_OK;
}
