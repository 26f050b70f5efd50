// api.cu -- the C ABI of include/gemmi.h: argument checks, workspace, dispatch.
//
// Dispatch (all paths bit-exact, see the kernels' headers):
//   int16, m <= skinny limit (16) : skinny.cu   (B streamed once, tensor-core limb products)
//   int16, n <= 64, A TMA-readable: gemm_fused.cu (A split on chip; B's planes from split.cu)
//   int16 / int8, otherwise       : split.cu (operands -> fp16 limb planes), then gemm_pair.cu
//                                   (tcgen05 on SM pairs) when C takes 16-byte reductions, else
//                                   gemm_tc.cu (one SM per tile)
//   *_host with m >= 1024         : the same, pipelined over row panels on copy streams
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "gemmi.h"
#include "internal.h"
#include "ptx.cuh"

namespace {

using gemmi::LimbPlanes;

thread_local std::string t_error;

int set_error(int code, const std::string& msg) {
  t_error = msg;
  return code;
}

int cuda_error(cudaError_t e, const char* where) {
  return set_error(GEMMI_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

constexpr int kMaxDevices = 64;
constexpr size_t kAlign = 256;

struct DeviceState {
  bool ready = false;
  bool arch_ok = false;
  int sm_count = 0;
  uint32_t* status = nullptr;   // device status word
  void* ws = nullptr;           // limb planes / aligned copies
  size_t ws_bytes = 0;
  void* host_buf = nullptr;     // device staging for the *_host entry points
  size_t host_buf_bytes = 0;
  void* sum_buf = nullptr;      // exact int64 sums for the requantising entry point
  size_t sum_buf_bytes = 0;
  void* conv_buf = nullptr;     // explicitly lowered convolution operand (fallback path)
  size_t conv_buf_bytes = 0;
  cudaEvent_t last_use = nullptr;
  cudaStream_t last_stream = nullptr;
  cudaStream_t h2d = nullptr;          // copy streams of the pipelined host-buffer path
  cudaStream_t d2h = nullptr;
  cudaEvent_t pipe_ev[12] = {};
  bool used = false;
  uint32_t last_detail = 0;
};

std::mutex g_mutex;
DeviceState g_dev[kMaxDevices];

// Optional per-kernel timing with CUDA events recorded on the launching stream.
struct KernelTimer {
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending;
  std::vector<cudaEvent_t> pool;
  double total_ms = 0.0;
  int64_t launches = 0;
};
bool g_timing = false;
KernelTimer g_timers[GEMMI_KERNEL_COUNT];

cudaEvent_t timer_event(KernelTimer& t) {
  if (!t.pool.empty()) {
    cudaEvent_t e = t.pool.back();
    t.pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

bool is_capturing(cudaStream_t s);

// Records the start event of a timed launch (returns null when timing is off or the stream is
// being captured: an event recorded into a graph cannot be timed from the host).
cudaEvent_t timer_begin(int kind, cudaStream_t s) {
  if (!g_timing || is_capturing(s)) return nullptr;
  cudaEvent_t e = timer_event(g_timers[kind]);
  cudaEventRecord(e, s);
  return e;
}

void timer_end(int kind, cudaEvent_t start, cudaStream_t s) {
  if (start == nullptr) return;
  cudaEvent_t e = timer_event(g_timers[kind]);
  cudaEventRecord(e, s);
  g_timers[kind].pending.emplace_back(start, e);
}

void timer_collect(KernelTimer& t) {
  for (auto& pr : t.pending) {
    cudaEventSynchronize(pr.second);
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess) {
      t.total_ms += ms;
      t.launches += 1;
    }
    t.pool.push_back(pr.first);
    t.pool.push_back(pr.second);
  }
  t.pending.clear();
}
cudaStream_t g_stream = nullptr;
int64_t g_skinny_max_m = 16;
int64_t g_timeout_us = 4000000;
int64_t g_skinny_ksplit = 0;
int64_t g_tc_chunk_scale = 2;
int64_t g_tc_group_m = 0;  // 0: automatic (raster_band())
int64_t g_tc_l2_hints = 0;
int64_t g_fused_max_n = 64;
int64_t g_tc_pair = 1;
int64_t g_split_ahead = 1;  // overlapped A split in the int16 pair kernel
int64_t g_conv_rows = 1;    // direct kernel for "same" convolutions with 64 input channels
// up to 2^28 multiply-adds the one-launch skinny path measured faster than split + tensor-core GEMM
// for every m <= 256 tried (4.9 against 11.0 us at 256^3, 12.1 against 14.0 us at 256 x 1024^2);
// at 2^29 they tie (256 x 2048 x 1024) and beyond the tensor cores win
int64_t g_small_max_macs = int64_t{1} << 28;
int64_t g_karatsuba = 0;

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Height of the tile raster's bands (in tile rows).  Automatic: 8 for the kernels on fp16 limb
// planes -- about sqrt(76) for the 76 SM pairs' concurrent 128 x 128 tiles, the fewest distinct A
// and B panels per wave; at int16 8192^3 it measured 1.2 % faster than 16, at burst clocks and
// under the power cap alike (less DRAM traffic) -- and 16 for int4, where 16 measured 0.5 % faster.
int raster_band(bool int4) {
  if (g_tc_group_m > 0) return static_cast<int>(g_tc_group_m);
  return int4 ? 16 : 8;
}

// Current device's state, initialised on first use (caller holds g_mutex).
int device_state(DeviceState** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(GEMMI_EINVAL, "device ordinal out of range");
  DeviceState& d = g_dev[dev];
  if (!d.ready) {
    cudaDeviceProp prop;
    e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetDeviceProperties");
    d.arch_ok = prop.major == 10 && prop.minor == 3;
    d.sm_count = prop.multiProcessorCount;
    if (d.arch_ok) {
      e = cudaMalloc(&d.status, 256);
      if (e != cudaSuccess) return set_error(GEMMI_ENOMEM, "cannot allocate the device status word");
      e = cudaMemset(d.status, 0, 256);
      if (e != cudaSuccess) return cuda_error(e, "cudaMemset(status)");
      e = cudaEventCreateWithFlags(&d.last_use, cudaEventDisableTiming);
      if (e != cudaSuccess) return cuda_error(e, "cudaEventCreate");
    }
    d.ready = true;
  }
  if (!d.arch_ok)
    return set_error(GEMMI_EARCH, "the current device is not an sm_103 (GB300) GPU; this library has no other path");
  *out = &d;
  return GEMMI_OK;
}

// Grows a device buffer to at least `bytes` (synchronising the device before freeing the old one).
int ensure_buffer(void** buf, size_t* have, size_t bytes) {
  if (*have >= bytes) return GEMMI_OK;
  if (*buf != nullptr) {
    cudaDeviceSynchronize();
    cudaFree(*buf);
    *buf = nullptr;
    *have = 0;
  }
  const size_t want = round_up(bytes, size_t(2) << 20);
  if (cudaMalloc(buf, want) != cudaSuccess) {
    cudaGetLastError();
    *buf = nullptr;
    return set_error(GEMMI_ENOMEM, "cannot allocate " + std::to_string(want) + " bytes of device workspace");
  }
  *have = want;
  return GEMMI_OK;
}

bool is_capturing(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &st) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return st != cudaStreamCaptureStatusNone;
}

// Orders this call's use of the workspace after the previous call's (which may be on another
// stream).  Inside a stream capture the library records and waits on no event of its own: the
// captured graph orders its nodes, and ordering graph launches against other work that uses
// the same workspace is the caller's (as for any captured work that shares memory).
int begin_workspace_use(DeviceState& d, cudaStream_t s) {
  if (d.used && d.last_stream != s && !is_capturing(s)) {
    cudaError_t e = cudaStreamWaitEvent(s, d.last_use, 0);
    if (e != cudaSuccess) return cuda_error(e, "cudaStreamWaitEvent");
  }
  return GEMMI_OK;
}

int end_workspace_use(DeviceState& d, cudaStream_t s) {
  if (is_capturing(s)) return GEMMI_OK;  // the event would belong to the graph, not to the stream
  cudaError_t e = cudaEventRecord(d.last_use, s);
  if (e != cudaSuccess) return cuda_error(e, "cudaEventRecord");
  d.last_stream = s;
  d.used = true;
  return GEMMI_OK;
}

bool overlaps(const void* a, size_t abytes, const void* b, size_t bbytes) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
  return a0 < b0 + bbytes && b0 < a0 + abytes;
}

// Bytes spanned by `rows` rows (rows >= 1) of `cols` elements at pitch `ld` elements, or false on
// 64-bit overflow (a huge leading dimension).
bool span_bytes(int64_t rows, int64_t ld, int64_t cols, size_t esize, size_t* out) {
  uint64_t a = 0, b = 0, c = 0;
  if (__builtin_mul_overflow(static_cast<uint64_t>(rows - 1), static_cast<uint64_t>(ld), &a)) return false;
  if (__builtin_add_overflow(a, static_cast<uint64_t>(cols), &b)) return false;
  if (__builtin_mul_overflow(b, static_cast<uint64_t>(esize), &c)) return false;
  *out = static_cast<size_t>(c);
  return true;
}

// Checks shared by every entry point.  Returns -1 to proceed, or a status to return.
int check_args(int64_t m, int64_t n, int64_t k, const void* A, int64_t lda, const void* B, int64_t ldb,
               const void* C, int64_t ldc, size_t op_size, size_t c_size) {
  if (m < 0 || n < 0 || k < 0) return set_error(GEMMI_EINVAL, "negative matrix dimension");
  if (ldc < std::max<int64_t>(1, n)) return set_error(GEMMI_EINVAL, "ldc < max(1, n)");
  if (lda < std::max<int64_t>(1, k)) return set_error(GEMMI_EINVAL, "lda < max(1, k)");
  if (ldb < std::max<int64_t>(1, n)) return set_error(GEMMI_EINVAL, "ldb < max(1, n)");
  if (m == 0 || n == 0) return GEMMI_OK;
  if (C == nullptr) return set_error(GEMMI_EINVAL, "C is null");
  if (k == 0) return GEMMI_OK;
  if (A == nullptr || B == nullptr) return set_error(GEMMI_EINVAL, "A or B is null");
  if (m > (int64_t(1) << 40) || n > (int64_t(1) << 31) || k > (int64_t(1) << 31))
    return set_error(GEMMI_EINVAL, "matrix dimension too large");
  size_t a_bytes = 0, b_bytes = 0, c_bytes = 0;
  if (!span_bytes(m, lda, k, op_size, &a_bytes) || !span_bytes(k, ldb, n, op_size, &b_bytes) ||
      !span_bytes(m, ldc, n, c_size, &c_bytes))
    return set_error(GEMMI_EINVAL, "leading dimension too large: the operand's extent overflows 64 bits");
  if (overlaps(C, c_bytes, A, a_bytes) || overlaps(C, c_bytes, B, b_bytes))
    return set_error(GEMMI_EINVAL, "C overlaps A or B");
  return -1;
}

uint64_t timeout_ns() { return static_cast<uint64_t>(g_timeout_us) * 1000u; }

struct Layout {
  size_t a0, a1, b0, b1, total;
};

Layout plane_layout(int64_t m, int64_t n, int64_t pitch, int nl) {
  Layout L{};
  const size_t a_plane = round_up(static_cast<size_t>(m) * pitch * 2, kAlign);
  const size_t b_plane = round_up(static_cast<size_t>(n) * pitch * 2, kAlign);
  L.a0 = 0;
  L.a1 = nl >= 2 ? a_plane : 0;
  L.b0 = a_plane * nl;
  L.b1 = nl >= 2 ? L.b0 + b_plane : L.b0;
  L.total = a_plane * nl + b_plane * nl;
  return L;
}

// The Karatsuba variant (GEMMI_OPT_KARATSUBA): h, l and s = h + l planes of both operands in the
// workspace, then the three-product kernel on one SM per tile.
int run_karatsuba(DeviceState& d, int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
                  int64_t ldb, int64_t* C, int64_t ldc, cudaStream_t s) {
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  const size_t a_plane = round_up(static_cast<size_t>(m) * pitch * 2, kAlign);
  const size_t b_plane = round_up(static_cast<size_t>(n) * pitch * 2, kAlign);
  int rc = ensure_buffer(&d.ws, &d.ws_bytes, 3 * (a_plane + b_plane));
  if (rc != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
  char* ws = static_cast<char*>(d.ws);
  LimbPlanes pa{{ws, ws + a_plane, ws + 2 * a_plane}, m, pitch};
  char* wb = ws + 3 * a_plane;
  LimbPlanes pb{{wb, wb + b_plane, wb + 2 * b_plane}, n, pitch};
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SPLIT, s);
  cudaError_t e = gemmi::split_i16(A, lda, B, ldb, m, n, k, pa, pb, s, d.status, timeout_ns());
  if (e == cudaSuccess) e = gemmi::limb_sum_planes(pa, pb, d.sm_count, s);
  timer_end(GEMMI_KERNEL_SPLIT, t0, s);
  if (e != cudaSuccess) return cuda_error(e, "limb split launch");
  gemmi::TcGemmArgs ta;
  ta.m = m;
  ta.n = n;
  ta.k = k;
  ta.a = pa;
  ta.b = pb;
  ta.C = C;
  ta.ldc = ldc;
  ta.status = d.status;
  ta.timeout_ns = timeout_ns();
  ta.num_sms = d.sm_count;
  ta.chunk_scale = static_cast<int>(g_tc_chunk_scale);
  ta.group_m = raster_band(false);
  ta.hint_a = static_cast<int>(g_tc_l2_hints & 3);
  ta.hint_b = static_cast<int>((g_tc_l2_hints >> 2) & 3);
  const char* why = "tcgen05 Karatsuba GEMM launch";
  cudaEvent_t t1 = timer_begin(GEMMI_KERNEL_TC_KARATSUBA, s);
  e = gemmi::tc_gemm_i16_karatsuba(ta, s, &why);
  timer_end(GEMMI_KERNEL_TC_KARATSUBA, t1, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  return end_workspace_use(d, s);
}

// The tensor-core path: split A (and B, unless `packed_b` already holds its planes) into the
// workspace, then run the tcgen05 GEMM.
// The narrow-n int16 path: only B is split (unless packed); A is read raw by the kernel, which
// splits it on chip.  TMA reads A, so its base must be 16-byte aligned and lda a multiple of 8;
// the kernel adds into C with 64-bit reductions, so C must be 8-byte aligned.
bool fused_applies(int nl, int64_t n, const void* A, int64_t lda, const void* C) {
  return nl == 2 && n <= g_fused_max_n && reinterpret_cast<uintptr_t>(A) % 16 == 0 && lda % 8 == 0 &&
         reinterpret_cast<uintptr_t>(C) % 8 == 0;
}

// A stride-1 convolution whose output has the input's height and width, read as an implicit
// IM2COL operand by the fused kernel (see FusedArgs).
struct ConvShape {
  int64_t N, H, W, Cin, S, ph, pw;
};

int run_fused(DeviceState& d, int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
              int64_t ldb, int64_t* C, int64_t ldc, cudaStream_t s, const LimbPlanes* packed_b,
              const ConvShape* conv = nullptr) {
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  const bool split_b = packed_b == nullptr;
  LimbPlanes pb{};
  if (split_b) {
    const Layout L = plane_layout(0, n, pitch, 2);
    int rc = ensure_buffer(&d.ws, &d.ws_bytes, L.total);
    if (rc != GEMMI_OK) return rc;
    if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
    char* ws = static_cast<char*>(d.ws);
    pb = LimbPlanes{{ws + L.b0, ws + L.b1}, n, pitch};
    const LimbPlanes none{{nullptr, nullptr}, 0, pitch};
    cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SPLIT, s);
    const cudaError_t e = gemmi::split_i16(nullptr, lda, B, ldb, m, n, k, none, pb, s, d.status, timeout_ns());
    timer_end(GEMMI_KERNEL_SPLIT, t0, s);
    if (e != cudaSuccess) return cuda_error(e, "limb split launch");
  } else {
    pb = *packed_b;
  }
  gemmi::FusedArgs fa;
  fa.m = m;
  fa.n = n;
  fa.k = k;
  fa.A = A;
  fa.lda = lda;
  fa.b = pb;
  fa.C = C;
  fa.ldc = ldc;
  fa.status = d.status;
  fa.timeout_ns = timeout_ns();
  fa.num_sms = d.sm_count;
  fa.chunk_scale = static_cast<int>(g_tc_chunk_scale);
  fa.group_m = raster_band(false);
  if (conv != nullptr) {
    fa.conv = 1;
    fa.conv_pixels = conv->N * conv->H * conv->W;
    fa.conv_cin = static_cast<int>(conv->Cin);
    fa.conv_h = static_cast<int>(conv->H);
    fa.conv_w = static_cast<int>(conv->W);
    fa.conv_s = static_cast<int>(conv->S);
    fa.conv_ph = static_cast<int>(conv->ph);
    fa.conv_pw = static_cast<int>(conv->pw);
  }
  const char* why = "fused tcgen05 GEMM launch";
  cudaEvent_t t1 = timer_begin(GEMMI_KERNEL_FUSED_I16, s);
  const cudaError_t e = gemmi::tc_gemm_fused_i16(fa, s, &why);
  timer_end(GEMMI_KERNEL_FUSED_I16, t1, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  return split_b ? end_workspace_use(d, s) : GEMMI_OK;
}

// The direct convolution (conv_rows.cu): the lowered weights (K x Cout) split once into limb planes
// in the workspace, then one launch over tiles of output rows.
int run_conv_rows(DeviceState& d, int64_t N, int64_t H, int64_t W, int64_t Cout, int64_t R, int64_t S,
                  const int16_t* X, const int16_t* Wt, int64_t* Y, cudaStream_t s) {
  const int64_t k = R * S * 64;
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  const Layout L = plane_layout(0, Cout, pitch, 2);
  int rc = ensure_buffer(&d.ws, &d.ws_bytes, L.total);
  if (rc != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
  char* ws = static_cast<char*>(d.ws);
  const LimbPlanes pb{{ws + L.b0, ws + L.b1}, Cout, pitch};
  const LimbPlanes none{{nullptr, nullptr}, 0, pitch};
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SPLIT, s);
  cudaError_t e = gemmi::split_i16(nullptr, k, Wt, Cout, 0, Cout, k, none, pb, s, d.status, timeout_ns());
  timer_end(GEMMI_KERNEL_SPLIT, t0, s);
  if (e != cudaSuccess) return cuda_error(e, "limb split launch");
  gemmi::ConvRowsArgs ca;
  ca.X = X;
  ca.N = N;
  ca.H = H;
  ca.W = W;
  ca.R = R;
  ca.S = S;
  ca.cout = Cout;
  ca.b = pb;
  ca.Y = Y;
  ca.status = d.status;
  ca.timeout_ns = timeout_ns();
  ca.num_sms = d.sm_count;
  ca.chunk_scale = static_cast<int>(g_tc_chunk_scale);
  const char* why = "direct convolution launch";
  cudaEvent_t t1 = timer_begin(GEMMI_KERNEL_CONV_ROWS, s);
  e = gemmi::conv_rows_i16(ca, s, &why);
  timer_end(GEMMI_KERNEL_CONV_ROWS, t1, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  return end_workspace_use(d, s);
}

int run_tc(DeviceState& d, int nl, int64_t m, int64_t n, int64_t k, const void* A, int64_t lda, const void* B,
           int64_t ldb, void* C, int64_t ldc, cudaStream_t s, const LimbPlanes* packed_b = nullptr) {
  if (fused_applies(nl, n, A, lda, C))
    return run_fused(d, m, n, k, static_cast<const int16_t*>(A), lda, static_cast<const int16_t*>(B), ldb,
                     static_cast<int64_t*>(C), ldc, s, packed_b);
  if (nl == 2 && g_karatsuba != 0 && packed_b == nullptr)
    return run_karatsuba(d, m, n, k, static_cast<const int16_t*>(A), lda, static_cast<const int16_t*>(B), ldb,
                         static_cast<int64_t*>(C), ldc, s);
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  // SM pairs (cta_group::2) unless switched off or C cannot take 16-byte bulk reductions
  const int64_t esz = nl == 2 ? 8 : 4;
  const bool pair = g_tc_pair != 0 && reinterpret_cast<uintptr_t>(C) % 16 == 0 && (ldc * esz) % 16 == 0;
  // Overlapped A split (int16 on SM pairs): the split launch converts B and only the row panels
  // of A that the first wave of tiles reads; the pair kernel's splitter warps convert the rest.
  const int64_t m_panels = (m + 127) / 128;
  int ahead_first = 0;
  if (nl == 2 && pair && g_split_ahead != 0 && reinterpret_cast<uintptr_t>(A) % 16 == 0 && lda % 8 == 0 &&
      k % 8 == 0 && m_panels < (int64_t{1} << 24)) {
    ahead_first = gemmi::pair_first_wave_panels(m, n, raster_band(false), d.sm_count);
    if (ahead_first >= m_panels) ahead_first = 0;
  }
  const bool ahead = ahead_first > 0;
  const Layout L = plane_layout(m, packed_b ? 0 : n, pitch, nl);
  const size_t ahead_off = round_up(L.total, kAlign);
  const size_t ahead_bytes = ahead ? static_cast<size_t>(2 + m_panels) * 4 : 0;
  int rc = ensure_buffer(&d.ws, &d.ws_bytes, ahead_off + ahead_bytes);
  if (rc != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
  char* ws = static_cast<char*>(d.ws);
  LimbPlanes pa{{ws + L.a0, ws + L.a1}, m, pitch};
  LimbPlanes pb = packed_b ? *packed_b : LimbPlanes{{ws + L.b0, ws + L.b1}, n, pitch};
  if (packed_b) B = nullptr;  // nothing to convert for B
  uint32_t* ahead_words = ahead ? reinterpret_cast<uint32_t*>(ws + ahead_off) : nullptr;
  cudaError_t e;
  if (ahead) {
    e = cudaMemsetAsync(ahead_words, 0, ahead_bytes, s);
    if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync(split counters)");
  }
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SPLIT, s);
  if (nl == 2) {
    const int64_t m_split = ahead ? std::min<int64_t>(m, static_cast<int64_t>(ahead_first) * 128) : m;
    e = gemmi::split_i16(static_cast<const int16_t*>(A), lda, static_cast<const int16_t*>(B), ldb, m_split, n, k, pa,
                         pb, s, d.status, timeout_ns());
  } else {
    e = gemmi::convert_i8(static_cast<const int8_t*>(A), lda, static_cast<const int8_t*>(B), ldb, m, n, k, pa, pb, s,
                          d.status, timeout_ns());
  }
  timer_end(GEMMI_KERNEL_SPLIT, t0, s);
  if (e != cudaSuccess) return cuda_error(e, "limb split launch");
  gemmi::TcGemmArgs ta;
  ta.m = m;
  ta.n = n;
  ta.k = k;
  ta.a = pa;
  ta.b = pb;
  ta.C = C;
  ta.ldc = ldc;
  ta.status = d.status;
  ta.timeout_ns = timeout_ns();
  ta.num_sms = d.sm_count;
  ta.chunk_scale = static_cast<int>(g_tc_chunk_scale);
  ta.group_m = raster_band(false);
  ta.hint_a = static_cast<int>(g_tc_l2_hints & 3);
  ta.hint_b = static_cast<int>((g_tc_l2_hints >> 2) & 3);
  if (ahead) {
    ta.a_raw = static_cast<const int16_t*>(A);
    ta.lda = lda;
    ta.ahead = ahead_words;
    ta.ahead_first = ahead_first;
  }
  const char* why = "tcgen05 GEMM launch";
  const int kind = pair ? (nl == 2 ? (ahead ? GEMMI_KERNEL_TC_PAIR_I16_AHEAD : GEMMI_KERNEL_TC_PAIR_I16)
                               : GEMMI_KERNEL_TC_PAIR_I8)
                        : (nl == 2 ? GEMMI_KERNEL_TC_I16 : GEMMI_KERNEL_TC_I8);
  cudaEvent_t t1 = timer_begin(kind, s);
  if (pair) e = nl == 2 ? gemmi::tc_pair_gemm_i16(ta, s, &why) : gemmi::tc_pair_gemm_i8(ta, s, &why);
  else e = nl == 2 ? gemmi::tc_gemm_i16(ta, s, &why) : gemmi::tc_gemm_i8(ta, s, &why);
  timer_end(kind, t1, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  return end_workspace_use(d, s);
}

int run_skinny(DeviceState& d, int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
               int64_t ldb, int64_t* C, int64_t ldc, cudaStream_t s) {
  // TMA needs 16-byte aligned row starts of B; a B without them is re-pitched into the workspace
  // (A is read with plain loads)
  const bool b_ok = reinterpret_cast<uintptr_t>(B) % 16 == 0 && (ldb * 2) % 16 == 0;
  const bool a_ok = true;
  const int16_t* Bs = B;
  const int16_t* As = A;
  int64_t ldbs = ldb, ldas = lda;
  const bool used_ws = !a_ok || !b_ok;
  int rc;
  if (used_ws) {
    const int64_t ldb_new = static_cast<int64_t>(round_up(static_cast<size_t>(n), 8));
    const int64_t lda_new = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
    const size_t b_bytes = b_ok ? 0 : round_up(static_cast<size_t>(k) * ldb_new * 2, kAlign);
    const size_t a_bytes = a_ok ? 0 : round_up(static_cast<size_t>(m) * lda_new * 2, kAlign);
    if ((rc = ensure_buffer(&d.ws, &d.ws_bytes, a_bytes + b_bytes)) != GEMMI_OK) return rc;
    if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
    char* ws = static_cast<char*>(d.ws);
    if (!b_ok) {
      cudaError_t e = cudaMemcpy2DAsync(ws, ldb_new * 2, B, ldb * 2, n * 2, k, cudaMemcpyDeviceToDevice, s);
      if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy2DAsync(B)");
      Bs = reinterpret_cast<const int16_t*>(ws);
      ldbs = ldb_new;
    }
    if (!a_ok) {
      cudaError_t e = cudaMemcpy2DAsync(ws + b_bytes, lda_new * 2, A, lda * 2, k * 2, m, cudaMemcpyDeviceToDevice, s);
      if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy2DAsync(A)");
      As = reinterpret_cast<const int16_t*>(ws + b_bytes);
      ldas = lda_new;
    }
  }
  gemmi::SkinnyArgs sa;
  sa.m = m;
  sa.n = n;
  sa.k = k;
  sa.A = As;
  sa.lda = ldas;
  sa.B = Bs;
  sa.ldb = ldbs;
  sa.C = C;
  sa.ldc = ldc;
  sa.status = d.status;
  sa.timeout_ns = timeout_ns();
  sa.num_sms = d.sm_count;
  sa.ksplit = static_cast<int>(g_skinny_ksplit);
  const char* why = "skinny GEMM launch";
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SKINNY, s);
  cudaError_t e = gemmi::skinny_gemm_i16(sa, s, &why);
  timer_end(GEMMI_KERNEL_SKINNY, t0, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  return used_ws ? end_workspace_use(d, s) : GEMMI_OK;
}

int gemm_i16_locked(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb,
                    int64_t* C, int64_t ldc, cudaStream_t s) {
  const int pre = check_args(m, n, k, A, lda, B, ldb, C, ldc, 2, 8);
  if (pre >= 0) return pre;
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  // small m, or a small problem of at most 256 rows: one launch of the skinny kernel (B split on
  // chip, one grid row per 16 rows of A) beats the split + tensor-core pair of launches
  const bool small = g_skinny_max_m > 0 && m <= 256 && m * n <= g_small_max_macs / std::max<int64_t>(k, 1);
  if (m <= g_skinny_max_m || small) return run_skinny(*d, m, n, k, A, lda, B, ldb, C, ldc, s);
  return run_tc(*d, 2, m, n, k, A, lda, B, ldb, C, ldc, s);
}

// The paper's micro-kernel output (Section 5.2): C16 += srs(A*B, shift).  The exact product goes
// into a zeroed int64 scratch through the regular int16 paths, then requant.cu applies the
// shift (rounding half up), the int16 saturation and the wrapping 16-bit addition.
int gemm_i16_srs_locked(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
                        int64_t ldb, int16_t* C, int64_t ldc, int shift, cudaStream_t s) {
  if (shift < 0 || shift > 62) return set_error(GEMMI_EINVAL, "shift must be in [0, 62]");
  const int pre = check_args(m, n, k, A, lda, B, ldb, C, ldc, 2, 2);
  if (pre >= 0) return pre;  // includes m == 0, n == 0 and k == 0 (srs of an empty sum adds 0)
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  const int64_t lds = static_cast<int64_t>(round_up(static_cast<size_t>(n), 8));
  const size_t bytes = static_cast<size_t>(m) * static_cast<size_t>(lds) * 8;
  if ((rc = ensure_buffer(&d->sum_buf, &d->sum_buf_bytes, bytes)) != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(*d, s)) != GEMMI_OK) return rc;
  int64_t* S = static_cast<int64_t*>(d->sum_buf);
  cudaError_t e = cudaMemsetAsync(S, 0, bytes, s);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync(sums)");
  rc = m <= g_skinny_max_m ? run_skinny(*d, m, n, k, A, lda, B, ldb, S, lds, s)
                           : run_tc(*d, 2, m, n, k, A, lda, B, ldb, S, lds, s);
  if (rc != GEMMI_OK) return rc;
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SRS, s);
  e = gemmi::srs_add_i16(S, lds, C, ldc, m, n, shift, s);
  timer_end(GEMMI_KERNEL_SRS, t0, s);
  if (e != cudaSuccess) return cuda_error(e, "srs launch");
  return end_workspace_use(*d, s);
}

// A convolution through the lowered GEMM (Sections 2 and 3 of the paper: the IM2COL transform
// casts the convolution as one large GEMM, and the transform may be applied on the fly as part of
// the packing).  "Same" stride-1 convolutions with Cin % 64 == 0 run the fused kernel straight
// from the NHWC tensor (each 64-wide K block is one filter tap of 64 channels, a shifted box of
// 128 pixels, with the converters zeroing the taps that fall outside the image); other shapes
// materialise the lowered matrix with im2col.cu and run the regular int16 path.
int conv2d_locked(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t R, int64_t S, int64_t ph,
                  int64_t pw, const int16_t* X, const int16_t* Wt, int64_t* Y, cudaStream_t s) {
  if (N < 0 || H < 0 || W < 0 || Cin < 0 || Cout < 0) return set_error(GEMMI_EINVAL, "negative tensor dimension");
  if (R < 1 || S < 1) return set_error(GEMMI_EINVAL, "filter height and width must be at least 1");
  if (ph < 0 || pw < 0) return set_error(GEMMI_EINVAL, "negative padding");
  const int64_t Ho = H + 2 * ph - R + 1, Wo = W + 2 * pw - S + 1;
  if (Ho < 0 || Wo < 0) return set_error(GEMMI_EINVAL, "filter larger than the padded input");
  const int64_t M = N * Ho * Wo, K = R * S * Cin;
  if (M == 0 || Cout == 0 || K == 0) return GEMMI_OK;
  if (X == nullptr || Wt == nullptr || Y == nullptr) return set_error(GEMMI_EINVAL, "X, Wt or Y is null");
  if (N > (int64_t(1) << 31) || H > (int64_t(1) << 20) || W > (int64_t(1) << 20) || Cin > (int64_t(1) << 20) ||
      Cout > (int64_t(1) << 20) || R > 64 || S > 64 || M > (int64_t(1) << 40) || K > (int64_t(1) << 31))
    return set_error(GEMMI_EINVAL, "tensor dimension too large");
  const size_t x_bytes = static_cast<size_t>(N * H * W * Cin) * 2;
  const size_t w_bytes = static_cast<size_t>(K * Cout) * 2;
  const size_t y_bytes = static_cast<size_t>(M * Cout) * 8;
  if (overlaps(Y, y_bytes, X, x_bytes) || overlaps(Y, y_bytes, Wt, w_bytes))
    return set_error(GEMMI_EINVAL, "Y overlaps X or Wt");
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  int geo[4];
  if (g_conv_rows != 0 && Ho == H && Wo == W && Cin == 64 && M > g_skinny_max_m && Cout % 2 == 0 && Cout <= 64 &&
      N * H * W < (int64_t(1) << 31) && reinterpret_cast<uintptr_t>(X) % 16 == 0 &&
      reinterpret_cast<uintptr_t>(Y) % 16 == 0 &&
      gemmi::conv_rows_geometry(W, R, S, static_cast<int>(g_tc_chunk_scale), &geo[0], &geo[1], &geo[2], &geo[3]))
    return run_conv_rows(*d, N, H, W, Cout, R, S, X, Wt, Y, s);
  const bool implicit = Ho == H && Wo == W && Cin % 64 == 0 && M > g_skinny_max_m && Cout <= 256 &&
                        N * H * W < (int64_t(1) << 31) && reinterpret_cast<uintptr_t>(X) % 16 == 0 &&
                        reinterpret_cast<uintptr_t>(Y) % 8 == 0;
  if (implicit) {
    const ConvShape cs{N, H, W, Cin, S, ph, pw};
    return run_fused(*d, M, Cout, K, X, K, Wt, Cout, Y, Cout, s, nullptr, &cs);
  }
  // explicit lowering into library-owned memory, then the int16 GEMM
  const int64_t lda = static_cast<int64_t>(round_up(static_cast<size_t>(K), 8));
  const size_t a_bytes = static_cast<size_t>(M) * static_cast<size_t>(lda) * 2;
  if ((rc = ensure_buffer(&d->conv_buf, &d->conv_buf_bytes, a_bytes)) != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(*d, s)) != GEMMI_OK) return rc;
  int16_t* A = static_cast<int16_t*>(d->conv_buf);
  cudaError_t e = gemmi::im2col_i16(X, A, lda, N, H, W, Cin, R, S, ph, pw, s);
  if (e != cudaSuccess) return cuda_error(e, "im2col launch");
  rc = M <= g_skinny_max_m ? run_skinny(*d, M, Cout, K, A, lda, Wt, Cout, Y, Cout, s)
                           : run_tc(*d, 2, M, Cout, K, A, lda, Wt, Cout, Y, Cout, s);
  if (rc != GEMMI_OK) return rc;
  return end_workspace_use(*d, s);
}

int gemm_i8_locked(int64_t m, int64_t n, int64_t k, const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb,
                   int32_t* C, int64_t ldc, cudaStream_t s) {
  const int pre = check_args(m, n, k, A, lda, B, ldb, C, ldc, 1, 4);
  if (pre >= 0) return pre;
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  return run_tc(*d, 1, m, n, k, A, lda, B, ldb, C, ldc, s);
}

// The int4 path (int4.cu, gemm_pair.cu): the packed operands become K-major E4M3 planes in the
// workspace (pitch k rounded up to 16 bytes), then the pair kernel runs on kind::f8f6f4.  A C that
// cannot take 16-byte bulk reductions gets a zeroed scratch result that one more pass adds into it.
// Checks of gemm_i4's arguments (lda, ldb in packed bytes); -1 to proceed, or a status to return.
// `b_bytes` > 0 replaces B's extent in the overlap check (the planes of a packed B).
int check_args_i4(int64_t m, int64_t n, int64_t k, const void* A, int64_t lda, const void* B, int64_t ldb,
                  const void* C, int64_t ldc, size_t b_bytes = 0) {
  if (m < 0 || n < 0 || k < 0) return set_error(GEMMI_EINVAL, "negative matrix dimension");
  const int64_t wa = (k + 1) / 2, wb = (n + 1) / 2;  // packed bytes per row of A and of B
  if (ldc < std::max<int64_t>(1, n)) return set_error(GEMMI_EINVAL, "ldc < max(1, n)");
  if (lda < std::max<int64_t>(1, wa)) return set_error(GEMMI_EINVAL, "lda < max(1, ceil(k/2)) bytes");
  if (ldb < std::max<int64_t>(1, wb)) return set_error(GEMMI_EINVAL, "ldb < max(1, ceil(n/2)) bytes");
  if (m == 0 || n == 0) return GEMMI_OK;
  if (C == nullptr) return set_error(GEMMI_EINVAL, "C is null");
  if (k == 0) return GEMMI_OK;
  if (A == nullptr || B == nullptr) return set_error(GEMMI_EINVAL, "A or B is null");
  if (m > (int64_t(1) << 40) || n > (int64_t(1) << 31) || k > (int64_t(1) << 31))
    return set_error(GEMMI_EINVAL, "matrix dimension too large");
  size_t a_bytes = 0, c_bytes = 0;
  if (!span_bytes(m, lda, wa, 1, &a_bytes) || !span_bytes(m, ldc, n, 4, &c_bytes) ||
      (b_bytes == 0 && !span_bytes(k, ldb, wb, 1, &b_bytes)))
    return set_error(GEMMI_EINVAL, "leading dimension too large: the operand's extent overflows 64 bits");
  if (overlaps(C, c_bytes, A, a_bytes) || overlaps(C, c_bytes, B, b_bytes))
    return set_error(GEMMI_EINVAL, "C overlaps A or B");
  return -1;
}

int run_i4(DeviceState& d, int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B,
           int64_t ldb, int32_t* C, int64_t ldc, cudaStream_t s, const LimbPlanes* packed_b = nullptr) {
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 16));
  const size_t a_plane = round_up(static_cast<size_t>(m) * pitch, kAlign);
  const size_t b_plane = packed_b ? 0 : round_up(static_cast<size_t>(n) * pitch, kAlign);
  const bool direct = reinterpret_cast<uintptr_t>(C) % 16 == 0 && ldc % 4 == 0;
  const int64_t ldt = static_cast<int64_t>(round_up(static_cast<size_t>(n), 4));
  const size_t t_bytes = direct ? 0 : static_cast<size_t>(m) * ldt * 4;
  int rc = ensure_buffer(&d.ws, &d.ws_bytes, a_plane + b_plane + t_bytes);
  if (rc != GEMMI_OK) return rc;
  if ((rc = begin_workspace_use(d, s)) != GEMMI_OK) return rc;
  char* ws = static_cast<char*>(d.ws);
  const LimbPlanes pa{{ws, nullptr}, m, pitch};
  const LimbPlanes pb = packed_b ? *packed_b : LimbPlanes{{ws + a_plane, nullptr}, n, pitch};
  int32_t* T = direct ? nullptr : reinterpret_cast<int32_t*>(ws + a_plane + b_plane);
  cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_CONVERT_I4, s);
  cudaError_t e = gemmi::convert_i4(A, lda, packed_b ? nullptr : B, ldb, m, n, k, pa, pb, d.sm_count, s);
  timer_end(GEMMI_KERNEL_CONVERT_I4, t0, s);
  if (e != cudaSuccess) return cuda_error(e, "int4 operand conversion launch");
  if (!direct && (e = cudaMemsetAsync(T, 0, t_bytes, s)) != cudaSuccess) return cuda_error(e, "cudaMemsetAsync");
  gemmi::TcGemmArgs ta;
  ta.m = m;
  ta.n = n;
  ta.k = k;
  ta.a = pa;
  ta.b = pb;
  ta.C = direct ? static_cast<void*>(C) : static_cast<void*>(T);
  ta.ldc = direct ? ldc : ldt;
  ta.status = d.status;
  ta.timeout_ns = timeout_ns();
  ta.num_sms = d.sm_count;
  ta.chunk_scale = static_cast<int>(g_tc_chunk_scale);
  ta.group_m = raster_band(true);
  ta.hint_a = static_cast<int>(g_tc_l2_hints & 3);
  ta.hint_b = static_cast<int>((g_tc_l2_hints >> 2) & 3);
  const char* why = "tcgen05 int4 GEMM launch";
  cudaEvent_t t1 = timer_begin(GEMMI_KERNEL_TC_PAIR_I4, s);
  e = gemmi::tc_pair_gemm_i4(ta, s, &why);
  timer_end(GEMMI_KERNEL_TC_PAIR_I4, t1, s);
  if (e != cudaSuccess) return cuda_error(e, why);
  if (!direct) {
    cudaEvent_t t2 = timer_begin(GEMMI_KERNEL_ADD_I32, s);
    e = gemmi::add_into_i32(C, ldc, T, ldt, m, n, d.sm_count, s);
    timer_end(GEMMI_KERNEL_ADD_I32, t2, s);
    if (e != cudaSuccess) return cuda_error(e, "int4 scratch add launch");
  }
  return end_workspace_use(d, s);
}

int gemm_i4_locked(int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb,
                   int32_t* C, int64_t ldc, cudaStream_t s) {
  const int pre = check_args_i4(m, n, k, A, lda, B, ldb, C, ldc);
  if (pre >= 0) return pre;
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  return run_i4(*d, m, n, k, A, lda, B, ldb, C, ldc, s);
}

// Reads the status words of the current device `dev` -- the library's own (when `d` is non-null)
// and the allocation-free entry point's (when that entry point has run on the device) -- after
// synchronising the device (s_only == false) or only stream `s`.  A non-zero word is cleared when
// `clear`; the first non-zero word decides the return code.
int read_status_words(int dev, DeviceState* d, bool clear, bool s_only, cudaStream_t s, bool with_noalloc = true) {
  cudaError_t e = s_only ? cudaStreamSynchronize(s) : cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_error(e, s_only ? "cudaStreamSynchronize" : "cudaDeviceSynchronize");
  uint32_t* words[2] = {d != nullptr ? d->status : nullptr, with_noalloc ? gemmi::noalloc_status_word(dev) : nullptr};
  uint32_t word = 0;
  for (uint32_t* w : words) {
    if (w == nullptr) continue;
    uint32_t v = 0;
    e = cudaMemcpyAsync(&v, w, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_error(e, "reading a device status word");
    if (clear && v != 0) {
      e = cudaMemsetAsync(w, 0, sizeof(v), s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
      if (e != cudaSuccess) return cuda_error(e, "clearing a device status word");
    }
    if (word == 0) word = v;
  }
  if (d != nullptr) d->last_detail = word;
  g_dev[dev].last_detail = word;
  if (word == 0) return GEMMI_OK;
  const int code = static_cast<int>(word & 0xFFu);
  char buf[160];
  std::snprintf(buf, sizeof(buf), "device status 0x%08x: a pipeline wait (site %u, block %u) ran out of time",
                word, (word >> 8) & 0xFFu, word >> 16);
  return set_error(code, buf);
}

// The library's own word only (the entry points that report their status themselves).
int read_status_locked(DeviceState& d, bool clear) {
  const int dev = static_cast<int>(&d - g_dev);
  return read_status_words(dev, &d, clear, false, nullptr, false);
}

// gemmi_device_status / gemmi_device_status_stream.  A device on which only the allocation-free
// entry point has run is read without setting up the library's own state (which allocates).
int device_status_impl(bool s_only, cudaStream_t s) {
  std::lock_guard<std::mutex> lock(g_mutex);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(GEMMI_EINVAL, "device ordinal out of range");
  if (!g_dev[dev].ready && gemmi::noalloc_status_word(dev) != nullptr)
    return read_status_words(dev, nullptr, true, s_only, s);
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  return read_status_words(dev, d, true, s_only, s);
}

int ensure_pipeline(DeviceState& d) {
  if (d.h2d != nullptr) return GEMMI_OK;
  cudaError_t e = cudaStreamCreateWithFlags(&d.h2d, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&d.d2h, cudaStreamNonBlocking);
  for (auto& ev : d.pipe_ev)
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
  return e == cudaSuccess ? GEMMI_OK : cuda_error(e, "creating the copy streams of the host-buffer path");
}

constexpr int kPipeSlots = 3;
constexpr int64_t kPanelMin = 512;

// First rows of the pipelined host path's row panels, then m: panels of at most mb rows, with a
// quarter and a half panel at each end when m has room for them.  The small first panel starts
// the copies out sooner; the small last panels shorten the end of the call, where the last GEMM
// and its copy out run with nothing left to overlap them.
std::vector<int64_t> panel_starts(int64_t m, int64_t mb) {
  std::vector<int64_t> starts{0};
  const int64_t q = mb / 4, h = mb / 2;
  if (q < 1 || m < 2 * (q + h) + mb) {
    for (int64_t r = mb; r < m; r += mb) starts.push_back(r);
  } else {
    starts.push_back(q);
    starts.push_back(q + h);
    // whole panels in the middle, the remainder of the rows as one panel in front of them
    const int64_t mid = m - 2 * (q + h);
    int64_t r = q + h + mid % mb;
    if (r > q + h) starts.push_back(r);
    for (r += mb; r < m - q - h; r += mb) starts.push_back(r);
    starts.push_back(m - q - h);
    starts.push_back(m - q);
  }
  starts.push_back(m);
  return starts;
}

// Host-buffer GEMM of m >= 2 * kPanelMin rows as a pipeline over row panels of A and C.  B is
// copied and split into limb planes once; then each panel's copy in (A and C rows), GEMM and
// copy out run on three streams (copy in, the caller's stream, copy out) through a ring of
// kPipeSlots device slots, so the host-link copies in both directions overlap each other and the
// tensor cores.  The link, not the GPU, bounds this path: about 0.2 TB/s each way.
template <typename OP, typename CT>
int host_gemm_pipelined(DeviceState& d, int nl, int64_t m, int64_t n, int64_t k, const OP* A, int64_t lda,
                        const OP* B, int64_t ldb, CT* C, int64_t ldc) {
  int rc = ensure_pipeline(d);
  if (rc != GEMMI_OK) return rc;
  cudaStream_t s = g_stream;
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 8));
  const int64_t mb = std::max<int64_t>(kPanelMin, static_cast<int64_t>(round_up(static_cast<size_t>((m + 15) / 16), 128)));
  const std::vector<int64_t> starts = panel_starts(m, mb);
  const int64_t panels = static_cast<int64_t>(starts.size()) - 1;
  const size_t b_raw = round_up(static_cast<size_t>(k) * n * sizeof(OP), kAlign);
  const size_t b_plane = round_up(static_cast<size_t>(n) * pitch * 2, kAlign);
  const size_t a_slot = round_up(static_cast<size_t>(mb) * k * sizeof(OP), kAlign);
  const size_t c_slot = round_up(static_cast<size_t>(mb) * n * sizeof(CT), kAlign);
  if ((rc = ensure_buffer(&d.host_buf, &d.host_buf_bytes, b_raw + nl * b_plane + kPipeSlots * (a_slot + c_slot))) !=
      GEMMI_OK)
    return rc;
  // the A planes of one panel, sized now so no panel has to grow the workspace mid-pipeline
  if ((rc = ensure_buffer(&d.ws, &d.ws_bytes, plane_layout(mb, 0, pitch, nl).total)) != GEMMI_OK) return rc;
  char* base = static_cast<char*>(d.host_buf);
  OP* dB = reinterpret_cast<OP*>(base);
  LimbPlanes pb{{base + b_raw, base + b_raw + (nl == 2 ? b_plane : 0)}, n, pitch};
  char* slots = base + b_raw + nl * b_plane;
  cudaEvent_t* ev = d.pipe_ev;  // 0 start, 1 B copied, 2-4 panel in, 5-7 panel done, 8-10 panel out, 11 end
  // on an error, let the copies already queued finish before the buffers can be reused
  auto settle = [&]() {
    cudaStreamSynchronize(d.h2d);
    cudaStreamSynchronize(s);
    cudaStreamSynchronize(d.d2h);
  };
  auto fail = [&](cudaError_t e, const char* what) {
    settle();
    return cuda_error(e, what);
  };
  cudaError_t e = cudaEventRecord(ev[0], s);  // after earlier work of the caller's stream
  if (e == cudaSuccess) e = cudaStreamWaitEvent(d.h2d, ev[0], 0);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(d.d2h, ev[0], 0);
  if (e == cudaSuccess)
    e = cudaMemcpy2DAsync(dB, n * sizeof(OP), B, ldb * sizeof(OP), n * sizeof(OP), k, cudaMemcpyHostToDevice, d.h2d);
  if (e == cudaSuccess) e = cudaEventRecord(ev[1], d.h2d);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[1], 0);
  if (e != cudaSuccess) return fail(e, "host-to-device copy of B");
  {
    const LimbPlanes none{{nullptr, nullptr}, 0, pitch};
    cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_SPLIT, s);
    e = nl == 2 ? gemmi::split_i16(nullptr, k, reinterpret_cast<const int16_t*>(dB), n, 0, n, k, none, pb, s, d.status,
                                   timeout_ns())
                : gemmi::convert_i8(nullptr, k, reinterpret_cast<const int8_t*>(dB), n, 0, n, k, none, pb, s, d.status,
                                    timeout_ns());
    timer_end(GEMMI_KERNEL_SPLIT, t0, s);
    if (e != cudaSuccess) return fail(e, "split of B");
  }
  for (int64_t p = 0; p < panels; ++p) {
    const int r = static_cast<int>(p % kPipeSlots);
    const int64_t r0 = starts[p], mi = starts[p + 1] - r0;
    OP* dA = reinterpret_cast<OP*>(slots + r * (a_slot + c_slot));
    CT* dC = reinterpret_cast<CT*>(slots + r * (a_slot + c_slot) + a_slot);
    e = p >= kPipeSlots ? cudaStreamWaitEvent(d.h2d, ev[8 + r], 0) : cudaSuccess;  // slot's last copy out
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(dA, k * sizeof(OP), A + r0 * lda, lda * sizeof(OP), k * sizeof(OP), mi,
                            cudaMemcpyHostToDevice, d.h2d);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(dC, n * sizeof(CT), C + r0 * ldc, ldc * sizeof(CT), n * sizeof(CT), mi,
                            cudaMemcpyHostToDevice, d.h2d);
    if (e == cudaSuccess) e = cudaEventRecord(ev[2 + r], d.h2d);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[2 + r], 0);
    if (e != cudaSuccess) return fail(e, "host-to-device copy of a panel");
    rc = run_tc(d, nl, mi, n, k, dA, k, nullptr, n, dC, n, s, &pb);
    if (rc != GEMMI_OK) {
      settle();
      return rc;
    }
    e = cudaEventRecord(ev[5 + r], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(d.d2h, ev[5 + r], 0);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(C + r0 * ldc, ldc * sizeof(CT), dC, n * sizeof(CT), n * sizeof(CT), mi,
                            cudaMemcpyDeviceToHost, d.d2h);
    if (e == cudaSuccess) e = cudaEventRecord(ev[8 + r], d.d2h);
    if (e != cudaSuccess) return fail(e, "device-to-host copy of a panel");
  }
  // the caller's stream continues after the last copy out
  e = cudaEventRecord(ev[11], d.d2h);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[11], 0);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(e, "cudaStreamSynchronize");
  return GEMMI_OK;
}

template <typename OP, typename CT, typename F>
int host_gemm(int64_t m, int64_t n, int64_t k, const OP* A, int64_t lda, const OP* B, int64_t ldb, CT* C,
              int64_t ldc, F device_call) {
  std::lock_guard<std::mutex> lock(g_mutex);
  const int pre = check_args(m, n, k, A, lda, B, ldb, C, ldc, sizeof(OP), sizeof(CT));
  if (pre >= 0) return pre;
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  constexpr int nl = sizeof(OP) == 2 ? 2 : 1;
  if (m >= 2 * kPanelMin && m > (nl == 2 ? g_skinny_max_m : 0)) {
    rc = host_gemm_pipelined(*d, nl, m, n, k, A, lda, B, ldb, C, ldc);
    if (rc != GEMMI_OK) return rc;
    uint32_t word = 0;
    const cudaError_t e = cudaMemcpy(&word, d->status, sizeof(word), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy(status)");
    if (word != 0) return read_status_locked(*d, true);
    return GEMMI_OK;
  }
  const size_t a_bytes = round_up(static_cast<size_t>(m) * k * sizeof(OP), kAlign);
  const size_t b_bytes = round_up(static_cast<size_t>(k) * n * sizeof(OP), kAlign);
  const size_t c_bytes = round_up(static_cast<size_t>(m) * n * sizeof(CT), kAlign);
  if ((rc = ensure_buffer(&d->host_buf, &d->host_buf_bytes, a_bytes + b_bytes + c_bytes)) != GEMMI_OK) return rc;
  char* base = static_cast<char*>(d->host_buf);
  OP* dA = reinterpret_cast<OP*>(base);
  OP* dB = reinterpret_cast<OP*>(base + a_bytes);
  CT* dC = reinterpret_cast<CT*>(base + a_bytes + b_bytes);
  cudaStream_t s = g_stream;
  cudaError_t e = cudaMemcpy2DAsync(dA, k * sizeof(OP), A, lda * sizeof(OP), k * sizeof(OP), m, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpy2DAsync(dB, n * sizeof(OP), B, ldb * sizeof(OP), n * sizeof(OP), k, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpy2DAsync(dC, n * sizeof(CT), C, ldc * sizeof(CT), n * sizeof(CT), m, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_error(e, "host-to-device copy");
  rc = device_call(m, n, k, dA, k, dB, n, dC, n, s);
  if (rc != GEMMI_OK) return rc;
  e = cudaMemcpy2DAsync(C, ldc * sizeof(CT), dC, n * sizeof(CT), n * sizeof(CT), m, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return cuda_error(e, "device-to-host copy");
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_error(e, "cudaStreamSynchronize");
  uint32_t word = 0;
  e = cudaMemcpy(&word, d->status, sizeof(word), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy(status)");
  if (word != 0) return read_status_locked(*d, true);
  return GEMMI_OK;
}

// gemm_i4 on host buffers with m >= 2 * kPanelMin, pipelined like host_gemm_pipelined: B is copied
// and converted to its E4M3 plane once, then row panels of A and C pass through kPipeSlots device
// slots, copies in and out on their own streams while each panel's GEMM runs on the caller's
// stream.  Device pitches (16 bytes for packed operands, 4 elements for C) keep every kernel on
// its aligned path.
int host_gemm_i4_pipelined(DeviceState& d, int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda,
                           const uint8_t* B, int64_t ldb, int32_t* C, int64_t ldc) {
  int rc = ensure_pipeline(d);
  if (rc != GEMMI_OK) return rc;
  cudaStream_t s = g_stream;
  const int64_t wa = (k + 1) / 2, wb = (n + 1) / 2;
  const int64_t dlda = static_cast<int64_t>(round_up(static_cast<size_t>(wa), 16));
  const int64_t dldb = static_cast<int64_t>(round_up(static_cast<size_t>(wb), 16));
  const int64_t dldc = static_cast<int64_t>(round_up(static_cast<size_t>(n), 4));
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), 16));
  const int64_t mb = std::max<int64_t>(kPanelMin, static_cast<int64_t>(round_up(static_cast<size_t>((m + 15) / 16), 128)));
  const std::vector<int64_t> starts = panel_starts(m, mb);
  const int64_t panels = static_cast<int64_t>(starts.size()) - 1;
  const size_t b_raw = round_up(static_cast<size_t>(k) * dldb, kAlign);
  const size_t b_plane = round_up(static_cast<size_t>(n) * pitch, kAlign);
  const size_t a_slot = round_up(static_cast<size_t>(mb) * dlda, kAlign);
  const size_t c_slot = round_up(static_cast<size_t>(mb) * dldc * 4, kAlign);
  if ((rc = ensure_buffer(&d.host_buf, &d.host_buf_bytes, b_raw + b_plane + kPipeSlots * (a_slot + c_slot))) !=
      GEMMI_OK)
    return rc;
  // one panel's A plane, sized now so no panel has to grow the workspace mid-pipeline
  if ((rc = ensure_buffer(&d.ws, &d.ws_bytes, round_up(static_cast<size_t>(mb) * pitch, kAlign))) != GEMMI_OK)
    return rc;
  char* base = static_cast<char*>(d.host_buf);
  uint8_t* dB = reinterpret_cast<uint8_t*>(base);
  const LimbPlanes pb{{base + b_raw, nullptr}, n, pitch};
  char* slots = base + b_raw + b_plane;
  cudaEvent_t* ev = d.pipe_ev;  // 0 start, 1 B copied, 2-4 panel in, 5-7 panel done, 8-10 panel out, 11 end
  auto settle = [&]() {
    cudaStreamSynchronize(d.h2d);
    cudaStreamSynchronize(s);
    cudaStreamSynchronize(d.d2h);
  };
  auto fail = [&](cudaError_t e, const char* what) {
    settle();
    return cuda_error(e, what);
  };
  cudaError_t e = cudaEventRecord(ev[0], s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(d.h2d, ev[0], 0);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(d.d2h, ev[0], 0);
  if (e == cudaSuccess) e = cudaMemcpy2DAsync(dB, dldb, B, ldb, wb, k, cudaMemcpyHostToDevice, d.h2d);
  if (e == cudaSuccess) e = cudaEventRecord(ev[1], d.h2d);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[1], 0);
  if (e != cudaSuccess) return fail(e, "host-to-device copy of B");
  {
    const LimbPlanes none{{nullptr, nullptr}, 0, pitch};
    cudaEvent_t t0 = timer_begin(GEMMI_KERNEL_CONVERT_I4, s);
    e = gemmi::convert_i4(nullptr, 1, dB, dldb, 0, n, k, none, pb, d.sm_count, s);
    timer_end(GEMMI_KERNEL_CONVERT_I4, t0, s);
    if (e != cudaSuccess) return fail(e, "conversion of B");
  }
  for (int64_t p = 0; p < panels; ++p) {
    const int r = static_cast<int>(p % kPipeSlots);
    const int64_t r0 = starts[p], mi = starts[p + 1] - r0;
    uint8_t* dA = reinterpret_cast<uint8_t*>(slots + r * (a_slot + c_slot));
    int32_t* dC = reinterpret_cast<int32_t*>(slots + r * (a_slot + c_slot) + a_slot);
    e = p >= kPipeSlots ? cudaStreamWaitEvent(d.h2d, ev[8 + r], 0) : cudaSuccess;  // slot's last copy out
    if (e == cudaSuccess) e = cudaMemcpy2DAsync(dA, dlda, A + r0 * lda, lda, wa, mi, cudaMemcpyHostToDevice, d.h2d);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(dC, dldc * 4, C + r0 * ldc, ldc * 4, n * 4, mi, cudaMemcpyHostToDevice, d.h2d);
    if (e == cudaSuccess) e = cudaEventRecord(ev[2 + r], d.h2d);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[2 + r], 0);
    if (e != cudaSuccess) return fail(e, "host-to-device copy of a panel");
    rc = run_i4(d, mi, n, k, dA, dlda, nullptr, dldb, dC, dldc, s, &pb);
    if (rc != GEMMI_OK) {
      settle();
      return rc;
    }
    e = cudaEventRecord(ev[5 + r], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(d.d2h, ev[5 + r], 0);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(C + r0 * ldc, ldc * 4, dC, dldc * 4, n * 4, mi, cudaMemcpyDeviceToHost, d.d2h);
    if (e == cudaSuccess) e = cudaEventRecord(ev[8 + r], d.d2h);
    if (e != cudaSuccess) return fail(e, "device-to-host copy of a panel");
  }
  e = cudaEventRecord(ev[11], d.d2h);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev[11], 0);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(e, "cudaStreamSynchronize");
  return GEMMI_OK;
}

// gemm_i4 on host buffers: packed A and B and C are copied into device buffers whose row pitches
// (16 bytes for the operands, 4 elements for C) keep the conversion and the pair kernel on their
// aligned paths, the GEMM runs, and C is copied back.
int host_gemm_i4(int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb,
                 int32_t* C, int64_t ldc) {
  std::lock_guard<std::mutex> lock(g_mutex);
  const int pre = check_args_i4(m, n, k, A, lda, B, ldb, C, ldc);
  if (pre >= 0) return pre;
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  if (m >= 2 * kPanelMin) {
    rc = host_gemm_i4_pipelined(*d, m, n, k, A, lda, B, ldb, C, ldc);
    if (rc != GEMMI_OK) return rc;
    uint32_t word = 0;
    const cudaError_t e = cudaMemcpy(&word, d->status, sizeof(word), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy(status)");
    if (word != 0) return read_status_locked(*d, true);
    return GEMMI_OK;
  }
  const int64_t wa = (k + 1) / 2, wb = (n + 1) / 2;
  const int64_t dlda = static_cast<int64_t>(round_up(static_cast<size_t>(wa), 16));
  const int64_t dldb = static_cast<int64_t>(round_up(static_cast<size_t>(wb), 16));
  const int64_t dldc = static_cast<int64_t>(round_up(static_cast<size_t>(n), 4));
  const size_t a_bytes = round_up(static_cast<size_t>(m) * dlda, kAlign);
  const size_t b_bytes = round_up(static_cast<size_t>(k) * dldb, kAlign);
  const size_t c_bytes = round_up(static_cast<size_t>(m) * dldc * 4, kAlign);
  if ((rc = ensure_buffer(&d->host_buf, &d->host_buf_bytes, a_bytes + b_bytes + c_bytes)) != GEMMI_OK) return rc;
  char* base = static_cast<char*>(d->host_buf);
  uint8_t* dA = reinterpret_cast<uint8_t*>(base);
  uint8_t* dB = reinterpret_cast<uint8_t*>(base + a_bytes);
  int32_t* dC = reinterpret_cast<int32_t*>(base + a_bytes + b_bytes);
  cudaStream_t s = g_stream;
  cudaError_t e = cudaMemcpy2DAsync(dA, dlda, A, lda, wa, m, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpy2DAsync(dB, dldb, B, ldb, wb, k, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpy2DAsync(dC, dldc * 4, C, ldc * 4, n * 4, m, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_error(e, "host-to-device copy");
  rc = run_i4(*d, m, n, k, dA, dlda, dB, dldb, dC, dldc, s);
  if (rc != GEMMI_OK) return rc;
  e = cudaMemcpy2DAsync(C, ldc * 4, dC, dldc * 4, n * 4, m, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return cuda_error(e, "device-to-host copy");
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_error(e, "cudaStreamSynchronize");
  uint32_t word = 0;
  e = cudaMemcpy(&word, d->status, sizeof(word), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemcpy(status)");
  if (word != 0) return read_status_locked(*d, true);
  return GEMMI_OK;
}

__global__ void wait_probe_kernel(uint32_t* status, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    gemmi::mbar_init(gemmi::smem_u32(&bar), 1);
    gemmi::fence_mbar_init();
  }
  __syncthreads();
  // nothing ever arrives on `bar`: the bounded wait must give up and report
  if (threadIdx.x == 0 && !gemmi::bounded_wait(gemmi::smem_u32(&bar), 0, timeout_ns))
    gemmi::report_status(status, GEMMI_ETIMEOUT, 99);
}

}  // namespace

namespace gemmi {
void record_error(const char* msg) { t_error = msg; }

cudaError_t launch_wait_timeout_probe(uint32_t* status, uint64_t timeout_ns, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(status, timeout_ns);
  return cudaGetLastError();
}
}  // namespace gemmi

extern "C" {

int gemm_i16_ex(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb,
                int64_t* C, int64_t ldc, void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i16_locked(m, n, k, A, lda, B, ldb, C, ldc, static_cast<cudaStream_t>(stream));
}

int gemm_i16(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb,
             int64_t* C, int64_t ldc) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i16_locked(m, n, k, A, lda, B, ldb, C, ldc, g_stream);
}

int gemm_i16_srs_ex(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B,
                    int64_t ldb, int16_t* C, int64_t ldc, int shift, void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i16_srs_locked(m, n, k, A, lda, B, ldb, C, ldc, shift, static_cast<cudaStream_t>(stream));
}

int gemm_i16_srs(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb,
                 int16_t* C, int64_t ldc, int shift) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i16_srs_locked(m, n, k, A, lda, B, ldb, C, ldc, shift, g_stream);
}

int gemmi_conv2d_i16(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t R, int64_t S,
                     int64_t pad_h, int64_t pad_w, const int16_t* X, const int16_t* Wt, int64_t* Y, void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return conv2d_locked(N, H, W, Cin, Cout, R, S, pad_h, pad_w, X, Wt, Y, static_cast<cudaStream_t>(stream));
}

int gemm_i8_ex(int64_t m, int64_t n, int64_t k, const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb,
               int32_t* C, int64_t ldc, void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i8_locked(m, n, k, A, lda, B, ldb, C, ldc, static_cast<cudaStream_t>(stream));
}

int gemm_i8(int64_t m, int64_t n, int64_t k, const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb,
            int32_t* C, int64_t ldc) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i8_locked(m, n, k, A, lda, B, ldb, C, ldc, g_stream);
}

int gemm_i4_ex(int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb,
               int32_t* C, int64_t ldc, void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i4_locked(m, n, k, A, lda, B, ldb, C, ldc, static_cast<cudaStream_t>(stream));
}

int gemm_i4(int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb,
            int32_t* C, int64_t ldc) {
  std::lock_guard<std::mutex> lock(g_mutex);
  return gemm_i4_locked(m, n, k, A, lda, B, ldb, C, ldc, g_stream);
}

int gemm_i16_host(int64_t m, int64_t n, int64_t k, const int16_t* A, int64_t lda, const int16_t* B, int64_t ldb,
                  int64_t* C, int64_t ldc) {
  return host_gemm(m, n, k, A, lda, B, ldb, C, ldc, gemm_i16_locked);
}

int gemm_i8_host(int64_t m, int64_t n, int64_t k, const int8_t* A, int64_t lda, const int8_t* B, int64_t ldb,
                 int32_t* C, int64_t ldc) {
  return host_gemm(m, n, k, A, lda, B, ldb, C, ldc, gemm_i8_locked);
}

int gemm_i4_host(int64_t m, int64_t n, int64_t k, const uint8_t* A, int64_t lda, const uint8_t* B, int64_t ldb,
                 int32_t* C, int64_t ldc) {
  return host_gemm_i4(m, n, k, A, lda, B, ldb, C, ldc);
}

}  // extern "C"

struct gemmi_packed_b {
  int nl;        // 2: int16 limb planes, 1: int8 values as fp16, 4: int4 values as E4M3 bytes
  int device;
  int64_t k, n, pitch;
  void* mem;     // the planes, owned by the handle
};

namespace {

int pack_b(int nl, int64_t k, int64_t n, const void* B, int64_t ldb, void* stream, gemmi_packed_b** out) {
  if (out == nullptr) return set_error(GEMMI_EINVAL, "null output handle");
  *out = nullptr;
  if (k < 1 || n < 1) return set_error(GEMMI_EINVAL, "packed operand needs k >= 1 and n >= 1");
  if (ldb < (nl == 4 ? (n + 1) / 2 : n)) return set_error(GEMMI_EINVAL, nl == 4 ? "ldb < ceil(n/2) bytes" : "ldb < n");
  if (B == nullptr) return set_error(GEMMI_EINVAL, "B is null");
  if (k > (int64_t(1) << 31) || n > (int64_t(1) << 31)) return set_error(GEMMI_EINVAL, "matrix dimension too large");
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  const bool i4 = nl == 4;
  const int64_t pitch = static_cast<int64_t>(round_up(static_cast<size_t>(k), i4 ? 16 : 8));
  const size_t plane = round_up(static_cast<size_t>(n) * pitch * (i4 ? 1 : 2), kAlign);
  void* mem = nullptr;
  if (cudaMalloc(&mem, plane * (nl == 2 ? 2 : 1)) != cudaSuccess) {
    cudaGetLastError();
    return set_error(GEMMI_ENOMEM, "cannot allocate the packed operand");
  }
  char* base = static_cast<char*>(mem);
  LimbPlanes pb{{base, base + (nl == 2 ? plane : 0)}, n, pitch};
  LimbPlanes none{{nullptr, nullptr}, 0, pitch};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e =
      nl == 2 ? gemmi::split_i16(nullptr, k, static_cast<const int16_t*>(B), ldb, 0, n, k, none, pb, s)
      : i4    ? gemmi::convert_i4(nullptr, 1, static_cast<const uint8_t*>(B), ldb, 0, n, k, none, pb, d->sm_count, s)
              : gemmi::convert_i8(nullptr, k, static_cast<const int8_t*>(B), ldb, 0, n, k, none, pb, s);
  if (e != cudaSuccess) {
    cudaFree(mem);
    return cuda_error(e, "packing launch");
  }
  *out = new gemmi_packed_b{nl, dev, k, n, pitch, mem};
  return GEMMI_OK;
}

int gemm_packed(int nl, int64_t m, const void* A, int64_t lda, const gemmi_packed_b* Bp, void* C, int64_t ldc,
                void* stream) {
  if (Bp == nullptr) return set_error(GEMMI_EINVAL, "null packed operand");
  if (Bp->nl != nl) return set_error(GEMMI_EINVAL, "packed operand has another element type");
  const int64_t n = Bp->n, k = Bp->k;
  const size_t op = nl == 2 ? 2 : 1, cs = nl == 2 ? 8 : 4;
  // the packed planes stand in for B in the overlap check (C must not overlap them either)
  const int pre = check_args(m, n, k, A, lda, Bp->mem, n, C, ldc, op, cs);
  if (pre >= 0) return pre;
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != Bp->device) return set_error(GEMMI_EINVAL, "packed operand belongs to another device");
  const size_t plane = round_up(static_cast<size_t>(n) * Bp->pitch * 2, kAlign);
  char* base = static_cast<char*>(Bp->mem);
  LimbPlanes pb{{base, base + (nl == 2 ? plane : 0)}, n, Bp->pitch};
  return run_tc(*d, nl, m, n, k, A, lda, nullptr, n, C, ldc, static_cast<cudaStream_t>(stream), &pb);
}

int gemm_i4_packed_impl(int64_t m, const uint8_t* A, int64_t lda, const gemmi_packed_b* Bp, int32_t* C, int64_t ldc,
                        void* stream) {
  if (Bp == nullptr) return set_error(GEMMI_EINVAL, "null packed operand");
  if (Bp->nl != 4) return set_error(GEMMI_EINVAL, "packed operand has another element type");
  const int64_t n = Bp->n, k = Bp->k;
  const size_t plane = round_up(static_cast<size_t>(n) * Bp->pitch, kAlign);
  // the packed plane stands in for B in the checks (C must not overlap it either)
  const int pre = check_args_i4(m, n, k, A, lda, Bp->mem, (n + 1) / 2, C, ldc, plane);
  if (pre >= 0) return pre;
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != Bp->device) return set_error(GEMMI_EINVAL, "packed operand belongs to another device");
  const LimbPlanes pb{{Bp->mem, nullptr}, n, Bp->pitch};
  return run_i4(*d, m, n, k, A, lda, nullptr, (n + 1) / 2, C, ldc, static_cast<cudaStream_t>(stream), &pb);
}

}  // namespace

extern "C" {

int gemmi_pack_b_i4(int64_t k, int64_t n, const uint8_t* B, int64_t ldb, void* stream, gemmi_packed_b** out) {
  return pack_b(4, k, n, B, ldb, stream, out);
}

int gemm_i4_packed(int64_t m, const uint8_t* A, int64_t lda, const gemmi_packed_b* B, int32_t* C, int64_t ldc,
                   void* stream) {
  return gemm_i4_packed_impl(m, A, lda, B, C, ldc, stream);
}

int gemmi_pack_b_i16(int64_t k, int64_t n, const int16_t* B, int64_t ldb, void* stream, gemmi_packed_b** out) {
  return pack_b(2, k, n, B, ldb, stream, out);
}

int gemmi_pack_b_i8(int64_t k, int64_t n, const int8_t* B, int64_t ldb, void* stream, gemmi_packed_b** out) {
  return pack_b(1, k, n, B, ldb, stream, out);
}

int gemm_i16_packed(int64_t m, const int16_t* A, int64_t lda, const gemmi_packed_b* B, int64_t* C, int64_t ldc,
                    void* stream) {
  return gemm_packed(2, m, A, lda, B, C, ldc, stream);
}

int gemm_i8_packed(int64_t m, const int8_t* A, int64_t lda, const gemmi_packed_b* B, int32_t* C, int64_t ldc,
                   void* stream) {
  return gemm_packed(1, m, A, lda, B, C, ldc, stream);
}

int gemmi_packed_b_free(gemmi_packed_b* packed) {
  if (packed == nullptr) return GEMMI_OK;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(packed->device);
  cudaDeviceSynchronize();
  cudaError_t e = cudaFree(packed->mem);
  cudaSetDevice(prev);
  delete packed;
  if (e != cudaSuccess) return cuda_error(e, "cudaFree(packed operand)");
  return GEMMI_OK;
}

int64_t gemmi_packed_b_k(const gemmi_packed_b* packed) { return packed ? packed->k : 0; }
int64_t gemmi_packed_b_n(const gemmi_packed_b* packed) { return packed ? packed->n : 0; }

void gemmi_set_stream(void* stream) {
  std::lock_guard<std::mutex> lock(g_mutex);
  g_stream = static_cast<cudaStream_t>(stream);
}

const char* gemmi_last_error(void) { return t_error.c_str(); }

int gemmi_device_status(void) { return device_status_impl(false, nullptr); }

int gemmi_device_status_stream(void* stream) { return device_status_impl(true, static_cast<cudaStream_t>(stream)); }

uint32_t gemmi_device_status_detail(void) {
  std::lock_guard<std::mutex> lock(g_mutex);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  return g_dev[dev].last_detail;
}

int gemmi_release_workspace(void) {
  std::lock_guard<std::mutex> lock(g_mutex);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(GEMMI_EINVAL, "device ordinal out of range");
  DeviceState& d = g_dev[dev];
  if (d.ws == nullptr && d.host_buf == nullptr && d.sum_buf == nullptr && d.conv_buf == nullptr) return GEMMI_OK;
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceSynchronize");
  if (d.ws) cudaFree(d.ws);
  if (d.host_buf) cudaFree(d.host_buf);
  if (d.sum_buf) cudaFree(d.sum_buf);
  if (d.conv_buf) cudaFree(d.conv_buf);
  d.ws = d.host_buf = d.sum_buf = d.conv_buf = nullptr;
  d.sum_buf_bytes = d.conv_buf_bytes = 0;
  d.ws_bytes = d.host_buf_bytes = 0;
  d.used = false;
  return GEMMI_OK;
}

size_t gemmi_workspace_bytes(void) {
  std::lock_guard<std::mutex> lock(g_mutex);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  return g_dev[dev].ws_bytes + g_dev[dev].host_buf_bytes + g_dev[dev].sum_buf_bytes + g_dev[dev].conv_buf_bytes;
}

int gemmi_set_option(int option, int64_t value) {
  std::lock_guard<std::mutex> lock(g_mutex);
  switch (option) {
    case GEMMI_OPT_SKINNY_MAX_M:
      if (value < 0 || value > 16) return set_error(GEMMI_EINVAL, "skinny limit must be in [0, 16]");
      g_skinny_max_m = value;
      return GEMMI_OK;
    case GEMMI_OPT_WAIT_TIMEOUT_US:
      // at least 1 ms: a CTA that gives up waits this long once more for its own copies in flight,
      // which land within microseconds, before it exits
      if (value < 1000 || value > 60000000) return set_error(GEMMI_EINVAL, "timeout must be in [1 ms, 60 s]");
      g_timeout_us = value;
      return GEMMI_OK;
    case GEMMI_OPT_SKINNY_KSPLIT:
      if (value < 0 || value > 4096) return set_error(GEMMI_EINVAL, "ksplit must be in [0, 4096]");
      g_skinny_ksplit = value;
      return GEMMI_OK;
    case GEMMI_OPT_TC_CHUNK_SCALE:
      if (value != 1 && value != 2) return set_error(GEMMI_EINVAL, "chunk scale must be 1 or 2");
      g_tc_chunk_scale = value;
      return GEMMI_OK;
    case GEMMI_OPT_TC_GROUP_M:
      if (value < 0 || value > 1024) return set_error(GEMMI_EINVAL, "raster band must be in [0, 1024]");
      g_tc_group_m = value;
      return GEMMI_OK;
    case GEMMI_OPT_TC_L2_HINTS:
      if (value < 0 || value > 15 || (value & 3) == 3 || ((value >> 2) & 3) == 3)
        return set_error(GEMMI_EINVAL, "L2 hints: 2 bits each for A and B, values 0..2");
      g_tc_l2_hints = value;
      return GEMMI_OK;
    case GEMMI_OPT_FUSED_MAX_N:
      if (value < 0 || value > 4096) return set_error(GEMMI_EINVAL, "fused-kernel n limit must be in [0, 4096]");
      g_fused_max_n = value;
      return GEMMI_OK;
    case GEMMI_OPT_TC_PAIR:
      if (value != 0 && value != 1) return set_error(GEMMI_EINVAL, "SM-pair option must be 0 or 1");
      g_tc_pair = value;
      return GEMMI_OK;
    case GEMMI_OPT_SMALL_MAX_MACS:
      if (value < 0 || value > (int64_t{1} << 40)) return set_error(GEMMI_EINVAL, "small-problem limit must be in [0, 2^40]");
      g_small_max_macs = value;
      return GEMMI_OK;
    case GEMMI_OPT_KARATSUBA:
      if (value != 0 && value != 1) return set_error(GEMMI_EINVAL, "Karatsuba option must be 0 or 1");
      g_karatsuba = value;
      return GEMMI_OK;
    case GEMMI_OPT_SPLIT_AHEAD:
      if (value != 0 && value != 1) return set_error(GEMMI_EINVAL, "overlapped-split option must be 0 or 1");
      g_split_ahead = value;
      return GEMMI_OK;
    case GEMMI_OPT_CONV_ROWS:
      if (value != 0 && value != 1) return set_error(GEMMI_EINVAL, "direct-convolution option must be 0 or 1");
      g_conv_rows = value;
      return GEMMI_OK;
    default:
      return set_error(GEMMI_EINVAL, "unknown option");
  }
}

int64_t gemmi_get_option(int option) {
  std::lock_guard<std::mutex> lock(g_mutex);
  switch (option) {
    case GEMMI_OPT_SKINNY_MAX_M: return g_skinny_max_m;
    case GEMMI_OPT_WAIT_TIMEOUT_US: return g_timeout_us;
    case GEMMI_OPT_SKINNY_KSPLIT: return g_skinny_ksplit;
    case GEMMI_OPT_TC_CHUNK_SCALE: return g_tc_chunk_scale;
    case GEMMI_OPT_TC_GROUP_M: return g_tc_group_m;
    case GEMMI_OPT_TC_L2_HINTS: return g_tc_l2_hints;
    case GEMMI_OPT_FUSED_MAX_N: return g_fused_max_n;
    case GEMMI_OPT_TC_PAIR: return g_tc_pair;
    case GEMMI_OPT_SMALL_MAX_MACS: return g_small_max_macs;
    case GEMMI_OPT_KARATSUBA: return g_karatsuba;
    case GEMMI_OPT_SPLIT_AHEAD: return g_split_ahead;
    case GEMMI_OPT_CONV_ROWS: return g_conv_rows;
    default: return -1;
  }
}

int gemmi_selftest_wait_timeout(int64_t timeout_us) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (timeout_us < 1 || timeout_us > 10000000) return set_error(GEMMI_EINVAL, "timeout must be in [1 us, 10 s]");
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  cudaError_t e = gemmi::launch_wait_timeout_probe(d->status, static_cast<uint64_t>(timeout_us) * 1000u, g_stream);
  if (e != cudaSuccess) return cuda_error(e, "wait probe launch");
  return read_status_locked(*d, true);
}

int gemmi_kernel_timing(int enable) {
  std::lock_guard<std::mutex> lock(g_mutex);
  g_timing = enable != 0;
  for (auto& t : g_timers) {
    timer_collect(t);
    t.total_ms = 0.0;
    t.launches = 0;
  }
  return GEMMI_OK;
}

int gemmi_kernel_time(int kernel, double* total_ms, int64_t* launches) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (kernel < 0 || kernel >= GEMMI_KERNEL_COUNT || total_ms == nullptr || launches == nullptr)
    return set_error(GEMMI_EINVAL, "bad kernel id or null output");
  timer_collect(g_timers[kernel]);
  *total_ms = g_timers[kernel].total_ms;
  *launches = g_timers[kernel].launches;
  return GEMMI_OK;
}

int gemmi_stream_read_probe(int64_t k, int64_t n, const int16_t* B, int64_t ldb, void* stream) {
  if (k < 0 || n < 0) return set_error(GEMMI_EINVAL, "negative matrix dimension");
  if (ldb < std::max<int64_t>(1, n)) return set_error(GEMMI_EINVAL, "ldb < max(1, n)");
  if (k == 0 || n == 0) return GEMMI_OK;
  if (B == nullptr) return set_error(GEMMI_EINVAL, "B is null");
  if (reinterpret_cast<uintptr_t>(B) % 16 != 0 || ldb % 8 != 0)
    return set_error(GEMMI_EINVAL, "the read probe needs a 16-byte aligned B with ldb % 8 == 0");
  if (k > (int64_t(1) << 31) || n > (int64_t(1) << 31)) return set_error(GEMMI_EINVAL, "matrix dimension too large");
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState* d = nullptr;
  int rc = device_state(&d);
  if (rc != GEMMI_OK) return rc;
  const char* why = "read probe launch";
  const cudaError_t e = gemmi::stream_read_probe(B, k, n, ldb, d->sm_count, d->status, timeout_ns(),
                                                 static_cast<cudaStream_t>(stream), &why);
  if (e != cudaSuccess) return cuda_error(e, why);
  return GEMMI_OK;
}

const char* gemmi_version(void) { return "gemmi 0.1 (sm_103a)"; }

}  // extern "C"
