// dvi_linear_noalloc: the projection kernel (Y = X W^T) for callers that
// cannot allocate device memory.
//
// Some callers may not call cudaMalloc at all, or may not own an allocator:
// code running inside another framework's memory pool or a fixed memory
// budget, plug-ins handed only input and output buffers, or processes that
// must not grow their device footprint after start-up.  dvi_linear needs a
// context whose workspace holds the split-K scratch; this variant keeps that
// scratch in fixed arrays of this file instead, so the caller passes only
// the weight, the input and the output.
//
// The arrays are static device memory: every GPU that loads the library
// holds them (8 MiB + 16 KiB) until the process exits.  Host code cannot use
// the array names as device addresses, so the first call on each device
// looks their addresses up with cudaGetSymbolAddress while that device is
// current, and later calls on that device reuse them.
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace {

// Capacity of the shared scratch: partial sums of K-split tiles, then the
// per-tile arrival counters (which must start every call at zero).
constexpr size_t kNoAllocPartFloats = static_cast<size_t>(1) << 21;   // 8 MiB
constexpr int kNoAllocCounters = 4096;

static __device__ __align__(256) float g_noalloc_part[kNoAllocPartFloats];
static __device__ __align__(256) int g_noalloc_counters[kNoAllocCounters];

struct DeviceScratch {
  bool ready = false;
  float* part = nullptr;
  int* counters = nullptr;
  int n_sms = 0;
};

constexpr int kMaxDevices = 64;
DeviceScratch g_scratch[kMaxDevices];
std::mutex g_scratch_mu;

// Addresses of the scratch arrays on the current device, looked up once per
// device (the lookup may load the module, so it must not happen while a
// stream is being captured).
dvi_status current_scratch(DeviceScratch* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return DVI_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  DeviceScratch& s = g_scratch[dev];
  if (!s.ready) {
    void* part = nullptr;
    void* ctr = nullptr;
    int n = 0;
    if (cudaGetSymbolAddress(&part, g_noalloc_part) != cudaSuccess) return DVI_ERR_CUDA;
    if (cudaGetSymbolAddress(&ctr, g_noalloc_counters) != cudaSuccess) return DVI_ERR_CUDA;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      return DVI_ERR_CUDA;
    s.part = static_cast<float*>(part);
    s.counters = static_cast<int*>(ctr);
    s.n_sms = n;
    s.ready = true;
  }
  *out = s;
  return DVI_OK;
}

}  // namespace

extern "C" dvi_status dvi_linear_noalloc(int dtype, const void* d_w, int n_out, int k_in, const float* d_x,
                                         int m_rows, float* d_y, dvi_stream stream) {
  using namespace dvi;
  if ((dtype != DVI_F32 && dtype != DVI_BF16) || !d_w || !d_x || !d_y || n_out < 1 || k_in < 1 || m_rows < 1 ||
      m_rows > kMaxTokens)
    return DVI_ERR_INVALID_ARG;
  const bool tc = dtype == DVI_BF16;
  if (tc && (k_in % 8 || (reinterpret_cast<uintptr_t>(d_w) & 15u) || (reinterpret_cast<uintptr_t>(d_x) & 15u)))
    return DVI_ERR_INVALID_ARG;
  // An error left pending by the caller's earlier CUDA work must not be
  // reported as this call's launch failure.
  cudaGetLastError();
  DeviceScratch s;
  const dvi_status rc = current_scratch(&s);
  if (rc != DVI_OK) return rc;

  ProjArgs a{};
  a.flavor = EPI_HEAD;
  a.dtype = dtype;
  a.M = m_rows;
  a.n_pad = (m_rows + 15) / 16 * 16;
  a.n_out = n_out;
  a.K = k_in;
  a.n_ttiles = 1;
  a.rows_per_seq = 1;
  a.b_mode = B_SOFT_F32;
  a.prefetch_a = 1;
  a.act = d_x;
  a.ld_act = k_in;
  a.w0 = d_w;
  a.logits_mode = 1;
  a.logits_out = d_y;
  a.ld_logits = n_out;
  a.part = s.part;
  a.counters = s.counters;
  plan_splits(a, s.n_sms, tc);
  const int n_counters = a.n_tiles * (tc ? 1 : (m_rows + kChunk - 1) / kChunk);
  if (proj_partial_floats(a, tc) > kNoAllocPartFloats || n_counters > kNoAllocCounters) {
    fprintf(stderr,
            "dvi_linear_noalloc: %d x %d weight with %d rows needs %zu floats of split-K scratch and %d "
            "counters; the fixed scratch holds %zu and %d\n",
            n_out, k_in, m_rows, proj_partial_floats(a, tc), n_counters, kNoAllocPartFloats, kNoAllocCounters);
    return DVI_ERR_CAPACITY;
  }
  ProjMaps maps{};
  if (tc && !make_weight_map(&maps.m0, d_w, n_out, k_in)) return DVI_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // A call that stopped early could leave counters raised; start from zero.
  if (cudaMemsetAsync(s.counters, 0, sizeof(int) * n_counters, st) != cudaSuccess) return DVI_ERR_CUDA;
  if (launch_proj(a, tc ? &maps : nullptr, st) != cudaSuccess) return DVI_ERR_CUDA;
  return DVI_OK;
}
