// k_noalloc.cu -- an allocation-free variant of the stand-alone adapter backward.
//
// ra_adapter_backward takes a caller-provided scratch buffer.  Some callers cannot provide
// one: plug-in hosts that hand a kernel only its input and output buffers (custom-operator
// slots of serving runtimes) have no allocator to call, and loops that forbid allocation
// once running cannot afford cudaMalloc, which can block, synchronise the device or fail
// at any time.  This variant keeps its scratch in a fixed device array instead.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/ringada.h"
#include "kernels.h"

namespace {

// Scratch shared by every call of ra_adapter_backward_noalloc on a device.  It lives as
// long as the library stays loaded on every GPU that loads it.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;  // 16 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
// per device: the array's address and the CUDA context it was looked up in.  A module
// variable's address belongs to the context; after a device reset (or any other teardown
// and re-creation of the primary context) the cached address would point into a dead
// context, so the lookup is redone whenever the current context differs.
void* g_scratch_ptr[kMaxDevices] = {};
CUcontext g_scratch_ctx[kMaxDevices] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  }
  return fn;
}

// Device address of the array on the current device (host code cannot use the array's
// name as an address: it names a host-side stand-in).  Looked up once per device and
// context.
ra_status scratch_on_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RA_ERR_CUDA;
  CtxGetCurrentFn get = ctx_get_current();
  if (!get) return RA_ERR_CUDA;
  CUcontext cur = nullptr;
  if (get(&cur) != CUDA_SUCCESS) return RA_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!cur || !g_scratch_ptr[dev] || g_scratch_ctx[dev] != cur) {
    // the lookup also makes the device's primary context current if none was
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return RA_ERR_CUDA;
    if (get(&cur) != CUDA_SUCCESS || !cur) return RA_ERR_CUDA;
    g_scratch_ptr[dev] = p;
    g_scratch_ctx[dev] = cur;
  }
  *out = g_scratch_ptr[dev];
  return RA_OK;
}

inline size_t up256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

extern "C" {

size_t ra_adapter_backward_noalloc_capacity(void) { return kNoAllocScratchBytes; }

ra_status ra_adapter_backward_noalloc(const float* g_dev, const float* h_dev, const float* z_dev,
                                      const float* W_down_dev, const float* W_up_dev, int32_t T,
                                      int32_t H, int32_t m, float* dW_down_dev, float* dW_up_dev,
                                      float* dh_dev, ra_stream_t stream) {
  if (!g_dev || !h_dev || !z_dev || !W_down_dev || !W_up_dev || !dW_down_dev || !dW_up_dev)
    return RA_ERR_ARG;
  if (T < 1 || H < 1 || m < 1) return RA_ERR_ARG;
  if (m > 128) return RA_ERR_SHAPE;
  const size_t part = up256(ra::adapter_bwd_partials_floats(T, H, m) * 4);
  const size_t dz = up256((size_t)T * m * 4);
  const size_t wt = up256((size_t)H * m * 4);
  if (part + dz + 2 * wt > kNoAllocScratchBytes) return RA_ERR_NOMEM;  // beyond the fixed array
  void* base = nullptr;
  ra_status s = scratch_on_current_device(&base);
  if (s != RA_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  char* p = (char*)base;
  float* partials = (float*)p;
  float* dzb = (float*)(p + part);
  float* WuT = (float*)(p + part + dz);
  float* WdT = (float*)(p + part + dz + wt);
  // every scratch element read below is written earlier in this same call, so nothing
  // left over from a previous call is ever read
  if (ra::transpose_f32(W_up_dev, WuT, ra::DT_F32, m, H, m, st) != cudaSuccess) return RA_ERR_CUDA;
  if (ra::transpose_f32(W_down_dev, WdT, ra::DT_F32, H, m, H, st) != cudaSuccess) return RA_ERR_CUDA;
  ra::AdapterBwdArgs a;
  a.T = T; a.H = H; a.m = m; a.dtype = ra::DT_F32;
  a.g = g_dev; a.h = h_dev; a.z = z_dev; a.WuT = WuT; a.WdT = WdT; a.dz = dzb;
  a.dh = dh_dev; a.dh_dtype = ra::DT_F32; a.dWd = dW_down_dev; a.dWu = dW_up_dev;
  a.partials = partials;
  return ra::adapter_bwd(a, st) == cudaSuccess ? RA_OK : RA_ERR_CUDA;
}

}  // extern "C"
