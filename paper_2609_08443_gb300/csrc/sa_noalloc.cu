// Allocation-free variant of the forward entry point.
//
// Some callers cannot hand this library a workspace: for example a plugin or
// custom-operator interface whose execute hook receives only its input and
// output buffers and must not allocate device memory itself, or a service that
// runs under a fixed device-memory budget planned ahead of time.  For them,
// sa_sketch_fwd_noalloc runs the same forward as sa_sketch_fwd but takes its
// scratch from a fixed array that lives in this library's device image.
#include <mutex>

#include <cuda.h>

#include "sa_kernels.cuh"

namespace {

// Upper bound of the scratch this entry point can use.  Every GPU on which the
// library is loaded holds this array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;  // 32 MiB

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

CtxGetCurrentFn ctx_get_current_fn() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  return fn;
}

struct ScratchAddr {
  CUcontext ctx = nullptr;
  void* ptr = nullptr;
};
std::mutex g_noalloc_mu;
ScratchAddr g_noalloc_addr[64];

// Device address of the array in the current device's context.  In host code
// the array's name is only a host-side stand-in, so the real address is looked
// up with the device current and cached per device, together with the context
// it belongs to: after a device reset the context changes and the address is
// looked up again instead of reusing one that points into freed memory.
sa_status noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SA_ERR_CUDA;
  CtxGetCurrentFn get = ctx_get_current_fn();
  if (!get) return SA_ERR_CUDA;
  CUcontext ctx = nullptr;  // null until the runtime has made a context current in this thread
  if (get(&ctx) != CUDA_SUCCESS) return SA_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  ScratchAddr& c = g_noalloc_addr[dev];
  if (ctx == nullptr || c.ptr == nullptr || c.ctx != ctx) {
    // the lookup makes the device's primary context current if none is
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return SA_ERR_CUDA;
    if (get(&ctx) != CUDA_SUCCESS || ctx == nullptr) return SA_ERR_CUDA;
    c.ctx = ctx;
    c.ptr = p;
  }
  *out = c.ptr;
  return SA_OK;
}

}  // namespace

extern "C" {

size_t sa_noalloc_scratch_bytes(void) { return kNoAllocScratchBytes; }

sa_status sa_sketch_fwd_noalloc(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                                const void* Q, int H, int P, int d, float scale, sa_dtype dt, float* sketch,
                                float* lse, void* stream) {
  const size_t need = sa_workspace_size(B, N, H, P, d, dt, 0);
  if (need == 0) return SA_ERR_UNSUPPORTED;
  if (need > kNoAllocScratchBytes) return SA_ERR_WORKSPACE;
  void* scratch = nullptr;
  const sa_status st = noalloc_scratch(&scratch);
  if (st != SA_OK) return st;
  // The planner kernel rewrites the array's header (error word, tile counts,
  // wait limit) at the start of every call, and every other section is written
  // before it is read within the call, so nothing carried over from the last
  // call is used -- including the error word of a call that failed.
  return sa_sketch_fwd(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, sketch, lse, scratch,
                       kNoAllocScratchBytes, stream);
}

sa_status sa_noalloc_get_device_error(void* stream) {
  void* scratch = nullptr;
  const sa_status st = noalloc_scratch(&scratch);
  if (st != SA_OK) return st;
  return sa_get_device_error(scratch, stream);
}

}  // extern "C"
