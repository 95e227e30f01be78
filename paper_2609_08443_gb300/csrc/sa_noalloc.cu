// Allocation-free variant of the forward entry point.
//
// Some callers cannot hand this library a workspace: for example a plugin or
// custom-operator interface whose execute hook receives only its input and
// output buffers and must not allocate device memory itself, or a service that
// runs under a fixed device-memory budget planned ahead of time.  For them,
// sa_sketch_fwd_noalloc runs the same forward as sa_sketch_fwd but takes its
// scratch from a fixed array that lives in this library's device image.
#include <mutex>

#include "sa_kernels.cuh"

namespace {

// Upper bound of the scratch this entry point can use.  Every GPU on which the
// library is loaded holds this array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;  // 32 MiB

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_addr[64] = {nullptr};

// Device address of the array on the current device.  In host code the
// array's name is only a host-side stand-in, so the real address is looked up
// once per device (with that device current) and cached.
sa_status noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SA_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return SA_ERR_CUDA;
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
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
  // The planner kernel rewrites the array's header (error word, tile counts)
  // at the start of every call, and every other section is written before it
  // is read within the call, so nothing carried over from the last call is used.
  return sa_sketch_fwd(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, sketch, lse, scratch,
                       kNoAllocScratchBytes, stream);
}

}  // extern "C"
