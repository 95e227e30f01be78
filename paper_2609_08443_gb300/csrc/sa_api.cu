// Host side of libsa_sketch: argument checks, workspace sizing, the choice of
// kernels for a shape, launches on the caller's stream and the measurement
// hooks.  Declarations and the meaning of every argument: include/sa_sketch.h.
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include <cuda.h>

#include "sa_kernels.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace {

std::atomic<int> g_path{0};  // 0 = choose per shape, 1 = CUDA cores only, 2 = lse pass + slices

std::atomic<uint64_t> g_launches{0};

constexpr uint64_t kDefaultWaitNs = 2000000000ull;  // 2 s
std::atomic<uint64_t> g_wait_ns{kDefaultWaitNs};

int device_sms() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev] = n;
  }
  return cache[dev];
}

// ------------------------------------------------------------------ timing
struct TimingRec {
  cudaEvent_t a = nullptr, b = nullptr;
  int cls = 0;
  bool used = false;
};
std::mutex g_tmu;
bool g_timing = false;
std::vector<TimingRec> g_recs;
size_t g_nrec = 0;
constexpr size_t kMaxRecords = 4096;

TimingRec* timing_begin(int cls, cudaStream_t st) {
  std::lock_guard<std::mutex> lk(g_tmu);
  if (!g_timing || g_nrec >= kMaxRecords) return nullptr;
  if (g_recs.size() <= g_nrec) {
    TimingRec r;
    if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return nullptr;
    g_recs.push_back(r);
  }
  TimingRec* r = &g_recs[g_nrec++];
  r->cls = cls;
  r->used = cudaEventRecord(r->a, st) == cudaSuccess;
  return r;
}

void timing_end(TimingRec* r, cudaStream_t st) {
  if (r && r->used) r->used = cudaEventRecord(r->b, st) == cudaSuccess;
}

template <class F>
sa_status launch(int cls, cudaStream_t st, F&& f) {
  TimingRec* rec = (cls == SA_KERNEL_AUX) ? nullptr : timing_begin(cls, st);
  const cudaError_t e = f();
  g_launches.fetch_add(1, std::memory_order_relaxed);
  timing_end(rec, st);
  return e == cudaSuccess ? SA_OK : SA_ERR_CUDA;
}

#define SA_TRY(x)                      \
  do {                                 \
    const sa_status s_ = (x);          \
    if (s_ != SA_OK) return s_;        \
  } while (0)

// ------------------------------------------------------------------ planning
enum class Path { Simt, TcFwd, TcBwd };

struct Plan {
  Path fwd_path, bwd_path;
  int T_fwd, W_fwd, T_bwd, W_bwd;
  sa::WsLayout lay;
};

bool shape_ok(int B, int64_t N, int H, int P, int d, sa_dtype dt) {
  if (B < 1 || N < 0 || N >= (int64_t(1) << 31) || H < 1 || H > sa::kMaxH) return false;
  if (P < 1 || P > sa::kMaxP || d < 1 || d > sa::kMaxD) return false;
  if (dt != SA_F32 && dt != SA_BF16) return false;
  return d % (dt == SA_BF16 ? 8 : 4) == 0;
}

// allow_tc = false keeps every kernel on the CUDA cores: the tensor-core
// kernels take the softmax maximum on the raw scores, which is the maximum of
// the scaled scores only for scale >= 0.  With shared prototypes a negative
// scale is folded into them instead (fold_negative_scale), so only per-user
// queries with a negative scale need the CUDA cores.
Plan make_plan(int B, int64_t N, int H, int P, int d, sa_dtype dt, bool bwd, bool allow_tc = true) {
  Plan p{};
  const int sms = device_sms() > 0 ? device_sms() : 1;
  p.fwd_path = allow_tc && sa::tc_fwd_supported(P, d, dt) ? Path::TcFwd : Path::Simt;
  p.bwd_path = allow_tc && sa::tc_bwd_supported(P, d, dt) ? Path::TcBwd : Path::Simt;
  if (p.fwd_path == Path::TcFwd) {
    p.T_fwd = sa::tc_tile_tokens();
    p.W_fwd = sa::tc_fwd_workers(sms, P, d);
  } else {
    p.T_fwd = sa::simt_tile_tokens();
    p.W_fwd = sa::simt_workers(sms, P);
  }
  if (p.bwd_path == Path::TcBwd) {
    p.T_bwd = sa::tc_tile_tokens();
    p.W_bwd = sa::tc_bwd_workers(sms, P, d);
  } else {
    p.T_bwd = sa::simt_tile_tokens();
    p.W_bwd = sa::simt_workers(sms, P);
  }
  const int W = (bwd && p.W_bwd > p.W_fwd) ? p.W_bwd : p.W_fwd;
  p.lay = sa::ws_layout(B, N, H, P, d, W, bwd);
  return p;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Checks every entry point applies before choosing kernels.
sa_status check_args(const void* K, const void* V, const int32_t* cu, int B, int64_t N, const void* Q, int H, int P,
                     int d, float scale, sa_dtype dt, const void* ws) {
  if (!cu || !Q || !ws) return SA_ERR_INVALID_ARG;
  if (N > 0 && (!K || !V)) return SA_ERR_INVALID_ARG;
  if (!std::isfinite(scale)) return SA_ERR_INVALID_ARG;
  if (B < 1 || N < 0 || H < 1 || P < 1 || d < 1) return SA_ERR_INVALID_ARG;
  if (!shape_ok(B, N, H, P, d, dt)) return SA_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SA_ERR_INVALID_ARG;
  if ((K && !aligned16(K)) || (V && !aligned16(V)) || !aligned16(Q)) return SA_ERR_INVALID_ARG;
  return SA_OK;
}

sa_status check_common(const void* K, const void* V, const int32_t* cu, int B, int64_t N, const void* Q,
                       int H, int P, int d, float scale, sa_dtype dt, const void* ws, size_t ws_bytes,
                       bool bwd, int uq, Plan* plan) {
  SA_TRY(check_args(K, V, cu, B, N, Q, H, P, d, scale, dt, ws));
  *plan = make_plan(B, N, H, P, d, dt, bwd, scale >= 0.f || !uq);
  if (ws_bytes < plan->lay.total) return SA_ERR_WORKSPACE;
  return SA_OK;
}

sa::Args make_args(const void* K, const void* V, const int32_t* cu, int B, int64_t N, const void* Q, int H,
                   int P, int d, float scale, sa_dtype dt, void* ws, const sa::WsLayout& L) {
  sa::Args a{};
  char* base = static_cast<char*>(ws);
  a.K = K;
  a.V = V;
  a.Q = Q;
  a.cu = cu;
  a.B = B;
  a.N = N;
  a.H = H;
  a.P = P;
  a.d = d;
  a.scale = scale;
  a.dt = dt;
  a.ws = ws;
  a.prefix = reinterpret_cast<int64_t*>(base + L.tile_prefix);
  a.partial = reinterpret_cast<float*>(base + L.partial);
  a.dq_partial = reinterpret_cast<float*>(base + L.dq_partial);
  a.lse_scratch = reinterpret_cast<float*>(base + L.lse);
  a.lse_part = reinterpret_cast<float2*>(base + L.lse_part);
  a.uq = 0;
  a.dq_user = nullptr;
  return a;
}

// A negative scale on the tensor cores: S = scale Q K^T = (-scale) (-Q) K^T,
// and negating Q is exact, so every score the kernels form -- and the maximum
// they shift by -- is the one of the caller's problem; the kernels then see a
// positive scale.  The forward's sketch and lse are unchanged; dK = scale dS Q
// is unchanged too, while the kernels' dQ is the gradient for -Q, so the caller's
// dQ is its negation (negate_dq).
sa_status fold_negative_scale(sa::Args& a, const sa::WsLayout& L, cudaStream_t st) {
  if (!(a.scale < 0.f)) return SA_OK;
  void* qn = static_cast<char*>(a.ws) + L.qneg;
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_negate(a.Q, qn, int64_t(a.H) * a.P * a.d, a.dt, st); }));
  a.Q = qn;
  a.scale = -a.scale;
  return SA_OK;
}

sa_status negate_dq(float* dQ, int H, int P, int d, cudaStream_t st) {
  return launch(SA_KERNEL_AUX, st, [&] { return sa::launch_negate(dQ, dQ, int64_t(H) * P * d, SA_F32, st); });
}

}  // namespace

// ------------------------------------------------------- tensor-core helpers
namespace sa {

bool tc_path_enabled() { return g_path.load() != 1; }
uint64_t wait_limit_ns() { return g_wait_ns.load(); }
bool tc_fwd_sliced_selected() { return g_path.load() == 2; }
bool tc_narrow_selected() { return g_path.load() == 3; }

namespace tcc {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// K or V [N, H, D] bf16 -> boxes of [128 tokens][1 head][64 features], 128-byte swizzle;
// rows past N read as zero.
bool make_kv_map(CUtensorMap* m, const void* base, int64_t N, int H, int D) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || N <= 0) return false;
  const cuuint64_t dims[3] = {cuuint64_t(D), cuuint64_t(H), cuuint64_t(N)};
  const cuuint64_t strides[2] = {cuuint64_t(D) * 2, cuuint64_t(H) * D * 2};
  const cuuint32_t box[3] = {64, 1, 128};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Q [H, P, D] bf16 -> boxes of [box_rows prototypes][64 features] of one head.
bool make_q_map(CUtensorMap* m, const void* Q, int H, int P, int D, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {cuuint64_t(D), cuuint64_t(P), cuuint64_t(H)};
  const cuuint64_t strides[2] = {cuuint64_t(D) * 2, cuuint64_t(P) * D * 2};
  const cuuint32_t box[3] = {64, cuuint32_t(box_rows), 1};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(Q), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool device_is_sm103() {
  int dev = 0, major = 0, minor = 0, smem = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return false;
  return major == 10 && minor == 3 && smem >= 232448;
}

int device_sm_count() { return device_sms() > 0 ? device_sms() : 1; }

}  // namespace tcc
}  // namespace sa

extern "C" {

size_t sa_workspace_size(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd) {
  if (!shape_ok(B, N, H, P, d, dt)) return 0;
  // enough for either plan (a negative scale runs on the CUDA cores)
  const size_t tc = make_plan(B, N, H, P, d, dt, bwd != 0, true).lay.total;
  const size_t cc = make_plan(B, N, H, P, d, dt, bwd != 0, false).lay.total;
  return tc > cc ? tc : cc;
}

}  // extern "C"

namespace {

// Forward of both entry points; uq = 1: Q holds one [H, P, d] block per user.
sa_status fwd_impl(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N, const void* Q, int H,
                   int P, int d, float scale, sa_dtype dt, float* sketch, float* lse, void* workspace,
                   size_t ws_bytes, void* stream, int uq) {
  if (!sketch) return SA_ERR_INVALID_ARG;
  Plan plan;
  SA_TRY(check_common(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, ws_bytes, false, uq, &plan));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  sa::Args a = make_args(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, plan.lay);
  a.uq = uq;
  char* base = static_cast<char*>(workspace);
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_plan(a, plan.T_fwd, st); }));
  if (plan.fwd_path == Path::TcFwd) SA_TRY(fold_negative_scale(a, plan.lay, st));
  if (plan.fwd_path == Path::TcFwd) {
    float* l = lse;
    if (sa::tc_fwd_needs_lse_pass_d(P, d)) {
      if (!l) l = a.lse_scratch;
      SA_TRY(launch(SA_KERNEL_FWD_LSE, st, [&] { return sa::launch_tc_lse(a, l, st); }));
    }
    SA_TRY(launch(SA_KERNEL_FWD_MAIN, st, [&] { return sa::launch_tc_fwd(a, plan.W_fwd, sketch, l, st); }));
  } else {
    float* l = lse ? lse : reinterpret_cast<float*>(base + plan.lay.lse);
    SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_simt_lse(a, l, st); }));
    SA_TRY(launch(SA_KERNEL_FWD_MAIN, st, [&] { return sa::launch_simt_fwd(a, plan.W_fwd, l, sketch, st); }));
  }
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_finalize_sketch(a, plan.W_fwd, sketch, st); }));
  return SA_OK;
}

// Backward of both entry points; uq = 1: Q and dQ hold one [H, P, d] block per
// user, whose pieces from different workers are summed like the sketch's.
sa_status bwd_impl(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N, const void* Q, int H,
                   int P, int d, float scale, sa_dtype dt, const float* dsketch, const float* lse, void* dK,
                   void* dV, float* dQ, void* workspace, size_t ws_bytes, void* stream, int uq) {
  if (!dsketch || !dQ || (N > 0 && (!dK || !dV))) return SA_ERR_INVALID_ARG;
  Plan plan;
  SA_TRY(check_common(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, ws_bytes, true, uq, &plan));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  sa::Args a = make_args(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, plan.lay);
  a.uq = uq;
  a.dq_user = uq ? dQ : nullptr;
  const bool folded = plan.bwd_path == Path::TcBwd && scale < 0.f;
  // dQ from the per-worker pieces: summed over workers per head (shared
  // queries) or, per user, only for segments cut across workers
  auto finalize_dq = [&](int W) -> sa_status {
    if (uq) return launch(SA_KERNEL_AUX, st, [&] { return sa::launch_finalize_sketch(a, W, dQ, st); });
    SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_finalize_dq(a, W, dQ, st); }));
    return folded ? negate_dq(dQ, H, P, d, st) : SA_OK;
  };
  char* base = static_cast<char*>(workspace);
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_plan(a, plan.T_bwd, st); }));
  if (folded) SA_TRY(fold_negative_scale(a, plan.lay, st));
  const float* l = lse;
  if (!l) {
    float* scratch = reinterpret_cast<float*>(base + plan.lay.lse);
    if (plan.bwd_path == Path::TcBwd) {
      SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_tc_lse(a, scratch, st); }));
    } else {
      SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_simt_lse(a, scratch, st); }));
    }
    l = scratch;
  }
  if (plan.bwd_path == Path::TcBwd && sa::tc_bwd_split(P, d)) {
    // token side (dV, dK, D_i) over all prototypes, then dQ per prototype slice
    __nv_bfloat16* gbf = reinterpret_cast<__nv_bfloat16*>(base + plan.lay.gbf);
    float* Dco = reinterpret_cast<float*>(base + plan.lay.dcoef);
    const int Wq = sa::tc_bwd_dq_workers(sa::tcc::device_sm_count(), P);
    SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_tc_g_bf16(a, dsketch, gbf, st); }));
    SA_TRY(launch(SA_KERNEL_BWD_MAIN, st,
                  [&] { return sa::launch_tc_bwd_tok(a, plan.W_bwd, dsketch, gbf, l, Dco, dK, dV, st); }));
    SA_TRY(launch(SA_KERNEL_BWD_DQ, st, [&] { return sa::launch_tc_bwd_dq(a, Wq, dsketch, l, Dco, st); }));
    return finalize_dq(Wq);
  }
  if (plan.bwd_path == Path::TcBwd) {
    SA_TRY(launch(SA_KERNEL_BWD_MAIN, st,
                  [&] { return sa::launch_tc_bwd(a, plan.W_bwd, dsketch, l, dK, dV, st); }));
  } else {
    float* Dco = reinterpret_cast<float*>(base + plan.lay.dcoef);
    SA_TRY(launch(SA_KERNEL_BWD_MAIN, st,
                  [&] { return sa::launch_simt_bwd_tokens(a, dsketch, l, dK, dV, Dco, st); }));
    SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_simt_bwd_dq(a, plan.W_bwd, dsketch, l, Dco, st); }));
  }
  return finalize_dq(plan.W_bwd);
}

}  // namespace

extern "C" {

sa_status sa_sketch_fwd(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                        const void* Q, int H, int P, int d, float scale, sa_dtype dt, float* sketch,
                        float* lse, void* workspace, size_t ws_bytes, void* stream) {
  return fwd_impl(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, sketch, lse, workspace, ws_bytes, stream, 0);
}

sa_status sa_sketch_bwd(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                        const void* Q, int H, int P, int d, float scale, sa_dtype dt, const float* dsketch,
                        const float* lse, void* dK, void* dV, float* dQ, void* workspace, size_t ws_bytes,
                        void* stream) {
  return bwd_impl(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, dsketch, lse, dK, dV, dQ, workspace, ws_bytes,
                  stream, 0);
}

sa_status sa_sketch_fwd_per_user(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                                 const void* Q, int H, int P, int d, float scale, sa_dtype dt, float* sketch,
                                 float* lse, void* workspace, size_t ws_bytes, void* stream) {
  return fwd_impl(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, sketch, lse, workspace, ws_bytes, stream, 1);
}

sa_status sa_sketch_bwd_per_user(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                                 const void* Q, int H, int P, int d, float scale, sa_dtype dt, const float* dsketch,
                                 const float* lse, void* dK, void* dV, float* dQ, void* workspace,
                                 size_t ws_bytes, void* stream) {
  return bwd_impl(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, dsketch, lse, dK, dV, dQ, workspace, ws_bytes,
                  stream, 1);
}

// ------------------------------------------- key projection (Sec. 3.1, K = X W_K)
static size_t x_elem(sa_dtype dt) { return dt == SA_BF16 ? 2 : 4; }

// Extra workspace of the X entry points, after the step's own: Q' = Q W_K^T
// [H,P,d] (dt); for the backward also dK' [N,H,d] (dt) and dQ' [H,P,d] (fp32).
static size_t x_extra(int64_t N, int H, int P, int d, sa_dtype dt, bool bwd) {
  size_t b = sa::align256(size_t(H) * P * d * x_elem(dt));
  if (bwd) b += sa::align256(size_t(N) * H * d * x_elem(dt)) + sa::align256(size_t(H) * P * d * 4);
  return b;
}

size_t sa_workspace_size_x(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd) {
  const size_t base = sa_workspace_size(B, N, H, P, d, dt, bwd);
  return base == 0 ? 0 : base + x_extra(N, H, P, d, dt, bwd != 0);
}

sa_status sa_sketch_fwd_x(const void* X, const int32_t* cu_seqlens, int B, int64_t N, const void* Q,
                          const void* Wk, int H, int P, int d, float scale, sa_dtype dt, float* sketch, float* lse,
                          void* workspace, size_t ws_bytes, void* stream) {
  if (!Q || !Wk || !workspace || (N > 0 && !X)) return SA_ERR_INVALID_ARG;
  const size_t base = sa_workspace_size(B, N, H, P, d, dt, 0);
  if (base == 0) return shape_ok(B, N, H, P, d, dt) ? SA_ERR_INVALID_ARG : SA_ERR_UNSUPPORTED;
  if (ws_bytes < base + x_extra(N, H, P, d, dt, false)) return SA_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 || !aligned16(Wk)) return SA_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* Qf = static_cast<char*>(workspace) + base;
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_fold_wk(Q, Wk, H, P, d, dt, Qf, st); }));
  return fwd_impl(X, X, cu_seqlens, B, N, Qf, H, P, d, scale, dt, sketch, lse, workspace, base, stream, 0);
}

sa_status sa_sketch_bwd_x(const void* X, const int32_t* cu_seqlens, int B, int64_t N, const void* Q,
                          const void* Wk, int H, int P, int d, float scale, sa_dtype dt, const float* dsketch,
                          const float* lse, void* dX, float* dQ, float* dWk, void* workspace, size_t ws_bytes,
                          void* stream) {
  if (!Q || !Wk || !dQ || !dWk || !workspace || (N > 0 && (!X || !dX))) return SA_ERR_INVALID_ARG;
  const size_t base = sa_workspace_size(B, N, H, P, d, dt, 1);
  if (base == 0) return shape_ok(B, N, H, P, d, dt) ? SA_ERR_INVALID_ARG : SA_ERR_UNSUPPORTED;
  if (ws_bytes < base + x_extra(N, H, P, d, dt, true)) return SA_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 || !aligned16(Wk)) return SA_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* Qf = static_cast<char*>(workspace) + base;
  char* dKf = Qf + sa::align256(size_t(H) * P * d * x_elem(dt));
  float* dQf = reinterpret_cast<float*>(dKf + sa::align256(size_t(N) * H * d * x_elem(dt)));
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_fold_wk(Q, Wk, H, P, d, dt, Qf, st); }));
  // the step with K = V = X and prototypes Q': dK' to the workspace, dV into dX
  SA_TRY(bwd_impl(X, X, cu_seqlens, B, N, Qf, H, P, d, scale, dt, dsketch, lse, N > 0 ? dKf : nullptr, dX, dQf,
                  workspace, base, stream, 0));
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_add_into(dX, dKf, N * H * int64_t(d), dt, st); }));
  return launch(SA_KERNEL_AUX, st, [&] { return sa::launch_wk_grads(dQf, Q, Wk, H, P, d, dt, dQ, dWk, st); });
}

// ------------------------------ token-wise normalisation (Sec. 5.1, App. C)
namespace {

// Workspace of the token-wise entry points: header | tile prefix | cut-segment
// pieces [Wf][2][P][d] | dQ pieces [Wq][H][P][d] (bwd) | piece statistics
// float2 [Wf][2][P] | lse_tok [B][H][P] | D [B][H][P] (bwd) | sketch recomputed
// by the backward [B][H][P][d] (bwd) | bf16 copy of dsketch (bwd, tensor cores).
// The forward runs on the tensor cores (128-token tiles, Wf workers) where
// tc_tw_fwd_supported, else on CUDA cores (32-token tiles); the backward on the
// tensor cores (token side with Wb workers, dQ with Wq) where
// tc_tw_bwd_supported, else on CUDA cores (Wb = Wq workers).
struct TwLayout {
  sa::WsLayout base;
  size_t stat_part, lse_tok, dcoef, sketch, gbf, total;
  bool tc_fwd, tc_bwd;
  int Tf, Wf, Tb, Wb, Wq;
};

TwLayout tw_layout(int B, int H, int P, int d, sa_dtype dt, float scale, bool bwd) {
  TwLayout t{};
  const int sms = device_sms() > 0 ? device_sms() : 1;
  // a negative scale is folded into negated prototypes (fold_negative_scale)
  t.tc_fwd = sa::tc_tw_fwd_supported(P, d, dt, scale < 0.f ? -scale : scale);
  t.tc_bwd = sa::tc_tw_bwd_supported(P, d, dt);
  t.Tf = t.tc_fwd ? sa::tc_tile_tokens() : sa::tw_tile_tokens();
  t.Wf = t.tc_fwd ? sa::tc_tw_fwd_workers(sms, P) : sa::simt_workers(sms, P);
  t.Tb = t.tc_bwd ? sa::tc_tile_tokens() : sa::tw_tile_tokens();
  t.Wb = t.tc_bwd ? sa::tc_bwd_workers(sms, P, d) : sa::simt_workers(sms, P);
  t.Wq = t.tc_bwd ? sa::tc_bwd_dq_workers(sms, P) : t.Wb;
  sa::WsLayout& L = t.base;
  size_t off = sizeof(sa::WsHeader);
  L.tile_prefix = off;
  off = sa::align256(off + sizeof(int64_t) * size_t(B + 1));
  L.partial = off;
  off = sa::align256(off + sizeof(float) * size_t(t.Wf) * 2 * P * d);
  L.dq_partial = off;
  if (bwd) off = sa::align256(off + sizeof(float) * size_t(t.Wq) * H * P * d);
  t.stat_part = off;
  off = sa::align256(off + sizeof(float2) * size_t(t.Wf) * 2 * P);
  t.lse_tok = off;
  off = sa::align256(off + sizeof(float) * size_t(B) * H * P);
  t.dcoef = t.sketch = t.gbf = off;
  if (bwd) {
    off = sa::align256(off + sizeof(float) * size_t(B) * H * P);
    t.sketch = off;
    off = sa::align256(off + sizeof(float) * size_t(B) * H * P * d);
    t.gbf = off;
    if (t.tc_bwd) off = sa::align256(off + 2 * size_t(B) * H * P * d);
  }
  L.qneg = off;
  off = sa::align256(off + 4 * size_t(H) * P * d);
  L.lse = L.dcoef = L.gbf = L.lse_part = off;  // unused on this path
  L.total = t.total = off;
  return t;
}

sa_status tw_check(const void* K, const void* V, const int32_t* cu, int B, int64_t N, const void* Q, int H, int P,
                   int d, float scale, sa_dtype dt, const void* ws, size_t ws_bytes, bool bwd, TwLayout* lay) {
  SA_TRY(check_args(K, V, cu, B, N, Q, H, P, d, scale, dt, ws));
  *lay = tw_layout(B, H, P, d, dt, scale, bwd);
  return ws_bytes < lay->total ? SA_ERR_WORKSPACE : SA_OK;
}

// Plan for the forward's tiles, online-softmax sweep, merge of cut segments:
// sketch and lse_tok.
sa_status tw_forward(const sa::Args& a_in, const TwLayout& lay, float* sketch, float* lse_tok, cudaStream_t st) {
  sa::Args a = a_in;
  float2* stat = reinterpret_cast<float2*>(static_cast<char*>(a.ws) + lay.stat_part);
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_plan(a, lay.Tf, st); }));
  if (lay.tc_fwd) SA_TRY(fold_negative_scale(a, lay.base, st));  // the backward needs no fold
  if (lay.tc_fwd) {
    SA_TRY(launch(SA_KERNEL_FWD_MAIN, st,
                  [&] { return sa::launch_tc_tw_fwd(a, lay.Wf, sketch, lse_tok, stat, st); }));
  } else {
    SA_TRY(launch(SA_KERNEL_FWD_MAIN, st, [&] { return sa::launch_tw_fwd(a, lay.Wf, sketch, lse_tok, stat, st); }));
  }
  return launch(SA_KERNEL_AUX, st, [&] { return sa::launch_tw_finalize(a, lay.Wf, stat, sketch, lse_tok, st); });
}

}  // namespace

size_t sa_workspace_size_tokenwise(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd) {
  if (!shape_ok(B, N, H, P, d, dt)) return 0;
  return tw_layout(B, H, P, d, dt, 1.f, bwd != 0).total;
}

sa_status sa_sketch_fwd_tokenwise(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                                  const void* Q, int H, int P, int d, float scale, sa_dtype dt, float* sketch,
                                  float* lse_tok, void* workspace, size_t ws_bytes, void* stream) {
  if (!sketch) return SA_ERR_INVALID_ARG;
  TwLayout lay;
  SA_TRY(tw_check(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, ws_bytes, false, &lay));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  sa::Args a = make_args(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, lay.base);
  if (!lse_tok) lse_tok = reinterpret_cast<float*>(static_cast<char*>(workspace) + lay.lse_tok);
  return tw_forward(a, lay, sketch, lse_tok, st);
}

sa_status sa_sketch_bwd_tokenwise(const void* K, const void* V, const int32_t* cu_seqlens, int B, int64_t N,
                                  const void* Q, int H, int P, int d, float scale, sa_dtype dt, const float* sketch,
                                  const float* lse_tok, const float* dsketch, void* dK, void* dV, float* dQ,
                                  void* workspace, size_t ws_bytes, void* stream) {
  if (!dsketch || !dQ || (N > 0 && (!dK || !dV))) return SA_ERR_INVALID_ARG;
  if ((sketch && !aligned16(sketch)) || (lse_tok && !aligned16(lse_tok)) || !aligned16(dsketch))
    return SA_ERR_INVALID_ARG;
  TwLayout lay;
  SA_TRY(tw_check(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, ws_bytes, true, &lay));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(workspace);
  sa::Args a = make_args(K, V, cu_seqlens, B, N, Q, H, P, d, scale, dt, workspace, lay.base);
  if (!sketch || !lse_tok) {  // recompute both from the inputs
    float* O = reinterpret_cast<float*>(base + lay.sketch);
    float* l = reinterpret_cast<float*>(base + lay.lse_tok);
    SA_TRY(tw_forward(a, lay, O, l, st));
    sketch = O;
    lse_tok = l;
  }
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_plan(a, lay.Tb, st); }));
  float* D = reinterpret_cast<float*>(base + lay.dcoef);
  SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_tw_dcoef(a, sketch, dsketch, lay.tc_bwd, D, st); }));
  if (lay.tc_bwd) {
    __nv_bfloat16* gbf = reinterpret_cast<__nv_bfloat16*>(base + lay.gbf);
    SA_TRY(launch(SA_KERNEL_AUX, st, [&] { return sa::launch_tc_g_bf16(a, dsketch, gbf, st); }));
    SA_TRY(launch(SA_KERNEL_BWD_MAIN, st,
                  [&] { return sa::launch_tc_tw_bwd_tok(a, lay.Wb, gbf, lse_tok, D, dK, dV, st); }));
    SA_TRY(launch(SA_KERNEL_BWD_DQ, st,
                  [&] { return sa::launch_tc_tw_bwd_dq(a, lay.Wq, dsketch, lse_tok, D, st); }));
  } else {
    SA_TRY(launch(SA_KERNEL_BWD_MAIN, st,
                  [&] { return sa::launch_tw_bwd_tokens(a, dsketch, lse_tok, D, dK, dV, st); }));
    SA_TRY(launch(SA_KERNEL_BWD_DQ, st,
                  [&] { return sa::launch_tw_bwd_dq(a, lay.Wb, dsketch, lse_tok, D, st); }));
  }
  return launch(SA_KERNEL_AUX, st, [&] { return sa::launch_finalize_dq(a, lay.Wq, dQ, st); });
}

sa_status sa_get_device_error(const void* workspace, void* stream) {
  if (!workspace) return SA_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return SA_ERR_CUDA;
  uint32_t err = 0;
  if (cudaMemcpy(&err, workspace, sizeof(err), cudaMemcpyDeviceToHost) != cudaSuccess) return SA_ERR_CUDA;
  return static_cast<sa_status>(err);
}

const char* sa_status_string(sa_status s) {
  switch (s) {
    case SA_OK: return "ok";
    case SA_ERR_INVALID_ARG: return "invalid argument (null pointer, misaligned buffer or bad size)";
    case SA_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case SA_ERR_WORKSPACE: return "workspace smaller than sa_workspace_size()";
    case SA_ERR_CUDA: return "CUDA runtime error";
    case SA_ERR_TIMEOUT: return "a device pipeline wait gave up (bounded wait expired)";
    case SA_ERR_BAD_SEQLENS: return "cu_seqlens is not 0..N non-decreasing";
  }
  return "unknown status";
}

sa_status sa_timing_enable(int on) {
  std::lock_guard<std::mutex> lk(g_tmu);
  g_timing = on != 0;
  g_nrec = 0;
  return SA_OK;
}

sa_status sa_timing_read(sa_kernel_class k, double* total_ms, int64_t* launches) {
  if (!total_ms || !launches) return SA_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_tmu);
  double tot = 0.0;
  int64_t n = 0;
  for (size_t i = 0; i < g_nrec; ++i) {
    TimingRec& r = g_recs[i];
    if (r.cls != int(k) || !r.used) continue;
    if (cudaEventSynchronize(r.b) != cudaSuccess) return SA_ERR_CUDA;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) return SA_ERR_CUDA;
    tot += ms;
    ++n;
  }
  *total_ms = tot;
  *launches = n;
  return SA_OK;
}

uint64_t sa_launch_count(void) { return g_launches.load(); }

sa_status sa_set_wait_limit_ns(uint64_t ns) {
  if (ns > 4000000000ull) return SA_ERR_INVALID_ARG;
  g_wait_ns.store(ns == 0 ? kDefaultWaitNs : ns);
  return SA_OK;
}

sa_status sa_select_path(int path) {
  if (path < 0 || path > 3) return SA_ERR_INVALID_ARG;
  g_path.store(path);
  return SA_OK;
}

const char* sa_main_kernel_name(int P, int d, sa_dtype dt, int bwd) {
  if (bwd) return sa::tc_bwd_supported(P, d, dt) ? sa::tc_bwd_name(P, d) : "simt_bwd_tokens_kernel";
  return sa::tc_fwd_supported(P, d, dt) ? sa::tc_fwd_name(P, d) : "simt_fwd_agg_kernel";
}

sa_status sa_plan_host(const int32_t* cu, int B, int H, int tile, int n_workers, int64_t* begin) {
  if (!cu || !begin || B < 1 || H < 1 || tile < 1 || n_workers < 1) return SA_ERR_INVALID_ARG;
  if (cu[0] != 0) return SA_ERR_BAD_SEQLENS;
  int64_t tph = 0;
  for (int b = 0; b < B; ++b) {
    const int64_t L = int64_t(cu[b + 1]) - int64_t(cu[b]);
    if (L < 0) return SA_ERR_BAD_SEQLENS;
    tph += (L + tile - 1) / tile;
  }
  const int64_t total = tph * H;
  for (int w = 0; w <= n_workers; ++w) begin[w] = sa::range_begin(total, n_workers, w);
  return SA_OK;
}

sa_status sa_walk_host(const int32_t* cu, int B, int H, int tile, int n_workers, int32_t* user, int32_t* head,
                       int64_t* tok0, int32_t* ntok, int64_t cap) {
  if (!cu || !user || !head || !tok0 || !ntok || B < 1 || H < 1 || tile < 1 || n_workers < 1)
    return SA_ERR_INVALID_ARG;
  if (cu[0] != 0) return SA_ERR_BAD_SEQLENS;
  std::vector<int64_t> prefix(size_t(B) + 1, 0);
  for (int b = 0; b < B; ++b) {
    const int64_t L = int64_t(cu[b + 1]) - int64_t(cu[b]);
    if (L < 0) return SA_ERR_BAD_SEQLENS;
    prefix[size_t(b) + 1] = prefix[size_t(b)] + (L + tile - 1) / tile;
  }
  const int64_t tph = prefix[size_t(B)], total = tph * H;
  if (cap < total) return SA_ERR_INVALID_ARG;
  // each worker's range as the kernels walk it: the first tile located by the
  // search, then 128-token steps inside a segment and the forward scan across
  // segment ends
  for (int w = 0; w < n_workers; ++w) {
    const int64_t tb = sa::range_begin(total, n_workers, w), te = sa::range_begin(total, n_workers, w + 1);
    sa::TileRef r{};
    for (int64_t t = tb; t < te; ++t) {
      if (t == tb) {
        r = sa::locate_tile(t, tph, prefix.data(), cu, B, tile);
      } else if (t < r.seg1) {
        r.tok0 += tile;
        const int64_t left = r.L - (t - r.seg0) * tile;
        r.n = int(left < tile ? left : tile);
      } else {
        r = sa::locate_next_segment(t, r.h, r.b, tph, prefix.data(), cu, B, tile);
      }
      user[t] = r.b;
      head[t] = r.h;
      tok0[t] = r.tok0;
      ntok[t] = r.n;
    }
  }
  return SA_OK;
}

}  // extern "C"
