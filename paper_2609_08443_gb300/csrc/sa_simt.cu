// CUDA-core kernels of the SA sketching step: the ragged planner, the
// fixed-order finalize reductions, and a fp32-arithmetic path used for fp32
// inputs and for shapes the tensor-core kernels do not cover.
//
// Forward (paper Sec. 3.1): per token the log-sum-exp over the P prototypes is
// computed first (sa_simt_lse), then blocks of 64 prototypes accumulate
// A[j,i] V_i with A[j,i] = exp(S[j,i] - lse_i) over a worker's tile range.
// Backward (chain rule of Sec. 3.1): per token tile dV and D_i = dV_i . v_i,
// then dK; dQ is accumulated per worker and head and reduced in worker order.
#include "sa_kernels.cuh"
#include "sa_simt_util.cuh"

namespace sa {

constexpr int ST = 32;    // tokens per tile on this path
constexpr int SPB = 64;   // prototypes per block
constexpr int SNT = 256;  // threads per block

// ------------------------------------------------------------------ planner
// One block: validates cu_seqlens and writes the per-head tile prefix.
__global__ void __launch_bounds__(1024) plan_kernel(const int32_t* __restrict__ cu, int B,
                                                    int64_t N, int T, void* ws,
                                                    int64_t* __restrict__ prefix, uint64_t wait_ns) {
  __shared__ int64_t warp_tot[32];
  __shared__ int64_t carry;
  __shared__ int bad;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) {
    carry = 0;
    bad = (cu[0] != 0) || (int64_t(cu[B]) != N);
    ws_header(ws)->timeout_site = 0;
    ws_header(ws)->wait_limit_ns = wait_ns;
  }
  __syncthreads();
  for (int base = 0; base < B; base += 1024) {
    const int b = base + tid;
    int64_t n = 0;
    if (b < B) {
      const int64_t L = int64_t(cu[b + 1]) - int64_t(cu[b]);
      if (L < 0) bad = 1;
      n = L > 0 ? (L + T - 1) / T : 0;
    }
    int64_t x = n;  // inclusive warp scan
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[wid] = x;
    __syncthreads();
    if (wid == 0) {
      int64_t s = warp_tot[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int64_t y = __shfl_up_sync(0xffffffffu, s, o);
        if (lane >= o) s += y;
      }
      warp_tot[lane] = s;  // inclusive over warps
    }
    __syncthreads();
    const int64_t before = carry + (wid > 0 ? warp_tot[wid - 1] : 0) + (x - n);
    if (b < B) prefix[b] = before;
    __syncthreads();
    if (tid == 0) carry += warp_tot[31];
    __syncthreads();
  }
  if (tid == 0) {
    prefix[B] = carry;
    ws_header(ws)->tiles_per_head = carry;
    ws_header(ws)->err = bad ? uint32_t(SA_ERR_BAD_SEQLENS) : 0u;
  }
}

// out[e] (+)= sum over k < n of src[off[k] + e] for e < PD, in k order; the
// first chunk of workers starts from zero, later chunks continue the running
// sum held in out (so the rounding is that of one sum in worker order).  A
// negative off[k] is a worker with an empty range.  float4 accesses when every
// address is 16-byte aligned.
__device__ __forceinline__ void sum_pieces(const float* __restrict__ src, const int64_t* off, int n,
                                           bool first, int64_t PD, float* __restrict__ out, int64_t e0,
                                           int64_t estep) {
  bool vec = (PD & 3) == 0 && ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(out)) & 15) == 0;
  if (vec) {
    const float4* s4 = reinterpret_cast<const float4*>(src);
    float4* o4 = reinterpret_cast<float4*>(out);
    for (int64_t e = e0; e < PD / 4; e += estep) {
      float4 s = first ? make_float4(0.f, 0.f, 0.f, 0.f) : o4[e];
      for (int k = 0; k < n; ++k) {
        if (off[k] < 0) continue;
        const float4 v = s4[off[k] / 4 + e];
        s.x += v.x;
        s.y += v.y;
        s.z += v.z;
        s.w += v.w;
      }
      o4[e] = s;
    }
    return;
  }
  for (int64_t e = e0; e < PD; e += estep) {
    float s = first ? 0.f : out[e];
    for (int k = 0; k < n; ++k)
      if (off[k] >= 0) s += src[off[k] + e];
    out[e] = s;
  }
}

// Sum of the pieces of every cut (user, head) segment, in worker order; zero
// sketch for empty users.  grid = B*H blocks.  The pieces' offsets are found
// once per block (range_begin divides in 64 bits), then summed element-wise.
__global__ void __launch_bounds__(256) finalize_sketch_kernel(const void* ws, const int64_t* prefix,
                                                              int B, int H, int P, int d, int W,
                                                              const float* __restrict__ partial,
                                                              float* __restrict__ sketch) {
  __shared__ int64_t off[256];
  if (ws_failed(ws)) return;
  const int64_t tph = reinterpret_cast<const WsHeader*>(ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int bh = blockIdx.x, b = bh / H, h = bh % H;
  const int64_t seg0 = int64_t(h) * tph + prefix[b], seg1 = int64_t(h) * tph + prefix[b + 1];
  const int64_t PD = int64_t(P) * d;
  float* out = sketch + int64_t(bh) * PD;
  if (seg0 == seg1) {
    for (int64_t e = threadIdx.x; e < PD; e += blockDim.x) out[e] = 0.f;
    return;
  }
  const int g0 = owner_of(total, W, seg0), g1 = owner_of(total, W, seg1 - 1);
  if (g0 == g1) return;  // written whole by its worker
  for (int c0 = g0; c0 <= g1; c0 += 256) {
    const int n = min(256, g1 - c0 + 1);
    __syncthreads();
    if (int(threadIdx.x) < n) {
      const int g = c0 + int(threadIdx.x);
      off[threadIdx.x] = range_begin(total, W, g) == range_begin(total, W, g + 1)
                             ? int64_t(-1)
                             : (int64_t(g) * 2 + partial_slot(total, W, g, seg0)) * PD;
    }
    __syncthreads();
    sum_pieces(partial, off, n, c0 == g0, PD, out, threadIdx.x, blockDim.x);
  }
}

// dQ[h] = sum over the workers whose range meets head h of their partial.
__global__ void __launch_bounds__(256) finalize_dq_kernel(const void* ws, int H, int P, int d, int W,
                                                          const float* __restrict__ dq_partial,
                                                          float* __restrict__ dQ) {
  __shared__ int64_t off[256];
  if (ws_failed(ws)) return;
  const int64_t tph = reinterpret_cast<const WsHeader*>(ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int h = blockIdx.y;
  const int64_t PD = int64_t(P) * d;
  float* out = dQ + int64_t(h) * PD;
  const int64_t e0 = blockIdx.x * int64_t(blockDim.x) + threadIdx.x, stride = int64_t(gridDim.x) * blockDim.x;
  if (tph == 0) {
    for (int64_t e = e0; e < PD; e += stride) out[e] = 0.f;
    return;
  }
  const int g0 = owner_of(total, W, int64_t(h) * tph), g1 = owner_of(total, W, int64_t(h + 1) * tph - 1);
  for (int c0 = g0; c0 <= g1; c0 += 256) {
    const int n = min(256, g1 - c0 + 1);
    __syncthreads();
    if (int(threadIdx.x) < n) {
      const int g = c0 + int(threadIdx.x);
      off[threadIdx.x] = range_begin(total, W, g) == range_begin(total, W, g + 1)
                             ? int64_t(-1)
                             : (int64_t(g) * H + h) * PD;
    }
    __syncthreads();
    sum_pieces(dq_partial, off, n, c0 == g0, PD, out, e0, stride);
  }
}

// ----------------------------------------------------------- lse (forward)
// One warp per (token, head): lse = log sum_j exp(scale * q_j . k), with the
// token's user's prototypes when the queries are per user.
template <typename T>
__global__ void __launch_bounds__(256) simt_lse_kernel(const T* __restrict__ K, const T* __restrict__ Q,
                                                       int64_t N, int H, int P, int d, float scale,
                                                       float* __restrict__ lse, const void* ws,
                                                       const int32_t* __restrict__ cu, int B, int uq) {
  __shared__ float ks[8][kMaxD];
  if (ws_failed(ws)) return;
  const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
  const int64_t w = int64_t(blockIdx.x) * 8 + wl;
  if (w >= N * H) return;
  const int64_t t = w / H;
  const int h = int(w - t * H);
  const T* krow = K + (t * H + h) * int64_t(d);
  for (int c = lane; c < d; c += 32) ks[wl][c] = ld_f32(krow + c);
  __syncwarp();
  constexpr int VN = Vec<T>::n;
  float m = -INFINITY, z = 0.f;
  const int qr = uq ? user_of_token(cu, B, t) * H + h : h;
  for (int j = lane; j < P; j += 32) {
    const T* q = Q + (int64_t(qr) * P + j) * d;
    float s = 0.f;
    for (int c = 0; c < d; c += VN) {
      float v[VN];
      Vec<T>::load(q + c, v);
#pragma unroll
      for (int k = 0; k < VN; ++k) s = fmaf(v[k], ks[wl][c + k], s);
    }
    s *= scale;
    if (s > m) {
      z = z * expf(m - s) + 1.f;
      m = s;
    } else {
      z += expf(s - m);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float z2 = __shfl_xor_sync(0xffffffffu, z, o);
    const float mm = fmaxf(m, m2);
    const float za = (m == -INFINITY) ? 0.f : z * expf(m - mm);
    const float zb = (m2 == -INFINITY) ? 0.f : z2 * expf(m2 - mm);
    m = mm;
    z = za + zb;
  }
  if (lane == 0) lse[t * H + h] = m + logf(z);
}

// --------------------------------------------------- aggregation (forward)
// grid = (W workers, ceil(P/64) prototype blocks).  Each block walks its
// worker's tile range and accumulates sketch rows p0..p0+63 in registers.
template <typename T>
__global__ void __launch_bounds__(SNT) simt_fwd_agg_kernel(Args a, const float* __restrict__ lse,
                                                           float* __restrict__ sketch) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  float* Qs = smem;              // [64][d+1]
  float* Ks = Qs + SPB * dp;     // [32][d+1]
  float* Vs = Ks + ST * dp;      // [32][d+1]
  float* As = Vs + ST * dp;      // [64][33]
  float* ls = As + SPB * 33;     // [32]
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int W = gridDim.x, w = blockIdx.x;
  const int p0 = blockIdx.y * SPB, np = min(SPB, P - p0);
  const int64_t tb = range_begin(total, W, w), te = range_begin(total, W, w + 1);
  if (tb >= te) return;
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const int tid = threadIdx.x, p = tid >> 2, cq = tid & 3;
  float acc[kMaxD / 4];
#pragma unroll
  for (int m = 0; m < kMaxD / 4; ++m) acc[m] = 0.f;
  int cur_q = -1;
  for (int64_t t = tb; t < te; ++t) {
    const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, ST);
    __syncthreads();
    const int qr = q_row(a, r.b, r.h);
    if (qr != cur_q) {
      stage_rows(Qs, Q + (int64_t(qr) * P + p0) * d, d, np, SPB, d);
      cur_q = qr;
    }
    stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
    stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
    if (tid < ST) ls[tid] = tid < r.n ? lse[(r.tok0 + tid) * H + r.h] : 0.f;
    __syncthreads();
    {
      float s[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] = 0.f;
      for (int c = 0; c < d; ++c) {
        const float q = Qs[p * dp + c];
#pragma unroll
        for (int k = 0; k < 8; ++k) s[k] = fmaf(q, Ks[(cq + 4 * k) * dp + c], s[k]);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = cq + 4 * k;
        As[p * 33 + i] = (i < r.n && p < np) ? expf(s[k] * a.scale - ls[i]) : 0.f;
      }
    }
    __syncthreads();
    for (int i = 0; i < ST; ++i) {
      const float w8 = As[p * 33 + i];
#pragma unroll
      for (int m = 0; m < kMaxD / 4; ++m) {
        const int c = cq + 4 * m;
        if (c < d) acc[m] = fmaf(w8, Vs[i * dp + c], acc[m]);
      }
    }
    if (t + 1 == te || t + 1 == r.seg1) {
      float* dst;
      if (r.seg0 >= tb && r.seg1 <= te) {
        dst = sketch + ((int64_t(r.b) * H + r.h) * P + p0 + p) * d;
      } else {
        const int slot = partial_slot(total, W, w, r.seg0);
        dst = a.partial + ((int64_t(w) * 2 + slot) * P + p0 + p) * d;
      }
#pragma unroll
      for (int m = 0; m < kMaxD / 4; ++m) {
        const int c = cq + 4 * m;
        if (c < d && p < np) dst[c] = acc[m];
        acc[m] = 0.f;
      }
    }
  }
}

// ----------------------------------------------------- backward per token
// One block per (head, user, tile of 32 tokens): dV, D_i = dV_i . v_i, dK.
template <typename T>
__global__ void __launch_bounds__(SNT) simt_bwd_tokens_kernel(Args a, const float* __restrict__ dsk,
                                                              const float* __restrict__ lse,
                                                              T* __restrict__ dK, T* __restrict__ dV,
                                                              float* __restrict__ Dco) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t t = blockIdx.x;
  if (t >= tph * H) return;
  float* Ks = smem;            // [32][d+1]
  float* Vs = Ks + ST * dp;    // [32][d+1]
  float* Qs = Vs + ST * dp;    // [64][d+1]
  float* Gs = Qs + SPB * dp;   // [64][d+1]
  float* As = Gs + SPB * dp;   // [64][33]
  float* ls = As + SPB * 33;   // [32]
  float* Ds = ls + ST;         // [32]
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, ST);
  const int tid = threadIdx.x;
  stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
  stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
  if (tid < ST) ls[tid] = tid < r.n ? lse[(r.tok0 + tid) * H + r.h] : 0.f;
  const float* G = dsk + (int64_t(r.b) * H + r.h) * int64_t(P) * d;
  const int ti = tid >> 3, cg = tid & 7;   // token / column group for dV, dK
  const int sp = tid >> 2, sq = tid & 3;   // prototype / token group for scores
  float acc[kMaxD / 8];
#pragma unroll
  for (int m = 0; m < kMaxD / 8; ++m) acc[m] = 0.f;
  // pass 1: dV_i = sum_j A[j,i] G_j
  for (int pc = 0; pc < P; pc += SPB) {
    const int np = min(SPB, P - pc);
    __syncthreads();
    stage_rows(Qs, Q + (int64_t(q_row(a, r.b, r.h)) * P + pc) * d, d, np, SPB, d);
    stage_rows_f32(Gs, G + int64_t(pc) * d, np, SPB, d);
    __syncthreads();
    {
      float s[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] = 0.f;
      for (int c = 0; c < d; ++c) {
        const float q = Qs[sp * dp + c];
#pragma unroll
        for (int k = 0; k < 8; ++k) s[k] = fmaf(q, Ks[(sq + 4 * k) * dp + c], s[k]);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = sq + 4 * k;
        As[sp * 33 + i] = (i < r.n && sp < np) ? expf(s[k] * a.scale - ls[i]) : 0.f;
      }
    }
    __syncthreads();
    for (int j = 0; j < np; ++j) {
      const float w8 = As[j * 33 + ti];
#pragma unroll
      for (int m = 0; m < kMaxD / 8; ++m) {
        const int c = cg + 8 * m;
        if (c < d) acc[m] = fmaf(w8, Gs[j * dp + c], acc[m]);
      }
    }
  }
  float part = 0.f;
#pragma unroll
  for (int m = 0; m < kMaxD / 8; ++m) {
    const int c = cg + 8 * m;
    if (c < d) part = fmaf(acc[m], Vs[ti * dp + c], part);
  }
  part += __shfl_xor_sync(0xffffffffu, part, 1);
  part += __shfl_xor_sync(0xffffffffu, part, 2);
  part += __shfl_xor_sync(0xffffffffu, part, 4);
  if (cg == 0) Ds[ti] = part;
  if (ti < r.n) {
    T* out = dV + ((r.tok0 + ti) * H + r.h) * int64_t(d);
#pragma unroll
    for (int m = 0; m < kMaxD / 8; ++m) {
      const int c = cg + 8 * m;
      if (c < d) st_from_f32(out + c, acc[m]);
    }
    if (cg == 0) Dco[(r.tok0 + ti) * H + r.h] = part;
  }
#pragma unroll
  for (int m = 0; m < kMaxD / 8; ++m) acc[m] = 0.f;
  // pass 2: dS = A o (G V^T - D), dK_i = scale sum_j dS[j,i] Q_j
  for (int pc = 0; pc < P; pc += SPB) {
    const int np = min(SPB, P - pc);
    __syncthreads();
    stage_rows(Qs, Q + (int64_t(q_row(a, r.b, r.h)) * P + pc) * d, d, np, SPB, d);
    stage_rows_f32(Gs, G + int64_t(pc) * d, np, SPB, d);
    __syncthreads();
    {
      float s[8], g[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] = g[k] = 0.f;
      for (int c = 0; c < d; ++c) {
        const float q = Qs[sp * dp + c], gg = Gs[sp * dp + c];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          s[k] = fmaf(q, Ks[(sq + 4 * k) * dp + c], s[k]);
          g[k] = fmaf(gg, Vs[(sq + 4 * k) * dp + c], g[k]);
        }
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = sq + 4 * k;
        const float A = expf(s[k] * a.scale - ls[i]);
        As[sp * 33 + i] = (i < r.n && sp < np) ? A * (g[k] - Ds[i]) : 0.f;
      }
    }
    __syncthreads();
    for (int j = 0; j < np; ++j) {
      const float ds = As[j * 33 + ti];
#pragma unroll
      for (int m = 0; m < kMaxD / 8; ++m) {
        const int c = cg + 8 * m;
        if (c < d) acc[m] = fmaf(ds, Qs[j * dp + c], acc[m]);
      }
    }
  }
  if (ti < r.n) {
    T* out = dK + ((r.tok0 + ti) * H + r.h) * int64_t(d);
#pragma unroll
    for (int m = 0; m < kMaxD / 8; ++m) {
      const int c = cg + 8 * m;
      if (c < d) st_from_f32(out + c, acc[m] * a.scale);
    }
  }
}

// ------------------------------------------------------------ backward dQ
// grid = (W workers, ceil(P/64)); per worker and head one fp32 partial of
// dQ[h] = scale sum_i dS[:, i] K_i, reduced later in worker order.
template <typename T>
__global__ void __launch_bounds__(SNT) simt_bwd_dq_kernel(Args a, const float* __restrict__ dsk,
                                                          const float* __restrict__ lse,
                                                          const float* __restrict__ Dco) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  float* Qs = smem;              // [64][d+1]
  float* Gs = Qs + SPB * dp;     // [64][d+1]
  float* Ks = Gs + SPB * dp;     // [32][d+1]
  float* Vs = Ks + ST * dp;      // [32][d+1]
  float* As = Vs + ST * dp;      // [64][33]
  float* ls = As + SPB * 33;     // [32]
  float* Ds = ls + ST;           // [32]
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int W = gridDim.x, w = blockIdx.x;
  const int p0 = blockIdx.y * SPB, np = min(SPB, P - p0);
  const int64_t tb = range_begin(total, W, w), te = range_begin(total, W, w + 1);
  if (tb >= te) return;
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const int tid = threadIdx.x, p = tid >> 2, cq = tid & 3;
  float acc[kMaxD / 4];
#pragma unroll
  for (int m = 0; m < kMaxD / 4; ++m) acc[m] = 0.f;
  int cur_h = -1, cur_b = -1, cur_q = -1;
  for (int64_t t = tb; t < te; ++t) {
    const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, ST);
    __syncthreads();
    const int qr = q_row(a, r.b, r.h);
    if (qr != cur_q) stage_rows(Qs, Q + (int64_t(qr) * P + p0) * d, d, np, SPB, d);
    cur_q = qr;
    if (r.h != cur_h || r.b != cur_b)
      stage_rows_f32(Gs, dsk + ((int64_t(r.b) * H + r.h) * P + p0) * d, np, SPB, d);
    cur_h = r.h;
    cur_b = r.b;
    stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
    stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, ST, d);
    if (tid < ST) {
      ls[tid] = tid < r.n ? lse[(r.tok0 + tid) * H + r.h] : 0.f;
      Ds[tid] = tid < r.n ? Dco[(r.tok0 + tid) * H + r.h] : 0.f;
    }
    __syncthreads();
    {
      float s[8], g[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] = g[k] = 0.f;
      for (int c = 0; c < d; ++c) {
        const float q = Qs[p * dp + c], gg = Gs[p * dp + c];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          s[k] = fmaf(q, Ks[(cq + 4 * k) * dp + c], s[k]);
          g[k] = fmaf(gg, Vs[(cq + 4 * k) * dp + c], g[k]);
        }
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = cq + 4 * k;
        const float A = expf(s[k] * a.scale - ls[i]);
        As[p * 33 + i] = (i < r.n && p < np) ? A * (g[k] - Ds[i]) : 0.f;
      }
    }
    __syncthreads();
    for (int i = 0; i < ST; ++i) {
      const float ds = As[p * 33 + i];
#pragma unroll
      for (int m = 0; m < kMaxD / 4; ++m) {
        const int c = cq + 4 * m;
        if (c < d) acc[m] = fmaf(ds, Ks[i * dp + c], acc[m]);
      }
    }
    // flush where the row of Q changes: at a head's end (shared queries: the
    // worker's partial of head h) or at a user segment's end (per-user queries:
    // dQ[b, h] when this worker holds the whole segment, else its partial slot)
    const bool flush = a.uq ? (t + 1 == te || t + 1 == r.seg1) : (t + 1 == te || (t + 1) / tph != t / tph);
    if (flush) {
      float* dst;
      if (!a.uq) {
        dst = a.dq_partial + ((int64_t(w) * H + r.h) * P + p0 + p) * d;
      } else if (r.seg0 >= tb && r.seg1 <= te) {
        dst = a.dq_user + ((int64_t(r.b) * H + r.h) * P + p0 + p) * d;
      } else {
        dst = a.partial + ((int64_t(w) * 2 + partial_slot(total, W, w, r.seg0)) * P + p0 + p) * d;
      }
#pragma unroll
      for (int m = 0; m < kMaxD / 4; ++m) {
        const int c = cq + 4 * m;
        if (c < d && p < np) dst[c] = acc[m] * a.scale;
        acc[m] = 0.f;
      }
    }
  }
}

// ------------------------------------------------------------------ launchers
static size_t smem_fwd_agg(int d) { return sizeof(float) * (size_t(SPB + 2 * ST) * (d + 1) + SPB * 33 + ST); }
static size_t smem_bwd_tok(int d) { return sizeof(float) * (size_t(2 * ST + 2 * SPB) * (d + 1) + SPB * 33 + 2 * ST); }
static size_t smem_bwd_dq(int d) { return smem_bwd_tok(d); }

cudaError_t launch_plan(const Args& a, int T, cudaStream_t st) {
  plan_kernel<<<1, 1024, 0, st>>>(a.cu, a.B, a.N, T, a.ws, a.prefix, wait_limit_ns());
  return cudaGetLastError();
}

cudaError_t launch_finalize_sketch(const Args& a, int W, float* sketch, cudaStream_t st) {
  if (a.B * int64_t(a.H) == 0) return cudaSuccess;
  finalize_sketch_kernel<<<a.B * a.H, 256, 0, st>>>(a.ws, a.prefix, a.B, a.H, a.P, a.d, W, a.partial, sketch);
  return cudaGetLastError();
}

cudaError_t launch_finalize_dq(const Args& a, int W, float* dQ, cudaStream_t st) {
  dim3 grid(32, a.H);
  finalize_dq_kernel<<<grid, 256, 0, st>>>(a.ws, a.H, a.P, a.d, W, a.dq_partial, dQ);
  return cudaGetLastError();
}

template <typename T>
static cudaError_t set_smem(const void* fn, size_t bytes) {
  return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
}

cudaError_t launch_simt_lse(const Args& a, float* lse, cudaStream_t st) {
  const int64_t warps = a.N * a.H;
  if (warps == 0) return cudaSuccess;
  const int64_t blocks = (warps + 7) / 8;
  if (a.dt == SA_BF16)
    simt_lse_kernel<__nv_bfloat16><<<unsigned(blocks), 256, 0, st>>>(
        static_cast<const __nv_bfloat16*>(a.K), static_cast<const __nv_bfloat16*>(a.Q), a.N, a.H, a.P, a.d,
        a.scale, lse, a.ws, a.cu, a.B, a.uq);
  else
    simt_lse_kernel<float><<<unsigned(blocks), 256, 0, st>>>(static_cast<const float*>(a.K),
                                                             static_cast<const float*>(a.Q), a.N, a.H, a.P,
                                                             a.d, a.scale, lse, a.ws, a.cu, a.B, a.uq);
  return cudaGetLastError();
}

cudaError_t launch_simt_fwd(const Args& a, int W, const float* lse, float* sketch, cudaStream_t st) {
  dim3 grid(W, (a.P + SPB - 1) / SPB);
  const size_t sm = smem_fwd_agg(a.d);
  cudaError_t e;
  if (a.dt == SA_BF16) {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_fwd_agg_kernel<__nv_bfloat16>), sm);
    if (e != cudaSuccess) return e;
    simt_fwd_agg_kernel<__nv_bfloat16><<<grid, SNT, sm, st>>>(a, lse, sketch);
  } else {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_fwd_agg_kernel<float>), sm);
    if (e != cudaSuccess) return e;
    simt_fwd_agg_kernel<float><<<grid, SNT, sm, st>>>(a, lse, sketch);
  }
  return cudaGetLastError();
}

cudaError_t launch_simt_bwd_tokens(const Args& a, const float* dsk, const float* lse, void* dK, void* dV,
                                   float* Dco, cudaStream_t st) {
  const int64_t max_tiles = int64_t(a.H) * ((a.N + ST - 1) / ST + a.B);
  if (a.N == 0) return cudaSuccess;
  const size_t sm = smem_bwd_tok(a.d);
  cudaError_t e;
  if (a.dt == SA_BF16) {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_bwd_tokens_kernel<__nv_bfloat16>), sm);
    if (e != cudaSuccess) return e;
    simt_bwd_tokens_kernel<__nv_bfloat16><<<unsigned(max_tiles), SNT, sm, st>>>(
        a, dsk, lse, static_cast<__nv_bfloat16*>(dK), static_cast<__nv_bfloat16*>(dV), Dco);
  } else {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_bwd_tokens_kernel<float>), sm);
    if (e != cudaSuccess) return e;
    simt_bwd_tokens_kernel<float><<<unsigned(max_tiles), SNT, sm, st>>>(a, dsk, lse, static_cast<float*>(dK),
                                                                        static_cast<float*>(dV), Dco);
  }
  return cudaGetLastError();
}

cudaError_t launch_simt_bwd_dq(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                               cudaStream_t st) {
  dim3 grid(W, (a.P + SPB - 1) / SPB);
  const size_t sm = smem_bwd_dq(a.d);
  cudaError_t e;
  if (a.dt == SA_BF16) {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_bwd_dq_kernel<__nv_bfloat16>), sm);
    if (e != cudaSuccess) return e;
    simt_bwd_dq_kernel<__nv_bfloat16><<<grid, SNT, sm, st>>>(a, dsk, lse, Dco);
  } else {
    e = set_smem<void>(reinterpret_cast<const void*>(&simt_bwd_dq_kernel<float>), sm);
    if (e != cudaSuccess) return e;
    simt_bwd_dq_kernel<float><<<grid, SNT, sm, st>>>(a, dsk, lse, Dco);
  }
  return cudaGetLastError();
}

int simt_tile_tokens() { return ST; }
int simt_workers(int num_sms, int P) {
  const int nb = (P + SPB - 1) / SPB;
  int w = (3 * num_sms + nb - 1) / nb;
  return w < 1 ? 1 : w;
}

}  // namespace sa
