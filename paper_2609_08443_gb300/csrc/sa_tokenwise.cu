// Token-wise ("vanilla") normalisation of the sketching step, the comparison of
// paper Sec. 5.1 and App. C: the same scores S = scale Q K_b^T, normalised over
// the user's tokens instead of over the prototypes,
//     A[j, :] = softmax over i of S[j, i]    (weights p(i | j)),
//     sketch[b, h] = A V_b.
// Each prototype row now needs a statistic over all of the user's tokens, which
// the ragged tiling spreads across workers, so the forward keeps per prototype
// a running maximum m_j and sum l_j (online softmax, as in FlashAttention with
// the P prototypes as queries) and rescales its accumulator when m_j grows.  A
// worker that holds a whole (user, head) segment writes O_j = acc_j / l_j and
// lse_j = m_j + log l_j; a cut segment leaves (acc_j, m_j, l_j) per worker, and
// tw_finalize merges those in worker order (bitwise reproducible).
//
// Backward (chain rule; the paper prints none), with G = dsketch[b, h]:
//     dV_i = sum_j A[j,i] G_j,    D_j = sum_i A[j,i] (G_j . v_i) = G_j . O_j,
//     dS[j,i] = A[j,i] (G_j . v_i - D_j),
//     dK_i = scale sum_j dS[j,i] q_j,    dQ[h] = scale sum_b sum_i dS[:, i] k_i.
// D_j depends only on the forward's output, so the token side (dV, dK) needs a
// single pass over the prototypes; dQ is accumulated per worker and head and
// reduced in worker order by the shared finalize kernel.
//
// CUDA cores, fp32 arithmetic, inputs fp32 or bf16 (widened on load).
#include "sa_simt_util.cuh"

namespace sa {

constexpr int TT = 32;    // tokens per tile (the plan's tile size on this path)
constexpr int TPB = 64;   // prototypes per block
constexpr int TNT = 256;  // threads per block

// ------------------------------------------------------------------ forward
// grid = (W workers, ceil(P / 64)); thread (p = tid / 4, cq = tid % 4) owns
// prototype p0 + p and the sketch columns cq, cq + 4, ...
template <typename T>
__global__ void __launch_bounds__(TNT) tw_fwd_kernel(Args a, float* __restrict__ sketch, float* __restrict__ lse_tok,
                                                     float2* __restrict__ stat_part) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  float* Qs = smem;             // [64][d+1]
  float* Ks = Qs + TPB * dp;    // [32][d+1]
  float* Vs = Ks + TT * dp;     // [32][d+1]
  float* As = Vs + TT * dp;     // [64][33]
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int W = gridDim.x, w = blockIdx.x;
  const int p0 = blockIdx.y * TPB, np = min(TPB, P - p0);
  const int64_t tb = range_begin(total, W, w), te = range_begin(total, W, w + 1);
  if (tb >= te) return;
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const int tid = threadIdx.x, p = tid >> 2, cq = tid & 3;
  float acc[kMaxD / 4];
#pragma unroll
  for (int k = 0; k < kMaxD / 4; ++k) acc[k] = 0.f;
  float m = -INFINITY, l = 0.f;  // running max of S[p, .] and this thread's share of the sum
  int cur_q = -1;
  for (int64_t t = tb; t < te; ++t) {
    const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, TT);
    __syncthreads();
    const int qr = q_row(a, r.b, r.h);
    if (qr != cur_q) {
      stage_rows(Qs, Q + (int64_t(qr) * P + p0) * d, d, np, TPB, d);
      cur_q = qr;
    }
    stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
    stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
    __syncthreads();
    float s[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) s[k] = 0.f;
    for (int c = 0; c < d; ++c) {
      const float q = Qs[p * dp + c];
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] = fmaf(q, Ks[(cq + 4 * k) * dp + c], s[k]);
    }
    float mt = -INFINITY;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      s[k] = (cq + 4 * k < r.n && p < np) ? s[k] * a.scale : -INFINITY;
      mt = fmaxf(mt, s[k]);
    }
    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 1));
    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 2));
    const float mn = fmaxf(m, mt);
    const float sh = (mn == -INFINITY) ? 0.f : mn;  // rows past P stay all-zero
    const float alpha = expf(m - sh);
    l *= alpha;
#pragma unroll
    for (int k = 0; k < kMaxD / 4; ++k) acc[k] *= alpha;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float e = expf(s[k] - sh);
      l += e;
      As[p * 33 + cq + 4 * k] = e;
    }
    m = mn;
    __syncthreads();
    for (int i = 0; i < TT; ++i) {
      const float e = As[p * 33 + i];
#pragma unroll
      for (int k = 0; k < kMaxD / 4; ++k) {
        const int c = cq + 4 * k;
        if (c < d) acc[k] = fmaf(e, Vs[i * dp + c], acc[k]);
      }
    }
    if (t + 1 == te || t + 1 == r.seg1) {
      float lt = l + __shfl_xor_sync(0xffffffffu, l, 1);
      lt += __shfl_xor_sync(0xffffffffu, lt, 2);
      const int64_t row = int64_t(r.b) * H + r.h;
      if (p < np) {
        if (r.seg0 >= tb && r.seg1 <= te) {
          float* dst = sketch + (row * P + p0 + p) * d;
          const float inv = 1.f / lt;
#pragma unroll
          for (int k = 0; k < kMaxD / 4; ++k) {
            const int c = cq + 4 * k;
            if (c < d) dst[c] = acc[k] * inv;
          }
          if (cq == 0) lse_tok[row * P + p0 + p] = m + logf(lt);
        } else {
          const int64_t slot = int64_t(w) * 2 + partial_slot(total, W, w, r.seg0);
          float* dst = a.partial + (slot * P + p0 + p) * d;
#pragma unroll
          for (int k = 0; k < kMaxD / 4; ++k) {
            const int c = cq + 4 * k;
            if (c < d) dst[c] = acc[k];
          }
          if (cq == 0) stat_part[slot * P + p0 + p] = make_float2(m, lt);
        }
      }
#pragma unroll
      for (int k = 0; k < kMaxD / 4; ++k) acc[k] = 0.f;
      m = -INFINITY;
      l = 0.f;
    }
  }
}

// Merge of the pieces of every cut (user, head) segment in worker order:
// M = max_g m_g, L = sum_g l_g e^(m_g - M), O = sum_g acc_g e^(m_g - M) / L,
// lse = M + log L.  Empty users: zero sketch and lse = -inf.  grid = B*H.
__global__ void __launch_bounds__(256) tw_finalize_kernel(const void* ws, const int64_t* prefix, int B, int H,
                                                          int P, int d, int W, const float* __restrict__ partial,
                                                          const float2* __restrict__ stat_part,
                                                          float* __restrict__ sketch, float* __restrict__ lse_tok) {
  if (ws_failed(ws)) return;
  const int64_t tph = reinterpret_cast<const WsHeader*>(ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int bh = blockIdx.x, b = bh / H, h = bh % H;
  const int64_t seg0 = int64_t(h) * tph + prefix[b], seg1 = int64_t(h) * tph + prefix[b + 1];
  const int64_t PD = int64_t(P) * d;
  float* out = sketch + int64_t(bh) * PD;
  if (seg0 == seg1) {
    for (int64_t e = threadIdx.x; e < PD; e += blockDim.x) out[e] = 0.f;
    for (int j = threadIdx.x; j < P; j += blockDim.x) lse_tok[int64_t(bh) * P + j] = -INFINITY;
    return;
  }
  const int g0 = owner_of(total, W, seg0), g1 = owner_of(total, W, seg1 - 1);
  if (g0 == g1) return;  // written whole by its worker
  for (int64_t e = threadIdx.x; e < PD; e += blockDim.x) {
    const int j = int(e / d);
    float M = -INFINITY;
    for (int g = g0; g <= g1; ++g) {
      if (range_begin(total, W, g) == range_begin(total, W, g + 1)) continue;
      const int64_t slot = int64_t(g) * 2 + partial_slot(total, W, g, seg0);
      M = fmaxf(M, stat_part[slot * P + j].x);
    }
    float L = 0.f, o = 0.f;
    for (int g = g0; g <= g1; ++g) {
      if (range_begin(total, W, g) == range_begin(total, W, g + 1)) continue;
      const int64_t slot = int64_t(g) * 2 + partial_slot(total, W, g, seg0);
      const float2 st = stat_part[slot * P + j];
      const float f = expf(st.x - M);
      L = fmaf(st.y, f, L);
      o = fmaf(partial[slot * PD + e], f, o);
    }
    out[e] = o / L;
    if (e - int64_t(j) * d == 0) lse_tok[int64_t(bh) * P + j] = M + logf(L);
  }
}

// D[r] = sum_c G[r, c] O[r, c] for every row r of [B*H*P, d]; one warp per row.
// With round_g, G is taken rounded to bf16: the tensor-core backward forms
// dA = G V^T from that rounded copy, and dS = A o (dA - D) cancels exactly
// only if D is built from the same G (a one-token user has dS = 0).
__global__ void __launch_bounds__(256) tw_dcoef_kernel(const void* ws, const float* __restrict__ O,
                                                       const float* __restrict__ G, int64_t rows, int d,
                                                       int round_g, float* __restrict__ D) {
  if (ws_failed(ws)) return;
  const int64_t r = int64_t(blockIdx.x) * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  float s = 0.f;
  for (int c = lane; c < d; c += 32) {
    const float g = round_g ? __bfloat162float(__float2bfloat16_rn(G[r * d + c])) : G[r * d + c];
    s = fmaf(g, O[r * d + c], s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) D[r] = s;
}

// ------------------------------------------------------ backward, token side
// One block per (head, user, tile of 32 tokens): dV and dK in one pass over the
// prototypes, 64 at a time.  Thread (ti = tid / 8, cg = tid % 8) owns token ti
// and columns cg, cg + 8, ...; for the scores thread (sp = tid / 4, sq = tid % 4)
// owns prototype sp and tokens sq, sq + 4, ...
template <typename T>
__global__ void __launch_bounds__(TNT) tw_bwd_tokens_kernel(Args a, const float* __restrict__ dsk,
                                                            const float* __restrict__ lse_tok,
                                                            const float* __restrict__ Dtw, T* __restrict__ dK,
                                                            T* __restrict__ dV) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t t = blockIdx.x;
  if (t >= tph * H) return;
  float* Ks = smem;              // [32][d+1]
  float* Vs = Ks + TT * dp;      // [32][d+1]
  float* Qs = Vs + TT * dp;      // [64][d+1]
  float* Gs = Qs + TPB * dp;     // [64][d+1]
  float* A1 = Gs + TPB * dp;     // [64][33]  A
  float* A2 = A1 + TPB * 33;     // [64][33]  dS / scale
  float* ls = A2 + TPB * 33;     // [64]
  float* Ds = ls + TPB;          // [64]
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, TT);
  const int tid = threadIdx.x;
  stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
  stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
  const int64_t row = int64_t(r.b) * H + r.h;
  const float* G = dsk + row * int64_t(P) * d;
  const int ti = tid >> 3, cg = tid & 7;
  const int sp = tid >> 2, sq = tid & 3;
  float av[kMaxD / 8], ak[kMaxD / 8];
#pragma unroll
  for (int k = 0; k < kMaxD / 8; ++k) av[k] = ak[k] = 0.f;
  for (int pc = 0; pc < P; pc += TPB) {
    const int np = min(TPB, P - pc);
    __syncthreads();
    stage_rows(Qs, Q + (int64_t(q_row(a, r.b, r.h)) * P + pc) * d, d, np, TPB, d);
    stage_rows_f32(Gs, G + int64_t(pc) * d, np, TPB, d);
    if (tid < TPB) {
      ls[tid] = tid < np ? lse_tok[row * P + pc + tid] : 0.f;
      Ds[tid] = tid < np ? Dtw[row * P + pc + tid] : 0.f;
    }
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
        const bool ok = i < r.n && sp < np;
        const float A = ok ? expf(s[k] * a.scale - ls[sp]) : 0.f;
        A1[sp * 33 + i] = A;
        A2[sp * 33 + i] = ok ? A * (g[k] - Ds[sp]) : 0.f;
      }
    }
    __syncthreads();
    for (int j = 0; j < np; ++j) {
      const float x = A1[j * 33 + ti], y = A2[j * 33 + ti];
#pragma unroll
      for (int k = 0; k < kMaxD / 8; ++k) {
        const int c = cg + 8 * k;
        if (c < d) {
          av[k] = fmaf(x, Gs[j * dp + c], av[k]);
          ak[k] = fmaf(y, Qs[j * dp + c], ak[k]);
        }
      }
    }
  }
  if (ti < r.n) {
    T* ov = dV + ((r.tok0 + ti) * H + r.h) * int64_t(d);
    T* ok = dK + ((r.tok0 + ti) * H + r.h) * int64_t(d);
#pragma unroll
    for (int k = 0; k < kMaxD / 8; ++k) {
      const int c = cg + 8 * k;
      if (c < d) {
        st_from_f32(ov + c, av[k]);
        st_from_f32(ok + c, ak[k] * a.scale);
      }
    }
  }
}

// --------------------------------------------------- backward, prototype side
// grid = (W workers, ceil(P / 64)); per worker and head one fp32 partial of
// dQ[h] = scale sum_i dS[:, i] k_i, flushed where the head changes.
template <typename T>
__global__ void __launch_bounds__(TNT) tw_bwd_dq_kernel(Args a, const float* __restrict__ dsk,
                                                        const float* __restrict__ lse_tok,
                                                        const float* __restrict__ Dtw) {
  extern __shared__ float smem[];
  if (ws_failed(a.ws)) return;
  const int d = a.d, P = a.P, H = a.H, dp = d + 1;
  float* Qs = smem;              // [64][d+1]
  float* Gs = Qs + TPB * dp;     // [64][d+1]
  float* Ks = Gs + TPB * dp;     // [32][d+1]
  float* Vs = Ks + TT * dp;      // [32][d+1]
  float* As = Vs + TT * dp;      // [64][33]
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * H;
  const int W = gridDim.x, w = blockIdx.x;
  const int p0 = blockIdx.y * TPB, np = min(TPB, P - p0);
  const int64_t tb = range_begin(total, W, w), te = range_begin(total, W, w + 1);
  if (tb >= te) return;
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const T* Q = static_cast<const T*>(a.Q);
  const int tid = threadIdx.x, p = tid >> 2, cq = tid & 3;
  float acc[kMaxD / 4];
#pragma unroll
  for (int k = 0; k < kMaxD / 4; ++k) acc[k] = 0.f;
  int cur_q = -1;
  int64_t cur_row = -1;
  float lp = 0.f, Dp = 0.f;  // lse and D of (user, head, prototype p0 + p)
  for (int64_t t = tb; t < te; ++t) {
    const TileRef r = locate_tile(t, tph, a.prefix, a.cu, a.B, TT);
    const int64_t row = int64_t(r.b) * H + r.h;
    __syncthreads();
    const int qr = q_row(a, r.b, r.h);
    if (qr != cur_q) stage_rows(Qs, Q + (int64_t(qr) * P + p0) * d, d, np, TPB, d);
    cur_q = qr;
    if (row != cur_row) {
      stage_rows_f32(Gs, dsk + (row * P + p0) * d, np, TPB, d);
      lp = p < np ? lse_tok[row * P + p0 + p] : 0.f;
      Dp = p < np ? Dtw[row * P + p0 + p] : 0.f;
      cur_row = row;
    }
    stage_rows(Ks, K + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
    stage_rows(Vs, V + (r.tok0 * H + r.h) * int64_t(d), int64_t(H) * d, r.n, TT, d);
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
        As[p * 33 + i] = (i < r.n && p < np) ? expf(s[k] * a.scale - lp) * (g[k] - Dp) : 0.f;
      }
    }
    __syncthreads();
    for (int i = 0; i < TT; ++i) {
      const float ds = As[p * 33 + i];
#pragma unroll
      for (int k = 0; k < kMaxD / 4; ++k) {
        const int c = cq + 4 * k;
        if (c < d) acc[k] = fmaf(ds, Ks[i * dp + c], acc[k]);
      }
    }
    if (t + 1 == te || (t + 1) / tph != t / tph) {
      float* dst = a.dq_partial + ((int64_t(w) * H + r.h) * P + p0 + p) * d;
#pragma unroll
      for (int k = 0; k < kMaxD / 4; ++k) {
        const int c = cq + 4 * k;
        if (c < d && p < np) dst[c] = acc[k] * a.scale;
        acc[k] = 0.f;
      }
    }
  }
}

// ------------------------------------------------------------------ launchers
static size_t smem_tw_fwd(int d) { return sizeof(float) * (size_t(TPB + 2 * TT) * (d + 1) + TPB * 33); }
static size_t smem_tw_tok(int d) {
  return sizeof(float) * (size_t(2 * TT + 2 * TPB) * (d + 1) + 2 * TPB * 33 + 2 * TPB);
}
static size_t smem_tw_dq(int d) { return sizeof(float) * (size_t(2 * TT + 2 * TPB) * (d + 1) + TPB * 33); }

template <class Fn, class... Xs>
static cudaError_t run(Fn* fn, dim3 grid, size_t sm, cudaStream_t st, Xs... xs) {
  const cudaError_t e = cudaFuncSetAttribute(reinterpret_cast<const void*>(fn),
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(sm));
  if (e != cudaSuccess) return e;
  fn<<<grid, TNT, sm, st>>>(xs...);
  return cudaGetLastError();
}

int tw_tile_tokens() { return TT; }

cudaError_t launch_tw_fwd(const Args& a, int W, float* sketch, float* lse_tok, float2* stat_part, cudaStream_t st) {
  const dim3 grid(W, (a.P + TPB - 1) / TPB);
  if (a.dt == SA_BF16) return run(&tw_fwd_kernel<__nv_bfloat16>, grid, smem_tw_fwd(a.d), st, a, sketch, lse_tok, stat_part);
  return run(&tw_fwd_kernel<float>, grid, smem_tw_fwd(a.d), st, a, sketch, lse_tok, stat_part);
}

cudaError_t launch_tw_finalize(const Args& a, int W, const float2* stat_part, float* sketch, float* lse_tok,
                               cudaStream_t st) {
  tw_finalize_kernel<<<a.B * a.H, 256, 0, st>>>(a.ws, a.prefix, a.B, a.H, a.P, a.d, W, a.partial, stat_part,
                                                sketch, lse_tok);
  return cudaGetLastError();
}

cudaError_t launch_tw_dcoef(const Args& a, const float* O, const float* G, bool round_g, float* D,
                            cudaStream_t st) {
  const int64_t rows = int64_t(a.B) * a.H * a.P;
  tw_dcoef_kernel<<<unsigned((rows + 7) / 8), 256, 0, st>>>(a.ws, O, G, rows, a.d, round_g ? 1 : 0, D);
  return cudaGetLastError();
}

cudaError_t launch_tw_bwd_tokens(const Args& a, const float* dsk, const float* lse_tok, const float* D, void* dK,
                                 void* dV, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  const dim3 grid(unsigned(int64_t(a.H) * ((a.N + TT - 1) / TT + a.B)));
  if (a.dt == SA_BF16)
    return run(&tw_bwd_tokens_kernel<__nv_bfloat16>, grid, smem_tw_tok(a.d), st, a, dsk, lse_tok, D,
               static_cast<__nv_bfloat16*>(dK), static_cast<__nv_bfloat16*>(dV));
  return run(&tw_bwd_tokens_kernel<float>, grid, smem_tw_tok(a.d), st, a, dsk, lse_tok, D, static_cast<float*>(dK),
             static_cast<float*>(dV));
}

cudaError_t launch_tw_bwd_dq(const Args& a, int W, const float* dsk, const float* lse_tok, const float* D,
                             cudaStream_t st) {
  const dim3 grid(W, (a.P + TPB - 1) / TPB);
  if (a.dt == SA_BF16) return run(&tw_bwd_dq_kernel<__nv_bfloat16>, grid, smem_tw_dq(a.d), st, a, dsk, lse_tok, D);
  return run(&tw_bwd_dq_kernel<float>, grid, smem_tw_dq(a.d), st, a, dsk, lse_tok, D);
}

}  // namespace sa
