// The key projection of the SA step (paper Sec. 3.1: S = (P W_Q)(X W_K)^T /
// sqrt(d), sketch A X; App. G.3: K = X W_K) folded into the prototypes.
//
// With keys k_i = x_i W_K and values x_i, the scores are
//     S[j,i] = q_j . (x_i W_K) = (q_j W_K^T) . x_i,
// so the sketching step runs unchanged on K = V = X with prototypes
// Q' = Q W_K^T: no K is materialised, X is the only per-token input, and the
// projection costs P d^2 per head instead of L d^2 per token range.  The
// backward maps the step's gradients (dK', dV, dQ' with respect to K = X, V = X
// and Q') back to the caller's parameters:
//     dX  = dV + dK'                 (X enters as the keys and as the values)
//     dQ  = dQ' W_K,   dW_K = dQ'^T Q   (chain rule through Q' = Q W_K^T)
// The three small kernels below (CUDA cores, fp32 accumulation) do exactly
// that; the heavy work stays in the sketching kernels.
#include "sa_kernels.cuh"

namespace sa {

// Q'[h, j, c] = sum_e Q[h, j, e] Wk[h, c, e]; one block per (head, 8 prototypes).
template <typename T>
__global__ void __launch_bounds__(256) fold_wk_kernel(const T* __restrict__ Q, const T* __restrict__ Wk, int P,
                                                      int d, T* __restrict__ Qf) {
  __shared__ float qs[8][kMaxD];
  const int h = blockIdx.y, j0 = blockIdx.x * 8;
  const T* Qh = Q + int64_t(h) * P * d;
  const T* Wh = Wk + int64_t(h) * d * d;
  for (int e = threadIdx.x; e < 8 * d; e += blockDim.x) {
    const int jj = e / d, c = e % d;
    qs[jj][c] = (j0 + jj < P) ? ld_f32(Qh + int64_t(j0 + jj) * d + c) : 0.f;
  }
  __syncthreads();
  for (int o = threadIdx.x; o < 8 * d; o += blockDim.x) {
    const int jj = o / d, c = o % d;
    if (j0 + jj >= P) continue;
    float s = 0.f;
    for (int e = 0; e < d; ++e) s = fmaf(qs[jj][e], ld_f32(Wh + int64_t(c) * d + e), s);
    st_from_f32(Qf + (int64_t(h) * P + j0 + jj) * d + c, s);
  }
}

// dX += dK' elementwise (both of type T).
template <typename T>
__global__ void add_into_kernel(T* __restrict__ dX, const T* __restrict__ dKf, int64_t n) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x)
    st_from_f32(dX + i, ld_f32(dX + i) + ld_f32(dKf + i));
}

// dst = -src elementwise (exact in bf16 and fp32).
template <typename T>
__global__ void negate_kernel(const T* __restrict__ src, T* __restrict__ dst, int64_t n) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x)
    dst[i] = -src[i];
}

// dQ[h] = dQ'[h] Wk[h]  (P x d),  dWk[h] = dQ'[h]^T Q[h]  (d x d); fp32 outputs.
// grid (ceil(max(P, d) / 8), H); each block computes 8 rows of both.
template <typename T>
__global__ void __launch_bounds__(256) wk_grads_kernel(const float* __restrict__ dQf, const T* __restrict__ Q,
                                                       const T* __restrict__ Wk, int P, int d,
                                                       float* __restrict__ dQ, float* __restrict__ dWk) {
  const int h = blockIdx.y, r0 = blockIdx.x * 8;
  const float* G = dQf + int64_t(h) * P * d;
  const T* Qh = Q + int64_t(h) * P * d;
  const T* Wh = Wk + int64_t(h) * d * d;
  for (int o = threadIdx.x; o < 8 * d; o += blockDim.x) {
    const int rr = r0 + o / d, e = o % d;
    if (rr < P) {  // dQ[rr, e] = sum_c dQ'[rr, c] Wk[c, e]
      float s = 0.f;
      for (int c = 0; c < d; ++c) s = fmaf(G[int64_t(rr) * d + c], ld_f32(Wh + int64_t(c) * d + e), s);
      dQ[(int64_t(h) * P + rr) * d + e] = s;
    }
    if (rr < d) {  // dWk[rr, e] = sum_j dQ'[j, rr] Q[j, e]
      float s = 0.f;
      for (int j = 0; j < P; ++j) s = fmaf(G[int64_t(j) * d + rr], ld_f32(Qh + int64_t(j) * d + e), s);
      dWk[(int64_t(h) * d + rr) * d + e] = s;
    }
  }
}

cudaError_t launch_fold_wk(const void* Q, const void* Wk, int H, int P, int d, sa_dtype dt, void* Qf,
                           cudaStream_t st) {
  dim3 grid((P + 7) / 8, H);
  if (dt == SA_BF16)
    fold_wk_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(Q),
                                                        static_cast<const __nv_bfloat16*>(Wk), P, d,
                                                        static_cast<__nv_bfloat16*>(Qf));
  else
    fold_wk_kernel<float><<<grid, 256, 0, st>>>(static_cast<const float*>(Q), static_cast<const float*>(Wk), P, d,
                                                static_cast<float*>(Qf));
  return cudaGetLastError();
}

cudaError_t launch_add_into(void* dX, const void* dKf, int64_t n, sa_dtype dt, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  if (dt == SA_BF16)
    add_into_kernel<__nv_bfloat16><<<2048, 256, 0, st>>>(static_cast<__nv_bfloat16*>(dX),
                                                         static_cast<const __nv_bfloat16*>(dKf), n);
  else
    add_into_kernel<float><<<2048, 256, 0, st>>>(static_cast<float*>(dX), static_cast<const float*>(dKf), n);
  return cudaGetLastError();
}

cudaError_t launch_negate(const void* src, void* dst, int64_t n, sa_dtype dt, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const int blocks = int((n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024);
  if (dt == SA_BF16)
    negate_kernel<__nv_bfloat16><<<blocks, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(src),
                                                         static_cast<__nv_bfloat16*>(dst), n);
  else
    negate_kernel<float><<<blocks, 256, 0, st>>>(static_cast<const float*>(src), static_cast<float*>(dst), n);
  return cudaGetLastError();
}

cudaError_t launch_wk_grads(const float* dQf, const void* Q, const void* Wk, int H, int P, int d, sa_dtype dt,
                            float* dQ, float* dWk, cudaStream_t st) {
  const int rows = P > d ? P : d;
  dim3 grid((rows + 7) / 8, H);
  if (dt == SA_BF16)
    wk_grads_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(dQf, static_cast<const __nv_bfloat16*>(Q),
                                                         static_cast<const __nv_bfloat16*>(Wk), P, d, dQ, dWk);
  else
    wk_grads_kernel<float><<<grid, 256, 0, st>>>(dQf, static_cast<const float*>(Q), static_cast<const float*>(Wk),
                                                 P, d, dQ, dWk);
  return cudaGetLastError();
}

}  // namespace sa
