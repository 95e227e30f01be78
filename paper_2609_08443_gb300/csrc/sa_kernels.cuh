// Internal interface between the host API (sa_api.cu) and the kernel files.
#pragma once
#include "sa_common.cuh"

namespace sa {

// Everything a kernel needs about one call (passed by value as a kernel arg).
struct Args {
  const void* K;
  const void* V;
  const void* Q;
  const int32_t* cu;
  int B;
  int64_t N;
  int H, P, d;
  float scale;
  sa_dtype dt;
  void* ws;            // workspace base (header)
  int64_t* prefix;     // per-head tile prefix [B + 1]
  float* partial;      // [W][2][P][d]
  float* dq_partial;   // [W][H][P][d]
  float* lse_scratch;  // [N][H] workspace copy of lse when the caller passes none
  float2* lse_part;    // [N][H][slices] per-slice (max, sum) of the lse pass when P >= 1024
  int uq;              // 1: per-user queries Q[B][H][P][d] and dQ[B][H][P][d] (stacked refinement)
  float* dq_user;      // per-user queries: the caller's dQ[B][H][P][d] (whole segments go there)
};

// Row of Q ([H or B*H][P][d]) that user b, head h reads.
SA_HD int q_row(const Args& a, int b, int h) { return a.uq ? b * a.H + h : h; }

// Limit of the bounded pipeline waits for calls enqueued from now on
// (sa_set_wait_limit_ns; the planner copies it into each call's workspace).
uint64_t wait_limit_ns();

// planner / finalize (sa_simt.cu)
cudaError_t launch_plan(const Args& a, int T, cudaStream_t st);
cudaError_t launch_finalize_sketch(const Args& a, int W, float* sketch, cudaStream_t st);
cudaError_t launch_finalize_dq(const Args& a, int W, float* dQ, cudaStream_t st);

// key projection folded into the prototypes (sa_xproj.cu)
cudaError_t launch_fold_wk(const void* Q, const void* Wk, int H, int P, int d, sa_dtype dt, void* Qf,
                           cudaStream_t st);
cudaError_t launch_add_into(void* dX, const void* dKf, int64_t n, sa_dtype dt, cudaStream_t st);
// dst = -src, n elements of type dt (src == dst allowed)
cudaError_t launch_negate(const void* src, void* dst, int64_t n, sa_dtype dt, cudaStream_t st);
cudaError_t launch_wk_grads(const float* dQf, const void* Q, const void* Wk, int H, int P, int d, sa_dtype dt,
                            float* dQ, float* dWk, cudaStream_t st);

// CUDA-core path (sa_simt.cu)
int simt_tile_tokens();
int simt_workers(int num_sms, int P);
cudaError_t launch_simt_lse(const Args& a, float* lse, cudaStream_t st);
cudaError_t launch_simt_fwd(const Args& a, int W, const float* lse, float* sketch, cudaStream_t st);
cudaError_t launch_simt_bwd_tokens(const Args& a, const float* dsk, const float* lse, void* dK, void* dV,
                                   float* Dco, cudaStream_t st);
cudaError_t launch_simt_bwd_dq(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                               cudaStream_t st);

// token-wise normalisation (sa_tokenwise.cu)
int tw_tile_tokens();
cudaError_t launch_tw_fwd(const Args& a, int W, float* sketch, float* lse_tok, float2* stat_part, cudaStream_t st);
cudaError_t launch_tw_finalize(const Args& a, int W, const float2* stat_part, float* sketch, float* lse_tok,
                               cudaStream_t st);
cudaError_t launch_tw_dcoef(const Args& a, const float* O, const float* G, bool round_g, float* D,
                            cudaStream_t st);
cudaError_t launch_tw_bwd_tokens(const Args& a, const float* dsk, const float* lse_tok, const float* D, void* dK,
                                 void* dV, cudaStream_t st);
cudaError_t launch_tw_bwd_dq(const Args& a, int W, const float* dsk, const float* lse_tok, const float* D,
                             cudaStream_t st);

}  // namespace sa
