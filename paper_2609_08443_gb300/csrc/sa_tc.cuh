// Interface of the tcgen05 / TMEM / TMA kernels (sm_103a).
#pragma once
#include "sa_kernels.cuh"

namespace sa {

bool tc_fwd_supported(int P, int d, sa_dtype dt);
bool tc_fwd_needs_lse_pass_d(int P, int d);  // lse pass, then 256-prototype slices
int tc_lse_slice(int P, int d);              // prototypes per slice of the lse pass
bool tc_path_enabled();
bool tc_fwd_sliced_selected();  // sa_select_path(2)
bool tc_narrow_selected();      // sa_select_path(3): the 8-softmax-warp pair forward for P = 512
// P = 512: the cluster-pair forward with 16 softmax warps (sa_tc_fwd_wide.cu)
cudaError_t launch_tc_fwd_wide(const Args& a, int W, float* sketch, float* lse, cudaStream_t st);
bool tc_bwd_supported(int P, int d, sa_dtype dt);
const char* tc_fwd_name(int P, int d);
const char* tc_bwd_name(int P, int d);
int tc_tile_tokens();
int tc_fwd_workers(int num_sms, int P, int d);
int tc_bwd_workers(int num_sms, int P, int d);
cudaError_t launch_tc_fwd(const Args& a, int W, float* sketch, float* lse, cudaStream_t st);
cudaError_t launch_tc_lse(const Args& a, float* lse, cudaStream_t st);
cudaError_t launch_tc_bwd(const Args& a, int W, const float* dsk, const float* lse, void* dK, void* dV,
                          cudaStream_t st);
// d = 128 with P in {256, 512}: token side (dV, dK, D_i) then prototype slices (dQ)
bool tc_bwd_split(int P, int d);
cudaError_t launch_tc_bwd_tok(const Args& a, int W, const float* dsk, __nv_bfloat16* gbf, const float* lse,
                              float* Dco, void* dK, void* dV, cudaStream_t st);
cudaError_t launch_tc_bwd_dq(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                             cudaStream_t st);
int tc_bwd_dq_workers(int num_sms, int P);
// token-wise normalisation (Sec. 5.1): tensor-core forward
bool tc_tw_fwd_supported(int P, int d, sa_dtype dt, float scale);
int tc_tw_fwd_workers(int num_sms, int P);
const char* tc_tw_fwd_name(int P, int d);
cudaError_t launch_tc_tw_fwd(const Args& a, int W, float* sketch, float* lse_tok, float2* stat_part,
                             cudaStream_t st);
bool tc_tw_bwd_supported(int P, int d, sa_dtype dt);
cudaError_t launch_tc_tw_bwd_tok(const Args& a, int W, const __nv_bfloat16* gbf, const float* lse_tok,
                                 const float* Dtw, void* dK, void* dV, cudaStream_t st);
cudaError_t launch_tc_tw_bwd_dq(const Args& a, int W, const float* dsk, const float* lse_tok, const float* Dtw,
                                cudaStream_t st);
cudaError_t launch_tc_g_bf16(const Args& a, const float* dsk, __nv_bfloat16* gbf, cudaStream_t st);

}  // namespace sa
