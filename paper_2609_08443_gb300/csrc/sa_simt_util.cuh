// Staging helpers of the CUDA-core kernels (sa_simt.cu, sa_tokenwise.cu):
// vector loads widened to fp32, rows copied into padded shared-memory tiles,
// and the user that holds a token.
#pragma once
#include "sa_kernels.cuh"

namespace sa {

// ------------------------------------------------------------ load helpers
template <typename T> struct Vec;
template <> struct Vec<float> {
  static constexpr int n = 4;
  static __device__ __forceinline__ void load(const float* p, float* o) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
  }
};
template <> struct Vec<__nv_bfloat16> {
  static constexpr int n = 8;
  static __device__ __forceinline__ void load(const __nv_bfloat16* p, float* o) {
    const uint4 v = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      o[2 * k] = __uint_as_float(w[k] << 16);
      o[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
    }
  }
};

// rows [0, nrows) of a [*, ld] source into smem [rows][d+1] as fp32; rows
// beyond nrows (up to rmax) are zero.
template <typename T>
__device__ __forceinline__ void stage_rows(float* dst, const T* src, int64_t src_ld, int nrows,
                                           int rmax, int d) {
  constexpr int VN = Vec<T>::n;
  const int per_row = d / VN;
  for (int e = threadIdx.x; e < rmax * per_row; e += blockDim.x) {
    const int r = e / per_row, c = (e - r * per_row) * VN;
    float v[VN];
    if (r < nrows) {
      Vec<T>::load(src + int64_t(r) * src_ld + c, v);
    } else {
#pragma unroll
      for (int k = 0; k < VN; ++k) v[k] = 0.f;
    }
#pragma unroll
    for (int k = 0; k < VN; ++k) dst[r * (d + 1) + c + k] = v[k];
  }
}

__device__ __forceinline__ void stage_rows_f32(float* dst, const float* src, int nrows, int rmax, int d) {
  for (int e = threadIdx.x; e < rmax * d; e += blockDim.x) {
    const int r = e / d, c = e - r * d;
    dst[r * (d + 1) + c] = r < nrows ? src[int64_t(r) * d + c] : 0.f;
  }
}

// User of token t: the largest b with cu[b] <= t (empty users before it share
// its offset, so the largest such b is the user that holds t).
__device__ __forceinline__ int user_of_token(const int32_t* cu, int B, int64_t t) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (int64_t(cu[mid]) <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

}  // namespace sa
