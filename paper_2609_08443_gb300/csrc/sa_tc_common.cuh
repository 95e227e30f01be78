// Pieces shared by the tensor-core kernels: the tile walker every warp role
// uses to follow its worker's range, TMA tensor maps, TMEM sizing and the
// epilogue that stores a sketch block from TMEM.
#pragma once
#include <cuda.h>

#include "sa_kernels.cuh"
#include "sa_ptx.cuh"

namespace sa {
namespace tcc {

constexpr int T = 128;           // tokens per tile = UMMA M
constexpr int kThreads = 384;    // 12 warps
constexpr int kSoftWarp0 = 4;    // warps 4..11: softmax / epilogue
constexpr int kSoftWarps = 8;

__host__ __device__ constexpr int tmem_cols_for(int c) {
  return c <= 32 ? 32 : c <= 64 ? 64 : c <= 128 ? 128 : c <= 256 ? 256 : 512;
}

// Follows worker tiles [tb, te) in (head, user, tile) order; all warp roles
// construct their own walker and see the same sequence.
struct TileWalker {
  const int64_t* prefix;
  const int32_t* cu;
  int B, Tt, H, uq;
  int64_t tph, t, tb, te;
  int h, b;
  int qk;  // row of Q this tile reads: h (shared queries) or b*H + h (per user)
  int64_t k, nk, tok0, seg0, seg1;
  int64_t cub, Lb;  // cu[b] and L_b of the current user, read once per segment
  int n;
  bool seg_first, seg_last;

  __device__ TileWalker(const Args& a, int64_t tb_, int64_t te_, int T_)
      : prefix(a.prefix), cu(a.cu), B(a.B), Tt(T_), H(a.H), uq(a.uq), t(tb_), tb(tb_), te(te_) {
    tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
    if (t < te) relocate();
  }
  __device__ void relocate() { set(locate_tile(t, tph, prefix, cu, B, Tt)); }
  __device__ void set(const TileRef& r) {
    h = r.h;
    b = r.b;
    qk = uq ? b * H + h : h;
    seg0 = r.seg0;
    seg1 = r.seg1;
    nk = seg1 - seg0;
    k = t - seg0;
    cub = r.tok0 - k * Tt;
    Lb = r.L;
    fields();
  }
  __device__ void fields() {
    tok0 = cub + k * Tt;
    const int64_t left = Lb - k * Tt;
    n = int(left < Tt ? left : Tt);
    seg_first = (k == 0) || (t == tb);
    seg_last = (k == nk - 1) || (t == te - 1);
  }
  // First token, size and head of the tile after this one (n = 0 past the range).
  __device__ void peek_next(int64_t& tok0_n, int& n_n, int& h_n) const {
    int qk_n;
    peek_next(tok0_n, n_n, h_n, qk_n);
  }
  // ... and the row of Q it reads (qk_n = qk past the range)
  __device__ void peek_next(int64_t& tok0_n, int& n_n, int& h_n, int& qk_n) const {
    if (t + 1 >= te) {
      tok0_n = 0;
      n_n = 0;
      h_n = h;
      qk_n = qk;
      return;
    }
    if (k + 1 < nk) {
      tok0_n = tok0 + Tt;
      const int64_t left = Lb - (k + 1) * Tt;
      n_n = int(left < Tt ? left : Tt);
      h_n = h;
      qk_n = qk;
    } else {
      const TileRef r = locate_next_segment(t + 1, h, b, tph, prefix, cu, B, Tt);
      tok0_n = r.tok0;
      n_n = r.n;
      h_n = r.h;
      qk_n = uq ? r.b * H + r.h : r.h;
    }
  }
  __device__ void next() {
    ++t;
    if (t >= te) return;
    if (k + 1 < nk) {
      ++k;
      fields();
    } else {
      set(locate_next_segment(t, h, b, tph, prefix, cu, B, Tt));
    }
  }
};

// The same walk with the binary search at every segment end instead of the
// forward scan.  The token-wise forward uses it: with the scan inlined in its
// roles' per-tile loops ptxas spilled more of its registers, and the 100K-token
// workload's token-wise forward ran 14 % slower; its segments are long there.
struct TileWalkerSearch : TileWalker {
  using TileWalker::TileWalker;
  __device__ void next() {
    ++t;
    if (t >= te) return;
    if (k + 1 < nk) {
      ++k;
      fields();
    } else {
      relocate();
    }
  }
};

// Where a worker's dQ block of prototypes [p0, p0 + PS) for the tiles ending
// at walker position w goes.  Shared queries: the worker's partial of head h
// ([W][H][P][d], summed over workers afterwards).  Per-user queries: dQ[b, h]
// itself when the worker holds the whole (user, head) segment, else the
// worker's partial slot of that segment ([W][2][P][d], summed like the sketch).
__device__ __forceinline__ float* dq_block_dst(const Args& a, int wk, int W, int64_t total, const TileWalker& w,
                                               int p0, int D) {
  if (!a.uq) return a.dq_partial + ((int64_t(wk) * a.H + w.h) * a.P + p0) * D;
  if (w.seg0 >= w.tb && w.seg1 <= w.te) return a.dq_user + ((int64_t(w.b) * a.H + w.h) * a.P + p0) * D;
  return a.partial + ((int64_t(wk) * 2 + partial_slot(total, W, wk, w.seg0)) * a.P + p0) * D;
}

__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = ptx::globaltimer();
  while (!ptx::mbar_try_wait(bar, parity))
    if (ptx::globaltimer() - t0 > limit_ns) return false;
  return true;
}

// Sketch block (PS prototypes x D) from TMEM to global memory.
//  TRANS (D = 128): TMEM holds O^T: lane = feature d, column = prototype.
//  else (D = 64):   TMEM holds O in PS/128 blocks: lane = prototype, column = d.
template <int D, int PS, bool TRANS, int O_COL>
__device__ __forceinline__ void store_sketch(uint32_t tmem, uint32_t lane_off, int sw, int q, int lane, float* dst) {
  float v[32];
  if (TRANS) {
    const int d = 32 * q + lane;
#pragma unroll 1
    for (int c = 0; c < PS / 2 / 32; ++c) {
      const int pbase = sw * (PS / 2) + 32 * c;
      ptx::tmem_ld32(tmem + lane_off + O_COL + pbase, v);
      ptx::tmem_ld_wait();
      float* col = dst + int64_t(pbase) * D + d;  // prototype pbase, feature d; the next prototype is D floats on
#pragma unroll
      for (int k = 0; k < 32; ++k) col[k * D] = v[k];
    }
  } else {
    constexpr int NB = PS / 128;
    const int blk = NB == 2 ? sw : 0;
    const int p = 128 * blk + 32 * q + lane;
    const int c0 = NB == 2 ? 0 : 32 * sw;
    const int c1 = NB == 2 ? D : c0 + 32;
#pragma unroll 1
    for (int c = c0; c < c1; c += 32) {
      ptx::tmem_ld32(tmem + lane_off + O_COL + blk * D + c, v);
      ptx::tmem_ld_wait();
      float4* o = reinterpret_cast<float4*>(dst + int64_t(p) * D + c);
#pragma unroll
      for (int k = 0; k < 8; ++k) o[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
    }
  }
}

// Prototype-major accumulator ([PS/128 blocks] lanes = prototype, columns = d)
// times `mul` to global rows [PS][D] (used for dQ partials).
template <int D, int PS, int O_COL>
__device__ __forceinline__ void store_sketch_scaled(uint32_t tmem, uint32_t lane_off, int sw, int q, int lane,
                                                    float* dst, float mul) {
  float v[32];
  constexpr int NB = PS / 128;
  const int blk = NB == 2 ? sw : 0;
  const int p = 128 * blk + 32 * q + lane;
  const int c0 = NB == 2 ? 0 : (D / 2) * sw;
  const int c1 = NB == 2 ? D : c0 + D / 2;
#pragma unroll 1
  for (int c = c0; c < c1; c += 32) {
    ptx::tmem_ld32(tmem + lane_off + O_COL + blk * D + c, v);
    ptx::tmem_ld_wait();
    float4* o = reinterpret_cast<float4*>(dst + int64_t(p) * D + c);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      o[k] = make_float4(v[4 * k] * mul, v[4 * k + 1] * mul, v[4 * k + 2] * mul, v[4 * k + 3] * mul);
  }
}

// ------------------------------------------------------------- host helpers
bool make_kv_map(CUtensorMap* m, const void* base, int64_t N, int H, int D);
bool make_q_map(CUtensorMap* m, const void* Q, int H, int P, int D, int box_rows);
bool device_is_sm103();
int device_sm_count();

}  // namespace tcc

bool tc_path_enabled();

}  // namespace sa
