// tcgen05 / TMEM / TMA forward of the token-wise ("vanilla") normalisation
// (paper Sec. 5.1, App. C): per user and head, A[j, :] = softmax over the
// user's tokens of S[j, :], sketch = A V.
//
// The roles of tokens and prototypes swap with respect to the prototype-wise
// kernels: the statistic is per prototype, so the scores are computed as
//     S = Q K^T     (UMMA M = 128 prototypes, N = 128 tokens, K = d)
// and every prototype's row lies in one TMEM lane, i.e. in one thread: the
// running maximum and sum over tokens stay in registers (online softmax, as in
// FlashAttention with the prototypes as queries).  The weights go to shared
// memory as bf16 in K-major order ([2 blocks of 64 tokens][PS prototypes][64],
// 128-byte swizzle) and
//     O += A V      (M = 128 prototypes, N = d, K = 128 tokens)
// accumulates in TMEM.  The shift of the exponentials is changed lazily: only
// when a tile's maximum exceeds the shift in use by more than 8 (log2 units,
// weights up to 2^8 are exact enough in bf16 and fp32 sums), and only then is
// the thread's row of O rescaled in TMEM (after the previous aggregation has
// completed, before the next is issued).  A user's sketch is normalised by the
// sum when its segment ends; a worker's piece of a segment cut across workers
// is left unnormalised with its (shift, sum) for tw_finalize_kernel.
//
// One CTA holds PS = 128 NM prototypes (grid.y = P / PS slices); warpgroup g of
// the softmax warps owns M-tile g.  Warp roles: 0 = TMA producer, 1 = UMMA
// issuer, 2 = TMEM allocator, 4..11 = softmax + epilogue.  Every wait is
// bounded (sa_ptx.cuh).
#include <cuda.h>

#include "sa_ptx.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace sa {
namespace tctw {

using namespace ptx;
using namespace tcc;

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLazy = 8.f;  // re-shift when a tile's max exceeds the shift by more (log2 units)

template <int D, int NM>
struct Cfg {
  static constexpr int PS = 128 * NM;
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = PS * D * 2;
  static constexpr int W_BYTES = PS * T * 2;
  static constexpr int NSLOT = (D == 128) ? 3 : 6;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_RING = OFF_Q + Q_BYTES;
  static constexpr int OFF_W = OFF_RING + NSLOT * KV_TILE;
  static constexpr int OFF_BAR = OFF_W + W_BYTES;
  static constexpr int NBAR = 2 * NSLOT + 9;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = OFF_MISC + 16;
  static_assert(SMEM <= 232448, "shared memory budget");
  static constexpr int S_COL = 0;
  static constexpr int O_COL = 128 * NM;
  static constexpr int TMEM_COLS = tmem_cols_for(O_COL + NM * D);
  static constexpr int SOFT_WARPS = 4 * NM;
};

template <int D, int NM>
__global__ void __launch_bounds__(kThreads, 1)
    tc_tw_fwd_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     const __grid_constant__ CUtensorMap tmQ, Args a, float* __restrict__ sketch,
                     float* __restrict__ lse_tok, float2* __restrict__ stat_part) {
  using C = Cfg<D, NM>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ws_failed(a.ws)) return;
  if (smem_u32(smem) & 1023u) {  // 128-byte swizzle atoms need 1024-byte alignment
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xA21u);
    return;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sRing = sbase + C::OFF_RING, sW = sbase + C::OFF_W;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto ring_full = [&](int s) { return bar0 + 8u * s; };
  auto ring_empty = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  const uint32_t q_full = bar0 + 8u * (2 * C::NSLOT + 0), q_empty = q_full + 8, s_full = q_full + 16,
                 s_empty = q_full + 24, w_full = q_full + 32, w_empty = q_full + 40, o_full = q_full + 48,
                 o_empty = q_full + 56, drain = q_full + 64;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);

  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = int(gridDim.x), wk = int(blockIdx.x);
  const int p0 = int(blockIdx.y) * C::PS;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  const int ntiles = int(te - tb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(ring_full(s), 1);
      mbar_init(ring_empty(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(s_full, 1);
    mbar_init(s_empty, C::SOFT_WARPS);
    mbar_init(w_full, C::SOFT_WARPS);
    mbar_init(w_empty, 1);
    mbar_init(o_full, 1);
    mbar_init(o_empty, C::SOFT_WARPS);
    mbar_init(drain, 1);
    wait_ctl_init(abort_flag, a.ws);
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Registers: the control warpgroup (warps 0-3) hands registers to the two
  // softmax warpgroups, which hold a row of 128 scores (128 x 88 + 256 x 208 =
  // 384 x 168, the launch allocation).
  if (ntiles > 0 && warp < kSoftWarp0) {
    setmaxnreg_dec<88>();
    if (warp == 0 && lane == 0) {
      // ------------------------------------------------------ TMA producer
      // K of tile li and V of tile li - 1 alternate in one ring of slots
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      TileWalkerSearch it(a, tb, te, T), pv(a, tb, te, T), pf(a, tb, te, T);
      pf.next();
      pf.next();
      int hc = 0, prev_q = -1;
      uint32_t e = 0;
      bool ok = true;
      for (int li = 0; li <= ntiles && ok; ++li) {
        if (li + 2 < ntiles) {
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) {
            tma_prefetch_l2_3d(&tmK, 64 * dh, pf.h, int(pf.tok0));
            tma_prefetch_l2_3d(&tmV, 64 * dh, pf.h, int(pf.tok0));
          }
          pf.next();
        }
        if (li < ntiles) {
          if (it.qk != prev_q) {
            if (hc > 0) ok = mbar_wait(q_empty, (hc - 1) & 1, abort_flag, a.ws, 0x901);
            if (!ok) break;
            mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
            for (int dh = 0; dh < D / 64; ++dh)
              tma_load_3d(sQ + dh * C::PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
            prev_q = it.qk;
            ++hc;
          }
          const int s = int(e % C::NSLOT);
          if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x902);
          if (!ok) break;
          mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh)
            tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, &tmK, ring_full(s), 64 * dh, it.h, int(it.tok0));
          ++e;
          it.next();
        }
        if (li >= 1) {
          const int s = int(e % C::NSLOT);
          if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x903);
          if (!ok) break;
          mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh)
            tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, &tmV, ring_full(s), 64 * dh, pv.h, int(pv.tok0));
          ++e;
          pv.next();
        }
      }
      if (!ok) {  // drain loads still in flight before the CTA may exit
        for (uint32_t k = (e > uint32_t(C::NSLOT) ? e - C::NSLOT : 0); k < e; ++k)
          mbar_wait_bounded(ring_full(int(k % C::NSLOT)), (k / C::NSLOT) & 1, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      // ------------------------------------------------------ UMMA issuer
      constexpr uint32_t idS = idesc_bf16(128, T, 0, 0);  // Q (K-major) x K^T (K-major)
      constexpr uint32_t idO = idesc_bf16(128, D, 0, 1);  // A (K-major) x V (MN-major)
      TileWalkerSearch cur(a, tb, te, T), nxt(a, tb, te, T);
      nxt.next();
      uint32_t e = 0;
      int hc = 0, sc = 0;
      bool ok = mbar_wait(q_full, 0, abort_flag, a.ws, 0xA01);
      // S[m-tile] = Q[m-tile] K^T over the d features, 16 per step
      auto issue_S = [&](uint32_t slot) {
        const uint32_t kaddr = sRing + slot * C::KV_TILE;
#pragma unroll
        for (int mt = 0; mt < NM; ++mt) {
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint64_t ad = sdesc(sQ + (k >> 2) * (C::PS * 128) + mt * (128 * 128) + (k & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc(kaddr + (k >> 2) * (T * 128) + (k & 3) * 32, 16, 1024);
            umma_ss(tmem + C::S_COL + mt * T, ad, bd, idS, k > 0 ? 1u : 0u);
          }
        }
      };
      if (ok) {
        ok = mbar_wait(ring_full(0), 0, abort_flag, a.ws, 0xA02);
        if (ok) {
          tc_fence_after();
          issue_S(0);
          umma_commit(s_full);
          umma_commit(ring_empty(0));
          if (ntiles == 1 || nxt.qk != cur.qk) umma_commit(q_empty);
          e = 1;
        }
      }
      for (int li = 0; li < ntiles && ok; ++li) {
        if (li + 1 < ntiles) {
          if (nxt.qk != cur.qk) {
            ++hc;
            ok = mbar_wait(q_full, hc & 1, abort_flag, a.ws, 0xA03);
            if (!ok) break;
          }
          ok = mbar_wait(s_empty, li & 1, abort_flag, a.ws, 0xA04);
          if (!ok) break;
          const int s = int(e % C::NSLOT);
          ok = mbar_wait(ring_full(s), (e / C::NSLOT) & 1, abort_flag, a.ws, 0xA05);
          if (!ok) break;
          tc_fence_after();
          issue_S(uint32_t(s));
          umma_commit(s_full);
          umma_commit(ring_empty(s));
          ++e;
          const int q_now = nxt.qk;
          nxt.next();
          if (li + 2 >= ntiles || nxt.qk != q_now) umma_commit(q_empty);
        }
        // O[m-tile] += A[m-tile] V over the tile's 128 tokens, 16 per step
        ok = mbar_wait(w_full, li & 1, abort_flag, a.ws, 0xA06);
        if (!ok) break;
        const int s = int(e % C::NSLOT);
        ok = mbar_wait(ring_full(s), (e / C::NSLOT) & 1, abort_flag, a.ws, 0xA07);
        if (!ok) break;
        if (cur.seg_first && sc > 0) {
          ok = mbar_wait(o_empty, (sc - 1) & 1, abort_flag, a.ws, 0xA08);
          if (!ok) break;
        }
        tc_fence_after();
        const uint32_t vaddr = sRing + s * C::KV_TILE;
#pragma unroll
        for (int k = 0; k < T / 16; ++k) {
          const uint32_t acc = (cur.seg_first && k == 0) ? 0u : 1u;
#pragma unroll
          for (int mt = 0; mt < NM; ++mt) {
            const uint64_t ad = sdesc(sW + (k >> 2) * (C::PS * 128) + mt * (128 * 128) + (k & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc(vaddr + k * 2048, T * 128, 1024);
            umma_ss(tmem + C::O_COL + mt * D, ad, bd, idO, acc);
          }
        }
        umma_commit(w_empty);
        umma_commit(ring_empty(s));
        ++e;
        if (cur.seg_last) {
          umma_commit(o_full);
          ++sc;
        }
        cur.next();
      }
      umma_commit(drain);  // no UMMA may still run when TMEM is released
      mbar_wait_bounded(drain, 0, 200000000ull);
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<208>();
    if (warp < kSoftWarp0 + C::SOFT_WARPS) {
      // ------------------------------------------- softmax + epilogue warps
      const int g = (warp - kSoftWarp0) >> 2;  // M-tile
      const int q = warp & 3;                  // TMEM lane quadrant
      const int pr = 128 * g + 32 * q + lane;  // prototype within the CTA's slice
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * kLog2e;
      TileWalkerSearch cur(a, tb, te, T);
      int seg_idx = 0;
      bool ok = true;
      float msh = 0.f, l = 0.f;  // shift in use (log2 units) and sum of 2^(S c2 - msh) so far
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      for (int li = 0; li < ntiles && ok; ++li) {
        ok = wwait(s_full, li & 1, 0xB01);
        if (!ok) break;
        tc_fence_after();
        float v[T];
#pragma unroll
        for (int c = 0; c < T / 32; ++c) tmem_ld32(tmem + lane_off + C::S_COL + g * T + 32 * c, v + 32 * c);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(s_empty);
        if (cur.n < T) {  // columns past the tile's tokens weigh exactly zero
#pragma unroll
          for (int c = 0; c < T; ++c)
            if (c >= cur.n) v[c] = -INFINITY;
        }
        const float mt = row_max<T>(v) * c2;
        float alpha = 1.f;
        if (cur.seg_first) {
          msh = mt;
          l = 0.f;
        } else if (mt > msh + kLazy) {
          alpha = ex2(msh - mt);
          msh = mt;
        }
        l = l * alpha + exp2_shift_sum<T>(v, c2, msh);
        if (li > 0) {  // the previous aggregation is done: W is free and O is at rest
          ok = wwait(w_empty, (li - 1) & 1, 0xB02);
          if (!ok) break;
        }
        // weights -> shared memory: [2 token blocks][PS prototypes][64 tokens], 128-byte swizzle
        uint8_t* wrow = smem + C::OFF_W + pr * 128;
#pragma unroll
        for (int k = 0; k < T / 8; ++k) {
          const int blk = k >> 3, chunk = k & 7;
          uint4 pk;
          pk.x = pack_bf16(v[8 * k + 0], v[8 * k + 1]);
          pk.y = pack_bf16(v[8 * k + 2], v[8 * k + 3]);
          pk.z = pack_bf16(v[8 * k + 4], v[8 * k + 5]);
          pk.w = pack_bf16(v[8 * k + 6], v[8 * k + 7]);
          *reinterpret_cast<uint4*>(wrow + blk * (C::PS * 128) + ((chunk ^ (pr & 7)) << 4)) = pk;
        }
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
          tc_fence_after();
          float o[32];
#pragma unroll 1
          for (int c = 0; c < D; c += 32) {
            const uint32_t ta = tmem + lane_off + C::O_COL + g * D + c;
            tmem_ld32(ta, o);
            tmem_ld_wait();
#pragma unroll
            for (int k = 0; k < 32; ++k) o[k] *= alpha;
            tmem_st16(ta, reinterpret_cast<const uint32_t*>(o));
            tmem_st16(ta + 16, reinterpret_cast<const uint32_t*>(o) + 16);
          }
          tmem_st_wait();
          tc_fence_before();
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(w_full);
        if (cur.seg_last) {
          ok = wwait(o_full, seg_idx & 1, 0xB03);
          if (!ok) break;
          tc_fence_after();
          const int64_t row = int64_t(cur.b) * a.H + cur.h;
          const bool whole = cur.seg0 >= tb && cur.seg1 <= te;
          const int64_t slot = int64_t(wk) * 2 + partial_slot(total, W, wk, cur.seg0);
          float* dst = whole ? sketch + (row * a.P + p0 + pr) * D : a.partial + (slot * a.P + p0 + pr) * D;
          const float mul = whole ? 1.f / l : 1.f;
          float o[32];
#pragma unroll 1
          for (int c = 0; c < D; c += 32) {
            tmem_ld32(tmem + lane_off + C::O_COL + g * D + c, o);
            tmem_ld_wait();
            float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
            for (int k = 0; k < 8; ++k)
              d4[k] = make_float4(o[4 * k] * mul, o[4 * k + 1] * mul, o[4 * k + 2] * mul, o[4 * k + 3] * mul);
          }
          if (whole)
            lse_tok[row * a.P + p0 + pr] = msh * kLn2 + logf(l);
          else
            stat_part[slot * a.P + p0 + pr] = make_float2(msh * kLn2, l);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(o_empty);
          ++seg_idx;
        }
        cur.next();
      }
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, int NM>
static cudaError_t launch_t(const Args& a, int W, float* sketch, float* lse_tok, float2* stat_part,
                            cudaStream_t st) {
  using C = Cfg<D, NM>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.H, a.P, D, C::PS))
    return cudaErrorInvalidValue;
  auto fn = &tc_tw_fwd_kernel<D, NM>;
  const cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const dim3 grid(W, a.P / C::PS);
  fn<<<grid, kThreads, C::SMEM, st>>>(tk, tv, tq, a, sketch, lse_tok, stat_part);
  return cudaGetLastError();
}

}  // namespace tctw

// Shapes served by the tensor-core token-wise forward: bf16, d in {64, 128},
// P a multiple of 128 up to 2048, a positive scale (the running maximum is
// taken on the raw scores).
bool tc_tw_fwd_supported(int P, int d, sa_dtype dt, float scale) {
  if (dt != SA_BF16 || (d != 64 && d != 128) || P % 128 != 0 || P > 2048 || !(scale > 0.f)) return false;
  return tcc::device_is_sm103() && tc_path_enabled();
}

static int tw_slice(int P) { return P % 256 == 0 ? 256 : 128; }

int tc_tw_fwd_workers(int num_sms, int P) {
  const int w = num_sms / (P / tw_slice(P));
  return w < 1 ? 1 : w;
}

const char* tc_tw_fwd_name(int P, int d) {
  if (tw_slice(P) == 256) return d == 128 ? "tc_tw_fwd_kernel<128,2>" : "tc_tw_fwd_kernel<64,2>";
  return d == 128 ? "tc_tw_fwd_kernel<128,1>" : "tc_tw_fwd_kernel<64,1>";
}

cudaError_t launch_tc_tw_fwd(const Args& a, int W, float* sketch, float* lse_tok, float2* stat_part,
                             cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  if (tw_slice(a.P) == 256)
    return a.d == 128 ? tctw::launch_t<128, 2>(a, W, sketch, lse_tok, stat_part, st)
                      : tctw::launch_t<64, 2>(a, W, sketch, lse_tok, stat_part, st);
  return a.d == 128 ? tctw::launch_t<128, 1>(a, W, sketch, lse_tok, stat_part, st)
                    : tctw::launch_t<64, 1>(a, W, sketch, lse_tok, stat_part, st);
}

}  // namespace sa
