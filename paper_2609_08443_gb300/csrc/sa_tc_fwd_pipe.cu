// Software-pipelined cluster-pair forward of the SA sketching step for
// P = 512 prototypes (paper Sec. 3.1; FlashSA's streaming scheme, Sec. 4.4).
//
// A cluster of two CTAs shares every 128-token tile; CTA r holds prototypes
// [256 r, 256 r + 256), so each token's softmax over all 512 prototypes needs
// the (max, sum) partials of four threads: the two warpgroups of each CTA,
// each holding 128 of the token's scores.  The exchange crosses SMs and takes
// longer than the rest of a tile's softmax, so the softmax warps overlap it
// with the next tile:
//
//   A(i):  scores of tile i from TMEM (twice: max, then exp2 with that max),
//          exponentials kept as fp16 pairs in registers, S released at once;
//          the thread's (max, sum) goes to shared memory and, with st.async,
//          into the peer CTA (four partials per token in each CTA).
//   B(i-1): the four partials of tile i-1 (landed while A(i) ran) are combined
//          in one fixed order -- bitwise the same (max, sum) in all four
//          threads of a token --, the weights of tile i-1 are scaled and
//          stored as bf16 for the aggregation UMMA.
//
// The UMMA issuer follows the same order: S(i+1) as soon as S(i) is released,
// then O(i-1) once its weights are stored.  K and V tiles come from two
// producers with rings of their own, so a V load held back by a pending
// aggregation never delays the next K.
// Warp roles: 0 = K producer (and prototypes), 1 = UMMA issuer, 2 = TMEM
// allocator, 3 = V producer, 4..11 = softmax + epilogue.  Every wait is
// bounded (sa_ptx.cuh).
#include <cuda.h>
#include <cuda_fp16.h>

#include "sa_ptx.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace sa {
namespace tcp {

using namespace ptx;
using namespace tcc;

constexpr uint32_t kRegsCtl = 88, kRegsSoft = 208;
static_assert(128 * kRegsCtl + 256 * kRegsSoft == 384 * 168, "register split = launch allocation");

template <int D>
struct PCfg {
  static constexpr int PS = 256;  // prototypes per CTA
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = PS * D * 2;
  static constexpr int W_BYTES = T * PS * 2;
  static constexpr int NK = (D == 128) ? 1 : 2;  // K slots
  static constexpr int NV = (D == 128) ? 1 : 2;  // V slots
  static constexpr int X_BYTES = 2 * 4 * T * 8;  // [2 buffers][4 partials][T] (max, sum)
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + NK * KV_TILE;
  static constexpr int OFF_W = OFF_V + NV * KV_TILE;
  static constexpr int OFF_X = OFF_W + W_BYTES;
  static constexpr int OFF_BAR = OFF_X + X_BYTES;
  static constexpr int NBAR = 2 * NK + 2 * NV + 15;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;  // TMEM address, abort flag + wait limit, skip flag
  static constexpr int SMEM = OFF_MISC + 16;
  static constexpr bool TRANS = (D == 128);  // O^T = V^T A (d on TMEM lanes)
  static constexpr int O_COLS = TRANS ? PS : (PS / 128) * D;
  static constexpr int S_COL = 0, O_COL = PS;
  static constexpr int TMEM_COLS = tmem_cols_for(PS + O_COLS);
  static constexpr int HALF = PS / 2;  // prototypes per softmax warpgroup
  static_assert(SMEM <= 232448 && TMEM_COLS <= 512, "budget");
  static_assert(OFF_K % 1024 == 0 && OFF_V % 1024 == 0 && OFF_W % 1024 == 0, "swizzle atoms");
};

__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ float2 unpack_f16(uint32_t w) {
  return __half22float2(*reinterpret_cast<const __half2*>(&w));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tc_fwd_pipe_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                       const __grid_constant__ CUtensorMap tmQ, Args a, float* __restrict__ sketch,
                       float* __restrict__ lse_out) {
  using C = PCfg<D>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Both CTAs of a pair must reach the cluster barriers below, so a failed
  // call or a misaligned base only skips the work.
  bool skip = ws_failed(a.ws);
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xA21u);
    skip = true;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sK = sbase + C::OFF_K, sV = sbase + C::OFF_V, sW = sbase + C::OFF_W;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto kfull = [&](int s) { return bar0 + 8u * s; };
  auto kempty = [&](int s) { return bar0 + 8u * (C::NK + s); };
  auto vfull = [&](int s) { return bar0 + 8u * (2 * C::NK + s); };
  auto vempty = [&](int s) { return bar0 + 8u * (2 * C::NK + C::NV + s); };
  const uint32_t b1 = bar0 + 8u * (2 * C::NK + 2 * C::NV);
  const uint32_t q_full = b1, q_empty = b1 + 8, s_full = b1 + 16, s_empty = b1 + 24, w_full = b1 + 32,
                 w_empty = b1 + 40, o_full = b1 + 48, o_empty = b1 + 56, drain = b1 + 64;
  // exchange buffer b: x_full = the four partials are in (8 local warp arrivals
  // + one arrival that expects the peer's 2 KB of st.async); x_free = this
  // CTA's warps have read it; r_free = the PEER's warps have read theirs (so
  // this CTA may push into it again)
  auto x_full = [&](int b) { return b1 + 72 + 8u * b; };
  auto x_free = [&](int b) { return b1 + 88 + 8u * b; };
  auto r_free = [&](int b) { return b1 + 104 + 8u * b; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  volatile uint32_t* skip_flag = reinterpret_cast<volatile uint32_t*>(smem + C::OFF_MISC + 8);
  const uint32_t rank = cluster_rank(), peer = rank ^ 1u;

  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = int(gridDim.x >> 1), wk = int(blockIdx.x >> 1);  // the two CTAs of cluster c are worker c
  const int p0 = int(rank) * C::PS;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  int ntiles = int(te - tb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NK; ++s) {
      mbar_init(kfull(s), 1);
      mbar_init(kempty(s), 1);
    }
    for (int s = 0; s < C::NV; ++s) {
      mbar_init(vfull(s), 1);
      mbar_init(vempty(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(s_full, 1);
    mbar_init(s_empty, kSoftWarps);
    mbar_init(w_full, kSoftWarps);
    mbar_init(w_empty, 1);
    mbar_init(o_full, 1);
    mbar_init(o_empty, kSoftWarps);
    mbar_init(drain, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(x_full(b), kSoftWarps + 1);
      mbar_init(x_free(b), kSoftWarps);
      mbar_init(r_free(b), kSoftWarps);
    }
    wait_ctl_init(abort_flag, a.ws);
    *skip_flag = skip ? 1u : 0u;
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  cluster_sync_all();  // barriers of both CTAs initialised; both skip if either must
  if (*skip_flag || ld_cluster_u32(mapa_shared(smem_u32(smem + C::OFF_MISC + 8), peer))) ntiles = 0;
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (ntiles > 0 && warp < kSoftWarp0) {
    setmaxnreg_dec<kRegsCtl>();
    if (warp == 0 && lane == 0) {
      // --------------------------------------------- K producer (+ prototypes)
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      TileWalker it(a, tb, te, T), pf(a, tb, te, T);
      pf.next();
      pf.next();
      int hc = 0, prev_q = -1, loaded = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        if (li + 2 < ntiles) {  // K and V of tile li + 2 into L2, so the ring loads hit L2
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) {
            tma_prefetch_l2_3d(&tmK, 64 * dh, pf.h, int(pf.tok0));
            tma_prefetch_l2_3d(&tmV, 64 * dh, pf.h, int(pf.tok0));
          }
          pf.next();
        }
        if (it.qk != prev_q) {  // a new head (or, with per-user queries, a new user)
          if (hc > 0) ok = mbar_wait(q_empty, uint32_t(hc - 1) & 1u, abort_flag, a.ws, 0x111);
          if (!ok) break;
          mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(sQ + dh * C::PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
          prev_q = it.qk;
          ++hc;
        }
        const int s = li % C::NK, use = li / C::NK;
        if (use > 0) ok = mbar_wait(kempty(s), uint32_t(use - 1) & 1u, abort_flag, a.ws, 0x112);
        if (!ok) break;
        mbar_arrive_expect_tx(kfull(s), C::KV_TILE);
#pragma unroll
        for (int dh = 0; dh < D / 64; ++dh)
          tma_load_3d(sK + s * C::KV_TILE + dh * T * 128, &tmK, kfull(s), 64 * dh, it.h, int(it.tok0));
        loaded = li + 1;
        it.next();
      }
      if (!ok) {  // the copies still in flight land before the CTA may exit
        for (int li = (loaded > C::NK ? loaded - C::NK : 0); li < loaded; ++li)
          mbar_wait_bounded(kfull(li % C::NK), uint32_t(li / C::NK) & 1u, 200000000ull);
        if (hc > 0) mbar_wait_bounded(q_full, uint32_t(hc - 1) & 1u, 200000000ull);
      }
    } else if (warp == 3 && lane == 0) {
      // ---------------------------------------------------------- V producer
      TileWalker it(a, tb, te, T);
      int loaded = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        const int s = li % C::NV, use = li / C::NV;
        if (use > 0) ok = mbar_wait(vempty(s), uint32_t(use - 1) & 1u, abort_flag, a.ws, 0x113);
        if (!ok) break;
        mbar_arrive_expect_tx(vfull(s), C::KV_TILE);
#pragma unroll
        for (int dh = 0; dh < D / 64; ++dh)
          tma_load_3d(sV + s * C::KV_TILE + dh * T * 128, &tmV, vfull(s), 64 * dh, it.h, int(it.tok0));
        loaded = li + 1;
        it.next();
      }
      if (!ok) {
        for (int li = (loaded > C::NV ? loaded - C::NV : 0); li < loaded; ++li)
          mbar_wait_bounded(vfull(li % C::NV), uint32_t(li / C::NV) & 1u, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      // ---------------------------------------------------------- UMMA issuer
      // Order: S(0); then per tile i: S(i+1) once S(i) is released, O(i-1)
      // once its weights are stored (the softmax warps' A(i+1) releases S(i+1)
      // before their B(i) stores the weights of tile i).
      constexpr uint32_t idS = idesc_bf16(128, C::PS, 0, 0);
      constexpr uint32_t idO = C::TRANS ? idesc_bf16(128, C::PS, 1, 1) : idesc_bf16(128, D, 1, 1);
      TileWalker ws_(a, tb, te, T), wo(a, tb, te, T);
      int hc = 0, sc = 0;
      bool ok = true;
      auto wt = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return ok = ok && mbar_wait(bar, par, abort_flag, a.ws, site);
      };
      int prev_q = -1;
      // S(li) = K(li) Q^T into the S columns; ws_ is at tile li
      auto issue_S = [&](int li) {
        if (ws_.qk != prev_q) {
          wt(q_full, uint32_t(hc) & 1u, 0x211);
          ++hc;
          prev_q = ws_.qk;
        }
        const int s = li % C::NK;
        wt(kfull(s), uint32_t(li / C::NK) & 1u, 0x212);
        if (!ok) return;
        tc_fence_after();
        const uint32_t kaddr = sK + s * C::KV_TILE;
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint64_t ad = sdesc(kaddr + (k >> 2) * (T * 128) + (k & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc(sQ + (k >> 2) * (C::PS * 128) + (k & 3) * 32, 16, 1024);
          umma_ss(tmem + C::S_COL, ad, bd, idS, k > 0 ? 1u : 0u);
        }
        umma_commit(s_full);
        umma_commit(kempty(s));
        int64_t t0n;
        int nn, hn, qn;
        ws_.peek_next(t0n, nn, hn, qn);
        if (li + 1 >= ntiles || qn != ws_.qk) umma_commit(q_empty);  // last S of these prototypes
        ws_.next();
      };
      // O(li) += V(li)^T A(li) (or A^T V); wo is at tile li
      auto issue_O = [&](int li) {
        wt(w_full, uint32_t(li) & 1u, 0x213);
        const int s = li % C::NV;
        wt(vfull(s), uint32_t(li / C::NV) & 1u, 0x214);
        if (wo.seg_first && sc > 0) wt(o_empty, uint32_t(sc - 1) & 1u, 0x215);
        if (!ok) return;
        tc_fence_after();
        const uint32_t vaddr = sV + s * C::KV_TILE;
#pragma unroll
        for (int k = 0; k < T / 16; ++k) {
          const uint32_t acc = (wo.seg_first && k == 0) ? 0u : 1u;
          if (C::TRANS) {
            // O^T[d, p] += sum_t V[t, d] A[t, p]: A-operand V^T (MN-major), B-operand A (MN-major)
            umma_ss(tmem + C::O_COL, sdesc(vaddr + k * 2048, T * 128, 1024), sdesc(sW + k * 2048, T * 128, 1024),
                    idO, acc);
          } else {
#pragma unroll
            for (int mb = 0; mb < C::PS / 128; ++mb)
              // O[p, d] += sum_t A[t, p] V[t, d]: A-operand A^T (MN-major), B-operand V (MN-major)
              umma_ss(tmem + C::O_COL + mb * D, sdesc(sW + mb * 2 * (T * 128) + k * 2048, T * 128, 1024),
                      sdesc(vaddr + k * 2048, T * 128, 1024), idO, acc);
          }
        }
        umma_commit(w_empty);
        umma_commit(vempty(s));
        if (wo.seg_last) {
          umma_commit(o_full);
          ++sc;
        }
        wo.next();
      };
      issue_S(0);
      for (int li = 0; li < ntiles && ok; ++li) {
        if (li + 1 < ntiles) {
          wt(s_empty, uint32_t(li) & 1u, 0x216);  // the softmax warps hold S(li)
          if (ok) issue_S(li + 1);
        }
        if (ok && li >= 1) issue_O(li - 1);
      }
      if (ok) issue_O(ntiles - 1);
      umma_commit(drain);  // no UMMA may still run when TMEM is released
      mbar_wait_bounded(drain, 0, 200000000ull);
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<kRegsSoft>();
    // ------------------------------------------------ softmax + epilogue warps
    const int sw = (warp - kSoftWarp0) >> 2;  // warpgroup: prototype half of this CTA
    const int q = warp & 3;                   // TMEM lane quadrant
    const int row = 32 * q + lane;            // token within the tile
    const uint32_t lane_off = uint32_t(32 * q) << 16;
    const float c2 = a.scale * 1.4426950408889634f;  // scale * log2(e)
    float2* X = reinterpret_cast<float2*>(smem + C::OFF_X);
    const uint32_t x_peer = mapa_shared(sbase + C::OFF_X, peer);
    const int slot = int(rank) * 2 + sw;  // this thread's partial among the four of its token
    TileWalker wb(a, tb, te, T);  // the tile of phase B
    bool ok = true;
    auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
      return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
    };
    auto wwait_cl = [&](uint32_t bar, uint32_t par, uint32_t site) {
      return __all_sync(0xffffffffu, mbar_wait_cluster(bar, par, abort_flag, a.ws, site));
    };
    uint32_t pk_prev[C::HALF / 2];  // exponentials of the previous tile, fp16 pairs
    float m_prev = 0.f;
    int seg_idx = 0;
    for (int it = 0; it <= ntiles && ok; ++it) {
      uint32_t pk[C::HALF / 2];
      float m = -INFINITY;
      if (it < ntiles) {
        // ------------------------------------------------------- A(it)
        ok = wwait(s_full, uint32_t(it) & 1u, 0x311);
        if (!ok) break;
        tc_fence_after();
        const uint32_t scol = tmem + lane_off + C::S_COL + sw * C::HALF;
        {
          float v[64];
#pragma unroll
          for (int c = 0; c < C::HALF / 64; ++c) {
            tmem_ld32(scol + 64 * c, v);
            tmem_ld32(scol + 64 * c + 32, v + 32);
            tmem_ld_wait();
            m = fmaxf(m, row_max<64>(v));
          }
        }
        const float sh = m * c2;
        float2 z0 = make_float2(0.f, 0.f), z1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < C::HALF / 32; ++c) {
          float v[32];
          tmem_ld32(scol + 32 * c, v);
          tmem_ld_wait();
          const float2 cc = make_float2(c2, c2), ns = make_float2(-sh, -sh);
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            float2 x0 = __ffma2_rn(make_float2(v[j], v[j + 1]), cc, ns);
            float2 x1 = __ffma2_rn(make_float2(v[j + 2], v[j + 3]), cc, ns);
            x0.x = ex2(x0.x);
            x0.y = ex2(x0.y);
            x1.x = ex2(x1.x);
            x1.y = ex2(x1.y);
            z0 = __fadd2_rn(z0, x0);
            z1 = __fadd2_rn(z1, x1);
            pk[16 * c + j / 2] = pack_f16(x0.x, x0.y);
            pk[16 * c + j / 2 + 1] = pack_f16(x1.x, x1.y);
          }
        }
        const float z = (z0.x + z0.y) + (z1.x + z1.y);
        // S(it) is in registers: its columns may take S(it+1)
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(s_empty);
        // publish this thread's partial: into this CTA's buffer and the peer's
        const int b = it & 1;
        if (it >= 2) {
          ok = wwait(x_free(b), uint32_t((it - 2) >> 1) & 1u, 0x312);  // this CTA's readers of tile it-2
          if (!ok) break;
        }
        X[(b * 4 + slot) * T + row] = make_float2(m, z);
        if (it >= 2) {
          ok = wwait_cl(r_free(b), uint32_t((it - 2) >> 1) & 1u, 0x313);  // the peer's readers of tile it-2
          if (!ok) break;
        }
        st_async_f2(x_peer + uint32_t(((b * 4 + slot) * T + row) * 8), make_float2(m, z),
                    mapa_shared(x_full(b), peer));
        __syncwarp();
        if (lane == 0) mbar_arrive(x_full(b));
        if (warp == kSoftWarp0 && lane == 0) mbar_arrive_expect_tx(x_full(b), 2u * T * 8u);
      }
      if (it >= 1) {
        // ----------------------------------------------------- B(it - 1)
        const int bp = (it - 1) & 1;
        ok = wwait_cl(x_full(bp), uint32_t((it - 1) >> 1) & 1u, 0x314);
        if (!ok) break;
        const float2 p0v = X[(bp * 4 + 0) * T + row], p1v = X[(bp * 4 + 1) * T + row];
        const float2 p2v = X[(bp * 4 + 2) * T + row], p3v = X[(bp * 4 + 3) * T + row];
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(x_free(bp));
          mbar_arrive_cluster(mapa_shared(r_free(bp), peer));
        }
        // the token's (max, sum) over all 512 prototypes, in partial order 0..3
        const float M = fmaxf(fmaxf(p0v.x, p1v.x), fmaxf(p2v.x, p3v.x));
        const float Z = ((p0v.y * ex2((p0v.x - M) * c2) + p1v.y * ex2((p1v.x - M) * c2)) +
                         p2v.y * ex2((p2v.x - M) * c2)) +
                        p3v.y * ex2((p3v.x - M) * c2);
        const bool valid = row < wb.n;
        // rows past the tile's tokens get exact zero weights
        const float f = valid ? ex2((m_prev - M) * c2) / Z : 0.f;
        if (rank == 0 && sw == 0 && valid && lse_out) lse_out[(wb.tok0 + row) * a.H + wb.h] = M * a.scale + logf(Z);
        if (it >= 2) {
          ok = wwait(w_empty, uint32_t(it - 2) & 1u, 0x315);  // O(it-2) has read the weights
          if (!ok) break;
        }
        // weights -> shared memory, [PS/64 blocks][128 tokens][64 prototypes], 128-byte swizzle
        uint8_t* wrow = smem + C::OFF_W + row * 128;
        const float2 ff = make_float2(f, f);
#pragma unroll
        for (int k = 0; k < C::HALF / 8; ++k) {
          const int p = sw * C::HALF + 8 * k;
          const int blk = p >> 6, chunk = (p & 63) >> 3;
          uint32_t o[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float2 e = __fmul2_rn(unpack_f16(pk_prev[4 * k + j]), ff);
            o[j] = pack_bf16(e.x, e.y);
          }
          *reinterpret_cast<uint4*>(wrow + blk * (T * 128) + ((chunk ^ (row & 7)) << 4)) =
              make_uint4(o[0], o[1], o[2], o[3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(w_full);
        if (wb.seg_last) {
          ok = wwait(o_full, uint32_t(seg_idx) & 1u, 0x316);
          if (!ok) break;
          tc_fence_after();
          const bool whole = wb.seg0 >= tb && wb.seg1 <= te;
          float* dst = whole ? sketch + ((int64_t(wb.b) * a.H + wb.h) * a.P + p0) * D
                             : a.partial + ((int64_t(wk) * 2 + partial_slot(total, W, wk, wb.seg0)) * a.P + p0) * D;
          store_sketch<D, C::PS, C::TRANS, C::O_COL>(tmem, lane_off, sw, q, lane, dst);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(o_empty);
          ++seg_idx;
        }
        wb.next();
      }
      if (it < ntiles) {
#pragma unroll
        for (int j = 0; j < C::HALF / 2; ++j) pk_prev[j] = pk[j];
        m_prev = m;
      }
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  // the peer may still push into this CTA's shared memory or arrive on its barriers
  cluster_sync_all();
}

template <int D>
static cudaError_t launch_pipe_t(const Args& a, int W, float* sketch, float* lse_out, cudaStream_t st) {
  using C = PCfg<D>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, C::PS))
    return cudaErrorInvalidValue;
  auto fn = &tc_fwd_pipe_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  // one cluster of two CTAs per worker; CTA rank r holds prototypes [256 r, 256 r + 256)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * W, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fn, tk, tv, tq, a, sketch, lse_out);
}

}  // namespace tcp

cudaError_t launch_tc_fwd_pipe(const Args& a, int W, float* sketch, float* lse, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  return a.d == 128 ? tcp::launch_pipe_t<128>(a, W, sketch, lse, st) : tcp::launch_pipe_t<64>(a, W, sketch, lse, st);
}

}  // namespace sa
