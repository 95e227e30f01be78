// Cluster-pair forward of the SA sketching step for P = 512 prototypes with
// sixteen softmax warps (paper Sec. 3.1; FlashSA's streaming scheme, Sec. 4.4).
//
// A cluster of two CTAs shares every 128-token tile; CTA r holds prototypes
// [256 r, 256 r + 256).  The per-token softmax over all 512 prototypes is the
// critical path of the step -- its exponentials alone keep an SM's MUFU busy
// for a quarter of a tile's tensor time, and with two softmax warps per SM
// sub-partition its dependent TMEM loads, max, exp, scale and stores left the
// tensor pipe idle more than half the time.  Here four warpgroups share the
// work: warpgroup g of CTA r holds, for every token of the tile, the 64 scores
// of prototypes [256 r + 64 g, +64) -- four warps per sub-partition to hide
// each other's latency, half the registers and instructions per thread.
//
// Per tile:
//   1. TMA: K and V tiles from two producers with rings of their own; the
//      prototype block Q ([256][d]) stays resident while the head does not
//      change.
//   2. UMMA  S^T = K Q^T  (M = 128 tokens, N = 256 prototypes, K = d) into TMEM.
//   3. Each softmax thread loads its 64 scores, releases S at once, and forms
//      exp2((s - m) c) with its own maximum m; its partial (m, sum) goes into
//      this CTA's exchange buffer and, with st.async, into the peer CTA's, so
//      both CTAs hold the eight partials of every token.  All four threads of
//      a token in each CTA combine the eight in one fixed order: bitwise the
//      same (max, sum) everywhere, and the per-token log-sum-exp.
//   4. The weights, scaled by exp2((m - M) c) / Z, go to shared memory as bf16
//      and UMMA accumulates the sketch: O^T += V^T A (d = 128) or O += A^T V.
//   5. When a user's segment ends the sketch (or a worker's piece of it) is
//      read back from TMEM and stored.
// Warp roles: 0 = K producer (and prototypes), 1 = UMMA issuer, 2 = TMEM
// allocator, 3 = V producer, 4..19 = softmax + epilogue.  Every wait is
// bounded (sa_ptx.cuh).
#include <cuda.h>

#include "sa_ptx.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace sa {
namespace tcq {

using namespace ptx;
using namespace tcc;

constexpr int kWThreads = 640;  // 20 warps
constexpr int kWSoft0 = 4;      // warps 4..19: softmax / epilogue
constexpr int kWSoftWarps = 16;
// Registers: 640 threads launch with 96 each; the control warpgroup (producers,
// issuer) keeps 64 and the four softmax warpgroups take 104.
constexpr uint32_t kWRegsCtl = 64, kWRegsSoft = 104;
static_assert(128 * kWRegsCtl + 512 * kWRegsSoft == 640 * 96, "register split = launch allocation");

template <int D>
struct WCfg {
  static constexpr int PS = 256;    // prototypes per CTA
  static constexpr int GP = 64;     // prototypes per softmax warpgroup
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = PS * D * 2;
  static constexpr int W_BYTES = T * PS * 2;
  static constexpr int NK = (D == 128) ? 1 : 2;  // K slots
  static constexpr int NV = (D == 128) ? 1 : 2;  // V slots
  static constexpr int NPART = 8;                // partials per token: 4 warpgroups x 2 CTAs
  static constexpr int X_BYTES = 2 * NPART * T * 8;  // [2 buffers][8 partials][T] (max, sum)
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + NK * KV_TILE;
  static constexpr int OFF_W = OFF_V + NV * KV_TILE;
  static constexpr int OFF_X = OFF_W + W_BYTES;
  static constexpr int OFF_BAR = OFF_X + X_BYTES;
  static constexpr int NBAR = 2 * NK + 2 * NV + 16;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;  // TMEM address, abort flag + wait limit, skip flag
  static constexpr int SMEM = OFF_MISC + 16;
  static constexpr bool TRANS = (D == 128);  // O^T = V^T A (d on TMEM lanes)
  static constexpr int O_COLS = TRANS ? PS : (PS / 128) * D;
  static constexpr int S_COL = 0, O_COL = PS;
  static constexpr int TMEM_COLS = tmem_cols_for(PS + O_COLS);
  static_assert(SMEM <= 232448 && TMEM_COLS <= 512, "budget");
  static_assert(OFF_K % 1024 == 0 && OFF_V % 1024 == 0 && OFF_W % 1024 == 0, "swizzle atoms");
};

// The CTA's sketch block (256 prototypes x D) from TMEM to global memory,
// shared by the 16 softmax warps: warp (g, q) takes TMEM lane quadrant q and
// the g-th quarter of the columns.
template <int D>
__device__ __forceinline__ void store_block(uint32_t tmem, uint32_t lane_off, int g, int q, int lane, float* dst) {
  using C = WCfg<D>;
  float v[32];
  if (C::TRANS) {  // lane = feature, column = prototype
    const int d = 32 * q + lane;
#pragma unroll 1
    for (int c = 0; c < C::GP / 32; ++c) {
      const int pbase = g * C::GP + 32 * c;
      tmem_ld32(tmem + lane_off + C::O_COL + pbase, v);
      tmem_ld_wait();
      float* col = dst + int64_t(pbase) * D + d;
#pragma unroll
      for (int k = 0; k < 32; ++k) col[k * D] = v[k];
    }
  } else {  // two blocks of 128 prototypes on lanes, D = 64 columns each
    const int blk = g >> 1, c = 32 * (g & 1);
    const int p = 128 * blk + 32 * q + lane;
    tmem_ld32(tmem + lane_off + C::O_COL + blk * D + c, v);
    tmem_ld_wait();
    float4* o = reinterpret_cast<float4*>(dst + int64_t(p) * D + c);
#pragma unroll
    for (int k = 0; k < 8; ++k) o[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
  }
}

template <int D>
__global__ void __launch_bounds__(kWThreads, 1)
    tc_fwd_wide_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                       const __grid_constant__ CUtensorMap tmQ, Args a, float* __restrict__ sketch,
                       float* __restrict__ lse_out) {
  using C = WCfg<D>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Both CTAs of a pair must reach the cluster barriers below, so a failed
  // call or a misaligned base only skips the work.
  bool skip = ws_failed(a.ws);
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xA31u);
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
  // exchange buffer b (tiles alternate): x_full = the eight partials are in
  // (16 local warp arrivals + one arrival expecting the peer's 4 KB of
  // st.async); x_free = this CTA's warps have read it; r_free = the PEER's
  // warps have read theirs, so this CTA may push into it again
  auto x_full = [&](int b) { return b1 + 72 + 8u * b; };
  auto x_free = [&](int b) { return b1 + 88 + 8u * b; };
  auto r_free = [&](int b) { return b1 + 104 + 8u * b; };
  const uint32_t never = b1 + 120;  // completed by nothing: the forced timeout of a test limit
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
    mbar_init(s_empty, kWSoftWarps);
    mbar_init(w_full, kWSoftWarps);
    mbar_init(w_empty, 1);
    mbar_init(o_full, 1);
    mbar_init(o_empty, kWSoftWarps);
    mbar_init(drain, 1);
    mbar_init(never, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(x_full(b), kWSoftWarps + 1);
      mbar_init(x_free(b), kWSoftWarps);
      mbar_init(r_free(b), kWSoftWarps);
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

  if (ntiles > 0 && warp < kWSoft0) {
    setmaxnreg_dec<kWRegsCtl>();
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
          if (hc > 0) ok = mbar_wait(q_empty, uint32_t(hc - 1) & 1u, abort_flag, a.ws, 0x121);
          if (!ok) break;
          mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(sQ + dh * C::PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
          prev_q = it.qk;
          ++hc;
        }
        const int s = li % C::NK, use = li / C::NK;
        if (use > 0) ok = mbar_wait(kempty(s), uint32_t(use - 1) & 1u, abort_flag, a.ws, 0x122);
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
        if (use > 0) ok = mbar_wait(vempty(s), uint32_t(use - 1) & 1u, abort_flag, a.ws, 0x123);
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
      // Order: S(0); then per tile i: S(i+1) once the softmax warps hold S(i)
      // in registers, O(i) once the weights of tile i are stored.
      constexpr uint32_t idS = idesc_bf16(128, C::PS, 0, 0);
      constexpr uint32_t idO = C::TRANS ? idesc_bf16(128, C::PS, 1, 1) : idesc_bf16(128, D, 1, 1);
      TileWalker ws_(a, tb, te, T), wo(a, tb, te, T);
      int hc = 0, sc = 0, prev_q = -1;
      // under a test limit (sa_set_wait_limit_ns) the issuer first waits for a
      // barrier nothing completes: the limit runs out and the CTA takes its
      // abort path (drains, TMEM freed, SA_ERR_TIMEOUT)
      bool ok = ctl_wait_limit(abort_flag) >= kPollLimitNs || mbar_wait(never, 0, abort_flag, a.ws, 0x220);
      auto wt = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return ok = ok && mbar_wait(bar, par, abort_flag, a.ws, site);
      };
      auto issue_S = [&](int li) {  // ws_ is at tile li
        if (ws_.qk != prev_q) {
          wt(q_full, uint32_t(hc) & 1u, 0x221);
          ++hc;
          prev_q = ws_.qk;
        }
        const int s = li % C::NK;
        wt(kfull(s), uint32_t(li / C::NK) & 1u, 0x222);
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
      auto issue_O = [&](int li) {  // wo is at tile li
        wt(w_full, uint32_t(li) & 1u, 0x223);
        const int s = li % C::NV;
        wt(vfull(s), uint32_t(li / C::NV) & 1u, 0x224);
        if (wo.seg_first && sc > 0) wt(o_empty, uint32_t(sc - 1) & 1u, 0x225);
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
          wt(s_empty, uint32_t(li) & 1u, 0x226);  // the softmax warps hold S(li)
          if (ok) issue_S(li + 1);
        }
        if (ok) issue_O(li);
      }
      umma_commit(drain);  // no UMMA may still run when TMEM is released
      mbar_wait_bounded(drain, 0, 200000000ull);
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<kWRegsSoft>();
    // ------------------------------------------------ softmax + epilogue warps
    const int g = (warp - kWSoft0) >> 2;  // warpgroup: prototypes [64 g, 64 g + 64) of this CTA
    const int q = warp & 3;               // TMEM lane quadrant
    const int row = 32 * q + lane;        // token within the tile
    const uint32_t lane_off = uint32_t(32 * q) << 16;
    const float c2 = a.scale * 1.4426950408889634f;  // scale * log2(e)
    float2* X = reinterpret_cast<float2*>(smem + C::OFF_X);
    const uint32_t x_peer = mapa_shared(sbase + C::OFF_X, peer);
    const int slot = int(rank) * 4 + g;  // this thread's partial among the eight of its token
    TileWalker cur(a, tb, te, T);
    bool ok = true;
    auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
      return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
    };
    auto wwait_cl = [&](uint32_t bar, uint32_t par, uint32_t site) {
      return __all_sync(0xffffffffu, mbar_wait_cluster(bar, par, abort_flag, a.ws, site));
    };
    int seg_idx = 0;
    for (int li = 0; li < ntiles && ok; ++li) {
      ok = wwait(s_full, uint32_t(li) & 1u, 0x321);
      if (!ok) break;
      tc_fence_after();
      float v[C::GP];
      tmem_ld32(tmem + lane_off + C::S_COL + g * C::GP, v);
      tmem_ld32(tmem + lane_off + C::S_COL + g * C::GP + 32, v + 32);
      tmem_ld_wait();
      // S is in registers: its columns may take the next tile's scores
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_empty);
      const float m = row_max<C::GP>(v);
      const float z = exp2_shift_sum<C::GP>(v, c2, m * c2);
      // this thread's partial into this CTA's exchange buffer and the peer's
      const int b = li & 1;
      if (li >= 2) {
        ok = wwait(x_free(b), uint32_t((li - 2) >> 1) & 1u, 0x322);  // this CTA's readers of tile li-2
        if (!ok) break;
        ok = wwait_cl(r_free(b), uint32_t((li - 2) >> 1) & 1u, 0x323);  // the peer's readers of tile li-2
        if (!ok) break;
      }
      const float2 part = make_float2(m, z);
      X[(b * C::NPART + slot) * T + row] = part;
      st_async_f2(x_peer + uint32_t(((b * C::NPART + slot) * T + row) * 8), part, mapa_shared(x_full(b), peer));
      __syncwarp();
      if (lane == 0) mbar_arrive(x_full(b));
      if (warp == kWSoft0 && lane == 0) mbar_arrive_expect_tx(x_full(b), 4u * T * 8u);
      ok = wwait_cl(x_full(b), uint32_t(li >> 1) & 1u, 0x324);
      if (!ok) break;
      // the token's (max, sum) over all 512 prototypes, partials in slot order
      float2 pp[C::NPART];
#pragma unroll
      for (int k = 0; k < C::NPART; ++k) pp[k] = X[(b * C::NPART + k) * T + row];
      const float M = fmaxf(fmaxf(fmax3(pp[0].x, pp[1].x, pp[2].x), fmax3(pp[3].x, pp[4].x, pp[5].x)),
                            fmaxf(pp[6].x, pp[7].x));
      float w[C::NPART];  // each partial's sum rescaled to the common maximum, all exponentials independent
      const float Mc = M * c2;
#pragma unroll
      for (int k = 0; k < C::NPART; ++k) w[k] = pp[k].y * ex2(fmaf(pp[k].x, c2, -Mc));
      const float Z = ((w[0] + w[1]) + (w[2] + w[3])) + ((w[4] + w[5]) + (w[6] + w[7]));  // fixed tree order
      // the partials are consumed (Z depends on every loaded value): the slots
      // of this buffer may be rewritten, locally and by the peer
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(x_free(b));
        mbar_arrive_relaxed_cluster(mapa_shared(r_free(b), peer));
      }
      const bool valid = row < cur.n;
      // rows past the tile's tokens get exact zero weights
      const float rz = __frcp_rn(Z);
      scale_row<C::GP>(v, valid ? ex2(fmaf(m, c2, -Mc)) * rz : 0.f);
      // natural log of Z through the log2 unit (Z lies in [1, 512])
      if (rank == 0 && g == 0 && valid && lse_out)
        lse_out[(cur.tok0 + row) * a.H + cur.h] = M * a.scale + __log2f(Z) * 0.6931471805599453f;
      if (li > 0) {
        ok = wwait(w_empty, uint32_t(li - 1) & 1u, 0x325);  // O(li-1) has read the weights
        if (!ok) break;
      }
      // weights -> shared memory, [PS/64 blocks][128 tokens][64 prototypes], 128-byte swizzle:
      // warpgroup g fills block g
      uint8_t* wrow = smem + C::OFF_W + g * (T * 128) + row * 128;
#pragma unroll
      for (int k = 0; k < C::GP / 8; ++k) {
        uint4 pk;
        pk.x = pack_bf16(v[8 * k + 0], v[8 * k + 1]);
        pk.y = pack_bf16(v[8 * k + 2], v[8 * k + 3]);
        pk.z = pack_bf16(v[8 * k + 4], v[8 * k + 5]);
        pk.w = pack_bf16(v[8 * k + 6], v[8 * k + 7]);
        *reinterpret_cast<uint4*>(wrow + ((k ^ (row & 7)) << 4)) = pk;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(w_full);
      if (cur.seg_last) {
        ok = wwait(o_full, uint32_t(seg_idx) & 1u, 0x326);
        if (!ok) break;
        tc_fence_after();
        const bool whole = cur.seg0 >= tb && cur.seg1 <= te;
        float* dst = whole ? sketch + ((int64_t(cur.b) * a.H + cur.h) * a.P + p0) * D
                           : a.partial + ((int64_t(wk) * 2 + partial_slot(total, W, wk, cur.seg0)) * a.P + p0) * D;
        store_block<D>(tmem, lane_off, g, q, lane, dst);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(o_empty);
        ++seg_idx;
      }
      cur.next();
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
static cudaError_t launch_wide_t(const Args& a, int W, float* sketch, float* lse_out, cudaStream_t st) {
  using C = WCfg<D>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, C::PS))
    return cudaErrorInvalidValue;
  auto fn = &tc_fwd_wide_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  // one cluster of two CTAs per worker; CTA rank r holds prototypes [256 r, 256 r + 256)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * W, 1, 1);
  cfg.blockDim = dim3(kWThreads, 1, 1);
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

}  // namespace tcq

cudaError_t launch_tc_fwd_wide(const Args& a, int W, float* sketch, float* lse, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  return a.d == 128 ? tcq::launch_wide_t<128>(a, W, sketch, lse, st) : tcq::launch_wide_t<64>(a, W, sketch, lse, st);
}

}  // namespace sa
