// tcgen05 / TMEM / TMA backward kernels of the SA sketching step (sm_103a).
//
// Chain rule of Sec. 3.1 with upstream G = dL/dsketch[b, h] and the forward's
// per-token log-sum-exp (FlashSA's softmax statistic, Sec. 4.4), so the
// weights are recomputed as A = exp(S - lse) without any reduction:
//   S^T  = K Q^T                 (UMMA, tokens on TMEM lanes)
//   A    = exp(scale S - lse)    (registers; bf16 copy in shared memory)
//   dA^T = V G^T                 (UMMA)
//   dV   = A G                   (UMMA, contraction over prototypes)
//   D_i  = dV_i . v_i            (= sum_j A[j,i] dA[j,i])
//   dS   = A o (dA - D)          (registers -> bf16 in shared memory)
//   dK   = scale dS Q            (UMMA)
//   dQ  += scale dS^T K          (UMMA, accumulated in TMEM over a worker's
//                                 tiles of one head; per-worker partials are
//                                 summed in worker order afterwards)
// Modes: kFull keeps all P prototypes in one CTA (TMEM: S/dA, dV, dK, dQ);
// kSlice handles one slice of prototypes and only dQ, with D_i read from the
// token-side kernel (tc_bwd_tok_kernel) that computes dV, dK and D_i for
// shapes whose four TMEM accumulators do not fit one SM.
// Warp roles: 0 TMA, 1 UMMA, 2-3 dsketch loader (fp32 -> bf16 swizzled),
// 4-11 softmax / epilogue.  Every wait is bounded.
#include <cuda.h>

#include "sa_ptx.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace sa {
namespace tcb {

using namespace ptx;
using namespace tcc;

enum Mode { kFull = 0, kSlice = 1 };

template <int D, int PS, int MODE>
struct BCfg {
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = PS * D * 2;
  static constexpr int AB_BYTES = T * PS * 2;
  static constexpr int NSLOT = 4;  // even: even slots hold K tiles, odd slots V tiles
  static constexpr int NBAR = 2 * NSLOT + 20;
  // two dsketch buffers where shared memory holds them, so the next user's
  // dsketch is converted while this user's tiles run
  static constexpr int NG = (3 * Q_BYTES + AB_BYTES + NSLOT * KV_TILE + NBAR * 8 + 16 <= 232448) ? 2 : 1;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_G = Q_BYTES;
  static constexpr int OFF_AB = OFF_G + NG * Q_BYTES;
  static constexpr int OFF_RING = OFF_AB + AB_BYTES;
  static constexpr int OFF_BAR = OFF_RING + NSLOT * KV_TILE;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = OFF_MISC + 16;
  static constexpr int NSD = (MODE == kSlice) ? 2 : 1;  // S/dA buffers (slice mode has TMEM to spare)
  static constexpr int SD_COL = 0;
  static constexpr int DV_COL = PS;
  static constexpr int DK_COL = PS + D;
  static constexpr int DQ_COL = (MODE == kFull) ? PS + 2 * D : NSD * PS;
  static constexpr int TMEM_COLS = tmem_cols_for(DQ_COL + (PS / 128) * D);
  static constexpr int HALF = PS / 2;
  static_assert(TMEM_COLS <= 512, "TMEM budget");
  static_assert(SMEM <= 232448, "shared memory budget");
};

// one token row of dV or dK (fp32 from TMEM) -> bf16 global row, columns
// [c0, c0 + NCOL) of this warpgroup's half
template <int NCOL>
__device__ __forceinline__ void store_row_bf16(uint32_t taddr, __nv_bfloat16* dst, float mul, bool valid) {
  float v[32];
#pragma unroll
  for (int c = 0; c < NCOL; c += 32) {
    tmem_ld32(taddr + c, v);
    tmem_ld_wait();
    if (valid) {
      uint4* o = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        uint4 pk;
        pk.x = pack_bf16(v[8 * k + 0] * mul, v[8 * k + 1] * mul);
        pk.y = pack_bf16(v[8 * k + 2] * mul, v[8 * k + 3] * mul);
        pk.z = pack_bf16(v[8 * k + 4] * mul, v[8 * k + 5] * mul);
        pk.w = pack_bf16(v[8 * k + 6] * mul, v[8 * k + 7] * mul);
        o[k] = pk;
      }
    }
  }
}

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

template <int D, int PS, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_bwd_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const __grid_constant__ CUtensorMap tmQ, Args a, const float* __restrict__ dsk,
                  const float* __restrict__ lse, const float* __restrict__ Dco_in, __nv_bfloat16* __restrict__ dK,
                  __nv_bfloat16* __restrict__ dV) {
  using C = BCfg<D, PS, MODE>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ws_failed(a.ws)) return;
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xB11u);
    return;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sG = sbase + C::OFF_G, sAB = sbase + C::OFF_AB, sRing = sbase + C::OFF_RING;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto ring_full = [&](int s) { return bar0 + 8u * s; };
  auto ring_empty = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  const uint32_t b1 = bar0 + 8u * (2 * C::NSLOT);
  const uint32_t q_full = b1, q_empty = b1 + 8, g_full = b1 + 16, g_empty = b1 + 24, s_full = b1 + 32,
                 sd_free_s = b1 + 40, da_full = b1 + 48, sd_free_da = b1 + 56, a_full = b1 + 64, dv_full = b1 + 72,
                 dv_empty = b1 + 80, ds_full = b1 + 88, ab_empty = b1 + 96, dk_empty = b1 + 104, dq_full = b1 + 112,
                 dq_empty = b1 + 120, drain = b1 + 128;
  // barriers of dsketch buffer gb
  auto g_full_of = [&](int gb) { return gb ? b1 + 136 : g_full; };
  auto g_empty_of = [&](int gb) { return gb ? b1 + 144 : g_empty; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);

  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = gridDim.x, wk = blockIdx.x, slice = blockIdx.y;
  const int p0 = slice * PS;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  const int ntiles = int(te - tb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(ring_full(s), 1);
      // V slots are released by the softmax warps once they have read v_i for D_i
      mbar_init(ring_empty(s), (MODE == kFull && (s & 1)) ? kSoftWarps : 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(g_full, 2);
    mbar_init(g_empty, 1);
    mbar_init(b1 + 136, 2);
    mbar_init(b1 + 144, 1);
    mbar_init(s_full, 1);
    mbar_init(sd_free_s, kSoftWarps);
    mbar_init(da_full, 1);
    mbar_init(sd_free_da, kSoftWarps);
    mbar_init(a_full, kSoftWarps);
    mbar_init(dv_full, 1);
    mbar_init(dv_empty, kSoftWarps);
    mbar_init(ds_full, kSoftWarps);
    mbar_init(ab_empty, 1);
    mbar_init(dk_empty, kSoftWarps);
    mbar_init(dq_full, 1);
    mbar_init(dq_empty, kSoftWarps);
    mbar_init(drain, 1);
    wait_ctl_init(abort_flag, a.ws);
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (ntiles > 0) {
    if (warp == 0 && lane == 0) {
      // ---------------------------------------------------------- TMA producer
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      TileWalker it(a, tb, te, T);
      int hc = 0, prev_h = -1;
      uint32_t e = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        if (it.qk != prev_h) {  // a new head (or, with per-user queries, a new user)
          if (hc > 0) ok = mbar_wait(q_empty, (hc - 1) & 1, abort_flag, a.ws, 0x401);
          if (!ok) break;
          mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(sQ + dh * PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
          prev_h = it.qk;
          ++hc;
        }
#pragma unroll
        for (int kv = 0; kv < 2; ++kv) {
          const int s = int(e % C::NSLOT);
          if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x402);
          if (!ok) break;
          mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh)
            tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, kv ? &tmV : &tmK, ring_full(s), 64 * dh, it.h,
                        int(it.tok0));
          ++e;
        }
        it.next();
      }
      if (!ok) {  // drain the ring loads and the prototype block still in flight
        for (uint32_t k = (e > uint32_t(C::NSLOT) ? e - C::NSLOT : 0); k < e; ++k)
          mbar_wait_bounded(ring_full(int(k % C::NSLOT)), (k / C::NSLOT) & 1, 200000000ull);
        if (hc > 0) mbar_wait_bounded(q_full, uint32_t(hc - 1) & 1u, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      // ---------------------------------------------------------- UMMA issuer
      constexpr uint32_t idSP = idesc_bf16(128, PS, 0, 0);      // [tok x P], K = d
      constexpr uint32_t idTD = idesc_bf16(128, D, 0, 1);       // [tok x d], K = prototypes
      constexpr uint32_t idQD = idesc_bf16(128, D, 1, 1);       // [proto x d], K = tokens
      TileWalker cur(a, tb, te, T), nxt(a, tb, te, T);
      nxt.next();
      int hc = 0, gc = 0, hp = 0, gbuf = 0;
      bool ok = true;
      auto wt = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return ok = ok && mbar_wait(bar, par, abort_flag, a.ws, site);
      };
      auto sdcol = [&](int i) { return uint32_t(C::SD_COL + (i % C::NSD) * PS); };
      // operand descriptors built once and stepped by constant offsets: each
      // instruction the issuing thread saves shortens the issue of a group (most
      // groups here are N = 64 or N = 128, a few dozen cycles of work per UMMA)
      const uint64_t dQk = sdesc(sQ, 16, 1024), dQm = sdesc(sQ, PS * 128, 1024);
      const uint64_t dABk = sdesc(sAB, 16, 1024), dABm = sdesc(sAB, T * 128, 1024);
      const uint64_t dRk = sdesc(sRing, 16, 1024), dRm = sdesc(sRing, T * 128, 1024);
      const uint64_t dGk = sdesc(sG, 16, 1024), dGm = sdesc(sG, PS * 128, 1024);
      // S(i) = K(i) Q^T into an S/dA buffer
      auto issue_S = [&](uint32_t kslot, uint32_t col) {
        const uint64_t dK = sdesc_add(dRk, kslot * C::KV_TILE);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          umma_ss(tmem + col, sdesc_add(dK, (k >> 2) * (T * 128) + (k & 3) * 32),
                  sdesc_add(dQk, (k >> 2) * (PS * 128) + (k & 3) * 32), idSP, k > 0 ? 1u : 0u);
      };
      TileWalker nx2(a, tb, te, T);
      nx2.next();
      nx2.next();
      wt(q_full, 0, 0x501);
      wt(ring_full(0), 0, 0x502);
      if (ok) {
        tc_fence_after();
        issue_S(0, sdcol(0));
        umma_commit(s_full);
        // slice mode: Q is read only by S, so it may be replaced after the last S of a head
        if (MODE == kSlice && (ntiles == 1 || nxt.qk != cur.qk)) umma_commit(q_empty);
      }
      bool first_of_hp = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        const uint32_t eK = 2u * li, eV = eK + 1;
        const int sK = int(eK % C::NSLOT), sV = int(eV % C::NSLOT);
        // ---- dA(i) = V(i) G^T
        if (cur.seg_first) {
          gbuf = gc % C::NG;
          wt(g_full_of(gbuf), uint32_t(gc / C::NG) & 1u, 0x503);
          ++gc;
        }
        wt(ring_full(sV), (eV / C::NSLOT) & 1, 0x504);
        wt(sd_free_s, li & 1, 0x505);
        if (!ok) break;
        tc_fence_after();
        const uint32_t gofs = uint32_t(gbuf * C::Q_BYTES);  // this segment's dsketch buffer
        {
          const uint64_t dVk = sdesc_add(dRk, uint32_t(sV) * C::KV_TILE), dG = sdesc_add(dGk, gofs);
#pragma unroll
          for (int k = 0; k < D / 16; ++k)
            umma_ss(tmem + sdcol(li), sdesc_add(dVk, (k >> 2) * (T * 128) + (k & 3) * 32),
                    sdesc_add(dG, (k >> 2) * (PS * 128) + (k & 3) * 32), idSP, k > 0 ? 1u : 0u);
        }
        umma_commit(da_full);
        if (MODE == kSlice) umma_commit(ring_empty(sV));
        // ---- dV(i) = A G
        if (MODE == kFull) {
          wt(a_full, li & 1, 0x506);
          if (li > 0) wt(dv_empty, (li - 1) & 1, 0x507);
          if (!ok) break;
          tc_fence_after();
          const uint64_t dG = sdesc_add(dGm, gofs);
#pragma unroll
          for (int k = 0; k < PS / 16; ++k)
            umma_ss(tmem + C::DV_COL, sdesc_add(dABk, (k >> 2) * (T * 128) + (k & 3) * 32), sdesc_add(dG, k * 2048),
                    idTD, k > 0 ? 1u : 0u);
          umma_commit(dv_full);
        }
        if (!ok) break;
        if (cur.seg_last) umma_commit(g_empty_of(gbuf));
        const bool more = li + 1 < ntiles;
        const bool newhead = more && nxt.qk != cur.qk;
        // ---- S(i+1) before dK/dQ(i) when its buffer and Q allow it
        const bool early = more && (C::NSD == 2 || !newhead);
        if (early) {
          if (C::NSD == 2) {
            if (newhead) {
              ++hc;
              wt(q_full, hc & 1, 0x508);
            }
            if (li >= 1) wt(sd_free_da, (li - 1) & 1, 0x509);
          } else {
            wt(sd_free_da, li & 1, 0x509);
          }
          wt(ring_full(int((eK + 2) % C::NSLOT)), ((eK + 2) / C::NSLOT) & 1, 0x50A);
          if (!ok) break;
          tc_fence_after();
          issue_S((eK + 2) % C::NSLOT, sdcol(li + 1));
          umma_commit(s_full);
          if (MODE == kSlice && (li + 2 >= ntiles || nx2.qk != nxt.qk)) umma_commit(q_empty);
        }
        // ---- dK(i) = dS Q, dQ += dS^T K
        wt(ds_full, li & 1, 0x50B);
        if (MODE == kFull && li > 0) wt(dk_empty, (li - 1) & 1, 0x50C);
        if (first_of_hp && hp > 0) wt(dq_empty, (hp - 1) & 1, 0x50D);
        if (!ok) break;
        tc_fence_after();
        if (MODE == kFull) {
#pragma unroll
          for (int k = 0; k < PS / 16; ++k)
            umma_ss(tmem + C::DK_COL, sdesc_add(dABk, (k >> 2) * (T * 128) + (k & 3) * 32), sdesc_add(dQm, k * 2048),
                    idTD, k > 0 ? 1u : 0u);
        }
        {
          const uint64_t dKm = sdesc_add(dRm, uint32_t(sK) * C::KV_TILE);
#pragma unroll
          for (int k = 0; k < T / 16; ++k)
#pragma unroll
            for (int mb = 0; mb < PS / 128; ++mb)
              umma_ss(tmem + C::DQ_COL + mb * D, sdesc_add(dABm, mb * 2 * (T * 128) + k * 2048),
                      sdesc_add(dKm, k * 2048), idQD, (first_of_hp && k == 0) ? 0u : 1u);
        }
        umma_commit(ab_empty);
        umma_commit(ring_empty(sK));
        const bool last_of_hp = !more || newhead;
        if (last_of_hp) {
          umma_commit(dq_full);
          if (MODE == kFull) umma_commit(q_empty);  // dK read Q up to here
          ++hp;
        }
        first_of_hp = last_of_hp;
        // ---- S(i+1) after a head change in full mode (Q replaced once dK(i) is done)
        if (more && !early) {
          ++hc;
          wt(q_full, hc & 1, 0x50E);
          wt(sd_free_da, li & 1, 0x50F);
          wt(ring_full(int((eK + 2) % C::NSLOT)), ((eK + 2) / C::NSLOT) & 1, 0x510);
          if (!ok) break;
          tc_fence_after();
          issue_S((eK + 2) % C::NSLOT, sdcol(li + 1));
          umma_commit(s_full);
        }
        cur.next();
        nxt.next();
        nx2.next();
      }
      umma_commit(drain);
      mbar_wait_bounded(drain, 0, 200000000ull);
    } else if (warp == 2 || warp == 3) {
      // ------------------------------------ dsketch rows -> bf16, swizzled [d/64][PS][64]
      const int t64 = threadIdx.x - 64;  // 0..63
      TileWalker cur(a, tb, te, T);
      int gc = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        if (cur.seg_first) {
          const int gb = gc % C::NG;
          if (gc >= C::NG)
            ok = __all_sync(0xffffffffu, mbar_wait(g_empty_of(gb), uint32_t((gc / C::NG) - 1) & 1u, abort_flag,
                                                   a.ws, 0x601));
          if (!ok) break;
          const float* src = dsk + ((int64_t(cur.b) * a.H + cur.h) * a.P + p0) * D;
          uint8_t* gdst = smem + C::OFF_G + gb * C::Q_BYTES;
          constexpr int CHUNKS = PS * D / 8;
#pragma unroll 8
          for (int c = t64; c < CHUNKS; c += 64) {
            const int p = c / (D / 8), dd = (c % (D / 8)) * 8;
            const float4 x = *reinterpret_cast<const float4*>(src + int64_t(p) * D + dd);
            const float4 y = *reinterpret_cast<const float4*>(src + int64_t(p) * D + dd + 4);
            uint4 pk;
            pk.x = pack_bf16(x.x, x.y);
            pk.y = pack_bf16(x.z, x.w);
            pk.z = pack_bf16(y.x, y.y);
            pk.w = pack_bf16(y.z, y.w);
            const int dh = dd >> 6, chunk = (dd & 63) >> 3;
            *reinterpret_cast<uint4*>(gdst + dh * PS * 128 + p * 128 + ((chunk ^ (p & 7)) << 4)) = pk;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(g_full_of(gb));
          ++gc;
        }
        cur.next();
      }
    } else if (warp >= kSoftWarp0) {
      // ------------------------------------------------ softmax + epilogue
      const int sw = (warp - kSoftWarp0) >> 2, q = warp & 3, row = 32 * q + lane;
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * 1.4426950408889634f;
      TileWalker cur(a, tb, te, T), prev(a, tb, te, T);
      bool ok = true;
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      int hp = 0;
      // dK of the previous tile and, at the end of a head piece, dQ
      auto finish_prev = [&](const TileWalker& pw, bool last_of_hp) {
        if (MODE == kFull) {
          __nv_bfloat16* dst = dK + ((pw.tok0 + row) * a.H + pw.h) * int64_t(D) + sw * (D / 2);
          store_row_bf16<D / 2>(tmem + lane_off + C::DK_COL + sw * (D / 2), dst, a.scale, row < pw.n);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(dk_empty);
        }
        if (last_of_hp) {
          float* dst = dq_block_dst(a, wk, W, total, pw, p0, D);
          store_sketch_scaled<D, PS, C::DQ_COL>(tmem, lane_off, sw, q, lane, dst, a.scale);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(dq_empty);
          ++hp;
        }
      };
      uint32_t apk[C::HALF / 2];  // this thread's A values, bf16 pairs
      // per-token lse (and D_i in slice mode), loaded one tile ahead
      float lse_cur = row < cur.n ? lse[(cur.tok0 + row) * a.H + cur.h] : 0.f;
      float d_cur = (MODE == kSlice && row < cur.n) ? Dco_in[(cur.tok0 + row) * a.H + cur.h] : 0.f;
      for (int li = 0; li < ntiles && ok; ++li) {
        const bool valid = row < cur.n;
        const int64_t tok = cur.tok0 + row;
        const uint32_t eV = 2u * li + 1;
        const int sV = int(eV % C::NSLOT);
        const uint32_t sdc = C::SD_COL + (li % C::NSD) * PS;
        float lse_nxt, d_nxt = 0.f;
        {
          int64_t t0n;
          int nn, hn;
          cur.peek_next(t0n, nn, hn);
          lse_nxt = row < nn ? lse[(t0n + row) * a.H + hn] : 0.f;
          if (MODE == kSlice) d_nxt = row < nn ? Dco_in[(t0n + row) * a.H + hn] : 0.f;
        }
        // ---- A = exp(scale S - lse)
        ok = wwait(s_full, li & 1, 0x701);
        if (!ok) break;
        tc_fence_after();
        {
          const float L2 = lse_cur * 1.4426950408889634f;
          float v[32];
#pragma unroll
          for (int c = 0; c < C::HALF / 32; ++c) {
            tmem_ld32(tmem + lane_off + sdc + sw * C::HALF + 32 * c, v);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float x0 = valid ? ex2(fmaf(v[2 * j], c2, -L2)) : 0.f;
              const float x1 = valid ? ex2(fmaf(v[2 * j + 1], c2, -L2)) : 0.f;
              apk[16 * c + j] = pack_bf16(x0, x1);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(sd_free_s);
        // ---- previous tile's dK / dQ (their MMAs also release the AB buffer)
        if (li > 0) {
          ok = wwait(ab_empty, (li - 1) & 1, 0x702);
          if (!ok) break;
          tc_fence_after();
          finish_prev(prev, prev.qk != cur.qk);
          prev.next();
        }
        // ---- A -> shared memory [PS/64][128 tokens][64], 128-byte swizzle
        if (MODE == kFull) {
          uint8_t* rowp = smem + C::OFF_AB + row * 128;
#pragma unroll
          for (int k = 0; k < C::HALF / 8; ++k) {
            const int p = sw * C::HALF + 8 * k;
            const int blk = p >> 6, chunk = (p & 63) >> 3;
            *reinterpret_cast<uint4*>(rowp + blk * (T * 128) + ((chunk ^ (row & 7)) << 4)) =
                make_uint4(apk[4 * k], apk[4 * k + 1], apk[4 * k + 2], apk[4 * k + 3]);
          }
        }
        if (MODE == kFull) {
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(a_full);
        }
        // ---- D_i
        float Dv = 0.f;
        if (MODE == kFull) {
          ok = wwait(dv_full, li & 1, 0x703);
          if (!ok) break;
          tc_fence_after();
          const uint8_t* vrow = smem + C::OFF_RING + sV * C::KV_TILE + row * 128;
          float v[32];
#pragma unroll
          for (int c = 0; c < D; c += 32) {
            tmem_ld32(tmem + lane_off + C::DV_COL + c, v);
            tmem_ld_wait();
            const int dh = c >> 6;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const int chunk = ((c & 63) >> 3) + k;
              const uint4 w = *reinterpret_cast<const uint4*>(vrow + dh * (T * 128) + ((chunk ^ (row & 7)) << 4));
              Dv = fmaf(v[8 * k + 0], bf16lo(w.x), Dv);
              Dv = fmaf(v[8 * k + 1], bf16hi(w.x), Dv);
              Dv = fmaf(v[8 * k + 2], bf16lo(w.y), Dv);
              Dv = fmaf(v[8 * k + 3], bf16hi(w.y), Dv);
              Dv = fmaf(v[8 * k + 4], bf16lo(w.z), Dv);
              Dv = fmaf(v[8 * k + 5], bf16hi(w.z), Dv);
              Dv = fmaf(v[8 * k + 6], bf16lo(w.w), Dv);
              Dv = fmaf(v[8 * k + 7], bf16hi(w.w), Dv);
            }
          }
          // dV rows of this tile
          __nv_bfloat16* dst = dV + (tok * a.H + cur.h) * int64_t(D) + sw * (D / 2);
          store_row_bf16<D / 2>(tmem + lane_off + C::DV_COL + sw * (D / 2), dst, 1.f, valid);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(dv_empty);
            mbar_arrive(ring_empty(sV));
          }
        } else {
          Dv = d_cur;
        }
        // ---- dS = A o (dA - D) -> shared memory (over A, whose readers are done)
        ok = wwait(da_full, li & 1, 0x704);
        if (!ok) break;
        tc_fence_after();
        {
          uint8_t* rowp = smem + C::OFF_AB + row * 128;
          float v[32];
#pragma unroll
          for (int c = 0; c < C::HALF / 32; ++c) {
            tmem_ld32(tmem + lane_off + sdc + sw * C::HALF + 32 * c, v);
            tmem_ld_wait();
            uint32_t o[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const uint32_t w = apk[16 * c + j];
              o[j] = pack_bf16(bf16lo(w) * (v[2 * j] - Dv), bf16hi(w) * (v[2 * j + 1] - Dv));
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const int p = sw * C::HALF + 32 * c + 8 * k;
              const int blk = p >> 6, chunk = (p & 63) >> 3;
              *reinterpret_cast<uint4*>(rowp + blk * (T * 128) + ((chunk ^ (row & 7)) << 4)) =
                  make_uint4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
            }
          }
        }
        tc_fence_before();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(sd_free_da);
          mbar_arrive(ds_full);
        }
        lse_cur = lse_nxt;
        d_cur = d_nxt;
        cur.next();
      }
      if (ok) {
        ok = wwait(ab_empty, (ntiles - 1) & 1, 0x705);
        if (ok) {
          tc_fence_after();
          finish_prev(prev, true);
        }
      }
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, int PS, int MODE>
static cudaError_t launch_bwd_t(const Args& a, int W, const float* dsk, const float* lse, const float* Dco, void* dK,
                                void* dV, cudaStream_t st) {
  using C = BCfg<D, PS, MODE>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, PS))
    return cudaErrorInvalidValue;
  auto fn = &tc_bwd_kernel<D, PS, MODE>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid(W, a.P / PS);
  fn<<<grid, kThreads, C::SMEM, st>>>(tk, tv, tq, a, dsk, lse, Dco, static_cast<__nv_bfloat16*>(dK),
                                      static_cast<__nv_bfloat16*>(dV));
  return cudaGetLastError();
}

}  // namespace tcb

// Tensor-core backward: bf16, all prototypes in one CTA when the four TMEM
// accumulators fit (d = 64 with P <= 256, d = 128 with P = 128), else the
// token-side kernel plus the dQ slices (tc_bwd_split).
bool tc_bwd_supported(int P, int d, sa_dtype dt) {
  if (dt != SA_BF16 || !tcc::device_is_sm103() || !tc_path_enabled()) return false;
  return ((d == 64 || d == 128) && (P == 128 || P == 256 || P == 512 || P == 1024 || P == 2048));
}

const char* tc_bwd_name(int P, int d) {
  if (d == 64 && P == 2048) return "tc_bwd_tok_kernel<64,2048>";
  if (d == 64 && P == 1024) return "tc_bwd_tok_kernel<64,1024>";
  if (d == 64 && P == 512) return "tc_bwd_tok_kernel<64,512>";
  if (d == 64) return P == 256 ? "tc_bwd_kernel<64,256,full>" : "tc_bwd_kernel<64,128,full>";
  if (P == 2048) return "tc_bwd_tok_kernel<128,2048>";
  if (P == 1024) return "tc_bwd_tok_kernel<128,1024>";
  if (P == 512) return "tc_bwd_tok_kernel<128,512>";
  if (P == 256) return "tc_bwd_tok_kernel<128,256>";
  return "tc_bwd_kernel<128,128,full>";
}

int tc_bwd_workers(int num_sms, int, int) { return num_sms; }

cudaError_t launch_tc_bwd(const Args& a, int W, const float* dsk, const float* lse, void* dK, void* dV,
                          cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  using namespace tcb;
  if (a.d == 64) {
    if (a.P == 256) return launch_bwd_t<64, 256, kFull>(a, W, dsk, lse, nullptr, dK, dV, st);
    if (a.P == 128) return launch_bwd_t<64, 128, kFull>(a, W, dsk, lse, nullptr, dK, dV, st);
  } else if (a.P == 128) {
    return launch_bwd_t<128, 128, kFull>(a, W, dsk, lse, nullptr, dK, dV, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sa

// ===================================================================== tokens
// Token side of the backward for shapes whose prototypes do not fit one CTA
// (d = 128 with P > 128): all P prototypes pass through the CTA in chunks of
// NC = 128 (Q and a bf16 copy of dsketch streamed by TMA), in one pass:
//   dV_i   = sum_j A[j,i] G_j                   (UMMA, accumulates over chunks)
//   u_i    = sum_j A[j,i] dA[j,i] Q_j            (UMMA on E = A o dA)
//   qbar_i = sum_j A[j,i] Q_j                    (UMMA)
//   D_i    = sum_j A[j,i] dA[j,i]                (registers)
//   dK_i   = scale (u_i - D_i qbar_i)            (= scale sum_j dS[j,i] Q_j)
// and D_i is written out for the prototype-side dQ kernel (kSlice mode above).
namespace sa {
namespace tcb {

template <int D, int P>
struct TokCfg {
  static constexpr int NC = 128;
  static constexpr int NCH = P / NC;
  static constexpr int SLOT = T * D * 2;  // one K, V, Q-chunk or G-chunk tile (NC == T)
  static constexpr int NSLOT = 6;         // three pairs: (K, V) of a tile or (G, Q) of a chunk
  static constexpr int OFF_SLOTS = 0;
  static constexpr int OFF_AB = NSLOT * SLOT;  // A, then E = A o dA, of one chunk; epilogue staging
  static constexpr int OFF_STATS = OFF_AB + T * NC * 2;
  static constexpr int OFF_BAR = OFF_STATS + 2 * T * 4;
  static constexpr int NBAR = 2 * NSLOT + 20;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = OFF_MISC + 16;
  // dV and qbar side by side: one N = 2D MMA against the adjacent G, Q chunks
  static constexpr int SD_COL = 0, DV_COL = NC, QB_COL = NC + D, U_COL = NC + 2 * D;
  static constexpr int TMEM_COLS = tmem_cols_for(NC + 3 * D);
  static constexpr int HALF = NC / 2;
  static_assert(NC == T && TMEM_COLS <= 512 && SMEM <= 232448, "budget");
};

// Where dA lands: with prototype-wise weights S and dA share SD_COL (TMEM is
// full); token-wise needs no qbar, so dA takes QB_COL and the two do not wait
// for each other.
template <int D, int P, bool TW>
__host__ __device__ constexpr int tok_da_col() {
  return TW ? TokCfg<D, P>::QB_COL : TokCfg<D, P>::SD_COL;
}

// Pair 0 holds the tile's K and V; the next tile's K loads into it once the
// tile's last S has read K, its V once the last dA has read V, and both tiles
// are pulled into L2 a tile ahead.  Chunks alternate between pairs 1 and 2
// (the chunk count per tile is even).  A chunk pair holds G in its first slot
// and Q in the second, so the four 64-column blocks of G and Q sit at one
// stride and [G | Q] is a single N = 2D operand.
__device__ __forceinline__ int tok_kv_pair(int) { return 0; }
__device__ __forceinline__ int tok_qg_pair(int, int c) { return 1 + (c & 1); }

// TW = false: prototype-wise weights (Sec. 3.1), lse and Dco per token [N][H]
// (Dco written here).  TW = true: token-wise weights (Sec. 5.1), lse and Dco
// per prototype [B][H][P] (both read), so dS = A o (dA - D_j) goes to shared
// memory in place of E and dK = scale dS Q needs no qbar.
template <int D, int P, bool TW>
__device__ __forceinline__ void bwd_tok_body(const CUtensorMap& tmK, const CUtensorMap& tmV, const CUtensorMap& tmQ,
                                             const CUtensorMap& tmG, const CUtensorMap& tmDK,
                                             const CUtensorMap& tmDV, const Args& a, const float* __restrict__ lse,
                                             float* __restrict__ Dco, __nv_bfloat16* __restrict__ dK,
                                             __nv_bfloat16* __restrict__ dV) {
  using C = TokCfg<D, P>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ws_failed(a.ws)) return;
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xB21u);
    return;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sSlots = sbase + C::OFF_SLOTS, sAB = sbase + C::OFF_AB;
  auto slot_addr = [&](int s) { return sSlots + uint32_t(s) * C::SLOT; };
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  const uint32_t b1 = bar0 + 8u * (2 * C::NSLOT);
  const uint32_t s_full = b1, sd_free_s = b1 + 8, da_full = b1 + 16, sd_free_da = b1 + 24, a_full = b1 + 32,
                 ab_free_a = b1 + 40, e_full = b1 + 48, ab_free_e = b1 + 56, acc_full = b1 + 64,
                 acc_empty = b1 + 72, st_ready = b1 + 80, st_used = b1 + 88, epi_ready = b1 + 96, epi_free = b1 + 104,
                 drain = b1 + 112;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = gridDim.x, wk = blockIdx.x;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  const int ntiles = int(te - tb);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(s_full, 1);
    mbar_init(sd_free_s, kSoftWarps);
    mbar_init(da_full, 1);
    mbar_init(sd_free_da, kSoftWarps);
    mbar_init(a_full, kSoftWarps);
    mbar_init(ab_free_a, 1);
    mbar_init(e_full, kSoftWarps);
    mbar_init(ab_free_e, 1);
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, kSoftWarps);
    mbar_init(st_ready, kSoftWarps);
    mbar_init(st_used, kSoftWarps);
    mbar_init(epi_ready, kSoftWarps);
    mbar_init(epi_free, 1);
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
  // softmax warpgroups (128 x 152 + 256 x 176 = 384 x 168, the launch allocation).
  if (ntiles > 0 && warp < kSoftWarp0) {
    setmaxnreg_dec<152>();
    if (warp == 0 && lane == 0) {
      // ---------------------------------------------------------- TMA producer
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmG);
      TileWalker it(a, tb, te, T), nx(a, tb, te, T);
      nx.next();
      static_assert(C::NCH % 2 == 0, "chunks alternate between two pairs");
      // per slot, as bits (registers, not an indexed array): loaded before, and
      // the parity of the wait for its next release
      uint32_t used = 0u, par = 0u;
      bool ok = true;
      // box origin (64*dh, c1, c2): K / V maps are (d, head, token); Q / G maps
      // are (d, prototype, head) and (d, prototype, user*H + head)
      auto load = [&](int s, const CUtensorMap* map, int c1, int c2) {
        if ((used >> s) & 1u) {
          ok = ok && mbar_wait(empty_bar(s), (par >> s) & 1u, abort_flag, a.ws, 0x801);
          par ^= 1u << s;
        }
        if (!ok) return;
        used |= 1u << s;
        mbar_arrive_expect_tx(full_bar(s), C::SLOT);
#pragma unroll
        for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(slot_addr(s) + dh * T * 128, map, full_bar(s), 64 * dh, c1, c2);
      };
      auto prefetch_kv = [&](const TileWalker& w) {
#pragma unroll
        for (int dh = 0; dh < D / 64; ++dh) {
          tma_prefetch_l2_3d(&tmK, 64 * dh, w.h, int(w.tok0));
          tma_prefetch_l2_3d(&tmV, 64 * dh, w.h, int(w.tok0));
        }
      };
      // Order of loads: ..., Q/G(li, last), K(li+1), Q/G(li+1, 0), V(li+1), ...:
      // K(li+1) waits for S(li, last), V(li+1) for dA(li, last).
      load(0, &tmK, it.h, int(it.tok0));
      load(1, &tmV, it.h, int(it.tok0));
      if (ntiles > 1) prefetch_kv(nx);
      for (int li = 0; li < ntiles && ok; ++li) {
        for (int c = 0; c < C::NCH && ok; ++c) {
          const int pr = tok_qg_pair(li, c);
          load(2 * pr + 1, &tmQ, c * C::NC, it.qk);
          load(2 * pr, &tmG, c * C::NC, int(it.b) * a.H + it.h);
          if (c == 0 && li > 0) load(1, &tmV, it.h, int(it.tok0));
          if (c == C::NCH - 1 && li + 1 < ntiles) load(0, &tmK, nx.h, int(nx.tok0));
        }
        it.next();
        nx.next();
        if (li + 2 < ntiles) prefetch_kv(nx);
      }
      if (!ok) {
        for (int s = 0; s < C::NSLOT; ++s)
          if ((used >> s) & 1u) mbar_wait_bounded(full_bar(s), (par >> s) & 1u, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      // ---------------------------------------------------------- UMMA issuer
      // Per chunk g: dA_g, [dV | qbar]_g, S_{g+1}, u_g.  Shared-memory
      // descriptors are built once per operand and stepped by constant offsets,
      // so the issue loop carries no address arithmetic.
      constexpr uint32_t idS = idesc_bf16(128, C::NC, 0, 0);    // [tok x chunk], K = d
      constexpr uint32_t idGQ = idesc_bf16(128, TW ? D : 2 * D, 0, 1);  // [tok x (d | d)] (TW: d), K = chunk
      constexpr uint32_t idU = idesc_bf16(128, D, 0, 1);        // [tok x d], K = chunk prototypes
      bool ok = true;
      uint32_t fpar = 0u;  // per slot, as bits: parity of the next "full" phase
      auto wt = [&](uint32_t bar, uint32_t parity, uint32_t site) {
        return ok = ok && mbar_wait(bar, parity, abort_flag, a.ws, site);
      };
      auto wfull = [&](int s, uint32_t site) {
        wt(full_bar(s), (fpar >> s) & 1u, site);
        fpar ^= 1u << s;
      };
      // K-major [128 rows x D] operand: K step k at +(k / 4) * 128 rows + (k % 4) * 32 B
      auto kmaj = [](uint32_t addr) { return sdesc(addr, 16, 1024); };
      auto kstep = [](int k) { return uint32_t((k >> 2) * (T * 128) + (k & 3) * 32); };
      const uint64_t dAB = kmaj(sAB);
      const uint32_t nchunks = uint32_t(ntiles) * C::NCH;
      auto issue_S = [&](uint32_t g) {
        const int li = int(g / C::NCH), c = int(g % C::NCH);
        const uint64_t dK = kmaj(slot_addr(2 * tok_kv_pair(li))), dQ = kmaj(slot_addr(2 * tok_qg_pair(li, c) + 1));
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          umma_ss(tmem + C::SD_COL, sdesc_add(dK, kstep(k)), sdesc_add(dQ, kstep(k)), idS, k > 0 ? 1u : 0u);
        umma_commit(s_full);
        if (c == C::NCH - 1) umma_commit(empty_bar(2 * tok_kv_pair(li)));  // last S: K free
      };
      wfull(2 * tok_kv_pair(0), 0x901);
      wfull(2 * tok_qg_pair(0, 0) + 1, 0x902);
      if (ok) {
        tc_fence_after();
        issue_S(0);
      }
      for (uint32_t g = 0; g < nchunks && ok; ++g) {
        const int li = int(g / C::NCH), c = int(g % C::NCH);
        const int kvp = tok_kv_pair(li), qgp = tok_qg_pair(li, c);
        const uint32_t aG = slot_addr(2 * qgp), aQ = slot_addr(2 * qgp + 1);
        // ---- dA_g = V G_g^T (into S's columns once S_g is read, or, token-wise,
        // into its own columns once dA_{g-1} is read)
        if (c == 0) wfull(2 * kvp + 1, 0x903);
        wfull(2 * qgp, 0x904);
        if (!TW) wt(sd_free_s, g & 1, 0x905);
        else if (g > 0) wt(sd_free_da, (g - 1) & 1, 0x905);
        if (!ok) break;
        tc_fence_after();
        {
          const uint64_t dV = kmaj(slot_addr(2 * kvp + 1)), dG = kmaj(aG);
#pragma unroll
          for (int k = 0; k < D / 16; ++k)
            umma_ss(tmem + tok_da_col<D, P, TW>(), sdesc_add(dV, kstep(k)), sdesc_add(dG, kstep(k)), idS,
                    k > 0 ? 1u : 0u);
        }
        umma_commit(da_full);
        if (c == C::NCH - 1) umma_commit(empty_bar(2 * kvp + 1));  // last dA: V free
        // ---- [dV | qbar] += A [G_g | Q_g]
        wt(a_full, g & 1, 0x906);
        if (c == 0 && li > 0) wt(acc_empty, (li - 1) & 1, 0x907);
        if (!ok) break;
        tc_fence_after();
        {
          const uint64_t dGQ = sdesc(aG, C::NC * 128, 1024);  // MN-major, 64-column blocks 16 KB apart
#pragma unroll
          for (int k = 0; k < C::NC / 16; ++k)
            umma_ss(tmem + C::DV_COL, sdesc_add(dAB, kstep(k)), sdesc_add(dGQ, k * 2048), idGQ,
                    (c == 0 && k == 0) ? 0u : 1u);
        }
        umma_commit(ab_free_a);
        umma_commit(empty_bar(2 * qgp));  // G chunk free
        // ---- S_{g+1}
        if (g + 1 < nchunks) {
          const uint32_t gn = g + 1;
          const int lin = int(gn / C::NCH), cn = int(gn % C::NCH);
          if (cn == 0) wfull(2 * tok_kv_pair(lin), 0x908);
          wfull(2 * tok_qg_pair(lin, cn) + 1, 0x909);
          wt(TW ? sd_free_s : sd_free_da, g & 1, 0x90A);  // S's columns read
          if (!ok) break;
          tc_fence_after();
          issue_S(gn);
        }
        // ---- u += E Q_g
        wt(e_full, g & 1, 0x90B);
        if (!ok) break;
        tc_fence_after();
        {
          const uint64_t dQm = sdesc(aQ, C::NC * 128, 1024);
#pragma unroll
          for (int k = 0; k < C::NC / 16; ++k)
            umma_ss(tmem + C::U_COL, sdesc_add(dAB, kstep(k)), sdesc_add(dQm, k * 2048), idU,
                    (c == 0 && k == 0) ? 0u : 1u);
        }
        umma_commit(ab_free_e);
        umma_commit(empty_bar(2 * qgp + 1));  // Q chunk free
        if (c == C::NCH - 1) umma_commit(acc_full);
      }
      umma_commit(drain);
      mbar_wait_bounded(drain, 0, 200000000ull);
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<176>();
    {
      // ------------------------------------------------ softmax + epilogue
      const int sw = (warp - kSoftWarp0) >> 2, q = warp & 3, row = 32 * q + lane;
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * 1.4426950408889634f;
      float* stats = reinterpret_cast<float*>(smem + C::OFF_STATS);
      TileWalker cur(a, tb, te, T);
      bool ok = true;
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      uint32_t g = 0;
      int epi = 0;  // staged epilogue stores so far
      auto put_tile = [&](const uint32_t* pk) {
        uint8_t* rowp = smem + C::OFF_AB + row * 128;
#pragma unroll
        for (int k = 0; k < C::HALF / 8; ++k) {
          const int p = sw * C::HALF + 8 * k;
          const int blk = p >> 6, chunk = (p & 63) >> 3;
          *reinterpret_cast<uint4*>(rowp + blk * (T * 128) + ((chunk ^ (row & 7)) << 4)) =
              make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]);
        }
      };
      // one staged [128 tokens][D] bf16 tile in AB -> global through TMA
      auto stage_and_store = [&](const CUtensorMap* map, const TileWalker& w) -> bool {
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(epi_ready);
        if (warp == kSoftWarp0 && lane == 0) {
          if (mbar_wait(epi_ready, epi & 1, abort_flag, a.ws, 0xA08)) {
#pragma unroll
            for (int dh = 0; dh < D / 64; ++dh) tma_store_3d(map, sAB + dh * T * 128, 64 * dh, w.h, int(w.tok0));
            bulk_commit_group();
            bulk_wait_read_all();
          }
          mbar_arrive(epi_free);
        }
        const bool r = wwait(epi_free, epi & 1, 0xA09);
        ++epi;
        return r;
      };
      float lse_cur = (!TW && row < cur.n) ? lse[(cur.tok0 + row) * a.H + cur.h] : 0.f;
      for (int li = 0; li < ntiles && ok; ++li) {
        const bool valid = row < cur.n;
        const int64_t tok = cur.tok0 + row;
        const float L2 = lse_cur * 1.4426950408889634f;
        if (!TW) {
          int64_t t0n;
          int nn, hn;
          cur.peek_next(t0n, nn, hn);
          lse_cur = row < nn ? lse[(t0n + row) * a.H + hn] : 0.f;
        }
        // token-wise: this segment's per-prototype lse and D_j (the same for
        // every thread: broadcast loads)
        const int64_t seg_row = (int64_t(cur.b) * a.H + cur.h) * a.P;
        float Dp = 0.f;
        for (int c = 0; c < C::NCH && ok; ++c, ++g) {
          uint32_t apk[C::HALF / 2];
          float v[C::HALF];  // this warpgroup's columns of S, then of dA (both loads before one wait)
          const int j0 = c * C::NC + sw * C::HALF;  // first prototype of this warpgroup's columns
          ok = wwait(s_full, g & 1, 0xA01);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < C::HALF / 32; ++cc) tmem_ld32(tmem + lane_off + C::SD_COL + sw * C::HALF + 32 * cc, v + 32 * cc);
          tmem_ld_wait();
          // S is in registers: its columns may take dA_g (or S_{g+1}) while the weights are formed
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sd_free_s);
#pragma unroll
          for (int cc = 0; cc < C::HALF / 32; ++cc) {
            if (TW) {
              const float4* l4 = reinterpret_cast<const float4*>(lse + seg_row + j0 + 32 * cc);
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                const float4 l = __ldg(l4 + j4);
                const float x0 = valid ? ex2(fmaf(v[32 * cc + 4 * j4 + 0], c2, -l.x * 1.4426950408889634f)) : 0.f;
                const float x1 = valid ? ex2(fmaf(v[32 * cc + 4 * j4 + 1], c2, -l.y * 1.4426950408889634f)) : 0.f;
                const float x2 = valid ? ex2(fmaf(v[32 * cc + 4 * j4 + 2], c2, -l.z * 1.4426950408889634f)) : 0.f;
                const float x3 = valid ? ex2(fmaf(v[32 * cc + 4 * j4 + 3], c2, -l.w * 1.4426950408889634f)) : 0.f;
                apk[16 * cc + 2 * j4] = pack_bf16(x0, x1);
                apk[16 * cc + 2 * j4 + 1] = pack_bf16(x2, x3);
              }
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float x0 = valid ? ex2(fmaf(v[32 * cc + 2 * j], c2, -L2)) : 0.f;
                const float x1 = valid ? ex2(fmaf(v[32 * cc + 2 * j + 1], c2, -L2)) : 0.f;
                apk[16 * cc + j] = pack_bf16(x0, x1);
              }
            }
          }
          if (g > 0) {
            ok = wwait(ab_free_e, (g - 1) & 1, 0xA02);  // u of the previous chunk has read E
            if (!ok) break;
          }
          put_tile(apk);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(a_full);
          // E = A o dA (token-wise: dS = A o (dA - D_j))
          ok = wwait(da_full, g & 1, 0xA03);
          if (!ok) break;
          tc_fence_after();
          uint32_t epk[C::HALF / 2];
#pragma unroll
          for (int cc = 0; cc < C::HALF / 32; ++cc)
            tmem_ld32(tmem + lane_off + tok_da_col<D, P, TW>() + sw * C::HALF + 32 * cc, v + 32 * cc);
          tmem_ld_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sd_free_da);
#pragma unroll
          for (int cc = 0; cc < C::HALF / 32; ++cc) {
            if (TW) {
              const float4* d4 = reinterpret_cast<const float4*>(Dco + seg_row + j0 + 32 * cc);
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                const float4 dd = __ldg(d4 + j4);
                const uint32_t w0 = apk[16 * cc + 2 * j4], w1 = apk[16 * cc + 2 * j4 + 1];
                epk[16 * cc + 2 * j4] = pack_bf16(bf16lo(w0) * (v[32 * cc + 4 * j4 + 0] - dd.x),
                                                  bf16hi(w0) * (v[32 * cc + 4 * j4 + 1] - dd.y));
                epk[16 * cc + 2 * j4 + 1] = pack_bf16(bf16lo(w1) * (v[32 * cc + 4 * j4 + 2] - dd.z),
                                                      bf16hi(w1) * (v[32 * cc + 4 * j4 + 3] - dd.w));
              }
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const uint32_t w = apk[16 * cc + j];
                const float e0 = bf16lo(w) * v[32 * cc + 2 * j], e1 = bf16hi(w) * v[32 * cc + 2 * j + 1];
                Dp += e0 + e1;
                epk[16 * cc + j] = pack_bf16(e0, e1);
              }
            }
          }
          ok = wwait(ab_free_a, g & 1, 0xA04);  // dV and qbar have read A
          if (!ok) break;
          put_tile(epk);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(e_full);
        }
        if (!ok) break;
        // D_i = (half from warpgroup 0) + (half from warpgroup 1), same order in
        // both; token-wise: u already is sum_j dS[j,i] Q_j, so D_i = 0 below
        float Dv = 0.f;
        if (!TW) {
          if (li > 0) {
            ok = wwait(st_used, (li - 1) & 1, 0xA05);
            if (!ok) break;
          }
          stats[sw * T + row] = Dp;
          __syncwarp();
          if (lane == 0) mbar_arrive(st_ready);
          ok = wwait(st_ready, li & 1, 0xA06);
          if (!ok) break;
          Dv = stats[row] + stats[T + row];
          __syncwarp();
          if (lane == 0) mbar_arrive(st_used);
          if (sw == 0 && valid) Dco[tok * a.H + cur.h] = Dv;
        }
        // epilogue: dV and dK = scale (u - D qbar); this warpgroup owns columns [sw*D/2, +D/2)
        ok = wwait(acc_full, li & 1, 0xA07);
        if (!ok) break;
        tc_fence_after();
        const bool whole = cur.n == T;  // a full tile is stored by TMA; a ragged tail row by row
        uint8_t* rowp = smem + C::OFF_AB + row * 128;
        auto put_half = [&](const float* x, int cc) {  // 32 columns [sw*D/2 + cc, +32) of this row
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int col = sw * (D / 2) + cc + 8 * k;
            const int dh = col >> 6, chunk = (col & 63) >> 3;
            *reinterpret_cast<uint4*>(rowp + dh * (T * 128) + ((chunk ^ (row & 7)) << 4)) =
                make_uint4(pack_bf16(x[8 * k], x[8 * k + 1]), pack_bf16(x[8 * k + 2], x[8 * k + 3]),
                           pack_bf16(x[8 * k + 4], x[8 * k + 5]), pack_bf16(x[8 * k + 6], x[8 * k + 7]));
          }
        };
        if (whole) {
          float x[32];
#pragma unroll
          for (int cc = 0; cc < D / 2; cc += 32) {
            tmem_ld32(tmem + lane_off + C::DV_COL + sw * (D / 2) + cc, x);
            tmem_ld_wait();
            put_half(x, cc);
          }
          ok = stage_and_store(&tmDV, cur);
          if (!ok) break;
          float uu[32], qb[32];
#pragma unroll
          for (int cc = 0; cc < D / 2; cc += 32) {
            tmem_ld32(tmem + lane_off + C::U_COL + sw * (D / 2) + cc, uu);
            if (!TW) tmem_ld32(tmem + lane_off + C::QB_COL + sw * (D / 2) + cc, qb);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 32; ++j) uu[j] = TW ? a.scale * uu[j] : a.scale * fmaf(-Dv, qb[j], uu[j]);
            put_half(uu, cc);
          }
          ok = stage_and_store(&tmDK, cur);
          if (!ok) break;
        } else {
          __nv_bfloat16* dvr = dV + (tok * a.H + cur.h) * int64_t(D) + sw * (D / 2);
          store_row_bf16<D / 2>(tmem + lane_off + C::DV_COL + sw * (D / 2), dvr, 1.f, valid);
          __nv_bfloat16* dkr = dK + (tok * a.H + cur.h) * int64_t(D) + sw * (D / 2);
          float uu[32], qb[32];
#pragma unroll
          for (int cc = 0; cc < D / 2; cc += 32) {
            tmem_ld32(tmem + lane_off + C::U_COL + sw * (D / 2) + cc, uu);
            if (!TW) tmem_ld32(tmem + lane_off + C::QB_COL + sw * (D / 2) + cc, qb);
            tmem_ld_wait();
            if (valid) {
              uint4* o = reinterpret_cast<uint4*>(dkr + cc);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                float x[8];
#pragma unroll
                for (int j = 0; j < 8; ++j)
                  x[j] = TW ? a.scale * uu[8 * k + j] : a.scale * fmaf(-Dv, qb[8 * k + j], uu[8 * k + j]);
                o[k] = make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]),
                                  pack_bf16(x[6], x[7]));
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty);
        cur.next();
      }
      if (warp == kSoftWarp0 && lane == 0) bulk_wait_all();  // stores complete before exit
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, int P>
__global__ void __launch_bounds__(kThreads, 1)
    tc_bwd_tok_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmG,
                      const __grid_constant__ CUtensorMap tmDK, const __grid_constant__ CUtensorMap tmDV, Args a,
                      const float* __restrict__ lse, float* __restrict__ Dco, __nv_bfloat16* __restrict__ dK,
                      __nv_bfloat16* __restrict__ dV) {
  bwd_tok_body<D, P, false>(tmK, tmV, tmQ, tmG, tmDK, tmDV, a, lse, Dco, dK, dV);
}

template <int D, int P>
__global__ void __launch_bounds__(kThreads, 1)
    tc_tw_bwd_tok_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                         const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmG,
                         const __grid_constant__ CUtensorMap tmDK, const __grid_constant__ CUtensorMap tmDV, Args a,
                         const float* __restrict__ lse_tok, float* __restrict__ Dtw, __nv_bfloat16* __restrict__ dK,
                         __nv_bfloat16* __restrict__ dV) {
  bwd_tok_body<D, P, true>(tmK, tmV, tmQ, tmG, tmDK, tmDV, a, lse_tok, Dtw, dK, dV);
}

// dsketch fp32 -> bf16 copy in the workspace, the layout TMA streams ([B*H][P][D])
__global__ void to_bf16_kernel(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst, int64_t n8,
                               const void* ws) {
  if (ws_failed(ws)) return;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n8; i += int64_t(gridDim.x) * blockDim.x) {
    const float4 x = reinterpret_cast<const float4*>(src)[2 * i];
    const float4 y = reinterpret_cast<const float4*>(src)[2 * i + 1];
    reinterpret_cast<uint4*>(dst)[i] =
        make_uint4(pack_bf16(x.x, x.y), pack_bf16(x.z, x.w), pack_bf16(y.x, y.y), pack_bf16(y.z, y.w));
  }
}

template <int D, int P, bool TW = false>
static cudaError_t launch_tok_t(const Args& a, int W, const __nv_bfloat16* gbf, const float* lse, float* Dco,
                                void* dK, void* dV, cudaStream_t st) {
  using C = TokCfg<D, P>;
  CUtensorMap tk, tv, tq, tg, tdk, tdv;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, C::NC) || !make_q_map(&tg, gbf, a.B * a.H, a.P, D, C::NC) ||
      !make_kv_map(&tdk, dK, a.N, a.H, D) || !make_kv_map(&tdv, dV, a.N, a.H, D))
    return cudaErrorInvalidValue;
  auto fn = TW ? &tc_tw_bwd_tok_kernel<D, P> : &tc_bwd_tok_kernel<D, P>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  fn<<<W, kThreads, C::SMEM, st>>>(tk, tv, tq, tg, tdk, tdv, a, lse, Dco, static_cast<__nv_bfloat16*>(dK),
                                   static_cast<__nv_bfloat16*>(dV));
  return cudaGetLastError();
}

}  // namespace tcb

bool tc_bwd_split(int P, int d) {
  return (d == 128 && (P == 256 || P == 512 || P == 1024 || P == 2048)) ||
         (d == 64 && (P == 512 || P == 1024 || P == 2048));
}

cudaError_t launch_tc_g_bf16(const Args& a, const float* dsk, __nv_bfloat16* gbf, cudaStream_t st) {
  const int64_t n8 = int64_t(a.B) * a.H * a.P * a.d / 8;
  tcb::to_bf16_kernel<<<1024, 256, 0, st>>>(dsk, gbf, n8, a.ws);
  return cudaGetLastError();
}

cudaError_t launch_tc_bwd_tok(const Args& a, int W, const float* dsk, __nv_bfloat16* gbf, const float* lse,
                              float* Dco, void* dK, void* dV, cudaStream_t st) {
  (void)dsk;
  if (a.N == 0) return cudaSuccess;
  if (a.d == 64) {
    if (a.P == 2048) return tcb::launch_tok_t<64, 2048>(a, W, gbf, lse, Dco, dK, dV, st);
    if (a.P == 1024) return tcb::launch_tok_t<64, 1024>(a, W, gbf, lse, Dco, dK, dV, st);
    return tcb::launch_tok_t<64, 512>(a, W, gbf, lse, Dco, dK, dV, st);
  }
  if (a.P == 2048) return tcb::launch_tok_t<128, 2048>(a, W, gbf, lse, Dco, dK, dV, st);
  if (a.P == 1024) return tcb::launch_tok_t<128, 1024>(a, W, gbf, lse, Dco, dK, dV, st);
  if (a.P == 512) return tcb::launch_tok_t<128, 512>(a, W, gbf, lse, Dco, dK, dV, st);
  return tcb::launch_tok_t<128, 256>(a, W, gbf, lse, Dco, dK, dV, st);
}

cudaError_t launch_tc_bwd_dq(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                             cudaStream_t st);

int tc_bwd_dq_workers(int num_sms, int P) {
  const int w = num_sms / (P / 128);
  return w < 1 ? 1 : w;
}

}  // namespace sa

// ================================================================ dQ (slices)
// Prototype side of the backward: one slice of PS = 128 prototypes per CTA,
// prototypes on TMEM lanes, tokens on columns:
//   S  = Q_r K^T,  dA = G_r V^T                (UMMA, [PS x 128 tokens])
//   dS = exp(scale S - lse_t) o (dA - D_t)     (registers; lse_t and D_t are
//                                               per-column values, no reduction)
//   dQ_r += dS K                               (UMMA with dS as the A operand
//                                               straight from TMEM)
// D_t comes from the token-side kernel.  Keeping dS in TMEM spares the
// shared-memory round trip that bounds the other kernels.
namespace sa {
namespace tcb {

template <int D, int PS>
struct QCfg {
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int QB = PS * D * 2;
  // K(i) is read by S(i) and, a tile later, by dQ(i); V(i) only by dA(i).  So
  // K gets four slots and V two: K(i+3) loads once dQ(i-1) is done and V(i+2)
  // once dA(i) is, a tile or more before they are needed.  (The dsketch slice
  // lives in TMEM as the A operand of dA, which leaves room for the fourth.)
  static constexpr int NK = 4, NV = 2;
  static constexpr int NSLOT = NK + NV;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_RING = QB;  // K slots 0..NK-1, then V slots
  static constexpr int OFF_COL = OFF_RING + NSLOT * KV_TILE;  // [2 bufs][lse2 | D][128] fp32
  static constexpr int OFF_BAR = OFF_COL + 2 * 2 * T * 4;
  static constexpr int NBAR = 2 * NSLOT + 16;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;  // TMEM base, abort flag
  static constexpr int OFF_FLAGS = OFF_MISC + 16;      // per K slot: control bits of the tile it holds
  static constexpr int SMEM = OFF_FLAGS + 4 * NK;
  // S^T and dA^T fp32; dS (bf16 pairs) and the dsketch slice G (bf16 pairs, the
  // A operand of dA^T = G V^T) 64 columns each; dQ fp32
  static constexpr int S_COL = 0, DA_COL = T, DS_COL = 2 * T, G_COL = 2 * T + T / 2, DQ_COL = 3 * T;
  static constexpr int TMEM_COLS = tmem_cols_for(DQ_COL + D);
  static_assert(PS == 128 && TMEM_COLS <= 512 && SMEM <= 232448, "budget");
};

// Per-tile control bits, written by the TMA producer next to the tile's K so
// the UMMA issuer follows the tile sequence without walking it.
enum : uint32_t { kNewHead = 1u, kHeadLast = 2u, kSegFirst = 4u, kSegLast = 8u };

// TW = false: prototype-wise weights, lse and D per token (column values
// staged by warps 2-3).  TW = true: token-wise weights (Sec. 5.1), lse and D
// per prototype [B][H][P]: per-row (per-thread) values, and columns past the
// tile's tokens are masked here.
template <int D, int PS, bool TW>
__device__ __forceinline__ void bwd_dq_body(const CUtensorMap& tmK, const CUtensorMap& tmV, const CUtensorMap& tmQ,
                                            const Args& a, const float* __restrict__ dsk,
                                            const float* __restrict__ lse, const float* __restrict__ Dco) {
  using C = QCfg<D, PS>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ws_failed(a.ws)) return;
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xB31u);
    return;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sRing = sbase + C::OFF_RING;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  // slot s < NK holds K tiles, slot NK + j holds V tiles
  auto ring_full = [&](int s) { return bar0 + 8u * s; };
  auto ring_empty = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  auto k_slot = [](int li) { return li % C::NK; };
  auto v_slot = [](int li) { return C::NK + li % C::NV; };
  const uint32_t b1 = bar0 + 8u * (2 * C::NSLOT);
  const uint32_t q_full = b1, q_empty = b1 + 8, g_full = b1 + 16, g_empty = b1 + 24, sda_full = b1 + 32,
                 sda_free = b1 + 40, ds_full = b1 + 48, ds_empty0 = b1 + 56, dq_empty = b1 + 72,
                 col_full0 = b1 + 80, col_empty0 = b1 + 96, drain = b1 + 112;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  uint32_t* tflags = reinterpret_cast<uint32_t*>(smem + C::OFF_FLAGS);
  float* cols = reinterpret_cast<float*>(smem + C::OFF_COL);
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = gridDim.x, wk = blockIdx.x, slice = blockIdx.y;
  const int p0 = slice * PS;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  const int ntiles = int(te - tb);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(ring_full(s), 1);
      mbar_init(ring_empty(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(g_full, kSoftWarps);
    mbar_init(g_empty, 1);
    mbar_init(sda_full, 1);
    mbar_init(sda_free, kSoftWarps);
    mbar_init(ds_full, kSoftWarps);
    mbar_init(ds_empty0, 1);
    mbar_init(ds_empty0 + 8, 1);  // unused (one dS buffer)
    mbar_init(dq_empty, kSoftWarps);
    mbar_init(col_full0, 2);
    mbar_init(col_full0 + 8, 2);
    mbar_init(col_empty0, kSoftWarps);
    mbar_init(col_empty0 + 8, kSoftWarps);
    mbar_init(drain, 1);
    wait_ctl_init(abort_flag, a.ws);
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Registers: the control warpgroup (warps 0-3: TMA, UMMA issuer, column loaders)
  // hands registers to the two softmax warpgroups (128 x 136 + 256 x 184 = 384 x 168).
  if (ntiles > 0 && warp < kSoftWarp0) {
    setmaxnreg_dec<136>();
    if (warp == 0 && lane == 0) {
      // ---------------------------------------------------------- TMA producer
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      TileWalker it(a, tb, te, T);
      int hc = 0, prev_h = -1, loaded = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        // "head" below = the run of tiles reading one row of Q: a head, or with
        // per-user queries one (user, head) segment
        const bool new_head = it.qk != prev_h;
        if (new_head) {
          if (hc > 0) ok = mbar_wait(q_empty, (hc - 1) & 1, abort_flag, a.ws, 0xC01);
          if (!ok) break;
          mbar_arrive_expect_tx(q_full, C::QB);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(sQ + dh * PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
          prev_h = it.qk;
          ++hc;
        }
        int64_t t0n;
        int nn, hn, qkn;
        it.peek_next(t0n, nn, hn, qkn);
        const uint32_t fl = (new_head ? kNewHead : 0u) | ((li + 1 >= ntiles || qkn != it.qk) ? kHeadLast : 0u) |
                            (it.seg_first ? kSegFirst : 0u) | (it.seg_last ? kSegLast : 0u);
#pragma unroll
        for (int kv = 0; kv < 2; ++kv) {
          const int nsl = kv ? C::NV : C::NK, use = li / nsl;
          const int s = kv ? v_slot(li) : k_slot(li);
          if (use > 0) ok = mbar_wait(ring_empty(s), (use + 1) & 1, abort_flag, a.ws, 0xC02);
          if (!ok) break;
          if (kv == 0) tflags[s] = fl;  // published by the arrive below
          mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh)
            tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, kv ? &tmV : &tmK, ring_full(s), 64 * dh, it.h,
                        int(it.tok0));
          loaded = li + 1;
        }
        it.next();
      }
      if (!ok) {  // let the copies in flight land before the CTA exits
        for (int li = (loaded > C::NK ? loaded - C::NK : 0); li < loaded; ++li) {
          mbar_wait_bounded(ring_full(k_slot(li)), (li / C::NK) & 1, 200000000ull);
          if (li + C::NV >= loaded) mbar_wait_bounded(ring_full(v_slot(li)), (li / C::NV) & 1, 200000000ull);
        }
      }
    } else if (warp == 1 && lane == 0) {
      // ---------------------------------------------------------- UMMA issuer
      // Order: S(0), dA(0);
      // then per tile i: S(i+1), dA(i+1), dQ(i), so the next tile's scores are
      // ready when the softmax warps finish tile i.  One commit announces S and
      // dA together (the softmax warps read both at once); descriptors are
      // built once per operand and stepped by constant offsets.
      constexpr uint32_t idPT = idesc_bf16(128, T, 0, 0);  // [proto x tok], K = d
      constexpr uint32_t idQ = idesc_bf16(128, D, 0, 1);   // [proto x d], K = tokens, A from TMEM
      const uint64_t dQs = sdesc(sQ, 16, 1024);
      auto step_p = [](int k) { return uint32_t((k >> 2) * (PS * 128) + (k & 3) * 32); };
      auto step_t = [](int k) { return uint32_t((k >> 2) * (T * 128) + (k & 3) * 32); };
      int hc = 0, gc = 0, hp = 0;
      bool ok = true;
      auto wt = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return ok = ok && mbar_wait(bar, par, abort_flag, a.ws, site);
      };
      // waits for tile li's K and V, returns its control bits
      auto wait_kv = [&](int li) -> uint32_t {
        wt(ring_full(k_slot(li)), (li / C::NK) & 1, 0xD02);
        wt(ring_full(v_slot(li)), (li / C::NV) & 1, 0xD04);
        return ok ? tflags[k_slot(li)] : 0u;
      };
      auto issue_sda = [&](int li, uint32_t fl) {
        if (fl & kNewHead) {
          wt(q_full, hc & 1, 0xD01);
          ++hc;
        }
        if (fl & kSegFirst) {
          wt(g_full, gc & 1, 0xD03);
          ++gc;
        }
        if (!ok) return;
        tc_fence_after();
        const int sK = k_slot(li), sV = v_slot(li);
        const uint64_t dK = sdesc(sRing + sK * C::KV_TILE, 16, 1024), dV = sdesc(sRing + sV * C::KV_TILE, 16, 1024);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          umma_ss(tmem + C::S_COL, sdesc_add(dQs, step_p(k)), sdesc_add(dK, step_t(k)), idPT, k > 0 ? 1u : 0u);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)  // G from TMEM: 8 columns (16 values of d) per step
          umma_ts(tmem + C::DA_COL, tmem + C::G_COL + 8 * k, sdesc_add(dV, step_t(k)), idPT, k > 0 ? 1u : 0u);
        umma_commit(sda_full);
        umma_commit(ring_empty(sV));                // V read by its only product
        if (fl & kHeadLast) umma_commit(q_empty);   // last S of this head piece
        if (fl & kSegLast) umma_commit(g_empty);    // last dA of this segment
      };
      uint32_t fl_cur = wait_kv(0);
      if (ok) issue_sda(0, fl_cur);
      for (int li = 0; li < ntiles && ok; ++li) {
        uint32_t fl_next = 0;
        if (li + 1 < ntiles) {
          wt(sda_free, li & 1, 0xD07);  // the softmax warps hold S(i), dA(i)
          fl_next = wait_kv(li + 1);
          if (!ok) break;
          issue_sda(li + 1, fl_next);
          if (!ok) break;
        }
        // ---- dQ += dS(i) K(i), dS read from TMEM
        const bool first_of_hp = (fl_cur & kNewHead) != 0;
        wt(ds_full, li & 1, 0xD09);
        if (first_of_hp && hp > 0) wt(dq_empty, (hp - 1) & 1, 0xD0A);
        if (!ok) break;
        tc_fence_after();
        {
          const int sK = k_slot(li);
          const uint64_t dK = sdesc(sRing + sK * C::KV_TILE, T * 128, 1024);  // MN-major: d blocks 16 KB apart
          const uint32_t dsb = tmem + C::DS_COL;
#pragma unroll
          for (int k = 0; k < T / 16; ++k)
            umma_ts(tmem + C::DQ_COL, dsb + 8 * k, sdesc_add(dK, k * 2048), idQ, (first_of_hp && k == 0) ? 0u : 1u);
          umma_commit(ds_empty0);
          umma_commit(ring_empty(sK));
        }
        if (fl_cur & kHeadLast) ++hp;
        fl_cur = fl_next;
      }
      umma_commit(drain);
      mbar_wait_bounded(drain, 0, 200000000ull);
    } else if (warp == 2 || warp == 3) {
      // ------------------------------------------------- per-token columns
      const int t64 = threadIdx.x - 64;
      TileWalker cur(a, tb, te, T);
      bool ok = true;
      auto hw = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      for (int li = 0; li < ntiles && ok; ++li) {
        if (!TW) {
          const int buf = li & 1;
          if (li >= 2) ok = hw(col_empty0 + 8 * buf, ((li >> 1) + 1) & 1, 0xE02);
          if (!ok) break;
          float* cl = cols + buf * 2 * T;
          for (int t = t64; t < T; t += 64) {
            const bool v = t < cur.n;
            const int64_t idx = (cur.tok0 + t) * a.H + cur.h;
            cl[t] = v ? lse[idx] * 1.4426950408889634f : INFINITY;  // exp2(x - inf) = 0 for padding
            cl[T + t] = v ? Dco[idx] : 0.f;
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(col_full0 + 8 * buf);
        }
        cur.next();
      }
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<184>();
    {
      // ------------------------------------------------ dS + dQ epilogue
      const int sw = (warp - kSoftWarp0) >> 2, q = warp & 3;
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * 1.4426950408889634f;
      TileWalker cur(a, tb, te, T);
      bool ok = true;
      int gc = 0;
      // The dsketch slice of user b, head h into TMEM as bf16 pairs (the A operand of
      // dA^T = G V^T): this thread's prototype row, warpgroup sw's half of the d columns.
      // Written once the last dA of the previous segment is done (g_empty).
      auto put_g = [&](int b, int h) -> bool {
        if (gc > 0 && !__all_sync(0xffffffffu, mbar_wait(g_empty, (gc - 1) & 1, abort_flag, a.ws, 0xF06)))
          return false;
        const float4* src = reinterpret_cast<const float4*>(
            dsk + ((int64_t(b) * a.H + h) * a.P + p0 + 32 * q + lane) * D + (D / 2) * sw);
#pragma unroll
        for (int half = 0; half < D / 64; ++half) {
          uint32_t pk[16];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 x = src[8 * half + j];
            pk[2 * j] = pack_bf16(x.x, x.y);
            pk[2 * j + 1] = pack_bf16(x.z, x.w);
          }
          tmem_st16(tmem + lane_off + C::G_COL + (D / 4) * sw + 16 * half, pk);
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(g_full);
        ++gc;
        return true;
      };
      ok = put_g(cur.b, cur.h);
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      int hp = 0;
      for (int li = 0; li < ntiles && ok; ++li) {
        const int buf = li & 1;
        float l2r = 0.f, dr = 0.f;  // token-wise: this row's lse (log2 units) and D
        if (TW) {
          const int64_t r = (int64_t(cur.b) * a.H + cur.h) * a.P + p0 + 32 * q + lane;
          l2r = lse[r] * 1.4426950408889634f;
          dr = Dco[r];
        } else {
          ok = wwait(col_full0 + 8 * buf, (li >> 1) & 1, 0xF01);
        }
        if (ok) ok = wwait(sda_full, li & 1, 0xF02);
        if (!ok) break;
        tc_fence_after();
        const float* cl = cols + buf * 2 * T;
        float sv[64], dv[64];  // this warpgroup's 64 token columns of S and dA
        tmem_ld32(tmem + lane_off + C::S_COL + 64 * sw, sv);
        tmem_ld32(tmem + lane_off + C::S_COL + 64 * sw + 32, sv + 32);
        tmem_ld32(tmem + lane_off + C::DA_COL + 64 * sw, dv);
        tmem_ld32(tmem + lane_off + C::DA_COL + 64 * sw + 32, dv + 32);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        // the next tile opens a new (user, head) segment: its dsketch slice goes in
        // before S and dA of that tile are issued (they wait for sda_free and g_full)
        if (li + 1 < ntiles && cur.seg_last) {
          const TileRef nx = locate_next_segment(cur.t + 1, cur.h, cur.b, cur.tph, a.prefix, a.cu, a.B, T);
          if (!put_g(nx.b, nx.h)) {
            ok = false;
            break;
          }
        }
        if (lane == 0) mbar_arrive(sda_free);  // the next tile's S and dA may now be written
        if (TW) {
          // per-row shift and D; columns past the tile's tokens weigh zero
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const int col = 64 * sw + 32 * c;
            uint32_t pk[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int jj = 32 * c + 2 * j;
              const float a0 = col + 2 * j < cur.n ? ex2(fmaf(sv[jj], c2, -l2r)) : 0.f;
              const float a1 = col + 2 * j + 1 < cur.n ? ex2(fmaf(sv[jj + 1], c2, -l2r)) : 0.f;
              pk[j] = pack_bf16(a0 * (dv[jj] - dr), a1 * (dv[jj + 1] - dr));
            }
            // dS(i) overwrites dS(i-1): dQ(i-1) must have read it
            if (c == 0 && li > 0 && !wwait(ds_empty0, (li - 1) & 1, 0xF04)) {
              ok = false;
              break;
            }
            tmem_st16(tmem + lane_off + C::DS_COL + col / 2, pk);
          }
          if (!ok) break;
        }
        // per-token values as 16-byte broadcasts: one shared-memory wavefront per 4 tokens
        const float4* cl4 = reinterpret_cast<const float4*>(cl);
#pragma unroll
        for (int c = 0; c < 2 && !TW; ++c) {
          const int col = 64 * sw + 32 * c;
          uint32_t pk[16];
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4) {
            const float4 l4 = cl4[(col >> 2) + j4];
            const float4 d4 = cl4[((T + col) >> 2) + j4];
            const int jj = 32 * c + 4 * j4;
            const float a0 = ex2(fmaf(sv[jj], c2, -l4.x)), a1 = ex2(fmaf(sv[jj + 1], c2, -l4.y));
            const float a2 = ex2(fmaf(sv[jj + 2], c2, -l4.z)), a3 = ex2(fmaf(sv[jj + 3], c2, -l4.w));
            pk[2 * j4] = pack_bf16(a0 * (dv[jj] - d4.x), a1 * (dv[jj + 1] - d4.y));
            pk[2 * j4 + 1] = pack_bf16(a2 * (dv[jj + 2] - d4.z), a3 * (dv[jj + 3] - d4.w));
          }
          if (c == 0 && li > 0 && !wwait(ds_empty0, (li - 1) & 1, 0xF04)) {
            ok = false;
            break;
          }
          tmem_st16(tmem + lane_off + C::DS_COL + col / 2, pk);
        }
        if (!ok) break;
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(ds_full);
          if (!TW) mbar_arrive(col_empty0 + 8 * buf);
        }
        // dQ partial of this worker and head (or user segment) at the end of its piece
        const bool more = li + 1 < ntiles;
        int64_t t0n;
        int nn, hn, qkn;
        cur.peek_next(t0n, nn, hn, qkn);
        if (!more || qkn != cur.qk) {
          ok = wwait(ds_empty0, li & 1, 0xF05);
          if (!ok) break;
          tc_fence_after();
          float* dst = dq_block_dst(a, wk, W, total, cur, p0, D);
          store_sketch_scaled<D, PS, C::DQ_COL>(tmem, lane_off, sw, q, lane, dst, a.scale);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(dq_empty);
          ++hp;
        }
        cur.next();
      }
      (void)hp;
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, int PS>
__global__ void __launch_bounds__(kThreads, 1)
    tc_bwd_dq_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     const __grid_constant__ CUtensorMap tmQ, Args a, const float* __restrict__ dsk,
                     const float* __restrict__ lse, const float* __restrict__ Dco) {
  bwd_dq_body<D, PS, false>(tmK, tmV, tmQ, a, dsk, lse, Dco);
}

template <int D, int PS>
__global__ void __launch_bounds__(kThreads, 1)
    tc_tw_bwd_dq_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                        const __grid_constant__ CUtensorMap tmQ, Args a, const float* __restrict__ dsk,
                        const float* __restrict__ lse_tok, const float* __restrict__ Dtw) {
  bwd_dq_body<D, PS, true>(tmK, tmV, tmQ, a, dsk, lse_tok, Dtw);
}

template <int D, int PS, bool TW = false>
static cudaError_t launch_dq_t(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                               cudaStream_t st) {
  using C = QCfg<D, PS>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, PS))
    return cudaErrorInvalidValue;
  auto fn = TW ? &tc_tw_bwd_dq_kernel<D, PS> : &tc_bwd_dq_kernel<D, PS>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid(W, a.P / PS);
  fn<<<grid, kThreads, C::SMEM, st>>>(tk, tv, tq, a, dsk, lse, Dco);
  return cudaGetLastError();
}

}  // namespace tcb
}  // namespace sa

namespace sa {
cudaError_t launch_tc_bwd_dq(const Args& a, int W, const float* dsk, const float* lse, const float* Dco,
                             cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  return a.d == 64 ? tcb::launch_dq_t<64, 128>(a, W, dsk, lse, Dco, st) : tcb::launch_dq_t<128, 128>(a, W, dsk, lse, Dco, st);
}

// Token-wise normalisation (Sec. 5.1): the same two kernels with per-prototype
// lse_tok and D_j = G_j . O_j ([B][H][P]); d = 128 and P in {256, ..., 2048}.
bool tc_tw_bwd_supported(int P, int d, sa_dtype dt) {
  return dt == SA_BF16 && d == 128 && (P == 256 || P == 512 || P == 1024 || P == 2048) && tcc::device_is_sm103() &&
         tc_path_enabled();
}

cudaError_t launch_tc_tw_bwd_tok(const Args& a, int W, const __nv_bfloat16* gbf, const float* lse_tok,
                                 const float* Dtw, void* dK, void* dV, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  float* Dp = const_cast<float*>(Dtw);  // read only in token-wise mode
  if (a.P == 2048) return tcb::launch_tok_t<128, 2048, true>(a, W, gbf, lse_tok, Dp, dK, dV, st);
  if (a.P == 1024) return tcb::launch_tok_t<128, 1024, true>(a, W, gbf, lse_tok, Dp, dK, dV, st);
  if (a.P == 512) return tcb::launch_tok_t<128, 512, true>(a, W, gbf, lse_tok, Dp, dK, dV, st);
  return tcb::launch_tok_t<128, 256, true>(a, W, gbf, lse_tok, Dp, dK, dV, st);
}

cudaError_t launch_tc_tw_bwd_dq(const Args& a, int W, const float* dsk, const float* lse_tok, const float* Dtw,
                                cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  return tcb::launch_dq_t<128, 128, true>(a, W, dsk, lse_tok, Dtw, st);
}
}  // namespace sa
