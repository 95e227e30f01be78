// tcgen05 / TMEM / TMA forward kernels of the SA sketching step (sm_103a).
//
// One CTA per SM walks a contiguous range of 128-token tiles (ragged tiling of
// sa_common.cuh).  Per tile (paper Sec. 3.1; FlashSA's streaming scheme of
// Sec. 4.4, S and A never leave the SM):
//   1. TMA brings the tile's K and V rows ([128 tokens][d] bf16, 128-byte
//      swizzle) into a ring of shared-memory slots; the prototype block Q
//      ([PS][d]) stays resident while the head does not change.
//   2. UMMA  S^T = K Q^T  (M = 128 tokens, N = PS prototypes, K = d) into TMEM,
//      so each token's P scores lie in one TMEM lane.
//   3. Eight softmax warps read the scores into registers (one token per
//      thread, half of the prototypes per warpgroup), normalise over the
//      prototypes -- either with their own max / sum (fused mode, all P in
//      this CTA) or with a given per-token log-sum-exp (sliced mode) -- and
//      write the weights A as bf16 into shared memory.
//   4. UMMA accumulates the sketch in TMEM:  O = A V  (d = 64: M = prototypes,
//      N = d) or  O^T = V^T A^T  (d = 128: M = d, N = prototypes).
//   5. When a user's segment ends the sketch (or a worker's piece of it) is
//      read back from TMEM and stored.
// Pair mode (P = 512): a cluster of two CTAs shares each tile; CTA r holds
// prototypes [256 r, 256 r + 256).  Per token, warpgroup 1 hands its (max,
// sum) to warpgroup 0 through shared memory; warpgroup 0 combines the CTA's
// two partials, pushes the result into the peer CTA's shared memory with
// st.async (whose completion is counted on the peer's mbarrier, so no
// cluster-scope fence is needed), combines its own and the peer's value in
// CTA order -- bitwise the same (max, sum) in both CTAs -- and hands the final
// pair back to warpgroup 1.
// Warp roles: 0 = TMA producer, 1 = UMMA issuer, 2 = TMEM allocator,
// 4..11 = softmax + epilogue.  Every wait is bounded (sa_ptx.cuh).
#include <cuda.h>
#include <cuda_fp16.h>

#include <cstdio>

#include "sa_ptx.cuh"
#include "sa_tc.cuh"
#include "sa_tc_common.cuh"

namespace sa {
namespace tcf {

using namespace ptx;
using namespace tcc;

enum Mode { kFused = 0, kSliced = 1, kPair = 2 };

constexpr uint32_t kRegsCtl = 104, kRegsSoft = 200;
static_assert(128 * kRegsCtl + 256 * kRegsSoft == 384 * 168, "register split = launch allocation");

template <int D, int PS, int MODE>
struct Cfg {
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = PS * D * 2;
  static constexpr int W_BYTES = T * PS * 2;
  static constexpr int NSLOT = (D == 128) ? 3 : 6;
  // fused: (max, sum) of each warpgroup [2][T] float2.  pair: each
  // warpgroup's max [2][T] fp32 and sum [2][T] fp16, then the peer CTA's pushed
  // (max, sum) [T] float2 at STATS_R
  static constexpr int STATS = (MODE == kSliced) ? 0 : (MODE == kPair) ? 2 * T * 4 + 2 * T * 2 + T * 8 : 2 * T * 8;
  static constexpr int STATS_Z = 2 * T * 4, STATS_R = 2 * T * 4 + 2 * T * 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_RING = OFF_Q + Q_BYTES;
  static constexpr int OFF_W = OFF_RING + NSLOT * KV_TILE;
  static constexpr int OFF_STATS = OFF_W + W_BYTES;
  static constexpr int OFF_BAR = OFF_STATS + STATS;
  static constexpr int NBAR = 2 * NSLOT + 16;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;  // tmem address, abort flag, skip flag (pair)
  static constexpr int SMEM = OFF_MISC + 16;
  static_assert(SMEM <= 232448, "shared memory budget");
  static constexpr bool TRANS = (D == 128);  // O^T = V^T A^T
  static constexpr int O_COLS = TRANS ? PS : (PS / 128) * D;
  static constexpr int S_COL = 0;
  static constexpr int O_COL = PS;
  // two sketch accumulators where TMEM holds them: a segment's sketch is stored
  // while the next segment accumulates into the other one
  static constexpr int NOB = (PS + 2 * O_COLS <= 512) ? 2 : 1;
  static constexpr int TMEM_COLS = tmem_cols_for(PS + NOB * O_COLS);
  static constexpr int HALF = PS / 2;  // prototypes per softmax warpgroup
};

template <int D, int PS, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_fwd_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const __grid_constant__ CUtensorMap tmQ, Args a, float* __restrict__ sketch,
                  float* __restrict__ lse_out, const float* __restrict__ lse_in) {
  using C = Cfg<D, PS, MODE>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr bool PAIR = (MODE == kPair);
  // A pair's CTAs must both reach the cluster barriers below, so pair mode
  // never returns early: a failed call or a misaligned base only skips work.
  bool skip = ws_failed(a.ws);
  if (smem_u32(smem) & 1023u) {  // 128-byte swizzle atoms need 1024-byte alignment
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xA11u);
    skip = true;
  }
  if (!PAIR && skip) return;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sRing = sbase + C::OFF_RING, sW = sbase + C::OFF_W;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto ring_full = [&](int s) { return bar0 + 8u * s; };
  auto ring_empty = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  const uint32_t q_full = bar0 + 8u * (2 * C::NSLOT + 0), q_empty = q_full + 8, s_full = q_full + 16,
                 s_empty = q_full + 24, w_full = q_full + 32, w_empty = q_full + 40, o_full = q_full + 48,
                 o_empty = q_full + 56, drain = q_full + 64, st_ready = q_full + 72, st_used = q_full + 80,
                 r_full = q_full + 88, r_used = q_full + 96, never = q_full + 104;
  // barriers of sketch accumulator ob
  auto o_full_of = [&](int ob) { return ob ? q_full + 112 : o_full; };
  auto o_empty_of = [&](int ob) { return ob ? q_full + 120 : o_empty; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  volatile uint32_t* skip_flag = reinterpret_cast<volatile uint32_t*>(smem + C::OFF_MISC + 8);
  const uint32_t rank = PAIR ? cluster_rank() : 0u, peer = rank ^ 1u;

  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  // pair mode: the two CTAs of cluster c are worker c; CTA rank r is slice r
  const int W = PAIR ? int(gridDim.x >> 1) : int(gridDim.x);
  const int wk = PAIR ? int(blockIdx.x >> 1) : int(blockIdx.x);
  const int slice = PAIR ? int(rank) : int(blockIdx.y);
  const int p0 = slice * PS;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  int ntiles = int(te - tb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(ring_full(s), 1);
      mbar_init(ring_empty(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(s_full, 1);
    mbar_init(s_empty, kSoftWarps);
    mbar_init(w_full, kSoftWarps);
    mbar_init(w_empty, 1);
    mbar_init(o_full, 1);
    mbar_init(o_empty, kSoftWarps);
    mbar_init(q_full + 112, 1);
    mbar_init(q_full + 120, kSoftWarps);
    mbar_init(drain, 1);
    // pair mode: st_ready = both warpgroups' partials are in (8 warps; st_used
    // is unused); r_full = the peer's pair has landed (one local expect_tx +
    // 1 KB of st.async), r_used = the peer has read what this CTA pushed (the
    // peer's 8 softmax warps)
    mbar_init(st_ready, kSoftWarps);
    mbar_init(st_used, kSoftWarps);
    mbar_init(r_full, 1);
    mbar_init(r_used, kSoftWarps);
    mbar_init(never, 1);  // completed by nothing: the forced timeout of a test limit
    wait_ctl_init(abort_flag, a.ws);
    *skip_flag = skip ? 1u : 0u;
    fence_mbar_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
  tc_fence_before();
  if (PAIR) {
    // barriers of both CTAs initialised; both CTAs skip if either must
    cluster_sync_all();
    if (*skip_flag || ld_cluster_u32(mapa_shared(smem_u32(smem + C::OFF_MISC + 8), peer))) ntiles = 0;
  } else {
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Registers: the control warpgroup (warps 0-3) gives up registers so that the
  // two softmax warpgroups can hold a tile row of 128 scores without spilling:
  // 128 x kRegsCtl + 256 x kRegsSoft = 384 x 168, the launch allocation.
  if (ntiles > 0 && warp < kSoftWarp0) {
    setmaxnreg_dec<kRegsCtl>();
    if (warp == 0 && lane == 0) {
      // ------------------------------------------------------ TMA producer
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmQ);
      TileWalker it(a, tb, te, T), pv(a, tb, te, T), pf(a, tb, te, T);
      pf.next();
      pf.next();
      int hc = 0, prev_h = -1;
      uint32_t e = 0;
      bool ok = true;
      for (int li = 0; li <= ntiles && ok; ++li) {
        if (li + 2 < ntiles) {
          // K and V of tile li + 2 into L2, so the ring loads hit L2
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh) {
            tma_prefetch_l2_3d(&tmK, 64 * dh, pf.h, int(pf.tok0));
            tma_prefetch_l2_3d(&tmV, 64 * dh, pf.h, int(pf.tok0));
          }
          pf.next();
        }
        if (li < ntiles) {
          if (it.qk != prev_h) {  // a new head (or, with per-user queries, a new user)
            if (hc > 0) ok = mbar_wait(q_empty, (hc - 1) & 1, abort_flag, a.ws, 0x101);
            if (!ok) break;
            mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
            for (int dh = 0; dh < D / 64; ++dh) tma_load_3d(sQ + dh * PS * 128, &tmQ, q_full, 64 * dh, p0, it.qk);
            prev_h = it.qk;
            ++hc;
          }
          const int s = int(e % C::NSLOT);
          if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x102);
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
          if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x103);
          if (!ok) break;
          mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
          for (int dh = 0; dh < D / 64; ++dh)
            tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, &tmV, ring_full(s), 64 * dh, pv.h, int(pv.tok0));
          ++e;
          pv.next();
        }
      }
      // drain loads still in flight before the CTA may exit: the last NSLOT
      // ring loads (every older slot was released by a completed reader) and
      // the last prototype block
      if (!ok) {
        for (uint32_t k = (e > uint32_t(C::NSLOT) ? e - C::NSLOT : 0); k < e; ++k)
          mbar_wait_bounded(ring_full(int(k % C::NSLOT)), (k / C::NSLOT) & 1, 200000000ull);
        if (hc > 0) mbar_wait_bounded(q_full, uint32_t(hc - 1) & 1u, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      // ------------------------------------------------------ UMMA issuer
      constexpr uint32_t idS = idesc_bf16(128, PS, 0, 0);
      constexpr uint32_t idO = C::TRANS ? idesc_bf16(128, PS, 1, 1) : idesc_bf16(128, D, 1, 1);
      TileWalker cur(a, tb, te, T), nxt(a, tb, te, T);
      nxt.next();
      uint32_t e = 0;
      int hc = 0, sc = 0;
      // under a test limit (sa_set_wait_limit_ns) the issuer first waits for a
      // barrier nothing completes: the limit runs out and the CTA takes its
      // abort path (drains, TMEM freed, SA_ERR_TIMEOUT)
      bool ok = ctl_wait_limit(abort_flag) >= kPollLimitNs || mbar_wait(never, 0, abort_flag, a.ws, 0x200);
      ok = ok && mbar_wait(q_full, 0, abort_flag, a.ws, 0x201);
      // operand descriptors built once and stepped by constant offsets: the
      // issuing thread shares its sub-partition with two softmax warps, and each
      // instruction it saves shortens the issue of a group
      const uint64_t dQ0 = sdesc(sQ, 16, 1024), dW0 = sdesc(sW, T * 128, 1024);
      const uint64_t dK0 = sdesc(sRing, 16, 1024), dV0 = sdesc(sRing, T * 128, 1024);
      auto issue_S = [&](uint32_t slot) {
        const uint64_t dK = sdesc_add(dK0, slot * C::KV_TILE);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          umma_ss(tmem + C::S_COL, sdesc_add(dK, (k >> 2) * (T * 128) + (k & 3) * 32),
                  sdesc_add(dQ0, (k >> 2) * (PS * 128) + (k & 3) * 32), idS, k > 0 ? 1u : 0u);
      };
      if (ok) {
        ok = mbar_wait(ring_full(0), 0, abort_flag, a.ws, 0x202);
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
            ok = mbar_wait(q_full, hc & 1, abort_flag, a.ws, 0x203);
            if (!ok) break;
          }
          ok = mbar_wait(s_empty, li & 1, abort_flag, a.ws, 0x204);
          if (!ok) break;
          const int s = int(e % C::NSLOT);
          ok = mbar_wait(ring_full(s), (e / C::NSLOT) & 1, abort_flag, a.ws, 0x205);
          if (!ok) break;
          tc_fence_after();
          issue_S(uint32_t(s));
          umma_commit(s_full);
          umma_commit(ring_empty(s));
          ++e;
          // last S of these prototypes: Q may be replaced once it completes
          const int q_now = nxt.qk;
          nxt.next();
          if (li + 2 >= ntiles || nxt.qk != q_now) umma_commit(q_empty);
        }
        // aggregation of tile li
        ok = mbar_wait(w_full, li & 1, abort_flag, a.ws, 0x206);
        if (!ok) break;
        const int s = int(e % C::NSLOT);
        ok = mbar_wait(ring_full(s), (e / C::NSLOT) & 1, abort_flag, a.ws, 0x207);
        if (!ok) break;
        // segment sc accumulates into buffer sc % NOB, free once the softmax
        // warps have stored the segment that used it last
        const int ob = sc % C::NOB;
        if (cur.seg_first && sc >= C::NOB) {
          ok = mbar_wait(o_empty_of(ob), uint32_t((sc / C::NOB) - 1) & 1u, abort_flag, a.ws, 0x208);
          if (!ok) break;
        }
        tc_fence_after();
        const uint64_t dV = sdesc_add(dV0, uint32_t(s) * C::KV_TILE);
        const uint32_t ocol = tmem + C::O_COL + uint32_t(ob * C::O_COLS);
#pragma unroll
        for (int k = 0; k < T / 16; ++k) {
          const uint32_t acc = (cur.seg_first && k == 0) ? 0u : 1u;
          if (C::TRANS) {
            // O^T[d, p] += sum_t V[t, d] A[t, p]:  A-operand V^T (MN-major), B-operand A (MN-major)
            umma_ss(ocol, sdesc_add(dV, k * 2048), sdesc_add(dW0, k * 2048), idO, acc);
          } else {
#pragma unroll
            for (int mb = 0; mb < PS / 128; ++mb)
              // O[p, d] += sum_t A[t, p] V[t, d]: A-operand A^T (MN-major), B-operand V (MN-major)
              umma_ss(ocol + mb * D, sdesc_add(dW0, mb * 2 * (T * 128) + k * 2048), sdesc_add(dV, k * 2048), idO,
                      acc);
          }
        }
        umma_commit(w_empty);
        umma_commit(ring_empty(s));
        ++e;
        if (cur.seg_last) {
          umma_commit(o_full_of(ob));
          ++sc;
        }
        cur.next();
      }
      // make sure no UMMA is still running when TMEM is released
      umma_commit(drain);
      mbar_wait_bounded(drain, 0, 200000000ull);
    }
  } else if (ntiles > 0) {
    setmaxnreg_inc<kRegsSoft>();
    {
      // ------------------------------------------- softmax + epilogue warps
      const int sw = (warp - kSoftWarp0) >> 2;  // warpgroup: prototype half
      const int q = warp & 3;                   // TMEM lane quadrant
      const int row = 32 * q + lane;            // token within the tile
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * 1.4426950408889634f;  // scale * log2(e)
      float2* stats = reinterpret_cast<float2*>(smem + C::OFF_STATS);
      TileWalker cur(a, tb, te, T);
      int seg_idx = 0;
      bool ok = true;
      // sliced mode: this token's lse, loaded one tile ahead
      float lse_cur = (MODE == kSliced && row < cur.n) ? lse_in[(cur.tok0 + row) * a.H + cur.h] : 0.f;
      // every wait result is made warp-uniform so a timeout never splits a warp
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      // sketch of segment seg_idx (accumulator seg_idx % NOB) waiting to be stored
      float* pend_dst = nullptr;
      auto store_pending = [&]() -> bool {
        const int ob = seg_idx % C::NOB;
        ok = wwait(o_full_of(ob), uint32_t(seg_idx / C::NOB) & 1u, 0x303);
        if (!ok) return false;
        tc_fence_after();
        store_sketch<D, PS, C::TRANS, C::O_COL>(tmem + uint32_t(ob * C::O_COLS), lane_off, sw, q, lane, pend_dst);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(o_empty_of(ob));
        ++seg_idx;
        pend_dst = nullptr;
        return true;
      };
      // pair mode: the peer's R buffer (second half of the stats area) and
      // its barriers, as shared::cluster addresses
      const uint32_t r_peer = PAIR ? mapa_shared(sbase + C::OFF_STATS + C::STATS_R, peer) : 0u;
      const uint32_t r_full_peer = PAIR ? mapa_shared(r_full, peer) : 0u;
      const uint32_t r_used_peer = PAIR ? mapa_shared(r_used, peer) : 0u;
      // (max, sum) of two disjoint prototype sets, a before b
      auto combine = [&](float2 x, float2 y) {
        const float M = fmaxf(x.x, y.x);
        return make_float2(M, x.y * ex2((x.x - M) * c2) + y.y * ex2((y.x - M) * c2));
      };
      for (int li = 0; li < ntiles && ok; ++li) {
        float lse_nxt = 0.f;
        if (MODE == kSliced) {  // next tile's lse, issued before this tile's scores are live
          int64_t t0n;
          int nn, hn;
          cur.peek_next(t0n, nn, hn);
          lse_nxt = row < nn ? lse_in[(t0n + row) * a.H + hn] : 0.f;
        }
        ok = wwait(s_full, li & 1, 0x301);
        if (!ok) break;
        tc_fence_after();
        float v[C::HALF];
#pragma unroll
        for (int c = 0; c < C::HALF / 32; ++c) tmem_ld32(tmem + lane_off + C::S_COL + sw * C::HALF + 32 * c, v + 32 * c);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        // pair mode frees S after the warpgroups have read each other's partials
        // (that orders every write of the partials after the reads of the last)
        if (lane == 0 && !PAIR) mbar_arrive(s_empty);
        const bool valid = row < cur.n;
        const int64_t tok = cur.tok0 + row;
        if (MODE == kFused || MODE == kPair) {
          const float m = row_max<C::HALF>(v);
          const float z = exp2_shift_sum<C::HALF>(v, c2, m * c2);
          float M, Z, f;
          if (PAIR) {
            // Both warpgroups publish their partial (max, sum) at once; both form
            // the CTA's pair from the two in warpgroup order, warpgroup 0 pushes
            // it into the peer CTA (st.async) and both read the peer's push, so
            // the local and the cluster exchange overlap and every thread of the
            // pair ends with bitwise the same (max, sum).  The sums travel as
            // fp16 inside the CTA (a warpgroup's sum lies in [1, 128]).
            float* lm = reinterpret_cast<float*>(smem + C::OFF_STATS);
            __half* lz = reinterpret_cast<__half*>(smem + C::OFF_STATS + C::STATS_Z);
            const float2* rs = reinterpret_cast<const float2*>(smem + C::OFF_STATS + C::STATS_R);
            lm[sw * T + row] = m;
            lz[sw * T + row] = __float2half_rn(z);
            __syncwarp();
            if (lane == 0) mbar_arrive(st_ready);
            ok = wwait(st_ready, li & 1, 0x305);
            if (!ok) break;
            const float2 loc = combine(make_float2(lm[row], __half2float(lz[row])),
                                       make_float2(lm[T + row], __half2float(lz[T + row])));
            __syncwarp();
            if (lane == 0) mbar_arrive(s_empty);
            if (sw == 0) {
              if (li > 0) {
                ok = wwait(r_used, (li - 1) & 1, 0x307);  // the peer has read the last push
                if (!ok) break;
              }
              if (warp == kSoftWarp0 && lane == 0) mbar_arrive_expect_tx(r_full, 8u * T);
              st_async_f2(r_peer + 8u * row, loc, r_full_peer);
            }
            ok = wwait(r_full, li & 1, 0x308);
            if (!ok) break;
            const float2 oth = rs[row];
            __syncwarp();
            if (lane == 0) mbar_arrive_relaxed_cluster(r_used_peer);
            const float2 fin = rank == 0 ? combine(loc, oth) : combine(oth, loc);
            M = fin.x;
            Z = fin.y;
            f = ex2((m - M) * c2) * rcp_approx(Z);
          } else {
            // exchange (max, sum) with the other warpgroup's thread of this token
            if (li > 0) {
              ok = wwait(st_used, (li - 1) & 1, 0x304);
              if (!ok) break;
            }
            stats[sw * T + row] = make_float2(m, z);
            __syncwarp();
            if (lane == 0) mbar_arrive(st_ready);
            ok = wwait(st_ready, li & 1, 0x305);
            if (!ok) break;
            const float2 o = stats[(1 - sw) * T + row];
            __syncwarp();
            if (lane == 0) mbar_arrive(st_used);
            M = fmaxf(m, o.x);
            const float f_self = ex2((m - M) * c2), f_other = ex2((o.x - M) * c2);
            Z = z * f_self + o.y * f_other;
            f = f_self * rcp_approx(Z);
          }
          // rows past the tile's tokens get exact zero weights
          scale_row<C::HALF>(v, valid ? f : 0.f);
          if (rank == 0 && sw == 0 && valid && lse_out) lse_out[tok * a.H + cur.h] = M * a.scale + logf(Z);
        } else {
          exp2_shift<C::HALF>(v, c2, valid ? lse_cur * 1.4426950408889634f : INFINITY);
        }
        if (li > 0) {
          ok = wwait(w_empty, (li - 1) & 1, 0x302);
          if (!ok) break;
        }
        // weights -> shared memory, [PS/64 blocks][128 tokens][64 prototypes], 128-byte swizzle
        uint8_t* wrow = smem + C::OFF_W + row * 128;
#pragma unroll
        for (int k = 0; k < C::HALF / 8; ++k) {
          const int p = sw * C::HALF + 8 * k;
          const int blk = p >> 6, chunk = (p & 63) >> 3;
          uint4 pk;
          pk.x = pack_bf16(v[8 * k + 0], v[8 * k + 1]);
          pk.y = pack_bf16(v[8 * k + 2], v[8 * k + 3]);
          pk.z = pack_bf16(v[8 * k + 4], v[8 * k + 5]);
          pk.w = pack_bf16(v[8 * k + 6], v[8 * k + 7]);
          *reinterpret_cast<uint4*>(wrow + blk * (T * 128) + ((chunk ^ (row & 7)) << 4)) = pk;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(w_full);
        lse_cur = lse_nxt;
        // two accumulators: the segment that ended with the previous tile is
        // stored now, after this tile's weights, so its last aggregation has had
        // a tile's time to finish and the next segment accumulates meanwhile;
        // one accumulator: the segment is stored when it ends (keeping the
        // pointer across tiles cost the softmax registers for no gain)
        if (C::NOB == 2 && pend_dst != nullptr && !store_pending()) break;
        if (cur.seg_last) {
          const bool whole = cur.seg0 >= tb && cur.seg1 <= te;
          pend_dst = whole ? sketch + ((int64_t(cur.b) * a.H + cur.h) * a.P + p0) * D
                           : a.partial + ((int64_t(wk) * 2 + partial_slot(total, W, wk, cur.seg0)) * a.P + p0) * D;
          if (C::NOB == 1 && !store_pending()) break;
        }
        cur.next();
      }
      if (ok && pend_dst != nullptr) store_pending();
    }
  }
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  // the peer may still read this CTA's statistics or arrive on its barriers
  if (PAIR) cluster_sync_all();
}

// ------------------------------------------------------------------ lse only
// Per-token log-sum-exp over NC * NCH prototypes in chunks of NC <= 256 (two
// TMEM buffers of NC columns alternate over (tile, chunk)).  With one slice
// (gridDim.y = 1) these are all P prototypes and the kernel writes lse; with
// gridDim.y = P / (NC * NCH) slices (P = 1024 or 2048: Q of all prototypes
// does not fit shared memory) slice y covers prototypes [y NC NCH, (y+1) NC NCH)
// and writes the token's partial (max of the raw scores, sum of exp2((s - max)
// scale log2 e)), which combine_lse_kernel folds into lse.
template <int D, int NC, int NCH>
struct LseCfg {
  static constexpr int P = NC * NCH;
  static constexpr int KV_TILE = T * D * 2;
  static constexpr int Q_BYTES = P * D * 2;
  static constexpr int NSLOT = (Q_BYTES + 4 * KV_TILE <= 200 * 1024) ? 4 : 3;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_RING = Q_BYTES;
  static constexpr int OFF_STATS = OFF_RING + NSLOT * KV_TILE;
  static constexpr int OFF_BAR = OFF_STATS + 2 * T * 8;
  static constexpr int NBAR = 2 * NSLOT + 9;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = OFF_MISC + 16;
  static constexpr int TMEM_COLS = tmem_cols_for(2 * NC);
  static constexpr int HALF = NC / 2;
};

template <int D, int NC, int NCH>
__global__ void __launch_bounds__(kThreads, 1)
    tc_lse_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ, Args a,
                  float* __restrict__ lse_out, float2* __restrict__ part_out) {
  using C = LseCfg<D, NC, NCH>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ws_failed(a.ws)) return;
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ws_set_error(a.ws, SA_ERR_CUDA, 0xA12u);
    return;
  }
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + C::OFF_Q, sRing = sbase + C::OFF_RING;
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto ring_full = [&](int s) { return bar0 + 8u * s; };
  auto ring_empty = [&](int s) { return bar0 + 8u * (C::NSLOT + s); };
  const uint32_t q_full = bar0 + 8u * (2 * C::NSLOT), q_empty = q_full + 8, s_full0 = q_full + 16,
                 s_empty0 = q_full + 32, drain = q_full + 48, st_ready = q_full + 56, st_used = q_full + 64;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int64_t tph = reinterpret_cast<const WsHeader*>(a.ws)->tiles_per_head;
  const int64_t total = tph * a.H;
  const int W = gridDim.x, wk = blockIdx.x;
  const int NS = gridDim.y, slice = blockIdx.y;  // prototype slices of C::P
  const int pb = slice * C::P;
  const int64_t tb = range_begin(total, W, wk), te = range_begin(total, W, wk + 1);
  const int ntiles = int(te - tb);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(ring_full(s), 1);
      mbar_init(ring_empty(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    mbar_init(s_full0, 1);
    mbar_init(s_full0 + 8, 1);
    mbar_init(s_empty0, kSoftWarps);
    mbar_init(s_empty0 + 8, kSoftWarps);
    mbar_init(drain, 1);
    mbar_init(st_ready, kSoftWarps);
    mbar_init(st_used, kSoftWarps);
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
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmQ);
      TileWalker it(a, tb, te, T);
      int hc = 0, prev_h = -1;
      uint32_t e = 0;
      bool ok = true;
      for (int li = 0; li < ntiles && ok; ++li) {
        if (it.qk != prev_h) {
          if (hc > 0) ok = mbar_wait(q_empty, (hc - 1) & 1, abort_flag, a.ws, 0x111);
          if (!ok) break;
          mbar_arrive_expect_tx(q_full, C::Q_BYTES);
#pragma unroll
          for (int c = 0; c < NCH; ++c)
#pragma unroll
            for (int dh = 0; dh < D / 64; ++dh)
              tma_load_3d(sQ + dh * C::P * 128 + c * NC * 128, &tmQ, q_full, 64 * dh, pb + c * NC, it.qk);
          prev_h = it.qk;
          ++hc;
        }
        const int s = int(e % C::NSLOT);
        if (e >= uint32_t(C::NSLOT)) ok = mbar_wait(ring_empty(s), ((e / C::NSLOT) + 1) & 1, abort_flag, a.ws, 0x112);
        if (!ok) break;
        mbar_arrive_expect_tx(ring_full(s), C::KV_TILE);
#pragma unroll
        for (int dh = 0; dh < D / 64; ++dh)
          tma_load_3d(sRing + s * C::KV_TILE + dh * T * 128, &tmK, ring_full(s), 64 * dh, it.h, int(it.tok0));
        ++e;
        it.next();
      }
      if (!ok) {
        for (uint32_t k = (e > uint32_t(C::NSLOT) ? e - C::NSLOT : 0); k < e; ++k)
          mbar_wait_bounded(ring_full(int(k % C::NSLOT)), (k / C::NSLOT) & 1, 200000000ull);
      }
    } else if (warp == 1 && lane == 0) {
      constexpr uint32_t idS = idesc_bf16(128, NC, 0, 0);
      TileWalker cur(a, tb, te, T);
      int hc = 0, prev_h = -1;
      bool ok = true;
      uint32_t g = 0;  // (tile, chunk) counter
      for (int li = 0; li < ntiles && ok; ++li) {
        const int h_now = cur.qk;
        if (h_now != prev_h) {
          prev_h = h_now;
          ok = mbar_wait(q_full, hc & 1, abort_flag, a.ws, 0x211);
          ++hc;
          if (!ok) break;
        }
        const int s = int(uint32_t(li) % C::NSLOT);
        ok = mbar_wait(ring_full(s), (uint32_t(li) / C::NSLOT) & 1, abort_flag, a.ws, 0x212);
        if (!ok) break;
        const uint32_t kaddr = sRing + s * C::KV_TILE;
        for (int c = 0; c < NCH && ok; ++c, ++g) {
          const int buf = int(g & 1);
          if (g >= 2) ok = mbar_wait(s_empty0 + 8 * buf, ((g >> 1) + 1) & 1, abort_flag, a.ws, 0x213);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint64_t ad = sdesc(kaddr + (k >> 2) * (T * 128) + (k & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc(sQ + (k >> 2) * (C::P * 128) + c * NC * 128 + (k & 3) * 32, 16, 1024);
            umma_ss(tmem + buf * NC, ad, bd, idS, k > 0 ? 1u : 0u);
          }
          umma_commit(s_full0 + 8 * buf);
        }
        if (!ok) break;
        umma_commit(ring_empty(s));
        cur.next();
        if (li + 1 >= ntiles || cur.qk != h_now) umma_commit(q_empty);
      }
      umma_commit(drain);
      mbar_wait_bounded(drain, 0, 200000000ull);
    } else if (warp >= kSoftWarp0) {
      const int sw = (warp - kSoftWarp0) >> 2, q = warp & 3, row = 32 * q + lane;
      const uint32_t lane_off = uint32_t(32 * q) << 16;
      const float c2 = a.scale * 1.4426950408889634f;
      float2* stats = reinterpret_cast<float2*>(smem + C::OFF_STATS);
      TileWalker cur(a, tb, te, T);
      bool ok = true;
      uint32_t g = 0;
      auto wwait = [&](uint32_t bar, uint32_t par, uint32_t site) {
        return __all_sync(0xffffffffu, mbar_wait(bar, par, abort_flag, a.ws, site));
      };
      for (int li = 0; li < ntiles && ok; ++li) {
        float m = -INFINITY, z = 0.f;
        for (int c = 0; c < NCH && ok; ++c, ++g) {
          const int buf = int(g & 1);
          ok = wwait(s_full0 + 8 * buf, (g >> 1) & 1, 0x311);
          if (!ok) break;
          tc_fence_after();
          float v[C::HALF];
#pragma unroll
          for (int k = 0; k < C::HALF / 32; ++k) tmem_ld32(tmem + lane_off + buf * NC + sw * C::HALF + 32 * k, v + 32 * k);
          tmem_ld_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(s_empty0 + 8 * buf);
          float mm = v[0];
#pragma unroll
          for (int j = 1; j < C::HALF; ++j) mm = fmaxf(mm, v[j]);
          const float M = fmaxf(m, mm), Mc = M * c2;
          float zz = 0.f;
#pragma unroll
          for (int j = 0; j < C::HALF; ++j) zz += ex2(fmaf(v[j], c2, -Mc));
          z = z * ex2((m - M) * c2) + zz;
          m = M;
        }
        if (!ok) break;
        if (li > 0) {
          ok = wwait(st_used, (li - 1) & 1, 0x312);
          if (!ok) break;
        }
        stats[sw * T + row] = make_float2(m, z);
        __syncwarp();
        if (lane == 0) mbar_arrive(st_ready);
        ok = wwait(st_ready, li & 1, 0x313);
        if (!ok) break;
        const float2 o = stats[(1 - sw) * T + row];
        __syncwarp();
        if (lane == 0) mbar_arrive(st_used);
        if (sw == 0 && row < cur.n) {
          const float M = fmaxf(m, o.x);
          const float Z = z * ex2((m - M) * c2) + o.y * ex2((o.x - M) * c2);
          const int64_t th = (cur.tok0 + row) * a.H + cur.h;
          if (NS == 1)
            lse_out[th] = M * a.scale + logf(Z);
          else
            part_out[th * NS + slice] = make_float2(M, Z);
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

// ------------------------------------------------------------- host side
template <int D, int PS, int MODE>
static cudaError_t launch_fwd_t(const Args& a, int W, float* sketch, float* lse_out, const float* lse_in,
                                cudaStream_t st) {
  using C = Cfg<D, PS, MODE>;
  CUtensorMap tk, tv, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_kv_map(&tv, a.V, a.N, a.H, D) ||
      !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, PS))
    return cudaErrorInvalidValue;
  auto fn = &tc_fwd_kernel<D, PS, MODE>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  if (MODE == kPair) {
    // one cluster of two CTAs per worker; CTA rank r holds prototypes [PS r, PS r + PS)
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
    return cudaLaunchKernelEx(&cfg, fn, tk, tv, tq, a, sketch, lse_out, lse_in);
  }
  dim3 grid(W, a.P / PS);
  fn<<<grid, kThreads, C::SMEM, st>>>(tk, tv, tq, a, sketch, lse_out, lse_in);
  return cudaGetLastError();
}

template <int D, int NC, int NCH>
static cudaError_t launch_lse_t(const Args& a, int W, float* lse_out, float2* part, cudaStream_t st) {
  using C = LseCfg<D, NC, NCH>;
  CUtensorMap tk, tq;
  if (!make_kv_map(&tk, a.K, a.N, a.H, D) || !make_q_map(&tq, a.Q, a.uq ? a.B * a.H : a.H, a.P, D, NC))
    return cudaErrorInvalidValue;
  auto fn = &tc_lse_kernel<D, NC, NCH>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int NS = a.P / C::P;
  dim3 grid(NS > 1 ? (W / NS > 0 ? W / NS : 1) : W, NS);
  fn<<<grid, kThreads, C::SMEM, st>>>(tk, tq, a, lse_out, part);
  return cudaGetLastError();
}

// lse[t, h] from the NS per-slice partials (max, sum), folded in slice order.
__global__ void combine_lse_kernel(const float2* __restrict__ part, int NS, int64_t nth, float scale,
                                   float* __restrict__ lse, const void* ws) {
  if (ws_failed(ws)) return;
  const float c2 = scale * 1.4426950408889634f;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < nth; i += int64_t(gridDim.x) * blockDim.x) {
    float2 acc = part[i * NS];
    for (int k = 1; k < NS; ++k) {
      const float2 y = part[i * NS + k];
      const float M = fmaxf(acc.x, y.x);
      acc = make_float2(M, acc.y * ex2((acc.x - M) * c2) + y.y * ex2((y.x - M) * c2));
    }
    lse[i] = acc.x * scale + logf(acc.y);
  }
}

}  // namespace tcf

// Shapes served by the tensor-core forward: bf16, d in {64, 128}, P in
// {128, 256} (one CTA holds all prototypes), P = 512 (a cluster pair) or
// P in {1024, 2048} (sliced lse pass, then 256-prototype slices).
bool tc_fwd_supported(int P, int d, sa_dtype dt) {
  if (dt != SA_BF16 || (d != 64 && d != 128)) return false;
  if (P != 128 && P != 256 && P != 512 && P != 1024 && P != 2048) return false;
  return tcc::device_is_sm103() && tc_path_enabled();
}

// Prototypes per slice of the lse pass (Q of one slice resident in shared memory).
int tc_lse_slice(int P, int d) {
  const int cap = d == 128 ? 512 : 1024;
  return P < cap ? P : cap;
}

// By default every supported shape normalises inside the forward kernel:
// P <= 256 in one CTA, P = 512 in a cluster pair.  Path 2 of sa_select_path
// runs P = 512 (and P = 256 with d = 128) as a per-token lse pass followed by
// 256-prototype slices that take that lse -- the same result computed another
// way, kept as a cross-check.
bool tc_fwd_needs_lse_pass_d(int P, int d) {
  return P >= 1024 || (tc_fwd_sliced_selected() && (P == 512 || (P == 256 && d == 128)));
}

const char* tc_fwd_name(int P, int d) {
  if (tc_fwd_needs_lse_pass_d(P, d)) return d == 128 ? "tc_fwd_kernel<128,256,sliced>" : "tc_fwd_kernel<64,256,sliced>";
  if (P == 512 && !tc_narrow_selected()) return d == 128 ? "tc_fwd_wide_kernel<128>" : "tc_fwd_wide_kernel<64>";
  if (P == 512) return d == 128 ? "tc_fwd_kernel<128,256,pair>" : "tc_fwd_kernel<64,256,pair>";
  if (P == 256) return d == 128 ? "tc_fwd_kernel<128,256,fused>" : "tc_fwd_kernel<64,256,fused>";
  return d == 128 ? "tc_fwd_kernel<128,128,fused>" : "tc_fwd_kernel<64,128,fused>";
}

int tc_tile_tokens() { return tcc::T; }

int tc_fwd_workers(int num_sms, int P, int) {
  const int slices = P > 256 ? P / 256 : 1;
  const int w = num_sms / slices;
  return w < 1 ? 1 : w;
}

cudaError_t launch_tc_lse(const Args& a, float* lse, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  const int W = tcc::device_sm_count();
  cudaError_t e = cudaErrorInvalidValue;
  if (a.d == 128) {
    if (a.P >= 512) e = tcf::launch_lse_t<128, 256, 2>(a, W, lse, a.lse_part, st);
    else if (a.P == 256) e = tcf::launch_lse_t<128, 256, 1>(a, W, lse, a.lse_part, st);
    else if (a.P == 128) e = tcf::launch_lse_t<128, 128, 1>(a, W, lse, a.lse_part, st);
  } else {
    if (a.P >= 1024) e = tcf::launch_lse_t<64, 256, 4>(a, W, lse, a.lse_part, st);
    else if (a.P == 512) e = tcf::launch_lse_t<64, 256, 2>(a, W, lse, a.lse_part, st);
    else if (a.P == 256) e = tcf::launch_lse_t<64, 256, 1>(a, W, lse, a.lse_part, st);
    else if (a.P == 128) e = tcf::launch_lse_t<64, 128, 1>(a, W, lse, a.lse_part, st);
  }
  if (e != cudaSuccess) return e;
  const int NS = a.P / tc_lse_slice(a.P, a.d);
  if (NS > 1) {
    tcf::combine_lse_kernel<<<1024, 256, 0, st>>>(a.lse_part, NS, a.N * a.H, a.scale, lse, a.ws);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t launch_tc_fwd(const Args& a, int W, float* sketch, float* lse, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  using namespace tcf;
  if (tc_fwd_needs_lse_pass_d(a.P, a.d))  // lse (from launch_tc_lse beforehand) is an input here
    return a.d == 128 ? launch_fwd_t<128, 256, kSliced>(a, W, sketch, nullptr, lse, st)
                      : launch_fwd_t<64, 256, kSliced>(a, W, sketch, nullptr, lse, st);
  if (a.P == 512 && !tc_narrow_selected()) return launch_tc_fwd_wide(a, W, sketch, lse, st);
  if (a.P == 512)
    return a.d == 128 ? launch_fwd_t<128, 256, kPair>(a, W, sketch, lse, nullptr, st)
                      : launch_fwd_t<64, 256, kPair>(a, W, sketch, lse, nullptr, st);
  if (a.P == 256)
    return a.d == 128 ? launch_fwd_t<128, 256, kFused>(a, W, sketch, lse, nullptr, st)
                      : launch_fwd_t<64, 256, kFused>(a, W, sketch, lse, nullptr, st);
  return a.d == 128 ? launch_fwd_t<128, 128, kFused>(a, W, sketch, lse, nullptr, st)
                    : launch_fwd_t<64, 128, kFused>(a, W, sketch, lse, nullptr, st);
}

}  // namespace sa
