// Thin inline-PTX layer for sm_103a: mbarriers with bounded waits, TMA tensor
// loads, tcgen05 (TMEM allocation, UMMA issue/commit, TMEM loads) and the
// shared-memory / instruction descriptors of tcgen05.mma kind::f16.
#pragma once
#include <cstdint>
#include <cuda.h>

#include "sa_common.cuh"

namespace sa {
namespace ptx {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Every wait in the tensor-core kernels is bounded: after the call's limit
// (the workspace header's wait_limit_ns, 2 s unless a test lowers it) the
// waiting thread raises the CTA's abort flag and records SA_ERR_TIMEOUT in the
// workspace; threads that see the flag stop waiting too.  A correct pipeline
// never gets near the limit.
//
// Each CTA keeps two control words in shared memory, reached through the
// `abort_flag` pointer every wait takes: abort_flag[0] is the abort flag and
// abort_flag[2] the limit in nanoseconds, copied from the workspace header by
// wait_ctl_init when the CTA starts (abort_flag[1] is left to the kernel).

__device__ __forceinline__ void wait_ctl_init(volatile int* abort_flag, const void* ws) {
  const uint64_t ns = reinterpret_cast<const WsHeader*>(ws)->wait_limit_ns;
  abort_flag[0] = 0;
  reinterpret_cast<volatile uint32_t*>(abort_flag)[2] = ns > 0xFFFFFFFFull ? 0xFFFFFFFFu : uint32_t(ns);
}

// Limits below this are test settings (sa_set_wait_limit_ns): kernels that
// support a forced timeout then wait on a barrier that nothing completes, so
// the limit runs out however fast the rest of the pipeline is.
constexpr uint32_t kPollLimitNs = 1000000u;  // 1 ms

__device__ __forceinline__ uint32_t ctl_wait_limit(volatile int* abort_flag) {
  return reinterpret_cast<volatile const uint32_t*>(abort_flag)[2];
}

__device__ __forceinline__ bool mbar_wait_timed_out(volatile int* abort_flag, void* ws, uint32_t site, uint64_t t0) {
  if (globaltimer() - t0 <= ctl_wait_limit(abort_flag)) return false;
  *abort_flag = 1;
  ws_set_error(ws, SA_ERR_TIMEOUT, site);
  return true;
}

// The flag and the clock are checked every 64 polls, so a handoff that is
// ready after a few polls costs nothing beyond the polls themselves.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, void* ws,
                                          uint32_t site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63u) == 0u) {
      if (*abort_flag) return false;
      if (mbar_wait_timed_out(abort_flag, ws, site, t0)) return false;
    }
  }
}

// ------------------------------------------------------------ CTA clusters
// Rank of this CTA in its cluster, the shared::cluster address of the same
// shared-memory offset in CTA `rank`, and the cluster-scope forms of the
// mbarrier operations used when two CTAs exchange per-token statistics.
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// arrive (release at cluster scope) on an mbarrier of this CTA or of a peer;
// `bar_cl` is a shared::cluster address (from mapa_shared)
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cl) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cl) : "memory");
}
// arrive without ordering prior memory operations (the peer only learns that
// values this thread already consumed may be overwritten)
__device__ __forceinline__ void mbar_arrive_relaxed_cluster(uint32_t bar_cl) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cl) : "memory");
}
// 8-byte store into a peer's shared memory that completes `bytes` of the
// transaction count of the peer's mbarrier `bar_cl` (no release fence needed:
// the data is visible to whoever observes that barrier phase complete)
__device__ __forceinline__ void st_async_f2(uint32_t dst_cl, float2 v, uint32_t bar_cl) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(dst_cl),
               "f"(v.x), "f"(v.y), "r"(bar_cl)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ float2 ld_cluster_f2(uint32_t addr_cl) {
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr_cl) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_cluster_u32(uint32_t addr_cl) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr_cl) : "memory");
  return v;
}
// Every thread of every CTA of the cluster must execute this (all CTAs of a
// cluster are resident together, so it completes once all have arrived).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Bounded wait with acquire at cluster scope (peers' writes become visible).
__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity, volatile int* abort_flag, void* ws,
                                                  uint32_t site) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 63u) == 0u) {
      if (*abort_flag) return false;
      if (mbar_wait_timed_out(abort_flag, ws, site, t0)) return false;
    }
  }
}

// ----------------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_prefetch_desc(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tmap, uint32_t bar, int c0, int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

// Pull a tile into L2 ahead of its shared-memory load (no completion tracking).
__device__ __forceinline__ void tma_prefetch_l2_3d(const void* tmap, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global [%0, {%1, %2, %3}];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(c0), "r"(c1), "r"(c2)
               : "memory");
}

// Shared -> global tile store (rows outside the tensor are not written).
__device__ __forceinline__ void tma_store_3d(const void* tmap, uint32_t src, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(src), "r"(c0), "r"(c1), "r"(c2)
               : "memory");
}
__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Wait until the shared-memory source of every committed bulk store was read.
__device__ __forceinline__ void bulk_wait_read_all() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// Wait until every committed bulk store has completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ------------------------------------------------------------------ tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem], kind::f16 (bf16 inputs, fp32 accumulate).
// No "memory" clobber: the issuing thread touches no memory the MMA reads, and
// volatile asm keeps its order against the mbarrier waits and tcgen05 fences,
// so the compiler can keep addresses and descriptors in registers between
// issues (an issue must cost far less than the 64 cycles of a 128x128x16 MMA).
__device__ __forceinline__ void umma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}
// D[tmem] (+)= A[tmem] * B[smem]: A is M x K with M on TMEM lanes and two bf16
// values per 32-bit column (lower K index in the low half).
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate));
}
// mbarrier arrives once every tcgen05 op issued so far by this thread is done
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp gets lane
// (quadrant base + i), columns col .. col+31.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 lanes x 16 consecutive 32-bit columns from registers into TMEM.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
      "%14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// ------------------------------------------------------------- descriptors
// Shared-memory matrix descriptor of tcgen05 (128-byte swizzle, version 1).
//   K-major operand: rows of 64 bf16 (128 B), 8-row atoms of 1024 B,
//     SBO = distance between 8-row groups, LBO unused.
//   MN-major operand: 64 MN-elements per 128-B row, one row per K index,
//     8 K-rows per 1024-B atom; LBO = distance between 64-element MN blocks,
//     SBO = distance between 8-row K groups.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= uint64_t((saddr & 0x3FFFFu) >> 4);
  d |= uint64_t((lbo_bytes & 0x3FFFFu) >> 4) << 16;
  d |= uint64_t((sbo_bytes & 0x3FFFFu) >> 4) << 32;
  d |= uint64_t(1) << 46;  // descriptor version for tcgen05
  d |= uint64_t(2) << 61;  // 128-byte swizzle
  return d;
}

// The same descriptor with its start address moved by `bytes` (a multiple of
// 16; the 14-bit address field cannot overflow inside 228 KB of shared memory).
__host__ __device__ __forceinline__ uint64_t sdesc_add(uint64_t desc, uint32_t bytes) {
  return desc + uint64_t(bytes >> 4);
}

// Instruction descriptor, kind::f16: bf16 A and B, fp32 D; a_mn / b_mn select
// MN-major (1) or K-major (0) operands.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, int a_mn, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(a_mn) << 15) | (uint32_t(b_mn) << 16) |
         (uint32_t(N >> 3) << 17) | (uint32_t(M >> 4) << 24);
}

// hardware approximate reciprocal (one MUFU operation; the weights it scales
// are rounded to bf16 afterwards)
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ------------------------------------------- per-thread softmax arithmetic
// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// max of v[0..N) with four independent chains (N a multiple of 8)
template <int N>
__device__ __forceinline__ float row_max(const float* v) {
  static_assert(N % 8 == 0, "row_max works on multiples of 8 values");
  float a0 = fmaxf(v[0], v[1]), a1 = fmaxf(v[2], v[3]), a2 = fmaxf(v[4], v[5]), a3 = fmaxf(v[6], v[7]);
#pragma unroll
  for (int j = 8; j < N; j += 8) {
    a0 = fmax3(a0, v[j], v[j + 1]);
    a1 = fmax3(a1, v[j + 2], v[j + 3]);
    a2 = fmax3(a2, v[j + 4], v[j + 5]);
    a3 = fmax3(a3, v[j + 6], v[j + 7]);
  }
  return fmaxf(fmax3(a0, a1, a2), a3);
}

// v[j] <- 2^(v[j] * c2 - sh) (one fused multiply-add per value, two values per
// instruction); returns the sum of the results, accumulated in four chains.
template <int N>
__device__ __forceinline__ float exp2_shift_sum(float* v, float c2, float sh) {
  static_assert(N % 4 == 0, "exp2_shift_sum works on multiples of 4 values");
  const float2 cc = make_float2(c2, c2), ns = make_float2(-sh, -sh);
  float2 z0 = make_float2(0.f, 0.f), z1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int j = 0; j < N; j += 4) {
    float2 x0 = __ffma2_rn(make_float2(v[j], v[j + 1]), cc, ns);
    float2 x1 = __ffma2_rn(make_float2(v[j + 2], v[j + 3]), cc, ns);
    x0.x = ex2(x0.x);
    x0.y = ex2(x0.y);
    x1.x = ex2(x1.x);
    x1.y = ex2(x1.y);
    v[j] = x0.x;
    v[j + 1] = x0.y;
    v[j + 2] = x1.x;
    v[j + 3] = x1.y;
    z0 = __fadd2_rn(z0, x0);
    z1 = __fadd2_rn(z1, x1);
  }
  return (z0.x + z0.y) + (z1.x + z1.y);
}

// v[j] <- 2^(v[j] * c2 - sh), no sum (sh = +inf gives exact zeros)
template <int N>
__device__ __forceinline__ void exp2_shift(float* v, float c2, float sh) {
  const float2 cc = make_float2(c2, c2), ns = make_float2(-sh, -sh);
#pragma unroll
  for (int j = 0; j < N; j += 2) {
    float2 x = __ffma2_rn(make_float2(v[j], v[j + 1]), cc, ns);
    v[j] = ex2(x.x);
    v[j + 1] = ex2(x.y);
  }
}

// v[j] <- v[j] * f, two values per instruction
template <int N>
__device__ __forceinline__ void scale_row(float* v, float f) {
  const float2 ff = make_float2(f, f);
#pragma unroll
  for (int j = 0; j < N; j += 2) {
    const float2 x = __fmul2_rn(make_float2(v[j], v[j + 1]), ff);
    v[j] = x.x;
    v[j + 1] = x.y;
  }
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Per-warpgroup register budget (all 128 threads of the warpgroup execute it).
// A kernel launched with R registers per thread may redistribute them among its
// warpgroups as long as the new budgets sum to at most threads x R.
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

}  // namespace ptx
}  // namespace sa
