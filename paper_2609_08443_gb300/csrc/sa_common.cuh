// Shared definitions of libsa_sketch: workspace layout, the ragged tiling and
// small device helpers.  Used by the host API and by every kernel.
//
// Ragged tiling ("ragged batching", paper Sec. 4.4): user b contributes
// ceil(L_b / T) tiles of T tokens per head.  The global tile list is ordered
// (head, user, tile); worker w of W owns the contiguous tile range
// [begin(w), begin(w+1)) with begin(w) = floor(total * w / W), so every worker
// gets the same number of tiles to within one.  A (user, head) segment that
// falls entirely inside one worker's range is finished by that worker; a
// segment cut by range boundaries leaves one fp32 partial per worker, and a
// finalize kernel adds them in worker order, which makes the result bitwise
// reproducible for a given W.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "../../include/sa_sketch.h"

#define SA_HD __host__ __device__ __forceinline__

namespace sa {

constexpr int kMaxP = 2048;
constexpr int kMaxD = 128;
constexpr int kMaxH = 64;

// ---------------------------------------------------------------- workspace
struct WsHeader {
  uint32_t err;           // sa_status written by device code (0 = OK)
  uint32_t pad0;
  int64_t tiles_per_head; // sum_b ceil(L_b / T) for the plan of this call
  uint32_t timeout_site;  // where a bounded wait gave up (diagnostics)
  uint32_t pad1;
  uint64_t wait_limit_ns; // limit of every bounded pipeline wait of this call
  uint32_t pad2[56];
};
static_assert(sizeof(WsHeader) == 256, "header is one 256-byte line");

SA_HD size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Byte offsets of the workspace sections for one call.
struct WsLayout {
  size_t tile_prefix;  // int64 [B + 1]: per-head tile prefix over users
  size_t partial;      // fp32 [W][2][P][d]: sketch pieces of cut segments
  size_t dq_partial;   // fp32 [W][H][P][d]: per-worker dQ per head (bwd)
  size_t lse;          // fp32 [N][H]: lse scratch when the caller passes none
  size_t dcoef;        // fp32 [N][H]: D_i = dV_i . v_i (bwd)
  size_t gbf;          // bf16 [B][H][P][d]: dsketch copy streamed by TMA (split backward)
  size_t lse_part;     // float2 [N][H][P / 512]: per-slice (max, sum) of the lse pass (P >= 1024)
  size_t qneg;         // [H][P][d] (4 bytes per element reserved): -Q, for a negative scale
  size_t total;
};

SA_HD WsLayout ws_layout(int B, int64_t N, int H, int P, int d, int W, bool bwd) {
  WsLayout L{};
  size_t off = sizeof(WsHeader);
  L.tile_prefix = off;
  off = align256(off + sizeof(int64_t) * size_t(B + 1));
  L.partial = off;
  off = align256(off + sizeof(float) * size_t(W) * 2 * size_t(P) * size_t(d));
  L.dq_partial = off;
  if (bwd) off = align256(off + sizeof(float) * size_t(W) * size_t(H) * size_t(P) * size_t(d));
  L.lse = off;
  off = align256(off + sizeof(float) * size_t(N) * size_t(H));
  L.dcoef = off;
  if (bwd) off = align256(off + sizeof(float) * size_t(N) * size_t(H));
  L.gbf = off;
  if (bwd && ((d == 128 && P > 128) || (d == 64 && P > 256)))
    off = align256(off + 2 * size_t(B) * size_t(H) * size_t(P) * size_t(d));
  L.lse_part = off;
  if (P >= 1024) off = align256(off + 8 * size_t(N) * size_t(H) * size_t((P + 511) / 512));
  L.qneg = off;
  off = align256(off + 4 * size_t(H) * size_t(P) * size_t(d));
  L.total = off;
  return L;
}

// ------------------------------------------------------------------ tiling
SA_HD int64_t range_begin(int64_t total, int W, int w) { return (total * int64_t(w)) / W; }

// Largest worker w with range_begin(w) <= t (so a worker with an empty range
// never owns a tile).  0 <= t < total.
SA_HD int owner_of(int64_t total, int W, int64_t t) {
  int64_t g = (t * int64_t(W)) / (total > 0 ? total : 1);
  if (g >= W) g = W - 1;
  while (g + 1 < W && range_begin(total, W, int(g + 1)) <= t) ++g;
  while (g > 0 && range_begin(total, W, int(g)) > t) --g;
  return int(g);
}

// Largest b in [0, B) with prefix[b] <= r (prefix non-decreasing, prefix[0]=0,
// r < prefix[B]); skips users with no tiles.
SA_HD int find_user(const int64_t* prefix, int B, int64_t r) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (prefix[mid] <= r) lo = mid; else hi = mid - 1;
  }
  return lo;
}

struct TileRef {
  int h;          // head
  int b;          // user
  int64_t tok0;   // first token row of the tile
  int n;          // tokens in the tile (1..T)
  int64_t seg0;   // global index of the segment's first tile
  int64_t seg1;   // one past the segment's last tile
  int64_t L;      // the user's tokens
};

SA_HD TileRef locate_tile(int64_t t, int64_t tph, const int64_t* prefix, const int32_t* cu,
                          int B, int T) {
  TileRef r;
  r.h = int(t / tph);
  int64_t rem = t - int64_t(r.h) * tph;
  r.b = find_user(prefix, B, rem);
  int64_t k = rem - prefix[r.b];
  int64_t L = int64_t(cu[r.b + 1]) - int64_t(cu[r.b]);
  r.tok0 = int64_t(cu[r.b]) + k * T;
  r.L = L;
  int64_t left = L - k * T;
  r.n = int(left < T ? left : T);
  r.seg0 = int64_t(r.h) * tph + prefix[r.b];
  r.seg1 = int64_t(r.h) * tph + prefix[r.b + 1];
  return r;
}

// locate_tile for tile t, the first tile of the segment that follows segment
// (h_prev, b_prev) in the tile order.  The user is found by a short forward
// scan from b_prev + 1 (or from 0 in a new head) instead of a binary search:
// consecutive segments are consecutive non-empty users, so the scan usually
// takes one step.  The answer is accepted only where it meets find_user's
// definition (prefix[b] <= r < prefix[b + 1]); a long run of empty users
// falls back to the search.
SA_HD TileRef locate_next_segment(int64_t t, int h_prev, int b_prev, int64_t tph, const int64_t* prefix,
                                  const int32_t* cu, int B, int T) {
  const int h = int(t / tph);
  const int64_t rem = t - int64_t(h) * tph;
  int c = h == h_prev ? b_prev + 1 : 0;
  if (c >= B) c = B - 1;
  for (int steps = 0; steps < 8 && c + 1 < B && prefix[c + 1] <= rem; ++steps) ++c;
  if (!(prefix[c] <= rem && (c + 1 >= B || prefix[c + 1] > rem))) return locate_tile(t, tph, prefix, cu, B, T);
  TileRef r;
  r.h = h;
  r.b = c;
  const int64_t k = rem - prefix[c];
  const int64_t cb = int64_t(cu[c]), L = int64_t(cu[c + 1]) - cb;
  r.tok0 = cb + k * T;
  r.L = L;
  const int64_t left = L - k * T;
  r.n = int(left < T ? left : T);
  r.seg0 = int64_t(h) * tph + prefix[c];
  r.seg1 = int64_t(h) * tph + prefix[c + 1];
  return r;
}

// Which of worker w's two partial slots holds its piece of segment [s0, s1):
// slot 0 if the piece is the first piece of w's range, slot 1 otherwise.
SA_HD int partial_slot(int64_t total, int W, int w, int64_t seg0) {
  return range_begin(total, W, w) >= seg0 ? 0 : 1;
}

// ---------------------------------------------------------- device helpers
#ifdef __CUDACC__
template <typename T> __device__ __forceinline__ float ld_f32(const T* p);
template <> __device__ __forceinline__ float ld_f32<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ld_f32<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}
template <typename T> __device__ __forceinline__ void st_from_f32(T* p, float v);
template <> __device__ __forceinline__ void st_from_f32<float>(float* p, float v) { *p = v; }
template <> __device__ __forceinline__ void st_from_f32<__nv_bfloat16>(__nv_bfloat16* p, float v) {
  *p = __float2bfloat16_rn(v);
}

__device__ __forceinline__ WsHeader* ws_header(void* ws) { return reinterpret_cast<WsHeader*>(ws); }
__device__ __forceinline__ bool ws_failed(const void* ws) {
  return *reinterpret_cast<const volatile uint32_t*>(ws) != 0u;
}
__device__ __forceinline__ void ws_set_error(void* ws, uint32_t code, uint32_t site) {
  WsHeader* h = ws_header(ws);
  if (atomicCAS(&h->err, 0u, code) == 0u) h->timeout_site = site;
}
#endif

}  // namespace sa
