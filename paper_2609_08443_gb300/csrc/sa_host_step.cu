// The training step (forward and backward of paper Sec. 3.1) on a batch that
// lives in host memory: users are grouped into chunks of about `chunk_tokens`
// tokens, and three streams overlap the host-to-device copy of one chunk, the
// step on the previous chunk and the device-to-host copy of the one before:
//
//   copy-in  : K, V, dsketch rows of chunk c -> staging buffer c % 2
//   compute  : sa_sketch_fwd + sa_sketch_bwd on the staging buffer; the chunk's
//              dQ is added into one fp32 accumulator in chunk order
//   copy-out : sketch, dK, dV rows of chunk c -> the caller's host arrays
//
// A staging buffer holds a chunk's inputs (K, V, dsketch) and, apart from
// them, its outputs and step workspace.  The step is the last reader of the
// inputs and the copy-out the last reader of the outputs, so a chunk's copy-in
// waits only for the step of the chunk that last used its buffer, and its step
// waits for that chunk's copy-out: the copy-in of chunk c + 2 runs beside the
// copy-out of chunk c, and the copies, not copy + step + copy, set the pace.
// dQ reaches the host after the last chunk.  The caller's
// stream waits for everything before the call returns, so synchronising it
// means the host outputs are complete.  With page-locked host arrays the
// copies run asynchronously; pageable arrays work but serialise the copies.
#include <mutex>
#include <vector>

#include "sa_kernels.cuh"

namespace sa {

// Keeps the first non-zero error word of a chunk's step workspace.
__global__ void sticky_error_kernel(const uint32_t* __restrict__ src, uint32_t* __restrict__ dst) {
  const uint32_t e = *reinterpret_cast<const volatile uint32_t*>(src);
  if (e != 0u && *dst == 0u) *dst = e;
}

}  // namespace sa

namespace {

struct StepStreams {
  cudaStream_t in = nullptr, cmp = nullptr, out = nullptr;
  cudaEvent_t entry = nullptr, fin = nullptr, in_done[2] = {}, cmp_done[2] = {}, out_done[2] = {};
  bool ready = false;
};

std::mutex g_step_mu;
StepStreams g_step[64];

// Streams and events of the pipeline on the current device, created on first use.
sa_status step_streams(StepStreams** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SA_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_step_mu);
  StepStreams& s = g_step[dev];
  if (!s.ready) {
    const unsigned sf = cudaStreamNonBlocking, ef = cudaEventDisableTiming;
    if (cudaStreamCreateWithFlags(&s.in, sf) != cudaSuccess || cudaStreamCreateWithFlags(&s.cmp, sf) != cudaSuccess ||
        cudaStreamCreateWithFlags(&s.out, sf) != cudaSuccess || cudaEventCreateWithFlags(&s.entry, ef) != cudaSuccess ||
        cudaEventCreateWithFlags(&s.fin, ef) != cudaSuccess)
      return SA_ERR_CUDA;
    for (int i = 0; i < 2; ++i)
      if (cudaEventCreateWithFlags(&s.in_done[i], ef) != cudaSuccess ||
          cudaEventCreateWithFlags(&s.cmp_done[i], ef) != cudaSuccess ||
          cudaEventCreateWithFlags(&s.out_done[i], ef) != cudaSuccess)
        return SA_ERR_CUDA;
    s.ready = true;
  }
  *out = &s;
  return SA_OK;
}

constexpr int kMaxChunkUsers = 1024;
constexpr int64_t kDefaultChunkTokens = 262144;

size_t elem(sa_dtype dt) { return dt == SA_BF16 ? 2 : 4; }

// Users [begin[c], begin[c+1]) form chunk c: consecutive users are added while
// the chunk stays within chunk_tokens tokens and max_users users (a longer user
// is a chunk of its own).
sa_status plan_chunks(const int32_t* cu, int B, int64_t chunk_tokens, int max_users, std::vector<int>* begin) {
  if (!cu || B < 1 || chunk_tokens < 1 || max_users < 1) return SA_ERR_INVALID_ARG;
  if (cu[0] != 0) return SA_ERR_BAD_SEQLENS;
  begin->assign(1, 0);
  int64_t tok = 0;
  int users = 0;
  for (int b = 0; b < B; ++b) {
    const int64_t L = int64_t(cu[b + 1]) - int64_t(cu[b]);
    if (L < 0) return SA_ERR_BAD_SEQLENS;
    if (users > 0 && (tok + L > chunk_tokens || users == max_users)) {
      begin->push_back(b);
      tok = 0;
      users = 0;
    }
    tok += L;
    ++users;
  }
  begin->push_back(B);
  return SA_OK;
}

// Device workspace of the pipeline, for chunks of at most Bc users and Nc tokens.
struct StepLayout {
  size_t q, dq, cu, stage[2], total;
  size_t k, v, g, sk, lse, dk, dv, dqc, ws;  // offsets inside one staging buffer
  size_t stage_bytes, ws_bytes;
};

StepLayout step_layout(int B, int n_chunks, int Bc, int64_t Nc, int H, int P, int d, sa_dtype dt) {
  StepLayout L{};
  const size_t e = elem(dt), hpd = size_t(H) * P * d;
  size_t off = 256;  // header: sticky error word
  L.q = off;
  off = sa::align256(off + hpd * e);
  L.dq = off;
  off = sa::align256(off + hpd * 4);
  L.cu = off;
  off = sa::align256(off + sizeof(int32_t) * size_t(B + n_chunks));
  size_t s = 0;
  L.k = s;
  s = sa::align256(s + size_t(Nc) * H * d * e);
  L.v = s;
  s = sa::align256(s + size_t(Nc) * H * d * e);
  L.g = s;
  s = sa::align256(s + size_t(Bc) * hpd * 4);
  L.sk = s;
  s = sa::align256(s + size_t(Bc) * hpd * 4);
  L.lse = s;
  s = sa::align256(s + size_t(Nc) * H * 4);
  L.dk = s;
  s = sa::align256(s + size_t(Nc) * H * d * e);
  L.dv = s;
  s = sa::align256(s + size_t(Nc) * H * d * e);
  L.dqc = s;
  s = sa::align256(s + hpd * 4);
  L.ws = s;
  L.ws_bytes = sa_workspace_size(Bc, Nc, H, P, d, dt, 1);
  s = sa::align256(s + L.ws_bytes);
  L.stage_bytes = s;
  L.stage[0] = off;
  L.stage[1] = off + s;
  L.total = off + 2 * s;
  return L;
}

// Largest chunk (users, tokens) of a plan.
void chunk_max(const int32_t* cu, const std::vector<int>& begin, int* Bc, int64_t* Nc) {
  *Bc = 1;
  *Nc = 1;
  for (size_t c = 0; c + 1 < begin.size(); ++c) {
    const int nb = begin[c + 1] - begin[c];
    const int64_t nt = int64_t(cu[begin[c + 1]]) - int64_t(cu[begin[c]]);
    if (nb > *Bc) *Bc = nb;
    if (nt > *Nc) *Nc = nt;
  }
}

#define STEP_CUDA(x)                          \
  do {                                        \
    if ((x) != cudaSuccess) return SA_ERR_CUDA; \
  } while (0)
#define STEP_TRY(x)                  \
  do {                               \
    const sa_status s_ = (x);        \
    if (s_ != SA_OK) return s_;      \
  } while (0)

}  // namespace

extern "C" {

sa_status sa_plan_chunks_host(const int32_t* cu_seqlens_host, int B, int64_t chunk_tokens, int* begin,
                              int* n_chunks) {
  if (!begin || !n_chunks) return SA_ERR_INVALID_ARG;
  std::vector<int> b;
  const sa_status st = plan_chunks(cu_seqlens_host, B, chunk_tokens > 0 ? chunk_tokens : kDefaultChunkTokens,
                                   kMaxChunkUsers, &b);
  if (st != SA_OK) return st;
  for (size_t i = 0; i < b.size(); ++i) begin[i] = b[i];
  *n_chunks = int(b.size()) - 1;
  return SA_OK;
}

size_t sa_step_host_workspace_size(const int32_t* cu_seqlens_host, int B, int H, int P, int d, sa_dtype dt,
                                   int64_t chunk_tokens) {
  std::vector<int> begin;
  if (plan_chunks(cu_seqlens_host, B, chunk_tokens > 0 ? chunk_tokens : kDefaultChunkTokens, kMaxChunkUsers,
                  &begin) != SA_OK)
    return 0;
  int Bc;
  int64_t Nc;
  chunk_max(cu_seqlens_host, begin, &Bc, &Nc);
  if (sa_workspace_size(Bc, Nc, H, P, d, dt, 1) == 0) return 0;
  return step_layout(B, int(begin.size()) - 1, Bc, Nc, H, P, d, dt).total;
}

sa_status sa_sketch_step_host(const void* K, const void* V, const int32_t* cu_seqlens_host, int B, int64_t N,
                              const void* Q, int H, int P, int d, float scale, sa_dtype dt, const float* dsketch,
                              float* sketch, void* dK, void* dV, float* dQ, int64_t chunk_tokens, void* workspace,
                              size_t ws_bytes, void* stream) {
  if (!cu_seqlens_host || !Q || !dsketch || !sketch || !dQ || !workspace) return SA_ERR_INVALID_ARG;
  if (N > 0 && (!K || !V || !dK || !dV)) return SA_ERR_INVALID_ARG;
  if (B < 1 || N < 0 || int64_t(cu_seqlens_host[B]) != N) return SA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SA_ERR_INVALID_ARG;
  std::vector<int> begin;
  STEP_TRY(plan_chunks(cu_seqlens_host, B, chunk_tokens > 0 ? chunk_tokens : kDefaultChunkTokens, kMaxChunkUsers,
                       &begin));
  const int nc = int(begin.size()) - 1;
  int Bc;
  int64_t Nc;
  chunk_max(cu_seqlens_host, begin, &Bc, &Nc);
  if (sa_workspace_size(Bc, Nc, H, P, d, dt, 1) == 0) return SA_ERR_UNSUPPORTED;
  const StepLayout L = step_layout(B, nc, Bc, Nc, H, P, d, dt);
  if (ws_bytes < L.total) return SA_ERR_WORKSPACE;
  StepStreams* S = nullptr;
  STEP_TRY(step_streams(&S));
  char* base = static_cast<char*>(workspace);
  const size_t e = elem(dt), row = size_t(H) * d * e, hpd = size_t(H) * P * d;
  cudaStream_t user = static_cast<cudaStream_t>(stream);

  // rebased offsets of every chunk, one host array copied once
  std::vector<int32_t> cu_all;
  cu_all.reserve(size_t(B + nc));
  for (int c = 0; c < nc; ++c)
    for (int b = begin[c]; b <= begin[c + 1]; ++b) cu_all.push_back(cu_seqlens_host[b] - cu_seqlens_host[begin[c]]);

  // start after the caller's earlier work and after the previous call's pipeline
  // (which may still read this workspace or these streams' buffers)
  STEP_CUDA(cudaEventRecord(S->entry, user));
  for (cudaStream_t t : {S->in, S->cmp, S->out}) {
    STEP_CUDA(cudaStreamWaitEvent(t, S->entry, 0));
    STEP_CUDA(cudaStreamWaitEvent(t, S->fin, 0));
  }
  STEP_CUDA(cudaMemsetAsync(base, 0, 256, S->cmp));
  STEP_CUDA(cudaMemsetAsync(base + L.dq, 0, hpd * 4, S->cmp));
  STEP_CUDA(cudaMemcpyAsync(base + L.q, Q, hpd * e, cudaMemcpyHostToDevice, S->in));
  STEP_CUDA(cudaMemcpyAsync(base + L.cu, cu_all.data(), cu_all.size() * sizeof(int32_t), cudaMemcpyHostToDevice,
                            S->in));
  int cu_off = 0;
  for (int c = 0; c < nc; ++c) {
    const int s = c & 1;
    const int b0 = begin[c], nb = begin[c + 1] - b0;
    const int64_t t0 = cu_seqlens_host[b0], nt = int64_t(cu_seqlens_host[begin[c + 1]]) - t0;
    char* st = base + L.stage[s];
    // copy-in, once the step of chunk c - 2 has read this buffer's inputs
    if (c >= 2) STEP_CUDA(cudaStreamWaitEvent(S->in, S->cmp_done[s], 0));
    if (nt > 0) {
      STEP_CUDA(cudaMemcpyAsync(st + L.k, static_cast<const char*>(K) + size_t(t0) * row, size_t(nt) * row,
                                cudaMemcpyHostToDevice, S->in));
      STEP_CUDA(cudaMemcpyAsync(st + L.v, static_cast<const char*>(V) + size_t(t0) * row, size_t(nt) * row,
                                cudaMemcpyHostToDevice, S->in));
    }
    STEP_CUDA(cudaMemcpyAsync(st + L.g, dsketch + size_t(b0) * hpd, size_t(nb) * hpd * 4, cudaMemcpyHostToDevice,
                              S->in));
    STEP_CUDA(cudaEventRecord(S->in_done[s], S->in));
    // the step on the chunk, once the copy-out of chunk c - 2 has read this
    // buffer's outputs
    STEP_CUDA(cudaStreamWaitEvent(S->cmp, S->in_done[s], 0));
    if (c >= 2) STEP_CUDA(cudaStreamWaitEvent(S->cmp, S->out_done[s], 0));
    const int32_t* cuc = reinterpret_cast<const int32_t*>(base + L.cu) + cu_off;
    float* skc = reinterpret_cast<float*>(st + L.sk);
    float* lsec = reinterpret_cast<float*>(st + L.lse);
    float* dqc = reinterpret_cast<float*>(st + L.dqc);
    STEP_TRY(sa_sketch_fwd(st + L.k, st + L.v, cuc, nb, nt, base + L.q, H, P, d, scale, dt, skc, lsec, st + L.ws,
                           L.ws_bytes, S->cmp));
    STEP_TRY(sa_sketch_bwd(st + L.k, st + L.v, cuc, nb, nt, base + L.q, H, P, d, scale, dt,
                           reinterpret_cast<const float*>(st + L.g), lsec, st + L.dk, st + L.dv, dqc, st + L.ws,
                           L.ws_bytes, S->cmp));
    STEP_CUDA(sa::launch_add_into(base + L.dq, dqc, int64_t(hpd), SA_F32, S->cmp));
    sa::sticky_error_kernel<<<1, 1, 0, S->cmp>>>(reinterpret_cast<const uint32_t*>(st + L.ws),
                                                 reinterpret_cast<uint32_t*>(base));
    STEP_CUDA(cudaGetLastError());
    STEP_CUDA(cudaEventRecord(S->cmp_done[s], S->cmp));
    // copy-out
    STEP_CUDA(cudaStreamWaitEvent(S->out, S->cmp_done[s], 0));
    STEP_CUDA(cudaMemcpyAsync(sketch + size_t(b0) * hpd, skc, size_t(nb) * hpd * 4, cudaMemcpyDeviceToHost, S->out));
    if (nt > 0) {
      STEP_CUDA(cudaMemcpyAsync(static_cast<char*>(dK) + size_t(t0) * row, st + L.dk, size_t(nt) * row,
                                cudaMemcpyDeviceToHost, S->out));
      STEP_CUDA(cudaMemcpyAsync(static_cast<char*>(dV) + size_t(t0) * row, st + L.dv, size_t(nt) * row,
                                cudaMemcpyDeviceToHost, S->out));
    }
    STEP_CUDA(cudaEventRecord(S->out_done[s], S->out));
    cu_off += nb + 1;
  }
  // dQ after the last chunk's addition (the copy-out stream follows the compute stream)
  STEP_CUDA(cudaMemcpyAsync(dQ, base + L.dq, hpd * 4, cudaMemcpyDeviceToHost, S->out));
  STEP_CUDA(cudaEventRecord(S->fin, S->out));
  STEP_CUDA(cudaStreamWaitEvent(user, S->fin, 0));
  return SA_OK;
}

}  // extern "C"
