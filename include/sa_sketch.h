/*
 * sa_sketch.h -- C ABI of libsa_sketch.so, the GB300 (sm_103a) implementation of
 * the Sketch Attention (SA) sketching step of SequenceO1.
 *
 * The operation (paper Sec. 3.1, equations for the affinity S, the prototype-wise
 * softmax A and the sketch eq:sa-sketch; App. B steps 1-3), for every user b and
 * head h, with K_b, V_b the user's rows cu_seqlens[b] .. cu_seqlens[b+1]-1:
 *
 *     S[j,i]     = scale * sum_c Q[h,j,c] * K_b[i,h,c]           (P x L_b)
 *     A[:,i]     = softmax over the P prototypes of S[:,i]       (each token
 *                  spreads unit mass over the prototypes)
 *     sketch[b,h]= A V_b                                         (P x d)
 *
 * No further normalisation is applied (the sketch is the plain weighted sum over
 * the user's tokens, Sec. 3.1).  Heads are independent copies of the paper's
 * single-head SA.  The backward is the chain rule of these three steps; the
 * prototypes are shared by all users (Sec. 3.1), so dQ sums over the batch.
 * FlashSA (Sec. 4.4) motivates the streaming design: S and A never reach HBM.
 *
 * Conventions shared by every entry point
 *   - All tensors are contiguous, row-major, in device memory, owned by the
 *     caller.  The library never allocates device memory and keeps no state
 *     besides per-device caches (kernel attributes, SM count, timing events).
 *   - K, V, Q, dK, dV all have element type `dt`.  sketch, dsketch, dQ and lse
 *     are float32.  Element offsets are 64-bit.
 *   - K, V   : [N, H, d]   packed rows of all users, N = cu_seqlens[B]
 *     Q      : [H, P, d]   prototypes
 *     cu     : [B + 1]     int32, cu[0] = 0, non-decreasing, cu[B] = N
 *     sketch : [B, H, P, d]      lse : [N, H]      dQ : [H, P, d]
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every call only enqueues work on it and returns; nothing
 *     synchronises the host.
 *   - Outputs are overwritten, never accumulated into.  A user with L_b = 0 gets
 *     an all-zero sketch and contributes nothing to dQ.
 *   - Inputs and outputs must not overlap.
 *   - Results are bitwise reproducible for the same inputs, device and
 *     arguments: every reduction runs in a fixed order (no float atomics).
 *   - Errors the host can see (NULL pointers, sizes, unsupported shapes, a small
 *     workspace) are returned synchronously before anything is enqueued.
 *     Errors only the device can see (bad cu_seqlens contents, a pipeline wait
 *     that gave up) are written to an error word inside the workspace; the
 *     kernels of that call then skip their work, and sa_get_device_error()
 *     reports the code.
 *   - Not thread-safe for concurrent calls that share one workspace.
 */
#ifndef SA_SKETCH_H
#define SA_SKETCH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SA_OK = 0,
  SA_ERR_INVALID_ARG = 1,  /* NULL pointer, negative size, scale not finite     */
  SA_ERR_UNSUPPORTED = 2,  /* shape or dtype outside what the kernels support   */
  SA_ERR_WORKSPACE = 3,    /* ws_bytes smaller than sa_workspace_size()          */
  SA_ERR_CUDA = 4,         /* a CUDA runtime call failed (launch, event, ...)    */
  SA_ERR_TIMEOUT = 5,      /* a device pipeline wait gave up (device-detected)   */
  SA_ERR_BAD_SEQLENS = 6   /* cu_seqlens not 0..N non-decreasing (device-detected) */
} sa_status;

typedef enum { SA_F32 = 0, SA_BF16 = 1 } sa_dtype;

/* Bytes of scratch the caller must pass as `workspace` (device memory, 256-byte
 * aligned) for a call with these sizes on the current device; `bwd` != 0 sizes
 * it for sa_sketch_bwd, which needs more.  Returns 0 for invalid sizes.
 * Supported: 1 <= P <= 2048, 1 <= d <= 128 (d a multiple of 8 for bf16, of 4 for
 * f32), 1 <= H <= 64, B >= 1, 0 <= N < 2^31. */
size_t sa_workspace_size(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd);

/* Forward: sketch[b,h] = softmax_proto(scale * Q[h] K_b[:,h]^T) V_b[:,h]
 * (Sec. 3.1).  `lse` may be NULL; when given it receives, per token and head,
 * log sum_j exp(S[j,i]) (the softmax statistic FlashSA keeps, Sec. 4.4) so the
 * backward can skip recomputing it.  `scale` is normally 1/sqrt(d); any finite
 * scale is valid.  A negative one runs on the same tensor-core kernels: the
 * call negates a copy of Q in the workspace (scale Q K^T = (-scale)(-Q) K^T,
 * exactly), and the backward negates dQ back. */
sa_status sa_sketch_fwd(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                        int64_t N, const void* Q, int H, int P, int d, float scale,
                        sa_dtype dt, float* sketch, float* lse, void* workspace,
                        size_t ws_bytes, void* stream);

/* Backward of the forward above for upstream gradient dsketch [B,H,P,d] (fp32):
 *   dV_i = sum_j A[j,i] G_j,   dS = A o (G V^T - colsum(A o G V^T)),
 *   dK_i = scale sum_j dS[j,i] Q_j,   dQ[h] = scale sum_b sum_i dS[:,i] K_b[i,h]
 * (chain rule of Sec. 3.1; the paper prints no backward).  `lse` is the forward's
 * statistic or NULL (then it is recomputed).  dK, dV have type `dt`; dQ is fp32
 * and fully overwritten (the sum over all users of the batch). */
sa_status sa_sketch_bwd(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                        int64_t N, const void* Q, int H, int P, int d, float scale,
                        sa_dtype dt, const float* dsketch, const float* lse, void* dK,
                        void* dV, float* dQ, void* workspace, size_t ws_bytes,
                        void* stream);

/* Per-user queries, the stacked refinement of Sec. 3.3: from the second SA step
 * on, the queries are each user's own refined sketch times W_Q^(l), so Q holds
 * one block of prototypes per user:
 *     Q : [B, H, P, d]  (type `dt`),    user b, head h reads Q[b, h] instead of Q[h].
 * Everything else -- arguments, layouts, ownership, `lse`, the workspace size
 * (sa_workspace_size with the same sizes), errors and determinism -- is as in
 * sa_sketch_fwd. */
sa_status sa_sketch_fwd_per_user(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                                 int64_t N, const void* Q, int H, int P, int d, float scale,
                                 sa_dtype dt, float* sketch, float* lse, void* workspace,
                                 size_t ws_bytes, void* stream);

/* Backward with per-user queries (chain rule of Sec. 3.3's steps): as
 * sa_sketch_bwd, except that Q is [B, H, P, d] and
 *     dQ : [B, H, P, d] fp32,  dQ[b, h] = scale sum_i dS[:, i] K_b[i, h]
 * holds only user b's tokens (no sum over the batch); fully overwritten, zero
 * for a user with L_b = 0. */
sa_status sa_sketch_bwd_per_user(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                                 int64_t N, const void* Q, int H, int P, int d, float scale,
                                 sa_dtype dt, const float* dsketch, const float* lse, void* dK,
                                 void* dV, float* dQ, void* workspace, size_t ws_bytes,
                                 void* stream);

/* The step with its key projection (Sec. 3.1: S = (P W_Q)(X W_K)^T / sqrt(d),
 * sketch A X; App. G.3: K = X W_K): the history X serves as the values and,
 * through W_K, as the keys.
 *     X  : [N, H, d]  (type `dt`)      Wk : [H, d, d] (type `dt`, k_i = x_i Wk[h])
 *     Q  : [H, P, d]  (type `dt`, the projected prototypes P W_Q)
 * Computed as the step with K = V = X and prototypes Q' = Q Wk^T (equal scores:
 * q_j . (x_i Wk) = (q_j Wk^T) . x_i); no K is formed.  The workspace must hold
 * sa_workspace_size_x() bytes (the step's own plus Q', and for the backward dK'
 * and dQ').  Other arguments, results and errors as in sa_sketch_fwd. */
size_t sa_workspace_size_x(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd);
sa_status sa_sketch_fwd_x(const void* X, const int32_t* cu_seqlens, int B, int64_t N, const void* Q,
                          const void* Wk, int H, int P, int d, float scale, sa_dtype dt, float* sketch,
                          float* lse, void* workspace, size_t ws_bytes, void* stream);

/* Backward of sa_sketch_fwd_x: dX [N,H,d] (type `dt`) = dV + dK W_K^T (X reaches
 * the sketch as the values and through the keys), dQ [H,P,d] fp32 and
 * dWk [H,d,d] fp32 = X^T dK per head (chain rule; the paper prints none).  All
 * outputs are overwritten; `lse` as in sa_sketch_bwd. */
sa_status sa_sketch_bwd_x(const void* X, const int32_t* cu_seqlens, int B, int64_t N, const void* Q,
                          const void* Wk, int H, int P, int d, float scale, sa_dtype dt, const float* dsketch,
                          const float* lse, void* dX, float* dQ, float* dWk, void* workspace, size_t ws_bytes,
                          void* stream);

/* Token-wise ("vanilla") normalisation, the comparison of Sec. 5.1 and App. C:
 * the same scores normalised over each user's tokens instead of the prototypes,
 *     A[j, :]      = softmax over i of S[j, i]     (weights p(i | j): every
 *                    prototype spreads unit mass over the user's tokens)
 *     sketch[b, h] = A V_b                          (P x d)
 *     lse_tok      : [B, H, P] fp32, log sum_i exp(S[j, i]) per user, head and
 *                    prototype (-inf for a user with L_b = 0, whose sketch is 0)
 * `lse_tok` may be NULL.  Shared prototypes Q [H, P, d] only.  Tensor cores
 * (tcgen05, fp32 accumulation) serve bf16 with d in {64, 128} and P a multiple
 * of 128 up to 2048, for any nonzero scale (a negative one is folded into a
 * negated copy of Q as in sa_sketch_fwd); other shapes, fp32 inputs and a zero
 * scale run on CUDA-core kernels (fp32 arithmetic).  The workspace must hold
 * sa_workspace_size_tokenwise() bytes; everything else (layouts, ownership,
 * errors, determinism) as in sa_sketch_fwd. */
size_t sa_workspace_size_tokenwise(int B, int64_t N, int H, int P, int d, sa_dtype dt, int bwd);
sa_status sa_sketch_fwd_tokenwise(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                                  int64_t N, const void* Q, int H, int P, int d, float scale,
                                  sa_dtype dt, float* sketch, float* lse_tok, void* workspace,
                                  size_t ws_bytes, void* stream);

/* Backward of sa_sketch_fwd_tokenwise for dsketch G [B,H,P,d] (chain rule; the
 * paper prints none), with D_j = G_j . sketch_j per user and head:
 *     dV_i = sum_j A[j,i] G_j,    dS[j,i] = A[j,i] (G_j . v_i - D_j),
 *     dK_i = scale sum_j dS[j,i] Q_j,    dQ[h] = scale sum_b sum_i dS[:,i] K_b[i,h].
 * `sketch` and `lse_tok` are the forward's outputs; when either is NULL both are
 * recomputed.  sketch, lse_tok and dsketch must be 16-byte aligned.  dK, dV have
 * type `dt`, dQ is fp32; all fully overwritten.  Tensor cores serve bf16 with
 * d = 128 and P in {256, 512, 1024, 2048}; other shapes run on CUDA cores. */
sa_status sa_sketch_bwd_tokenwise(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                                  int64_t N, const void* Q, int H, int P, int d, float scale,
                                  sa_dtype dt, const float* sketch, const float* lse_tok,
                                  const float* dsketch, void* dK, void* dV, float* dQ,
                                  void* workspace, size_t ws_bytes, void* stream);

/* The training step (forward and backward, Sec. 3.1) on a batch held in HOST
 * memory (the paper has no counterpart; a runtime convenience).  K, V, Q and
 * dsketch are host arrays, sketch, dK, dV and dQ host arrays the call fills;
 * shapes, dtypes and the results are those of sa_sketch_fwd followed by
 * sa_sketch_bwd (lse is kept internal).  cu_seqlens_host is a host array.
 *   - Users are grouped into chunks of at most chunk_tokens tokens (<= 0: 262144;
 *     a longer user is a chunk of its own; at most 1024 users per chunk).  Three
 *     internal streams overlap the host-to-device copy of a chunk, the step on
 *     the previous chunk and the device-to-host copy of the one before, through
 *     two staging buffers in the workspace (a chunk's copy-in waits for the step
 *     of the chunk that last used its buffer, its step for that chunk's
 *     copy-out, so that copy-in and copy-out run side by side); dQ is
 *     summed over the chunks in chunk order (bitwise reproducible for a given
 *     chunk_tokens, but not bitwise equal to one sa_sketch_bwd call on the
 *     whole batch: the summation groups differ).
 *   - Asynchronous with respect to the host: the call enqueues everything and
 *     makes `stream` wait for it, so synchronising `stream` means the host
 *     outputs are written.  Page-locked host arrays give overlapped copies;
 *     pageable ones are correct but serialise the copies.  Host arrays must stay
 *     valid and unchanged until then.
 *   - `workspace` is device memory of sa_step_host_workspace_size() bytes
 *     (256-byte aligned); sa_get_device_error(workspace, stream) reports the
 *     first device-detected error of any chunk.
 *   - Not thread-safe: the pipeline's streams are shared per device; serialise
 *     calls on one device. */
size_t sa_step_host_workspace_size(const int32_t* cu_seqlens_host, int B, int H, int P, int d, sa_dtype dt,
                                   int64_t chunk_tokens);
sa_status sa_sketch_step_host(const void* K, const void* V, const int32_t* cu_seqlens_host, int B,
                              int64_t N, const void* Q, int H, int P, int d, float scale, sa_dtype dt,
                              const float* dsketch, float* sketch, void* dK, void* dV, float* dQ,
                              int64_t chunk_tokens, void* workspace, size_t ws_bytes, void* stream);

/* Allocation-free forward (the paper has no counterpart; this is a library
 * convenience).  For callers that cannot provide a workspace: for example a
 * plugin or custom-operator hook that receives only its input and output
 * buffers and may not allocate device memory, or a service running inside a
 * device-memory budget fixed in advance.  Same arguments and results as
 * sa_sketch_fwd without the workspace: the scratch comes from one fixed array
 * of sa_noalloc_scratch_bytes() bytes (32 MiB) that this library keeps in
 * device memory on every GPU where it is loaded, until the process exits.
 *   - Returns SA_ERR_WORKSPACE, before launching anything, when the call would
 *     need more scratch than that; use sa_sketch_fwd then.  The scratch holds
 *     per-worker sketch pieces (2 x P x d fp32 per SM) and per-token
 *     statistics (4 bytes per token and head), so on a 152-SM GB300 the array
 *     serves, for example, P = 256 with d = 64 or P = 128 with d = 128 for
 *     batches of up to about 3 million token-heads (tokens x heads); the
 *     100K-token workload's P = 512 with d = 128 does not fit.
 *   - It allocates nothing itself.  The array belongs to the current device
 *     (cudaGetDevice), not to the device of `stream` or of the tensors: make
 *     the device that owns the stream and all buffers current before calling.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current) and caches it with the
 *     device's context (a reset context is looked up again).  Under CUDA's
 *     default lazy module loading that first call is also when the driver
 *     commits the array's 32 MiB, so it can fail with SA_ERR_CUDA if the
 *     device is out of memory: make one warm-up call at set-up, before the
 *     memory budget is fully used and before any stream capture.
 *   - All calls share the one array: two calls whose work overlaps on the GPU
 *     (different streams, or different host threads) race and may corrupt each
 *     other's results; serialise them.  Each call rewrites everything it
 *     reads, including the error word, so a call after a failed one starts
 *     clean.
 *   - Errors only the device can see (bad cu_seqlens contents, a pipeline wait
 *     that gave up) make the call's kernels skip their work and are reported
 *     by sa_noalloc_get_device_error(), not by the return value. */
sa_status sa_sketch_fwd_noalloc(const void* K, const void* V, const int32_t* cu_seqlens, int B,
                                int64_t N, const void* Q, int H, int P, int d, float scale,
                                sa_dtype dt, float* sketch, float* lse, void* stream);

/* Size in bytes of the fixed scratch array used by sa_sketch_fwd_noalloc. */
size_t sa_noalloc_scratch_bytes(void);

/* Synchronises `stream` and returns the device-detected status of the last
 * sa_sketch_fwd_noalloc call on the current device (SA_OK, SA_ERR_BAD_SEQLENS
 * or SA_ERR_TIMEOUT), or SA_ERR_CUDA if the stream reports an error.  The
 * counterpart of sa_get_device_error() for callers that hold no workspace. */
sa_status sa_noalloc_get_device_error(void* stream);

/* Synchronises `stream` and returns the device-detected status of the last call
 * that used this workspace (SA_OK, SA_ERR_BAD_SEQLENS or SA_ERR_TIMEOUT), or
 * SA_ERR_CUDA if the stream itself reports an error. */
sa_status sa_get_device_error(const void* workspace, void* stream);

/* Static English description of a status code. */
const char* sa_status_string(sa_status s);

/* ---- measurement hooks (used by bench.py; not needed for normal use) ------- */

/* Kernel classes whose launches can be timed with CUDA events: the forward's
 * main kernel, the backward's main (token-side) kernel, small helpers, the
 * per-token lse pass, and the backward's prototype-side dQ kernel. */
typedef enum {
  SA_KERNEL_FWD_MAIN = 0,
  SA_KERNEL_BWD_MAIN = 1,
  SA_KERNEL_AUX = 2,
  SA_KERNEL_FWD_LSE = 3,
  SA_KERNEL_BWD_DQ = 4
} sa_kernel_class;

/* Turn event timing of the main kernels on (1) or off (0) and clear the record.
 * When on, every main-kernel launch is bracketed by CUDA events recorded on the
 * launching stream (at most 4096 launches are recorded). */
sa_status sa_timing_enable(int on);

/* Synchronises the recorded events and returns, for kernel class `k`, the sum of
 * launch durations in milliseconds and the number of launches recorded. */
sa_status sa_timing_read(sa_kernel_class k, double* total_ms, int64_t* launches);

/* Number of kernels this library has launched in this process. */
uint64_t sa_launch_count(void);

/* Time limit, in nanoseconds, of every bounded wait inside the tensor-core
 * kernels, for calls enqueued after this one (0 restores the default of 2 s;
 * at most 4 s, else SA_ERR_INVALID_ARG).  A correct pipeline never waits
 * anywhere near 2 s; a lower limit exists so that tests can make a wait run
 * out on purpose and check the recovery: the call's kernels stop, drain their
 * copies and tensor-core work still in flight, release their tensor memory,
 * and sa_get_device_error() reports SA_ERR_TIMEOUT.  Under a limit below
 * 1 ms the tensor-core forwards first wait on a barrier that nothing
 * completes, so such a call always times out (a try-wait may otherwise sleep
 * until its barrier completes and never see a short limit).  The limit is
 * copied into each call's workspace when the call is enqueued. */
sa_status sa_set_wait_limit_ns(uint64_t ns);

/* Kernel selection for all later calls in this process: 0 (default) lets each
 * call pick the tensor-core kernels where its shape is supported, 1 forces the
 * CUDA-core kernels everywhere (a cross-check of the two), 2 keeps the
 * tensor cores but runs the forward for P = 512 (and P = 256 with d = 128) as a
 * per-token lse pass followed by prototype slices instead of the cluster-pair
 * kernel (another cross-check), 3 runs the P = 512 forward on the
 * cluster-pair kernel with eight softmax warps per CTA instead of sixteen
 * (its earlier form, a third cross-check).  The workspace size depends on the selection: size it after
 * choosing. */
sa_status sa_select_path(int path);

/* Name of the kernel that a forward (bwd = 0) or backward (bwd = 1) call with
 * these shapes would use as its main kernel ("tc..." = tcgen05 tensor cores,
 * "simt..." = CUDA cores).  Static string. */
const char* sa_main_kernel_name(int P, int d, sa_dtype dt, int bwd);

/* ---- host-side planning (pure C, no GPU; exported for tests) -------------- */

/* The tiling every call applies: user b contributes ceil(L_b / tile) tiles per
 * head, tiles are ordered (head, user, tile), and worker w of n_workers owns
 * the contiguous tile range [begin[w], begin[w+1]).  Fills begin[0..n_workers]
 * from host cu_seqlens; returns SA_ERR_BAD_SEQLENS for invalid offsets. */
sa_status sa_plan_host(const int32_t* cu_seqlens_host, int B, int H, int tile, int n_workers,
                       int64_t* begin);

/* The tile sequence as the tensor-core kernels walk it: worker w of n_workers
 * takes its range [begin[w], begin[w+1]) (sa_plan_host), locates its first
 * tile by a binary search over the users, steps `tile` tokens at a time inside
 * a (user, head) segment and finds the next segment's user by a forward scan
 * over the users (falling back to the search after a run of empty users).
 * Writes, for every tile t of the batch (t < H * tiles per head <= cap), its
 * user, head, first token row and token count.  Pure C, no GPU; exported for
 * tests.  SA_ERR_INVALID_ARG if cap is too small, SA_ERR_BAD_SEQLENS for
 * invalid offsets. */
sa_status sa_walk_host(const int32_t* cu_seqlens_host, int B, int H, int tile, int n_workers, int32_t* user,
                       int32_t* head, int64_t* tok0, int32_t* ntok, int64_t cap);

/* The chunks sa_sketch_step_host forms: users [begin[c], begin[c+1]) are chunk
 * c, for c < *n_chunks; `begin` must hold B + 1 entries. */
sa_status sa_plan_chunks_host(const int32_t* cu_seqlens_host, int B, int64_t chunk_tokens, int* begin,
                              int* n_chunks);

#ifdef __cplusplus
}
#endif
#endif /* SA_SKETCH_H */
