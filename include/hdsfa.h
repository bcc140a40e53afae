/*
 * hdsfa.h -- C ABI of libhdsfa.so: GB300 (sm_103a) kernels for Hidden Decoding's
 * multi-stream token expansion and Stream-Factorized Attention (SFA).
 *
 * Notation (0-indexed): a batch holds B sequences of L tokens; each token is
 * expanded into n streams, giving nL positions.  Token t, stream s sits at
 * position p = t*n + s (the paper's 1-indexed t = (i-1)n + k, Eq. 1).
 *
 * Conventions shared by every entry point
 *   - Ownership: the caller allocates and owns every buffer (device memory).
 *     The library never allocates, frees or synchronises; all work is enqueued
 *     asynchronously on `stream` (0 = legacy default stream).
 *   - Layout: dense row-major, no padding.  bf16 is IEEE bfloat16 (uint16 bits).
 *       tables  [n][V][D]        ids [B][L] int32      expanded [B][nL][D]
 *       q, o, dout, dq  [B][nL][Hq][Dh]      k, v, dk, dv  [B][nL][Hkv][Dh]
 *       lse [B][Hq][nL] float32, natural-log log-sum-exp of each softmax row.
 *   - Grouped K/V: query head h reads K/V head h / (Hq / Hkv).
 *   - Host-side argument errors return before anything is enqueued.
 *   - dev_status (nullable): a device int32 the kernels OR error bits into
 *     (HD_DEVBIT_*); the caller zeroes it, synchronises, then reads it.
 *     Kernels never trap.
 *   - Pointers must be 16-byte aligned; D and Dh must make rows a multiple of
 *     16 bytes.
 */
#ifndef HDSFA_H
#define HDSFA_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  HD_OK = 0,
  HD_ERR_INVALID_ARG = 1, /* null / misaligned pointer, non-positive size, Hq % Hkv != 0 */
  HD_ERR_UNSUPPORTED = 2, /* valid but not implemented (e.g. Dh not in {64, 128, 256}) */
  HD_ERR_CUDA = 3,        /* a CUDA runtime/driver call or kernel launch failed */
  HD_ERR_WORKSPACE = 4,   /* workspace null or smaller than sfa_bwd_workspace_bytes() */
  HD_ERR_TIMEOUT = 5,     /* reserved: a bounded device wait expired (see HD_DEVBIT_TIMEOUT) */
  HD_ERR_INDEX = 6,       /* reserved: an index was out of range (see HD_DEVBIT_INDEX) */
  HD_ERR_SCRATCH_LIMIT = 7 /* sfa_bwd_noalloc: sizes need more than SFA_BWD_NOALLOC_MAX_BYTES */
} hd_status_t;

/* Bits the kernels OR into *dev_status. */
#define HD_DEVBIT_INDEX 1   /* a token id outside [0, V): hd_expand_embed zeroed its n output
                               rows; hd_expand_embed_bwd left it out of the sums.  A sequence
                               length outside its range in sfa_decode / sfa_kv_append */
#define HD_DEVBIT_TIMEOUT 2 /* a bounded pipeline wait expired; outputs are invalid */

/* Attention mask of one SFA layer (Sec. 2.2, Eq. 4 and Fig. 2). */
typedef enum {
  SFA_WITHIN = 0, /* intra-stream: p' <= p and p' = p (mod n)                 (Eq. 4, Fig. 2c) */
  SFA_CROSS = 1,  /* full cross-stream: standard causal mask over nL, p' <= p (Fig. 2a)        */
  SFA_LOCAL = 2,  /* local cross-stream: causal window, p - window < p' <= p  (Fig. 2b)        */
  SFA_WITHIN_NAIVE = 3 /* measurement mode: the SFA_WITHIN result (same mask, same outputs)
                          computed over the full causal tile schedule of nL positions, with
                          the stream condition applied per pair instead of skipping the
                          other streams' tiles: n times the work, what the skipping saves.
                          sfa_fwd / sfa_bwd (and their parts) at Dh = 128 only.          */
} sfa_mode_t;

/*
 * hd_expand_embed -- multi-stream token expansion (Eq. 1, Sec. 2.1):
 *   out[b][t*n + s][:] = tables[s][ids[b][t]][:]   for t < L, s < n.
 * tables: bf16 [n][V][D] (read-only); ids: int32 [B][L]; out: bf16 [B][n*L][D].
 * An id outside [0, V) writes zero rows and sets HD_DEVBIT_INDEX.
 * Requires D % 8 == 0 (16-byte rows) and 16-byte aligned tables/out.
 * Bit-exact copy; HBM-bound.
 */
hd_status_t hd_expand_embed(const void* tables, const int32_t* ids, void* out, int B, int L, int n,
                            int V, int D, int32_t* dev_status, cudaStream_t stream);

/*
 * hd_expand_embed_bwd -- backward of the expansion (adjoint of Eq. 1, Sec. 2.1):
 *   dtables[s][v][:] += sum over (b, t) with ids[b][t] = v of dout[b][t*n + s][:]
 * for every s < n and every v in [0, V) that occurs in ids.
 *   dout: bf16 [B][n*L][D] (read-only); ids: int32 [B][L]; dtables: float32 [n][V][D],
 *   accumulated in place (rows of ids that do not occur are not touched; zero the
 *   tables first for a plain gradient).
 *   Deterministic: every element of dtables is read and written once, by one thread,
 *   which sums the occurrences of its id in fp32 in an order fixed by their number
 *   (ascending token order b*L + t; for ids with more than 32 occurrences, eight
 *   consecutive token blocks, each in ascending order, whose sums are added in
 *   block order) and adds the sum to dtables: repeated calls on the same inputs give
 *   identical bits.
 *   An id outside [0, V) contributes nothing and sets HD_DEVBIT_INDEX.
 *   workspace: device memory of at least hd_expand_embed_bwd_workspace_bytes(B, L)
 *   bytes, 16-byte aligned, overwritten (no contents need to survive between calls;
 *   the size is independent of n, V and D).
 *   Requires D % 8 == 0, B*L < 2^31, n*D < 2^31, 16-byte aligned dout/dtables;
 *   HBM-bound.
 */
size_t hd_expand_embed_bwd_workspace_bytes(int B, int L); /* 0 for invalid sizes */
hd_status_t hd_expand_embed_bwd(const void* dout, const int32_t* ids, float* dtables, int B, int L,
                                int n, int V, int D, void* workspace, size_t workspace_bytes,
                                int32_t* dev_status, cudaStream_t stream);
/*
 * The same in two parts.  hd_expand_embed_bwd_plan reads only ids: it sorts the
 * tokens by id and lists each id's run of tokens in the workspace (the "plan"), so a
 * caller can build it as soon as the ids are known (e.g. on a side stream during the
 * forward pass) and keep it for several applies.  hd_expand_embed_bwd_apply adds the
 * gradient rows into dtables following a plan of the same ids, B, L and V; the
 * workspace must hold that plan, unmodified, when the apply runs (order a plan on
 * another stream before the apply with an event).  plan + apply == hd_expand_embed_bwd.
 * An apply on a workspace that does not hold such a plan gives meaningless sums but
 * never reads or writes outside dout, dtables and the workspace: records and token
 * indexes outside the plan's ranges are skipped.
 */
hd_status_t hd_expand_embed_bwd_plan(const int32_t* ids, int B, int L, int V, void* workspace,
                                     size_t workspace_bytes, int32_t* dev_status, cudaStream_t stream);
hd_status_t hd_expand_embed_bwd_apply(const void* dout, float* dtables, int B, int L, int n, int V,
                                      int D, const void* workspace, size_t workspace_bytes,
                                      cudaStream_t stream);

/*
 * hd_select_final_stream -- the positions the loss reads (Eq. 2, Sec. 2.1): the loss
 * is taken only on each token's final stream, 0-indexed position t*n + n-1.
 *   y[b][t][:] = x[b][t*n + n-1][:]   x: bf16 [B][n*L][D], y: bf16 [B][L][D].
 * hd_select_final_stream_bwd -- its adjoint:
 *   dx[b][t*n + n-1][:] = dy[b][t][:], every other row of dx is set to zero.
 * Bit-exact copies; D % 8 == 0, 16-byte aligned pointers; HBM-bound.
 */
hd_status_t hd_select_final_stream(const void* x, void* y, int B, int L, int n, int D,
                                   cudaStream_t stream);
hd_status_t hd_select_final_stream_bwd(const void* dy, void* dx, int B, int L, int n, int D,
                                       cudaStream_t stream);

/*
 * sfa_fwd -- SFA forward over the expanded sequence (Sec. 2.2; Eq. 3-4; Fig. 2):
 *   O[b][p][h] = sum_{p' visible from p} softmax_p'(scale * q_p . k_p') v_p',
 *   lse[b][h][p] = log sum_{p' visible} exp(scale * q_p . k_p').
 * q: bf16 [B][nL][Hq][Dh]; k, v: bf16 [B][nL][Hkv][Dh]; o: bf16 like q (written);
 * lse: float32 [B][Hq][nL] (written).  softmax_scale <= 0 selects 1/sqrt(Dh).
 * window is used only by SFA_LOCAL (must be >= 1 there).  Dh in {64, 128, 256}: the
 * forward and the backward run on tcgen05 kernels at every head dim (256 is the
 * paper's 80B configuration, Table 6).
 * Every position sees itself, so no softmax row is empty.
 */
hd_status_t sfa_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B, int L,
                    int n, int Hq, int Hkv, int Dh, float softmax_scale, sfa_mode_t mode,
                    int window, int32_t* dev_status, cudaStream_t stream);

/* Bytes of device workspace sfa_bwd needs for these sizes and mode (fp32 dQ
 * accumulator [B][nL][Hq][Dh] plus two fp32 row terms of about B*Hq*nL each; when the
 * backward's grid would leave SMs idle, also fp32 dK and dV partial sums [B][nL][Hkv][Dh]
 * for each of the query-head chunks it then splits the work into).
 * Returns 0 for invalid sizes. */
size_t sfa_bwd_workspace_bytes(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode);

/*
 * sfa_bwd -- gradient of sfa_fwd (the paper trains with SFA but does not write
 * the gradient; this is the derivative of the forward above):
 *   P = exp(scale q k^T - lse) on visible pairs, dP = dO v^T,
 *   dS = P * (dP - rowsum(dO * O)),
 *   dq = scale dS k,  dk = scale sum_{h in group} dS^T q,  dv = sum_{h in group} P^T dO.
 * Inputs q, k, v, o, dout (bf16) and lse (float32, as written by sfa_fwd).
 * Outputs dq [B][nL][Hq][Dh], dk, dv [B][nL][Hkv][Dh] (bf16, overwritten).
 * workspace: device buffer of at least sfa_bwd_workspace_bytes(...) bytes, 256-byte
 * aligned; its contents on entry do not matter.
 */
hd_status_t sfa_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                    const void* dout, void* dq, void* dk, void* dv, int B, int L, int n, int Hq,
                    int Hkv, int Dh, float softmax_scale, sfa_mode_t mode, int window,
                    void* workspace, size_t workspace_bytes, int32_t* dev_status,
                    cudaStream_t stream);

/*
 * The three phases sfa_bwd runs, in order on one stream, exported so a caller
 * can overlap or time them separately.  Same sizes, mode and workspace as sfa_bwd.
 *   sfa_bwd_prep     : delta = rowsum(dO * O) and lse * log2(e) into the workspace
 *                      (fp32, stream-major), and zero its fp32 dQ accumulator.
 *   sfa_bwd_main     : recompute P on visible pairs, add every dQ contribution
 *                      into the accumulator and write dk, dv (overwritten).
 *   sfa_bwd_finalize : dq = bf16(scale * accumulator).
 * A later phase reads what the earlier one left in the workspace.
 * sfa_bwd_prep is itself the two halves below, for a caller that overlaps them:
 *   sfa_bwd_row_terms: the delta and lse terms only (needs o, so after sfa_fwd);
 *   sfa_bwd_clear    : only the zeroing of the dQ accumulator.  It needs nothing from
 *                      the forward, so it may run on another stream beside sfa_fwd,
 *                      ordered after the previous sfa_bwd_finalize that read the same
 *                      workspace and before sfa_bwd_main.
 */
hd_status_t sfa_bwd_prep(const void* o, const void* dout, const float* lse, int B, int L, int n, int Hq,
                         int Hkv, int Dh, sfa_mode_t mode, void* workspace, size_t workspace_bytes,
                         cudaStream_t stream);
hd_status_t sfa_bwd_row_terms(const void* o, const void* dout, const float* lse, int B, int L, int n,
                              int Hq, int Hkv, int Dh, sfa_mode_t mode, void* workspace,
                              size_t workspace_bytes, cudaStream_t stream);
hd_status_t sfa_bwd_clear(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode, void* workspace,
                          size_t workspace_bytes, cudaStream_t stream);
hd_status_t sfa_bwd_main(const void* q, const void* k, const void* v, const void* dout, void* dk, void* dv,
                         int B, int L, int n, int Hq, int Hkv, int Dh, float softmax_scale,
                         sfa_mode_t mode, int window, void* workspace, size_t workspace_bytes,
                         int32_t* dev_status, cudaStream_t stream);
hd_status_t sfa_bwd_finalize(void* dq, int B, int L, int n, int Hq, int Hkv, int Dh,
                             float softmax_scale, sfa_mode_t mode, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream);

/*
 * sfa_fwd_final / sfa_bwd_final -- attention of the final-stream queries only (the
 * positions t*n + n-1 the loss reads, Eq. 2) against the layer's keys over all nL
 * positions: the layers that run only the final stream while the other streams' K/V
 * stay as context (Sec. 3.1, KV-mirror layers).  The mask is the layer's own (Eq. 4,
 * Fig. 2): the query of token t at position p = t*n + n-1 sees key p' iff
 *   WITHIN  p' <= p and p' = n-1 (mod n)   (only stream n-1's keys)
 *   CROSS   p' <= p
 *   LOCAL   p - window < p' <= p
 * which equals rows t*n + n-1 of sfa_fwd over the full sequence.
 *   q, o, dout, dq : bf16 [B][L][Hq][Dh]  (dense: only the final-stream rows)
 *   k, v, dk, dv   : bf16 [B][n*L][Hkv][Dh]
 *   lse            : float32 [B][Hq][L], natural log (written by sfa_fwd_final)
 * dk, dv are fully overwritten (zero for keys no final-stream query sees).
 * workspace: >= sfa_bwd_final_workspace_bytes(...) bytes, 256-byte aligned.
 * Dh in {64, 128, 256}, on the same tcgen05 kernels as sfa_fwd / sfa_bwd.
 */
hd_status_t sfa_fwd_final(const void* q, const void* k, const void* v, void* o, float* lse, int B, int L,
                          int n, int Hq, int Hkv, int Dh, float softmax_scale, sfa_mode_t mode, int window,
                          int32_t* dev_status, cudaStream_t stream);
size_t sfa_bwd_final_workspace_bytes(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode);
hd_status_t sfa_bwd_final(const void* q, const void* k, const void* v, const void* o, const float* lse,
                          const void* dout, void* dq, void* dk, void* dv, int B, int L, int n, int Hq,
                          int Hkv, int Dh, float softmax_scale, sfa_mode_t mode, int window,
                          void* workspace, size_t workspace_bytes, int32_t* dev_status,
                          cudaStream_t stream);

/*
 * sfa_decode -- one decoding step over the expanded KV cache (Sec. 3.2 "Inference
 * Cost"; masks of Eq. 4 and Fig. 2).  Generation runs each new token's n streams
 * together: with T = lens[b] tokens in sequence b's cache (the new token included,
 * its K/V rows already appended, see sfa_kv_append), the new token's positions
 * p = (T-1)*n + s attend to the cached positions p' < T*n that the layer's mask lets
 * them see: WITHIN p' = s (mod n) and p' <= p (only stream s's rows are read for it),
 * CROSS p' <= p, LOCAL p - window < p' <= p.  The result equals rows (T-1)*n .. T*n-1
 * of sfa_fwd over the sequence.
 *   q, o     : bf16 [B][n][Hq][Dh], the new token's n positions.
 *   k_cache, v_cache : bf16 [B][Lcap*n][Hkv][Dh], position p at row p (the layout of
 *              sfa_fwd's k / v, so a prefilled forward's K/V is a cache); read-only.
 *   lens     : int32 device array [B], tokens in each sequence's cache (ragged batch).
 *   lse      : float32 [B][Hq][n] natural-log LSE of each row, or NULL.
 *   max_tokens: a bound on every lens[b] (<= Lcap); the work is split for it.
 *   workspace: device memory of >= sfa_decode_workspace_bytes(B, max_tokens, n, Hq,
 *              Hkv, Dh, mode, window) bytes, 16-byte aligned (partial results).
 * A sequence with lens outside [1, max_tokens] gets zero rows, LSE = -inf and
 * HD_DEVBIT_INDEX.  Dh in {64, 128, 256}; Lcap*n <= 2^30.  HBM-bound (reads the
 * visible cached rows once per step).
 */
size_t sfa_decode_workspace_bytes(int B, int max_tokens, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode,
                                  int window); /* 0 for invalid sizes */
hd_status_t sfa_decode(const void* q, const void* k_cache, const void* v_cache, const int32_t* lens, void* o,
                       float* lse, int B, int max_tokens, int Lcap, int n, int Hq, int Hkv, int Dh,
                       float softmax_scale, sfa_mode_t mode, int window, void* workspace,
                       size_t workspace_bytes, int32_t* dev_status, cudaStream_t stream);

/*
 * sfa_kv_append -- the new token's n K and V rows into the cache (Sec. 3.2: each
 * decoded token adds n stream positions):
 *   k_cache[b][(T-1)*n + s] = k_new[b][s], likewise v, with T = lens[b] (the length
 *   including the new token), s < n.
 *   k_new, v_new: bf16 [B][n][Hkv][Dh]; caches as in sfa_decode.  Bit copy.
 * A length outside [1, Lcap] writes nothing for that sequence and sets HD_DEVBIT_INDEX.
 */
hd_status_t sfa_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                          const int32_t* lens, int B, int Lcap, int n, int Hkv, int Dh,
                          int32_t* dev_status, cudaStream_t stream);

/*
 * sfa_bwd_noalloc -- sfa_bwd without a caller-supplied workspace.  The paper has no
 * counterpart: this is an interface for callers that cannot hand the library device
 * memory of their own (a runtime that commits its whole device-memory budget at
 * start-up and forbids allocation while serving, or C code with no device allocator).
 * Same arguments, outputs and status codes as sfa_bwd, minus the workspace.
 *
 * The workspace lives in a fixed device array of the library, SFA_BWD_NOALLOC_MAX_BYTES
 * long, present in every CUDA context that loads the library's module; the call
 * allocates and frees nothing.  Sizes whose sfa_bwd_workspace_bytes() exceeds that
 * limit return HD_ERR_SCRATCH_LIMIT before anything is enqueued (use sfa_bwd there).
 *   - Set-up: every call looks up the array's device address in the calling thread's
 *     current CUDA context (the address belongs to that context, so it is not cached);
 *     the first call in a context also loads the library's module there, so make that
 *     first call before any stream capture.  A failed look-up returns HD_ERR_CUDA.
 *   - Sharing: every call on a device uses the same array, which keeps the last call's
 *     contents; each call clears what it reads before reading it.  Calls that may run
 *     concurrently on one device (unordered streams, several host threads) race on
 *     the array: the caller must order them.
 */
#define SFA_BWD_NOALLOC_MAX_BYTES ((size_t)64 << 20)
hd_status_t sfa_bwd_noalloc(const void* q, const void* k, const void* v, const void* o,
                            const float* lse, const void* dout, void* dq, void* dk, void* dv, int B,
                            int L, int n, int Hq, int Hkv, int Dh, float softmax_scale,
                            sfa_mode_t mode, int window, int32_t* dev_status, cudaStream_t stream);

/* Human-readable name of a status code (static string). */
const char* hd_status_string(hd_status_t status);

/*
 * hd_selftest_bounded_wait -- diagnostic of the failure path shared by the tensor-core
 * kernels (no counterpart in the paper).  Launches one warp that waits, with the same
 * bounded mbarrier wait those kernels use, on a barrier nothing arrives on.  After the
 * bound (about a second) the wait gives up: HD_DEVBIT_TIMEOUT is ORed into *dev_status
 * and *dev_result is set to 0 (1 would mean the wait completed).  No fault, no trap: the
 * kernel returns and the context stays usable.
 *   dev_status, dev_result: device int32 words (dev_status may be NULL; dev_result not).
 */
hd_status_t hd_selftest_bounded_wait(int32_t* dev_status, int32_t* dev_result, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* HDSFA_H */
