// C ABI of libhdsfa.so (declared in include/hdsfa.h): host-side validation,
// problem geometry and kernel dispatch.  No allocation, no synchronisation.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "common.cuh"
#include "decode_plan.cuh"
#include "nvtx_range.h"

namespace hdsfa {
cudaError_t launch_expand_embed(const void* tables, const int32_t* ids, void* out, int B, int L,
                                int n, int V, int D, int32_t* status, cudaStream_t stream);
size_t expand_bwd_ws_bytes(long long N);
cudaError_t launch_expand_bwd_plan(const int32_t* ids, int B, int L, int V, void* ws, int32_t* status,
                                   cudaStream_t st);
cudaError_t launch_expand_bwd_apply(const void* dx, float* de, int B, int L, int n, int V, int D, const void* ws,
                                    cudaStream_t st);
cudaError_t launch_select_final(const void* x, void* y, int B, int L, int n, int D, cudaStream_t st);
cudaError_t launch_select_final_bwd(const void* dy, void* dx, int B, int L, int n, int D, cudaStream_t st);
cudaError_t launch_sfa_decode(const void* q, const void* kc, const void* vc, const int32_t* lens, void* o,
                              float* lse, int B, int maxT, int Lcap, int n, int Hq, int Hkv, int Dh, float scale,
                              int mode, int window, void* ws, int32_t* status, cudaStream_t st);
cudaError_t launch_bounded_wait_selftest(int32_t* status, int32_t* result, cudaStream_t st);
cudaError_t launch_kv_append(const void* kn, const void* vn, void* kc, void* vc, const int32_t* lens, int B,
                             int Lcap, int n, int Hkv, int Dh, int32_t* status, cudaStream_t st);
cudaError_t launch_sfa_fwd_tc(const void* q, const void* k, const void* v, void* o, float* lse,
                              const SfaGeom& g, int Dh, float scale, int32_t* status, cudaStream_t st);
cudaError_t launch_sfa_fwd_tc256(const void* q, const void* k, const void* v, void* o, float* lse,
                                 const SfaGeom& g, float scale, int32_t* status, cudaStream_t st);
cudaError_t launch_sfa_bwd_prep(const void* o, const void* dout, const float* lse, float* lse2_ws,
                                float* delta_ws, float* dq_ws, const SfaGeom& g, int Dh,
                                cudaStream_t st, bool zero = true);
cudaError_t launch_sfa_bwd_clear(float* dq_ws, const SfaGeom& g, int Dh, cudaStream_t st);
cudaError_t launch_sfa_bwd_main_tc(const void* q, const void* k, const void* v, const void* dout, void* dk,
                                   void* dv, const float* lse2_ws, const float* delta_ws, float* dq_ws,
                                   float* dkv_ws, const SfaGeom& g, int Dh, float scale, int32_t* status,
                                   cudaStream_t st);
cudaError_t launch_sfa_bwd_main_tc256(const void* q, const void* k, const void* v, const void* dout, void* dk,
                                      void* dv, const float* lse2_ws, const float* delta_ws, float* dq_ws,
                                      float* dkv_ws, const SfaGeom& g, float scale, int32_t* status,
                                      cudaStream_t st);
cudaError_t launch_sfa_bwd_finalize(void* dq, const float* dq_ws, const SfaGeom& g, int Dh,
                                    float scale, cudaStream_t st);
}  // namespace hdsfa

namespace {

bool aligned16(const void* p) { return p != nullptr && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Validates sizes shared by sfa_fwd / sfa_bwd and builds the virtual-problem geometry.

hd_status_t make_geom(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode, int window,
                      SfaGeom* g) {
  if (B <= 0 || L <= 0 || n <= 0 || Hq <= 0 || Hkv <= 0 || Dh <= 0) return HD_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return HD_ERR_INVALID_ARG;
  if (mode != SFA_WITHIN && mode != SFA_CROSS && mode != SFA_LOCAL && mode != SFA_WITHIN_NAIVE)
    return HD_ERR_INVALID_ARG;
  if (mode == SFA_LOCAL && window <= 0) return HD_ERR_INVALID_ARG;
  if (Dh != 64 && Dh != 128 && Dh != 256) return HD_ERR_UNSUPPORTED;
  // the naive schedule exists on the head-dim-128 kernels only
  if (mode == SFA_WITHIN_NAIVE && Dh != 128) return HD_ERR_UNSUPPORTED;
  const long long nL = (long long)n * L;
  // Every row index, head product and tile count must fit the kernels' int math.
  if (nL > (1LL << 30) || (long long)B * nL * Hq > (1LL << 31) / 2) return HD_ERR_UNSUPPORTED;
  g->B = B;
  g->nL = (int)nL;
  g->Hq = Hq;
  g->Hkv = Hkv;
  g->n = n;
  if (mode == SFA_WITHIN) {
    g->Lv = L;
    g->ns = n;
    g->rs = n;
    g->window = 0;
  } else {  // CROSS, LOCAL, and the naive WITHIN schedule
    g->Lv = (int)nL;
    g->ns = 1;
    g->rs = 1;
    g->window = mode == SFA_LOCAL ? window : 0;
  }
  g->smod = mode == SFA_WITHIN_NAIVE ? n : 0;
  // queries are the key rows themselves
  g->Lq = g->Lv;
  g->qstep = 1;
  g->qoff = 0;
  g->q_nL = g->nL;
  g->q_ns = g->ns;
  g->q_rs = g->rs;
  g->kv_s0 = 0;
  return HD_OK;
}

// A final-stream problem: the L final-stream queries (positions t*n + n-1, the rows
// the loss reads, Eq. 2) in dense [B][L] tensors against the keys of the layer's mask.
hd_status_t make_final_geom(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode, int window,
                            SfaGeom* g) {
  if (mode == SFA_WITHIN_NAIVE) return HD_ERR_UNSUPPORTED;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, window, g);
  if (st != HD_OK) return st;
  g->Lq = L;
  g->q_nL = L;
  g->q_ns = 1;
  g->q_rs = 1;
  if (mode == SFA_WITHIN) {  // the problem of stream n-1: query row t is its key row t
    g->qstep = 1;
    g->qoff = 0;
    g->kv_s0 = n - 1;
  } else {  // query row t at position t*n + n-1 of the nL key rows
    g->qstep = n;
    g->qoff = n - 1;
    g->kv_s0 = 0;
  }
  return HD_OK;
}

float resolve_scale(float s, int Dh) { return s > 0.f ? s : 1.0f / sqrtf((float)Dh); }

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Workspace layout: fp32 dQ accumulator [B][nL][Hq][Dh], then -lse*log2(e) and
// -delta, each fp32 [B][Hq][ns][Lvp] (stream-major rows, Lvp = row_terms_pitch(Lv)),
// then on small grids the fp32 dV / dK partial sums of the head chunks, one slice per
// chunk (bwd_dkv_slice elements each).
struct BwdWs {
  float* dq;
  float* lse2;
  float* delta;
  float* dkv;
};

// Sizes follow the query side (query_geom): the accumulator and row terms are per query row.
size_t ws_bytes(const SfaGeom& gk, int Dh) {
  const SfaGeom g = query_geom(gk);
  const size_t rows = (size_t)g.B * g.nL * g.Hq;
  const size_t trows = (size_t)g.B * g.Hq * g.ns * (size_t)row_terms_pitch(g.Lv);
  const size_t dkv = (size_t)bwd_head_chunks(gk, Dh) * 2 * bwd_dkv_slice(gk, Dh) * sizeof(float);
  return align256(rows * Dh * sizeof(float)) + 2 * align256(trows * sizeof(float)) + align256(dkv);
}

hd_status_t split_ws(const SfaGeom& gk, int Dh, void* ws, size_t bytes, BwdWs* out) {
  if (ws == nullptr || bytes < ws_bytes(gk, Dh) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return HD_ERR_WORKSPACE;
  const SfaGeom g = query_geom(gk);
  const size_t rows = (size_t)g.B * g.nL * g.Hq;
  const size_t trows = (size_t)g.B * g.Hq * g.ns * (size_t)row_terms_pitch(g.Lv);
  char* p = static_cast<char*>(ws);
  out->dq = reinterpret_cast<float*>(p);
  p += align256(rows * Dh * sizeof(float));
  out->lse2 = reinterpret_cast<float*>(p);
  p += align256(trows * sizeof(float));
  out->delta = reinterpret_cast<float*>(p);
  p += align256(trows * sizeof(float));
  out->dkv = bwd_dkv_slice(gk, Dh) > 0 ? reinterpret_cast<float*>(p) : nullptr;
  return HD_OK;
}

hd_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? HD_OK : HD_ERR_CUDA; }

}  // namespace

extern "C" {

hd_status_t hd_expand_embed(const void* tables, const int32_t* ids, void* out, int B, int L, int n,
                            int V, int D, int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("hd_expand_embed");
  if (!aligned16(tables) || !aligned16(out) || ids == nullptr) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || n <= 0 || V <= 0 || D <= 0 || D % 8 != 0) return HD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(ids) & 3u) != 0) return HD_ERR_INVALID_ARG;
  return hdsfa::launch_expand_embed(tables, ids, out, B, L, n, V, D, dev_status, stream) == cudaSuccess
             ? HD_OK
             : HD_ERR_CUDA;
}

size_t hd_expand_embed_bwd_workspace_bytes(int B, int L) {
  if (B <= 0 || L <= 0 || (long long)B * L >= (1LL << 31)) return 0;
  return hdsfa::expand_bwd_ws_bytes((long long)B * L);
}

hd_status_t hd_expand_embed_bwd_plan(const int32_t* ids, int B, int L, int V, void* workspace,
                                     size_t workspace_bytes, int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("hd_expand_embed_bwd_plan");
  if (ids == nullptr || (reinterpret_cast<uintptr_t>(ids) & 3u) != 0) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || V <= 0) return HD_ERR_INVALID_ARG;
  const size_t need = hd_expand_embed_bwd_workspace_bytes(B, L);
  if (need == 0) return HD_ERR_UNSUPPORTED;
  if (!aligned16(workspace) || workspace_bytes < need) return HD_ERR_WORKSPACE;
  return cuda_status(hdsfa::launch_expand_bwd_plan(ids, B, L, V, workspace, dev_status, stream));
}

hd_status_t hd_expand_embed_bwd_apply(const void* dout, float* dtables, int B, int L, int n, int V, int D,
                                      const void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  HD_NVTX_RANGE("hd_expand_embed_bwd_apply");
  if (!aligned16(dout) || !aligned16(dtables)) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || n <= 0 || V <= 0 || D <= 0 || D % 8 != 0) return HD_ERR_INVALID_ARG;
  const size_t need = hd_expand_embed_bwd_workspace_bytes(B, L);
  if (need == 0 || (long long)n * D >= (1LL << 31)) return HD_ERR_UNSUPPORTED;
  if (!aligned16(workspace) || workspace_bytes < need) return HD_ERR_WORKSPACE;
  return cuda_status(hdsfa::launch_expand_bwd_apply(dout, dtables, B, L, n, V, D, workspace, stream));
}

hd_status_t hd_expand_embed_bwd(const void* dout, const int32_t* ids, float* dtables, int B, int L, int n,
                                int V, int D, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                                cudaStream_t stream) {
  HD_NVTX_RANGE("hd_expand_embed_bwd");
  // every argument is checked before the plan is enqueued
  if (!aligned16(dout) || !aligned16(dtables) || ids == nullptr) return HD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(ids) & 3u) != 0) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || n <= 0 || V <= 0 || D <= 0 || D % 8 != 0) return HD_ERR_INVALID_ARG;
  const size_t need = hd_expand_embed_bwd_workspace_bytes(B, L);
  if (need == 0 || (long long)n * D >= (1LL << 31)) return HD_ERR_UNSUPPORTED;
  if (!aligned16(workspace) || workspace_bytes < need) return HD_ERR_WORKSPACE;
  hd_status_t st = hd_expand_embed_bwd_plan(ids, B, L, V, workspace, workspace_bytes, dev_status, stream);
  if (st != HD_OK) return st;
  return hd_expand_embed_bwd_apply(dout, dtables, B, L, n, V, D, workspace, workspace_bytes, stream);
}

hd_status_t hd_select_final_stream(const void* x, void* y, int B, int L, int n, int D, cudaStream_t stream) {
  HD_NVTX_RANGE("hd_select_final_stream");
  if (!aligned16(x) || !aligned16(y)) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || n <= 0 || D <= 0 || D % 8 != 0) return HD_ERR_INVALID_ARG;
  return cuda_status(hdsfa::launch_select_final(x, y, B, L, n, D, stream));
}

hd_status_t hd_select_final_stream_bwd(const void* dy, void* dx, int B, int L, int n, int D,
                                       cudaStream_t stream) {
  HD_NVTX_RANGE("hd_select_final_stream_bwd");
  if (!aligned16(dy) || !aligned16(dx)) return HD_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || n <= 0 || D <= 0 || D % 8 != 0) return HD_ERR_INVALID_ARG;
  return cuda_status(hdsfa::launch_select_final_bwd(dy, dx, B, L, n, D, stream));
}

hd_status_t sfa_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B, int L,
                    int n, int Hq, int Hkv, int Dh, float softmax_scale, sfa_mode_t mode,
                    int window, int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_fwd");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse))
    return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, window, &g);
  if (st != HD_OK) return st;
  const float scale = resolve_scale(softmax_scale, Dh);
  // head dim 256: one query tile per CTA (its O takes half of TMEM)
  if (Dh == 256) return cuda_status(hdsfa::launch_sfa_fwd_tc256(q, k, v, o, lse, g, scale, dev_status, stream));
  return cuda_status(hdsfa::launch_sfa_fwd_tc(q, k, v, o, lse, g, Dh, scale, dev_status, stream));
}

size_t sfa_bwd_workspace_bytes(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode) {
  SfaGeom g;
  if (make_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g) != HD_OK) return 0;
  return ws_bytes(g, Dh);
}

hd_status_t sfa_bwd_prep(const void* o, const void* dout, const float* lse, int B, int L, int n, int Hq,
                         int Hkv, int Dh, sfa_mode_t mode, void* workspace, size_t workspace_bytes,
                         cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_prep");
  if (!aligned16(o) || !aligned16(dout) || !aligned16(lse)) return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  return cuda_status(hdsfa::launch_sfa_bwd_prep(o, dout, lse, ws.lse2, ws.delta, ws.dq, query_geom(g), Dh, stream));
}

hd_status_t sfa_bwd_row_terms(const void* o, const void* dout, const float* lse, int B, int L, int n, int Hq,
                              int Hkv, int Dh, sfa_mode_t mode, void* workspace, size_t workspace_bytes,
                              cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_row_terms");
  if (!aligned16(o) || !aligned16(dout) || !aligned16(lse)) return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  return cuda_status(
      hdsfa::launch_sfa_bwd_prep(o, dout, lse, ws.lse2, ws.delta, ws.dq, query_geom(g), Dh, stream, false));
}

hd_status_t sfa_bwd_clear(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode, void* workspace,
                          size_t workspace_bytes, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_clear");
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  return cuda_status(hdsfa::launch_sfa_bwd_clear(ws.dq, query_geom(g), Dh, stream));
}

hd_status_t sfa_bwd_main(const void* q, const void* k, const void* v, const void* dout, void* dk, void* dv,
                         int B, int L, int n, int Hq, int Hkv, int Dh, float softmax_scale,
                         sfa_mode_t mode, int window, void* workspace, size_t workspace_bytes,
                         int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_main");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(dout) || !aligned16(dk) ||
      !aligned16(dv))
    return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, window, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  const float scale = resolve_scale(softmax_scale, Dh);
  // tcgen05 kernels at every head dim (at 256 as two CTAs per key tile, one per half
  // of the dK / dV / dQ columns)
  if (Dh == 256)
    return cuda_status(hdsfa::launch_sfa_bwd_main_tc256(q, k, v, dout, dk, dv, ws.lse2, ws.delta, ws.dq, ws.dkv, g,
                                                        scale, dev_status, stream));
  return cuda_status(hdsfa::launch_sfa_bwd_main_tc(q, k, v, dout, dk, dv, ws.lse2, ws.delta, ws.dq, ws.dkv, g, Dh,
                                                   scale, dev_status, stream));
}

hd_status_t sfa_bwd_finalize(void* dq, int B, int L, int n, int Hq, int Hkv, int Dh,
                             float softmax_scale, sfa_mode_t mode, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_finalize");
  if (!aligned16(dq)) return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  return cuda_status(hdsfa::launch_sfa_bwd_finalize(dq, ws.dq, query_geom(g), Dh,
                                                    resolve_scale(softmax_scale, Dh), stream));
}

hd_status_t sfa_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                    const void* dout, void* dq, void* dk, void* dv, int B, int L, int n, int Hq,
                    int Hkv, int Dh, float softmax_scale, sfa_mode_t mode, int window,
                    void* workspace, size_t workspace_bytes, int32_t* dev_status,
                    cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse) ||
      !aligned16(dout) || !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
    return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_geom(B, L, n, Hq, Hkv, Dh, mode, window, &g);
  if (st != HD_OK) return st;
  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  st = sfa_bwd_prep(o, dout, lse, B, L, n, Hq, Hkv, Dh, mode, workspace, workspace_bytes, stream);
  if (st != HD_OK) return st;
  st = sfa_bwd_main(q, k, v, dout, dk, dv, B, L, n, Hq, Hkv, Dh, softmax_scale, mode, window, workspace,
                    workspace_bytes, dev_status, stream);
  if (st != HD_OK) return st;
  return sfa_bwd_finalize(dq, B, L, n, Hq, Hkv, Dh, softmax_scale, mode, workspace,
                          workspace_bytes, stream);
}

// Sizes of a decode step: max_tokens bounds every sequence's length and the cache
// capacity Lcap bounds max_tokens.
static hd_status_t decode_sizes(int B, int maxT, int Lcap, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode,
                                int window) {
  if (B <= 0 || maxT <= 0 || Lcap <= 0 || n <= 0 || Hq <= 0 || Hkv <= 0 || Dh <= 0) return HD_ERR_INVALID_ARG;
  if (Hq % Hkv != 0 || maxT > Lcap) return HD_ERR_INVALID_ARG;
  if (mode != SFA_WITHIN && mode != SFA_CROSS && mode != SFA_LOCAL) return HD_ERR_INVALID_ARG;
  if (mode == SFA_LOCAL && window <= 0) return HD_ERR_INVALID_ARG;
  if (Dh != 64 && Dh != 128 && Dh != 256) return HD_ERR_UNSUPPORTED;
  if ((long long)Lcap * n > (1LL << 30) || (long long)n * Hq > (1LL << 20)) return HD_ERR_UNSUPPORTED;
  return HD_OK;
}

size_t sfa_decode_workspace_bytes(int B, int max_tokens, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode,
                                  int window) {
  if (decode_sizes(B, max_tokens, max_tokens, n, Hq, Hkv, Dh, mode, window) != HD_OK) return 0;
  return hdsfa::decode_ws_bytes(hdsfa::decode_plan(B, max_tokens, n, Hq, Hkv, Dh, mode, window));
}

hd_status_t sfa_decode(const void* q, const void* k_cache, const void* v_cache, const int32_t* lens, void* o,
                       float* lse, int B, int max_tokens, int Lcap, int n, int Hq, int Hkv, int Dh,
                       float softmax_scale, sfa_mode_t mode, int window, void* workspace, size_t workspace_bytes,
                       int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_decode");
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(o)) return HD_ERR_INVALID_ARG;
  if (lens == nullptr || (reinterpret_cast<uintptr_t>(lens) & 3u) != 0) return HD_ERR_INVALID_ARG;
  if (lse != nullptr && (reinterpret_cast<uintptr_t>(lse) & 3u) != 0) return HD_ERR_INVALID_ARG;
  hd_status_t st = decode_sizes(B, max_tokens, Lcap, n, Hq, Hkv, Dh, mode, window);
  if (st != HD_OK) return st;
  const size_t need = sfa_decode_workspace_bytes(B, max_tokens, n, Hq, Hkv, Dh, mode, window);
  if (!aligned16(workspace) || workspace_bytes < need) return HD_ERR_WORKSPACE;
  return cuda_status(hdsfa::launch_sfa_decode(q, k_cache, v_cache, lens, o, lse, B, max_tokens, Lcap, n, Hq, Hkv,
                                              Dh, resolve_scale(softmax_scale, Dh), (int)mode,
                                              mode == SFA_LOCAL ? window : 0, workspace, dev_status, stream));
}

hd_status_t sfa_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache, const int32_t* lens,
                          int B, int Lcap, int n, int Hkv, int Dh, int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_kv_append");
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache))
    return HD_ERR_INVALID_ARG;
  if (lens == nullptr || (reinterpret_cast<uintptr_t>(lens) & 3u) != 0) return HD_ERR_INVALID_ARG;
  if (B <= 0 || Lcap <= 0 || n <= 0 || Hkv <= 0 || Dh <= 0 || Dh % 8 != 0) return HD_ERR_INVALID_ARG;
  if ((long long)Lcap * n > (1LL << 30)) return HD_ERR_UNSUPPORTED;
  return cuda_status(hdsfa::launch_kv_append(k_new, v_new, k_cache, v_cache, lens, B, Lcap, n, Hkv, Dh,
                                             dev_status, stream));
}

// ---- final-stream problems (Eq. 2 rows; Sec. 3.1 final-stream-only layers) ----
hd_status_t sfa_fwd_final(const void* q, const void* k, const void* v, void* o, float* lse, int B, int L, int n,
                          int Hq, int Hkv, int Dh, float softmax_scale, sfa_mode_t mode, int window,
                          int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_fwd_final");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse))
    return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_final_geom(B, L, n, Hq, Hkv, Dh, mode, window, &g);
  if (st != HD_OK) return st;
  const float scale = resolve_scale(softmax_scale, Dh);
  if (Dh == 256) return cuda_status(hdsfa::launch_sfa_fwd_tc256(q, k, v, o, lse, g, scale, dev_status, stream));
  return cuda_status(hdsfa::launch_sfa_fwd_tc(q, k, v, o, lse, g, Dh, scale, dev_status, stream));
}

size_t sfa_bwd_final_workspace_bytes(int B, int L, int n, int Hq, int Hkv, int Dh, sfa_mode_t mode) {
  SfaGeom g;
  if (make_final_geom(B, L, n, Hq, Hkv, Dh, mode, mode == SFA_LOCAL ? 1 : 0, &g) != HD_OK) return 0;
  return ws_bytes(g, Dh);
}

hd_status_t sfa_bwd_final(const void* q, const void* k, const void* v, const void* o, const float* lse,
                          const void* dout, void* dq, void* dk, void* dv, int B, int L, int n, int Hq, int Hkv,
                          int Dh, float softmax_scale, sfa_mode_t mode, int window, void* workspace,
                          size_t workspace_bytes, int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_final");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse) ||
      !aligned16(dout) || !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
    return HD_ERR_INVALID_ARG;
  SfaGeom g;
  hd_status_t st = make_final_geom(B, L, n, Hq, Hkv, Dh, mode, window, &g);
  if (st != HD_OK) return st;

  BwdWs ws;
  if ((st = split_ws(g, Dh, workspace, workspace_bytes, &ws)) != HD_OK) return st;
  const float scale = resolve_scale(softmax_scale, Dh);
  const SfaGeom gq = query_geom(g);
  cudaError_t e = hdsfa::launch_sfa_bwd_prep(o, dout, lse, ws.lse2, ws.delta, ws.dq, gq, Dh, stream);
  if (e == cudaSuccess && mode == SFA_WITHIN) {
    // only stream n-1's keys are seen by the final-stream queries: the other rows are zero
    const size_t bytes = (size_t)B * n * L * Hkv * Dh * 2;
    e = cudaMemsetAsync(dk, 0, bytes, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(dv, 0, bytes, stream);
  }
  if (e == cudaSuccess) {
    if (Dh == 256)
      e = hdsfa::launch_sfa_bwd_main_tc256(q, k, v, dout, dk, dv, ws.lse2, ws.delta, ws.dq, ws.dkv, g, scale, dev_status,
                                           stream);
    else
      e = hdsfa::launch_sfa_bwd_main_tc(q, k, v, dout, dk, dv, ws.lse2, ws.delta, ws.dq, ws.dkv, g, Dh, scale, dev_status,
                                        stream);
  }
  if (e == cudaSuccess) e = hdsfa::launch_sfa_bwd_finalize(dq, ws.dq, gq, Dh, scale, stream);
  return cuda_status(e);
}

hd_status_t hd_selftest_bounded_wait(int32_t* dev_status, int32_t* dev_result, cudaStream_t stream) {
  HD_NVTX_RANGE("hd_selftest_bounded_wait");
  if (dev_result == nullptr || (reinterpret_cast<uintptr_t>(dev_result) & 3u) != 0) return HD_ERR_INVALID_ARG;
  if (dev_status != nullptr && (reinterpret_cast<uintptr_t>(dev_status) & 3u) != 0) return HD_ERR_INVALID_ARG;
  return cuda_status(hdsfa::launch_bounded_wait_selftest(dev_status, dev_result, stream));
}

const char* hd_status_string(hd_status_t s) {
  switch (s) {
    case HD_OK: return "HD_OK";
    case HD_ERR_INVALID_ARG: return "HD_ERR_INVALID_ARG: invalid argument";
    case HD_ERR_UNSUPPORTED: return "HD_ERR_UNSUPPORTED: configuration not supported";
    case HD_ERR_CUDA: return "HD_ERR_CUDA: CUDA launch or runtime error";
    case HD_ERR_WORKSPACE: return "HD_ERR_WORKSPACE: workspace missing, misaligned or too small";
    case HD_ERR_TIMEOUT: return "HD_ERR_TIMEOUT: bounded device wait expired";
    case HD_ERR_INDEX: return "HD_ERR_INDEX: index out of range";
    case HD_ERR_SCRATCH_LIMIT:
      return "HD_ERR_SCRATCH_LIMIT: sizes need more workspace than sfa_bwd_noalloc's fixed array";
  }
  return "unknown hd_status_t";
}

}  // extern "C"
