/*
 * hdsfa_oracle.c -- fp64 CPU oracle for Hidden Decoding's stream expansion and
 * Stream-Factorized Attention (SFA).
 *
 * TEST INFRASTRUCTURE ONLY.  This file exists so the CUDA path can be checked
 * against a plain, slow, obviously correct restatement of the method.  Only the
 * tests, the smoke check and the benchmark's CPU-baseline leg load it; the
 * product library never links, loads or calls it, and it shares no code,
 * header, table or helper with the CUDA sources.
 *
 * What it computes (all citations are to the Hidden Decoding paper):
 *   - Eq. 1  : the expanded sequence S_t = E_k(x_i) at position t = (i-1)n + k, and
 *              its adjoint (the gradient with respect to the n tables).
 *   - Eq. 2  : the final-stream positions t = i n that the loss reads, and their
 *              adjoint.
 *   - Sec. 3.2 "Inference Cost": decoding, where each new token's n positions
 *              attend to the expanded KV cache (the forward's rows for that token),
 *              and the cache append of the new token's n K/V rows.
 *   - Eq. 3  : token index i(t) = ceil(t/n) and stream index s(t) = ((t-1) mod n) + 1.
 *   - Eq. 4  : the intra-stream mask M[t,t'] = 1[t' <= t and s(t') = s(t)] (WITHIN).
 *   - Fig. 2a: the full cross-stream layer, the standard causal mask over all
 *              nL positions (CROSS); Sec. 2.1 feeds the expanded sequence to the
 *              backbone "under standard causal attention".
 *   - Fig. 2b: the local cross-stream layer, a causal sliding window (LOCAL);
 *              the paper gives no window size, so it is a parameter w counted in
 *              expanded positions: t - w < t' <= t.
 *   - Sec. 2 "Setup": the backbone's standard (masked) softmax attention with
 *              grouped K/V heads (Table 6 "Q/KV heads"): query head h reads K/V
 *              head g(h) = h / (Hq / Hkv).
 *   The paper never writes the attention gradient; the backward here is the
 *   derivative of that forward, written out from the softmax Jacobian.
 *
 * Arithmetic is fp64 throughout; bf16 inputs are upcast exactly by the caller.
 * Layouts (0-indexed, row-major, contiguous):
 *   q, o, dout, dq : [B][nL][Hq][Dh]      k, v, dk, dv : [B][nL][Hkv][Dh]
 *   lse, delta     : [B][Hq][nL]          (natural-log log-sum-exp)
 * Position p (0-indexed) is the paper's t = p + 1.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { HDO_WITHIN = 0, HDO_CROSS = 1, HDO_LOCAL = 2 };

typedef struct {
  int64_t B, L, n, Hq, Hkv, Dh;
  int mode;
  int64_t window; /* LOCAL only: key t' visible iff t - window < t' <= t */
  double scale;
} hdo_dims;

/* ---- Eq. 3: token and stream index of a 1-indexed expanded position t ---- */
int64_t hdo_token_index(int64_t t, int64_t n) { return (t + n - 1) / n; } /* ceil(t/n) */
int64_t hdo_stream_index(int64_t t, int64_t n) { return ((t - 1) % n) + 1; }

/* ---- Eq. 4 and Fig. 2: may query position t attend to key position tk? ----
 * t and tk are the paper's 1-indexed expanded positions. */
int hdo_visible(int64_t t, int64_t tk, int64_t n, int mode, int64_t window) {
  switch (mode) {
    case HDO_WITHIN: /* Eq. 4 */
      return tk <= t && hdo_stream_index(tk, n) == hdo_stream_index(t, n);
    case HDO_CROSS: /* Fig. 2a: causal over the whole expanded sequence */
      return tk <= t;
    case HDO_LOCAL: /* Fig. 2b: causal sliding window of w positions */
      return tk <= t && tk > t - window;
    default:
      return 0;
  }
}

/* ---- Eq. 1: expansion gather ----
 * tables: bf16 bit patterns [n][V][D]; ids: [B][L]; out: [B][n*L][D].
 * A token id outside [0, V) yields a zero row; the return value counts them. */
int64_t hdo_expand(const uint16_t* tables, const int32_t* ids, uint16_t* out,
                   int64_t B, int64_t L, int64_t n, int64_t V, int64_t D) {
  int64_t bad = 0;
  for (int64_t b = 0; b < B; ++b) {
    for (int64_t i = 1; i <= L; ++i) {     /* token x_i, 1-indexed */
      int32_t x = ids[b * L + (i - 1)];
      for (int64_t k = 1; k <= n; ++k) {   /* stream k, 1-indexed */
        int64_t t = (i - 1) * n + k;       /* physical position (Eq. 1) */
        uint16_t* dst = out + (b * n * L + (t - 1)) * D;
        if (x < 0 || x >= V) {
          memset(dst, 0, (size_t)D * sizeof(uint16_t));
          if (k == 1) ++bad;
          continue;
        }
        const uint16_t* src = tables + ((k - 1) * V + x) * D; /* E_k(x_i) */
        memcpy(dst, src, (size_t)D * sizeof(uint16_t));
      }
    }
  }
  return bad;
}

/* ---- Eq. 1 backward: the adjoint of the expansion gather ----
 * The forward copies E_k(x_i) to position t = (i-1)n + k, so the gradient of the
 * loss with respect to row x of table k is the sum of the position gradients of
 * every token i with x_i = x, taken at stream k:
 *   dE_k[x] += sum_{i : x_i = x} dS_{(i-1)n+k}.
 * dX: [B][n*L][D] fp64; ids: [B][L]; dE: [n][V][D] fp64, accumulated (not cleared).
 * An id outside [0, V) contributes nothing (its rows were zero in the forward). */
void hdo_expand_bwd(const double* dX, const int32_t* ids, double* dE, int64_t B, int64_t L,
                    int64_t n, int64_t V, int64_t D) {
  for (int64_t b = 0; b < B; ++b) {
    for (int64_t i = 1; i <= L; ++i) {
      int32_t x = ids[b * L + (i - 1)];
      if (x < 0 || x >= V) continue;
      for (int64_t k = 1; k <= n; ++k) {
        int64_t t = (i - 1) * n + k;
        const double* src = dX + (b * n * L + (t - 1)) * D;
        double* dst = dE + ((k - 1) * V + x) * D;
        for (int64_t c = 0; c < D; ++c) dst[c] += src[c];
      }
    }
  }
}

/* ---- Eq. 2: the supervised (final-stream) positions ----
 * Only the final stream of each token is supervised: the loss reads the hidden
 * state at 1-indexed position t = i n.  select: Y[b][i-1] = X[b][i n - 1] (0-indexed
 * rows of D bf16 bit patterns); its adjoint writes dY back to those rows and zero
 * to every other position. */
void hdo_select_final(const uint16_t* X, uint16_t* Y, int64_t B, int64_t L, int64_t n, int64_t D) {
  for (int64_t b = 0; b < B; ++b)
    for (int64_t i = 1; i <= L; ++i)
      memcpy(Y + (b * L + (i - 1)) * D, X + (b * n * L + (i * n - 1)) * D, (size_t)D * sizeof(uint16_t));
}

void hdo_select_final_bwd(const uint16_t* dY, uint16_t* dX, int64_t B, int64_t L, int64_t n, int64_t D) {
  memset(dX, 0, (size_t)(B * n * L * D) * sizeof(uint16_t));
  for (int64_t b = 0; b < B; ++b)
    for (int64_t i = 1; i <= L; ++i)
      memcpy(dX + (b * n * L + (i * n - 1)) * D, dY + (b * L + (i - 1)) * D, (size_t)D * sizeof(uint16_t));
}

/* ---------------------------------------------------------------- helpers */
static inline const double* qrow(const double* q, const hdo_dims* d, int64_t b, int64_t p, int64_t h) {
  return q + ((b * d->n * d->L + p) * d->Hq + h) * d->Dh;
}
static inline const double* kvrow(const double* k, const hdo_dims* d, int64_t b, int64_t p, int64_t g) {
  return k + ((b * d->n * d->L + p) * d->Hkv + g) * d->Dh;
}
static inline double dot(const double* a, const double* b, int64_t n) {
  double s = 0.0;
  for (int64_t i = 0; i < n; ++i) s += a[i] * b[i];
  return s;
}
static inline int64_t kv_head(const hdo_dims* d, int64_t h) { return h / (d->Hq / d->Hkv); }
static inline int vis0(const hdo_dims* d, int64_t p, int64_t pk) {
  return hdo_visible(p + 1, pk + 1, d->n, d->mode, d->window);
}

/* Scores z[p'] = scale * q_p . k_p' over the visible keys of row p, and the row's
 * natural-log log-sum-exp.  Invisible entries of z are left untouched. */
static double row_scores(const double* q, const double* k, const hdo_dims* d,
                         int64_t b, int64_t h, int64_t p, double* z) {
  const int64_t nL = d->n * d->L, g = kv_head(d, h);
  const double* qp = qrow(q, d, b, p, h);
  double m = -INFINITY;
  for (int64_t pk = 0; pk < nL; ++pk) {
    if (!vis0(d, p, pk)) continue;
    z[pk] = d->scale * dot(qp, kvrow(k, d, b, pk, g), d->Dh);
    if (z[pk] > m) m = z[pk];
  }
  double sum = 0.0;
  for (int64_t pk = 0; pk < nL; ++pk)
    if (vis0(d, p, pk)) sum += exp(z[pk] - m);
  return m + log(sum);
}

/* ---- Decoding with the expanded KV cache (Sec. 3.2 "Inference Cost") ----
 * Generation processes each new token's n streams together in one forward pass.
 * With i = lens[b] tokens of sequence b in the cache (the new token i included, its
 * K/V already stored), the new token's positions t = (i-1)n + k, k = 1..n, attend
 * under the layer's mask (Eq. 4, Fig. 2) to the cached positions 1 .. i n: the same
 * masked softmax attention as the forward, for the new token's rows only.  Intra-stream
 * layers thus read only their own stream's cached keys; cross-stream layers read all.
 *   q, o   : [B][n][Hq][Dh] (row k-1 = stream k of the new token)
 *   kc, vc : [B][Lcap n][Hkv][Dh] (position t at row t-1)
 *   lens   : [B], tokens in the cache, valid in [1, Lcap]
 *   lse    : [B][Hq][n] natural log
 * A sequence whose lens is outside [1, Lcap] gets zero rows and lse = -inf; the
 * return value counts such sequences. */
int64_t hdo_decode(const double* q, const double* kc, const double* vc, const int32_t* lens, double* o,
                   double* lse, int64_t B, int64_t Lcap, int64_t n, int64_t Hq, int64_t Hkv, int64_t Dh,
                   double scale, int mode, int64_t window) {
  int64_t bad = 0;
  for (int64_t b = 0; b < B; ++b) {
    const int64_t i = lens[b];
    const int valid = i >= 1 && i <= Lcap;
    if (!valid) ++bad;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t k = 1; k <= n; ++k) {
      for (int64_t h = 0; h < Hq; ++h) {
        const double* qr = q + ((b * n + (k - 1)) * Hq + h) * Dh;
        double* orow = o + ((b * n + (k - 1)) * Hq + h) * Dh;
        double* l = lse + (b * Hq + h) * n + (k - 1);
        for (int64_t e = 0; e < Dh; ++e) orow[e] = 0.0;
        if (!valid) {
          *l = -INFINITY;
          continue;
        }
        const int64_t t = (i - 1) * n + k, g = h / (Hq / Hkv);
        double m = -INFINITY;
        for (int64_t tk = 1; tk <= i * n; ++tk) {
          if (!hdo_visible(t, tk, n, mode, window)) continue;
          const double z = scale * dot(qr, kc + ((b * Lcap * n + tk - 1) * Hkv + g) * Dh, Dh);
          if (z > m) m = z;
        }
        double sum = 0.0;
        for (int64_t tk = 1; tk <= i * n; ++tk) {
          if (!hdo_visible(t, tk, n, mode, window)) continue;
          const double z = scale * dot(qr, kc + ((b * Lcap * n + tk - 1) * Hkv + g) * Dh, Dh);
          const double w = exp(z - m);
          sum += w;
          const double* vr = vc + ((b * Lcap * n + tk - 1) * Hkv + g) * Dh;
          for (int64_t e = 0; e < Dh; ++e) orow[e] += w * vr[e];
        }
        for (int64_t e = 0; e < Dh; ++e) orow[e] /= sum;
        *l = m + log(sum);
      }
    }
  }
  return bad;
}

/* The new token's K (or V) rows enter the cache at its n positions:
 * cache[b][(i-1)n + k - 1] = new[b][k-1] with i = lens[b] (bf16 bit patterns, rows of
 * Hkv*Dh).  Sequences with lens outside [1, Lcap] are left untouched (counted). */
int64_t hdo_kv_append(const uint16_t* nw, uint16_t* cache, const int32_t* lens, int64_t B, int64_t Lcap,
                      int64_t n, int64_t row) {
  int64_t bad = 0;
  for (int64_t b = 0; b < B; ++b) {
    const int64_t i = lens[b];
    if (i < 1 || i > Lcap) {
      ++bad;
      continue;
    }
    for (int64_t k = 1; k <= n; ++k)
      memcpy(cache + (b * Lcap * n + (i - 1) * n + k - 1) * row, nw + (b * n + k - 1) * row,
             (size_t)row * sizeof(uint16_t));
  }
  return bad;
}

/* ---- forward for one row: O[b,p,h] = sum_p' P[p,p'] V[p'], P = softmax over visible keys */
static void fwd_row(const double* q, const double* k, const double* v, const hdo_dims* d,
                    int64_t b, int64_t h, int64_t p, double* o_row, double* lse_out, double* z) {
  const int64_t nL = d->n * d->L, g = kv_head(d, h);
  double lse = row_scores(q, k, d, b, h, p, z);
  for (int64_t e = 0; e < d->Dh; ++e) o_row[e] = 0.0;
  for (int64_t pk = 0; pk < nL; ++pk) {
    if (!vis0(d, p, pk)) continue;
    double P = exp(z[pk] - lse);
    const double* vr = kvrow(v, d, b, pk, g);
    for (int64_t e = 0; e < d->Dh; ++e) o_row[e] += P * vr[e];
  }
  *lse_out = lse;
}

/* Full forward: every (b, h, p). */
void hdo_sfa_fwd(const double* q, const double* k, const double* v, double* o, double* lse,
                 const hdo_dims* d) {
  const int64_t nL = d->n * d->L;
  const int64_t rows = d->B * d->Hq * nL;
#pragma omp parallel
  {
    double* z = (double*)malloc((size_t)nL * sizeof(double));
#pragma omp for schedule(dynamic, 16)
    for (int64_t r = 0; r < rows; ++r) {
      int64_t b = r / (d->Hq * nL), h = (r / nL) % d->Hq, p = r % nL;
      fwd_row(q, k, v, d, b, h, p, o + ((b * nL + p) * d->Hq + h) * d->Dh,
              lse + (b * d->Hq + h) * nL + p, z);
    }
    free(z);
  }
}

/* Forward for a list of rows; rows[3r..3r+2] = (b, h, p).  o_rows: [nrows][Dh]. */
void hdo_sfa_fwd_rows(const double* q, const double* k, const double* v, const hdo_dims* d,
                      int64_t nrows, const int64_t* rows, double* o_rows, double* lse_rows) {
  const int64_t nL = d->n * d->L;
#pragma omp parallel
  {
    double* z = (double*)malloc((size_t)nL * sizeof(double));
#pragma omp for schedule(dynamic, 1)
    for (int64_t r = 0; r < nrows; ++r)
      fwd_row(q, k, v, d, rows[3 * r], rows[3 * r + 1], rows[3 * r + 2], o_rows + r * d->Dh,
              lse_rows + r, z);
    free(z);
  }
}

/* ---- backward, per query row, reduced softmax-Jacobian form ----
 * With P the row's softmax over visible keys and dP[p'] = dO_p . V[p'], the
 * Jacobian J = diag(P) - P P^T gives dz = J dP = P * (dP - D), D = sum_p' P dP.
 * dQ_p = scale * sum_p' dz[p'] K[p'].
 * Writes dq_row (nullable), and the row statistics lse and D (nullable). */
static void bwd_q_row(const double* q, const double* k, const double* v, const double* dout,
                      const hdo_dims* d, int64_t b, int64_t h, int64_t p, double* dq_row,
                      double* lse_out, double* D_out, double* z, double* dP) {
  const int64_t nL = d->n * d->L, g = kv_head(d, h);
  const double* dop = qrow(dout, d, b, p, h);
  double lse = row_scores(q, k, d, b, h, p, z);
  double D = 0.0;
  for (int64_t pk = 0; pk < nL; ++pk) {
    if (!vis0(d, p, pk)) continue;
    z[pk] = exp(z[pk] - lse); /* z now holds P */
    dP[pk] = dot(dop, kvrow(v, d, b, pk, g), d->Dh);
    D += z[pk] * dP[pk];
  }
  if (dq_row) {
    for (int64_t e = 0; e < d->Dh; ++e) dq_row[e] = 0.0;
    for (int64_t pk = 0; pk < nL; ++pk) {
      if (!vis0(d, p, pk)) continue;
      double dz = z[pk] * (dP[pk] - D);
      const double* kr = kvrow(k, d, b, pk, g);
      for (int64_t e = 0; e < d->Dh; ++e) dq_row[e] += d->scale * dz * kr[e];
    }
  }
  if (lse_out) *lse_out = lse;
  if (D_out) *D_out = D;
}

/* dQ rows plus row statistics for a list of (b, h, p). */
void hdo_sfa_bwd_q_rows(const double* q, const double* k, const double* v, const double* dout,
                        const hdo_dims* d, int64_t nrows, const int64_t* rows, double* dq_rows,
                        double* lse_rows, double* D_rows) {
  const int64_t nL = d->n * d->L;
#pragma omp parallel
  {
    double* z = (double*)malloc((size_t)nL * sizeof(double));
    double* dP = (double*)malloc((size_t)nL * sizeof(double));
#pragma omp for schedule(dynamic, 1)
    for (int64_t r = 0; r < nrows; ++r)
      bwd_q_row(q, k, v, dout, d, rows[3 * r], rows[3 * r + 1], rows[3 * r + 2],
                dq_rows ? dq_rows + r * d->Dh : NULL, lse_rows ? lse_rows + r : NULL,
                D_rows ? D_rows + r : NULL, z, dP);
    free(z);
    free(dP);
  }
}

/* ---- backward, per key row ----
 * For key position p' of K/V head g: the gradient sums, over the query heads h of
 * the group and the query rows p that see p',
 *   dV[p'] = sum P[p,p'] dO_p,   dK[p'] = scale * sum dz[p,p'] Q_p,
 * with P[p,p'] = exp(scale q_p.k_p' - lse[p]) and dz = P (dO_p.v_p' - D[p]).
 * lse and D are full [B][Hq][nL] arrays; only entries of rows that see a
 * requested key are read.  rows[3r..3r+2] = (b, g, p'). */
void hdo_sfa_bwd_kv_rows(const double* q, const double* k, const double* v, const double* dout,
                         const double* lse, const double* D, const hdo_dims* d, int64_t nrows,
                         const int64_t* rows, double* dk_rows, double* dv_rows) {
  const int64_t nL = d->n * d->L, grp = d->Hq / d->Hkv;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < nrows; ++r) {
    int64_t b = rows[3 * r], g = rows[3 * r + 1], pk = rows[3 * r + 2];
    double* dk = dk_rows + r * d->Dh;
    double* dv = dv_rows + r * d->Dh;
    for (int64_t e = 0; e < d->Dh; ++e) dk[e] = dv[e] = 0.0;
    const double* kr = kvrow(k, d, b, pk, g);
    const double* vr = kvrow(v, d, b, pk, g);
    for (int64_t h = g * grp; h < (g + 1) * grp; ++h) {
      for (int64_t p = 0; p < nL; ++p) {
        if (!vis0(d, p, pk)) continue;
        const double* qp = qrow(q, d, b, p, h);
        const double* dop = qrow(dout, d, b, p, h);
        double P = exp(d->scale * dot(qp, kr, d->Dh) - lse[(b * d->Hq + h) * nL + p]);
        double dz = P * (dot(dop, vr, d->Dh) - D[(b * d->Hq + h) * nL + p]);
        for (int64_t e = 0; e < d->Dh; ++e) {
          dv[e] += P * dop[e];
          dk[e] += d->scale * dz * qp[e];
        }
      }
    }
  }
}

/* Full backward: first every query row (dQ, lse, D), then every key row (dK, dV).
 * lse_ws and D_ws are caller-provided [B][Hq][nL] scratch arrays. */
void hdo_sfa_bwd(const double* q, const double* k, const double* v, const double* dout,
                 double* dq, double* dk, double* dv, double* lse_ws, double* D_ws,
                 const hdo_dims* d) {
  const int64_t nL = d->n * d->L;
  const int64_t qrows = d->B * d->Hq * nL, krows = d->B * d->Hkv * nL;
#pragma omp parallel
  {
    double* z = (double*)malloc((size_t)nL * sizeof(double));
    double* dP = (double*)malloc((size_t)nL * sizeof(double));
#pragma omp for schedule(dynamic, 16)
    for (int64_t r = 0; r < qrows; ++r) {
      int64_t b = r / (d->Hq * nL), h = (r / nL) % d->Hq, p = r % nL;
      bwd_q_row(q, k, v, dout, d, b, h, p, dq + ((b * nL + p) * d->Hq + h) * d->Dh,
                lse_ws + (b * d->Hq + h) * nL + p, D_ws + (b * d->Hq + h) * nL + p, z, dP);
    }
    free(z);
    free(dP);
  }
  int64_t* rows = (int64_t*)malloc((size_t)krows * 3 * sizeof(int64_t));
  double* dk_rows = (double*)malloc((size_t)krows * d->Dh * sizeof(double));
  double* dv_rows = (double*)malloc((size_t)krows * d->Dh * sizeof(double));
  for (int64_t r = 0; r < krows; ++r) {
    rows[3 * r] = r / (d->Hkv * nL);
    rows[3 * r + 1] = (r / nL) % d->Hkv;
    rows[3 * r + 2] = r % nL;
  }
  hdo_sfa_bwd_kv_rows(q, k, v, dout, lse_ws, D_ws, d, krows, rows, dk_rows, dv_rows);
  for (int64_t r = 0; r < krows; ++r) {
    int64_t b = rows[3 * r], g = rows[3 * r + 1], pk = rows[3 * r + 2];
    memcpy(dk + ((b * nL + pk) * d->Hkv + g) * d->Dh, dk_rows + r * d->Dh, (size_t)d->Dh * sizeof(double));
    memcpy(dv + ((b * nL + pk) * d->Hkv + g) * d->Dh, dv_rows + r * d->Dh, (size_t)d->Dh * sizeof(double));
  }
  free(rows);
  free(dk_rows);
  free(dv_rows);
}

/* ---- backward with the softmax Jacobian formed explicitly (small inputs only) ----
 * Per query row: J[a][c] = P_a (delta_ac - P_c) over the row's m visible keys,
 * dz = J dP, then dQ_p = scale sum dz K, dK += scale dz Q_p, dV += P dO_p.
 * Single-threaded accumulation into dq, dk, dv (zeroed here). */
void hdo_sfa_bwd_jacobian(const double* q, const double* k, const double* v, const double* dout,
                          double* dq, double* dk, double* dv, const hdo_dims* d) {
  const int64_t nL = d->n * d->L;
  memset(dq, 0, (size_t)(d->B * nL * d->Hq * d->Dh) * sizeof(double));
  memset(dk, 0, (size_t)(d->B * nL * d->Hkv * d->Dh) * sizeof(double));
  memset(dv, 0, (size_t)(d->B * nL * d->Hkv * d->Dh) * sizeof(double));
  double* z = (double*)malloc((size_t)nL * sizeof(double));
  int64_t* idx = (int64_t*)malloc((size_t)nL * sizeof(int64_t));
  double* P = (double*)malloc((size_t)nL * sizeof(double));
  double* dP = (double*)malloc((size_t)nL * sizeof(double));
  double* dz = (double*)malloc((size_t)nL * sizeof(double));
  double* J = (double*)malloc((size_t)nL * nL * sizeof(double));
  for (int64_t b = 0; b < d->B; ++b)
    for (int64_t h = 0; h < d->Hq; ++h) {
      int64_t g = kv_head(d, h);
      for (int64_t p = 0; p < nL; ++p) {
        double lse = row_scores(q, k, d, b, h, p, z);
        int64_t m = 0;
        for (int64_t pk = 0; pk < nL; ++pk)
          if (vis0(d, p, pk)) idx[m++] = pk;
        const double* dop = qrow(dout, d, b, p, h);
        for (int64_t a = 0; a < m; ++a) {
          P[a] = exp(z[idx[a]] - lse);
          dP[a] = dot(dop, kvrow(v, d, b, idx[a], g), d->Dh);
        }
        for (int64_t a = 0; a < m; ++a)
          for (int64_t c = 0; c < m; ++c) J[a * m + c] = P[a] * ((a == c ? 1.0 : 0.0) - P[c]);
        for (int64_t a = 0; a < m; ++a) {
          dz[a] = 0.0;
          for (int64_t c = 0; c < m; ++c) dz[a] += J[a * m + c] * dP[c];
        }
        double* dqp = dq + ((b * nL + p) * d->Hq + h) * d->Dh;
        const double* qp = qrow(q, d, b, p, h);
        for (int64_t a = 0; a < m; ++a) {
          const double* kr = kvrow(k, d, b, idx[a], g);
          double* dkr = dk + ((b * nL + idx[a]) * d->Hkv + g) * d->Dh;
          double* dvr = dv + ((b * nL + idx[a]) * d->Hkv + g) * d->Dh;
          for (int64_t e = 0; e < d->Dh; ++e) {
            dqp[e] += d->scale * dz[a] * kr[e];
            dkr[e] += d->scale * dz[a] * qp[e];
            dvr[e] += P[a] * dop[e];
          }
        }
      }
    }
  free(z);
  free(idx);
  free(P);
  free(dP);
  free(dz);
  free(J);
}

/* Threads an OpenMP parallel region would use (for reporting the CPU baseline). */
int hdo_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
