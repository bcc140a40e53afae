// Stream-Factorized Attention forward and backward on warp-level mma.sync
// (m16n8k16 bf16, fp32 accumulate): FlashAttention-2-style tiles, cp.async
// double buffering, XOR-swizzled shared memory.
//
// Each CTA works on one virtual causal problem (see SfaGeom): WITHIN mode gives
// one problem per stream (rows p = r*n + s, Eq. 4), so a query tile visits only
// its own stream's key tiles; CROSS gives one causal problem over nL positions
// (Fig. 2a); LOCAL adds the window bound (Fig. 2b); a final-stream problem maps
// query row r to key row r*qstep + qoff.  Key tiles beyond the causal
// diagonal (or before the window) are never visited; only tiles that straddle a
// mask edge are masked in registers.
#include "common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int BM = 64, BN = 64, NT = 128;

struct MmaFwdArgs {
  const bf16* q;
  const bf16* k;
  const bf16* v;
  bf16* o;
  float* lse;
  SfaGeom g;
  float scale_log2;
};

struct MmaBwdArgs {
  const bf16* q;
  const bf16* k;
  const bf16* v;
  const bf16* dout;
  const float* lse2;   // [B][Hq][ns][Lvp] -lse * log2(e), stream-major (see sfa_bwd_prep.cu)
  const float* delta;  // [B][Hq][ns][Lvp] -rowsum(dO * O)
  float* dq_acc;       // [B][nL][Hq][Dh] fp32, pre-zeroed; gets sum dS K (unscaled)
  bf16* dk;
  bf16* dv;
  SfaGeom g;
  float scale;
  float scale_log2;
};

// rows [r0, r0 + ROWS) of a [*][DH] row set (row stride rstride elements) -> swizzled smem.
template <int DH, int ROWS>
HD_DEVINLINE void load_rows(bf16* s, const bf16* base, long long rstride, int r0, int Lv, int tid) {
  constexpr int CPR = DH / 8;
#pragma unroll
  for (int i = tid; i < ROWS * CPR; i += NT) {
    const int r = i / CPR, c = i % CPR;
    const int gr = r0 + r;
    const bool ok = gr < Lv;
    const bf16* src = base + (long long)(ok ? gr : 0) * rstride + c * 8;
    cp_async_16(smem_u32(s + swz<DH>(r, c * 8)), src, ok);
  }
}

// Key row c visible from the query at key row rq (query row r sits at key row
// r*qstep + qoff of its problem: r itself unless it is a final-stream problem).
HD_DEVINLINE bool visible(int rq, int c, int Lv, int window) {
  return c <= rq && c < Lv && (window <= 0 || rq - c < window);
}

// ----------------------------------------------------------------- forward
template <int DH>
__global__ void __launch_bounds__(NT) sfa_fwd_mma_kernel(MmaFwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);  // [BM][DH]
  bf16* sK = sQ + BM * DH;                        // [2][BN][DH]
  bf16* sV = sK + 2 * BN * DH;                    // [2][BN][DH]
  const SfaGeom G = a.g;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ntile = (G.Lq + BM - 1) / BM;
  const int mt = ntile - 1 - (int)blockIdx.x;  // longest rows first
  const int m0 = mt * BM;
  const int h = blockIdx.y / G.q_ns, s = blockIdx.y % G.q_ns, b = blockIdx.z;
  const int sk = s + G.kv_s0;  // stream of the key problem
  const int kvh = h / (G.Hq / G.Hkv);
  const long long q_rs = (long long)G.q_rs * G.Hq * DH, kv_rs = (long long)G.rs * G.Hkv * DH;
  const bf16* qb = a.q + (((long long)b * G.q_nL + s) * G.Hq + h) * DH;
  const bf16* kb = a.k + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;
  const bf16* vb = a.v + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;
  const int rq_first = m0 * G.qstep + G.qoff, rq_last = (min(m0 + BM, G.Lq) - 1) * G.qstep + G.qoff;
  const int n_lo = G.window > 0 ? max(0, rq_first - G.window + 1) / BN : 0;
  const int n_hi = min(rq_last / BN, (G.Lv - 1) / BN);

  load_rows<DH, BM>(sQ, qb, q_rs, m0, G.Lq, tid);
  load_rows<DH, BN>(sK, kb, kv_rs, n_lo * BN, G.Lv, tid);
  load_rows<DH, BN>(sV, vb, kv_rs, n_lo * BN, G.Lv, tid);
  cp_async_commit();

  // Q fragments stay in registers up to head dim 128; at 256 the O accumulator needs
  // those registers and the fragments are reloaded from shared memory per key tile.
  constexpr bool kHoldQ = DH <= 128;
  uint32_t qf[kHoldQ ? DH / 16 : 1][4];
  float oacc[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  float mx[2] = {-INFINITY, -INFINITY}, lsum[2] = {0.f, 0.f};
  const int g4 = lane >> 2, t4 = lane & 3;
  const int r_lo = m0 + warp * 16 + g4;

  for (int nt_i = n_lo; nt_i <= n_hi; ++nt_i) {
    const int buf = (nt_i - n_lo) & 1;
    cp_async_wait<0>();
    __syncthreads();
    if (kHoldQ && nt_i == n_lo) {
#pragma unroll
      for (int kk = 0; kk < (kHoldQ ? DH / 16 : 0); ++kk)
        ldsm_x4(smem_u32(sQ + swz<DH>(warp * 16 + (lane & 15), kk * 16 + (lane >> 4) * 8)),
                qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
    }
    if (nt_i < n_hi) {
      load_rows<DH, BN>(sK + (buf ^ 1) * BN * DH, kb, kv_rs, (nt_i + 1) * BN, G.Lv, tid);
      load_rows<DH, BN>(sV + (buf ^ 1) * BN * DH, vb, kv_rs, (nt_i + 1) * BN, G.Lv, tid);
      cp_async_commit();
    }
    const bf16* cK = sK + buf * BN * DH;
    const bf16* cV = sV + buf * BN * DH;
    const int n0 = nt_i * BN;

    float sacc[BN / 8][4];
#pragma unroll
    for (int i = 0; i < BN / 8; ++i) sacc[i][0] = sacc[i][1] = sacc[i][2] = sacc[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
      uint32_t qr[4];
      if (kHoldQ) {
        qr[0] = qf[kHoldQ ? kk : 0][0];
        qr[1] = qf[kHoldQ ? kk : 0][1];
        qr[2] = qf[kHoldQ ? kk : 0][2];
        qr[3] = qf[kHoldQ ? kk : 0][3];
      } else {
        ldsm_x4(smem_u32(sQ + swz<DH>(warp * 16 + (lane & 15), kk * 16 + (lane >> 4) * 8)), qr[0], qr[1], qr[2],
                qr[3]);
      }
#pragma unroll
      for (int np = 0; np < BN / 16; ++np) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(cK + swz<DH>(np * 16 + (lane & 7) + (lane >> 4) * 8,
                                      kk * 16 + ((lane >> 3) & 1) * 8)),
                b0, b1, b2, b3);
        mma_bf16_16816(sacc[2 * np], qr, b0, b1);
        mma_bf16_16816(sacc[2 * np + 1], qr, b2, b3);
      }
    }
    // tiles with a key past the first query's key row, a key at or below the last
    // query's window edge, or ragged
    const bool need_mask = (nt_i + 1) * BN - 1 > rq_first || (G.window > 0 && nt_i * BN <= rq_last - G.window) ||
                           (nt_i + 1) * BN > G.Lv;
    float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int i = 0; i < BN / 8; ++i) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float x = sacc[i][e] * a.scale_log2;
        if (need_mask) {
          const int r = r_lo + (e >> 1) * 8, c = n0 + i * 8 + 2 * t4 + (e & 1);
          if (!visible(r * G.qstep + G.qoff, c, G.Lv, G.window)) x = -INFINITY;
        }
        sacc[i][e] = x;
        tmax[e >> 1] = fmaxf(tmax[e >> 1], x);
      }
    }
    float corr[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      tmax[hh] = fmaxf(tmax[hh], __shfl_xor_sync(0xffffffffu, tmax[hh], 1));
      tmax[hh] = fmaxf(tmax[hh], __shfl_xor_sync(0xffffffffu, tmax[hh], 2));
      const float mnew = fmaxf(mx[hh], tmax[hh]);
      const float muse = (mnew == -INFINITY) ? 0.f : mnew;
      corr[hh] = exp2f(mx[hh] - muse);
      mx[hh] = mnew;
      lsum[hh] *= corr[hh];
      tmax[hh] = muse;
    }
#pragma unroll
    for (int i = 0; i < BN / 8; ++i) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(sacc[i][e] - tmax[e >> 1]);
        sacc[i][e] = p;
        lsum[e >> 1] += p;
      }
    }
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      oacc[i][0] *= corr[0];
      oacc[i][1] *= corr[0];
      oacc[i][2] *= corr[1];
      oacc[i][3] *= corr[1];
    }
#pragma unroll
    for (int kk = 0; kk < BN / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(sacc[2 * kk][0], sacc[2 * kk][1]);
      pa[1] = pack_bf16(sacc[2 * kk][2], sacc[2 * kk][3]);
      pa[2] = pack_bf16(sacc[2 * kk + 1][0], sacc[2 * kk + 1][1]);
      pa[3] = pack_bf16(sacc[2 * kk + 1][2], sacc[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < DH / 16; ++dp) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(cV + swz<DH>(kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8,
                                        dp * 16 + (lane >> 4) * 8)),
                  b0, b1, b2, b3);
        mma_bf16_16816(oacc[2 * dp], pa, b0, b1);
        mma_bf16_16816(oacc[2 * dp + 1], pa, b2, b3);
      }
    }
  }

  // epilogue: normalise, stage through shared memory, coalesced 16-byte stores
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    lsum[hh] += __shfl_xor_sync(0xffffffffu, lsum[hh], 1);
    lsum[hh] += __shfl_xor_sync(0xffffffffu, lsum[hh], 2);
  }
  const float inv0 = 1.f / lsum[0], inv1 = 1.f / lsum[1];
  __syncthreads();
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) {
    const int row = warp * 16 + g4, col = i * 8 + 2 * t4;
    *reinterpret_cast<uint32_t*>(sQ + swz<DH>(row, col)) = pack_bf16(oacc[i][0] * inv0, oacc[i][1] * inv0);
    *reinterpret_cast<uint32_t*>(sQ + swz<DH>(row + 8, col)) = pack_bf16(oacc[i][2] * inv1, oacc[i][3] * inv1);
  }
  if (t4 == 0) {
    float* lrow = a.lse + ((long long)b * G.Hq + h) * G.q_nL + s;
    if (r_lo < G.Lq) lrow[(long long)r_lo * G.q_rs] = (mx[0] + log2f(lsum[0])) * kLn2;
    if (r_lo + 8 < G.Lq) lrow[(long long)(r_lo + 8) * G.q_rs] = (mx[1] + log2f(lsum[1])) * kLn2;
  }
  __syncthreads();
  bf16* ob = a.o + (((long long)b * G.q_nL + s) * G.Hq + h) * DH;
  constexpr int CPR = DH / 8;
  for (int i = tid; i < BM * CPR; i += NT) {
    const int r = i / CPR, c = i % CPR;
    if (m0 + r < G.Lq)
      *reinterpret_cast<uint4*>(ob + (long long)(m0 + r) * q_rs + c * 8) =
          *reinterpret_cast<const uint4*>(sQ + swz<DH>(r, c * 8));
  }
}

// ----------------------------------------------------------------- backward
// One CTA per (key tile j, b, K/V head g, stream s).  It keeps dK_j, dV_j in
// registers while looping over the group's query heads and the query tiles that
// can see tile j; dQ contributions go to the fp32 accumulator with atomics.
// Warp w owns key rows [16w, 16w + 16) of the tile for S^T, dP^T, dK, dV.
// DO: the head-dim columns of dK, dV, dQ one CTA accumulates (starting at d0); S^T and
// dP^T always take the full head dim.  DO = DH, or DO = DH / 2 at head dim 256 (whose
// dK and dV would not fit the registers at once), the two slices of a key tile being
// separate CTAs of one launch.
template <int DH, int DO>
__global__ void __launch_bounds__(NT, 1) sfa_bwd_mma_kernel(MmaBwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  bf16* sK = reinterpret_cast<bf16*>(smem_raw);  // [BN][DH]
  bf16* sV = sK + BN * DH;                        // [BN][DH]
  bf16* sQ = sV + BN * DH;                        // [2][BM][DH]
  bf16* sdO = sQ + 2 * BM * DH;                   // [2][BM][DH]
  bf16* sdS = sdO + 2 * BM * DH;                  // [BN][BM]  (dS^T, key-major)
  float* sL = reinterpret_cast<float*>(sdS + BN * BM);  // [2][BM] -lse * log2(e)
  float* sD = sL + 2 * BM;                               // [2][BM] -delta

  const SfaGeom G = a.g;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g4 = lane >> 2, t4 = lane & 3;
  const int ntile = (G.Lq + BM - 1) / BM;
  const int j = blockIdx.x;  // key tile; tile 0 sees the most query tiles, so it starts first
  const int n0 = j * BN;
  const int kvh = blockIdx.y / G.q_ns, s = blockIdx.y % G.q_ns;
  // blockIdx.z: batch and head-dim slice (the DO columns of dK, dV, dQ from d0 this CTA
  // writes; the slices of one key tile run side by side)
  const int b = blockIdx.z / (DH / DO), d0 = (blockIdx.z % (DH / DO)) * DO;
  const int sk = s + G.kv_s0;  // stream of the key problem
  const int grp = G.Hq / G.Hkv;
  // query tiles that can see a key of this tile: query row r stands at key row
  // r*qstep + qoff >= n0, and under a window r*qstep + qoff < n0 + BN - 1 + window
  const int mi_lo = (n0 <= G.qoff ? 0 : (n0 - G.qoff + G.qstep - 1) / G.qstep) / BM;
  int mi_hi = ntile - 1;
  if (G.window > 0) mi_hi = min(mi_hi, ((n0 + BN - 2 + G.window - G.qoff) / G.qstep) / BM);
  const int nq = mi_hi - mi_lo + 1;
  const int total = grp * max(nq, 0);
  const long long q_rs = (long long)G.q_rs * G.Hq * DH, kv_rs = (long long)G.rs * G.Hkv * DH;
  const bf16* kb = a.k + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;
  const bf16* vb = a.v + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;

  auto q_base = [&](const bf16* t, int h) {
    return t + (((long long)b * G.q_nL + s) * G.Hq + h) * DH;
  };
  const int Lqp = row_terms_pitch(G.Lq);
  auto row_terms = [&](int it, int r, float& l2, float& dl) {
    const int h = kvh * grp + it / nq, m0 = (mi_lo + it % nq) * BM;
    const long long idx = (((long long)b * G.Hq + h) * G.q_ns + s) * Lqp + m0 + r;
    const bool ok = m0 + r < G.Lq;
    l2 = ok ? a.lse2[idx] : 0.f;
    dl = ok ? a.delta[idx] : 0.f;
  };

  load_rows<DH, BN>(sK, kb, kv_rs, n0, G.Lv, tid);
  load_rows<DH, BN>(sV, vb, kv_rs, n0, G.Lv, tid);
  if (total > 0) {
    const int h = kvh * grp;
    load_rows<DH, BM>(sQ, q_base(a.q, h), q_rs, mi_lo * BM, G.Lq, tid);
    load_rows<DH, BM>(sdO, q_base(a.dout, h), q_rs, mi_lo * BM, G.Lq, tid);
  }
  cp_async_commit();
  if (tid < BM && total > 0) {
    float l2, dl;
    row_terms(0, tid, l2, dl);
    sL[tid] = l2;
    sD[tid] = dl;
  }

  float dK[DO / 8][4], dV[DO / 8][4];
#pragma unroll
  for (int i = 0; i < DO / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dK[i][e] = dV[i][e] = 0.f;

  for (int it = 0; it < total; ++it) {
    const int buf = it & 1;
    cp_async_wait<0>();
    __syncthreads();
    const bool has_next = it + 1 < total;
    float nl2 = 0.f, ndl = 0.f;
    if (has_next) {
      const int h1 = kvh * grp + (it + 1) / nq, m1 = (mi_lo + (it + 1) % nq) * BM;
      load_rows<DH, BM>(sQ + (buf ^ 1) * BM * DH, q_base(a.q, h1), q_rs, m1, G.Lq, tid);
      load_rows<DH, BM>(sdO + (buf ^ 1) * BM * DH, q_base(a.dout, h1), q_rs, m1, G.Lq, tid);
      cp_async_commit();
      if (tid < BM) row_terms(it + 1, tid, nl2, ndl);
    }
    const int h = kvh * grp + it / nq;
    const int m0 = (mi_lo + it % nq) * BM;
    const bf16* cQ = sQ + buf * BM * DH;
    const bf16* cdO = sdO + buf * BM * DH;
    const float* cL = sL + buf * BM;
    const float* cD = sD + buf * BM;

#pragma unroll
    for (int half = 0; half < 2; ++half) {
      float sacc[4][4], dpacc[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e) sacc[i][e] = dpacc[i][e] = 0.f;
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
        uint32_t ka[4], va[4];
        ldsm_x4(smem_u32(sK + swz<DH>(warp * 16 + (lane & 15), kk * 16 + (lane >> 4) * 8)),
                ka[0], ka[1], ka[2], ka[3]);
        ldsm_x4(smem_u32(sV + swz<DH>(warp * 16 + (lane & 15), kk * 16 + (lane >> 4) * 8)),
                va[0], va[1], va[2], va[3]);
#pragma unroll
        for (int np = 0; np < 2; ++np) {
          const int qr = half * 32 + np * 16 + (lane & 7) + (lane >> 4) * 8;
          const int qc = kk * 16 + ((lane >> 3) & 1) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(smem_u32(cQ + swz<DH>(qr, qc)), b0, b1, b2, b3);
          mma_bf16_16816(sacc[2 * np], ka, b0, b1);
          mma_bf16_16816(sacc[2 * np + 1], ka, b2, b3);
          ldsm_x4(smem_u32(cdO + swz<DH>(qr, qc)), b0, b1, b2, b3);
          mma_bf16_16816(dpacc[2 * np], va, b0, b1);
          mma_bf16_16816(dpacc[2 * np + 1], va, b2, b3);
        }
      }
      // P^T and dS^T for rows (key) kr, columns (query) qc
#pragma unroll
      for (int i = 0; i < 4; ++i) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int kr = n0 + warp * 16 + g4 + (e >> 1) * 8;
          const int ql = half * 32 + i * 8 + 2 * t4 + (e & 1);
          const int qr = m0 + ql;
          float p = 0.f;
          if (qr < G.Lq && visible(qr * G.qstep + G.qoff, kr, G.Lv, G.window))
            p = exp2f(fmaf(sacc[i][e], a.scale_log2, cL[ql]));
          sacc[i][e] = p;
          dpacc[i][e] = p * (dpacc[i][e] + cD[ql]);
        }
      }
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        uint32_t pa[4], da[4];
        pa[0] = pack_bf16(sacc[2 * kk][0], sacc[2 * kk][1]);
        pa[1] = pack_bf16(sacc[2 * kk][2], sacc[2 * kk][3]);
        pa[2] = pack_bf16(sacc[2 * kk + 1][0], sacc[2 * kk + 1][1]);
        pa[3] = pack_bf16(sacc[2 * kk + 1][2], sacc[2 * kk + 1][3]);
        da[0] = pack_bf16(dpacc[2 * kk][0], dpacc[2 * kk][1]);
        da[1] = pack_bf16(dpacc[2 * kk][2], dpacc[2 * kk][3]);
        da[2] = pack_bf16(dpacc[2 * kk + 1][0], dpacc[2 * kk + 1][1]);
        da[3] = pack_bf16(dpacc[2 * kk + 1][2], dpacc[2 * kk + 1][3]);
        const int qrow = half * 32 + kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
        for (int dp = 0; dp < DO / 16; ++dp) {
          const int dcol = d0 + dp * 16 + (lane >> 4) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(smem_u32(cdO + swz<DH>(qrow, dcol)), b0, b1, b2, b3);
          mma_bf16_16816(dV[2 * dp], pa, b0, b1);
          mma_bf16_16816(dV[2 * dp + 1], pa, b2, b3);
          ldsm_x4_t(smem_u32(cQ + swz<DH>(qrow, dcol)), b0, b1, b2, b3);
          mma_bf16_16816(dK[2 * dp], da, b0, b1);
          mma_bf16_16816(dK[2 * dp + 1], da, b2, b3);
        }
        // dS^T (bf16) to shared memory for the dQ product
        const int krow = warp * 16 + g4;
        const int qcol = half * 32 + kk * 16 + 2 * t4;
        *reinterpret_cast<uint32_t*>(sdS + swz<BM>(krow, qcol)) = da[0];
        *reinterpret_cast<uint32_t*>(sdS + swz<BM>(krow + 8, qcol)) = da[1];
        *reinterpret_cast<uint32_t*>(sdS + swz<BM>(krow, qcol + 8)) = da[2];
        *reinterpret_cast<uint32_t*>(sdS + swz<BM>(krow + 8, qcol + 8)) = da[3];
      }
    }
    __syncthreads();
    // dQ[q rows of warp] += dS K  (unscaled; the post kernel applies the scale)
    {
      float* dqb = a.dq_acc + (((long long)b * G.q_nL + s) * G.Hq + h) * DH;
      const int qa = m0 + warp * 16 + g4;
#pragma unroll
      for (int dh = 0; dh < 2; ++dh) {
        float qacc[DO / 16][4];
#pragma unroll
        for (int i = 0; i < DO / 16; ++i) qacc[i][0] = qacc[i][1] = qacc[i][2] = qacc[i][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk) {
          uint32_t aa[4];
          ldsm_x4_t(smem_u32(sdS + swz<BM>(kk * 16 + (lane & 7) + (lane >> 4) * 8,
                                           warp * 16 + ((lane >> 3) & 1) * 8)),
                    aa[0], aa[1], aa[2], aa[3]);
#pragma unroll
          for (int dp = 0; dp < DO / 32; ++dp) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(smem_u32(sK + swz<DH>(kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8,
                                            d0 + dh * (DO / 2) + dp * 16 + (lane >> 4) * 8)),
                      b0, b1, b2, b3);
            mma_bf16_16816(qacc[2 * dp], aa, b0, b1);
            mma_bf16_16816(qacc[2 * dp + 1], aa, b2, b3);
          }
        }
#pragma unroll
        for (int i = 0; i < DO / 16; ++i) {
          const int col = d0 + dh * (DO / 2) + i * 8 + 2 * t4;
          if (qa < G.Lq)
            atomicAdd(reinterpret_cast<float2*>(dqb + (long long)qa * q_rs + col),
                      make_float2(qacc[i][0], qacc[i][1]));
          if (qa + 8 < G.Lq)
            atomicAdd(reinterpret_cast<float2*>(dqb + (long long)(qa + 8) * q_rs + col),
                      make_float2(qacc[i][2], qacc[i][3]));
        }
      }
    }
    if (has_next && tid < BM) {
      sL[(buf ^ 1) * BM + tid] = nl2;
      sD[(buf ^ 1) * BM + tid] = ndl;
    }
  }

  cp_async_wait<0>();  // a key tile that no query sees still loaded K and V
  // epilogue: dK *= scale, write dK and dV rows of this key tile
  bf16* dkb = a.dk + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;
  bf16* dvb = a.dv + (((long long)b * G.nL + sk) * G.Hkv + kvh) * DH;
  const int kr = n0 + warp * 16 + g4;
#pragma unroll
  for (int i = 0; i < DO / 8; ++i) {
    const int col = d0 + i * 8 + 2 * t4;
    if (kr < G.Lv) {
      *reinterpret_cast<uint32_t*>(dkb + (long long)kr * kv_rs + col) =
          pack_bf16(dK[i][0] * a.scale, dK[i][1] * a.scale);
      *reinterpret_cast<uint32_t*>(dvb + (long long)kr * kv_rs + col) = pack_bf16(dV[i][0], dV[i][1]);
    }
    if (kr + 8 < G.Lv) {
      *reinterpret_cast<uint32_t*>(dkb + (long long)(kr + 8) * kv_rs + col) =
          pack_bf16(dK[i][2] * a.scale, dK[i][3] * a.scale);
      *reinterpret_cast<uint32_t*>(dvb + (long long)(kr + 8) * kv_rs + col) =
          pack_bf16(dV[i][2], dV[i][3]);
    }
  }
}

// ----------------------------------------------------------------- launchers
template <int DH>
static cudaError_t fwd_impl(const MmaFwdArgs& a, cudaStream_t st) {
  const int smem = (BM + 4 * BN) * DH * (int)sizeof(bf16);
  cudaError_t e = cudaFuncSetAttribute(sfa_fwd_mma_kernel<DH>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.g.Lq + BM - 1) / BM, a.g.Hq * a.g.q_ns, a.g.B);
  sfa_fwd_mma_kernel<DH><<<grid, NT, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_sfa_fwd_mma(const void* q, const void* k, const void* v, void* o, float* lse,
                               const SfaGeom& g, int Dh, float scale, cudaStream_t st) {
  MmaFwdArgs a{(const bf16*)q, (const bf16*)k, (const bf16*)v, (bf16*)o, lse, g, scale * kLog2e};
  if (Dh == 64) return fwd_impl<64>(a, st);
  if (Dh == 256) return fwd_impl<256>(a, st);
  return fwd_impl<128>(a, st);
}

template <int DH, int DO>
static cudaError_t bwd_impl(MmaBwdArgs a, cudaStream_t st) {
  const SfaGeom& g = a.g;
  const int smem = (2 * BN * DH + 4 * BM * DH + BN * BM) * (int)sizeof(bf16) + 4 * BM * (int)sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(sfa_bwd_mma_kernel<DH, DO>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  // the DH / DO head-dim slices of every key tile in one launch
  dim3 grid((g.Lv + BN - 1) / BN, g.Hkv * g.q_ns, g.B * (DH / DO));
  sfa_bwd_mma_kernel<DH, DO><<<grid, NT, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_sfa_bwd_main_mma(const void* q, const void* k, const void* v, const void* dout,
                                    void* dk, void* dv, const float* lse2_ws, const float* delta_ws,
                                    float* dq_ws, const SfaGeom& g, int Dh, float scale,
                                    cudaStream_t st) {
  MmaBwdArgs a{(const bf16*)q, (const bf16*)k, (const bf16*)v, (const bf16*)dout, lse2_ws, delta_ws,
               dq_ws, (bf16*)dk, (bf16*)dv, g, scale, scale * kLog2e};
  if (Dh == 64) return bwd_impl<64, 64>(a, st);
  if (Dh == 256) return bwd_impl<256, 128>(a, st);
  return bwd_impl<128, 128>(a, st);
}

}  // namespace hdsfa
