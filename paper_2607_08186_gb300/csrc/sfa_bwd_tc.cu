// Stream-Factorized Attention backward (main pass) on the sm_103a tensor cores,
// head dim 128.
//
// One CTA owns a 128-row key tile j of one virtual causal problem (SfaGeom) and
// one K/V head; it loops over the group's query heads and over the 64-row query
// tiles that can see tile j (causal: query tiles at or after the key tile; LOCAL:
// also within the window).  Per query tile, with TMEM lane = key row:
//   S^T  = K Q^T,  dP^T = V dO^T                      (SS MMA, M=128 N=64 K=128)
//   P^T  = exp2(S^T * scale*log2e - lse2),  dS^T = P^T (dP^T - delta)   (softmax)
//   dV  += P^T dO,  dK += dS^T Q                      (TS MMA: P^T, dS^T bf16 in TMEM)
//   dQ^T = K^T dS^T                                   (SS MMA, M=128 (head dim) N=64)
// dQ^T leaves TMEM through the dQ warpgroup: shared memory, then a TMA tensor
// reduce-add (fp32) into the workspace accumulator.  dK, dV stay in TMEM for
// the whole loop and are written once (dK scaled).
//
// Issue order of the MMA thread for tile t:
//   dP(t+1) | wait P(t) | dV(t) S(t+1) dK(t) | wait dQ^T read-out of t-1 | dQ(t)
// so the softmax of tile t+1 (which needs S(t+1), dP(t+1)) runs while the tensor
// pipe works on dK(t), dQ(t) and dP(t+2).  S(t+1) reuses the S^T columns that hold
// P^T(t) only after dV(t) has been issued (tcgen05 MMAs of one thread run in order).
//
// Roles (448 threads): warp 0 TMA producer (+ TMEM owner), warp 1 MMA issuer,
// warps 2..5 and 6..9 softmax (key row = TMEM lane; query columns 0..31 and
// 32..63), warps 10..13 dQ flush (one head-dim row each).  Every mbarrier wait
// is bounded.
//
// TMEM columns: S^T at 0 (P^T bf16 over its first 32), dP^T[st] at 64 + 64*st
// (dS^T bf16 over its first 32), dQ^T at 192, dV at 256, dK at 384.
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcbwd {
constexpr int BK = 128, BQ = 64, DH = 128, NST = 2, NTHREADS = 448;
constexpr uint32_t COL_ST = 0, COL_DQ = 192, COL_DV = 256, COL_DK = 384;
HD_DEVINLINE uint32_t col_dpt(int st) { return 64u + 64u * st; }

struct Smem {
  bf16 k[BK * DH];          // 2 swizzle blocks of [128 key rows][64]
  bf16 v[BK * DH];
  bf16 q[NST][BQ * DH];     // 2 swizzle blocks of [64 query rows][64]
  bf16 dO[NST][BQ * DH];
  bf16 ds[NST][BK * BQ];    // dS^T [128 key rows][64 queries], one swizzle block
  float dq[4][BQ * 32];     // per dQ warp: [64 queries][32 head-dim] fp32 staging
  float lse2[NST][BQ];
  float delta[NST][BQ];
  uint64_t kv_full, qd_full[NST], qd_empty[NST], s_full, dp_full[NST], p_ready, dq_full, dq_free,
      ds_free[NST], s_read, kv_done, drain;
  uint32_t tmem_base;
  int abort;
};

struct Params {
  CUtensorMap tm_q, tm_do, tm_k, tm_v, tm_dq;
  const float* lse2;   // [B][Hq][ns][Lvp]
  const float* delta;  // [B][Hq][ns][Lvp]
  bf16* dk;
  bf16* dv;
  SfaGeom g;
  float scale, scale_log2;
  int32_t* status;
};

HD_DEVINLINE bool visible(int r, int c, int Lv, int window) {
  return c <= r && r < Lv && c < Lv && (window <= 0 || r - c < window);
}

__global__ void __launch_bounds__(NTHREADS, 1) bwd_kernel(const __grid_constant__ Params P) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SfaGeom& G = P.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.x;  // key tile; tile 0 sees the most query tiles and starts first
  const int n0 = j * BK;
  const int kvh = blockIdx.y / G.ns, s = blockIdx.y % G.ns, b = blockIdx.z;
  const int grp = G.Hq / G.Hkv;
  const int i_lo = n0 / BQ;
  int i_hi = (G.Lv - 1) / BQ;
  if (G.window > 0) i_hi = min(i_hi, (n0 + BK - 1 + G.window - 1) / BQ);
  const int nq = i_hi - i_lo + 1;
  const int T = grp * nq;
  const int Lvp = (G.Lv + 63) & ~63;

  if (threadIdx.x == 0) {
    mbar_init(&sm.kv_full, 1);
    for (int i = 0; i < NST; ++i) {
      mbar_init(&sm.qd_full[i], 1);
      mbar_init(&sm.qd_empty[i], 1);
      mbar_init(&sm.dp_full[i], 1);
      mbar_init(&sm.ds_free[i], 1);
    }
    mbar_init(&sm.s_full, 1);
    mbar_init(&sm.p_ready, 256);
    mbar_init(&sm.s_read, 256);
    mbar_init(&sm.dq_full, 1);
    mbar_init(&sm.dq_free, 128);
    mbar_init(&sm.kv_done, 1);
    mbar_init(&sm.drain, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch(&P.tm_q);
      tma_prefetch(&P.tm_do);
      tma_prefetch(&P.tm_k);
      tma_prefetch(&P.tm_v);
      mbar_arrive_expect_tx(&sm.kv_full, 2 * BK * DH * 2);
      for (int c = 0; c < DH / 64; ++c) {
        tma_load_5d(sm.k + c * BK * 64, &P.tm_k, &sm.kv_full, c * 64, kvh, s, n0, b);
        tma_load_5d(sm.v + c * BK * 64, &P.tm_v, &sm.kv_full, c * 64, kvh, s, n0, b);
      }
      int issued = 0;
      for (int t = 0; t < T; ++t, ++issued) {
        const int st = t & 1;
        if (t >= NST && !mbar_wait(&sm.qd_empty[st], ((t - NST) >> 1) & 1, abort, P.status)) break;
        const int h = kvh * grp + t / nq, q0 = (i_lo + t % nq) * BQ;
        mbar_arrive_expect_tx(&sm.qd_full[st], 2 * BQ * DH * 2 + 2 * BQ * 4);
        for (int c = 0; c < DH / 64; ++c) {
          tma_load_5d(sm.q[st] + c * BQ * 64, &P.tm_q, &sm.qd_full[st], c * 64, h, s, q0, b);
          tma_load_5d(sm.dO[st] + c * BQ * 64, &P.tm_do, &sm.qd_full[st], c * 64, h, s, q0, b);
        }
        const long long off = (((long long)b * G.Hq + h) * G.ns + s) * Lvp + q0;
        bulk_load(sm.lse2[st], P.lse2 + off, BQ * 4, &sm.qd_full[st]);
        bulk_load(sm.delta[st], P.delta + off, BQ * 4, &sm.qd_full[st]);
      }
      mbar_drain(&sm.kv_full, 0);
      for (int t = max(0, issued - NST); t < issued; ++t) mbar_drain(&sm.qd_full[t & 1], (t >> 1) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(128, BQ, 0, 0);   // S^T, dP^T: A = K/V, B = Q/dO (K-major)
      constexpr uint32_t idKV = idesc_bf16(128, DH, 0, 1);  // dV, dK: A in TMEM, B = dO/Q MN-major
      constexpr uint32_t idQ = idesc_bf16(128, BQ, 1, 1);   // dQ^T: A = K^T, B = dS^T, both MN-major
      const uint32_t ka = smem_u32(sm.k), va = smem_u32(sm.v);
      // S^T = K Q^T or dP^T = V dO^T of tile t into TMEM column col
      auto issue_sdp = [&](uint32_t aa, const bf16* bt, uint32_t col) {
        const uint32_t ba = smem_u32(bt);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(aa + (kk >> 2) * (BK * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc_sw128(ba + (kk >> 2) * (BQ * 128) + (kk & 3) * 32, 16, 1024);
          tc_mma_ss(tmem + col, ad, bd, idS, kk > 0 ? 1u : 0u);
        }
      };
      // dV (a_col = P^T) or dK (a_col = dS^T) += A * B, B = dO or Q of the tile (MN-major)
      auto issue_kv = [&](uint32_t a_col, const bf16* bt, uint32_t d_col, bool acc) {
        const uint32_t ba = smem_u32(bt);
#pragma unroll
        for (int kk = 0; kk < BQ / 16; ++kk) {
          const uint64_t bd = sdesc_sw128(ba + kk * 16 * 128, BQ * 128, 1024);
          tc_mma_ts(tmem + d_col, tmem + a_col + kk * 8, bd, idKV, (acc || kk > 0) ? 1u : 0u);
        }
      };
      bool ok = mbar_wait(&sm.kv_full, 0, abort, P.status) && mbar_wait(&sm.qd_full[0], 0, abort, P.status);
      if (ok) {
        tc_fence_after();
        issue_sdp(ka, sm.q[0], COL_ST);
        tc_commit(&sm.s_full);
        issue_sdp(va, sm.dO[0], col_dpt(0));
        tc_commit(&sm.dp_full[0]);
      }
      for (int t = 0; ok && t < T; ++t) {
        const int st = t & 1, sn = st ^ 1;
        if (t + 1 < T) {
          // dP^T(t+1): its columns last held dS^T(t-1), read by dK(t-1) issued earlier
          if (!mbar_wait(&sm.qd_full[sn], ((t + 1) >> 1) & 1, abort, P.status)) { ok = false; break; }
          tc_fence_after();
          issue_sdp(va, sm.dO[sn], col_dpt(sn));
          tc_commit(&sm.dp_full[sn]);
        }
        if (!mbar_wait(&sm.p_ready, t & 1, abort, P.status)) { ok = false; break; }
        tc_fence_after();
        issue_kv(COL_ST, sm.dO[st], COL_DV, t > 0);
        if (t + 1 < T) {
          issue_sdp(ka, sm.q[sn], COL_ST);  // after dV(t) read P^T(t)
          tc_commit(&sm.s_full);
        }
        issue_kv(col_dpt(st), sm.q[st], COL_DK, t > 0);
        tc_commit(&sm.qd_empty[st]);
        if (t >= 1 && !mbar_wait(&sm.dq_free, (t - 1) & 1, abort, P.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t dsa = smem_u32(sm.ds[st]);
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(ka + kk * 16 * 128, BK * 128, 1024);
          const uint64_t bd = sdesc_sw128(dsa + kk * 16 * 128, BK * 128, 1024);
          tc_mma_ss(tmem + COL_DQ, ad, bd, idQ, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sm.dq_full);
        tc_commit(&sm.ds_free[st]);
      }
      tc_commit(&sm.kv_done);
      tc_commit(&sm.drain);
      mbar_drain(&sm.drain, 0);
    }
  } else if (warp < 10) {
    // ------------------------------------------------------------ softmax (key rows)
    const int half = (warp - 2) >> 2;  // query columns [32*half, 32*half + 32)
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int kr = n0 + row;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const float c2 = P.scale_log2;
    bool ok = true;
    for (int t = 0; t < T; ++t) {
      const int st = t & 1;
      const int q0 = (i_lo + t % nq) * BQ + 32 * half;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full, t & 1, abort, P.status) &&
                                       mbar_wait(&sm.dp_full[st], (t >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[32], dr[32];
      tmem_ld32(tl + COL_ST + 32 * half, sr);
      tmem_ld32(tl + col_dpt(st) + 32 * half, dr);
      tmem_ld_wait();
      // both halves have read their S^T / dP^T columns before either packs bf16 over them
      // (an mbarrier rather than bar.sync, so an aborted peer cannot strand this warp)
      tc_fence_before();
      mbar_arrive(&sm.s_read);
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_read, t & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float4* l2 = reinterpret_cast<const float4*>(sm.lse2[st] + 32 * half);
      const float4* dl = reinterpret_cast<const float4*>(sm.delta[st] + 32 * half);
      const bool need_mask = (q0 < n0 + BK) || G.window > 0 || (n0 + BK > G.Lv) || (q0 + 32 > G.Lv);
      if (need_mask) {
        // zero the scores of invisible pairs up front: exp2(-inf) = 0 below
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (!visible(q0 + c, kr, G.Lv, G.window)) sr[c] = __float_as_uint(-INFINITY);
      }
      uint32_t pp[16], dd[16];
#pragma unroll
      for (int c4 = 0; c4 < 8; ++c4) {
        const float4 lv = l2[c4], dv = dl[c4];
        const float la[4] = {lv.x, lv.y, lv.z, lv.w}, da[4] = {dv.x, dv.y, dv.z, dv.w};
        float p[4], d[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int c = c4 * 4 + e;
          p[e] = ex2_approx(fmaf(__uint_as_float(sr[c]), c2, -la[e]));
          d[e] = p[e] * (__uint_as_float(dr[c]) - da[e]);
        }
        pp[2 * c4] = cvt_bf16x2(p[0], p[1]);
        pp[2 * c4 + 1] = cvt_bf16x2(p[2], p[3]);
        dd[2 * c4] = cvt_bf16x2(d[0], d[1]);
        dd[2 * c4 + 1] = cvt_bf16x2(d[2], d[3]);
      }
      // P^T and dS^T (bf16 pairs) over the first 32 columns of S^T and dP^T[st]
      tmem_st16(tl + COL_ST + 16 * half, pp);
      tmem_st16(tl + col_dpt(st) + 16 * half, dd);
      // dS^T -> shared memory for the dQ MMA; this buffer was last read by dQ(t-2)
      if (t >= NST &&
          !__all_sync(0xffffffffu, mbar_wait(&sm.ds_free[st], ((t - NST) >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      uint8_t* dsrow = reinterpret_cast<uint8_t*>(sm.ds[st]) + row * 128;
#pragma unroll
      for (int c = 0; c < 4; ++c)
        *reinterpret_cast<uint4*>(dsrow + (((4 * half + c) ^ (row & 7)) << 4)) =
            make_uint4(dd[4 * c], dd[4 * c + 1], dd[4 * c + 2], dd[4 * c + 3]);
      fence_async_smem();
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&sm.p_ready);
    }
    // epilogue: half 0 writes this key row of dV, half 1 of dK (scaled)
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.kv_done, 0, abort, P.status))) {
      tc_fence_after();
      const long long orow = (((long long)b * G.nL + (long long)kr * G.rs + s) * G.Hkv + kvh) * DH;
      const float mul = half ? P.scale : 1.f;
      bf16* dst = (half ? P.dk : P.dv) + orow;
      const uint32_t col = half ? COL_DK : COL_DV;
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tl + col + c * 32, o);
        tmem_ld_wait();
        if (kr < G.Lv) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = cvt_bf16x2(__uint_as_float(o[e + 0]) * mul, __uint_as_float(o[e + 1]) * mul);
            w.y = cvt_bf16x2(__uint_as_float(o[e + 2]) * mul, __uint_as_float(o[e + 3]) * mul);
            w.z = cvt_bf16x2(__uint_as_float(o[e + 4]) * mul, __uint_as_float(o[e + 5]) * mul);
            w.w = cvt_bf16x2(__uint_as_float(o[e + 6]) * mul, __uint_as_float(o[e + 7]) * mul);
            *reinterpret_cast<uint4*>(dst + c * 32 + e) = w;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ dQ flush (head-dim rows)
    const int q4 = warp & 3;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    float* stage = sm.dq[q4];
    for (int t = 0; t < T; ++t) {
      const int h = kvh * grp + t / nq, q0 = (i_lo + t % nq) * BQ;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.dq_full, t & 1, abort, P.status))) break;
      tc_fence_after();
      uint32_t v[BQ];
      tmem_ld32(tl + COL_DQ, v);
      tmem_ld32(tl + COL_DQ + 32, v + 32);
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(&sm.dq_free);
      // the previous reduce must have finished reading the staging buffer
      if (lane == 0) bulk_wait_read0();
      __syncwarp();
#pragma unroll
      for (int c = 0; c < BQ; ++c) stage[c * 32 + lane] = __uint_as_float(v[c]);
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_reduce_add_5d(&P.tm_dq, stage, q4 * 32, h, s, q0, b);
        bulk_commit();
      }
    }
    if (lane == 0) bulk_wait0();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}
}  // namespace tcbwd

cudaError_t launch_sfa_bwd_main_tc(const void* q, const void* k, const void* v, const void* dout, void* dk,
                                   void* dv, const float* lse2_ws, const float* delta_ws, float* dq_ws,
                                   const SfaGeom& g, float scale, int32_t* status, cudaStream_t st) {
  using namespace tcbwd;
  Params p;
  if (!make_rows_tmap(&p.tm_q, q, g, g.Hq, DH, BQ) || !make_rows_tmap(&p.tm_do, dout, g, g.Hq, DH, BQ) ||
      !make_rows_tmap(&p.tm_k, k, g, g.Hkv, DH, BK) || !make_rows_tmap(&p.tm_v, v, g, g.Hkv, DH, BK) ||
      !make_rows_tmap(&p.tm_dq, dq_ws, g, g.Hq, DH, BQ, 4, 32, false))
    return cudaErrorInvalidValue;
  p.lse2 = lse2_ws;
  p.delta = delta_ws;
  p.dk = (bf16*)dk;
  p.dv = (bf16*)dv;
  p.g = g;
  p.scale = scale;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.status = status;
  const int smem = (int)sizeof(Smem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((g.Lv + BK - 1) / BK, g.Hkv * g.ns, g.B);
  bwd_kernel<<<grid, NTHREADS, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace hdsfa
