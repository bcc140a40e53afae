// Stream-Factorized Attention backward (main pass) on the sm_103a tensor cores,
// head dim 128.
//
// One CTA owns a 128-row key tile j of one virtual causal problem (SfaGeom) and
// one K/V head; it loops over the group's query heads and over the 64-row query
// tiles that can see tile j (causal: query tiles at or after the key tile; LOCAL:
// also within the window).  Per query tile, with TMEM lane = key row:
//   S^T  = K Q^T,  dP^T = V dO^T                      (SS MMA, M=128 N=64 K=128)
//   P^T  = exp2(S^T * scale*log2e - lse2),  dS^T = P^T (dP^T - delta)   (softmax WG)
//   dV  += P^T dO,  dK += dS^T Q                      (TS MMA: P^T, dS^T bf16 in TMEM)
//   dQ^T = K^T dS^T                                   (SS MMA, M=128 (head dim) N=64)
// dQ^T leaves TMEM through the dQ warpgroup: shared memory, then a TMA tensor
// reduce-add (fp32) into the workspace accumulator.  dK, dV stay in TMEM for
// the whole loop and are written once (dK scaled).
//
// Roles (320 threads): warp 0 TMA producer (+ TMEM owner), warp 1 MMA issuer,
// warps 2..5 softmax (one key row each), warps 6..9 dQ flush (one head-dim row
// each).  Q/dO/lse2/delta tiles and the S^T/dP^T/dQ^T TMEM buffers are
// double-buffered; every mbarrier wait is bounded.
//
// TMEM columns: S^T[st] at 64*st (P^T bf16 over its first 32), dP^T[st] at
// 128 + 64*st (dS^T bf16 over its first 32, then dQ^T fp32), dV at 256, dK at 384.
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcbwd {
constexpr int BK = 128, BQ = 64, DH = 128, NST = 2, NTHREADS = 320;
constexpr uint32_t COL_DV = 256, COL_DK = 384;
HD_DEVINLINE uint32_t col_st(int st) { return 64u * st; }
HD_DEVINLINE uint32_t col_dpt(int st) { return 128u + 64u * st; }

struct Smem {
  bf16 k[BK * DH];          // 2 swizzle blocks of [128 key rows][64]
  bf16 v[BK * DH];
  bf16 q[NST][BQ * DH];     // 2 swizzle blocks of [64 query rows][64]
  bf16 dO[NST][BQ * DH];
  bf16 ds[NST][BK * BQ];    // dS^T [128 key rows][64 queries], one swizzle block
  float dq[4][BQ * 32];     // per dQ warp: [64 queries][32 head-dim] fp32 staging
  float lse2[NST][BQ];
  float delta[NST][BQ];
  uint64_t kv_full, qd_full[NST], qd_empty[NST], sdp_full[NST], p_ready[NST], dq_full[NST], dq_free[NST],
      kv_done, drain;
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
      mbar_init(&sm.sdp_full[i], 1);
      mbar_init(&sm.p_ready[i], 128);
      mbar_init(&sm.dq_full[i], 1);
      mbar_init(&sm.dq_free[i], 128);
    }
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
      bool ok = mbar_wait(&sm.kv_full, 0, abort, P.status);
      auto issue_rest = [&](int u) -> bool {
        const int su = u & 1;
        if (!mbar_wait(&sm.p_ready[su], (u >> 1) & 1, abort, P.status)) return false;
        tc_fence_after();
        const uint32_t qa = smem_u32(sm.q[su]), da = smem_u32(sm.dO[su]), dsa = smem_u32(sm.ds[su]);
#pragma unroll
        for (int kk = 0; kk < BQ / 16; ++kk) {
          const uint64_t bd = sdesc_sw128(da + kk * 16 * 128, BQ * 128, 1024);
          tc_mma_ts(tmem + COL_DV, tmem + col_st(su) + kk * 8, bd, idKV, (u > 0 || kk > 0) ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < BQ / 16; ++kk) {
          const uint64_t bd = sdesc_sw128(qa + kk * 16 * 128, BQ * 128, 1024);
          tc_mma_ts(tmem + COL_DK, tmem + col_dpt(su) + kk * 8, bd, idKV, (u > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&sm.qd_empty[su]);
        // dQ^T overwrites the dP^T / dS^T columns only after the dK MMA above read them
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(ka + kk * 16 * 128, BK * 128, 1024);
          const uint64_t bd = sdesc_sw128(dsa + kk * 16 * 128, BK * 128, 1024);
          tc_mma_ss(tmem + col_dpt(su), ad, bd, idQ, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sm.dq_full[su]);
        return true;
      };
      for (int t = 0; ok && t < T; ++t) {
        const int st = t & 1;
        if (!mbar_wait(&sm.qd_full[st], (t >> 1) & 1, abort, P.status)) break;
        if (t >= NST && !mbar_wait(&sm.dq_free[st], ((t - NST) >> 1) & 1, abort, P.status)) break;
        tc_fence_after();
        const uint32_t qa = smem_u32(sm.q[st]), da = smem_u32(sm.dO[st]);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t ak = sdesc_sw128(ka + (kk >> 2) * (BK * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bq = sdesc_sw128(qa + (kk >> 2) * (BQ * 128) + (kk & 3) * 32, 16, 1024);
          tc_mma_ss(tmem + col_st(st), ak, bq, idS, kk > 0 ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t av = sdesc_sw128(va + (kk >> 2) * (BK * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bo = sdesc_sw128(da + (kk >> 2) * (BQ * 128) + (kk & 3) * 32, 16, 1024);
          tc_mma_ss(tmem + col_dpt(st), av, bo, idS, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sm.sdp_full[st]);
        if (t >= 1 && !issue_rest(t - 1)) { ok = false; break; }
      }
      if (ok && T > 0) ok = issue_rest(T - 1);
      tc_commit(&sm.kv_done);
      tc_commit(&sm.drain);
      mbar_drain(&sm.drain, 0);
    }
  } else if (warp < 6) {
    // ------------------------------------------------------------ softmax (key rows)
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int kr = n0 + row;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const float c2 = P.scale_log2;
    uint8_t* dsrow0 = reinterpret_cast<uint8_t*>(sm.ds[0]) + row * 128;
    uint8_t* dsrow1 = reinterpret_cast<uint8_t*>(sm.ds[1]) + row * 128;
    bool ok = true;
    for (int t = 0; t < T; ++t) {
      const int st = t & 1;
      const int q0 = (i_lo + t % nq) * BQ;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.sdp_full[st], (t >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[BQ], dr[BQ];
      tmem_ld32(tl + col_st(st), sr);
      tmem_ld32(tl + col_st(st) + 32, sr + 32);
      tmem_ld32(tl + col_dpt(st), dr);
      tmem_ld32(tl + col_dpt(st) + 32, dr + 32);
      tmem_ld_wait();
      const float* l2 = sm.lse2[st];
      const float* dl = sm.delta[st];
      const bool need_mask = (q0 < n0 + BK) || G.window > 0 || (n0 + BK > G.Lv) || (q0 + BQ > G.Lv);
      uint32_t pp[BQ / 2], dd[BQ / 2];
#pragma unroll
      for (int c = 0; c < BQ; c += 2) {
        float p0 = ex2_approx(fmaf(__uint_as_float(sr[c]), c2, -l2[c]));
        float p1 = ex2_approx(fmaf(__uint_as_float(sr[c + 1]), c2, -l2[c + 1]));
        if (need_mask) {
          if (!visible(q0 + c, kr, G.Lv, G.window)) p0 = 0.f;
          if (!visible(q0 + c + 1, kr, G.Lv, G.window)) p1 = 0.f;
        }
        const float d0 = p0 * (__uint_as_float(dr[c]) - dl[c]);
        const float d1 = p1 * (__uint_as_float(dr[c + 1]) - dl[c + 1]);
        pp[c >> 1] = cvt_bf16x2(p0, p1);
        dd[c >> 1] = cvt_bf16x2(d0, d1);
      }
      tmem_st16(tl + col_st(st), pp);
      tmem_st16(tl + col_st(st) + 16, pp + 16);
      tmem_st16(tl + col_dpt(st), dd);
      tmem_st16(tl + col_dpt(st) + 16, dd + 16);
      // dS^T row -> shared memory for the dQ MMA; the buffer was last read by tile t-2's dQ MMA
      if (t >= NST && !__all_sync(0xffffffffu, mbar_wait(&sm.dq_full[st], ((t - NST) >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      uint8_t* dsrow = st ? dsrow1 : dsrow0;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        *reinterpret_cast<uint4*>(dsrow + ((c ^ (row & 7)) << 4)) =
            make_uint4(dd[4 * c], dd[4 * c + 1], dd[4 * c + 2], dd[4 * c + 3]);
      fence_async_smem();
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&sm.p_ready[st]);
    }
    // dK, dV epilogue: this thread's key row
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.kv_done, 0, abort, P.status))) {
      tc_fence_after();
      const long long orow = (((long long)b * G.nL + (long long)kr * G.rs + s) * G.Hkv + kvh) * DH;
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        const float mul = which ? P.scale : 1.f;
        bf16* dst = (which ? P.dk : P.dv) + orow;
        const uint32_t col = which ? COL_DK : COL_DV;
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
    }
  } else {
    // ------------------------------------------------------------ dQ flush (head-dim rows)
    const int q4 = warp & 3;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    float* stage = sm.dq[q4];
    for (int t = 0; t < T; ++t) {
      const int st = t & 1;
      const int h = kvh * grp + t / nq, q0 = (i_lo + t % nq) * BQ;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.dq_full[st], (t >> 1) & 1, abort, P.status))) break;
      tc_fence_after();
      uint32_t v[BQ];
      tmem_ld32(tl + col_dpt(st), v);
      tmem_ld32(tl + col_dpt(st) + 32, v + 32);
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(&sm.dq_free[st]);
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
