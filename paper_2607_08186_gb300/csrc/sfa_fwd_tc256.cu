// Stream-Factorized Attention forward on the sm_103a tensor cores, head dim 256
// (the 80B configuration's heads, Table 6).
//
// Same problem and masks as the head-dim <= 128 forward (Eq. 4, Fig. 2a/2b, and the
// final-stream query geometry of Sec. 3.1); the tile plan differs because a 128-row
// query tile's O accumulator alone takes 256 of the 512 TMEM columns and its Q tile
// 64 KB of shared memory:
//   TMEM   S in two 128-column buffers (S of key tile j+1 is computed while the
//          softmax of tile j runs; P packed bf16 over the first 64 columns of its S
//          buffer), O over columns 256..511.
//   smem   Q (four [128][64] swizzle blocks, 64 KB) and a ring of five 32 KB slots;
//          a slot holds one half of a K or V tile (head-dim columns [0,128) or
//          [128,256), two [128][64] swizzle blocks).  The producer fills the slots in
//          the order the MMA issuer consumes them:
//            K(lo); then for each key tile j: K(j+1), V(j)
//          which is the issue order S(lo), S(lo+1), PV(lo), S(lo+2), PV(lo+1), ...
//          A slot is released by a tcgen05 commit after the MMAs that read it.
// Roles (192 threads, one CTA per 128-row query tile):
//   warp 0      TMA producer (Q once, then K / V halves into the ring); owns TMEM.
//   warp 1      MMA issuer (the whole warp runs the loop, one elected lane issues):
//               S = Q K^T (SS, 16 k-steps over the two K halves), then after the
//               softmax has written P: O[:, 0:128] += P V_a, O[:, 128:256] += P V_b
//               (TS, P read from TMEM, V MN-major).
//   warps 2..5  online softmax, one thread per query row (its TMEM lane), fp32 with
//               exp2; O is rescaled in TMEM only when the running max grows by more
//               than 2^8, and only after the previous tile's PV has completed (the
//               issuer runs S(j+1) ahead of PV(j)); epilogue writes O (bf16) and LSE.
// Every mbarrier wait is bounded.
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcfwd256 {
constexpr int DH = 256, BM = 128, BN = 128, NSLOT = 5, NTHREADS = 192;
constexpr uint32_t COL_O = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: P stays <= 256 between O rescales

struct Smem {
  bf16 q[DH / 64][BM * 64];        // Q tile: four [128 rows][64] swizzle blocks
  bf16 ring[NSLOT][2][BN * 64];    // per slot: two [128 rows][64] swizzle blocks
  uint64_t q_full, full[NSLOT], empty[NSLOT], s_full[2], p_full[2], pv_done, drain;
  uint32_t tmem_base;
  int abort;
};

struct Params {
  CUtensorMap tm_q, tm_k, tm_v;
  bf16* o;
  float* lse;
  SfaGeom g;
  float scale_log2;
  int32_t* status;
};

HD_DEVINLINE bool visible(int rq, int c, int Lv, int window) {
  return c <= rq && c < Lv && (window <= 0 || rq - c < window);
}

// Unit u of the ring sequence K(lo), K(lo+1), V(lo), K(lo+2), V(lo+1), ..., V(hi), two
// units (halves) per tile: its key tile, tensor (0 = K, 1 = V) and half.
HD_DEVINLINE void unit_of(int u, int lo, int hi, int& j, int& isv, int& half) {
  half = u & 1;
  const int p = u >> 1;  // pair index: 0 = K(lo); then 2i+1 = K(lo+1+i) (if any), 2i+2 = V(lo+i)
  if (p == 0) {
    j = lo;
    isv = 0;
    return;
  }
  const int ntk = hi - lo;  // K tiles after the first
  const int i = (p - 1) >> 1;
  if (((p - 1) & 1) == 0 && i < ntk) {
    j = lo + 1 + i;
    isv = 0;
    return;
  }
  // V tiles: before the K tiles run out they alternate; afterwards only V remains
  const int vi = i < ntk ? i : (p - 1) - ntk;
  j = lo + vi;
  isv = 1;
}

__global__ void __launch_bounds__(NTHREADS, 1) fwd256_kernel(const __grid_constant__ Params P) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SfaGeom& G = P.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ncta = (G.Lq + BM - 1) / BM;
  // query-tile rank slowest, last tiles (most key tiles) first
  const int per_rank = G.Hq * G.q_ns * G.B;
  const int mt = ncta - 1 - (int)blockIdx.x / per_rank;
  const int hsb = (int)blockIdx.x % per_rank;
  const int m0 = mt * BM;
  const int b = hsb / (G.Hq * G.q_ns), h = (hsb / G.q_ns) % G.Hq, s = hsb % G.q_ns;
  const int sk = s + G.kv_s0;
  const int kvh = h / (G.Hq / G.Hkv);
  const int rq_first = m0 * G.qstep + G.qoff, rq_last = (min(m0 + BM, G.Lq) - 1) * G.qstep + G.qoff;
  const int lo = G.window > 0 ? max(0, rq_first - G.window + 1) / BN : 0;
  const int hi = min(rq_last / BN, (G.Lv - 1) / BN);
  const int ntiles = hi - lo + 1;  // >= 1: every query sees its own key row
  const int nunits = 4 * ntiles;

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    for (int i = 0; i < NSLOT; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.s_full[i], 1);
      mbar_init(&sm.p_full[i], 128);
    }
    mbar_init(&sm.pv_done, 1);
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
      tma_prefetch(&P.tm_k);
      tma_prefetch(&P.tm_v);
      mbar_arrive_expect_tx(&sm.q_full, BM * DH * 2);
      for (int c = 0; c < DH / 64; ++c) tma_load_5d(sm.q[c], &P.tm_q, &sm.q_full, c * 64, h, s, m0, b);
      int issued = 0;
      for (int u = 0; u < nunits; ++u, ++issued) {
        const int slot = u % NSLOT;
        if (u >= NSLOT && !mbar_wait(&sm.empty[slot], ((u / NSLOT) - 1) & 1, abort, P.status)) break;
        int j, isv, half;
        unit_of(u, lo, hi, j, isv, half);
        const CUtensorMap* tm = isv ? &P.tm_v : &P.tm_k;
        mbar_arrive_expect_tx(&sm.full[slot], BN * 128 * 2);
        tma_load_5d(sm.ring[slot][0], tm, &sm.full[slot], half * 128, kvh, sk, j * BN, b);
        tma_load_5d(sm.ring[slot][1], tm, &sm.full[slot], half * 128 + 64, kvh, sk, j * BN, b);
      }
      // every copy this thread started lands before the CTA may exit
      mbar_drain(&sm.q_full, 0);
      for (int u = max(0, issued - NSLOT); u < issued; ++u) mbar_drain(&sm.full[u % NSLOT], (u / NSLOT) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idS = idesc_bf16(BM, BN, 0, 0);   // S[q][kv] = Q K^T (both K-major)
    constexpr uint32_t idO = idesc_bf16(BM, 128, 0, 1);  // O[q][d half] += P V (V MN-major)
    bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.q_full, 0, abort, P.status));
    int u = 0;  // next ring unit to consume
    auto wait_unit = [&](int x) -> bool {
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.full[x % NSLOT], (x / NSLOT) & 1, abort, P.status))) return false;
      tc_fence_after();
      return true;
    };
    // Descriptors are encoded once at the first block / slot; a block, slot or k-step
    // adds its byte offset / 16 (the address field; shared addresses stay below 256 KB).
    // The Q blocks and the ring slots are contiguous: block c at +16 KB * c, slot i at
    // +32 KB * i.
    static_assert(sizeof(Smem::q[0]) == 16384 && sizeof(Smem::ring[0]) == 32768, "descriptor strides");
    const uint64_t qd = sdesc_sw128(smem_u32(sm.q[0]), 16, 1024);
    const uint64_t rd = sdesc_sw128(smem_u32(sm.ring[0][0]), 16, 1024);        // K half, K-major
    const uint64_t rv = sdesc_sw128(smem_u32(sm.ring[0][0]), BN * 128, 1024);  // V half, MN-major (LBO: next 64 columns)
    // S(j) into buffer sb: k-steps 0..7 from the K half in unit u, 8..15 from unit u+1
    auto issue_s = [&](int sb) -> bool {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        if (!wait_unit(u + hf)) return false;
        const int slot = (u + hf) % NSLOT;
        const uint64_t kd = rd + (uint64_t)(slot * (32768 / 16));
#pragma unroll
        for (int k8 = 0; k8 < 8; ++k8) {
          const int kk = hf * 8 + k8;
          const uint64_t qo = (uint64_t)((kk >> 2) * (16384 / 16) + (kk & 3) * 2);
          const uint64_t ko = (uint64_t)((k8 >> 2) * (16384 / 16) + (k8 & 3) * 2);
          tc_mma_ss_w(tmem + sb * 128, qd + qo, kd + ko, idS, kk > 0 ? 1u : 0u);
        }
        tc_commit_w(&sm.empty[slot]);
      }
      u += 2;
      tc_commit_w(&sm.s_full[sb]);
      return true;
    };
    // PV(j) from buffer sb: O[:, 128*hf ..] += P V_hf over the 128 keys (8 k-steps)
    auto issue_pv = [&](int sb, bool acc0) -> bool {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        if (!wait_unit(u + hf)) return false;
        const int slot = (u + hf) % NSLOT;
        const uint64_t vd = rv + (uint64_t)(slot * (32768 / 16));
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          tc_mma_ts_w(tmem + COL_O + hf * 128, tmem + sb * 128 + kk * 8, vd + (uint64_t)(kk * 16 * 128 / 16), idO,
                      (acc0 || kk > 0) ? 1u : 0u);
        tc_commit_w(&sm.empty[slot]);
      }
      u += 2;
      tc_commit_w(&sm.pv_done);
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int i = 0; ok && i < ntiles; ++i) {
      if (i + 1 < ntiles && !issue_s((i + 1) & 1)) {
        ok = false;
        break;
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.p_full[i & 1], (i >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (!issue_pv(i & 1, i > 0)) ok = false;
    }
    // every MMA issued above completes before TMEM / smem are released
    tc_commit_w(&sm.drain);
    mbar_drain(&sm.drain, 0);
  } else {
    // ------------------------------------------------------------ softmax / epilogue
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int r = m0 + row;
    const int rq = r * G.qstep + G.qoff;
    const int rq0 = rq_first;
    const int rq1 = rq_last;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t tO = tl + COL_O;
    const float c2 = P.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int i = 0; i < ntiles; ++i) {
      const int j = lo + i;
      const uint32_t tS = tl + (uint32_t)((i & 1) * 128);
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[i & 1], (i >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float x[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_ld32(tS + c * 32, reinterpret_cast<uint32_t*>(x) + c * 32);
      tmem_ld_wait();
      const bool need_mask = (j + 1) * BN - 1 > rq0 || (G.window > 0 && j * BN <= rq1 - G.window) ||
                             (j + 1) * BN > G.Lv;
      if (need_mask) {
#pragma unroll
        for (int e = 0; e < BN; ++e)
          if (!visible(rq, j * BN + e, G.Lv, G.window)) x[e] = -INFINITY;
      }
      float mx[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = x[e];
#pragma unroll
      for (int e = 8; e < BN; ++e) mx[e & 7] = fmaxf(mx[e & 7], x[e]);
      const float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                               fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      const float m_new = fmaxf(m_run, tmax);
      const bool rescale = (m_run == -INFINITY) || ((m_new - m_run) * c2 > kRescaleThreshold);
      const float m_use = rescale ? m_new : m_run;
      const float neg = (m_use == -INFINITY) ? 0.f : -m_use * c2;
      const uint64_t c2x2 = f2pack(c2, c2), neg2 = f2pack(neg, neg);
      uint64_t sum2[4] = {0, 0, 0, 0};
      uint32_t pk[BN / 2];
#pragma unroll
      for (int e = 0; e < BN; e += 2) {
        float a0, a1;
        f2unpack(ffma2(f2pack(x[e], x[e + 1]), c2x2, neg2), a0, a1);
        const float p0 = ex2_approx(a0), p1 = ex2_approx(a1);
        sum2[(e >> 1) & 3] = fadd2(sum2[(e >> 1) & 3], f2pack(p0, p1));
        pk[e >> 1] = cvt_bf16x2(p0, p1);
      }
      float s0, s1, s2, s3, s4, s5, s6, s7;
      f2unpack(sum2[0], s0, s1);
      f2unpack(sum2[1], s2, s3);
      f2unpack(sum2[2], s4, s5);
      f2unpack(sum2[3], s6, s7);
      const float rsum = ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
      // O holds the PVs of tiles < i only once PV(i-1) has completed (S(i) was issued
      // before it): wait for it before touching O
      if (i > 0) {
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.pv_done, (i - 1) & 1, abort, P.status))) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      const bool mine = rescale && m_run != -INFINITY && i > 0;
      if (__any_sync(0xffffffffu, mine)) {
        const float alpha = mine ? ex2_approx((m_run - m_use) * c2) : 1.f;
        l_run *= alpha;
#pragma unroll
        for (int c = 0; c < DH / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(tO + c * 32, o);
        }
      }
      m_run = m_use;
      l_run += rsum;
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_st16(tS + c * 16, pk + c * 16);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&sm.p_full[i & 1]);
    }
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.pv_done, (ntiles - 1) & 1, abort, P.status))) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      bf16* orow = P.o + (((long long)b * G.q_nL + (long long)r * G.q_rs + s) * G.Hq + h) * DH;
#pragma unroll 1
      for (int c = 0; c < DH / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_ld_wait();
        if (r < G.Lq) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = cvt_bf16x2(__uint_as_float(o[e + 0]) * inv, __uint_as_float(o[e + 1]) * inv);
            w.y = cvt_bf16x2(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
            w.z = cvt_bf16x2(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv);
            w.w = cvt_bf16x2(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + c * 32 + e) = w;
          }
        }
      }
      if (r < G.Lq)
        P.lse[((long long)b * G.Hq + h) * G.q_nL + (long long)r * G.q_rs + s] = (m_run * c2 + log2f(l_run)) * kLn2;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}
}  // namespace tcfwd256

cudaError_t launch_sfa_fwd_tc256(const void* q, const void* k, const void* v, void* o, float* lse,
                                 const SfaGeom& g, float scale, int32_t* status, cudaStream_t st) {
  using namespace tcfwd256;
  Params p;
  if (!make_rows_tmap(&p.tm_q, q, query_geom(g), g.Hq, DH, BM) || !make_rows_tmap(&p.tm_k, k, g, g.Hkv, DH, BN) ||
      !make_rows_tmap(&p.tm_v, v, g, g.Hkv, DH, BN))
    return cudaErrorInvalidValue;
  p.o = (bf16*)o;
  p.lse = lse;
  p.g = g;
  p.scale_log2 = scale * kLog2e;
  p.status = status;
  const int smem = (int)sizeof(Smem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(fwd256_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const unsigned grid = (unsigned)((g.Lq + BM - 1) / BM) * (unsigned)(g.Hq * g.q_ns * g.B);
  fwd256_kernel<<<grid, NTHREADS, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace hdsfa
