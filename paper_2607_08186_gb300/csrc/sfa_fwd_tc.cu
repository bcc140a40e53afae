// Stream-Factorized Attention forward on the sm_103a tensor cores.
//
// One CTA computes a 128-row query tile of one virtual causal problem (SfaGeom):
// in WITHIN mode the problem is one stream (rows p = t*n + s, Eq. 4), so the tile
// visits only that stream's key tiles; CROSS is causal over all nL positions
// (Fig. 2a); LOCAL adds the window (Fig. 2b).  Key tiles past the diagonal (or
// before the window) are skipped; tiles straddling a mask edge are masked in
// registers.  A final-stream problem has only the L final-stream queries (dense
// [B][L] tensors) against the same keys: query row r stands at key row
// r*qstep + qoff, which sets its tile range and mask.
//
// A CTA owns two 128-row query tiles (groups g = 0, 1).  Where a K/V group has an
// even number of query heads (GQA), they are the same rows of two of its heads, so
// both see the same key tiles and finish together; otherwise rows m0 and m0 + 128 of
// one head (the second tile then runs one key tile longer: measured as about 2 us of
// a WITHIN CTA's 35 us, the first tile's softmax warps idle meanwhile).
// Roles (320 threads):
//   warp 0      TMA producer: both Q tiles once, then K/V tiles into a 2-stage ring;
//               owns TMEM.
//   warp 1      MMA issuer: the whole warp runs the issue loop, one elected lane
//               issues.  Per key tile and group: S_g = Q_g K^T (SS) into the group's
//               128 TMEM columns, O_g += P_g V (TS: P_g read from TMEM) into its O
//               columns; the next S_g is issued after the PV that reads P_g.
//   warps 2..5, 6..9  softmax of group 0 / 1: one thread per query row (its TMEM
//               lane); online softmax in fp32 with exp2 (packed f32x2 arithmetic),
//               P packed to bf16 over the first 64 columns of S_g, O_g rescaled in
//               TMEM only when the running max grows by more than 2^8, epilogue.
// K/V tiles use the 128-byte swizzle written by TMA.  Every mbarrier wait is bounded.
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcfwd {
constexpr int BM = 128, BN = 128, NST = 2, NG = 2, NTHREADS = 64 + NG * 128;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: P stays <= 256 between O rescales

template <int DH>
struct Smem {
  bf16 q[NG][BM * DH];  // per query tile: DH/64 swizzle blocks of [BM][64]
  bf16 k[NST][BN * DH];
  bf16 v[NST][BN * DH];
  uint64_t q_full, kv_full[NST], kv_empty[NST], s_full[NG], p_full[NG], o_done[NG], drain;
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
  int head_pairs;  // 1: a CTA's two query tiles are the same rows of two heads of one K/V group
};

// Key row c visible from the query at key row rq (= r*qstep + qoff).
HD_DEVINLINE bool visible(int rq, int c, int Lv, int window) {
  return c <= rq && c < Lv && (window <= 0 || rq - c < window);
}

// Key-tile range [lo, hi] of the query tile starting at row m0 (hi < lo: no rows).
HD_DEVINLINE void tile_range(const SfaGeom& G, int m0, int& lo, int& hi) {
  if (m0 >= G.Lq) {
    lo = 0;
    hi = -1;
    return;
  }
  const int rq_first = m0 * G.qstep + G.qoff, rq_last = (min(m0 + BM, G.Lq) - 1) * G.qstep + G.qoff;
  lo = G.window > 0 ? max(0, rq_first - G.window + 1) / BN : 0;
  hi = min(rq_last / BN, (G.Lv - 1) / BN);
}

// TMEM columns: S_g at g*128 (P_g packed bf16 over its first 64 columns), O_g at 256 + g*DH.
// NAIVE: the naive intra-stream schedule (G.smod > 1): every tile is masked, a pair
// also needing key row = query row (mod smod); its own instantiation, so the other
// modes' softmax carries none of that code.
template <int DH, bool NAIVE>
__global__ void __launch_bounds__(NTHREADS, 1) fwd_kernel(const __grid_constant__ Params P) {
  extern __shared__ uint8_t smem_raw[];
  Smem<DH>& sm = *reinterpret_cast<Smem<DH>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SfaGeom& G = P.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // A CTA's two query tiles: with head_pairs the same 128 rows of heads 2x and 2x+1
  // (one K/V group: both tiles see exactly the same key tiles and finish together),
  // else rows m0 and m0 + 128 of one head (the second tile sees one more key tile).
  const int hp = P.head_pairs;
  const int rows_per_cta = hp ? BM : NG * BM;
  const int ncta = (G.Lq + rows_per_cta - 1) / rows_per_cta;
  const int nh = hp ? G.Hq / NG : G.Hq;  // head slots of the grid
  // linear grid, query-tile rank slowest: the last query tiles (the most key tiles to
  // visit) of every head, stream and batch launch first
  const int per_rank = nh * G.q_ns * G.B;
  const int mt = ncta - 1 - (int)blockIdx.x / per_rank;
  const int hsb = (int)blockIdx.x % per_rank;
  const int b = hsb / (nh * G.q_ns), hx = (hsb / G.q_ns) % nh, s = hsb % G.q_ns;
  int qm[NG], hd[NG];  // first query row and head of each group's tile
#pragma unroll
  for (int g = 0; g < NG; ++g) {
    qm[g] = hp ? mt * BM : mt * NG * BM + g * BM;
    hd[g] = hp ? NG * hx + g : hx;
  }
  const int h = hd[0];
  const int sk = s + G.kv_s0;  // stream of the key problem
  const int kvh = h / (G.Hq / G.Hkv);
  int lo[NG], hi[NG];
#pragma unroll
  for (int g = 0; g < NG; ++g) tile_range(G, qm[g], lo[g], hi[g]);
  const int n_lo = lo[0];
  int n_hi = hi[0];
#pragma unroll
  for (int g = 1; g < NG; ++g) n_hi = max(n_hi, hi[g]);

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    for (int i = 0; i < NST; ++i) {
      mbar_init(&sm.kv_full[i], 1);
      mbar_init(&sm.kv_empty[i], 1);
    }
    for (int g = 0; g < NG; ++g) {
      mbar_init(&sm.s_full[g], 1);
      mbar_init(&sm.p_full[g], 128);
      mbar_init(&sm.o_done[g], 1);
    }
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
      mbar_arrive_expect_tx(&sm.q_full, NG * BM * DH * 2);
      for (int g = 0; g < NG; ++g)
        for (int c = 0; c < DH / 64; ++c)
          tma_load_5d(sm.q[g] + c * BM * 64, &P.tm_q, &sm.q_full, c * 64, hd[g], s, qm[g], b);
      int issued = 0;
      for (int j = n_lo; j <= n_hi; ++j, ++issued) {
        const int it = j - n_lo, st = it % NST;
        if (it >= NST && !mbar_wait(&sm.kv_empty[st], ((it / NST) - 1) & 1, abort, P.status)) break;
        mbar_arrive_expect_tx(&sm.kv_full[st], 2 * BN * DH * 2);
        for (int c = 0; c < DH / 64; ++c) {
          tma_load_5d(sm.k[st] + c * BN * 64, &P.tm_k, &sm.kv_full[st], c * 64, kvh, sk, j * BN, b);
          tma_load_5d(sm.v[st] + c * BN * 64, &P.tm_v, &sm.kv_full[st], c * 64, kvh, sk, j * BN, b);
        }
      }
      // every copy this thread started lands before the CTA may exit
      mbar_drain(&sm.q_full, 0);
      for (int it = max(0, issued - NST); it < issued; ++it) mbar_drain(&sm.kv_full[it % NST], (it / NST) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs the loop (warp-uniform operands); one elected lane issues.
    {
      constexpr uint32_t idS = idesc_bf16(BM, BN, 0, 0);  // S[q][kv] = Q K^T (both K-major)
      constexpr uint32_t idO = idesc_bf16(BM, DH, 0, 1);  // O[q][d] += P V   (P in TMEM, V MN-major)
      int ps[NG] = {0, 0};                                  // per-group P phases consumed
      bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.q_full, 0, abort, P.status));
      int kv_ready = n_lo - 1;                              // highest key tile known loaded
      auto wait_kv = [&](int j) -> bool {
        if (j <= kv_ready) return true;
        const int it = j - n_lo;
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.kv_full[it % NST], (it / NST) & 1, abort, P.status))) return false;
        kv_ready = j;
        tc_fence_after();
        return true;
      };
      // Operand descriptors are encoded once; k-step kk adds its byte offset / 16 to the
      // 64-bit descriptor (the address field; shared addresses stay below 256 KB), which
      // keeps the instructions between consecutive MMAs (and so the issue gaps) small.
      static_assert(BM == 128 && BN == 128 && NST == 2 && NG == 2, "descriptor bases below");
      const uint64_t qK0 = sdesc_sw128(smem_u32(sm.q[0]), 16, 1024), qK1 = sdesc_sw128(smem_u32(sm.q[1]), 16, 1024);
      const uint64_t kK0 = sdesc_sw128(smem_u32(sm.k[0]), 16, 1024), kK1 = sdesc_sw128(smem_u32(sm.k[1]), 16, 1024);
      const uint64_t vM0 = sdesc_sw128(smem_u32(sm.v[0]), BN * 128, 1024),
                     vM1 = sdesc_sw128(smem_u32(sm.v[1]), BN * 128, 1024);
      auto issue_s = [&](int g, int j) {
        const uint64_t qd = g ? qK1 : qK0, kd = ((j - n_lo) & 1) ? kK1 : kK0;
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t off = (uint64_t)((kk >> 2) * (128 * 128 / 16) + (kk & 3) * 2);
          tc_mma_ss_w(tmem + g * 128, qd + off, kd + off, idS, kk > 0 ? 1u : 0u);
        }
        tc_commit_w(&sm.s_full[g]);
      };
      auto issue_pv = [&](int g, int j) -> bool {
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.p_full[g], ps[g] & 1, abort, P.status))) return false;
        ++ps[g];
        tc_fence_after();
        const uint64_t vd = ((j - n_lo) & 1) ? vM1 : vM0;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          tc_mma_ts_w(tmem + 256 + g * DH, tmem + g * 128 + kk * 8, vd + (uint64_t)(kk * 16 * 128 / 16), idO,
                    (j > lo[g] || kk > 0) ? 1u : 0u);
        return true;
      };
      if (ok && n_hi >= n_lo && wait_kv(n_lo)) {
        for (int g = 0; g < NG; ++g)
          if (lo[g] <= n_lo && n_lo <= hi[g]) issue_s(g, n_lo);
        for (int j = n_lo; ok && j <= n_hi; ++j) {
          for (int g = 0; ok && g < NG; ++g) {
            if (lo[g] <= j && j <= hi[g]) {
              if (!issue_pv(g, j)) { ok = false; break; }
              if (j == hi[g]) tc_commit_w(&sm.o_done[g]);
            }
            // S of the next tile for this group reuses its S/P columns: issued after its PV
            if (j + 1 <= hi[g] && lo[g] <= j + 1) {
              if (!wait_kv(j + 1)) { ok = false; break; }
              issue_s(g, j + 1);
            }
          }
          tc_commit_w(&sm.kv_empty[(j - n_lo) % NST]);
        }
      }
      // every MMA issued above completes before TMEM / smem are released
      tc_commit_w(&sm.drain);
      mbar_drain(&sm.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax / epilogue
    const int g = (warp - 2) >> 2;
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int r = qm[g] + row;
    const int hg = hd[g];
    const int rq = r * G.qstep + G.qoff;                      // its key row
    const int rq0 = qm[g] * G.qstep + G.qoff;                 // key row of the tile's first query
    // key row of its last query (a key tile above rq1 - window is inside every row's window)
    const int rq1 = (min(qm[g] + BM, G.Lq) - 1) * G.qstep + G.qoff;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t tS = tl + g * 128, tO = tl + 256 + g * DH;
    const float c2 = P.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;  // m_run in raw score units
    bool ok = true;
    for (int j = lo[g]; j <= hi[g]; ++j) {
      const int i = j - lo[g];
      // tcgen05.ld/st are warp-collective: every wait result is made warp-uniform
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[g], i & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float x[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_ld32(tS + c * 32, reinterpret_cast<uint32_t*>(x) + c * 32);
      tmem_ld_wait();
      // tiles holding a key past the first query's key row (the diagonal band), a key at
      // or below the last query's window edge, and the ragged last tile
      const bool need_mask = (j + 1) * BN - 1 > rq0 || (G.window > 0 && j * BN <= rq1 - G.window) ||
                             (j + 1) * BN > G.Lv;
      if constexpr (NAIVE) {
        // causal (no window in this schedule) and k = (rq - key row) mod smod == 0,
        // k stepped down the tile's columns
        int k = (rq - j * BN) % G.smod;
        if (k < 0) k += G.smod;
#pragma unroll
        for (int e = 0; e < BN; ++e) {
          if (k != 0 || j * BN + e > rq || j * BN + e >= G.Lv) x[e] = -INFINITY;
          k = k == 0 ? G.smod - 1 : k - 1;
        }
      } else if (need_mask) {
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
      // O_g already holds every earlier tile's PV (its S of this tile was issued after them)
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
      // P (bf16 pairs) over the first 64 columns of this group's S
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_st16(tS + c * 16, pk + c * 16);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&sm.p_full[g]);
    }
    if (ok && hi[g] >= lo[g] && __all_sync(0xffffffffu, mbar_wait(&sm.o_done[g], 0, abort, P.status))) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      // O rows leave through shared memory: each thread writes its row (normalised,
      // bf16) into this warp's 32 rows of the group's Q buffer (no longer read: the last
      // S MMA of the group completed before o_done), 16-byte units XOR-swizzled by the
      // row; then every store instruction writes whole rows (DH*2 bytes each, 2 rows at
      // DH = 128), instead of one 16-byte piece of 32 different rows.
      constexpr int UPR = DH * 2 / 16;  // 16-byte units per row
      uint8_t* stg = reinterpret_cast<uint8_t*>(sm.q[g]) + q4 * (32 * DH * 2);
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; e += 8) {
          uint4 w;
          w.x = cvt_bf16x2(__uint_as_float(o[e + 0]) * inv, __uint_as_float(o[e + 1]) * inv);
          w.y = cvt_bf16x2(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
          w.z = cvt_bf16x2(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv);
          w.w = cvt_bf16x2(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv);
          const int u = c * 4 + e / 8;
          *reinterpret_cast<uint4*>(stg + lane * (DH * 2) + ((u ^ (lane & 7)) << 4)) = w;
        }
      }
      __syncwarp();
      {
        const long long rstride = (long long)G.q_rs * G.Hq * DH;  // elements between query rows
        bf16* obase = P.o + (((long long)b * G.q_nL + s) * G.Hq + hg) * DH;
        const int r0 = qm[g] + q4 * 32;  // this warp's first row
#pragma unroll
        for (int i = 0; i < 32 * UPR / 32; ++i) {
          const int rr = (i * 32 + lane) / UPR, u = (i * 32 + lane) % UPR;  // row within the warp, unit
          if (r0 + rr < G.Lq)
            *reinterpret_cast<uint4*>(obase + (long long)(r0 + rr) * rstride + u * 8) =
                *reinterpret_cast<const uint4*>(stg + rr * (DH * 2) + ((u ^ (rr & 7)) << 4));
        }
      }
      if (r < G.Lq)
        P.lse[((long long)b * G.Hq + hg) * G.q_nL + (long long)r * G.q_rs + s] = (m_run * c2 + log2f(l_run)) * kLn2;
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
}  // namespace tcfwd

// --------------------------------------------------------------------- host
template <int DH, bool NAIVE>
static cudaError_t tc_fwd_impl(tcfwd::Params& p, cudaStream_t st) {
  const int smem = (int)sizeof(tcfwd::Smem<DH>) + 1024;
  cudaError_t e =
      cudaFuncSetAttribute(tcfwd::fwd_kernel<DH, NAIVE>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int rows_per_cta = p.head_pairs ? tcfwd::BM : tcfwd::NG * tcfwd::BM;
  const int nh = p.head_pairs ? p.g.Hq / tcfwd::NG : p.g.Hq;
  const unsigned grid = (unsigned)((p.g.Lq + rows_per_cta - 1) / rows_per_cta) * (unsigned)(nh * p.g.q_ns * p.g.B);
  tcfwd::fwd_kernel<DH, NAIVE><<<grid, tcfwd::NTHREADS, smem, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_sfa_fwd_tc(const void* q, const void* k, const void* v, void* o, float* lse,
                              const SfaGeom& g, int Dh, float scale, int32_t* status, cudaStream_t st) {
  tcfwd::Params p;
  if (!make_rows_tmap(&p.tm_q, q, query_geom(g), g.Hq, Dh, tcfwd::BM) ||
      !make_rows_tmap(&p.tm_k, k, g, g.Hkv, Dh, tcfwd::BN) ||
      !make_rows_tmap(&p.tm_v, v, g, g.Hkv, Dh, tcfwd::BN))
    return cudaErrorInvalidValue;
  p.o = (bf16*)o;
  p.lse = lse;
  p.g = g;
  p.scale_log2 = scale * tcfwd::kLog2e;
  p.status = status;
  p.head_pairs = (g.Hq / g.Hkv) % tcfwd::NG == 0;
  if (Dh == 64) return tc_fwd_impl<64, false>(p, st);
  return g.smod > 1 ? tc_fwd_impl<128, true>(p, st) : tc_fwd_impl<128, false>(p, st);
}

}  // namespace hdsfa
