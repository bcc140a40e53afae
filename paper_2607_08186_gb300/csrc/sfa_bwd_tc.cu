// Stream-Factorized Attention backward (main pass) on the sm_103a tensor cores,
// head dims 64 and 128 (template parameter DH).
//
// One CTA owns a 128-row key tile j of one virtual causal problem (SfaGeom) and
// one K/V head; it loops over the group's query heads and over the 128-row query
// tiles that can see tile j (causal: query tiles at or after the key tile; LOCAL:
// also within the window; a final-stream problem maps query row r to key row
// r*qstep + qoff).  Every GEMM is a 128 x 128 x 16k tcgen05 MMA (N = 128
// runs at full tensor rate; N = 64 does not):
//   S'^T = K Q^T - lse2/c2 (-inf on masked pairs),  dP'^T = V dO^T - delta
//                                       SS: A = K / V (K-major), B = Q / dO (K-major),
//                                       accumulated onto TMEM pre-filled with the
//                                       per-query terms and the mask (c2 = scale*log2e,
//                                       lse2 = lse*log2e)
//   P^T  = exp2(c2 S'^T)      (softmax phase A: needs S'^T only)
//   dS^T = P^T dP'^T          (phase B: P^T read back as the bf16 the dV MMA uses)
//                             packed f32x2 arithmetic, exp2 on the SFU
//   dV  += P^T dO,  dK += dS^T Q        TS: A = P^T / dS^T packed bf16 in TMEM
//   dQ   = dS K                         SS: A = dS^T tile in smem read MN-major,
//                                           B = K read MN-major; TMEM lane = query row
// dK and dV stay in TMEM for the whole loop and are written once (dK scaled).  dQ
// of each tile is read out by the dQ warpgroup, staged in shared
// memory (128-byte swizzle) and added into the fp32 workspace accumulator by TMA
// tensor reduce-add.
//
// TMEM: two 128-column regions R0, R1 swap roles with the tile parity p:
//   S^T(t) in R[p] (P^T packed bf16 over its first 64 columns, then dQ(t)),
//   dP^T(t) in R[p^1] (dS^T packed bf16 over its first 64 columns);  dV at 256, dK at 384.
// MMA issue order, issuer X:  for each quarter u of the query columns: wait P^T(t)
//                   quarter u | dV(t) k-steps of u;  then per quarter: wait dS^T(t)
//                   quarter u | dK(t) k-steps of u
//                 issuer Y:  wait dS^T(t) complete and dV(t) done | dQ(t) | wait R[p^1]
//                   pre-filled | S(t+1) | wait dQ(t) read out and R[p] pre-filled | dP(t+1)
// Phase A of tile t+1 needs only S'^T(t+1), so it overlaps the dQ(t) read-out, the
// dP(t+1) pre-fill and the dP(t+1) MMA; dV / dK k-steps run under the later quarters.
// The pre-fills (every TMEM lane gets the same 128 per-query values) are written
// by the dQ warps: R[p^1] once dK(t) has read dS^T(t) (under dQ(t)), R[p] right
// after they have read dQ(t) out of it.
// S(t+1) lands in R[p^1], whose dS^T(t) dK(t) has already consumed (tcgen05 MMAs of
// one thread execute in order), so it overlaps the dQ(t) read-out; dP(t+1) lands in
// R[p] only after that read-out.
//
// Small grids (fewer CTAs than SMs) also split the group's query heads into chunks, one
// CTA each; each chunk writes its fp32
// dK / dV partial sums to a workspace slice of its own, which dkv_finalize_kernel adds
// in chunk order (bwd_head_chunks in common.cuh).
// Roles (480 threads, 128 registers each): warp 0 TMA producer (+ TMEM owner);
// warp 1 MMA issuer X (dV, dK per query quarter; one lane); warp 14 MMA issuer Y
// (dQ, S, dP; the whole warp runs its loop, one elected lane issues, 0.7 % faster than
// one lane; the same for X was 1.7 % slower):
// two issuing threads on different schedulers, because an MMA thread sharing its
// scheduler with a busy softmax warp gets few issue slots, and one thread for all 40
// MMAs and 12 barrier waits of a tile became the critical path; warps 2..5 softmax
// (TMEM lane = key row; 128 query columns in eight 16-column chunks per phase);
// warps 6..9 / 10..13 dQ flush and pre-fill for columns 0..63 / 64..127: each loads
// its 64 dQ columns (TMEM lane = query row), pre-fills the region for the next dP^T,
// then stages two 4 KB rounds through its own buffer.
// Every mbarrier wait is bounded.
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcbwd {
constexpr int BK = 128, BQ = 128, NTHREADS = 480;
constexpr uint32_t COL_DV = 256, COL_DK = 384;
HD_DEVINLINE uint32_t col_r(int r) { return 128u * r; }

template <int DH>
struct Smem {
  bf16 k[BK * DH];        // DH/64 swizzle blocks of [128 key rows][64]
  bf16 v[BK * DH];
  bf16 q[2][BQ * DH];     // double-buffered query tile: DH/64 swizzle blocks of [128 rows][64]
  bf16 dO[BQ * DH];
  bf16 ds[BK * BQ];       // dS^T [128 key rows][128 queries]: 2 swizzle blocks of [128][64]
  float dqs[8][32 * 32];  // per dQ warp: [32 query rows][32 head-dim] fp32, 128-byte swizzle
  float nlse2[2][BQ];     // -lse*log2(e) of the query tile in q[i], loaded with it
  float ndelta[2][BQ];    // -delta of the query tile in q[i], loaded with it
  uint64_t kv_full, q_full[2], q_empty[2], do_full, do_empty, s_full, dp_full, pa_part[4], pb_part[4], dq_full, s_init,
      dp_init, dk_done, dv_done, kv_done, drain;
  uint64_t dq_read[DH == 64 ? 4 : 1];  // DH = 64: both dQ warps of a lane quadrant have read dQ(t)
  uint32_t tmem_base;
  int abort;
};

// The layout, 1024-byte aligned inside the dynamic shared memory, must fit the 227 KB
// per-block limit; the kernel checks the actual alignment pad on entry.
template <int DH>
constexpr int smem_bytes() { return (int)sizeof(Smem<DH>) + 1024 < 232448 ? (int)sizeof(Smem<DH>) + 1024 : 232448; }
static_assert(sizeof(Smem<128>) <= 232448, "backward shared-memory layout exceeds 227 KB");

struct Params {
  CUtensorMap tm_q, tm_do, tm_k, tm_v, tm_dq;
  const float* lse2;   // [B][Hq][ns][Lvp]
  const float* delta;  // [B][Hq][ns][Lvp]
  bf16* dk;
  bf16* dv;
  float* dkv;   // head chunks > 1: fp32 partial sums [chunks][2][B][q_ns][Lv][Hkv][DH] (dV, dK)
  int hchunks;  // query-head chunks per K/V head (bwd_head_chunks)
  SfaGeom g;
  float scale, scale_log2;
  int32_t* status;
};


// WIN: a windowed (LOCAL) problem, whose pre-fill masks only tiles that reach the
// window edge; the other modes keep a separate instantiation.  DH = 64: dQ, dK and
// dV are 64 columns wide (N = 64 MMAs for dV, dK, dQ) and each dQ warp reads out 32
// of them instead of 64; S^T, dP^T and the pre-fills are as at 128.
template <int DH, bool WIN>
__global__ void __launch_bounds__(NTHREADS, 1) bwd_kernel(const __grid_constant__ Params P) {
  static_assert(DH == 64 || DH == 128, "head dim 64 or 128");
  extern __shared__ uint8_t smem_raw[];
  {
    uint32_t dyn;
    asm("mov.u32 %0, %%dynamic_smem_size;\n" : "=r"(dyn));
    const uintptr_t base = reinterpret_cast<uintptr_t>(smem_raw);
    if (((base + 1023) & ~uintptr_t(1023)) - base + sizeof(Smem<DH>) > dyn) {  // uniform: nothing touched yet
      if (threadIdx.x == 0) set_status(P.status, HD_DEVBIT_TIMEOUT);
      return;
    }
  }
  Smem<DH>& sm = *reinterpret_cast<Smem<DH>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SfaGeom& G = P.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // linear grid, key tile slowest: every CTA of key tile 0 (the most query tiles to
  // visit) launches before any of tile 1, and so on, over all heads, streams and batches
  // (and head chunks, neighbours)
  const int HC = P.hchunks;
  const int per_tile = HC * G.Hkv * G.q_ns * G.B;
  const int j = (int)blockIdx.x / per_tile;
  const int rem = (int)blockIdx.x % per_tile;
  const int hc = rem % HC, hsb = rem / HC;
  const int n0 = j * BK;
  const int b = hsb / (G.Hkv * G.q_ns), kvh = (hsb / G.q_ns) % G.Hkv, s = hsb % G.q_ns;
  const int sk = s + G.kv_s0;  // stream of the key problem
  // this CTA's query heads: chunk hc of the group's heads
  const int grp_all = G.Hq / G.Hkv, hper = (grp_all + HC - 1) / HC;
  const int grp = min(hper, grp_all - hc * hper);  // heads of this chunk (>= 1)
  const int h_base = kvh * grp_all + hc * hper;
  // query rows that can see a key of the tile: key row r*qstep + qoff >= n0, and under
  // a window r*qstep + qoff < n0 + BK - 1 + window
  const int i_lo = (n0 <= G.qoff ? 0 : (n0 - G.qoff + G.qstep - 1) / G.qstep) / BQ;
  int i_hi = (G.Lq - 1) / BQ;
  if (G.window > 0) i_hi = min(i_hi, ((n0 + BK - 2 + G.window - G.qoff) / G.qstep) / BQ);
  const int nq = i_hi - i_lo + 1;
  const int T = grp * nq;
  const int Lqp = row_terms_pitch(G.Lq);
  if (nq <= 0) {  // no query sees this key tile: its dK and dV rows are zero
    if (HC > 1) {  // this chunk's slice rows are zero
      const size_t half = (size_t)G.B * G.q_ns * G.Lv * G.Hkv * DH;
      for (int i = threadIdx.x; i < BK * (DH / 4); i += NTHREADS) {
        const int kr = n0 + i / (DH / 4), c4 = i % (DH / 4);
        if (kr >= G.Lv) continue;
        const long long wrow = ((((long long)b * G.q_ns + s) * G.Lv + kr) * G.Hkv + kvh) * DH + c4 * 4;
        *reinterpret_cast<float4*>(P.dkv + (2 * hc) * half + wrow) = make_float4(0.f, 0.f, 0.f, 0.f);
        *reinterpret_cast<float4*>(P.dkv + (2 * hc + 1) * half + wrow) = make_float4(0.f, 0.f, 0.f, 0.f);
      }
      return;
    }
    for (int i = threadIdx.x; i < BK * (DH / 8); i += NTHREADS) {
      const int kr = n0 + i / (DH / 8), c = i % (DH / 8);
      if (kr >= G.Lv) continue;
      const long long orow = (((long long)b * G.nL + (long long)kr * G.rs + sk) * G.Hkv + kvh) * DH + c * 8;
      *reinterpret_cast<uint4*>(P.dk + orow) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(P.dv + orow) = make_uint4(0, 0, 0, 0);
    }
    return;
  }

  if (threadIdx.x == 0) {
    mbar_init(&sm.kv_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.q_full[i], 1);
      mbar_init(&sm.q_empty[i], 1);
    }
    mbar_init(&sm.do_full, 1);
    mbar_init(&sm.do_empty, 2);  // dV(t) (issuer X) and dP(t) (issuer Y) both read dO(t)
    mbar_init(&sm.s_full, 1);
    mbar_init(&sm.dp_full, 1);
    for (int i = 0; i < 4; ++i) {
      mbar_init(&sm.pa_part[i], 128);
      mbar_init(&sm.pb_part[i], 128);
    }
    mbar_init(&sm.dq_full, 1);
    mbar_init(&sm.s_init, 256);
    mbar_init(&sm.dp_init, 256);
    mbar_init(&sm.dk_done, 1);
    mbar_init(&sm.dv_done, 1);
    mbar_init(&sm.kv_done, 1);
    mbar_init(&sm.drain, 2);
    if (DH == 64)
      for (int i = 0; i < 4; ++i) mbar_init(&sm.dq_read[i], 64);
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
        tma_load_5d(sm.k + c * BK * 64, &P.tm_k, &sm.kv_full, c * 64, kvh, sk, n0, b);
        tma_load_5d(sm.v + c * BK * 64, &P.tm_v, &sm.kv_full, c * 64, kvh, sk, n0, b);
      }
      int nq_issued = 0, ndo_issued = 0;
      // query tiles (with their row terms) run up to two ahead (double buffer); dO one ahead
      for (int t = 0; t < T; ++t) {
        const int h = h_base + t / nq, q0 = (i_lo + t % nq) * BQ;
        const int qb = t & 1;
        if (t >= 2 && !mbar_wait(&sm.q_empty[qb], ((t - 2) >> 1) & 1, abort, P.status)) break;
        mbar_arrive_expect_tx(&sm.q_full[qb], BQ * DH * 2 + 2 * BQ * 4);
        for (int c = 0; c < DH / 64; ++c)
          tma_load_5d(sm.q[qb] + c * BQ * 64, &P.tm_q, &sm.q_full[qb], c * 64, h, s, q0, b);
        const long long off = (((long long)b * G.Hq + h) * G.q_ns + s) * Lqp + q0;
        bulk_load(sm.nlse2[qb], P.lse2 + off, BQ * 4, &sm.q_full[qb]);
        bulk_load(sm.ndelta[qb], P.delta + off, BQ * 4, &sm.q_full[qb]);
        ++nq_issued;
        if (t >= 1 && !mbar_wait(&sm.do_empty, (t - 1) & 1, abort, P.status)) break;
        mbar_arrive_expect_tx(&sm.do_full, BQ * DH * 2);
        for (int c = 0; c < DH / 64; ++c)
          tma_load_5d(sm.dO + c * BQ * 64, &P.tm_do, &sm.do_full, c * 64, h, s, q0, b);
        ++ndo_issued;
      }
      // every copy this thread started lands before the CTA may exit
      mbar_drain(&sm.kv_full, 0);
      for (int t = max(0, nq_issued - 2); t < nq_issued; ++t) mbar_drain(&sm.q_full[t & 1], (t >> 1) & 1);
      if (ndo_issued > 0) mbar_drain(&sm.do_full, (ndo_issued - 1) & 1);
    }
  } else if (warp == 1 || warp == NTHREADS / 32 - 1) {
    // ------------------------------------------------------------ MMA issuers
    if (lane == 0 || warp != 1) {  // issuer X: one lane; issuer Y: the whole warp, elected lanes issue
      constexpr uint32_t idSP = idesc_bf16(128, BQ, 0, 0);  // S^T, dP^T: A = K / V, B = Q / dO (K-major)
      constexpr uint32_t idKV = idesc_bf16(128, DH, 0, 1);  // dV, dK: A in TMEM, B = dO / Q MN-major
      constexpr uint32_t idQ = idesc_bf16(128, DH, 1, 1);   // dQ: A = dS (dS^T tile MN-major), B = K MN-major
      // Operand descriptors are encoded once; k-step kk adds its byte offset / 16 to the
      // 64-bit descriptor (the address field; shared addresses stay below 256 KB).  The
      // fewer instructions between consecutive MMAs, the better the tensor pipe is fed:
      // encoding a descriptor per k-step cost ~30-40 cycles of issue per MMA.
      static_assert(BK == 128 && BQ == 128, "one 128-row swizzle block is 16 KB");
      const uint64_t kK = sdesc_sw128(smem_u32(sm.k), 16, 1024), vK = sdesc_sw128(smem_u32(sm.v), 16, 1024);
      const uint64_t doK = sdesc_sw128(smem_u32(sm.dO), 16, 1024);
      const uint64_t qK0 = sdesc_sw128(smem_u32(sm.q[0]), 16, 1024), qK1 = sdesc_sw128(smem_u32(sm.q[1]), 16, 1024);
      const uint64_t doM = sdesc_sw128(smem_u32(sm.dO), BQ * 128, 1024);
      const uint64_t qM0 = sdesc_sw128(smem_u32(sm.q[0]), BQ * 128, 1024),
                     qM1 = sdesc_sw128(smem_u32(sm.q[1]), BQ * 128, 1024);
      const uint64_t dsM = sdesc_sw128(smem_u32(sm.ds), BK * 128, 1024), kM = sdesc_sw128(smem_u32(sm.k), BK * 128, 1024);
      // K-major k-step: 32 bytes inside a 64-column block, 16 KB per block; MN-major: 16 rows of 128 bytes
      auto koff = [](int kk) { return (uint64_t)((kk >> 2) * (128 * 128 / 16) + (kk & 3) * 2); };
      auto moff = [](int kk) { return (uint64_t)(kk * 16 * 128 / 16); };
      // S'^T / dP'^T: accumulated from the first k-step onto the pre-filled region
      auto issue_sp = [&](uint64_t ad0, uint64_t bd0, uint32_t col) {
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) tc_mma_ss_w(tmem + col, ad0 + koff(kk), bd0 + koff(kk), idSP, 1u);
      };
      // dV (a_col = P^T) or dK (a_col = dS^T) += A * B over query k-steps [k0, k0+2);
      // B = dO or Q [query rows][d], MN-major
      auto issue_kv = [&](uint32_t a_col, uint64_t bd0, uint32_t d_col, bool acc, int k0) {
#pragma unroll
        for (int kk = k0; kk < k0 + 2; ++kk)
          tc_mma_ts(tmem + d_col, tmem + a_col + kk * 8, bd0 + moff(kk), idKV, (acc || kk > 0) ? 1u : 0u);
      };
      bool ok = true;
      if (warp == 1) {
        // ---- issuer X: dV(t) and dK(t), one query quarter at a time
        for (int t = 0; ok && t < T; ++t) {
          const int p = t & 1;
          const uint64_t qM = p ? qM1 : qM0;
          // dO(t) has landed (issuer Y waits for it too, but only before dP(t), which it
          // may issue after phase A(t) has already released P^T(t) here)
          if (!mbar_wait(&sm.do_full, t & 1, abort, P.status)) { ok = false; break; }
          for (int u = 0; u < 4; ++u) {
            if (!mbar_wait(&sm.pa_part[u], t & 1, abort, P.status)) { ok = false; break; }
            tc_fence_after();
            issue_kv(col_r(p), doM, COL_DV, t > 0, 2 * u);       // reads P^T(t) and dO(t)
          }
          if (!ok) break;
          tc_commit(&sm.do_empty);
          tc_commit(&sm.dv_done);  // issuer Y may write dQ(t) over P^T(t) in R[p]
          for (int u = 0; u < 4; ++u) {
            if (!mbar_wait(&sm.pb_part[u], t & 1, abort, P.status)) { ok = false; break; }
            tc_fence_after();
            issue_kv(col_r(p ^ 1), qM, COL_DK, t > 0, 2 * u);    // reads dS^T(t) and Q(t)
          }
          if (!ok) break;
          tc_commit(&sm.q_empty[p]);
          tc_commit(&sm.dk_done);  // R[p^1] free for the S'^T(t+1) pre-fill
        }
        tc_commit(&sm.kv_done);
      } else {
        // ---- issuer Y: S(0), dP(0), then per tile dQ(t), S(t+1), dP(t+1)
        ok = __all_sync(0xffffffffu, mbar_wait(&sm.kv_full, 0, abort, P.status)) && __all_sync(0xffffffffu, mbar_wait(&sm.q_full[0], 0, abort, P.status)) &&
             __all_sync(0xffffffffu, mbar_wait(&sm.s_init, 0, abort, P.status));
        if (ok) {
          tc_fence_after();
          issue_sp(kK, qK0, col_r(0));
          tc_commit_w(&sm.s_full);
          ok = __all_sync(0xffffffffu, mbar_wait(&sm.do_full, 0, abort, P.status)) && __all_sync(0xffffffffu, mbar_wait(&sm.dp_init, 0, abort, P.status));
          if (ok) {
            tc_fence_after();
            issue_sp(vK, doK, col_r(1));
            tc_commit_w(&sm.dp_full);
            tc_commit_w(&sm.do_empty);  // with issuer X's arrival after dV(0)
          }
        }
        for (int t = 0; ok && t < T; ++t) {
          const int p = t & 1;
          // dQ(t) = dS K into R[p]: dS^T(t) complete in smem, phase B(t) and dV(t)
          // (issuer X) done reading P^T(t) there
          if (!__all_sync(0xffffffffu, mbar_wait(&sm.pb_part[3], t & 1, abort, P.status)) ||
              !__all_sync(0xffffffffu, mbar_wait(&sm.dv_done, t & 1, abort, P.status))) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc_mma_ss_w(tmem + col_r(p), dsM + moff(kk), kM + moff(kk), idQ, kk > 0 ? 1u : 0u);
          tc_commit_w(&sm.dq_full);
          if (t + 1 < T) {
            // S^T(t+1) into R[p^1]: s_init follows dK(t) (issuer X) having read dS^T(t) there
            if (!__all_sync(0xffffffffu, mbar_wait(&sm.q_full[p ^ 1], ((t + 1) >> 1) & 1, abort, P.status)) ||
                !__all_sync(0xffffffffu, mbar_wait(&sm.s_init, (t + 1) & 1, abort, P.status))) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_sp(kK, p ? qK0 : qK1, col_r(p ^ 1));
            tc_commit_w(&sm.s_full);
            // dP^T(t+1) into R[p]: dQ(t) read out and R[p] pre-filled, dO(t+1) loaded
            if (!__all_sync(0xffffffffu, mbar_wait(&sm.dp_init, (t + 1) & 1, abort, P.status)) ||
                !__all_sync(0xffffffffu, mbar_wait(&sm.do_full, (t + 1) & 1, abort, P.status))) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_sp(vK, doK, col_r(p));
            tc_commit_w(&sm.dp_full);
            tc_commit_w(&sm.do_empty);  // with issuer X's arrival after dV(t+1)
          }
        }
      }
      // every MMA either issuer started completes before TMEM / smem are released
      if (warp == 1)
        tc_commit(&sm.drain);
      else
        tc_commit_w(&sm.drain);
      mbar_drain(&sm.drain, 0);
    }
  } else if (warp < 6) {
    // ------------------------------------------------------------ softmax
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;    // TMEM lane
    const int kr = n0 + row;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const float c2 = P.scale_log2;
    uint8_t* dsrow = reinterpret_cast<uint8_t*>(sm.ds) + row * 128;
    bool ok = true;
    for (int t = 0; t < T; ++t) {
      const int p = t & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full, t & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      // Eight chunks of 16 query columns per phase; the TMEM loads of chunk c+1 are in
      // flight while chunk c is computed.  Chunk c packs into columns [8c, 8c+8), which
      // hold data this thread has already read.  Each quarter is published with its
      // stores landed, so the MMAs of that quarter may start.
      const uint64_t c2x2 = f2pack(c2, c2);
      // ---- phase A: P^T = exp2(c2 S'^T), S'^T already carrying -lse2/c2 (or -inf
      // where masked), packed bf16 into R[p]
      {
        uint32_t sbuf[2][16];
        auto chunk_a = [&](int c, uint32_t* sr, uint32_t* sn) {
          tmem_ld_wait();
          if (c + 1 < 8) tmem_ld16(tl + col_r(p) + 16 * (c + 1), sn);
          float x[16], pv[16];
#pragma unroll
          for (int e = 0; e < 16; e += 2)
            f2unpack(fmul2(f2pack(__uint_as_float(sr[e]), __uint_as_float(sr[e + 1])), c2x2), x[e], x[e + 1]);
#pragma unroll
          for (int e = 0; e < 16; ++e) pv[e] = ex2_approx(x[e]);
          uint32_t pp[8];
#pragma unroll
          for (int e = 0; e < 16; e += 2) pp[e >> 1] = cvt_bf16x2(pv[e], pv[e + 1]);
          tmem_st8(tl + col_r(p) + 8 * c, pp);
        };
        tmem_ld16(tl + col_r(p), sbuf[0]);
#pragma unroll
        for (int c = 0; c < 8; c += 2) {
          chunk_a(c, sbuf[0], sbuf[1]);
          chunk_a(c + 1, sbuf[1], sbuf[0]);
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&sm.pa_part[c >> 1]);
        }
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.dp_full, t & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      // ---- phase B: dS^T = P^T dP'^T (P^T as packed bf16 from R[p], dP'^T already
      // carrying -delta), packed bf16 into R[p^1] and into shared memory for dQ(t)
      {
        uint32_t dbuf[2][16], pbuf[2][8];
        auto chunk_b = [&](int c, uint32_t* dr, uint32_t* pr, uint32_t* dn, uint32_t* pn) {
          tmem_ld_wait();
          if (c + 1 < 8) {
            tmem_ld16(tl + col_r(p ^ 1) + 16 * (c + 1), dn);
            tmem_ld8(tl + col_r(p) + 8 * (c + 1), pn);
          }
          // dS pair = bf16(P pair) * bf16(dP' pair) in one packed bf16 multiply: one more
          // rounding (of dP', relative 2^-9) than an fp32 product rounded to bf16
          uint32_t dd[8];
#pragma unroll
          for (int e = 0; e < 16; e += 2)
            dd[e >> 1] = mul_bf16x2(pr[e >> 1], cvt_bf16x2(__uint_as_float(dr[e]), __uint_as_float(dr[e + 1])));
          tmem_st8(tl + col_r(p ^ 1) + 8 * c, dd);
          // dS^T -> shared memory for dQ(t): block c/4, 16-byte chunks 2(c%4), 2(c%4)+1
          uint8_t* blk = dsrow + (c >> 2) * (BK * 128);
#pragma unroll
          for (int k = 0; k < 2; ++k)
            *reinterpret_cast<uint4*>(blk + (((2 * (c & 3) + k) ^ (row & 7)) << 4)) =
                make_uint4(dd[4 * k], dd[4 * k + 1], dd[4 * k + 2], dd[4 * k + 3]);
        };
        tmem_ld16(tl + col_r(p ^ 1), dbuf[0]);
        tmem_ld8(tl + col_r(p), pbuf[0]);
#pragma unroll
        for (int c = 0; c < 8; c += 2) {
          chunk_b(c, dbuf[0], pbuf[0], dbuf[1], pbuf[1]);
          chunk_b(c + 1, dbuf[1], pbuf[1], dbuf[0], pbuf[0]);
          // after the last quarter the whole dS^T tile is also in shared memory for dQ(t)
          if (c == 6) fence_async_smem();
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&sm.pb_part[c >> 1]);
        }
      }
    }
    // epilogue: this key row of dV, then of dK (scaled); with head chunks, into this
    // chunk's fp32 workspace slice instead
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.kv_done, 0, abort, P.status))) {
      tc_fence_after();
      const long long orow = (((long long)b * G.nL + (long long)kr * G.rs + sk) * G.Hkv + kvh) * DH;
      const size_t half = (size_t)G.B * G.q_ns * G.Lv * G.Hkv * DH;
      const long long wrow = ((((long long)b * G.q_ns + s) * G.Lv + kr) * G.Hkv + kvh) * DH;
#pragma unroll 1
      for (int c = 0; c < 2 * DH / 32; ++c) {
        const int which = c >= DH / 32;
        const float mul = which ? P.scale : 1.f;
        bf16* dst = (which ? P.dk : P.dv) + orow + (c % (DH / 32)) * 32;
        const uint32_t col = (which ? COL_DK : COL_DV) + (c % (DH / 32)) * 32;
        uint32_t o[32];
        tmem_ld32(tl + col, o);
        tmem_ld_wait();
        if (HC > 1) {
          if (kr < G.Lv) {
            float* wdst = P.dkv + (2 * hc + which) * half + wrow + (c % (DH / 32)) * 32;
#pragma unroll
            for (int e = 0; e < 32; e += 4)
              *reinterpret_cast<float4*>(wdst + e) =
                  make_float4(__uint_as_float(o[e]) * mul, __uint_as_float(o[e + 1]) * mul,
                              __uint_as_float(o[e + 2]) * mul, __uint_as_float(o[e + 3]) * mul);
          }
        } else if (kr < G.Lv) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = cvt_bf16x2(__uint_as_float(o[e + 0]) * mul, __uint_as_float(o[e + 1]) * mul);
            w.y = cvt_bf16x2(__uint_as_float(o[e + 2]) * mul, __uint_as_float(o[e + 3]) * mul);
            w.z = cvt_bf16x2(__uint_as_float(o[e + 4]) * mul, __uint_as_float(o[e + 5]) * mul);
            w.w = cvt_bf16x2(__uint_as_float(o[e + 6]) * mul, __uint_as_float(o[e + 7]) * mul);
            *reinterpret_cast<uint4*>(dst + e) = w;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ dQ flush, pre-fills
    // Pre-fill, columns [64*dhalf, +64) of a region, this warp's TMEM lanes (key rows):
    // -lse2/c2 of the next query tile before its S^T MMA, with -inf where the key row
    // does not see the query (the mask: exp2 then gives P = 0 whatever the MMA adds);
    // -delta before its dP^T MMA.
    // dQ: TMEM lane = query row q0 + 32*q4 + lane; this warp's 64 head-dim columns
    // leave TMEM first, then two 32-column rounds are staged (128-byte swizzle) and
    // added into the fp32 accumulator by TMA reduce.
    const int dhalf = (warp - 6) >> 2;
    const int q4 = warp & 3;
    constexpr int DQC = DH / 2;  // dQ columns read out and reduced by this warp
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    float* stage = sm.dqs[warp - 6];
    const float inv_c2 = 1.f / P.scale_log2;
    const int kr = n0 + q4 * 32 + lane;  // key row of this thread's TMEM lane
    // Pre-fill values for this warp's 64 columns are read from shared memory and
    // masked before the region is free (those loads would otherwise queue behind the
    // MMAs' operand reads on the critical path); only the TMEM stores follow the wait.
    // S'^T of the query tile starting at qm: -lse2/c2, -inf where not visible.
    auto s_values = [&](uint32_t* w, const float* src, int qm) {
      const float4* s4 = reinterpret_cast<const float4*>(src + 64 * dhalf);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float4 x = s4[i];
        w[4 * i] = __float_as_uint(x.x * inv_c2);
        w[4 * i + 1] = __float_as_uint(x.y * inv_c2);
        w[4 * i + 2] = __float_as_uint(x.z * inv_c2);
        w[4 * i + 3] = __float_as_uint(x.w * inv_c2);
      }
      // masked where a pair can fall outside: the diagonal band, (LOCAL) the last query's
      // window edge at or above the tile's first key, ragged tiles
      const bool win_edge =
          WIN ? (qm + BQ - 1) * G.qstep + G.qoff - G.window >= n0 : G.window > 0;
      if ((qm * G.qstep + G.qoff < n0 + BK) || win_edge || (n0 + BK > G.Lv) || (qm + BQ > G.Lq) || G.smod > 1) {
        // key row kr sees the queries q in [vis_lo, vis_hi): q*qstep + qoff >= kr
        // (causal), q < Lq, and for LOCAL q*qstep + qoff < kr + window (an empty range
        // when kr itself is past Lv)
        const int vis_lo = kr <= G.qoff ? 0 : (kr - G.qoff + G.qstep - 1) / G.qstep;
        int vis_hi = G.Lq;
        if (G.window > 0) {
          const int e = kr + G.window - G.qoff;  // q*qstep < e
          vis_hi = min(vis_hi, e <= 0 ? 0 : (e + G.qstep - 1) / G.qstep);
        }
        if (kr >= G.Lv) vis_hi = 0;
        const int qb = qm + 64 * dhalf;
#pragma unroll
        for (int i = 0; i < 64; ++i)
          if (qb + i < vis_lo || qb + i >= vis_hi) w[i] = __float_as_uint(-INFINITY);
        if (G.smod > 1) {  // the naive intra-stream schedule (CROSS rows: query row = key row)
          int k = (qb - kr) % G.smod;  // (query row - key row) mod smod, stepped along the columns
          if (k < 0) k += G.smod;
#pragma unroll
          for (int i = 0; i < 64; ++i) {
            if (k != 0) w[i] = __float_as_uint(-INFINITY);
            k = k + 1 == G.smod ? 0 : k + 1;
          }
        }
      }
    };
    auto d_values = [&](uint32_t* w, const float* src) {  // dP'^T: -delta
      const uint4* s4 = reinterpret_cast<const uint4*>(src + 64 * dhalf);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const uint4 x = s4[i];
        w[4 * i] = x.x;
        w[4 * i + 1] = x.y;
        w[4 * i + 2] = x.z;
        w[4 * i + 3] = x.w;
      }
    };
    auto store64 = [&](uint32_t col, const uint32_t* w) {
      tmem_st32(tl + col + 64 * dhalf, w);
      tmem_st32(tl + col + 64 * dhalf + 32, w + 32);
    };
    auto publish = [&](uint64_t* bar) {  // stores landed, then signal the MMA thread
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(bar);
    };
    // tile 0: S'^T(0) region R0, dP'^T(0) region R1
    bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.q_full[0], 0, abort, P.status));
    if (ok) {
      uint32_t w[64];
      s_values(w, sm.nlse2[0], i_lo * BQ);
      store64(col_r(0), w);
      publish(&sm.s_init);
      d_values(w, sm.ndelta[0]);
      store64(col_r(1), w);
      publish(&sm.dp_init);
    }
    for (int t = 0; ok && t < T; ++t) {
      const int p = t & 1;
      const int h = h_base + t / nq, q0 = (i_lo + t % nq) * BQ;
      const bool next = t + 1 < T;
      if (next) {
        // R[p^1] for S'^T(t+1): row terms of tile t+1 loaded; dK(t) has read dS^T(t) there
        uint32_t w[64];
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.q_full[p ^ 1], ((t + 1) >> 1) & 1, abort, P.status))) {
          ok = false;
          break;
        }
        s_values(w, sm.nlse2[p ^ 1], (i_lo + (t + 1) % nq) * BQ);
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.dk_done, t & 1, abort, P.status))) {
          ok = false;
          break;
        }
        tc_fence_after();
        store64(col_r(p ^ 1), w);
        publish(&sm.s_init);
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.dq_full, t & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      // this warp's DH/2 dQ columns [DQC*dhalf, +DQC)
      uint32_t v[DQC];
#pragma unroll
      for (int r2 = 0; r2 < DQC / 32; ++r2) tmem_ld32(tl + col_r(p) + DQC * dhalf + 32 * r2, v + 32 * r2);
      tmem_ld_wait();
      if constexpr (DH == 64) {
        // the pre-fill below covers query columns [64*dhalf, +64) of R[p], which at DH = 64
        // hold the other dQ warp's dQ columns: both warps of this quadrant read theirs first
        mbar_arrive(&sm.dq_read[q4]);
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.dq_read[q4], t & 1, abort, P.status))) {
          ok = false;
          break;
        }
      }
      if (next) {
        // dQ(t) is out of R[p]: pre-fill it for dP'^T(t+1), 16 columns at a time
#pragma unroll 1
        for (int h4 = 0; h4 < 4; ++h4) {
          const uint4* s4 = reinterpret_cast<const uint4*>(sm.ndelta[p ^ 1] + 64 * dhalf + 16 * h4);
          uint32_t w[16];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const uint4 x = s4[i];
            w[4 * i] = x.x;
            w[4 * i + 1] = x.y;
            w[4 * i + 2] = x.z;
            w[4 * i + 3] = x.w;
          }
          tmem_st16(tl + col_r(p) + 64 * dhalf + 16 * h4, w);
        }
        publish(&sm.dp_init);
      }
#pragma unroll
      for (int r2 = 0; r2 < DQC / 32; ++r2) {
        // the previous reduce from this warp's buffer must have read it
        if (lane == 0) bulk_wait_read0();
        __syncwarp();
        uint8_t* srow = reinterpret_cast<uint8_t*>(stage) + lane * 128;
#pragma unroll
        for (int c = 0; c < 8; ++c)
          *reinterpret_cast<uint4*>(srow + ((c ^ (lane & 7)) << 4)) =
              make_uint4(v[32 * r2 + 4 * c], v[32 * r2 + 4 * c + 1], v[32 * r2 + 4 * c + 2], v[32 * r2 + 4 * c + 3]);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_reduce_add_5d(&P.tm_dq, stage, DQC * dhalf + 32 * r2, h, s, q0 + q4 * 32, b);
          bulk_commit();
        }
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
// Head chunks: dv / dk rows (bf16) from the chunks' fp32 partial sums, added in chunk
// order, 8 columns per thread.
template <int DH>
__global__ void __launch_bounds__(256) dkv_finalize_kernel(const float* __restrict__ dkv, bf16* __restrict__ dk,
                                                           bf16* __restrict__ dv, SfaGeom g, int chunks) {
  const long long n8 = (long long)g.B * g.q_ns * g.Lv * g.Hkv * (DH / 8);
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n8) return;
  const int c8 = (int)(i % (DH / 8));
  long long r = i / (DH / 8);
  const int kvh = (int)(r % g.Hkv);
  r /= g.Hkv;
  const int kr = (int)(r % g.Lv);
  r /= g.Lv;
  const int s = (int)(r % g.q_ns), b = (int)(r / g.q_ns);
  const long long orow = (((long long)b * g.nL + (long long)kr * g.rs + s + g.kv_s0) * g.Hkv + kvh) * DH + c8 * 8;
  const size_t half = (size_t)n8 * 8;
#pragma unroll
  for (int which = 0; which < 2; ++which) {
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f), y = x;
    for (int hc = 0; hc < chunks; ++hc) {
      const float4* src = reinterpret_cast<const float4*>(dkv + (2 * hc + which) * half + i * 8);
      const float4 a = src[0], e = src[1];
      x.x += a.x; x.y += a.y; x.z += a.z; x.w += a.w;
      y.x += e.x; y.y += e.y; y.z += e.z; y.w += e.w;
    }
    uint4 w;
    w.x = cvt_bf16x2(x.x, x.y);
    w.y = cvt_bf16x2(x.z, x.w);
    w.z = cvt_bf16x2(y.x, y.y);
    w.w = cvt_bf16x2(y.z, y.w);
    *reinterpret_cast<uint4*>((which ? dk : dv) + orow) = w;
  }
}
}  // namespace tcbwd

template <int DH>
static cudaError_t bwd_tc_impl(tcbwd::Params& p, const SfaGeom& g, cudaStream_t st) {
  using namespace tcbwd;
  const size_t nkv = bwd_dkv_slice(g, DH);
  if (p.hchunks > 1 && p.dkv == nullptr) return cudaErrorInvalidValue;
  const int smem = smem_bytes<DH>();
  auto kern = g.window > 0 ? bwd_kernel<DH, true> : bwd_kernel<DH, false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const unsigned grid = (unsigned)((g.Lv + BK - 1) / BK) * (unsigned)(p.hchunks * g.Hkv * g.q_ns * g.B);
  kern<<<grid, NTHREADS, smem, st>>>(p);
  e = cudaGetLastError();
  if (e != cudaSuccess || p.hchunks == 1) return e;
  const long long n8 = (long long)nkv / 8;
  dkv_finalize_kernel<DH><<<(unsigned)((n8 + 255) / 256), 256, 0, st>>>(p.dkv, p.dk, p.dv, g, p.hchunks);
  return cudaGetLastError();
}

// Dh: 64 or 128.
cudaError_t launch_sfa_bwd_main_tc(const void* q, const void* k, const void* v, const void* dout, void* dk,
                                   void* dv, const float* lse2_ws, const float* delta_ws, float* dq_ws,
                                   float* dkv_ws, const SfaGeom& g, int Dh, float scale, int32_t* status,
                                   cudaStream_t st) {
  using namespace tcbwd;
  Params p;
  const int DH = Dh;
  const SfaGeom gq = query_geom(g);
  if (!make_rows_tmap(&p.tm_q, q, gq, g.Hq, DH, BQ) || !make_rows_tmap(&p.tm_do, dout, gq, g.Hq, DH, BQ) ||
      !make_rows_tmap(&p.tm_k, k, g, g.Hkv, DH, BK) || !make_rows_tmap(&p.tm_v, v, g, g.Hkv, DH, BK) ||
      !make_rows_tmap(&p.tm_dq, dq_ws, gq, g.Hq, DH, 32, 4, 32, true))
    return cudaErrorInvalidValue;
  p.lse2 = lse2_ws;
  p.delta = delta_ws;
  p.dk = (bf16*)dk;
  p.dv = (bf16*)dv;
  p.hchunks = bwd_head_chunks(g, Dh);
  p.dkv = dkv_ws;
  p.g = g;
  p.scale = scale;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.status = status;
  return Dh == 64 ? bwd_tc_impl<64>(p, g, st) : bwd_tc_impl<128>(p, g, st);
}

}  // namespace hdsfa
