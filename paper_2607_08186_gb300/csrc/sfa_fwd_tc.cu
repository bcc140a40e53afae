// Stream-Factorized Attention forward on the sm_103a tensor cores.
//
// One CTA computes a 128-row query tile of one virtual causal problem (SfaGeom):
// in WITHIN mode the problem is one stream (rows p = t*n + s, Eq. 4), so the tile
// visits only that stream's key tiles; CROSS is causal over all nL positions
// (Fig. 2a); LOCAL adds the window (Fig. 2b).  Key tiles past the diagonal (or
// before the window) are skipped; tiles straddling a mask edge are masked in
// registers.
//
// Roles (192 threads):
//   warp 0      TMA producer: Q once, then K/V tiles into a 2-stage ring; owns TMEM.
//   warp 1      MMA issuer (one thread): S = Q K^T into one of two TMEM S buffers,
//               O += P V into the TMEM O accumulator.
//   warps 2..5  softmax: one thread per query row (its TMEM lane); online softmax
//               in fp32 with exp2, P (bf16) to shared memory, O rescaled in TMEM
//               only when the running max grows by more than 2^8, epilogue.
// Shared-memory tiles use the 128-byte swizzle written by TMA; P is written by
// the softmax threads in the same layout.  Every mbarrier wait is bounded.
#include <cudaTypedefs.h>

#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace tcfwd {
constexpr int BM = 128, BN = 128, NST = 2, NTHREADS = 192;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: P stays <= 256 between rescales

template <int DH>
struct Smem {
  bf16 q[BM * DH];        // DH/64 swizzle blocks of [BM][64]
  bf16 k[NST][BN * DH];
  bf16 v[NST][BN * DH];
  bf16 p[BM * BN];        // 2 swizzle blocks of [BM][64]
  uint64_t q_full, kv_full[NST], kv_empty[NST], s_full[2], s_free[2], p_full, o_done, drain;
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

HD_DEVINLINE bool visible(int r, int c, int Lv, int window) {
  return c <= r && c < Lv && (window <= 0 || r - c < window);
}

template <int DH>
__global__ void __launch_bounds__(NTHREADS, 1) fwd_kernel(const __grid_constant__ Params P) {
  extern __shared__ uint8_t smem_raw[];
  Smem<DH>& sm = *reinterpret_cast<Smem<DH>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SfaGeom& G = P.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ntile = (G.Lv + BM - 1) / BM;
  const int mt = ntile - 1 - (int)blockIdx.x;  // longest rows first
  const int m0 = mt * BM;
  const int h = blockIdx.y / G.ns, s = blockIdx.y % G.ns, b = blockIdx.z;
  const int kvh = h / (G.Hq / G.Hkv);
  const int n_lo = G.window > 0 ? max(0, m0 - G.window + 1) / BN : 0;
  const int n_hi = min(mt, (G.Lv - 1) / BN);
  const int nkv = n_hi - n_lo + 1;

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    for (int i = 0; i < NST; ++i) {
      mbar_init(&sm.kv_full[i], 1);
      mbar_init(&sm.kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.s_full[i], 1);
      mbar_init(&sm.s_free[i], 128);
    }
    mbar_init(&sm.p_full, 128);
    mbar_init(&sm.o_done, 1);
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
      for (int c = 0; c < DH / 64; ++c)
        tma_load_5d(sm.q + c * BM * 64, &P.tm_q, &sm.q_full, c * 64, h, s, m0, b);
      int issued = 0;
      for (int it = 0; it < nkv; ++it) {
        const int st = it % NST;
        if (it >= NST && !mbar_wait(&sm.kv_empty[st], ((it / NST) - 1) & 1, abort, P.status)) break;
        const int r0 = (n_lo + it) * BN;
        mbar_arrive_expect_tx(&sm.kv_full[st], 2 * BN * DH * 2);
        for (int c = 0; c < DH / 64; ++c) {
          tma_load_5d(sm.k[st] + c * BN * 64, &P.tm_k, &sm.kv_full[st], c * 64, kvh, s, r0, b);
          tma_load_5d(sm.v[st] + c * BN * 64, &P.tm_v, &sm.kv_full[st], c * 64, kvh, s, r0, b);
        }
        ++issued;
      }
      // let every copy this thread started land before the CTA can exit
      mbar_drain(&sm.q_full, 0);
      for (int it = max(0, issued - NST); it < issued; ++it)
        mbar_drain(&sm.kv_full[it % NST], (it / NST) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(BM, BN, 0, 0);  // S[q][kv] = Q K^T, both K-major
      constexpr uint32_t idO = idesc_bf16(BM, DH, 0, 1);  // O[q][d] += P V, V MN-major
      const uint32_t qa = smem_u32(sm.q), pa = smem_u32(sm.p);
      bool ok = mbar_wait(&sm.q_full, 0, abort, P.status);
      auto issue_pv = [&](int jt) -> bool {
        const int pst = jt % NST;
        if (!mbar_wait(&sm.p_full, jt & 1, abort, P.status)) return false;
        tc_fence_after();
        const uint32_t va = smem_u32(sm.v[pst]);
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(pa + (kk >> 2) * (BM * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc_sw128(va + kk * 16 * 128, BN * 128, 1024);
          tc_mma_ss(tmem + 256, ad, bd, idO, (jt > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&sm.o_done);
        tc_commit(&sm.kv_empty[pst]);
        return true;
      };
      for (int it = 0; ok && it < nkv; ++it) {
        const int st = it % NST, sb = it & 1;
        if (!mbar_wait(&sm.kv_full[st], (it / NST) & 1, abort, P.status)) break;
        if (it >= 2 && !mbar_wait(&sm.s_free[sb], ((it - 2) >> 1) & 1, abort, P.status)) break;
        tc_fence_after();
        const uint32_t ka = smem_u32(sm.k[st]);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(qa + (kk >> 2) * (BM * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc_sw128(ka + (kk >> 2) * (BN * 128) + (kk & 3) * 32, 16, 1024);
          tc_mma_ss(tmem + sb * 128, ad, bd, idS, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sm.s_full[sb]);
        if (it >= 1 && !issue_pv(it - 1)) break;
        if (it == nkv - 1) issue_pv(it);
      }
      // every MMA issued above has finished before TMEM / smem are released
      tc_commit(&sm.drain);
      mbar_drain(&sm.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax / epilogue
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int r = m0 + row;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    uint8_t* prow = reinterpret_cast<uint8_t*>(sm.p) + row * 128;
    for (int it = 0; it < nkv; ++it) {
      const int sb = it & 1;
      const int j = n_lo + it;
      // tcgen05.ld/st are warp-collective: every wait result is made warp-uniform
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[sb], (it >> 1) & 1, abort, P.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sraw[BN];
      float x[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_ld32(tl + sb * 128 + c * 32, sraw + c * 32);
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(&sm.s_free[sb]);
      const bool need_mask = (j == n_hi) || G.window > 0 || (j + 1) * BN > G.Lv;
      float tmax = -INFINITY;
#pragma unroll
      for (int i = 0; i < BN; ++i) {
        float y = __uint_as_float(sraw[i]) * P.scale_log2;
        if (need_mask && !visible(r, j * BN + i, G.Lv, G.window)) y = -INFINITY;
        x[i] = y;
        tmax = fmaxf(tmax, y);
      }
      const float m_new = fmaxf(m_run, tmax);
      const bool rescale = (m_run == -INFINITY) || (m_new > m_run + kRescaleThreshold);
      const float m_use = rescale ? m_new : m_run;
      const float m_sub = (m_use == -INFINITY) ? 0.f : m_use;
      float rsum = 0.f;
#pragma unroll
      for (int i = 0; i < BN; ++i) {
        x[i] = exp2f(x[i] - m_sub);
        rsum += x[i];
      }
      if (it > 0) {
        // PV of the previous tile must be done: it reads the P buffer and writes O
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.o_done, (it - 1) & 1, abort, P.status))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const bool mine = rescale && m_run != -INFINITY;
        if (__any_sync(0xffffffffu, mine)) {
          const float alpha = mine ? exp2f(m_run - m_use) : 1.f;
          l_run *= alpha;
#pragma unroll
          for (int c = 0; c < DH / 32; ++c) {
            uint32_t o[32];
            tmem_ld32(tl + 256 + c * 32, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st32(tl + 256 + c * 32, o);
          }
          tmem_st_wait();
        }
      }
      m_run = m_use;
      l_run += rsum;
      // P row -> shared memory, 128-byte swizzle, two 64-column blocks
#pragma unroll
      for (int c = 0; c < BN / 8; ++c) {
        uint4 w;
        w.x = pack_bf16(x[c * 8 + 0], x[c * 8 + 1]);
        w.y = pack_bf16(x[c * 8 + 2], x[c * 8 + 3]);
        w.z = pack_bf16(x[c * 8 + 4], x[c * 8 + 5]);
        w.w = pack_bf16(x[c * 8 + 6], x[c * 8 + 7]);
        const int blk = c >> 3, ch = (c & 7) ^ (row & 7);
        *reinterpret_cast<uint4*>(prow + blk * (BM * 128) + ch * 16) = w;
      }
      fence_async_smem();
      tc_fence_before();
      mbar_arrive(&sm.p_full);
    }
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.o_done, (nkv - 1) & 1, abort, P.status))) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      bf16* orow = P.o + (((long long)b * G.nL + (long long)r * G.rs + s) * G.Hq + h) * DH;
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tl + 256 + c * 32, o);
        tmem_ld_wait();
        if (r < G.Lv) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = pack_bf16(__uint_as_float(o[e + 0]) * inv, __uint_as_float(o[e + 1]) * inv);
            w.y = pack_bf16(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
            w.z = pack_bf16(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv);
            w.w = pack_bf16(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + c * 32 + e) = w;
          }
        }
      }
      if (r < G.Lv)
        P.lse[((long long)b * G.Hq + h) * G.nL + (long long)r * G.rs + s] = (m_run + log2f(l_run)) * kLn2;
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
static PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// Tensor map over a [B][nL][H][Dh] bf16 tensor seen as the 5-D array
// {Dh, H, ns, Lv, B} (innermost first): virtual row r of stream s is position
// r*rs + s.  Box = 64 head-dim elements (one 128-byte swizzle row) x box_rows rows.
bool make_rows_tmap(CUtensorMap* m, const void* base, const SfaGeom& g, int H, int Dh, int box_rows) {
  auto enc = tmap_encoder();
  if (enc == nullptr) return false;
  const cuuint64_t e = 2;
  cuuint64_t dims[5] = {(cuuint64_t)Dh, (cuuint64_t)H, (cuuint64_t)g.ns, (cuuint64_t)g.Lv, (cuuint64_t)g.B};
  cuuint64_t strides[4] = {Dh * e, (cuuint64_t)H * Dh * e, (cuuint64_t)g.rs * H * Dh * e,
                           (cuuint64_t)g.nL * H * Dh * e};
  cuuint32_t box[5] = {64, 1, 1, (cuuint32_t)box_rows, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int DH>
static cudaError_t tc_fwd_impl(tcfwd::Params& p, cudaStream_t st) {
  const int smem = (int)sizeof(tcfwd::Smem<DH>) + 1024;
  cudaError_t e = cudaFuncSetAttribute(tcfwd::fwd_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((p.g.Lv + tcfwd::BM - 1) / tcfwd::BM, p.g.Hq * p.g.ns, p.g.B);
  tcfwd::fwd_kernel<DH><<<grid, tcfwd::NTHREADS, smem, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_sfa_fwd_tc(const void* q, const void* k, const void* v, void* o, float* lse,
                              const SfaGeom& g, int Dh, float scale, int32_t* status, cudaStream_t st) {
  tcfwd::Params p;
  if (!make_rows_tmap(&p.tm_q, q, g, g.Hq, Dh, tcfwd::BM) || !make_rows_tmap(&p.tm_k, k, g, g.Hkv, Dh, tcfwd::BN) ||
      !make_rows_tmap(&p.tm_v, v, g, g.Hkv, Dh, tcfwd::BN))
    return cudaErrorInvalidValue;
  p.o = (bf16*)o;
  p.lse = lse;
  p.g = g;
  p.scale_log2 = scale * tcfwd::kLog2e;
  p.status = status;
  return Dh == 64 ? tc_fwd_impl<64>(p, st) : tc_fwd_impl<128>(p, st);
}

}  // namespace hdsfa
