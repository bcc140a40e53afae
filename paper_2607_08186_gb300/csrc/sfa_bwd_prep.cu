// Backward pre- and post-processing (bandwidth kernels).
//
// prep:     -delta[p] = -sum_d dO[p,d] * O[p,d] (fp32) and -lse2[p] = -lse[p] * log2(e),
//           both written stream-major, [B][Hq][ns][Lvp] with row r of stream s at
//           position p = r*ns + s and Lvp = row_terms_pitch(Lv), so one query tile
//           of any stream is contiguous floats (a single bulk copy).  Negated so the
//           backward folds them in with one add / fused multiply-add.  Rows in
//           [Lv, Lvp) get -lse2 = -inf and -delta = 0 (their P and dS vanish).
//           Also zeroes the fp32 dQ accumulator (or leaves that to clear, which needs
//           nothing from the forward and may run beside it on another stream).
// finalize: dq = bf16(scale * accumulator), round to nearest even.
#include "common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

// One warp takes RPW consecutive (b, p, h) rows: DH/8 lanes per row (16 bytes of O and
// of dO each), 32*8/DH rows side by side, ITER such row groups with every load issued
// before the first dot product, so each warp keeps several KB in flight.  With ZERO the
// warp then zeroes the same rows of the fp32 dQ accumulator (contiguous, 16-byte stores).
template <int DH, bool ZERO>
__global__ void __launch_bounds__(256) sfa_bwd_prep_kernel(const bf16* __restrict__ o,
                                                           const bf16* __restrict__ dout,
                                                           const float* __restrict__ lse,
                                                           float* __restrict__ lse2_t,
                                                           float* __restrict__ delta_t,
                                                           float* __restrict__ dq_acc, SfaGeom g) {
  constexpr int LPR = DH / 8;        // lanes per row
  constexpr int RPG = 32 / LPR;      // rows per group of the warp
  constexpr int ITER = 4;            // row groups per warp
  constexpr int RPW = RPG * ITER;    // rows per warp
  const int lane = threadIdx.x & 31, sub = lane / LPR, l = lane % LPR;
  // row indices fit 32 bits (the host caps B*nL*Hq below 2^30): 32-bit index math, whose
  // divisions cost a fraction of 64-bit ones
  const long long nrows = (long long)g.B * g.nL * g.Hq;
  const long long row0 = (((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * RPW;
  if (row0 >= nrows) return;
  uint4 xo[ITER], xd[ITER];
#pragma unroll
  for (int i = 0; i < ITER; ++i) {
    const long long row = row0 + i * RPG + sub;
    if (row < nrows) {
      xo[i] = *reinterpret_cast<const uint4*>(o + row * DH + l * 8);
      xd[i] = *reinterpret_cast<const uint4*>(dout + row * DH + l * 8);
    } else {
      xo[i] = make_uint4(0, 0, 0, 0);
      xd[i] = make_uint4(0, 0, 0, 0);
    }
  }
  const int Lvp = row_terms_pitch(g.Lv);
#pragma unroll
  for (int i = 0; i < ITER; ++i) {
    const bf16* xa = reinterpret_cast<const bf16*>(&xo[i]);
    const bf16* ya = reinterpret_cast<const bf16*>(&xd[i]);
    float acc = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc += __bfloat162float(xa[e]) * __bfloat162float(ya[e]);
#pragma unroll
    for (int off = LPR / 2; off; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    const long long row = row0 + i * RPG + sub;
    if (l == 0 && row < nrows) {
      const unsigned ur = (unsigned)row, Hq = (unsigned)g.Hq, nL = (unsigned)g.nL, ns = (unsigned)g.ns;
      const unsigned bp = ur / Hq, h = ur - bp * Hq, b = bp / nL, p = bp - b * nL;
      const unsigned r = p / ns, s = p - r * ns;
      const long long t = (((long long)b * Hq + h) * ns + s) * Lvp + r;
      delta_t[t] = -acc;
      lse2_t[t] = -lse[((long long)b * Hq + h) * nL + p] * 1.4426950408889634f;
    }
  }
  if (ZERO) {  // zero dQ accumulator rows [row0, row0 + RPW): RPW * DH floats, contiguous
    const long long nz = (min(nrows, row0 + RPW) - row0) * DH / 4;
    float4* dz = reinterpret_cast<float4*>(dq_acc + row0 * DH);
    for (long long c = lane; c < nz; c += 32) dz[c] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

// The fp32 dQ accumulator alone, zeroed with 16-byte stores (grid-stride).
__global__ void __launch_bounds__(256) sfa_bwd_clear_kernel(float4* __restrict__ acc, long long n4) {
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (long long)gridDim.x * blockDim.x)
    acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
}

__global__ void sfa_bwd_pad_kernel(float* __restrict__ lse2_t, float* __restrict__ delta_t, SfaGeom g) {
  const int Lvp = row_terms_pitch(g.Lv), pad = Lvp - g.Lv;
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)g.B * g.Hq * g.ns * pad) return;
  const long long t = (i / pad) * Lvp + g.Lv + i % pad;
  lse2_t[t] = -INFINITY;
  delta_t[t] = 0.f;
}

__global__ void __launch_bounds__(256) sfa_bwd_finalize_kernel(const float* __restrict__ dq_acc,
                                                               bf16* __restrict__ dq, long long n8,
                                                               float scale) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n8) return;
  const float4 a = reinterpret_cast<const float4*>(dq_acc)[2 * i];
  const float4 c = reinterpret_cast<const float4*>(dq_acc)[2 * i + 1];
  uint4 r;
  r.x = pack_bf16(a.x * scale, a.y * scale);
  r.y = pack_bf16(a.z * scale, a.w * scale);
  r.z = pack_bf16(c.x * scale, c.y * scale);
  r.w = pack_bf16(c.z * scale, c.w * scale);
  reinterpret_cast<uint4*>(dq)[i] = r;
}

cudaError_t launch_sfa_bwd_prep(const void* o, const void* dout, const float* lse, float* lse2_ws,
                                float* delta_ws, float* dq_ws, const SfaGeom& g, int Dh,
                                cudaStream_t st, bool zero) {
  const long long rows = (long long)g.B * g.nL * g.Hq;
  const long long rpw = 4LL * (32 / (Dh / 8));  // rows per warp (ITER * rows per group)
  const long long warps = (rows + rpw - 1) / rpw;
  const unsigned blocks = (unsigned)((warps * 32 + 255) / 256);
  const bf16 *ob = (const bf16*)o, *db = (const bf16*)dout;
  if (Dh == 256) {
    if (zero)
      sfa_bwd_prep_kernel<256, true><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
    else
      sfa_bwd_prep_kernel<256, false><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
  } else if (Dh == 64) {
    if (zero)
      sfa_bwd_prep_kernel<64, true><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
    else
      sfa_bwd_prep_kernel<64, false><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
  } else {
    if (zero)
      sfa_bwd_prep_kernel<128, true><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
    else
      sfa_bwd_prep_kernel<128, false><<<blocks, 256, 0, st>>>(ob, db, lse, lse2_ws, delta_ws, dq_ws, g);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int pad = row_terms_pitch(g.Lv) - g.Lv;
  if (pad > 0) {
    const long long n = (long long)g.B * g.Hq * g.ns * pad;
    sfa_bwd_pad_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(lse2_ws, delta_ws, g);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t launch_sfa_bwd_clear(float* dq_ws, const SfaGeom& g, int Dh, cudaStream_t st) {
  const long long n4 = (long long)g.B * g.nL * g.Hq * Dh / 4;
  long long blocks = (n4 + 255) / 256;
  if (blocks > 152LL * 16) blocks = 152LL * 16;
  sfa_bwd_clear_kernel<<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<float4*>(dq_ws), n4);
  return cudaGetLastError();
}

cudaError_t launch_sfa_bwd_finalize(void* dq, const float* dq_ws, const SfaGeom& g, int Dh,
                                    float scale, cudaStream_t st) {
  const long long n8 = (long long)g.B * g.nL * g.Hq * Dh / 8;
  sfa_bwd_finalize_kernel<<<(unsigned)((n8 + 255) / 256), 256, 0, st>>>(dq_ws, (bf16*)dq, n8, scale);
  return cudaGetLastError();
}

}  // namespace hdsfa
