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

// One warp takes the 8 consecutive rows r0..r0+7 of one (b, head h, stream s) problem
// (positions p = r*ns + s): each row's O and dO are DH*2 contiguous bytes (DH/8 lanes,
// 16 bytes each, 32*8/DH rows per load instruction, every load issued before the
// first dot product); the rows' LSE values lie within 8*ns floats and their row terms
// are 8 consecutive floats of the stream-major arrays, so lanes 0..7 load the LSE
// together and, after the dot products are gathered to them, store both row terms
// as one 32-byte run each.  Warps are ordered head-fastest, so a CTA's eight warps
// read the eight heads' rows that share positions (adjacent in memory).  With ZERO the
// warp then zeroes its rows of the fp32 dQ accumulator.
template <int DH, bool ZERO>
__global__ void __launch_bounds__(256) sfa_bwd_prep_kernel(const bf16* __restrict__ o,
                                                           const bf16* __restrict__ dout,
                                                           const float* __restrict__ lse,
                                                           float* __restrict__ lse2_t,
                                                           float* __restrict__ delta_t,
                                                           float* __restrict__ dq_acc, SfaGeom g) {
  constexpr int LPR = DH / 8;      // lanes per row
  constexpr int RPG = 32 / LPR;    // rows per load instruction
  constexpr int RPW = 8;           // rows per warp
  constexpr int ITER = RPW / RPG;  // load instructions per tensor
  const int lane = threadIdx.x & 31, sub = lane / LPR, l = lane % LPR;
  // warp -> (b, s, r-block, h), h fastest; 32-bit index math (the host caps B*nL*Hq
  // below 2^30)
  const unsigned Hq = (unsigned)g.Hq, ns = (unsigned)g.ns, Lv = (unsigned)g.Lv, nL = (unsigned)g.nL;
  const unsigned nrb = (Lv + RPW - 1) / RPW;
  const unsigned w = (unsigned)(((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if ((long long)w >= (long long)g.B * ns * nrb * Hq) return;
  const unsigned h = w % Hq, w1 = w / Hq, rb = w1 % nrb, w2 = w1 / nrb, s = w2 % ns, b = w2 / ns;
  const unsigned r0 = rb * RPW;
  uint4 xo[ITER], xd[ITER];
#pragma unroll
  for (int i = 0; i < ITER; ++i) {
    const unsigned r = r0 + i * RPG + sub;
    xo[i] = make_uint4(0, 0, 0, 0);
    xd[i] = make_uint4(0, 0, 0, 0);
    if (r < Lv) {
      const long long row = ((long long)b * nL + (long long)r * ns + s) * Hq + h;
      xo[i] = *reinterpret_cast<const uint4*>(o + row * DH + l * 8);
      xd[i] = *reinterpret_cast<const uint4*>(dout + row * DH + l * 8);
    }
  }
  const long long bh = (long long)b * Hq + h;
  const bool mine = lane < RPW && r0 + lane < Lv;  // lane j: row r0 + j's LSE and row terms
  const float lv = mine ? lse[bh * nL + (long long)(r0 + lane) * ns + s] : 0.f;
  float acc[ITER];
#pragma unroll
  for (int i = 0; i < ITER; ++i) {
    const bf16* xa = reinterpret_cast<const bf16*>(&xo[i]);
    const bf16* ya = reinterpret_cast<const bf16*>(&xd[i]);
    float a = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) a += __bfloat162float(xa[e]) * __bfloat162float(ya[e]);
#pragma unroll
    for (int off = LPR / 2; off; off >>= 1) a += __shfl_xor_sync(0xffffffffu, a, off);
    acc[i] = a;  // row r0 + i*RPG + sub, in every lane of its group
  }
  float dl = 0.f;  // lane j < 8: the dot product of row r0 + j
#pragma unroll
  for (int i = 0; i < ITER; ++i)
#pragma unroll
    for (int sb = 0; sb < RPG; ++sb) {
      const float v = __shfl_sync(0xffffffffu, acc[i], sb * LPR);
      if (lane == i * RPG + sb) dl = v;
    }
  if (mine) {
    const long long t = (bh * ns + s) * row_terms_pitch(g.Lv) + r0 + lane;
    delta_t[t] = -dl;
    lse2_t[t] = -lv * 1.4426950408889634f;
  }
  if (ZERO) {  // this warp's rows of the dQ accumulator, DH contiguous floats each
#pragma unroll
    for (int j = 0; j < RPW; ++j) {
      const unsigned r = r0 + j;
      if (r < Lv) {
        float4* dz = reinterpret_cast<float4*>(dq_acc + (((long long)b * nL + (long long)r * ns + s) * Hq + h) * DH);
        for (int c = lane; c < DH / 4; c += 32) dz[c] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
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
  const long long warps = (long long)g.B * g.ns * ((g.Lv + 7) / 8) * g.Hq;  // 8 rows of one problem each
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
