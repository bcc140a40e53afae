// Decoding over the expanded KV cache (Sec. 3.2 "Inference Cost").  (Head dim 256 with up
// to 128 query rows per K/V head runs on the tcgen05 kernel further below.)
//
// Generation feeds each new token's n streams through the model together: its n
// positions p = (T-1)n + s (T = tokens in the cache, the new one included, whose K/V
// rows are already stored) attend, under the layer's mask, to the cached positions
// 0 .. Tn-1.  An intra-stream layer (Eq. 4) reads only stream s's cached rows for
// the queries of stream s; a cross-stream layer (Fig. 2a) reads all of them; a local
// one (Fig. 2b) the last `window` positions.  The cache has the training layout,
// [B][Lcap*n][Hkv][Dh] with position p at row p, so the forward pass's K/V tensors
// are a filled cache.
//
// Memory-bound: every step streams the visible cached rows of K and V once.  Per K/V
// head the queries are the n streams x (Hq/Hkv) heads of the group, 16 to 32 rows (a
// CTA takes up to 32; more rows take several CTAs): far below a tcgen05 tile, so the
// contractions use warp-level mma.sync m16n8k16 (bf16, fp32 accumulate), which keeps
// up with HBM.  Split over the cached positions (flash-decoding):
//   decode_kernel : CTA (split c, K/V head x row group, sequence): a 3-stage cp.async
//                   ring of 64-position K/V tiles; warp w takes keys [16w, 16w+16) of
//                   each tile with its own online softmax; the 4 warps merge in shared
//                   memory and write an unnormalised partial (O, running max, sum).
//                   At head dim 256 the tiles are 32 positions and the warps pair up:
//                   both warps of a pair compute the same scores and softmax for their
//                   16 keys, each accumulates O for one half of the head dim.
//   combine_kernel: merges a row's partials, writes O (bf16) and the natural-log LSE.
// Masking is per element (the new token's own positions, the stream condition of an
// intra-stream layer, the window); rows past the group's query count and positions
// past the sequence are zero-filled and masked.  A sequence whose length is outside
// [1, max_tokens] gets zero rows, LSE = -inf and HD_DEVBIT_INDEX.
#include <algorithm>

#include "decode_plan.cuh"
#include "tc_common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

// Defined in tmap.cu: the decoding step's queries [B][n][Hq][Dh] as {Dh, Hq, n, B}, box
// 64 columns x G heads x n streams.
bool make_qgroup_tmap(CUtensorMap* m, const void* base, int B, int n, int Hq, int Dh, int G);

namespace dec {
constexpr int NT = 128;      // 4 warps
constexpr int STAGES = 3;
// Head-dim split of the warps: at head dim 256 the four warps form two key groups x two
// halves of the head dim (a warp's O accumulator would not fit its registers whole);
// otherwise four key groups.  A stage holds 16 cached positions per key group.
template <int DH>
constexpr int dsplit() { return DH == 256 ? 2 : 1; }
template <int DH>
constexpr int ktile() { return 64 / dsplit<DH>(); }  // cached positions per pipeline stage
constexpr int RG = 32;       // query rows per CTA at most (two m16 tiles)
constexpr int kMaxSplit = 128;

struct DecodeArgs {
  const bf16* q;        // [B][n][Hq][Dh]
  const bf16* kc;       // [B][Lcap*n][Hkv][Dh]
  const bf16* vc;
  const int32_t* lens;  // [B] tokens in the cache
  bf16* o;              // [B][n][Hq][Dh]
  float* lse;           // [B][Hq][n] or null
  float* part_o;        // [B][Hkv][ngroups][nsplit][rg][Dh]
  float2* part_ml;      // [B][Hkv][ngroups][nsplit][rg]: (max in log2 units, sum)
  int32_t* status;
  int B, Lcap, maxT, n, Hq, Hkv, G, M, ngroups, nsplit, chunk, mode, window;
  int rg;               // query rows per row group (the partials' row pitch)
  float scale_log2;
};

// Programmatic dependent launch: both kernels are launched so that they may start
// while the kernel before them in the stream is finishing; each waits for that
// kernel's results before its first read of them, and the decode kernel lets the
// combine kernel launch at once, so the combine's launch and start overlap the
// decode's tail.  Without the launch attribute both are no-ops.
HD_DEVINLINE void grid_dep_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
HD_DEVINLINE void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

// Visible position range [lo, hi) of a sequence of T tokens (the new token's rows
// see nothing outside it; per-row conditions are applied per element).
HD_DEVINLINE void seq_range(const DecodeArgs& a, int T, int& lo, int& hi) {
  hi = T * a.n;
  lo = a.mode == SFA_LOCAL ? max(0, (T - 1) * a.n - a.window + 1) : 0;
}

template <int DH, int MT>
__global__ void __launch_bounds__(NT) decode_kernel(DecodeArgs a) {
  constexpr int DS = dsplit<DH>(), KT = ktile<DH>(), KW = 4 / DS, DC = DH / DS;  // DC: O columns per warp
  extern __shared__ __align__(128) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);  // [MT*16][DH]
  bf16* sK = sQ + MT * 16 * DH;                   // [STAGES][KT][DH]
  bf16* sV = sK + STAGES * KT * DH;               // [STAGES][KT][DH]
  constexpr int CPR = DH / 8;
  const int c = blockIdx.x, g = blockIdx.y / a.ngroups, rg = blockIdx.y % a.ngroups, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g4 = lane >> 2, t4 = lane & 3;
  const int kw = warp / DS, dw = warp % DS;  // key group and head-dim part of this warp
  const size_t pidx = (((size_t)b * a.Hkv + g) * a.ngroups + rg) * a.nsplit + c;
  float* po = a.part_o + pidx * RG * DH;
  float2* pml = a.part_ml + pidx * RG;
  grid_dep_wait();
  grid_dep_launch();
  const int T = a.lens[b];
  int k0 = 0, k1 = 0;
  if (T >= 1 && T <= a.maxT) {
    int lo, hi;
    seq_range(a, T, lo, hi);
    k0 = lo + c * a.chunk;
    k1 = min(k0 + a.chunk, hi);
  }
  if (k0 >= k1) {  // nothing of this sequence in this split: an empty partial
    for (int i = tid; i < RG; i += NT) pml[i] = make_float2(-INFINITY, 0.f);
    return;
  }
  const long long pbase = (long long)b * a.Lcap * a.n;  // cache row of position 0

  // query rows of the group -> smem (rows past M zero-filled)
  for (int i = tid; i < MT * 16 * CPR; i += NT) {
    const int rr = i / CPR, cc = i % CPR, r = rg * RG + rr;
    const bool ok = r < a.M;
    const int s = ok ? r / a.G : 0, h = g * a.G + (ok ? r % a.G : 0);
    cp_async_16(smem_u32(sQ + swz<DH>(rr, cc * 8)), a.q + (((long long)b * a.n + s) * a.Hq + h) * DH + cc * 8,
                ok);
  }
  auto load_stage = [&](int st, int kp0) {
    bf16* dK = sK + st * KT * DH;
    bf16* dV = sV + st * KT * DH;
    for (int i = tid; i < KT * CPR; i += NT) {
      const int rr = i / CPR, cc = i % CPR, p = kp0 + rr;
      const bool ok = p < k1;
      const long long off = ((pbase + (ok ? p : k0)) * a.Hkv + g) * DH + cc * 8;
      cp_async_16(smem_u32(dK + swz<DH>(rr, cc * 8)), a.kc + off, ok);
      cp_async_16(smem_u32(dV + swz<DH>(rr, cc * 8)), a.vc + off, ok);
    }
  };
  const int nsub = (k1 - k0 + KT - 1) / KT;
  load_stage(0, k0);
  cp_async_commit();
  if (nsub > 1) load_stage(1, k0 + KT);
  cp_async_commit();

  // this thread's query rows: (mt, half) -> local row mt*16 + g4 + 8*half
  int rs_[MT][2], rq[MT][2];  // stream of the row (-1: padding row) and its position
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      const int r = rg * RG + mt * 16 + g4 + 8 * hf;
      rs_[mt][hf] = r < a.M ? r / a.G : -1;
      rq[mt][hf] = (T - 1) * a.n + (r < a.M ? r / a.G : 0);
    }
  // stream of this thread's keys: when n divides 16 and k0, every warp's first key is a
  // multiple of n, so the stream of key kb + j*8 + 2*t4 + e is fixed per thread
  const bool kst_fixed = (16 % a.n) == 0 && (k0 % a.n) == 0;
  int kst0[2][2];
#pragma unroll
  for (int j = 0; j < 2; ++j)
#pragma unroll
    for (int e = 0; e < 2; ++e) kst0[j][e] = (j * 8 + 2 * t4 + e) % a.n;
  float mx[MT][2], ls[MT][2], oacc[MT][DC / 8][4];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    mx[mt][0] = mx[mt][1] = -INFINITY;
    ls[mt][0] = ls[mt][1] = 0.f;
#pragma unroll
    for (int i = 0; i < DC / 8; ++i) oacc[mt][i][0] = oacc[mt][i][1] = oacc[mt][i][2] = oacc[mt][i][3] = 0.f;
  }

  for (int it = 0; it < nsub; ++it) {
    cp_async_wait<STAGES - 2>();  // stage `it` has landed
    __syncthreads();              // ... for every thread, and stage it-1 is no longer read
    if (it + 2 < nsub) load_stage((it + 2) % STAGES, k0 + (it + 2) * KT);
    cp_async_commit();
    const bf16* cK = sK + (it % STAGES) * KT * DH;
    const bf16* cV = sV + (it % STAGES) * KT * DH;

    float sacc[MT][2][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
      for (int j = 0; j < 2; ++j) sacc[mt][j][0] = sacc[mt][j][1] = sacc[mt][j][2] = sacc[mt][j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
      uint32_t b0, b1, b2, b3;
      ldsm_x4(smem_u32(cK + swz<DH>(kw * 16 + (lane & 7) + (lane >> 4) * 8, kk * 16 + ((lane >> 3) & 1) * 8)),
              b0, b1, b2, b3);
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        uint32_t qa[4];
        ldsm_x4(smem_u32(sQ + swz<DH>(mt * 16 + (lane & 15), kk * 16 + (lane >> 4) * 8)), qa[0], qa[1], qa[2],
                qa[3]);
        mma_bf16_16816(sacc[mt][0], qa, b0, b1);
        mma_bf16_16816(sacc[mt][1], qa, b2, b3);
      }
    }
    // mask + online softmax (log2 domain)
    const int kb = k0 + it * KT + kw * 16;
    int kp[2][2], kst[2][2];
#pragma unroll
    for (int j = 0; j < 2; ++j)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        kp[j][e] = kb + j * 8 + 2 * t4 + e;
        kst[j][e] = a.mode != SFA_WITHIN ? 0 : (kst_fixed ? kst0[j][e] : kp[j][e] % a.n);
      }
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int j = 0; j < 2; ++j)
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const int hf = e4 >> 1, e = e4 & 1, p = kp[j][e], pq = rq[mt][hf];
          bool vis = rs_[mt][hf] >= 0 && p < k1 && p <= pq;
          if (a.mode == SFA_WITHIN) vis = vis && kst[j][e] == rs_[mt][hf];
          if (a.mode == SFA_LOCAL) vis = vis && p > pq - a.window;
          const float x = vis ? sacc[mt][j][e4] * a.scale_log2 : -INFINITY;
          sacc[mt][j][e4] = x;
          tmax[hf] = fmaxf(tmax[hf], x);
        }
      float corr[2], muse[2];
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        tmax[hf] = fmaxf(tmax[hf], __shfl_xor_sync(0xffffffffu, tmax[hf], 1));
        tmax[hf] = fmaxf(tmax[hf], __shfl_xor_sync(0xffffffffu, tmax[hf], 2));
        const float mnew = fmaxf(mx[mt][hf], tmax[hf]);
        muse[hf] = mnew == -INFINITY ? 0.f : mnew;
        corr[hf] = exp2f(mx[mt][hf] - muse[hf]);
        mx[mt][hf] = mnew;
        ls[mt][hf] *= corr[hf];
      }
#pragma unroll
      for (int j = 0; j < 2; ++j)
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const float p = exp2f(sacc[mt][j][e4] - muse[e4 >> 1]);
          sacc[mt][j][e4] = p;
          ls[mt][e4 >> 1] += p;
        }
#pragma unroll
      for (int i = 0; i < DC / 8; ++i) {
        oacc[mt][i][0] *= corr[0];
        oacc[mt][i][1] *= corr[0];
        oacc[mt][i][2] *= corr[1];
        oacc[mt][i][3] *= corr[1];
      }
    }
    // O += P V over this warp's 16 keys
    uint32_t pa[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      pa[mt][0] = pack_bf16(sacc[mt][0][0], sacc[mt][0][1]);
      pa[mt][1] = pack_bf16(sacc[mt][0][2], sacc[mt][0][3]);
      pa[mt][2] = pack_bf16(sacc[mt][1][0], sacc[mt][1][1]);
      pa[mt][3] = pack_bf16(sacc[mt][1][2], sacc[mt][1][3]);
    }
#pragma unroll
    for (int dp = 0; dp < DC / 16; ++dp) {
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(smem_u32(cV + swz<DH>(kw * 16 + (lane & 7) + ((lane >> 3) & 1) * 8,
                                      dw * DC + dp * 16 + (lane >> 4) * 8)),
                b0, b1, b2, b3);
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        mma_bf16_16816(oacc[mt][2 * dp], pa[mt], b0, b1);
        mma_bf16_16816(oacc[mt][2 * dp + 1], pa[mt], b2, b3);
      }
    }
  }

  // merge the 4 warps' partials in shared memory (the K/V ring is free now)
  cp_async_wait<0>();
  __syncthreads();
  // [KW][MT*16][DH]: key group kw's O, its head-dim parts side by side; then the key
  // groups' running max and sum (the DS warps of a key group hold the same ones)
  static_assert((KW * MT * 16 * DH + 2 * KW * MT * 16) * 4 <= 2 * STAGES * KT * DH * 2, "merge fits the ring");
  float* sO = reinterpret_cast<float*>(sK);
  float* sM = sO + KW * MT * 16 * DH;  // [KW][MT*16]
  float* sL = sM + KW * MT * 16;       // [KW][MT*16]
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      ls[mt][hf] += __shfl_xor_sync(0xffffffffu, ls[mt][hf], 1);
      ls[mt][hf] += __shfl_xor_sync(0xffffffffu, ls[mt][hf], 2);
      const int row = mt * 16 + g4 + 8 * hf;
      if (t4 == 0 && dw == 0) {
        sM[kw * MT * 16 + row] = mx[mt][hf];
        sL[kw * MT * 16 + row] = ls[mt][hf];
      }
    }
#pragma unroll
    for (int i = 0; i < DC / 8; ++i)
#pragma unroll
      for (int e4 = 0; e4 < 4; ++e4) {
        const int row = mt * 16 + g4 + 8 * (e4 >> 1), col = dw * DC + i * 8 + 2 * t4 + (e4 & 1);
        sO[(kw * MT * 16 + row) * DH + col] = oacc[mt][i][e4];
      }
  }
  __syncthreads();
  for (int idx = tid; idx < MT * 16 * DH; idx += NT) {
    const int row = idx / DH, col = idx % DH;
    float m = -INFINITY;
#pragma unroll
    for (int w = 0; w < KW; ++w) m = fmaxf(m, sM[w * MT * 16 + row]);
    float o = 0.f, l = 0.f;
    if (m != -INFINITY) {
#pragma unroll
      for (int w = 0; w < KW; ++w) {
        const float mw = sM[w * MT * 16 + row];
        const float f = mw == -INFINITY ? 0.f : exp2f(mw - m);
        o += f * sO[(w * MT * 16 + row) * DH + col];
        l += f * sL[w * MT * 16 + row];
      }
    }
    po[row * DH + col] = o;
    if (col == 0) pml[row] = make_float2(m, l);
  }
}

// CTA (K/V head x row group, sequence, 8-column slice x block of 8 rows); one warp per
// query row, its lanes over the splits: the row's max and sum by warp reductions, then
// the slice of O as the weighted sum of the splits' partial slices, written as bf16
// (round to nearest even); the first slice's CTAs also write the natural-log LSE.
template <int DH>
__global__ void __launch_bounds__(256) combine_kernel(DecodeArgs a) {
  const int g = blockIdx.x / a.ngroups, rg = blockIdx.x % a.ngroups, b = blockIdx.y;
  const int c8 = blockIdx.z % (DH / 8), rb = blockIdx.z / (DH / 8);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rows = min(a.rg, a.M - rg * a.rg);
  const size_t pidx0 = (((size_t)b * a.Hkv + g) * a.ngroups + rg) * a.nsplit;
  grid_dep_wait();  // every partial of the decode kernel is written
  const int T = a.lens[b];
  const bool valid = T >= 1 && T <= a.maxT;
  if (!valid && blockIdx.x == 0 && blockIdx.z == 0 && threadIdx.x == 0) set_status(a.status, HD_DEVBIT_INDEX);
  const int row = rb * 8 + warp;
  if (row < rows) {
    float m = -INFINITY;
    for (int c = lane; c < a.nsplit; c += 32) m = fmaxf(m, a.part_ml[(pidx0 + c) * a.rg + row].x);
#pragma unroll
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    float l = 0.f, acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int c = lane; c < a.nsplit; c += 32) {
      const float2 ml = a.part_ml[(pidx0 + c) * a.rg + row];
      const float f = (ml.x == -INFINITY || m == -INFINITY) ? 0.f : exp2f(ml.x - m);
      l += f * ml.y;
      if (f != 0.f) {
        const float4* src = reinterpret_cast<const float4*>(a.part_o + ((pidx0 + c) * a.rg + row) * DH + c8 * 8);
        const float4 x0 = src[0], x1 = src[1];
        acc[0] += f * x0.x;
        acc[1] += f * x0.y;
        acc[2] += f * x0.z;
        acc[3] += f * x0.w;
        acc[4] += f * x1.x;
        acc[5] += f * x1.y;
        acc[6] += f * x1.z;
        acc[7] += f * x1.w;
      }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      l += __shfl_xor_sync(0xffffffffu, l, off);
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], off);
    }
    if (lane == 0) {
      const bool ok = valid && l > 0.f;
      const float inv = ok ? 1.f / l : 0.f;
      const int r = rg * a.rg + row, s = r / a.G, h = g * a.G + r % a.G;
      uint4 out;
      out.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      out.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      out.z = pack_bf16(acc[4] * inv, acc[5] * inv);
      out.w = pack_bf16(acc[6] * inv, acc[7] * inv);
      *reinterpret_cast<uint4*>(a.o + (((long long)b * a.n + s) * a.Hq + h) * DH + c8 * 8) = out;
      if (c8 == 0 && a.lse != nullptr)
        a.lse[((long long)b * a.Hq + h) * a.n + s] = ok ? (m + __log2f(l)) * 0.6931471805599453f : -INFINITY;
    }
  }
}

// The new token's n K and V rows into the cache at positions (T-1)n + s: one warp per
// (sequence, stream), 16-byte vectors.  A length outside [1, Lcap] writes nothing and
// sets HD_DEVBIT_INDEX.
__global__ void __launch_bounds__(256) append_kernel(const uint4* __restrict__ kn, const uint4* __restrict__ vn,
                                                     uint4* __restrict__ kc, uint4* __restrict__ vc,
                                                     const int32_t* __restrict__ lens, int B, int Lcap, int n,
                                                     int row16, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const long long w = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (w >= (long long)B * n) return;
  const int b = (int)(w / n), s = (int)(w % n);
  const int T = lens[b];
  if (T < 1 || T > Lcap) {
    if (lane == 0 && s == 0) set_status(status, HD_DEVBIT_INDEX);
    return;
  }
  const long long dst = ((long long)b * Lcap * n + (long long)(T - 1) * n + s) * row16;
  const long long src = w * row16;
  for (int i = lane; i < row16; i += 32) {
    kc[dst + i] = kn[src + i];
    vc[dst + i] = vn[src + i];
  }
}
}  // namespace dec

// ------------------------------------------------------------------ tcgen05 path
// Head dim 256 with up to 128 query rows per K/V head (the 80B configuration: 4 streams x
// 12 heads = 48): the mma.sync kernel would take two row groups (reading the cache twice)
// and its warp-level products would limit the step, so this path runs the whole group on
// the tensor cores.  CTA (split c, K/V head, sequence): the group's M = n*G query rows
// (row s*G + head offset, zero rows up to 128) are one 128-row tile against 128-position
// tiles of the split's cached rows, with the head-dim-256 forward's plan: S in two
// 128-column TMEM buffers, O in columns 256..511, K / V halves (128 head-dim columns)
// through a five-slot ring in the issuer's order K(0), then K(j+1), V(j) per tile; warp 0
// TMA, warp 1 MMA issue, warps 2..5 the online softmax of one row each (per-element mask:
// position <= the row's own position, its stream in an intra-stream layer, the window in
// a local one) and the unnormalised partial (O, running max in log2 units, sum) that
// combine_kernel merges.  Every mbarrier wait is bounded.
namespace dectc {
constexpr int DH = 256, BM = 128, BN = 128, NSLOT = 5, NTHREADS = 192;
constexpr uint32_t COL_O = 256;
constexpr float kRescaleThreshold = 8.0f;

struct Smem {
  bf16 q[DH / 64][BM * 64];      // the group's query rows: four [128][64] swizzle blocks
  bf16 ring[NSLOT][2][BN * 64];  // per slot: one K or V half, two [128][64] blocks
  uint64_t q_full, full[NSLOT], empty[NSLOT], s_full[2], p_full[2], pv_done, drain;
  uint32_t tmem_base;
  int abort;
};

struct Params {
  CUtensorMap tm_q, tm_k, tm_v;
  dec::DecodeArgs a;
};

// Unit u of the ring sequence K(0), K(1), V(0), K(2), V(1), ..., V(nt-1), two halves per
// tile: its tile, tensor (0 = K, 1 = V) and half.
HD_DEVINLINE void unit_of(int u, int nt, int& j, int& isv, int& half) {
  half = u & 1;
  const int p = u >> 1;
  if (p == 0) {
    j = 0;
    isv = 0;
    return;
  }
  const int i = (p - 1) >> 1;
  if (((p - 1) & 1) == 0 && i < nt - 1) {
    j = i + 1;
    isv = 0;
    return;
  }
  j = i < nt - 1 ? i : (p - 1) - (nt - 1);
  isv = 1;
}

__global__ void __launch_bounds__(NTHREADS, 1) decode_tc_kernel(const __grid_constant__ Params P) {
  const dec::DecodeArgs& a = P.a;
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int c = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t pidx = ((size_t)b * a.Hkv + g) * a.nsplit + c;
  float* po = a.part_o + pidx * a.rg * DH;
  float2* pml = a.part_ml + pidx * a.rg;
  dec::grid_dep_wait();
  dec::grid_dep_launch();
  const int T = a.lens[b];
  int k0 = 0, k1 = 0;
  if (T >= 1 && T <= a.maxT) {
    int lo, hi;
    dec::seq_range(a, T, lo, hi);
    k0 = lo + c * a.chunk;
    k1 = min(k0 + a.chunk, hi);
  }
  if (k0 >= k1) {  // nothing of this sequence in this split: an empty partial
    for (int i = threadIdx.x; i < a.M; i += NTHREADS) pml[i] = make_float2(-INFINITY, 0.f);
    return;
  }
  const int nt = (k1 - k0 + BN - 1) / BN, nunits = 4 * nt;

  // rows M..127 of the query tile are zero (their scores are masked; no NaN enters O)
  for (int i = threadIdx.x; i < (DH / 64) * (BM - a.M) * 8; i += NTHREADS) {
    const int blk = i / ((BM - a.M) * 8), rem = i % ((BM - a.M) * 8);
    reinterpret_cast<uint4*>(sm.q[blk] + (a.M + rem / 8) * 64)[rem % 8] = make_uint4(0, 0, 0, 0);
  }
  fence_async_smem();
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
      mbar_arrive_expect_tx(&sm.q_full, a.M * DH * 2);
      for (int cb = 0; cb < DH / 64; ++cb) {
        asm volatile(
            "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5, %6}], [%2];\n" ::"r"(smem_u32(sm.q[cb])),
            "l"(reinterpret_cast<uint64_t>(&P.tm_q)), "r"(smem_u32(&sm.q_full)), "r"(cb * 64), "r"(g * a.G),
            "r"(0), "r"(b)
            : "memory");
      }
      int issued = 0;
      for (int u = 0; u < nunits; ++u, ++issued) {
        const int slot = u % NSLOT;
        if (u >= NSLOT && !mbar_wait(&sm.empty[slot], ((u / NSLOT) - 1) & 1, abort, a.status)) break;
        int j, isv, half;
        unit_of(u, nt, j, isv, half);
        const CUtensorMap* tm = isv ? &P.tm_v : &P.tm_k;
        mbar_arrive_expect_tx(&sm.full[slot], BN * 128 * 2);
        tma_load_5d(sm.ring[slot][0], tm, &sm.full[slot], half * 128, g, 0, k0 + j * BN, b);
        tma_load_5d(sm.ring[slot][1], tm, &sm.full[slot], half * 128 + 64, g, 0, k0 + j * BN, b);
      }
      mbar_drain(&sm.q_full, 0);
      for (int u = max(0, issued - NSLOT); u < issued; ++u) mbar_drain(&sm.full[u % NSLOT], (u / NSLOT) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idS = idesc_bf16(BM, BN, 0, 0);
    constexpr uint32_t idO = idesc_bf16(BM, 128, 0, 1);
    bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.q_full, 0, abort, a.status));
    int u = 0;
    auto wait_unit = [&](int x) -> bool {
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.full[x % NSLOT], (x / NSLOT) & 1, abort, a.status))) return false;
      tc_fence_after();
      return true;
    };
    // descriptors encoded once; a block, slot or k-step adds its byte offset / 16
    const uint64_t qd = sdesc_sw128(smem_u32(sm.q[0]), 16, 1024);
    const uint64_t rd = sdesc_sw128(smem_u32(sm.ring[0][0]), 16, 1024);
    const uint64_t rv = sdesc_sw128(smem_u32(sm.ring[0][0]), BN * 128, 1024);
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
    for (int i = 0; ok && i < nt; ++i) {
      if (i + 1 < nt && !issue_s((i + 1) & 1)) {
        ok = false;
        break;
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.p_full[i & 1], (i >> 1) & 1, abort, a.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (!issue_pv(i & 1, i > 0)) ok = false;
    }
    tc_commit_w(&sm.drain);
    mbar_drain(&sm.drain, 0);
  } else {
    // ------------------------------------------------------------ softmax / partial
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const bool rv = row < a.M;
    const int s = rv ? row / a.G : 0;
    const int pq = (T - 1) * a.n + s;  // the row's own position
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t tO = tl + COL_O;
    const float c2 = a.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int i = 0; i < nt; ++i) {
      const uint32_t tS = tl + (uint32_t)((i & 1) * 128);
      if (!__all_sync(0xffffffffu, mbar_wait(&sm.s_full[i & 1], (i >> 1) & 1, abort, a.status))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float x[BN];
#pragma unroll
      for (int cc = 0; cc < BN / 32; ++cc) tmem_ld32(tS + cc * 32, reinterpret_cast<uint32_t*>(x) + cc * 32);
      tmem_ld_wait();
      {
        const int base = k0 + i * BN;
        // (position - s) mod n, stepped along the columns (intra-stream layers keep 0)
        int kres = (base - s) % a.n;
        if (kres < 0) kres += a.n;
        const int lim = min(k1 - 1, pq), wlo = a.mode == SFA_LOCAL ? pq - a.window : -1;
        const bool within = a.mode == SFA_WITHIN;
#pragma unroll
        for (int e = 0; e < BN; ++e) {
          const int p = base + e;
          if (!rv || p > lim || p <= wlo || (within && kres != 0)) x[e] = -INFINITY;
          kres = kres + 1 == a.n ? 0 : kres + 1;
        }
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
      // O holds the earlier tiles' PVs only once PV(i-1) has completed
      if (i > 0) {
        if (!__all_sync(0xffffffffu, mbar_wait(&sm.pv_done, (i - 1) & 1, abort, a.status))) {
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
        for (int cc = 0; cc < DH / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(tO + cc * 32, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(tO + cc * 32, o);
        }
      }
      m_run = m_use;
      l_run += rsum;
#pragma unroll
      for (int cc = 0; cc < BN / 32; ++cc) tmem_st16(tS + cc * 16, pk + cc * 16);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&sm.p_full[i & 1]);
    }
    if (ok && __all_sync(0xffffffffu, mbar_wait(&sm.pv_done, (nt - 1) & 1, abort, a.status))) {
      tc_fence_after();
      float* orow = po + (size_t)row * DH;
#pragma unroll 1
      for (int cc = 0; cc < DH / 32; ++cc) {
        uint32_t o[32];
        tmem_ld32(tO + cc * 32, o);
        tmem_ld_wait();
        if (rv) {
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<float4*>(orow + cc * 32 + e) =
                make_float4(__uint_as_float(o[e]), __uint_as_float(o[e + 1]), __uint_as_float(o[e + 2]),
                            __uint_as_float(o[e + 3]));
        }
      }
      if (rv) pml[row] = make_float2(m_run * c2, l_run);
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
}  // namespace dectc

// ------------------------------------------------------------------ host side

DecodePlan decode_plan(int B, int maxT, int n, int Hq, int Hkv, int Dh, int mode, int window) {
  using namespace dec;
  DecodePlan p;
  p.G = Hq / Hkv;
  p.M = n * p.G;
  p.tc = Dh == 256 && p.M <= dectc::BM;
  p.rg = p.tc ? p.M : RG;
  p.ngroups = p.tc ? 1 : (p.M + RG - 1) / RG;
  const long long range = mode == SFA_LOCAL ? std::min<long long>((long long)maxT * n, (long long)window + n - 1)
                                            : (long long)maxT * n;
  const int KT = p.tc ? dectc::BN : Dh == 256 ? ktile<256>() : ktile<128>();
  const long long tiles = (range + KT - 1) / KT;
  const long long ctas = (long long)B * Hkv * p.ngroups;
  // resident decode CTAs: two per SM at head dim 128 (104 KB of shared memory) and 256
  // (112 KB), four at 64
  const long long resident = 152LL * (p.tc ? 1 : Dh == 64 ? 4 : 2);  // the tcgen05 kernel: one per SM
  // split count: least (waves x (tiles per CTA + a fixed cost of about two tiles))
  long long best = 1, best_cost = -1;
  for (long long ns = 1; ns <= std::min(tiles, (long long)kMaxSplit); ++ns) {
    const long long per = (tiles + ns - 1) / ns, used = (tiles + per - 1) / per;
    if (used != ns) continue;  // another ns gives the same chunks
    const long long cost = ((ctas * ns + resident - 1) / resident) * (per + 2);
    if (best_cost < 0 || cost < best_cost) {
      best = ns;
      best_cost = cost;
    }
  }
  const long long tiles_per = (tiles + best - 1) / best;
  p.chunk = (int)(tiles_per * KT);
  p.nsplit = (int)((tiles + tiles_per - 1) / tiles_per);
  const size_t parts = (size_t)B * Hkv * p.ngroups * p.nsplit;
  p.part_o_bytes = parts * p.rg * Dh * sizeof(float);
  p.part_ml_bytes = parts * p.rg * sizeof(float2);
  return p;
}

size_t decode_ws_bytes(const DecodePlan& p) { return ((p.part_o_bytes + 255) & ~size_t(255)) + p.part_ml_bytes; }

template <int DH, int MT>
static cudaError_t launch_decode_t(const dec::DecodeArgs& a, cudaStream_t st) {
  using namespace dec;
  const size_t smem = (size_t)(MT * 16 + 2 * STAGES * ktile<DH>()) * DH * sizeof(bf16);
  cudaError_t e = cudaFuncSetAttribute(decode_kernel<DH, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.nsplit, a.Hkv * a.ngroups, a.B);
  cfg.blockDim = dim3(NT);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decode_kernel<DH, MT>, a);
  if (e != cudaSuccess) return e;
  cfg.gridDim = dim3(a.Hkv * a.ngroups, a.B, (DH / 8) * ((std::min(a.rg, a.M) + 7) / 8));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  return cudaLaunchKernelEx(&cfg, combine_kernel<DH>, a);
}

static cudaError_t launch_decode_tc(const dec::DecodeArgs& a, cudaStream_t st) {
  using namespace dectc;
  Params p;
  p.a = a;
  SfaGeom gk = {};  // the cache as one problem of Lcap*n rows per sequence
  gk.B = a.B;
  gk.nL = a.Lcap * a.n;
  gk.Hq = a.Hq;
  gk.Hkv = a.Hkv;
  gk.n = a.n;
  gk.Lv = a.Lcap * a.n;
  gk.ns = 1;
  gk.rs = 1;
  if (!make_qgroup_tmap(&p.tm_q, a.q, a.B, a.n, a.Hq, DH, a.G) || !make_rows_tmap(&p.tm_k, a.kc, gk, a.Hkv, DH, BN) ||
      !make_rows_tmap(&p.tm_v, a.vc, gk, a.Hkv, DH, BN))
    return cudaErrorInvalidValue;
  const int smem = (int)sizeof(Smem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(decode_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.nsplit, a.Hkv, a.B);
  cfg.blockDim = dim3(NTHREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decode_tc_kernel, p);
  if (e != cudaSuccess) return e;
  cfg.gridDim = dim3(a.Hkv, a.B, (DH / 8) * ((std::min(a.rg, a.M) + 7) / 8));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  return cudaLaunchKernelEx(&cfg, dec::combine_kernel<DH>, a);
}

cudaError_t launch_sfa_decode(const void* q, const void* kc, const void* vc, const int32_t* lens, void* o,
                              float* lse, int B, int maxT, int Lcap, int n, int Hq, int Hkv, int Dh, float scale,
                              int mode, int window, void* ws, int32_t* status, cudaStream_t st) {
  const DecodePlan p = decode_plan(B, maxT, n, Hq, Hkv, Dh, mode, window);
  dec::DecodeArgs a;
  a.q = (const bf16*)q;
  a.kc = (const bf16*)kc;
  a.vc = (const bf16*)vc;
  a.lens = lens;
  a.o = (bf16*)o;
  a.lse = lse;
  a.part_o = static_cast<float*>(ws);
  a.part_ml = reinterpret_cast<float2*>(static_cast<char*>(ws) + ((p.part_o_bytes + 255) & ~size_t(255)));
  a.status = status;
  a.B = B;
  a.Lcap = Lcap;
  a.maxT = maxT;
  a.n = n;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = p.G;
  a.M = p.M;
  a.ngroups = p.ngroups;
  a.nsplit = p.nsplit;
  a.chunk = p.chunk;
  a.rg = p.rg;
  a.mode = mode;
  a.window = window;
  a.scale_log2 = scale * 1.4426950408889634f;
  if (p.tc) return launch_decode_tc(a, st);
  const bool two = p.M > 16;  // a row group of more than 16 rows takes two m16 tiles
  if (Dh == 64) return two ? launch_decode_t<64, 2>(a, st) : launch_decode_t<64, 1>(a, st);
  if (Dh == 256) return two ? launch_decode_t<256, 2>(a, st) : launch_decode_t<256, 1>(a, st);
  return two ? launch_decode_t<128, 2>(a, st) : launch_decode_t<128, 1>(a, st);
}

cudaError_t launch_kv_append(const void* kn, const void* vn, void* kc, void* vc, const int32_t* lens, int B,
                             int Lcap, int n, int Hkv, int Dh, int32_t* status, cudaStream_t st) {
  const long long warps = (long long)B * n;
  dec::append_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(
      (const uint4*)kn, (const uint4*)vn, (uint4*)kc, (uint4*)vc, lens, B, Lcap, n, Hkv * Dh / 8, status);
  return cudaGetLastError();
}

}  // namespace hdsfa
