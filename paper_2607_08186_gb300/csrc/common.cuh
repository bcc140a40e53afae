// Device helpers shared by the sm_103a kernels of libhdsfa.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/hdsfa.h"

#define HD_DEVINLINE __device__ __forceinline__

// One attention problem seen by a kernel: plain causal attention over a "virtual"
// sequence of Lv rows whose row r lives at expanded position p = r*rs + s.
//   WITHIN: one problem per stream s, Lv = L, rs = n   (Eq. 4: stream s sees only
//           its own earlier positions, which are exactly every n-th row).
//   CROSS : one problem, Lv = nL, rs = 1, s = 0       (Fig. 2a: causal over nL).
//   LOCAL : as CROSS plus the window lower bound       (Fig. 2b).
//
// Query side.  In the modes above the queries are the same virtual rows as the keys.
// A final-stream problem (the loss rows of Eq. 2 / the final-stream-only layers of
// Sec. 3.1) has only the L final-stream queries, in their own dense [B][L] tensors,
// against the keys above: query row r stands at key row r*qstep + qoff of its
// problem (CROSS / LOCAL over nL: qstep = n, qoff = n-1; WITHIN: the problem of
// stream n-1 alone, qstep = 1, qoff = 0, kv_s0 = n-1).
struct SfaGeom {
  int B, nL, Hq, Hkv, n;
  int Lv;       // key rows of each virtual problem
  int ns;       // problems per (b, head): n for WITHIN, 1 otherwise
  int rs;       // expanded-position step between consecutive virtual rows
  int window;   // > 0 only for LOCAL: key r' visible iff r - window < r' <= r
  int Lq;       // query rows of each problem (= Lv when queries are the key rows)
  int qstep, qoff;         // query row r sits at key row r*qstep + qoff (1, 0)
  int q_nL, q_ns, q_rs;    // rows per batch, problems, row step of the query tensors (nL, ns, rs)
  int kv_s0;               // stream of the first key problem (0)
  int smod;                // > 1: a pair is visible only if its key and query rows are
                           // congruent mod smod (the intra-stream mask of Eq. 4 over the
                           // CROSS schedule, SFA_WITHIN_NAIVE); 0 otherwise
};

// Geometry of the query-side tensors (Q, O, dO, dQ, LSE, row terms) of a problem.
__host__ __device__ inline SfaGeom query_geom(const SfaGeom& g) {
  SfaGeom q = g;
  q.nL = g.q_nL;
  q.ns = g.q_ns;
  q.rs = g.q_rs;
  q.Lv = g.Lq;
  q.Lq = g.Lq;
  q.qstep = 1;
  q.qoff = 0;
  q.kv_s0 = 0;
  return q;
}

// Stream-major backward row terms (-lse*log2e, -delta) are padded per (b, h, stream)
// to a multiple of the largest query tile any backward kernel reads at once.
constexpr int kRowTermAlign = 128;
__host__ __device__ inline int row_terms_pitch(int Lv) { return (Lv + kRowTermAlign - 1) / kRowTermAlign * kRowTermAlign; }

// Head chunks of the tensor-core backward.  Its grid is one CTA (two at head dim 256)
// per 128-row key tile and (b, K/V head, stream); when that leaves SMs idle (short or
// final-stream problems with few K/V heads), each CTA takes only a chunk of the group's
// query heads, for up to about four CTAs per SM.  (With one to two CTAs per SM, as in the n = 1
// and the final-stream intra-stream layers with 8 K/V heads, the partial sums' extra
// traffic cost more than the better balance gained: 3 % slower.)  Chunk hc writes its dK / dV partial sums (fp32,
// dK already scaled) to its own slice of a workspace [chunks][2][B][q_ns][Lv][Hkv][Dh]
// (dV, then dK), and a finalize pass adds the slices in chunk order: the same result,
// bit for bit, on every run.
constexpr int kSmCount = 152;
__host__ __device__ inline int bwd_head_chunks(const SfaGeom& g, int Dh) {
  const long long ctas = (long long)((g.Lv + 127) / 128) * (Dh == 256 ? 2 : 1) * g.Hkv * g.q_ns * g.B;
  const int grp = g.Hq / g.Hkv;
  if (ctas >= kSmCount || grp < 2) return 1;
  long long want = (4 * kSmCount + ctas - 1) / ctas;  // 2 or 6 per SM: 3.5 % / 1 % slower
  const int hs = (int)(want < grp ? want : grp);
  const int per = (grp + hs - 1) / hs;
  return (grp + per - 1) / per;
}
// Elements of one slice half (dV or dK of one chunk); 0 without chunks.
__host__ __device__ inline size_t bwd_dkv_slice(const SfaGeom& g, int Dh) {
  return bwd_head_chunks(g, Dh) > 1 ? (size_t)g.B * g.q_ns * g.Lv * g.Hkv * Dh : 0;
}

HD_DEVINLINE uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

HD_DEVINLINE void cp_async_16(uint32_t dst, const void* src, bool pred) {
  int sz = pred ? 16 : 0;  // src-size 0 zero-fills the 16 destination bytes
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(sz));
}
HD_DEVINLINE void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
HD_DEVINLINE void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

HD_DEVINLINE void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
HD_DEVINLINE void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}

// D(16x8 f32) += A(16x16 bf16, row) * B(16x8 bf16, col)
HD_DEVINLINE void mma_bf16_16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

HD_DEVINLINE uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Element offset of (row, col) in a [rows][RL] bf16 tile whose 16-byte chunks are
// XOR-swizzled by (row & 7), so 8 consecutive rows of one chunk hit 8 distinct
// bank groups (conflict-free ldmatrix and cp.async).  RL must be >= 64.
template <int RL>
HD_DEVINLINE int swz(int row, int col) {
  return row * RL + ((((col >> 3) ^ (row & 7))) << 3) + (col & 7);
}

HD_DEVINLINE void set_status(int32_t* st, int bit) {
  if (st) atomicOr(st, bit);
}
