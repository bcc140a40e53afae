// Backward of the multi-stream token expansion (Eq. 1) and the final-stream
// selection the loss reads (Eq. 2).
//
// expand backward: dE[s][v][:] += sum over tokens t with ids[t] = v of dX[t*n + s][:].
//   Deterministic: the tokens are sorted by the 64-bit key (id << 32 | token index),
//   a total order, so the sum of each (s, v) row is taken in ascending token order by
//   one CTA and added to dE once (no floating-point atomics).
//   1. sort the keys, ascending (ids outside [0, V) get the largest keys and sort to
//      the end).  Up to kRankMax tokens by rank: each key's sorted position is the
//      number of keys below it, counted by a 2-D grid of tiles.  Beyond that, bitonic:
//      keys built and sorted in shared memory in chunks of kChunk (padding up to a
//      power of two sorts last); for every larger sequence size the strides >= kChunk
//      run as global compare-exchange steps and the strides below it in shared
//      memory again.
//   2. runs: each run of equal ids is listed once with its start, length and first
//      token, light (<= kHeavy tokens) and heavy runs apart (by the rank pass itself,
//      or by a pass over the bitonic result).  Steps 1-2 depend on the ids only: the
//      "plan", which a caller may build once, off the critical path, and apply later.
//   3. rows: CTAs over column slices of a run's n rows sum the run's token rows in
//      fp32 and add the sums into dE (read-modify-write of fp32 rows).  A light run
//      is summed in ascending token order; a heavy one in kHeavyBlocks consecutive
//      token blocks (one warp each, ascending order within a block) whose sums are
//      added in block order.  The order depends only on the run's length: repeated
//      calls give identical bits.  An id outside [0, V) contributes nothing and
//      sets HD_DEVBIT_INDEX.
// select final: y[b][t] = x[b][t*n + n-1];  its adjoint writes dy to those rows and
//   zero to every other position.
#include "common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace ebwd {
constexpr int kChunk = 4096;          // keys per shared-memory bitonic block (32 KB)
constexpr int kSortThreads = 1024;    // two compare-exchanges per thread and stage
constexpr int kRowThreads = 256;
constexpr int kHeavy = 32;            // runs longer than this take the split-token path
constexpr int kLightItems = 2 * kRowThreads;  // 16-byte chunks per light unit, two per thread
constexpr int kHeavyItems = 32;               // chunks per heavy unit, one per lane
constexpr int kHeavyBlocks = kRowThreads / 32;  // consecutive token blocks of a heavy run
constexpr int kRankTile = 256;         // keys per tile of the rank count
constexpr long long kRankMax = 16384;  // up to this many tokens: rank count, else bitonic sort
constexpr unsigned long long kNoKey = ~0ull;
constexpr uint32_t kNoId = 0xFFFFFFFFu;

// Key of token i: (id << 32) | i, ids outside [0, V) and the padding up to N2 last.
HD_DEVINLINE unsigned long long make_key(const int32_t* ids, long long i, long long N, int V, int32_t* status) {
  if (i >= N) return kNoKey;
  const int32_t x = ids[i];
  const bool ok = x >= 0 && x < V;
  if (!ok) set_status(status, HD_DEVBIT_INDEX);
  return ((ok ? (unsigned long long)(uint32_t)x : 0xFFFFFFFFull) << 32) | (unsigned long long)(uint32_t)i;
}

// Compare-exchange of positions i < l: ascending when (i & seq) == 0 (bitonic network).
HD_DEVINLINE void cmpx(unsigned long long& a, unsigned long long& b, bool asc) {
  if ((a > b) == asc) {
    const unsigned long long t = a;
    a = b;
    b = t;
  }
}

// seq_hi == 0: build the keys of the chunk from ids and sort it completely
//              (sequence sizes 2 .. kChunk); block 0 also clears the run counters.
// seq_hi  > 0: finish sequence size seq_hi inside each chunk (strides kChunk/2 .. 1).
__global__ void __launch_bounds__(kSortThreads) chunk_kernel(unsigned long long* __restrict__ keys,
                                                             const int32_t* __restrict__ ids, long long N, int V,
                                                             long long seq_hi, unsigned* __restrict__ counts,
                                                             int32_t* status) {
  __shared__ unsigned long long sk[kChunk];
  const long long base = (long long)blockIdx.x * kChunk;
  if (seq_hi == 0) {
    if (blockIdx.x == 0 && threadIdx.x < 2) counts[threadIdx.x] = 0;
    for (int i = threadIdx.x; i < kChunk; i += kSortThreads) sk[i] = make_key(ids, base + i, N, V, status);
  } else {
    for (int i = threadIdx.x; i < kChunk; i += kSortThreads) sk[i] = keys[base + i];
  }
  __syncthreads();
  const long long k0 = seq_hi ? seq_hi : 2, k1 = seq_hi ? seq_hi : kChunk;
  for (long long seq = k0; seq <= k1; seq <<= 1) {
    for (int j = (int)(seq < kChunk ? seq : kChunk) >> 1; j > 0; j >>= 1) {
      for (int p = threadIdx.x; p < kChunk / 2; p += kSortThreads) {
        const int i = 2 * j * (p / j) + (p % j), l = i + j;
        unsigned long long a = sk[i], b = sk[l];
        cmpx(a, b, ((base + i) & seq) == 0);
        sk[i] = a;
        sk[l] = b;
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < kChunk; i += kSortThreads) keys[base + i] = sk[i];
}

// Sorting by rank, for up to kRankMax tokens: the keys are distinct, so the sorted
// position of key i is the number of keys below it.  Tile (x, y) counts, for each
// key i of tile x and the keys of tile y: the keys below key i, the keys with its
// id, and the keys with its id below it, packed in 21-bit fields of partial[y][i].
// The scatter pass adds a key's counts in tile order, stores the key at its rank and,
// for the first key of an id (no key of its id below it), appends the id's run
// record.  Block (0, 0) also clears the run counters.
constexpr int kField = 21;
__global__ void __launch_bounds__(kRankTile) rank_kernel(const int32_t* __restrict__ ids, long long N, int V,
                                                        unsigned long long* __restrict__ partial,
                                                        unsigned* __restrict__ counts, int32_t* status) {
  __shared__ ulonglong2 sj[kRankTile / 2];
  const long long j0 = (long long)blockIdx.y * kRankTile;
  const long long i = (long long)blockIdx.x * kRankTile + threadIdx.x;
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x < 2) counts[threadIdx.x] = 0;
  // keys past N are kNoKey, above every real key; ids are checked once (tile row x = 0)
  reinterpret_cast<unsigned long long*>(sj)[threadIdx.x] =
      make_key(ids, j0 + threadIdx.x, N, V, blockIdx.x == 0 ? status : nullptr);
  __syncthreads();
  if (i >= N) return;
  const unsigned long long ki = make_key(ids, i, N, V, nullptr);
  const uint32_t vi = (uint32_t)(ki >> 32);
  unsigned below = 0, same = 0, same_below = 0;
#pragma unroll 8
  for (int t = 0; t < kRankTile / 2; ++t) {
    const ulonglong2 p = sj[t];
    const bool bx = p.x < ki, by = p.y < ki;
    const bool sx = (uint32_t)(p.x >> 32) == vi, sy = (uint32_t)(p.y >> 32) == vi;
    below += bx + by;
    same += sx + sy;
    same_below += (sx && bx) + (sy && by);
  }
  partial[blockIdx.y * N + i] = (unsigned long long)below | ((unsigned long long)same << kField) |
                                ((unsigned long long)same_below << (2 * kField));
}

__global__ void __launch_bounds__(256) scatter_kernel(const int32_t* __restrict__ ids, long long N, int V,
                                                      const unsigned long long* __restrict__ partial, int tiles,
                                                      unsigned long long* __restrict__ keys, uint4* __restrict__ light,
                                                      uint4* __restrict__ heavy, unsigned* __restrict__ counts) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  unsigned long long acc = 0;  // fields stay below 2^15 (N <= kRankMax): no carries
#pragma unroll 8
  for (int y = 0; y < tiles; ++y) acc += partial[(long long)y * N + i];
  const unsigned mask = (1u << kField) - 1;
  const unsigned r = (unsigned)acc & mask, m = (unsigned)(acc >> kField) & mask;
  const unsigned first = (unsigned)(acc >> (2 * kField)) & mask;
  const unsigned long long key = make_key(ids, i, N, V, nullptr);
  keys[r] = key;
  const uint32_t v = (uint32_t)(key >> 32);
  if (v != kNoId && first == 0) {
    const uint4 rec = make_uint4(r, m, (uint32_t)i, v);
    if (m <= (unsigned)kHeavy)
      light[atomicAdd(counts, 1u)] = rec;
    else
      heavy[atomicAdd(counts + 1, 1u)] = rec;
  }
}

// One global step of sequence size seq, stride j >= kChunk.
__global__ void step_kernel(unsigned long long* __restrict__ keys, long long N2, long long seq, long long j) {
  for (long long p = (long long)blockIdx.x * blockDim.x + threadIdx.x; p < N2 / 2;
       p += (long long)gridDim.x * blockDim.x) {
    const long long i = 2 * j * (p / j) + (p % j), l = i + j;
    unsigned long long a = keys[i], b = keys[l];
    const unsigned long long a0 = a;
    cmpx(a, b, (i & seq) == 0);
    if (a != a0) {
      keys[i] = a;
      keys[l] = b;
    }
  }
}

// Runs of equal ids in the sorted keys: one warp per sorted position; the warp of a
// run's first position measures the run with ballots and appends {start, length,
// first token, id} to the light (length <= kHeavy) or heavy list.  The order of a
// list depends on scheduling; the sums do not (each run is summed by itself).
__global__ void __launch_bounds__(256) runs_kernel(const unsigned long long* __restrict__ keys, long long N,
                                                   uint4* __restrict__ light, uint4* __restrict__ heavy,
                                                   unsigned* __restrict__ counts) {
  const int lane = threadIdx.x & 31;
  const long long nw = ((long long)gridDim.x * blockDim.x) >> 5;
  for (long long i = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < N; i += nw) {
    const unsigned long long key = keys[i];
    const uint32_t v = (uint32_t)(key >> 32);
    if (v == kNoId) break;  // the sorted tail: invalid ids and padding
    if (i > 0 && (uint32_t)(keys[i - 1] >> 32) == v) continue;
    long long m = 1;
    for (long long r = i + 1;; r += 32) {
      const long long j = r + lane;
      const unsigned b = __ballot_sync(0xffffffffu, j < N && (uint32_t)(keys[j] >> 32) == v);
      m += __popc(b);
      if (b != 0xffffffffu) break;
    }
    if (lane == 0) {
      const uint4 rec = make_uint4((uint32_t)i, (uint32_t)m, (uint32_t)key, v);
      if (m <= kHeavy)
        light[atomicAdd(counts, 1u)] = rec;
      else
        heavy[atomicAdd(counts + 1, 1u)] = rec;
    }
  }
}

HD_DEVINLINE void add_bf16x8(float* acc, const uint4& w) {
  const bf16* h = reinterpret_cast<const bf16*>(&w);
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] += __bfloat162float(h[e]);
}

HD_DEVINLINE void rmw_add(float* dst, const float4& a0, const float4& a1, const float* acc) {
  float4 x0 = a0, x1 = a1;
  x0.x += acc[0];
  x0.y += acc[1];
  x0.z += acc[2];
  x0.w += acc[3];
  x1.x += acc[4];
  x1.y += acc[5];
  x1.z += acc[6];
  x1.w += acc[7];
  reinterpret_cast<float4*>(dst)[0] = x0;
  reinterpret_cast<float4*>(dst)[1] = x1;
}

// Work units: heavy run r, slice z of kHeavyItems chunks, then light run r, slice z
// of kLightItems chunks (two per thread).  Chunk `it` of a token's n*D row lies at
// element it*8 of the token's n*D gradient block (stream it / (D/8)).
//   light: each thread sums its chunk over the run's tokens in ascending order.
//   heavy: warp w sums the chunk over the w-th of kHeavyBlocks consecutive token
//          blocks; warp 0 adds the block sums in block order.
// Every element of dE is read and written by exactly one thread.
__global__ void __launch_bounds__(kRowThreads, 3) rows_kernel(const bf16* __restrict__ dx,
                                                          const unsigned long long* __restrict__ keys,
                                                          const uint4* __restrict__ light,
                                                          const uint4* __restrict__ heavy,
                                                          const unsigned* __restrict__ counts,
                                                          float* __restrict__ de, long long N, int n, int V,
                                                          int D) {
  __shared__ float part[kHeavyBlocks][kHeavyItems][9];  // padded against bank conflicts
  const int d8 = D / 8, items = n * d8;
  const long long nD = (long long)n * D;
  const int SL = (items + kLightItems - 1) / kLightItems, SH = (items + kHeavyItems - 1) / kHeavyItems;
  // heavy units first: they take longest, so they start before the light ones
  // The run lists hold at most N records each; a record or a key outside the plan's
  // ranges (a workspace the plan did not write) is skipped, so every access stays in
  // bounds whatever the workspace holds.
  const long long nl = counts[0] < N ? counts[0] : N, nh = counts[1] < N ? counts[1] : N;
  const long long hunits = nh * SH, units = hunits + nl * SL;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (long long w = blockIdx.x; w < units; w += gridDim.x) {
    if (w >= hunits) {
      const long long lw = w - hunits, r = lw / SL;
      const int z = (int)(lw - r * SL);
      const uint4 rec = light[r];
      const uint32_t start = rec.x, m = rec.y, v = rec.w;
      if (start >= N || m > N - start || v >= (uint32_t)V || rec.z >= N) continue;
      int it[2];
      float* drow[2];
      float4 e0[2], e1[2];
      float acc[2][8];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        it[q] = z * kLightItems + q * kRowThreads + tid;
        drow[q] = nullptr;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[q][e] = 0.f;
        if (it[q] < items) {
          const int s = it[q] / d8, c = it[q] - s * d8;
          drow[q] = de + ((long long)s * V + v) * D + c * 8;
          e0[q] = reinterpret_cast<const float4*>(drow[q])[0];
          e1[q] = reinterpret_cast<const float4*>(drow[q])[1];
        }
      }
      // first token from the record, the others from the sorted keys
      for (uint32_t j0 = 0; j0 < m; j0 += 4) {
        uint4 x[4][2];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t j = j0 + u;
          long long tok = -1;
          if (j < m) tok = j == 0 ? (long long)rec.z : (long long)(uint32_t)keys[start + j];
          if (tok >= N) tok = -1;
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            x[u][q] = make_uint4(0, 0, 0, 0);
            if (tok >= 0 && drow[q] != nullptr)
              x[u][q] = *reinterpret_cast<const uint4*>(dx + tok * nD + (long long)it[q] * 8);
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (j0 + u < m) {
#pragma unroll
            for (int q = 0; q < 2; ++q) add_bf16x8(acc[q], x[u][q]);
          }
      }
#pragma unroll
      for (int q = 0; q < 2; ++q)
        if (drow[q] != nullptr) rmw_add(drow[q], e0[q], e1[q], acc[q]);
    } else {
      const long long r = w / SH;
      const int z = (int)(w - r * SH);
      const uint4 rec = heavy[r];
      const uint32_t start = rec.x, m = rec.y, v = rec.w;
      if (start >= N || m > N - start || v >= (uint32_t)V) continue;  // uniform over the block
      const int itm = z * kHeavyItems + lane;
      const bool live = itm < items;
      // token block of this warp: [m*warp/8, m*(warp+1)/8)
      const uint32_t jb = (uint32_t)((unsigned long long)m * warp / kHeavyBlocks);
      const uint32_t je = (uint32_t)((unsigned long long)m * (warp + 1) / kHeavyBlocks);
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (uint32_t j0 = jb; j0 < je; j0 += 8) {
        uint4 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          x[u] = make_uint4(0, 0, 0, 0);
          if (j0 + u < je && live) {
            const long long tok = (long long)(uint32_t)keys[start + j0 + u];
            if (tok < N) x[u] = *reinterpret_cast<const uint4*>(dx + tok * nD + (long long)itm * 8);
          }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (j0 + u < je) add_bf16x8(acc, x[u]);
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) part[warp][lane][e] = acc[e];
      __syncthreads();
      if (warp == 0 && live) {
        const int s = itm / d8, c = itm - s * d8;
        float* drow = de + ((long long)s * V + v) * D + c * 8;
        const float4 a0 = reinterpret_cast<const float4*>(drow)[0], a1 = reinterpret_cast<const float4*>(drow)[1];
        float sum[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) sum[e] = part[0][lane][e];
#pragma unroll
        for (int b = 1; b < kHeavyBlocks; ++b)
#pragma unroll
          for (int e = 0; e < 8; ++e) sum[e] += part[b][lane][e];
        rmw_add(drow, a0, a1, sum);
      }
      __syncthreads();
    }
  }
}

// y[b][t] = x[b][t*n + n-1]: one warp per output row, 16-byte vectors.
__global__ void __launch_bounds__(256) select_kernel(const uint4* __restrict__ x, uint4* __restrict__ y,
                                                     long long rows, int n, int d16) {
  const int lane = threadIdx.x & 31;
  const long long nw = ((long long)gridDim.x * blockDim.x) >> 5;
  for (long long r = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += nw) {
    const uint4* src = x + (r * n + (n - 1)) * d16;
    uint4* dst = y + r * d16;
    for (int c = lane; c < d16; c += 32) dst[c] = __ldg(src + c);
  }
}

// dx[b][p] = dy[b][p / n] when p % n == n-1, else zero: one warp per row of dx.
__global__ void __launch_bounds__(256) select_bwd_kernel(const uint4* __restrict__ dy, uint4* __restrict__ dx,
                                                         long long rows_x, int n, int d16) {
  const int lane = threadIdx.x & 31;
  const long long nw = ((long long)gridDim.x * blockDim.x) >> 5;
  for (long long p = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; p < rows_x; p += nw) {
    uint4* dst = dx + p * d16;
    if (p % n == n - 1) {
      const uint4* src = dy + (p / n) * d16;
      for (int c = lane; c < d16; c += 32) dst[c] = __ldg(src + c);
    } else {
      for (int c = lane; c < d16; c += 32) dst[c] = make_uint4(0, 0, 0, 0);
    }
  }
}
}  // namespace ebwd

// Keys padded to a power of two, at least one shared-memory chunk.
long long expand_bwd_sort_len(long long N) {
  long long N2 = ebwd::kChunk;
  while (N2 < N) N2 <<= 1;
  return N2;
}

// Workspace: sorted keys [N2] u64, light and heavy run lists [N] uint4 each, two
// counters (16 bytes), then, up to kRankMax tokens, the rank counts [tiles][N] u64.
size_t expand_bwd_ws_bytes(long long N) {
  const long long tiles = (N + ebwd::kRankTile - 1) / ebwd::kRankTile;
  return (size_t)expand_bwd_sort_len(N) * 8 + 2 * (size_t)N * 16 + 16 +
         (N <= ebwd::kRankMax ? (size_t)tiles * N * 8 : 0);
}

static unsigned grid_for(long long work, int per_block, long long cap) {
  long long g = (work + per_block - 1) / per_block;
  if (g < 1) g = 1;
  return (unsigned)(g < cap ? g : cap);
}

struct ExpandBwdWs {
  unsigned long long* keys;
  uint4* light;
  uint4* heavy;
  unsigned* counts;
  unsigned long long* partial;
};

static ExpandBwdWs split_ws(void* ws, long long N) {
  ExpandBwdWs w;
  w.keys = static_cast<unsigned long long*>(ws);
  w.light = reinterpret_cast<uint4*>(w.keys + expand_bwd_sort_len(N));
  w.heavy = w.light + N;
  w.counts = reinterpret_cast<unsigned*>(w.heavy + N);
  w.partial = reinterpret_cast<unsigned long long*>(w.counts + 4);
  return w;
}

// Plan: sorted keys and run lists of the ids (depends on ids only).
cudaError_t launch_expand_bwd_plan(const int32_t* ids, int B, int L, int V, void* ws, int32_t* status,
                                   cudaStream_t st) {
  using namespace ebwd;
  const long long N = (long long)B * L, N2 = expand_bwd_sort_len(N);
  const ExpandBwdWs w = split_ws(ws, N);
  if (N <= kRankMax) {
    const int tiles = (int)((N + kRankTile - 1) / kRankTile);
    rank_kernel<<<dim3(tiles, tiles), kRankTile, 0, st>>>(ids, N, V, w.partial, w.counts, status);
    scatter_kernel<<<tiles, kRankTile, 0, st>>>(ids, N, V, w.partial, tiles, w.keys, w.light, w.heavy,
                                                w.counts);
    return cudaGetLastError();
  }
  const unsigned nchunks = (unsigned)(N2 / kChunk);
  chunk_kernel<<<nchunks, kSortThreads, 0, st>>>(w.keys, ids, N, V, 0, w.counts, status);
  for (long long seq = 2LL * kChunk; seq <= N2; seq <<= 1) {
    for (long long j = seq >> 1; j >= kChunk; j >>= 1)
      step_kernel<<<grid_for(N2 / 2, 256, 152LL * 16), 256, 0, st>>>(w.keys, N2, seq, j);
    chunk_kernel<<<nchunks, kSortThreads, 0, st>>>(w.keys, ids, N, V, seq, w.counts, status);
  }
  runs_kernel<<<grid_for(N, 8, 152LL * 64), 256, 0, st>>>(w.keys, N, w.light, w.heavy, w.counts);
  return cudaGetLastError();
}

// Apply: the row sums of a plan into dE.
cudaError_t launch_expand_bwd_apply(const void* dx, float* de, int B, int L, int n, int V, int D, const void* ws,
                                    cudaStream_t st) {
  using namespace ebwd;
  const ExpandBwdWs w = split_ws(const_cast<void*>(ws), (long long)B * L);
  rows_kernel<<<152 * 3, kRowThreads, 0, st>>>((const bf16*)dx, w.keys, w.light, w.heavy, w.counts, de,
                                                 (long long)B * L, n, V, D);
  return cudaGetLastError();
}

cudaError_t launch_select_final(const void* x, void* y, int B, int L, int n, int D, cudaStream_t st) {
  const long long rows = (long long)B * L;
  ebwd::select_kernel<<<grid_for(rows, 8, 152LL * 64), 256, 0, st>>>((const uint4*)x, (uint4*)y, rows, n,
                                                                     D / 8);
  return cudaGetLastError();
}

cudaError_t launch_select_final_bwd(const void* dy, void* dx, int B, int L, int n, int D, cudaStream_t st) {
  const long long rows_x = (long long)B * L * n;
  ebwd::select_bwd_kernel<<<grid_for(rows_x, 8, 152LL * 64), 256, 0, st>>>((const uint4*)dy, (uint4*)dx,
                                                                           rows_x, n, D / 8);
  return cudaGetLastError();
}

}  // namespace hdsfa
