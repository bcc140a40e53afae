// Backward of the multi-stream token expansion (Eq. 1) and the final-stream
// selection the loss reads (Eq. 2).
//
// expand backward: dE[s][v][:] += sum over tokens t with ids[t] = v of dX[t*n + s][:].
//   Deterministic: the tokens are sorted by the 64-bit key (id << 32 | token index),
//   a total order, so the sum of each (s, v) row is taken in ascending token order by
//   one CTA and added to dE once (no floating-point atomics).
//   1. keys:  one key per token; ids outside [0, V) and the padding up to a power of
//      two get the largest keys and sort to the end.
//   2. bitonic sort, ascending: chunks of kChunk keys sorted in shared memory, then
//      for every larger sequence size the strides >= kChunk as global compare-exchange
//      steps and the strides below it in shared memory again.
//   3. rows: for each id present, CTAs over column slices of its n rows sum the id's
//      token rows in fp32, ascending token order, and add the sums into dE
//      (read-modify-write of fp32 rows).  An id outside [0, V) contributes nothing
//      and sets HD_DEVBIT_INDEX.
// select final: y[b][t] = x[b][t*n + n-1];  its adjoint writes dy to those rows and
//   zero to every other position.
#include "common.cuh"

namespace hdsfa {

typedef __nv_bfloat16 bf16;

namespace ebwd {
constexpr int kChunk = 2048;          // keys per shared-memory bitonic block
constexpr int kSortThreads = kChunk / 2;
constexpr int kRowThreads = 256;
constexpr unsigned long long kNoKey = ~0ull;

__global__ void keys_kernel(const int32_t* __restrict__ ids, unsigned long long* __restrict__ keys,
                            long long N, long long N2, int V, int32_t* status) {
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < N2;
       i += (long long)gridDim.x * blockDim.x) {
    unsigned long long k = kNoKey;
    if (i < N) {
      const int32_t x = ids[i];
      const bool ok = x >= 0 && x < V;
      if (!ok) set_status(status, HD_DEVBIT_INDEX);
      const unsigned long long hi = ok ? (unsigned long long)(uint32_t)x : 0xFFFFFFFFull;
      k = (hi << 32) | (unsigned long long)(uint32_t)i;
    }
    keys[i] = k;
  }
}

// Compare-exchange of positions i < l: ascending when (i & seq) == 0 (bitonic network).
HD_DEVINLINE void cmpx(unsigned long long& a, unsigned long long& b, bool asc) {
  if ((a > b) == asc) {
    const unsigned long long t = a;
    a = b;
    b = t;
  }
}

// seq_hi == 0: sort each chunk completely (sequence sizes 2 .. kChunk).
// seq_hi  > 0: finish sequence size seq_hi inside each chunk (strides kChunk/2 .. 1).
__global__ void __launch_bounds__(kSortThreads) chunk_kernel(unsigned long long* __restrict__ keys, long long seq_hi) {
  __shared__ unsigned long long sk[kChunk];
  const long long base = (long long)blockIdx.x * kChunk;
  for (int i = threadIdx.x; i < kChunk; i += kSortThreads) sk[i] = keys[base + i];
  __syncthreads();
  const long long k0 = seq_hi ? seq_hi : 2, k1 = seq_hi ? seq_hi : kChunk;
  for (long long seq = k0; seq <= k1; seq <<= 1) {
    for (int j = (int)(seq < kChunk ? seq : kChunk) >> 1; j > 0; j >>= 1) {
      const int p = threadIdx.x;  // one pair per thread
      const int i = 2 * j * (p / j) + (p % j), l = i + j;
      const bool asc = ((base + i) & seq) == 0;
      unsigned long long a = sk[i], b = sk[l];
      cmpx(a, b, asc);
      sk[i] = a;
      sk[l] = b;
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < kChunk; i += kSortThreads) keys[base + i] = sk[i];
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

// Work unit w = i * slices + z: sorted position i, column slice z of the n*D/8
// 16-byte chunks of a row (kRowThreads chunks per slice, one per thread).  Only a
// position that starts an id's run of keys does work; it sums the chunk over the
// run's tokens in ascending token order and adds the sum into dE once.  A frequent
// id's slices run on different SMs; every element still has a single writer.
__global__ void __launch_bounds__(kRowThreads) rows_kernel(const bf16* __restrict__ dx,
                                                          const unsigned long long* __restrict__ keys,
                                                          float* __restrict__ de, long long N, int n, int V,
                                                          int D, int slices) {
  const int d8 = D / 8;
  const long long units = N * slices;
  for (long long w = blockIdx.x; w < units; w += gridDim.x) {
    const long long i = w / slices;
    const int z = (int)(w - i * slices);
    const uint32_t v = (uint32_t)(keys[i] >> 32);
    if (v == 0xFFFFFFFFu) break;  // ids outside [0, V) and padding: the sorted tail
    if (i > 0 && (uint32_t)(keys[i - 1] >> 32) == v) continue;  // inside a run
    // run length m: keys are sorted, so the matches after i form a prefix
    long long m = 1;
    for (;;) {
      const long long j = i + m + threadIdx.x;
      const int hit = (j < N && (uint32_t)(keys[j] >> 32) == v) ? 1 : 0;
      const int cnt = __syncthreads_count(hit);
      m += cnt;
      if (cnt < kRowThreads) break;
    }
    const int it = z * kRowThreads + threadIdx.x;  // chunk of the n*D/8 of this id
    if (it < n * d8) {
      const int s = it / d8, c = it - s * d8;
      const bf16* src = dx + (long long)s * D + c * 8;
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (long long j0 = i; j0 < i + m; j0 += 8) {
        uint4 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          x[u] = make_uint4(0, 0, 0, 0);
          if (j0 + u < i + m) {
            const long long tok = (long long)(uint32_t)keys[j0 + u];  // b*L + t
            x[u] = *reinterpret_cast<const uint4*>(src + tok * n * (long long)D);
          }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          if (j0 + u < i + m) {  // ascending token order, one add per token
            const bf16* h = reinterpret_cast<const bf16*>(&x[u]);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] += __bfloat162float(h[e]);
          }
        }
      }
      float4* dst = reinterpret_cast<float4*>(de + ((long long)s * V + v) * D + c * 8);
      float4 a = dst[0], b = dst[1];
      a.x += acc[0];
      a.y += acc[1];
      a.z += acc[2];
      a.w += acc[3];
      b.x += acc[4];
      b.y += acc[5];
      b.z += acc[6];
      b.w += acc[7];
      dst[0] = a;
      dst[1] = b;
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

static unsigned grid_for(long long work, int per_block, long long cap) {
  long long g = (work + per_block - 1) / per_block;
  if (g < 1) g = 1;
  return (unsigned)(g < cap ? g : cap);
}

cudaError_t launch_expand_bwd(const void* dx, const int32_t* ids, float* de, int B, int L, int n, int V, int D,
                              void* keys_ws, int32_t* status, cudaStream_t st) {
  using namespace ebwd;
  const long long N = (long long)B * L, N2 = expand_bwd_sort_len(N);
  unsigned long long* keys = static_cast<unsigned long long*>(keys_ws);
  keys_kernel<<<grid_for(N2, 256, 152LL * 16), 256, 0, st>>>(ids, keys, N, N2, V, status);
  const unsigned nchunks = (unsigned)(N2 / kChunk);
  chunk_kernel<<<nchunks, kSortThreads, 0, st>>>(keys, 0);
  for (long long seq = 2LL * kChunk; seq <= N2; seq <<= 1) {
    for (long long j = seq >> 1; j >= kChunk; j >>= 1)
      step_kernel<<<grid_for(N2 / 2, 256, 152LL * 16), 256, 0, st>>>(keys, N2, seq, j);
    chunk_kernel<<<nchunks, kSortThreads, 0, st>>>(keys, seq);
  }
  const int slices = (int)(((long long)n * (D / 8) + kRowThreads - 1) / kRowThreads);
  rows_kernel<<<grid_for(N * slices, 1, 152LL * 8), kRowThreads, 0, st>>>((const bf16*)dx, keys, de, N, n, V,
                                                                          D, slices);
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
