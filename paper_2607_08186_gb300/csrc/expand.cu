// Multi-stream token expansion (Eq. 1): out[b][t*n + s][:] = tables[s][ids[b][t]][:].
//
// HBM-bound bit copy.  One warp per output row (b, t, s): it reads the table row
// with 16-byte non-coherent loads (the tables are read-only during the kernel) and
// writes the contiguous output row with 16-byte stores, four vectors in flight per
// lane.  Output rows are visited in memory order, so consecutive warps write
// consecutive rows.
#include "common.cuh"

namespace hdsfa {

__global__ void __launch_bounds__(256) expand_embed_kernel(const uint4* __restrict__ tables,
                                                           const int32_t* __restrict__ ids,
                                                           uint4* __restrict__ out, long long rows,
                                                           int n, int V, int D16, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const long long warp0 = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
  for (long long row = warp0; row < rows; row += nwarps) {
    const int s = (int)(row % n);
    const int id = __ldg(ids + row / n);
    uint4* dst = out + row * D16;
    if (id < 0 || id >= V) {
      for (int c = lane; c < D16; c += 32) dst[c] = make_uint4(0, 0, 0, 0);
      if (lane == 0 && s == 0) set_status(status, HD_DEVBIT_INDEX);
      continue;
    }
    const uint4* src = tables + ((long long)s * V + id) * D16;
    int c = lane;
    for (; c + 96 < D16; c += 128) {
      uint4 a0 = __ldg(src + c), a1 = __ldg(src + c + 32), a2 = __ldg(src + c + 64),
            a3 = __ldg(src + c + 96);
      dst[c] = a0;
      dst[c + 32] = a1;
      dst[c + 64] = a2;
      dst[c + 96] = a3;
    }
    for (; c < D16; c += 32) dst[c] = __ldg(src + c);
  }
}

cudaError_t launch_expand_embed(const void* tables, const int32_t* ids, void* out, int B, int L,
                                int n, int V, int D, int32_t* status, cudaStream_t stream) {
  const long long rows = (long long)B * L * n;
  const int threads = 256;
  long long blocks = (rows + (threads / 32) - 1) / (threads / 32);
  if (blocks > 152LL * 64) blocks = 152LL * 64;  // grid-stride beyond 64 waves of the 152 SMs
  expand_embed_kernel<<<(unsigned)blocks, threads, 0, stream>>>(
      (const uint4*)tables, ids, (uint4*)out, rows, n, V, D / 8, status);
  return cudaGetLastError();
}

}  // namespace hdsfa
