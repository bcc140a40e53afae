// sfa_bwd_noalloc: the SFA backward of sfa_bwd with its workspace held in a fixed
// device array of this module instead of a buffer the caller passes in.
//
// For callers that cannot hand the library device memory of their own: a runtime
// that commits its whole device-memory budget at start-up and forbids allocation
// once it is serving, or plain C code with no device allocator at hand.  The call
// allocates nothing: the array below is part of this module's static device image
// (SFA_BWD_NOALLOC_MAX_BYTES of device memory in every CUDA context that loads the
// module), and the entry point only looks up its address in the current context.
//
// The array is shared by every call on a device and keeps the previous call's
// contents.  Nothing stale is ever read: the prep pass of each call zeroes the fp32
// dQ accumulator and rewrites every row term (padding rows included) before the
// main pass reads them.  Two calls that may run at the same time on one device
// (different streams without an ordering event, or different host threads) use the
// same array and race; the caller orders them.
#include "common.cuh"
#include "nvtx_range.h"

namespace {

constexpr size_t kScratchBytes = SFA_BWD_NOALLOC_MAX_BYTES;
static_assert(kScratchBytes % 256 == 0, "scratch size keeps the workspace split 256-byte aligned");

static __device__ __align__(256) unsigned char g_sfa_bwd_scratch[kScratchBytes];

bool aligned16(const void* p) { return p != nullptr && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Device address of the array in the calling thread's current CUDA context.  The
// address belongs to that context (a non-primary context on the same device, or the
// primary context created again after cudaDeviceReset, holds the array elsewhere), so
// it is looked up on every call instead of being cached per device; once the module
// is loaded in the context the look-up is a table query.  The first call in a context
// loads the module there.
hd_status_t scratch_address(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_sfa_bwd_scratch);
  if (e != cudaSuccess || p == nullptr) {
    cudaGetLastError();  // leave no error behind for the caller's next check
    return HD_ERR_CUDA;
  }
  *out = p;
  return HD_OK;
}

}  // namespace

extern "C" hd_status_t sfa_bwd_noalloc(const void* q, const void* k, const void* v, const void* o,
                                       const float* lse, const void* dout, void* dq, void* dk, void* dv,
                                       int B, int L, int n, int Hq, int Hkv, int Dh,
                                       float softmax_scale, sfa_mode_t mode, int window,
                                       int32_t* dev_status, cudaStream_t stream) {
  HD_NVTX_RANGE("sfa_bwd_noalloc");
  // argument errors answer as sfa_bwd does, before the array is looked at
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse) ||
      !aligned16(dout) || !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
    return HD_ERR_INVALID_ARG;
  const size_t need = sfa_bwd_workspace_bytes(B, L, n, Hq, Hkv, Dh, mode);
  // invalid or unsupported sizes, or a LOCAL call without a window: sfa_bwd's own
  // status (its checks come before any workspace use; nothing is enqueued)
  if (need == 0 || (mode == SFA_LOCAL && window <= 0))
    return sfa_bwd(q, k, v, o, lse, dout, dq, dk, dv, B, L, n, Hq, Hkv, Dh, softmax_scale, mode, window,
                   nullptr, 0, dev_status, stream);
  if (need > kScratchBytes) return HD_ERR_SCRATCH_LIMIT;
  void* scratch = nullptr;
  const hd_status_t st = scratch_address(&scratch);
  if (st != HD_OK) return st;
  return sfa_bwd(q, k, v, o, lse, dout, dq, dk, dv, B, L, n, Hq, Hkv, Dh, softmax_scale, mode, window,
                 scratch, kScratchBytes, dev_status, stream);
}
