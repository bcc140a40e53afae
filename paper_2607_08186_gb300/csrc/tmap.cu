// Host-side TMA tensor-map construction (driver entry point fetched through the
// runtime, so the library needs no link-time libcuda dependency).
#include <cudaTypedefs.h>

#include "tc_common.cuh"

namespace hdsfa {

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

bool make_rows_tmap(CUtensorMap* m, const void* base, const SfaGeom& g, int H, int Dh, int box_rows,
                    int esize, int box_d, bool swizzle128) {
  auto enc = tmap_encoder();
  if (enc == nullptr) return false;
  const cuuint64_t e = (cuuint64_t)esize;
  cuuint64_t dims[5] = {(cuuint64_t)Dh, (cuuint64_t)H, (cuuint64_t)g.ns, (cuuint64_t)g.Lv, (cuuint64_t)g.B};
  cuuint64_t strides[4] = {Dh * e, (cuuint64_t)H * Dh * e, (cuuint64_t)g.rs * H * Dh * e,
                           (cuuint64_t)g.nL * H * Dh * e};
  cuuint32_t box[5] = {(cuuint32_t)box_d, 1, 1, (cuuint32_t)box_rows, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  const CUtensorMapDataType dt = esize == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUresult r = enc(m, dt, 5, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Tensor map over the decoding step's queries q [B][n][Hq][Dh] seen as {Dh, Hq, n, B};
// box = 64 columns x G heads x n streams of one sequence, so one load per 64 columns
// brings the n*G query rows of a K/V head's group, row s*G + (head - first head).
bool make_qgroup_tmap(CUtensorMap* m, const void* base, int B, int n, int Hq, int Dh, int G) {
  auto enc = tmap_encoder();
  if (enc == nullptr) return false;
  cuuint64_t dims[4] = {(cuuint64_t)Dh, (cuuint64_t)Hq, (cuuint64_t)n, (cuuint64_t)B};
  cuuint64_t strides[3] = {(cuuint64_t)Dh * 2, (cuuint64_t)Hq * Dh * 2, (cuuint64_t)n * Hq * Dh * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)G, (cuuint32_t)n, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace hdsfa
