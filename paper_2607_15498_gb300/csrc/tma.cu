// Host-side TMA tensor maps (cuTensorMapEncodeTiled reached through the runtime's driver entry
// point, so the library does not link libcuda directly).
#include <atomic>

#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace vr {

bool make_tmap_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  // driver entry point, looked up once per process (every thread that looks it up finds the same)
  static std::atomic<PFN_cuTensorMapEncodeTiled_v12000> cached{nullptr};
  PFN_cuTensorMapEncodeTiled_v12000 encode = cached.load(std::memory_order_acquire);
  if (encode == nullptr) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
      return false;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    cached.store(encode, std::memory_order_release);
  }
  // [rows][128] bf16, row-major; boxes of 64 columns (128 B, one swizzle span) x box_rows rows
  const cuuint64_t dims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)kHeadDim * 2};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace vr
