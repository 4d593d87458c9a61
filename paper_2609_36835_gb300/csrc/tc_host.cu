// Host side of the tensor-core kernels: TMA tensor-map encoding through the
// driver entry point (no link-time dependency on libcuda).
#include <cudaTypedefs.h>
#include <map>
#include <mutex>
#include <utility>

#include "tc.cuh"

namespace arckv {

namespace {
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_once;
}  // namespace

static bool encoder_ready() {
  std::call_once(g_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  });
  return g_encode != nullptr;
}

bool encode_bf16_map_3d(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint64_t dim2,
                        uint32_t box1) {
  if (!encoder_ready()) return false;
  // TMA requires a 16-byte aligned base and row strides that are multiples of 16 bytes
  if (((uintptr_t)base & 15u) != 0 || (dim0 * 2) % 16 != 0) return false;
  const cuuint64_t gdim[3] = {dim0, dim1, dim2};
  const cuuint64_t gstride[2] = {dim0 * 2, dim0 * dim1 * 2};
  const cuuint32_t box[3] = {64, box1, 1};
  const cuuint32_t estride[3] = {1, 1, 1};
  const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride, box,
                              estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_bf16_map_3d_sw64(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint64_t dim2,
                             uint64_t ld, uint32_t box1) {
  if (!encoder_ready()) return false;
  if (((uintptr_t)base & 15u) != 0 || (ld * 2) % 16 != 0 || ld < dim0 || box1 == 0 || box1 > 256) return false;
  const cuuint64_t gdim[3] = {dim0, dim1, dim2};
  const cuuint64_t gstride[2] = {ld * 2, ld * dim1 * 2};
  const cuuint32_t box[3] = {32, box1, 1};
  const cuuint32_t estride[3] = {1, 1, 1};
  const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride, box,
                              estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_f32_map_3d(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1, uint64_t dim2,
                       uint32_t box0, uint32_t box1, uint64_t ld, uint64_t bs, bool swz128) {
  if (!encoder_ready()) return false;
  if (ld == 0) ld = dim0;
  if (bs == 0) bs = ld * dim1;
  if (((uintptr_t)base & 15u) != 0 || (ld * 4) % 16 != 0 || (bs * 4) % 16 != 0 || (box0 * 4) % 16 != 0 ||
      box0 > 256 || box1 > 256 || ld < dim0 || (swz128 && box0 * 4 != 128))
    return false;
  const cuuint64_t gdim[3] = {dim0, dim1, dim2};
  const cuuint64_t gstride[2] = {ld * 4, bs * 4};
  const cuuint32_t box[3] = {box0, box1, 1};
  const cuuint32_t estride[3] = {1, 1, 1};
  const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), gdim, gstride, box,
                              estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              swz128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

cudaError_t set_dyn_smem(const void* kern, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> done;   // (kernel, device) -> bytes already allowed
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) dev = -1;
  std::lock_guard<std::mutex> lock(mu);
  auto it = done.find({kern, dev});
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done[{kern, dev}] = bytes;
  return e;
}

int tc_gemm_sm_count() {
  static std::mutex mu;
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == 0) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    cache[dev] = v > 0 ? v : 1;
  }
  return cache[dev];
}

}  // namespace arckv
