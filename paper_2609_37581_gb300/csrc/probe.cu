// A measurement kernel beside the method: the scoring grid's Z copies without its consumers.
#include <cuda.h>

#include "common.cuh"
#include "sm100.cuh"

namespace trevs {

// The scoring grid's copy geometry (pre_llm.cu): 128-row tiles, stages of four 64-column
// slices (64 KB), boxes of 8 rows x four slices.
constexpr int kTileRows = 128;
constexpr int kChunk = 64;
constexpr int kZSlices = 4;
constexpr int kZBoxRows = 8;
constexpr int kZBoxBytes = kZBoxRows * kZSlices * 128;
constexpr int kZStageBytes = kTileRows * kZSlices * 128;

// ------------------------------------------------------------------ streaming probe
//
// A measurement kernel, not part of the method: Z streams through shared memory exactly as
// in the scoring grid (3D boxes of 8 rows x four 64-column slices, a ring of two 64 KB
// stages, each CTA a contiguous range of (128-row tile, 256-column stage) units), and every
// stage is released as soon as it has landed. Its rate is what the scoring grid's copies
// reach without the grid's consumers.
__global__ void __launch_bounds__(64, 1) stream_probe_kernel(const __grid_constant__ CUtensorMap tmZ3, int tiles,
                                                            int nzs, uint32_t* err) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[2], empty[2];
  __shared__ volatile int s_abort;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    s_abort = 0;
    mbar_fence_init();
  }
  __syncthreads();
  const long long W = (long long)tiles * nzs, P = gridDim.x;
  const long long u0 = W * blockIdx.x / P, u1 = W * (blockIdx.x + 1) / P;
  const uint64_t lim = 2000000000ull;
  int issued = 0;
  if (tid == 0) {
    const uint64_t pz = l2_policy_evict_first();
    for (long long u = u0; u < u1; ++u, ++issued) {
      const int g = (int)(u - u0), s = g & 1, it = g >> 1;
      if (g >= 2 && !mbar_wait(smem_u32(&empty[s]), (it - 1) & 1, &s_abort, lim)) {
        s_abort = 1;
        break;
      }
      const int t = (int)(u / nzs), zs = (int)(u - (long long)t * nzs);
      const uint32_t fb = smem_u32(&full[s]);
      mbar_arrive_expect_tx(fb, (uint32_t)kZStageBytes);
      for (int zb = 0; zb < kTileRows / kZBoxRows; ++zb)
        tma_load_3d(smem_u32(smem) + s * kZStageBytes + zb * kZBoxBytes, &tmZ3, 0, t * kTileRows + zb * kZBoxRows,
                    zs * kZSlices, fb, pz);
    }
  } else if (tid == 32) {
    for (long long u = u0; u < u1; ++u) {
      const int g = (int)(u - u0), s = g & 1, it = g >> 1;
      if (!mbar_wait(smem_u32(&full[s]), it & 1, &s_abort, lim)) {
        s_abort = 1;
        break;
      }
      mbar_arrive(smem_u32(&empty[s]));
    }
  }
  __syncthreads();
  if (s_abort && tid == 0) {
    // let the copies already issued land before the block's shared memory is released
    const volatile int no_abort = 0;
    for (int g = issued - 2 > 0 ? issued - 2 : 0; g < issued; ++g)
      mbar_wait(smem_u32(&full[g & 1]), (g >> 1) & 1, &no_abort, 500000000ull);
    atomicOr(err, 1u);
  }
}

// ------------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// Z [rows][cols] as [cols / 64][rows][64], boxes of 8 rows x four slices, 128-byte swizzle,
// zero fill past the last row: the scoring grid's map of Z.
static cudaError_t make_probe_map(CUtensorMap* tm, const void* base, long long rows, int cols, long long stride) {
  static EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {(cuuint64_t)kChunk, (cuuint64_t)rows, (cuuint64_t)(cols / kChunk)};
  const cuuint64_t strides[2] = {(cuuint64_t)stride * 2, (cuuint64_t)kChunk * 2};
  const cuuint32_t box[3] = {(cuuint32_t)kChunk, (cuuint32_t)kZBoxRows, (cuuint32_t)kZSlices};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult res = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// One pass of the streaming probe over Z [rows][d] (d a multiple of 256) on `ctas` CTAs.
cudaError_t launch_stream_probe(const void* Z, long long z_stride, long long rows, int d, int ctas, uint32_t* err,
                                cudaStream_t st) {
  CUtensorMap tm;
  cudaError_t e = make_probe_map(&tm, Z, rows, d, z_stride);
  if (e != cudaSuccess) return e;
  const int smem = 2 * kZStageBytes + 1024;
  e = ensure_dynamic_smem(stream_probe_kernel, smem);
  if (e != cudaSuccess) return e;
  const int tiles = (int)((rows + kTileRows - 1) / kTileRows), nzs = d / (kChunk * kZSlices);
  if (launch_fault_injected()) return cudaErrorLaunchFailure;
  stream_probe_kernel<<<ctas, 64, smem, st>>>(tm, tiles, nzs, err);
  return cudaGetLastError();
}

}  // namespace trevs
