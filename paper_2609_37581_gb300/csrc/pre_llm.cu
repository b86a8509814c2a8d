// Stage 1 (pre-LLM, Sec. 4.1): textual-relevance scores (Eq. 4-5), selection (Sec. 3.1 ratio
// split or Eq. 6-7 fused score) and gather of the kept feature rows.
#include "pre_llm.cuh"
#include "sm100.cuh"

namespace trevs {

// ------------------------------------------------------------------ scoring contraction
//
// One CTA scores a tile of 128 visual rows of one request against the M text rows of that
// request. G = Z_tile . T^T runs on the 5th-generation tensor cores: TMA streams 64-column
// chunks of Z and T into a ring of 128-byte-swizzled shared-memory stages, one thread
// issues UMMA (M = 128, N = M rounded up to 16, K = 16 per instruction) into a TMEM
// accumulator, and four warps compute the fp32 squared norms ||z_i||^2, ||t_j||^2 from the
// same stages. The epilogue reads the accumulator row by row from TMEM and forms
// m_ji = max(G_ji / (||t_j|| ||z_i||), 0) and s^t_i = sqrt(sum_j m_ji^2 / M); the [M, N]
// similarity never reaches memory. The last tile of a request to finish (ticket counter,
// no waiting) runs that request's selection.
//
// Warp roles: 0 = TMA producer, 1 = TMEM owner and MMA issuer, 2..7 = squared norms of the
// 128 Z rows and the M T rows of every stage (row units spread over 192 threads, four
// independent accumulators each); 2..5 then run the epilogue (warp w reads TMEM lanes
// 32*(w%4) .. 32*(w%4)+31, i.e. those tile rows). All eight warps run the selection.

constexpr int kTileRows = kScoreTileRows;
constexpr int kChunk = 64;                     // d' columns per stage (one 128-byte swizzle row)
constexpr int kMaxStages = 8;
constexpr int kZBoxRows = 64;
constexpr int kTBoxRows = 32;
constexpr int kZStageBytes = kTileRows * kChunk * 2;
constexpr int kScoreThreads = 256;

struct ScoreLaunch {
  int stages;
  int stage_bytes;
  int tmem_cols;
  int smem_bytes;   // dynamic shared memory actually requested (for the selection)
};

__global__ void __launch_bounds__(kScoreThreads, 1)
    pre_score_kernel(const __grid_constant__ CUtensorMap tmZ, const __grid_constant__ CUtensorMap tmT,
                     const __grid_constant__ PreMeta meta, const PreArgs a, const ScoreLaunch L) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ uint32_t tmem_base_s;
  __shared__ float rinv_t[256];
  __shared__ float zsq_s[kTileRows];
  __shared__ SelShared ss;
  __shared__ int s_last;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_issued;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int sel_bytes = L.smem_bytes - (int)(smem - smem_raw);
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x;
  const int b = find_request(meta.B, tile, [&](int i) { return meta.r[i].tile_off; });
  const PreReq r = meta.r[b];
  const int row0 = (tile - r.tile_off) * kTileRows;
  const int m = r.m;
  const int nk = (a.d + kChunk - 1) / kChunk;
  const int S = L.stages;
  const int nz_box = (row0 + kZBoxRows < r.n) ? 2 : 1;
  const int nt_box = (m + kTBoxRows - 1) / kTBoxRows;
  const int n_mma = (m + 15) & ~15;
  const uint32_t stage_tx = (uint32_t)(nz_box * kZBoxRows + nt_box * kTBoxRows) * kChunk * 2;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1 + 6);   // MMA commit + six norm warps
    }
    mbar_init(smem_u32(&acc_bar), 1);
    s_abort = 0;
    s_issued = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), (uint32_t)L.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  pdl_launch_dependents();   // later grids of the stream may start launching

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmZ);
      tma_prefetch_desc(&tmT);
      const uint64_t pz = l2_policy_evict_first();   // Z is streamed once
      const uint64_t pt = l2_policy_evict_last();    // T is re-read by every tile of the request
      for (int kc = 0; kc < nk; ++kc) {
        const int s = kc % S, it = kc / S;
        if (kc >= S && !mbar_wait(smem_u32(&empty_bar[s]), (it - 1) & 1, &s_abort)) {
          s_abort = 1;
          break;
        }
        const uint32_t A = sbase + s * L.stage_bytes, B = A + kZStageBytes;
        const uint32_t fb = smem_u32(&full_bar[s]);
        mbar_arrive_expect_tx(fb, stage_tx);
        const int x = kc * kChunk;
        tma_load_2d(A, &tmZ, x, r.n_off + row0, fb, pz);
        if (nz_box == 2) tma_load_2d(A + kZBoxRows * 128, &tmZ, x, r.n_off + row0 + kZBoxRows, fb, pz);
        for (int tb = 0; tb < nt_box; ++tb) tma_load_2d(B + tb * kTBoxRows * 128, &tmT, x, r.m_off + tb * kTBoxRows, fb, pt);
        s_issued = kc + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kTileRows, n_mma);
      for (int kc = 0; kc < nk; ++kc) {
        const int s = kc % S, it = kc / S;
        if (!mbar_wait(smem_u32(&full_bar[s]), it & 1, &s_abort)) {
          s_abort = 1;
          break;
        }
        tc_fence_after();
        const uint32_t A = sbase + s * L.stage_bytes, B = A + kZStageBytes;
#pragma unroll
        for (int k = 0; k < kChunk / 16; ++k)
          umma_bf16(tmem, umma_desc_sw128(A + 32 * k), umma_desc_sw128(B + 32 * k), idesc, (kc | k) != 0);
        umma_commit(smem_u32(&empty_bar[s]));   // frees the stage once these MMAs have read it
      }
      umma_commit(smem_u32(&acc_bar));          // accumulator complete (also on abort)
    }
  } else {
    // row units u = t, t + 192 (t = tid - 64; 128 + M <= 384): u < 128 is Z row u, else T row u - 128
    const int t = tid - 64;
    const int units = kTileRows + m;
    float acc[2][4];
#pragma unroll
    for (int x = 0; x < 2; ++x)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[x][j] = 0.f;
    for (int kc = 0; kc < nk; ++kc) {
      const int s = kc % S, it = kc / S;
      if (!mbar_wait(smem_u32(&full_bar[s]), it & 1, &s_abort)) {
        s_abort = 1;
        break;
      }
      const uint8_t* A = smem + s * L.stage_bytes;
#pragma unroll
      for (int x = 0; x < 2; ++x) {
        const int u = t + 192 * x;
        if (u < units) {
          // T row u - 128 sits right after the 128 Z rows of the stage
          const uint8_t* rowp = A + u * 128;
#pragma unroll
          for (int j = 0; j < 8; ++j) bf16_sq_acc8(*reinterpret_cast<const uint4*>(rowp + (swz(u, j) << 4)), acc[x]);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty_bar[s]));
    }
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      const int u = t + 192 * x;
      const float sq = (acc[x][0] + acc[x][1]) + (acc[x][2] + acc[x][3]);
      if (u < kTileRows) zsq_s[u] = sq;
      else if (u < units) rinv_t[u - kTileRows] = sq > 0.f ? 1.0f / sqrtf(sq) : 0.f;
    }
    asm volatile("bar.sync 1, 192;" ::: "memory");   // the six norm warps
  }
  if (warp >= 2 && warp < 6) {
    const int q = warp & 3;             // TMEM lane quarter of this warp
    const int row = 32 * q + lane;      // tile row owned by this thread
    const float zacc = zsq_s[row];
    bool ok = mbar_wait(smem_u32(&acc_bar), 0, &s_abort);
    ok = __all_sync(0xffffffffu, ok && !s_abort);
    tc_fence_after();
    if (ok) {
      const float rz = zacc > 0.f ? 1.0f / sqrtf(zacc) : 0.f;
      float sum = 0.f;
      for (int c0 = 0; c0 < m; c0 += 32) {
        float v[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          if (c0 + j < m) {
            const float x = fmaxf(v[j] * rinv_t[c0 + j] * rz, 0.f);
            sum = fmaf(x, x, sum);
          }
        }
      }
      if (row0 + row < r.n) a.s_t[r.n_off + row0 + row] = sqrtf(sum / (float)m);
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)L.tmem_cols);
  }
  if (s_abort) {
    // let the copies already issued land before the block's shared memory is released
    if (tid == 0) {
      const int issued = s_issued;
      const volatile int no_abort = 0;
      for (int kc = issued - S > 0 ? issued - S : 0; kc < issued; ++kc)
        mbar_wait(smem_u32(&full_bar[kc % S]), (kc / S) & 1, &no_abort, 500000000ull);
      atomicOr(a.err, 1u);
    }
    return;
  }

  if (a.action == kActScores) return;
  // last finished tile of this request runs its selection
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned ntiles = (unsigned)((r.n + kTileRows - 1) / kTileRows);
    const unsigned prev = atomicAdd(&a.counters[b], 1u);
    s_last = (prev == ntiles - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) a.counters[b] = 0u;
  select_request(a, r, b, smem, sel_bytes, ss, a.mode == kModeFused, a.action == kActSelect);
}

// One CTA per request: selection from scores already in memory.
__global__ void __launch_bounds__(512) pre_select_kernel(const __grid_constant__ PreMeta meta,
                                                         const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  const PreReq r = meta.r[blockIdx.x];
  select_request(a, r, blockIdx.x, smem, smem_bytes, ss, a.mode == kModeFused && !a.s_fused_given, true);
}

// One CTA per request: the saliency side of the selection (inputs only), run ahead of the
// scoring grid so that the last tile of a request only ranks textual relevance.
__global__ void __launch_bounds__(512) pre_saliency_kernel(const __grid_constant__ PreMeta meta,
                                                           const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  pdl_launch_dependents();
  const int b = blockIdx.x;
  const PreReq r = meta.r[b];
  const bool in_smem = (size_t)r.n * 4 + 16 <= (size_t)smem_bytes;
  const size_t gbase = ((size_t)r.n_off + 4 * (size_t)b + 3) & ~(size_t)3;
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + gbase;
  const int4 rule = saliency_prepare(a, r, keys, ss);
  if (threadIdx.x == 0) a.sal[b] = rule;
}

// ------------------------------------------------------------------ row gather
//
// One warp per destination row: dst[row] = src[off + idx[row]] for every head segment,
// 16-byte vector loads with eight in flight per lane.
__global__ void __launch_bounds__(256) gather_rows_kernel(const __grid_constant__ GatherMeta gm) {
  pdl_wait();   // the indices come from the preceding grids
  const GatherJob& j = gm.job[blockIdx.y];
  const GatherTable& t = gm.t[j.tab];
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= j.rows) return;
  const int b = find_request(t.B, row, [&](int i) { return t.dst_off[i]; });
  const int li = __ldcg(j.idx + row);
  if (li < 0 || li >= t.src_rows[b]) return;
  const long long srow = (long long)t.src_off[b] + li;
  const int U = j.row_bytes >> 4;
  const int total = U * j.heads;
  const uint8_t* src = j.src + srow * j.src_tok;
  uint8_t* dst = j.dst + (long long)row * j.dst_tok;
  for (int x0 = lane; x0 < total; x0 += 256) {
    uint4 v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int x = x0 + 32 * q;
      if (x < total) {
        const int h = x / U, u = x - h * U;
        v[q] = __ldg(reinterpret_cast<const uint4*>(src + h * j.src_head + u * 16));
      }
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int x = x0 + 32 * q;
      if (x < total) {
        const int h = x / U, u = x - h * U;
        *reinterpret_cast<uint4*>(dst + h * j.dst_head + u * 16) = v[q];
      }
    }
  }
}

// ------------------------------------------------------------------ host-side launchers

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

// Tensor map of a [rows, cols] bf16 matrix (row stride in elements), boxes of
// box_rows x 64 columns, 128-byte swizzle, zero fill outside the matrix.
static cudaError_t make_tmap(CUtensorMap* tm, const void* base, long long rows, int cols, long long stride,
                             int box_rows) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)(rows > 0 ? rows : 1)};
  const cuuint64_t strides[1] = {(cuuint64_t)stride * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kChunk, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult res = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t launch_pre_score(const PreMeta& meta, const PreArgs& a, int max_m, int max_n, long long z_rows,
                             long long t_rows_total, cudaStream_t st) {
  if (meta.total_tiles == 0) return cudaSuccess;
  const int t_rows = ((max_m + kTBoxRows - 1) / kTBoxRows) * kTBoxRows;
  ScoreLaunch L;
  L.stage_bytes = kZStageBytes + t_rows * 128;
  int stages = (106 * 1024 - 1024) / L.stage_bytes;   // two CTAs per SM
  if (stages < 3) stages = (200 * 1024) / L.stage_bytes;   // one CTA per SM, deeper ring
  L.stages = stages > kMaxStages ? kMaxStages : (stages < 2 ? 2 : stages);
  int cols = 32;
  while (cols < ((max_m + 15) & ~15)) cols <<= 1;
  L.tmem_cols = cols;
  int smem = L.stages * L.stage_bytes + 1024;
  const int sel = (int)((size_t)max_n * 5 + 16) + 1024;
  if (a.action != kActScores && sel > smem && sel <= 200 * 1024) smem = sel;
  L.smem_bytes = smem;
  CUtensorMap tmZ, tmT;
  cudaError_t e = make_tmap(&tmZ, a.Z, z_rows, a.d, a.z_stride, kZBoxRows);
  if (e != cudaSuccess) return e;
  e = make_tmap(&tmT, a.T, t_rows_total, a.d, a.t_stride, kTBoxRows);
  if (e != cudaSuccess) return e;
  e = ensure_dynamic_smem(pre_score_kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(pre_score_kernel, dim3(meta.total_tiles), dim3(kScoreThreads), smem, st, a.sal_ready != 0,
                       tmZ, tmT, meta, a, L);
}

cudaError_t launch_pre_saliency(const PreMeta& meta, const PreArgs& a, int max_n, cudaStream_t st) {
  if (meta.B == 0) return cudaSuccess;
  int smem = (int)((size_t)max_n * 4 + 16);
  if (smem > 160 * 1024) smem = 0;   // keys stay in the global scratch
  cudaError_t e = ensure_dynamic_smem(pre_saliency_kernel, smem);
  if (e != cudaSuccess) return e;
  pre_saliency_kernel<<<meta.B, 512, smem, st>>>(meta, a, smem);
  return cudaGetLastError();
}

cudaError_t launch_pre_select(const PreMeta& meta, const PreArgs& a, int max_n, cudaStream_t st) {
  if (meta.B == 0) return cudaSuccess;
  int smem = (int)((size_t)max_n * 5 + 16);
  if (smem > 160 * 1024) smem = 0;   // keys stay in the global scratch
  cudaError_t e = ensure_dynamic_smem(pre_select_kernel, smem);
  if (e != cudaSuccess) return e;
  pre_select_kernel<<<meta.B, 512, smem, st>>>(meta, a, smem);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherMeta& gm, cudaStream_t st, bool pdl) {
  int rows = 0;
  for (int i = 0; i < gm.njobs; ++i) rows = rows > gm.job[i].rows ? rows : gm.job[i].rows;
  if (rows == 0 || gm.njobs == 0) return cudaSuccess;
  return launch_kernel(gather_rows_kernel, dim3((rows + 7) / 8, gm.njobs), dim3(256), 0, st, pdl, gm);
}

}  // namespace trevs
