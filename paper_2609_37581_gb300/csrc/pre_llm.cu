// Stage 1 (pre-LLM, Sec. 4.1): textual-relevance scores (Eq. 4-5), selection (Sec. 3.1 ratio
// split or Eq. 6-7 fused score) and gather of the kept feature rows.
#include "pre_llm.cuh"

namespace trevs {

// ------------------------------------------------------------------ scoring contraction
//
// One CTA scores a tile of 64 visual rows of one request against all M text rows of that
// request: G = Z_tile . T^T on the tensor cores (bf16 x bf16 -> fp32), while the same
// shared-memory stages feed the fp32 squared norms ||z_i||^2 and ||t_j||^2. The epilogue
// forms m_ji = max(G_ji / (||t_j|| ||z_i||), 0) and s^t_i = sqrt(sum_j m_ji^2 / M) in
// registers; the [M, N] similarity never reaches memory. The last tile of a request to
// finish (ticket counter, no waiting) runs that request's selection.

constexpr int kTileRows = 64;
constexpr int kChunk = 64;         // d' columns per pipeline stage
constexpr int kStages = 3;
constexpr int kZStageBytes = kTileRows * kChunk * 2;

template <int NT>  // text columns padded to 8*NT (NT even, 8*NT <= 256)
__global__ void __launch_bounds__(128) pre_score_kernel(const __grid_constant__ PreMeta meta,
                                                        const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  __shared__ float zsq_s[kTileRows];
  __shared__ float rinv_t[8 * NT];
  __shared__ int s_last;

  constexpr int kMRows = 8 * NT;
  constexpr int kTStageBytes = kMRows * kChunk * 2;
  constexpr int kStageBytes = kZStageBytes + kTStageBytes;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int tile = blockIdx.x;
  const int b = find_request(meta.B, tile, [&](int i) { return meta.r[i].tile_off; });
  const PreReq r = meta.r[b];
  const int row0 = (tile - r.tile_off) * kTileRows;
  const int m = r.m;
  const int nk = (a.d + kChunk - 1) / kChunk;
  const __nv_bfloat16* Zb = a.Z + (long long)r.n_off * a.z_stride;
  const __nv_bfloat16* Tb = a.T + (long long)r.m_off * a.t_stride;

  auto load_stage = [&](int st, int kc) {
    uint8_t* zs = smem + st * kStageBytes;
    uint8_t* ts = zs + kZStageBytes;
    const int kbase = kc * kChunk;
#pragma unroll
    for (int it = 0; it < (kTileRows * 8) / 128; ++it) {
      int idx = tid + it * 128;
      int rr = idx >> 3, c = idx & 7;
      int grow = row0 + rr, col = kbase + c * 8;
      bool ok = grow < r.n && col < a.d;
      const void* src = ok ? (const void*)(Zb + (long long)grow * a.z_stride + col) : (const void*)a.Z;
      cp_async16(smem_u32(zs + rr * 128 + swz(rr, c) * 16), src, ok ? 16 : 0);
    }
    for (int idx = tid; idx < kMRows * 8; idx += 128) {
      int rr = idx >> 3, c = idx & 7;
      int col = kbase + c * 8;
      bool ok = rr < m && col < a.d;
      const void* src = ok ? (const void*)(Tb + (long long)rr * a.t_stride + col) : (const void*)a.T;
      cp_async16(smem_u32(ts + rr * 128 + swz(rr, c) * 16), src, ok ? 16 : 0);
    }
  };

  float acc[NT][4];
#pragma unroll
  for (int i = 0; i < NT; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  float zacc = 0.f, tacc0 = 0.f, tacc1 = 0.f;

#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < nk) load_stage(s, s);
    cp_async_commit();
  }
  for (int kc = 0; kc < nk; ++kc) {
    cp_async_wait<kStages - 2>();
    __syncthreads();
    const int nxt = kc + kStages - 1;
    if (nxt < nk) load_stage(nxt % kStages, nxt);
    cp_async_commit();

    const uint8_t* zs = smem + (kc % kStages) * kStageBytes;
    const uint8_t* ts = zs + kZStageBytes;
    {  // ||z_i||^2: two threads per row, four 16-byte chunks each
      const int rr = tid >> 1, h = tid & 1;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        zacc += bf16_sq_sum8(*reinterpret_cast<const uint4*>(zs + rr * 128 + swz(rr, 4 * h + j) * 16));
    }
    if (tid < m && tid < kMRows) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        tacc0 += bf16_sq_sum8(*reinterpret_cast<const uint4*>(ts + tid * 128 + swz(tid, j) * 16));
    }
    if (kMRows > 128 && tid + 128 < m && tid + 128 < kMRows) {
      const int rr = tid + 128;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        tacc1 += bf16_sq_sum8(*reinterpret_cast<const uint4*>(ts + rr * 128 + swz(rr, j) * 16));
    }
#pragma unroll
    for (int ks = 0; ks < kChunk / 16; ++ks) {
      uint32_t af[4];
      {
        const int rr = 16 * warp + (lane & 15), c = 2 * ks + (lane >> 4);
        ldmatrix_x4(smem_u32(zs + rr * 128 + swz(rr, c) * 16), af[0], af[1], af[2], af[3]);
      }
#pragma unroll
      for (int p = 0; p < NT / 2; ++p) {
        if (16 * p < m) {
          const int mi = lane >> 3;
          const int rr = 16 * p + 8 * (mi >> 1) + (lane & 7), c = 2 * ks + (mi & 1);
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4(smem_u32(ts + rr * 128 + swz(rr, c) * 16), b0, b1, b2, b3);
          mma_bf16_16816(acc[2 * p], af, b0, b1);
          mma_bf16_16816(acc[2 * p + 1], af, b2, b3);
        }
      }
    }
  }
  cp_async_wait<0>();

  zacc += __shfl_xor_sync(0xffffffffu, zacc, 1);
  if ((tid & 1) == 0) zsq_s[tid >> 1] = zacc;
  if (tid < kMRows) rinv_t[tid] = tacc0 > 0.f ? 1.0f / sqrtf(tacc0) : 0.f;
  if (kMRows > 128 && tid + 128 < kMRows) rinv_t[tid + 128] = tacc1 > 0.f ? 1.0f / sqrtf(tacc1) : 0.f;
  __syncthreads();

  {
    const int ra = 16 * warp + (lane >> 2), rb = ra + 8;
    const float za = zsq_s[ra], zb = zsq_s[rb];
    const float iza = za > 0.f ? 1.0f / sqrtf(za) : 0.f;
    const float izb = zb > 0.f ? 1.0f / sqrtf(zb) : 0.f;
    float sa = 0.f, sb = 0.f;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int j0 = 8 * nt + 2 * (lane & 3);
      if (j0 < m) {
        const float t = rinv_t[j0];
        const float ca = fmaxf(acc[nt][0] * t * iza, 0.f), cb = fmaxf(acc[nt][2] * t * izb, 0.f);
        sa = fmaf(ca, ca, sa);
        sb = fmaf(cb, cb, sb);
      }
      if (j0 + 1 < m) {
        const float t = rinv_t[j0 + 1];
        const float ca = fmaxf(acc[nt][1] * t * iza, 0.f), cb = fmaxf(acc[nt][3] * t * izb, 0.f);
        sa = fmaf(ca, ca, sa);
        sb = fmaf(cb, cb, sb);
      }
    }
    sa += __shfl_xor_sync(0xffffffffu, sa, 1);
    sa += __shfl_xor_sync(0xffffffffu, sa, 2);
    sb += __shfl_xor_sync(0xffffffffu, sb, 1);
    sb += __shfl_xor_sync(0xffffffffu, sb, 2);
    if ((lane & 3) == 0) {
      const float inv_m = 1.0f / (float)m;
      if (row0 + ra < r.n) a.s_t[r.n_off + row0 + ra] = sqrtf(sa * inv_m);
      if (row0 + rb < r.n) a.s_t[r.n_off + row0 + rb] = sqrtf(sb * inv_m);
    }
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
  select_request(a, r, smem, smem_bytes, ss, a.mode == kModeFused, a.action == kActSelect);
}

// One CTA per request: selection from scores already in memory.
__global__ void __launch_bounds__(512) pre_select_kernel(const __grid_constant__ PreMeta meta,
                                                         const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  const PreReq r = meta.r[blockIdx.x];
  select_request(a, r, smem, smem_bytes, ss, a.mode == kModeFused && !a.s_fused_given, true);
}

// ------------------------------------------------------------------ row gather
//
// One warp per destination row: dst[row] = src[off + idx[row]] for every head segment,
// 16-byte vector loads with four in flight per lane.
__global__ void __launch_bounds__(256) gather_rows_kernel(const __grid_constant__ GatherMeta gm) {
  const GatherJob& j = gm.job[blockIdx.y];
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= j.rows) return;
  const int b = find_request(gm.B, row, [&](int i) { return gm.dst_off[i]; });
  const int li = __ldg(j.idx + row);
  if (li < 0 || li >= gm.src_rows[b]) return;
  const long long srow = (long long)gm.src_off[b] + li;
  const int U = j.row_bytes >> 4;
  const int total = U * j.heads;
  const uint8_t* src = j.src + srow * j.src_tok;
  uint8_t* dst = j.dst + (long long)row * j.dst_tok;
  for (int x0 = lane; x0 < total; x0 += 128) {
    uint4 v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int x = x0 + 32 * q;
      if (x < total) {
        const int h = x / U, u = x - h * U;
        v[q] = __ldg(reinterpret_cast<const uint4*>(src + h * j.src_head + u * 16));
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int x = x0 + 32 * q;
      if (x < total) {
        const int h = x / U, u = x - h * U;
        *reinterpret_cast<uint4*>(dst + h * j.dst_head + u * 16) = v[q];
      }
    }
  }
}

// ------------------------------------------------------------------ host-side launchers

int pre_score_smem_bytes(int max_m) {
  const int nt = max_m <= 16 ? 2 : max_m <= 32 ? 4 : max_m <= 64 ? 8 : max_m <= 128 ? 16 : 32;
  return kStages * (kZStageBytes + 8 * nt * kChunk * 2);
}

cudaError_t launch_pre_score(const PreMeta& meta, const PreArgs& a, int max_m, int max_n,
                             cudaStream_t st) {
  if (meta.total_tiles == 0) return cudaSuccess;
  int smem = pre_score_smem_bytes(max_m);
  // room for the selection's keys and flags when a request fits
  const int sel = (int)((size_t)max_n * 5 + 16);
  if (a.action != kActScores && sel > smem && sel <= 160 * 1024) smem = sel;
  const int nt = max_m <= 16 ? 2 : max_m <= 32 ? 4 : max_m <= 64 ? 8 : max_m <= 128 ? 16 : 32;
  const dim3 grid(meta.total_tiles), block(128);
#define TREVS_LAUNCH_SCORE(NT_)                                                                \
  case NT_: {                                                                                  \
    cudaError_t e = ensure_dynamic_smem(pre_score_kernel<NT_>, smem);                          \
    if (e != cudaSuccess) return e;                                                            \
    pre_score_kernel<NT_><<<grid, block, smem, st>>>(meta, a, smem);                           \
    break;                                                                                     \
  }
  switch (nt) {
    TREVS_LAUNCH_SCORE(2)
    TREVS_LAUNCH_SCORE(4)
    TREVS_LAUNCH_SCORE(8)
    TREVS_LAUNCH_SCORE(16)
    TREVS_LAUNCH_SCORE(32)
  }
#undef TREVS_LAUNCH_SCORE
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

cudaError_t launch_gather(const GatherMeta& gm, cudaStream_t st) {
  int rows = 0;
  for (int i = 0; i < gm.njobs; ++i) rows = rows > gm.job[i].rows ? rows : gm.job[i].rows;
  if (rows == 0 || gm.njobs == 0) return cudaSuccess;
  gather_rows_kernel<<<dim3((rows + 7) / 8, gm.njobs), 256, 0, st>>>(gm);
  return cudaGetLastError();
}

}  // namespace trevs
