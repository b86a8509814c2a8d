// Stage 2 (in-LLM at layer l*, Sec. 4.2): text-to-vision attention statistics, head
// variance (Eq. 8), high-variance head set H*, token scores (Eq. 9), TopK and compaction.
#include "in_llm.cuh"

namespace trevs {

constexpr int kQB = kTextBlockRows;
constexpr int kKB = kKeyBlock;
constexpr int kDh = 128;       // head width
constexpr int kRowBytes = kDh * 2;

// Row q of a [rows][128] bf16 tile: 16 chunks of 16 bytes, XOR-swizzled on the low 3 bits.
__device__ __forceinline__ uint32_t tile_addr(uint32_t base, int row, int chunk) {
  return base + row * kRowBytes + ((chunk ^ (row & 7)) << 4);
}

__device__ __forceinline__ void load_rows(uint32_t dst, const __nv_bfloat16* base, long long row_stride,
                                          int row0, int rows, int valid, int tid, int nthr) {
  for (int idx = tid; idx < rows * 16; idx += nthr) {
    const int rr = idx >> 4, c = idx & 15;
    const bool ok = row0 + rr < valid;
    const void* src = ok ? (const void*)(base + (long long)(row0 + rr) * row_stride + c * 8) : (const void*)base;
    cp_async16(tile_addr(dst, rr, c), src, ok ? 16 : 0);
  }
}

// A fragments of a 16 x 128 tile for all 8 k-steps.
__device__ __forceinline__ void load_afrag(uint32_t qs, int lane, uint32_t (&af)[8][4]) {
#pragma unroll
  for (int ks = 0; ks < 8; ++ks)
    ldmatrix_x4(tile_addr(qs, lane & 15, 2 * ks + (lane >> 4)), af[ks][0], af[ks][1], af[ks][2], af[ks][3]);
}

// acc[2][4] = Q_tile(16 x 128) . K_rows(key0 .. key0+15)^T
__device__ __forceinline__ void qk_16x16(const uint32_t (&af)[8][4], uint32_t ks_base, int key0, int lane,
                                         float (&acc)[2][4]) {
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int mi = lane >> 3;
    const int rr = key0 + 8 * (mi >> 1) + (lane & 7), c = 2 * ks + (mi & 1);
    uint32_t b0, b1, b2, b3;
    ldmatrix_x4(tile_addr(ks_base, rr, c), b0, b1, b2, b3);
    mma_bf16_16816(acc[0], af[ks], b0, b1);
    mma_bf16_16816(acc[1], af[ks], b2, b3);
  }
}

// ------------------------------------------------------------------ attention statistics
//
// Block (request, head h, 16-row block of text queries): logits Q_h . K_g^T * scale for all
// K1 keys into shared memory (tensor cores), then per row the max, the sum of exp and the
// two-pass variance of the softmax row about its mean 1/K1 (Eq. 8). The last block of a
// request averages the row variances into u_h.
__global__ void __launch_bounds__(128) in_head_stats_kernel(const __grid_constant__ InMeta meta,
                                                            const InArgs a, int k1_ld) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_last;
  if (!a.overlap) pdl_wait();   // Q, K may come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].hs_off; });
  const InReq r = meta.r[b];
  const int nqb = (r.l + kQB - 1) / kQB;
  const int t = blockIdx.x - r.hs_off;
  const int h = t / nqb, qb = t - h * nqb;
  const int g = (h * a.Hkv) / a.Hq;
  const int q0 = qb * kQB;

  uint8_t* qs = smem;                              // 16 x 256 B
  uint8_t* kbuf = smem + kQB * kRowBytes;          // 2 x 64 x 256 B
  float* lg = reinterpret_cast<float*>(kbuf + 2 * kKB * kRowBytes);   // [16][k1_ld]
  const uint32_t qs_a = smem_u32(qs), kb_a = smem_u32(kbuf);

  const __nv_bfloat16* Qb = a.Q + (long long)r.l_off * a.q_ts + (long long)h * a.q_hs;
  const __nv_bfloat16* Kb = a.K + (long long)r.k1_off * a.k_ts + (long long)g * a.k_hs;
  const int nkc = (r.k1 + kKB - 1) / kKB;

  load_rows(qs_a, Qb, a.q_ts, q0, kQB, r.l, tid, 128);
  load_rows(kb_a, Kb, a.k_ts, 0, kKB, r.k1, tid, 128);
  cp_async_commit();
  uint32_t af[8][4];
  for (int kc = 0; kc < nkc; ++kc) {
    if (kc + 1 < nkc) load_rows(kb_a + ((kc + 1) & 1) * kKB * kRowBytes, Kb, a.k_ts, (kc + 1) * kKB, kKB, r.k1, tid, 128);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (kc == 0) load_afrag(qs_a, lane, af);
    float acc[2][4];
    qk_16x16(af, kb_a + (kc & 1) * kKB * kRowBytes, 16 * warp, lane, acc);
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      const int key = kc * kKB + 16 * warp + 8 * nt + 2 * (lane & 3);
      const int row = lane >> 2;
      *reinterpret_cast<float2*>(lg + row * k1_ld + key) = make_float2(acc[nt][0] * a.scale, acc[nt][1] * a.scale);
      *reinterpret_cast<float2*>(lg + (row + 8) * k1_ld + key) = make_float2(acc[nt][2] * a.scale, acc[nt][3] * a.scale);
    }
    __syncthreads();
  }

  const int k1 = r.k1;
  const float mean = 1.0f / (float)k1;
  for (int rr = warp; rr < kQB; rr += 4) {
    const int q = q0 + rr;
    if (q >= r.l) break;
    float* row = lg + rr * k1_ld;
    float mx = -INFINITY;
    for (int i = lane; i < k1; i += 32) mx = fmaxf(mx, row[i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
    for (int i = lane; i < k1; i += 32) {
      const float e = expf(row[i] - mx);
      row[i] = e;
      sum += e;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float inv = 1.0f / sum;
    float v = 0.f;
    for (int i = lane; i < k1; i += 32) {
      const float dlt = row[i] * inv - mean;
      v = fmaf(dlt, dlt, v);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) {
      const long long o = (long long)h * a.stats_ld + r.l_off + q;
      a.row_stats[o] = make_float2(mx, inv);
      a.row_var[o] = v / (float)k1;
    }
  }

  // completion of this grid implies completion of the preceding one
  if (a.overlap) pdl_wait();
  if (!a.hs_finalize) return;
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned prev = atomicAdd(&a.cnt_hs[b], 1u);
    s_last = (prev == (unsigned)(a.Hq * nqb) - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) a.cnt_hs[b] = 0u;
  for (int hh = tid; hh < a.Hq; hh += 128) {
    const float* rv = a.row_var + (long long)hh * a.stats_ld + r.l_off;
    float s = 0.f;
    for (int q = 0; q < r.l; ++q) s += __ldcg(rv + q);
    a.u[(long long)b * a.u_ld + hh] = s / (float)r.l;
  }
  if (a.zero_p)
    for (int i = tid; i < r.k1; i += 128) a.p_bits[r.k1_off + i] = 0u;
}

// ------------------------------------------------------------------ token scores
//
// Block (request, 16-row text block, 64-key block): for each head of H* in ascending order
// recompute the logits on the tensor cores, turn them into attention with the row
// statistics, and accumulate the head sum; the max over the block's text rows of the head
// mean (Eq. 9) is merged across text blocks with an integer atomicMax on the (non-negative)
// float bits, which is exact and order independent. The last block of a request selects
// TopK(p, K2) and writes H*.
__global__ void __launch_bounds__(128) in_token_score_kernel(const __grid_constant__ InMeta meta,
                                                             const InArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  __shared__ int s_heads[kMaxHeads];
  __shared__ int s_sel[kMaxHeads];
  __shared__ int s_nh, s_last;
  pdl_wait();   // u, row statistics and the cleared p come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].ts_off; });
  const InReq r = meta.r[b];
  const int nib = (r.k1 + kKB - 1) / kKB;
  const int t = blockIdx.x - r.ts_off;
  const int qb = t / nib, ib = t - qb * nib;
  const int q0 = qb * kQB, i0 = ib * kKB;

  // H*: the n_keep heads of largest u, ties to the lower head
  const float* u = a.u + (long long)b * a.u_ld;
  for (int hh = tid; hh < a.Hq; hh += 128) {
    const float uh = __ldcg(u + hh);
    int rank = 0;
    for (int x = 0; x < a.Hq; ++x) {
      const float ux = __ldcg(u + x);
      rank += (ux > uh) || (ux == uh && x < hh);
    }
    s_sel[hh] = rank < a.n_keep;
  }
  __syncthreads();
  if (tid == 0) {  // ascending list; at most n_keep entries even if u holds NaN
    int cnt = 0;
    for (int hh = 0; hh < a.Hq && cnt < a.n_keep; ++hh)
      if (s_sel[hh]) s_heads[cnt++] = hh;
    s_nh = cnt;
  }
  __syncthreads();

  uint8_t* qs = smem;
  uint8_t* ks = smem + kQB * kRowBytes;
  const uint32_t qs_a = smem_u32(qs), ks_a = smem_u32(ks);
  float psum[2][4];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) psum[i][j] = 0.f;
  const int ra = q0 + (lane >> 2), rb = ra + 8;
  int g_loaded = -1;
  for (int hi = 0; hi < s_nh; ++hi) {
    const int h = s_heads[hi];
    const int g = (h * a.Hkv) / a.Hq;
    load_rows(qs_a, a.Q + (long long)r.l_off * a.q_ts + (long long)h * a.q_hs, a.q_ts, q0, kQB, r.l, tid, 128);
    if (g != g_loaded)
      load_rows(ks_a, a.K + (long long)r.k1_off * a.k_ts + (long long)g * a.k_hs, a.k_ts, i0, kKB, r.k1, tid, 128);
    g_loaded = g;
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    uint32_t af[8][4];
    load_afrag(qs_a, lane, af);
    float acc[2][4];
    qk_16x16(af, ks_a, 16 * warp, lane, acc);
    const long long so = (long long)h * a.stats_ld + r.l_off;
    const float2 sa = ra < r.l ? __ldcg(a.row_stats + so + ra) : make_float2(0.f, 0.f);
    const float2 sb = rb < r.l ? __ldcg(a.row_stats + so + rb) : make_float2(0.f, 0.f);
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      psum[nt][0] += expf(acc[nt][0] * a.scale - sa.x) * sa.y;
      psum[nt][1] += expf(acc[nt][1] * a.scale - sa.x) * sa.y;
      psum[nt][2] += expf(acc[nt][2] * a.scale - sb.x) * sb.y;
      psum[nt][3] += expf(acc[nt][3] * a.scale - sb.x) * sb.y;
    }
    __syncthreads();
  }
  // rows past L contribute nothing; attention is positive, so 0 never wins the max
  const float inv_nh = s_nh > 0 ? 1.0f / (float)s_nh : 0.f;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    float m0 = fmaxf(ra < r.l ? psum[nt][0] : 0.f, rb < r.l ? psum[nt][2] : 0.f);
    float m1 = fmaxf(ra < r.l ? psum[nt][1] : 0.f, rb < r.l ? psum[nt][3] : 0.f);
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, o));
      m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
    }
    if (lane < 4) {
      const int i = i0 + 16 * warp + 8 * nt + 2 * lane;
      if (i < r.k1) atomicMax(a.p_bits + r.k1_off + i, __float_as_uint(m0 * inv_nh));
      if (i + 1 < r.k1) atomicMax(a.p_bits + r.k1_off + i + 1, __float_as_uint(m1 * inv_nh));
    }
  }

  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int nqb = (r.l + kQB - 1) / kQB;
    const unsigned prev = atomicAdd(&a.cnt_ts[b], 1u);
    s_last = (prev == (unsigned)(nqb * nib) - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) a.cnt_ts[b] = 0u;
  if (a.heads_out)
    for (int x = tid; x < s_nh; x += 128) a.heads_out[(long long)b * a.n_keep + x] = s_heads[x];
  if (r.k2 <= 0) return;
  const int n = r.k1;
  const bool in_smem = (size_t)n * 5 <= (size_t)smem_bytes;
  const size_t gbase = ((size_t)r.k1_off + 4 * (size_t)b + 3) & ~(size_t)3;   // 16-byte aligned
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + gbase;
  uint8_t* flags = in_smem ? smem + (size_t)n * 4 : a.flags + gbase;
  for (int i = tid; i < n; i += 128) flags[i] = 0;
  uint32_t lo, hi, tau;
  int need, n_eq;
  block_fill_keys(keys, reinterpret_cast<const float*>(a.p_bits + r.k1_off), n,
                  [&](float x, int) { return score_key(x); }, ss, lo, hi);
  block_kth_largest(keys, n, r.k2, ss, lo, hi, tau, need, n_eq);
  block_mark_selected(keys, n, tau, need, n_eq, flags, ss);
  block_compact_flags(flags, n, a.kept_local + r.k2_off, ss);
}

// ------------------------------------------------------------------ host-side launchers

int in_head_stats_ld(int max_k1) { return ((max_k1 + kKB - 1) / kKB) * kKB + 8; }

cudaError_t launch_in_head_stats(const InMeta& meta, const InArgs& a, int max_k1, cudaStream_t st) {
  if (meta.total_hs == 0) return cudaSuccess;
  const int ld = in_head_stats_ld(max_k1);
  const int smem = kQB * kRowBytes + 2 * kKB * kRowBytes + kQB * ld * 4;
  cudaError_t e = ensure_dynamic_smem(in_head_stats_kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(in_head_stats_kernel, dim3(meta.total_hs), dim3(128), smem, st, true, meta, a, ld);
}

cudaError_t launch_in_token_score(const InMeta& meta, const InArgs& a, int max_k1, cudaStream_t st) {
  if (meta.total_ts == 0) return cudaSuccess;
  int smem = kQB * kRowBytes + kKB * kRowBytes;
  if (max_k1 * 5 > smem) smem = max_k1 * 5;
  cudaError_t e = ensure_dynamic_smem(in_token_score_kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(in_token_score_kernel, dim3(meta.total_ts), dim3(128), smem, st, true, meta, a, smem);
}

}  // namespace trevs
