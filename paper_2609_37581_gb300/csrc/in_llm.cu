// Stage 2 (in-LLM at layer l*, Sec. 4.2): text-to-vision attention statistics, head
// variance (Eq. 8), high-variance head set H*, token scores (Eq. 9), TopK and compaction.
#include "in_llm.cuh"

namespace trevs {

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

// A fragments of the 16 x 128 m-tile starting at `row0` of a tile, for all 8 k-steps.
__device__ __forceinline__ void load_afrag(uint32_t qs, int row0, int lane, uint32_t (&af)[8][4]) {
#pragma unroll
  for (int ks = 0; ks < 8; ++ks)
    ldmatrix_x4(tile_addr(qs, row0 + (lane & 15), 2 * ks + (lane >> 4)), af[ks][0], af[ks][1], af[ks][2],
                af[ks][3]);
}

// acc[NT][4] = Q m-tile (16 x 128) . K_rows(key0 .. key0 + 8*NT - 1)^T, NT even.
template <int NT>
__device__ __forceinline__ void qk_tile(const uint32_t (&af)[8][4], uint32_t ks_base, int key0, int lane,
                                        float (&acc)[NT][4]) {
#pragma unroll
  for (int i = 0; i < NT; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int p = 0; p < NT / 2; ++p) {
      const int mi = lane >> 3;
      const int rr = key0 + 16 * p + 8 * (mi >> 1) + (lane & 7), c = 2 * ks + (mi & 1);
      uint32_t b0, b1, b2, b3;
      ldmatrix_x4(tile_addr(ks_base, rr, c), b0, b1, b2, b3);
      mma_bf16_16816(acc[2 * p], af[ks], b0, b1);
      mma_bf16_16816(acc[2 * p + 1], af[ks], b2, b3);
    }
  }
}

// ------------------------------------------------------------------ attention statistics
//
// Block (request, head h, chunk of QC = 16*MT text rows): logits Q_h . K_g^T * scale for all
// K1 keys into shared memory (tensor cores; K streamed once in 64-key chunks through a
// two-buffer cp.async ring), then per row the max, the sum of exp and the two-pass
// variance of the softmax row about its mean 1/K1 (Eq. 8). The last block of a request
// averages the row variances into u_h and clears p for the token-score pass.
// Warp w computes m-tile (w % MT) against key slice (w / MT) of each chunk.
template <int MT>
__global__ void __launch_bounds__(128) in_head_stats_kernel(const __grid_constant__ InMeta meta,
                                                            const InArgs a, int k1_ld) {
  constexpr int QC = 16 * MT;
  constexpr int KW = 16 * MT;          // keys per warp in a 64-key chunk
  constexpr int NT = KW / 8;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_last;
  if (!a.overlap && !a.independent) pdl_wait();   // Q, K may come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].hs_off; });
  const InReq r = meta.r[b];
  const int nqc = (r.l + QC - 1) / QC;
  const int t = blockIdx.x - r.hs_off;
  const int h = t / nqc, qc = t - h * nqc;
  const int g = (h * a.Hkv) / a.Hq;
  const int q0 = qc * QC;

  uint8_t* qs = smem;                              // QC x 256 B
  uint8_t* kbuf = smem + QC * kRowBytes;           // 2 x 64 x 256 B
  float* lg = reinterpret_cast<float*>(kbuf + 2 * kKB * kRowBytes);   // [QC][k1_ld]
  const uint32_t qs_a = smem_u32(qs), kb_a = smem_u32(kbuf);

  const __nv_bfloat16* Qb = a.Q + (long long)r.l_off * a.q_ts + (long long)h * a.q_hs;
  const __nv_bfloat16* Kb = a.K + (long long)r.k1_off * a.k_ts + (long long)g * a.k_hs;
  const int nkc = (r.k1 + kKB - 1) / kKB;
  const int mt = warp % MT, kslice = warp / MT;
  const float sc = a.scale * 1.4426950408889634f;   // logits in log2 units: exp(x) = exp2(x * log2 e)

  load_rows(qs_a, Qb, a.q_ts, q0, QC, r.l, tid, 128);
  load_rows(kb_a, Kb, a.k_ts, 0, kKB, r.k1, tid, 128);
  cp_async_commit();
  uint32_t af[8][4];
  for (int kc = 0; kc < nkc; ++kc) {
    if (kc + 1 < nkc) load_rows(kb_a + ((kc + 1) & 1) * kKB * kRowBytes, Kb, a.k_ts, (kc + 1) * kKB, kKB, r.k1, tid, 128);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (kc == 0) load_afrag(qs_a, 16 * mt, lane, af);
    float acc[NT][4];
    qk_tile<NT>(af, kb_a + (kc & 1) * kKB * kRowBytes, kslice * KW, lane, acc);
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int key = kc * kKB + kslice * KW + 8 * nt + 2 * (lane & 3);
      const int row = 16 * mt + (lane >> 2);
      *reinterpret_cast<float2*>(lg + row * k1_ld + key) = make_float2(acc[nt][0] * sc, acc[nt][1] * sc);
      *reinterpret_cast<float2*>(lg + (row + 8) * k1_ld + key) = make_float2(acc[nt][2] * sc, acc[nt][3] * sc);
    }
    __syncthreads();
  }

  // row statistics, TPR threads per row (all rows of the chunk in parallel)
  constexpr int TPR = 128 / QC;
  __shared__ float s_inv[64];
  __shared__ float s_mean[64];
  const int k1 = r.k1;
  {
    const int rr = tid / TPR, sub = tid % TPR;
    float* row = lg + rr * k1_ld;
    // full-sequence variant: the row's non-visual mass joins the denominator (log2 units)
    float other = -INFINITY;
    if (a.lse && q0 + rr < r.l)
      other = __ldg(a.lse + (long long)h * a.lse_hs + (long long)(r.l_off + q0 + rr) * a.lse_rs) *
              1.4426950408889634f;
    float mx = -INFINITY;
#pragma unroll 4
    for (int i = sub; i < k1; i += TPR) mx = fmaxf(mx, row[i]);
#pragma unroll
    for (int o = 1; o < TPR; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    mx = fmaxf(mx, other);
    float sum = 0.f;
#pragma unroll 4
    for (int i = sub; i < k1; i += TPR) {
      const float e = exp2f(row[i] - mx);
      row[i] = e;
      sum += e;
    }
#pragma unroll
    for (int o = 1; o < TPR; o <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (sub == 0) {
      const float tot = sum + exp2f(other - mx);   // + 0 without the variant
      s_inv[rr] = 1.0f / tot;
      // Eq. 8 takes the variance about the row's mean: 1 / K1, or its visual mass / K1
      s_mean[rr] = a.lse ? (sum / tot) / (float)k1 : 1.0f / (float)k1;
    }
  }
  __syncthreads();
  // A[h][q][i] = e / sum, written along i by whole warps, and the two-pass variance of the
  // row about its mean (Eq. 8)
  {
    const int rows = min(QC, r.l - q0);
    float* A = a.attn + r.attn_off + ((long long)h * r.l + q0) * k1;
    for (int rr = warp; rr < rows; rr += 4) {
      const float inv = s_inv[rr];
      const float mean = s_mean[rr];
      const float* row = lg + rr * k1_ld;
      float* out = A + (long long)rr * k1;
      float v = 0.f;
#pragma unroll 2
      for (int i = lane; i < k1; i += 32) {
        const float p = row[i] * inv;
        out[i] = p;
        const float dlt = p - mean;
        v = fmaf(dlt, dlt, v);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) a.row_var[(long long)h * a.stats_ld + r.l_off + q0 + rr] = v / (float)k1;
    }
  }

  // completion of this grid implies completion of the preceding one
  if (a.overlap && !a.independent) pdl_wait();
  if (!a.hs_finalize) return;
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned prev = atomicAdd(&a.cnt_hs[b], 1u);
    s_last = (prev == (unsigned)(a.Hq * nqc) - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) a.cnt_hs[b] = 0u;
  // u_h = mean over text rows of the row variances: one warp per head, lanes over rows
  for (int hh = warp; hh < a.Hq; hh += 4) {
    const float* rv = a.row_var + (long long)hh * a.stats_ld + r.l_off;
    float s = 0.f;
    for (int q = lane; q < r.l; q += 32) s += __ldcg(rv + q);
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) a.u[(long long)b * a.u_ld + hh] = s / (float)r.l;
  }
  if (a.zero_p)
    for (int i = tid; i < r.k1; i += 128) a.p_bits[r.k1_off + i] = 0u;
}

// ------------------------------------------------------------------ token scores
//
// Block (request, 16-row text chunk, 64-key block): for each head of H* in ascending order
// sum the stored attention probabilities (Eq. 9, head mean), then take the max over the
// chunk's text rows; chunks merge with an integer atomicMax on the (non-negative) float
// bits, which is exact and order independent. Thread t owns key t % 64 and rows
// t / 64, t / 64 + 2, ...; every load is a 256-byte row segment. The last block of a
// request selects TopK(p, K2) and writes H*.
__global__ void __launch_bounds__(128) in_token_score_kernel(const __grid_constant__ InMeta meta,
                                                             const InArgs a, int smem_bytes) {
  constexpr int QC = kScoreTextRows;
  constexpr int RPT = QC / 2;         // rows per thread
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  __shared__ int s_heads[kMaxHeads];
  __shared__ int s_sel[kMaxHeads];
  __shared__ float s_half[kKB];
  __shared__ int s_nh, s_last;
  pdl_wait();   // u, the attention probabilities and the cleared p come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].ts_off; });
  const InReq r = meta.r[b];
  const int nib = (r.k1 + kKB - 1) / kKB;
  const int t = blockIdx.x - r.ts_off;
  const int qc = t / nib, ib = t - qc * nib;
  const int q0 = qc * QC, i0 = ib * kKB;

  // H*: the n_keep heads of largest u, ties to the lower head
  __shared__ float s_u[kMaxHeads];
  const float* u = a.u + (long long)b * a.u_ld;
  for (int hh = tid; hh < a.Hq; hh += 128) s_u[hh] = __ldcg(u + hh);
  __syncthreads();
  for (int hh = tid; hh < a.Hq; hh += 128) {
    const float uh = s_u[hh];
    int rank = 0;
    for (int x = 0; x < a.Hq; ++x) {
      const float ux = s_u[x];
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
  const int nh = s_nh;

  const int key = i0 + (tid & (kKB - 1));
  const int rbase = tid / kKB;
  float psum[RPT];
#pragma unroll
  for (int j = 0; j < RPT; ++j) psum[j] = 0.f;
  if (key < r.k1) {
    // four heads' rows in flight at a time; heads are still summed in ascending order
    const float* A0 = a.attn + r.attn_off + key;
    const long long hstride = (long long)r.l * r.k1;
    for (int h0 = 0; h0 < nh; h0 += 4) {
      float v[4][RPT];
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const float* A = A0 + (long long)s_heads[min(h0 + x, nh - 1)] * hstride;
#pragma unroll
        for (int j = 0; j < RPT; ++j) {
          const int q = q0 + rbase + 2 * j;
          v[x][j] = (h0 + x < nh && q < r.l) ? __ldcg(A + (long long)q * r.k1) : 0.f;
        }
      }
#pragma unroll
      for (int x = 0; x < 4; ++x)
#pragma unroll
        for (int j = 0; j < RPT; ++j) psum[j] += v[x][j];
    }
  }
  // rows past L contribute nothing; attention is positive, so 0 never wins the max
  float m = 0.f;
#pragma unroll
  for (int j = 0; j < RPT; ++j) m = fmaxf(m, psum[j]);
  if (rbase == 1) s_half[tid & (kKB - 1)] = m;
  __syncthreads();
  if (rbase == 0 && key < r.k1) {
    const float inv_nh = nh > 0 ? 1.0f / (float)nh : 0.f;
    atomicMax(a.p_bits + r.k1_off + key, __float_as_uint(fmaxf(m, s_half[tid]) * inv_nh));
  }

  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int nqc = (r.l + QC - 1) / QC;
    const unsigned prev = atomicAdd(&a.cnt_ts[b], 1u);
    s_last = (prev == (unsigned)(nqc * nib) - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) a.cnt_ts[b] = 0u;
  if (a.heads_out)
    for (int x = tid; x < nh; x += 128) a.heads_out[(long long)b * a.n_keep + x] = s_heads[x];
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
  if (n <= 128) {
    block_mark_topk_small(keys, n, r.k2, flags);
  } else {
    block_kth_largest(keys, n, r.k2, ss, lo, hi, tau, need, n_eq);
    block_mark_selected(keys, n, tau, need, n_eq, flags, ss);
  }
  block_compact_flags(flags, n, a.kept_local + r.k2_off, ss);
}

// ------------------------------------------------------------------ stage 2 for small requests
//
// Requests with L <= 64 text rows and K1 <= 128 visual tokens take two grids.
//
// in_attn_small_kernel: one block per (request, head). Q_h (64 rows) and K_g (K1 rows) are
// copied into shared memory once; each warp computes the logits of 16 text rows against all
// keys on the tensor cores and keeps them in registers (a quad of lanes holds two rows), so
// the softmax max and sum and the two-pass Eq. 8 row variance need only quad shuffles. The
// block writes the attention probabilities A_h[q][i] and u_h.
//
// in_select_small_kernel: one block per (request, 16 keys). Each block forms H* from u and
// Eq. 9 p_i = max_q of the mean over H* (heads summed in ascending order) for its keys, with
// thread (key, row group) and all of a thread's loads in flight: a request's 4 L K1 |H*|
// bytes of probabilities are spread over several SMs. The last block of a request to
// finish (a ticket per request, reset by that block) ranks the K1 scores, TopK(p, K2) with
// ties to the lower index, and writes the ordered kept list.
template <int NCH>   // 64-key chunks: K1 <= 64 * NCH
__global__ void __launch_bounds__(128) in_attn_small_kernel(const __grid_constant__ InMeta meta, const InArgs a) {
  constexpr int QR = 64;              // text rows (four m16 tiles, one per warp)
  constexpr int NT = 8;               // n-tiles of a 64-key chunk
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ float s_upart[4];
  if (!a.independent) pdl_wait();     // Q, K may come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x / a.Hq, h = blockIdx.x - b * a.Hq;
  const int g = (h * a.Hkv) / a.Hq;
  const InReq r = meta.r[b];
  const int L = r.l, K1 = r.k1;
  const uint32_t qs_a = smem_u32(smem), ks_a = qs_a + QR * kRowBytes;
  load_rows(qs_a, a.Q + (long long)r.l_off * a.q_ts + (long long)h * a.q_hs, a.q_ts, 0, QR, L, tid, 128);
  load_rows(ks_a, a.K + (long long)r.k1_off * a.k_ts + (long long)g * a.k_hs, a.k_ts, 0, 64 * NCH, K1, tid, 128);
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();
  float acc[NCH][NT][4];
  {
    uint32_t af[8][4];
    load_afrag(qs_a, 16 * warp, lane, af);
#pragma unroll
    for (int ch = 0; ch < NCH; ++ch) qk_tile<NT>(af, ks_a + ch * 64 * kRowBytes, 0, lane, acc[ch]);
  }
  const float sc = a.scale * 1.4426950408889634f;       // logits in log2 units
  const int ra = 16 * warp + (lane >> 2), rb = ra + 8;
  // full-sequence variant: the non-visual mass of rows ra, rb joins their denominators
  float oa = -INFINITY, ob = -INFINITY;
  if (a.lse) {
    const float* lr = a.lse + (long long)h * a.lse_hs + (long long)r.l_off * a.lse_rs;
    if (ra < L) oa = __ldg(lr + (long long)ra * a.lse_rs) * 1.4426950408889634f;
    if (rb < L) ob = __ldg(lr + (long long)rb * a.lse_rs) * 1.4426950408889634f;
  }
  float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
  for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = 64 * ch + 8 * nt + 2 * (lane & 3) + e;
        if (key < K1) {
          mxa = fmaxf(mxa, acc[ch][nt][e] * sc);
          mxb = fmaxf(mxb, acc[ch][nt][2 + e] * sc);
        }
      }
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, o));
    mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, o));
  }
  mxa = fmaxf(mxa, oa);
  mxb = fmaxf(mxb, ob);
  float sa = 0.f, sb = 0.f;
#pragma unroll
  for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = 64 * ch + 8 * nt + 2 * (lane & 3) + e;
        const float ea = key < K1 ? exp2f(acc[ch][nt][e] * sc - mxa) : 0.f;
        const float eb = key < K1 ? exp2f(acc[ch][nt][2 + e] * sc - mxb) : 0.f;
        acc[ch][nt][e] = ea;
        acc[ch][nt][2 + e] = eb;
        sa += ea;
        sb += eb;
      }
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    sa += __shfl_xor_sync(0xffffffffu, sa, o);
    sb += __shfl_xor_sync(0xffffffffu, sb, o);
  }
  const float ta = sa + exp2f(oa - mxa), tb = sb + exp2f(ob - mxb);   // + 0 without the variant
  const float ia = 1.0f / ta, ib = 1.0f / tb;
  // Eq. 8 takes the variance about each row's mean: 1 / K1, or its visual mass / K1
  const float mean_a = a.lse ? (sa * ia) / (float)K1 : 1.0f / (float)K1;
  const float mean_b = a.lse ? (sb * ib) / (float)K1 : 1.0f / (float)K1;
  float* A = a.attn + r.attn_off + (long long)h * L * K1;
  float* Aa = A + (long long)ra * K1;
  float* Ab = A + (long long)rb * K1;
  // (key, key + 1) pairs go out as one 8-byte store when every row start is 8-byte aligned
  const bool pairs = (K1 & 1) == 0 && ((reinterpret_cast<uintptr_t>(A) & 7) == 0);
  const bool wa = ra < L, wb = rb < L;
  float va = 0.f, vb = 0.f;
#pragma unroll
  for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int key = 64 * ch + 8 * nt + 2 * (lane & 3);
      const float pa0 = acc[ch][nt][0] * ia, pa1 = acc[ch][nt][1] * ia;
      const float pb0 = acc[ch][nt][2] * ib, pb1 = acc[ch][nt][3] * ib;
      if (key < K1) {
        va = fmaf(pa0 - mean_a, pa0 - mean_a, va);
        vb = fmaf(pb0 - mean_b, pb0 - mean_b, vb);
      }
      if (key + 1 < K1) {
        va = fmaf(pa1 - mean_a, pa1 - mean_a, va);
        vb = fmaf(pb1 - mean_b, pb1 - mean_b, vb);
      }
      if (pairs) {
        if (key < K1) {
          if (wa) *reinterpret_cast<float2*>(Aa + key) = make_float2(pa0, pa1);
          if (wb) *reinterpret_cast<float2*>(Ab + key) = make_float2(pb0, pb1);
        }
      } else if (key < K1) {
        if (wa) {
          Aa[key] = pa0;
          if (key + 1 < K1) Aa[key + 1] = pa1;
        }
        if (wb) {
          Ab[key] = pb0;
          if (key + 1 < K1) Ab[key + 1] = pb1;
        }
      }
    }
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    va += __shfl_xor_sync(0xffffffffu, va, o);
    vb += __shfl_xor_sync(0xffffffffu, vb, o);
  }
  // Eq. 8 numerator: sum over this warp's valid rows of Var_i A[q, i]
  float vs = ((lane & 3) == 0) ? ((ra < L ? va : 0.f) + (rb < L ? vb : 0.f)) / (float)K1 : 0.f;
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) vs += __shfl_xor_sync(0xffffffffu, vs, o);
  if (lane == 0) s_upart[warp] = vs;
  __syncthreads();
  if (tid == 0) a.u[(long long)b * a.u_ld + h] = (((s_upart[0] + s_upart[1]) + s_upart[2]) + s_upart[3]) / (float)L;
}

constexpr int kSelThreads = 128;
constexpr int kSelKeys = 16;                       // keys per block
constexpr int kSelGroups = kSelThreads / kSelKeys; // row groups per block
__global__ void __launch_bounds__(kSelThreads) in_select_small_kernel(const __grid_constant__ InMeta meta,
                                                                       const InArgs a) {
  __shared__ float s_u[kMaxHeads];
  __shared__ int s_heads[kMaxHeads];
  __shared__ int s_wc[kSelThreads / 32];
  __shared__ float s_red[kSelThreads];
  __shared__ uint32_t s_keys[128];
  __shared__ int s_last;
  pdl_wait();                         // u and the attention probabilities come from the preceding grid
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int kblocks = (int)gridDim.y;
  const int b = blockIdx.x, kb = blockIdx.y;
  const InReq r = meta.r[b];
  const int L = r.l, K1 = r.k1, Hq = a.Hq;
  if (kb * kSelKeys < K1) {
    const float* u = a.u + (long long)b * a.u_ld;
    for (int hh = tid; hh < Hq; hh += kSelThreads) s_u[hh] = __ldcg(u + hh);
    __syncthreads();
    // H*: the n_keep largest u, ties to the lower head, listed in ascending head order
    int nh = 0;
    for (int h0 = 0; h0 < Hq; h0 += kSelThreads) {
      const int hh = h0 + tid;
      bool sel = false;
      if (hh < Hq) {
        const float uh = s_u[hh];
        int rank = 0;
        for (int x = 0; x < Hq; ++x) rank += (s_u[x] > uh) || (s_u[x] == uh && x < hh);
        sel = rank < a.n_keep;
      }
      const uint32_t bal = __ballot_sync(0xffffffffu, sel);
      if (lane == 0) s_wc[warp] = __popc(bal);
      __syncthreads();
      int before = nh;
      for (int w = 0; w < warp; ++w) before += s_wc[w];
      for (int w = 0; w < kSelThreads / 32; ++w) nh += s_wc[w];
      if (sel) s_heads[before + __popc(bal & lanemask_lt())] = hh;
      __syncthreads();
    }
    // at most n_keep heads, the lowest of those ranked first, even if u holds NaN (a NaN
    // compares false with everything, so its head ranks 0 and joins the n_keep best)
    nh = min(nh, a.n_keep);
    // Eq. 9 for key i: rows rg, rg + 8, ... (L <= 64: eight rows), every head's loads in flight
    const int i = kb * kSelKeys + (tid % kSelKeys), rg = tid / kSelKeys;
    const float* A = a.attn + r.attn_off + i;
    const long long hstride = (long long)L * K1;
    float m = 0.f;                    // probabilities are positive: 0 never wins the max
    if (i < K1) {
      constexpr int RPT = 64 / kSelGroups;
      float psum[RPT];
#pragma unroll
      for (int j = 0; j < RPT; ++j) psum[j] = 0.f;
      for (int h0 = 0; h0 < nh; h0 += 8) {
        float v[8][RPT];
#pragma unroll
        for (int x = 0; x < 8; ++x) {
          const float* Ah = A + (long long)s_heads[min(h0 + x, nh - 1)] * hstride;
#pragma unroll
          for (int j = 0; j < RPT; ++j) {
            const int q = rg + kSelGroups * j;
            v[x][j] = (h0 + x < nh && q < L) ? __ldcg(Ah + (long long)q * K1) : 0.f;
          }
        }
#pragma unroll
        for (int x = 0; x < 8; ++x)
#pragma unroll
          for (int j = 0; j < RPT; ++j) psum[j] += v[x][j];
      }
#pragma unroll
      for (int j = 0; j < RPT; ++j) m = fmaxf(m, psum[j]);
    }
    s_red[tid] = m;
    __syncthreads();
    if (tid < kSelKeys && i < K1) {
      float mx = 0.f;
      for (int x = 0; x < kSelGroups; ++x) mx = fmaxf(mx, s_red[x * kSelKeys + tid]);
      a.p_bits[r.k1_off + i] = __float_as_uint(mx * (nh > 0 ? 1.0f / (float)nh : 0.f));
    }
    if (kb == 0 && a.heads_out)
      for (int x = tid; x < nh; x += kSelThreads) a.heads_out[(long long)b * a.n_keep + x] = s_heads[x];
  }
  // the last block of the request ranks all K1 scores
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t done = atomicAdd(a.cnt_ts + b, 1u) + 1u;
    s_last = done == (uint32_t)kblocks;
    if (s_last) a.cnt_ts[b] = 0u;     // ready for the next launch
  }
  __syncthreads();
  if (!s_last || r.k2 <= 0) return;
  __threadfence();
  uint32_t key = 0u;
  if (tid < K1) {
    key = score_key(__uint_as_float(__ldcg(a.p_bits + r.k1_off + tid)));
    s_keys[tid] = key;
  }
  __syncthreads();
  bool keep = false;
  if (tid < K1) {
    int rank = 0;
#pragma unroll 4
    for (int j = 0; j < K1; ++j) {
      const uint32_t o = s_keys[j];
      rank += (o > key) || (o == key && j < tid);
    }
    keep = rank < r.k2;
  }
  const uint32_t kbal = __ballot_sync(0xffffffffu, keep);
  if (lane == 0) s_wc[warp] = __popc(kbal);
  __syncthreads();
  int pos = 0;
  for (int w = 0; w < warp; ++w) pos += s_wc[w];
  if (keep) a.kept_local[r.k2_off + pos + __popc(kbal & lanemask_lt())] = tid;
}

// ------------------------------------------------------------------ host-side launchers

// Row stride of the logits tile: 2 mod 32 words keeps the row-parallel passes conflict-free.
int in_head_stats_ld(int max_k1) { return ((max_k1 + kKB - 1) / kKB) * kKB + 2; }

cudaError_t launch_in_head_stats(const InMeta& meta, const InArgs& a, int max_k1, cudaStream_t st) {
  if (meta.total_hs == 0) return cudaSuccess;
  const int ld = in_head_stats_ld(max_k1);
  const int qc = stats_text_rows(max_k1);
  const int smem = qc * kRowBytes + 2 * kKB * kRowBytes + qc * ld * 4;   // two K chunk buffers
  cudaError_t e;
  switch (qc) {
    case 64:
      e = ensure_dynamic_smem(in_head_stats_kernel<4>, smem);
      if (e != cudaSuccess) return e;
      return launch_kernel(in_head_stats_kernel<4>, dim3(meta.total_hs), dim3(128), smem, st, true, meta, a, ld);
    case 32:
      e = ensure_dynamic_smem(in_head_stats_kernel<2>, smem);
      if (e != cudaSuccess) return e;
      return launch_kernel(in_head_stats_kernel<2>, dim3(meta.total_hs), dim3(128), smem, st, true, meta, a, ld);
    default:
      e = ensure_dynamic_smem(in_head_stats_kernel<1>, smem);
      if (e != cudaSuccess) return e;
      return launch_kernel(in_head_stats_kernel<1>, dim3(meta.total_hs), dim3(128), smem, st, true, meta, a, ld);
  }
}

// The two-grid small path when every request has L <= 64 and K1 <= 128.
bool in_small_fits(int Hq, int max_l, int max_k1) { return max_l <= 64 && max_k1 <= 128 && Hq <= kMaxHeads; }

cudaError_t launch_in_small(const InMeta& meta, const InArgs& a, int max_k1, cudaStream_t st) {
  if (meta.B == 0) return cudaSuccess;
  const int nch = max_k1 <= 64 ? 1 : 2;
  const int smem = 64 * kRowBytes + 64 * nch * kRowBytes;
  const dim3 grid((unsigned)(meta.B * a.Hq));
  cudaError_t e = nch == 1 ? launch_kernel(in_attn_small_kernel<1>, grid, dim3(128), smem, st, true, meta, a)
                           : launch_kernel(in_attn_small_kernel<2>, grid, dim3(128), smem, st, true, meta, a);
  if (e != cudaSuccess) return e;
  const dim3 sgrid((unsigned)meta.B, (unsigned)((max_k1 + kSelKeys - 1) / kSelKeys));
  return launch_kernel(in_select_small_kernel, sgrid, dim3(kSelThreads), 0, st, true, meta, a);
}

cudaError_t launch_in_token_score(const InMeta& meta, const InArgs& a, int max_k1, cudaStream_t st) {
  if (meta.total_ts == 0) return cudaSuccess;
  const int smem = max_k1 * 5 + 16;
  cudaError_t e = ensure_dynamic_smem(in_token_score_kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(in_token_score_kernel, dim3(meta.total_ts), dim3(128), smem, st, true, meta, a, smem);
}

}  // namespace trevs
