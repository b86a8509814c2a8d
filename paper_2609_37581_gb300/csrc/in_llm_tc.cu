// Stage 2 (in-LLM at layer l*, Sec. 4.2) for requests too large for the small path, on the
// 5th-generation tensor cores. Two grids; the [Hq, L, K1] attention probabilities never reach
// memory.
//
// in_stats_tc_kernel, one block per (request, head h, 128 text rows): the logits
// S = Q_h . K_g^T (UMMA M = 128 rows, N = 128 keys, K = 128 dims) of the block's rows, chunk by
// chunk of 128 keys, into a double-buffered TMEM accumulator. TMEM lane r holds text row r, so
// each epilogue thread owns a whole row. Per chunk the thread takes the row's maximum, then
// the sum of e = exp(logit - max), and the sum of squared deviations of e about the chunk's
// mean (shifted sums, shift = the chunk's first e); the chunks merge by the pairwise update
// of Chan, Golub and LeVeque (1979), rescaled to the running maximum. One pass over the keys
// thus gives each row's softmax normaliser and the Eq. 8 variance of its probabilities about
// their mean (1 / K1, or the row's visual mass / K1 with the full-sequence variant). Each row's
// (max, 1 / total) goes to the workspace for the token scores; the last block of a request
// averages the row variances into u_h (Eq. 8) and clears p.
//
// in_score_tc_kernel, one block per (request, 128 text rows, 64 visual keys): H* from u, then
// for each head of H* in ascending order the logits of the block's rows and keys again (UMMA
// M = 128, N = 64), the probabilities from the rows' (max, 1 / total), summed per (row, key)
// in registers (Eq. 9, head mean); the max over the rows merges across blocks with an integer
// atomicMax on the (non-negative) float bits. The last block of a request takes
// TopK(p, K2) and writes H*.
//
// Operands: Q_h and K_g tiles arrive by TMA (two 64-dim boxes of 128-byte swizzled rows per
// tile, from a [rows][heads][128] tensor map), in the K-major layout the UMMA descriptors
// state. Rows past the request (the next request's rows or the zero fill past the tensor)
// produce logits that no thread reads. Warps: 0 = TMA producer, 1 = TMEM owner and MMA
// issuer, 2..9 = epilogue, two per TMEM lane quarter (warp w reads lanes 32 (w % 4) .. + 31
// and half of the columns; tree reductions keep the dependent chains short). Every wait is bounded
// by the limit in word 1 of the status words (2 s when 0); a wait that gives up stops the
// block, drains its MMAs and copies, and sets bit 0 of the status word.
#include "in_llm.cuh"
#include "sm100.cuh"

namespace trevs {

namespace {

constexpr int kTcRows = 128;                     // text rows per block (UMMA M)
constexpr int kSlice = kTcRows * 128;            // one 64-dim slice of 128 rows: 16 KB
constexpr int kTile = 2 * kSlice;                // 128 rows x 128 dims: 32 KB
constexpr int kStatKeys = 128;                   // keys per statistics chunk (UMMA N)
constexpr int kStatStages = 2;
constexpr int kScoreKeys = 64;                   // keys per token-score block (UMMA N)
constexpr int kScoreKSlice = kScoreKeys * 128;   // one 64-dim slice of 64 keys: 8 KB
constexpr int kScoreStage = kTile + 2 * kScoreKSlice;
constexpr int kScoreStages = 2;
constexpr int kEpiWarps = 8;                     // two warps per TMEM lane quarter
constexpr int kTcThreads = 64 + 32 * kEpiWarps;  // producer, MMA issuer, epilogue
constexpr int kStatHalf = kStatKeys / 2;         // columns of a chunk per epilogue warp
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint64_t wait_limit_ns(const uint32_t* err) {
  const uint32_t us = err ? __ldcg(err + 1) : 0u;
  return us ? (uint64_t)us * 1000ull : 2000000000ull;
}

// D (+)= the 128-row tile at `a` (two 16 KB slices) times the `n`-row tile at `b` (two
// slices of n * 128 bytes), K = 128 dims: two slices x four 16-dim steps.
__device__ __forceinline__ void mma_tile_128(uint32_t d, uint32_t a, uint32_t b, int n, uint32_t idesc) {
  using namespace sm100;
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int k = 0; k < 4; ++k)
      umma_bf16(d, umma_desc_sw128(a + c * kSlice + 32 * k), umma_desc_sw128(b + c * n * 128 + 32 * k), idesc,
                (c | k) != 0 ? 1u : 0u);
}

// Reductions of 32 values in a tree of depth 5 (the array is overwritten).
__device__ __forceinline__ float tree_max32(float (&w)[32]) {
#pragma unroll
  for (int s = 16; s; s >>= 1)
#pragma unroll
    for (int i = 0; i < s; ++i) w[i] = fmaxf(w[i], w[i + s]);
  return w[0];
}
__device__ __forceinline__ float tree_sum32(float (&w)[32]) {
#pragma unroll
  for (int s = 16; s; s >>= 1)
#pragma unroll
    for (int i = 0; i < s; ++i) w[i] += w[i + s];
  return w[0];
}

// Pairwise merge (Chan, Golub and LeVeque) of two partial states of a row: n values
// e = exp2(y - m) with sum S and sum of squared deviations about their mean M2; n = 0 is an
// empty state. The result is in units of exp2(y - max(m, m2)).
__device__ __forceinline__ void merge_state(float& m, float& n, float& S, float& M2, float m2, float n2, float S2,
                                            float M22) {
  if (n2 == 0.f) return;
  if (n == 0.f) {
    m = m2; n = n2; S = S2; M2 = M22;
    return;
  }
  const float mx = fmaxf(m, m2);
  const float f = exp2f(m - mx), f2 = exp2f(m2 - mx);
  const float dm = S2 * f2 / n2 - S * f / n;   // difference of the two means
  const float nn = n + n2;
  M2 = M2 * f * f + M22 * f2 * f2 + dm * dm * (n * n2 / nn);
  S = S * f + S2 * f2;
  m = mx;
  n = nn;
}

// Rows of the Q box for a chunk with `rows` text rows: 32, 64 or 128. The MMA still reads
// 128 rows of each slice; rows past the box hold stale data and yield logits no thread reads.
__device__ __forceinline__ int q_box_rows(int rows) { return rows <= 32 ? 32 : (rows <= 64 ? 64 : kTcRows); }
__device__ __forceinline__ const CUtensorMap* q_map(const InQMaps& m, int qb) {
  return qb == 32 ? &m.q32 : (qb == 64 ? &m.q64 : &m.q128);
}

}  // namespace

__global__ void __launch_bounds__(kTcThreads, 2)
    in_stats_tc_kernel(const __grid_constant__ InQMaps tq, const __grid_constant__ CUtensorMap tmK,
                       const __grid_constant__ InMeta meta, const InArgs a) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t qfull, kfull[kStatStages], kempty[kStatStages];
  __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2], mma_drain;
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_kissued;
  __shared__ int s_last;
  __shared__ float4 s_state[2][kTcRows];   // (m, n, S, M2) of each row, per column half
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t qs = smem_u32(smem), ks = qs + kTile;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].hs_off; });
  const InReq r = meta.r[b];
  const int nqc = (r.l + kTcRows - 1) / kTcRows;
  const int t = blockIdx.x - r.hs_off;
  const int h = t / nqc, qc = t - h * nqc;
  const int g = (h * a.Hkv) / a.Hq;
  const int q0 = qc * kTcRows;
  const int K1 = r.k1, L = r.l, nkc = (K1 + kStatKeys - 1) / kStatKeys;
  const uint64_t lim = wait_limit_ns(a.err);

  if (tid == 0) {
    mbar_init(smem_u32(&qfull), 1);
    for (int s = 0; s < kStatStages; ++s) {
      mbar_init(smem_u32(&kfull[s]), 1);
      mbar_init(smem_u32(&kempty[s]), 1);          // MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&acc_full[i]), 1);
      mbar_init(smem_u32(&acc_empty[i]), kEpiWarps);
    }
    mbar_init(smem_u32(&mma_drain), 1);
    s_abort = 0;
    s_kissued = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), 2 * kStatKeys);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  if (!a.overlap && !a.independent) pdl_wait();   // Q, K may come from the preceding grid
  pdl_launch_dependents();

  if (warp == 0) {
    if (lane == 0) {
      const int qb = q_box_rows(L - q0);
      const CUtensorMap* tmQ = q_map(tq, qb);
      tma_prefetch_desc(tmQ);
      tma_prefetch_desc(&tmK);
      const uint64_t pol = l2_policy_evict_last();   // K_g serves every head of its group
      const int qrow = r.l_off + q0;
      mbar_arrive_expect_tx(smem_u32(&qfull), (uint32_t)(qb * 256));
      tma_load_3d(qs, tmQ, 0, qrow, h, smem_u32(&qfull), pol);
      tma_load_3d(qs + kSlice, tmQ, 64, qrow, h, smem_u32(&qfull), pol);
      for (int j = 0; j < nkc; ++j) {
        const int s = j % kStatStages, ph = j / kStatStages;
        if (j >= kStatStages && !mbar_wait(smem_u32(&kempty[s]), (ph - 1) & 1, &s_abort, lim)) {
          s_abort = 1;
          break;
        }
        const uint32_t dst = ks + s * kTile, fb = smem_u32(&kfull[s]);
        mbar_arrive_expect_tx(fb, (uint32_t)kTile);
        tma_load_3d(dst, &tmK, 0, r.k1_off + j * kStatKeys, g, fb, pol);
        tma_load_3d(dst + kSlice, &tmK, 64, r.k1_off + j * kStatKeys, g, fb, pol);
        s_kissued = j + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kTcRows, kStatKeys);
      bool ok = mbar_wait(smem_u32(&qfull), 0, &s_abort, lim);
      for (int j = 0; ok && j < nkc; ++j) {
        const int s = j % kStatStages, ph = j / kStatStages, buf = j & 1, use = j >> 1;
        ok = mbar_wait(smem_u32(&kfull[s]), ph & 1, &s_abort, lim);
        if (ok && j >= 2) ok = mbar_wait(smem_u32(&acc_empty[buf]), (use - 1) & 1, &s_abort, lim);
        if (!ok) break;
        tc_fence_after();
        mma_tile_128(tmem + (uint32_t)(buf * kStatKeys), qs, ks + s * kTile, kStatKeys, idesc);
        umma_commit(smem_u32(&kempty[s]));     // frees the K stage once these MMAs have read it
        umma_commit(smem_u32(&acc_full[buf]));
      }
      if (!ok) {
        s_abort = 1;
        // no MMA may still write TMEM when it is released: wait for every one issued
        const volatile int no_abort = 0;
        umma_commit(smem_u32(&mma_drain));
        mbar_wait(smem_u32(&mma_drain), 0, &no_abort, 500000000ull);
      }
    }
  } else {
    // epilogue warp w: TMEM lane quarter w % 4 (the text rows), column half (w - 2) / 4 of
    // every chunk; a warp whose 32 rows all lie past the request's L only keeps pace
    const int q = warp & 3, row = 32 * q + lane, half = (warp - 2) >> 2;
    const bool live = 32 * q < L - q0;
    const float sc = a.scale * kLog2e;            // logits in log2 units: exp(x) = exp2(x log2 e)
    // running state over this thread's keys so far (see merge_state)
    float m = -INFINITY, n = 0.f, S = 0.f, M2 = 0.f;
    for (int j = 0; j < nkc; ++j) {
      const int buf = j & 1, use = j >> 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_full[buf]), use & 1, &s_abort, lim) && !s_abort);
      if (!ok) {
        s_abort = 1;
        break;
      }
      tc_fence_after();
      const int nv = min(kStatKeys, K1 - j * kStatKeys) - half * kStatHalf;   // valid keys of this half
      const uint32_t lb = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * kStatKeys + half * kStatHalf);
      if (live && nv > 0) {
        const int nh = min(nv, kStatHalf);
        float v[32], w[32];
        float cm = -INFINITY;
        for (int g0 = 0; g0 < nh; g0 += 32) {
          tmem_ld_32x32b_x32(lb + (uint32_t)g0, v);
#pragma unroll
          for (int e = 0; e < 32; ++e) w[e] = g0 + e < nh ? v[e] * sc : -INFINITY;
          cm = fmaxf(cm, tree_max32(w));
        }
        float se = 0.f, sd = 0.f, sd2 = 0.f, shift = 0.f;
        for (int g0 = 0; g0 < nh; g0 += 32) {
          tmem_ld_32x32b_x32(lb + (uint32_t)g0, v);
          if (g0 == 0) shift = exp2f(v[0] * sc - cm);   // shifted sums: about the first e
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const bool in = g0 + e < nh;
            const float x = in ? exp2f(v[e] * sc - cm) : 0.f;
            w[e] = in ? x - shift : 0.f;
            v[e] = x;
          }
          se += tree_sum32(v);
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = w[e] * w[e];
          sd2 += tree_sum32(v);
          sd += tree_sum32(w);
        }
        const float fv = (float)nh;
        merge_state(m, n, S, M2, cm, fv, se, fmaxf(sd2 - sd * sd / fv, 0.f));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&acc_empty[buf]));
    }
    s_state[half][row] = make_float4(m, n, S, M2);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * kStatKeys);
  }
  if (s_abort) {
    // let the copies already issued land before the block's shared memory is released
    if (tid == 0) {
      const volatile int no_abort = 0;
      mbar_wait(smem_u32(&qfull), 0, &no_abort, 500000000ull);
      const int ki = s_kissued;
      for (int j = ki - kStatStages > 0 ? ki - kStatStages : 0; j < ki; ++j)
        mbar_wait(smem_u32(&kfull[j % kStatStages]), (j / kStatStages) & 1, &no_abort, 500000000ull);
      atomicOr(a.err, 1u);
    }
    return;
  }

  // each row: its two column halves merged, then (T, 1 / total) and the Eq. 8 variance
  if (tid < kTcRows && q0 + tid < L) {
    const int rq = q0 + tid;
    float4 st = s_state[0][tid];
    const float4 s1 = s_state[1][tid];
    merge_state(st.x, st.y, st.z, st.w, s1.x, s1.y, s1.z, s1.w);
    // full-sequence variant: the row's non-visual mass joins the denominator
    const float o = a.lse ? __ldg(a.lse + (long long)h * a.lse_hs + (long long)(r.l_off + rq) * a.lse_rs) * kLog2e
                          : -INFINITY;
    const float tm = fmaxf(st.x, o);
    const float f = exp2f(st.x - tm);
    const float inv = 1.0f / (st.z * f + exp2f(o - tm));   // + 0 without the variant
    const float fp = f * inv;                                // p = e * fp
    a.rstat[(long long)h * a.stats_ld + r.l_off + rq] = make_float2(tm, inv);
    // Eq. 8: the variance of the row's K1 probabilities about their mean
    a.row_var[(long long)h * a.stats_ld + r.l_off + rq] = st.w * fp * fp / (float)K1;
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
  for (int hh = warp; hh < a.Hq; hh += kTcThreads / 32) {
    const float* rv = a.row_var + (long long)hh * a.stats_ld + r.l_off;
    float s = 0.f;
    for (int x = lane; x < L; x += 32) s += __ldcg(rv + x);
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) a.u[(long long)b * a.u_ld + hh] = s / (float)L;
  }
  if (a.zero_p)
    for (int i = tid; i < K1; i += kTcThreads) a.p_bits[r.k1_off + i] = 0u;
}

__global__ void __launch_bounds__(kTcThreads, 2)
    in_score_tc_kernel(const __grid_constant__ InQMaps tq, const __grid_constant__ CUtensorMap tmK,
                       const __grid_constant__ InMeta meta, const InArgs a, int smem_bytes) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t sfull[kScoreStages], sempty[kScoreStages];
  __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2], mma_drain;
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_issued;
  __shared__ SelShared ss;
  __shared__ float s_u[kMaxHeads];
  __shared__ int s_heads[kMaxHeads];
  __shared__ int s_sel[kMaxHeads];
  __shared__ int s_nh, s_last;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t ring = smem_u32(smem);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].ts_off; });
  const InReq r = meta.r[b];
  const int K1 = r.k1, L = r.l;
  const int nkb = (K1 + kScoreKeys - 1) / kScoreKeys;
  const int t = blockIdx.x - r.ts_off;
  const int qc = t / nkb, kb = t - qc * nkb;
  const int q0 = qc * kTcRows, i0 = kb * kScoreKeys;
  const int nv = min(kScoreKeys, K1 - i0);
  const uint64_t lim = wait_limit_ns(a.err);

  if (tid == 0) {
    for (int s = 0; s < kScoreStages; ++s) {
      mbar_init(smem_u32(&sfull[s]), 1);
      mbar_init(smem_u32(&sempty[s]), 1);          // MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&acc_full[i]), 1);
      mbar_init(smem_u32(&acc_empty[i]), kEpiWarps);
    }
    mbar_init(smem_u32(&mma_drain), 1);
    s_abort = 0;
    s_issued = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), 2 * kScoreKeys);
    tmem_relinquish();
  }
  pdl_wait();   // u, the row statistics and the cleared p come from the preceding grid

  // H*: the n_keep heads of largest u, ties to the lower head, in ascending head order; at
  // most n_keep even if u holds NaN (a NaN compares false with everything and ranks 0)
  const float* u = a.u + (long long)b * a.u_ld;
  for (int hh = tid; hh < a.Hq; hh += kTcThreads) s_u[hh] = __ldcg(u + hh);
  __syncthreads();
  for (int hh = tid; hh < a.Hq; hh += kTcThreads) {
    const float uh = s_u[hh];
    int rank = 0;
    for (int x = 0; x < a.Hq; ++x) {
      const float ux = s_u[x];
      rank += (ux > uh) || (ux == uh && x < hh);
    }
    s_sel[hh] = rank < a.n_keep;
  }
  __syncthreads();
  if (tid == 0) {
    int cnt = 0;
    for (int hh = 0; hh < a.Hq && cnt < a.n_keep; ++hh)
      if (s_sel[hh]) s_heads[cnt++] = hh;
    s_nh = cnt;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const int nh = s_nh;

  if (warp == 0) {
    if (lane == 0) {
      const int qb = q_box_rows(L - q0);
      const CUtensorMap* tmQ = q_map(tq, qb);
      const uint32_t stage_bytes = (uint32_t)(qb * 256 + 2 * kScoreKSlice);
      tma_prefetch_desc(tmQ);
      tma_prefetch_desc(&tmK);
      const uint64_t pol = l2_policy_evict_last();
      for (int j = 0; j < nh; ++j) {
        const int s = j % kScoreStages, ph = j / kScoreStages;
        if (j >= kScoreStages && !mbar_wait(smem_u32(&sempty[s]), (ph - 1) & 1, &s_abort, lim)) {
          s_abort = 1;
          break;
        }
        const int h = s_heads[j], g = (h * a.Hkv) / a.Hq;
        const uint32_t dst = ring + s * kScoreStage, fb = smem_u32(&sfull[s]);
        mbar_arrive_expect_tx(fb, stage_bytes);
        tma_load_3d(dst, tmQ, 0, r.l_off + q0, h, fb, pol);
        tma_load_3d(dst + kSlice, tmQ, 64, r.l_off + q0, h, fb, pol);
        tma_load_3d(dst + kTile, &tmK, 0, r.k1_off + i0, g, fb, pol);
        tma_load_3d(dst + kTile + kScoreKSlice, &tmK, 64, r.k1_off + i0, g, fb, pol);
        s_issued = j + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kTcRows, kScoreKeys);
      bool ok = true;
      for (int j = 0; ok && j < nh; ++j) {
        const int s = j % kScoreStages, ph = j / kScoreStages, buf = j & 1, use = j >> 1;
        ok = mbar_wait(smem_u32(&sfull[s]), ph & 1, &s_abort, lim);
        if (ok && j >= 2) ok = mbar_wait(smem_u32(&acc_empty[buf]), (use - 1) & 1, &s_abort, lim);
        if (!ok) break;
        tc_fence_after();
        const uint32_t st = ring + s * kScoreStage;
        mma_tile_128(tmem + (uint32_t)(buf * kScoreKeys), st, st + kTile, kScoreKeys, idesc);
        umma_commit(smem_u32(&sempty[s]));
        umma_commit(smem_u32(&acc_full[buf]));
      }
      if (!ok) {
        s_abort = 1;
        const volatile int no_abort = 0;
        umma_commit(smem_u32(&mma_drain));
        mbar_wait(smem_u32(&mma_drain), 0, &no_abort, 500000000ull);
      }
    }
  }
  // epilogue: thread (warp 2..9, lane) owns text row 32 (warp % 4) + lane of the block and
  // the keys of column half (warp - 2) / 4; a warp whose 32 rows all lie past L only keeps pace
  constexpr int kHalf = kScoreKeys / 2;
  float acc[kHalf];
#pragma unroll
  for (int c = 0; c < kHalf; ++c) acc[c] = 0.f;
  const int q = warp & 3, row = 32 * q + lane, rq = q0 + row, half = (warp - 2) >> 2;
  if (warp >= 2) {
    const float sc = a.scale * kLog2e;
    const float2* rstat = a.rstat + r.l_off + rq;
    float2 rs_next = make_float2(0.f, 0.f);
    if (nh > 0 && rq < L) rs_next = __ldcg(rstat + (long long)s_heads[0] * a.stats_ld);
    for (int j = 0; j < nh; ++j) {
      const int buf = j & 1, use = j >> 1;
      const float2 rs = rs_next;   // the next head's row statistics load while this one waits
      if (j + 1 < nh && rq < L) rs_next = __ldcg(rstat + (long long)s_heads[j + 1] * a.stats_ld);
      const bool ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&acc_full[buf]), use & 1, &s_abort, lim) && !s_abort);
      if (!ok) {
        s_abort = 1;
        break;
      }
      tc_fence_after();
      if (32 * q < L - q0) {
        float v[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * kScoreKeys + half * kHalf), v);
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[e] += exp2f(v[e] * sc - rs.x) * rs.y;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&acc_empty[buf]));
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * kScoreKeys);
  }
  if (s_abort) {
    if (tid == 0) {
      const volatile int no_abort = 0;
      const int ji = s_issued;
      for (int j = ji - kScoreStages > 0 ? ji - kScoreStages : 0; j < ji; ++j)
        mbar_wait(smem_u32(&sfull[j % kScoreStages]), (j / kScoreStages) & 1, &no_abort, 500000000ull);
      atomicOr(a.err, 1u);
    }
    return;
  }
  // every copy has landed and every MMA completed: the ring holds the [128][65] row sums
  float* colbuf = reinterpret_cast<float*>(smem);
  if (warp >= 2) {
#pragma unroll
    for (int c = 0; c < kHalf; ++c) colbuf[row * (kScoreKeys + 1) + half * kHalf + c] = rq < L ? acc[c] : 0.f;
  }
  __syncthreads();
  if (tid < nv) {
    // rows past L contribute 0; probabilities are positive, so 0 never wins the max
    float mx = 0.f;
    for (int x = 0; x < kTcRows; ++x) mx = fmaxf(mx, colbuf[x * (kScoreKeys + 1) + tid]);
    const float inv_nh = nh > 0 ? 1.0f / (float)nh : 0.f;
    atomicMax(a.p_bits + r.k1_off + i0 + tid, __float_as_uint(mx * inv_nh));
  }

  // the last block of the request ranks all K1 scores
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int nqc = (L + kTcRows - 1) / kTcRows;
    const unsigned prev = atomicAdd(&a.cnt_ts[b], 1u);
    s_last = (prev == (unsigned)(nqc * nkb) - 1);
  }
  __syncthreads();
  if (!s_last) return;
  pdl_launch_dependents();   // the compaction may launch now, onto the SMs the other blocks left
  __threadfence();
  if (tid == 0) a.cnt_ts[b] = 0u;
  if (a.heads_out)
    for (int x = tid; x < nh; x += kTcThreads) a.heads_out[(long long)b * a.n_keep + x] = s_heads[x];
  if (r.k2 <= 0) return;
  const int n = K1;
  const bool in_smem = (size_t)n * 5 <= (size_t)smem_bytes;
  const size_t gbase = ((size_t)r.k1_off + 4 * (size_t)b + 3) & ~(size_t)3;   // 16-byte aligned
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + gbase;
  uint8_t* flags = in_smem ? smem + (size_t)n * 4 : a.flags + gbase;
  __syncthreads();   // colbuf is read no more
  for (int i = tid; i < n; i += kTcThreads) flags[i] = 0;
  uint32_t lo, hi, tau;
  int need, n_eq;
  block_fill_keys(keys, reinterpret_cast<const float*>(a.p_bits + r.k1_off), n,
                  [&](float x, int) { return score_key(x); }, ss, lo, hi);
  if (n <= kTcThreads) {
    block_mark_topk_small(keys, n, r.k2, flags);
  } else {
    block_kth_largest(keys, n, r.k2, ss, lo, hi, tau, need, n_eq);
    block_mark_selected(keys, n, tau, need, n_eq, flags, ss);
  }
  block_compact_flags(flags, n, a.kept_local + r.k2_off, ss);
}

// ------------------------------------------------------------------ host-side launchers

// Tensor maps of Q (128-row boxes) and K (128- and 64-row boxes) for the two grids; fails
// (and the caller takes the store-once kernels) when the strides do not suit TMA.
cudaError_t make_in_tc_maps(const InArgs& a, long long q_rows, long long k_rows, InTcMaps& m) {
  cudaError_t e = make_tmap_heads(&m.q.q128, a.Q, q_rows, a.Hq, a.q_ts, a.q_hs, kTcRows);
  if (e == cudaSuccess) e = make_tmap_heads(&m.q.q64, a.Q, q_rows, a.Hq, a.q_ts, a.q_hs, 64);
  if (e == cudaSuccess) e = make_tmap_heads(&m.q.q32, a.Q, q_rows, a.Hq, a.q_ts, a.q_hs, 32);
  if (e == cudaSuccess) e = make_tmap_heads(&m.k128, a.K, k_rows, a.Hkv, a.k_ts, a.k_hs, kStatKeys);
  if (e == cudaSuccess) e = make_tmap_heads(&m.k64, a.K, k_rows, a.Hkv, a.k_ts, a.k_hs, kScoreKeys);
  return e;
}

int in_tc_text_rows() { return kTcRows; }
int in_tc_score_keys() { return kScoreKeys; }

cudaError_t launch_in_stats_tc(const InMeta& meta, const InArgs& a, const InTcMaps& m, cudaStream_t st) {
  if (meta.total_hs == 0) return cudaSuccess;
  const int smem = (1 + kStatStages) * kTile + 1024;
  return launch_kernel(in_stats_tc_kernel, dim3(meta.total_hs), dim3(kTcThreads), smem, st, true, m.q, m.k128, meta,
                       a);
}

cudaError_t launch_in_score_tc(const InMeta& meta, const InArgs& a, const InTcMaps& m, cudaStream_t st) {
  if (meta.total_ts == 0) return cudaSuccess;
  const int ring = kScoreStages * kScoreStage;
  return launch_kernel(in_score_tc_kernel, dim3(meta.total_ts), dim3(kTcThreads), ring + 1024, st, true, m.q, m.k64,
                       meta, a, ring);
}

}  // namespace trevs
