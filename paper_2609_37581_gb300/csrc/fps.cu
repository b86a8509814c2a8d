// Stage 1 context preservation (Sec. 3.1): S_d = FPS({z_i | i in C}, K_d), C = [N] minus S_r.
//
// Each step of farthest point sampling takes the candidate whose smallest cosine distance
// 1 - cos(z_i, z_s) to the tokens selected so far (the pivots S_r and the earlier picks) is
// largest, ties to the lower index. The distances to the pivots come from the scoring
// contraction run with the pivot rows in place of the text rows (max of the cosines). One
// block of 512 threads per request then draws the K_d tokens:
//
//   * The pool: the W candidates farthest from the pivots (W <= 128, about 2 K_d). Their
//     pairwise cosines are one small contraction (mma.sync over 256-column chunks of the
//     gathered rows, streamed through a ring of up to four chunks with cp.async) kept in
//     shared memory, so a step inside the pool costs an argmax over W and one row of it.
//   * Every candidate outside the pool keeps an upper bound of its distance (the distance to
//     the pivots, lowered when refreshed) and the number of picks the bound accounts for.
//     A distance only falls as picks are added, so the best pool candidate is the exact
//     FPS choice whenever it beats the largest bound outside (ties to the lower index).
//     Otherwise the outside candidate with the largest bound is brought up to date against
//     the picks it has not seen (one warp per pick): if it still leads it is drawn, and the
//     pool's distances are lowered by its cosines. Each candidate is refreshed at most once
//     per step, so a step ends after at most N rounds; the draw is exact for any W.
//
// Without pivots every candidate starts at distance +inf, so the first draw is row 0 (the
// lowest index); the host then runs the contraction with row 0 as the one pivot and the
// block records it as draw 0, so that no bound starts at +inf.
#include "fps.cuh"

namespace trevs {

constexpr int kFpsSlices = 4;                 // 64-column slices per staged chunk (256 columns)
constexpr int kFpsRingBytes = 128 * 1024;     // ring of staged chunks of the pool rows
constexpr int kFpsGramLd = kFpsMaxPool + 4;   // fp32 row stride of the pool cosines
constexpr int kFpsSmem = kFpsRingBytes + kFpsMaxPool * kFpsGramLd * 4 + 4 * kFpsMaxPool * 4;

// (d_a, i_a) comes before (d_b, i_b): farther, or as far and a lower index.
__device__ __forceinline__ bool fps_before(float da, int ia, float db, int ib) {
  return da > db || (da == db && ia < ib);
}

// cos(x, y) of two bf16 rows by one warp (0 when either row is zero).
__device__ float warp_row_cos(const __nv_bfloat16* x, const __nv_bfloat16* y, int d, int lane) {
  float dot = 0.f, xx = 0.f, yy = 0.f;
  for (int c = lane * 8; c < d; c += 256) {
    const uint4 u = *reinterpret_cast<const uint4*>(x + c);
    const uint4 v = *reinterpret_cast<const uint4*>(y + c);
    const uint32_t p[4] = {u.x, u.y, u.z, u.w}, q[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float pl = __uint_as_float(p[j] << 16), ph = __uint_as_float(p[j] & 0xFFFF0000u);
      const float ql = __uint_as_float(q[j] << 16), qh = __uint_as_float(q[j] & 0xFFFF0000u);
      dot = fmaf(pl, ql, dot); dot = fmaf(ph, qh, dot);
      xx = fmaf(pl, pl, xx);   xx = fmaf(ph, ph, xx);
      yy = fmaf(ql, ql, yy);   yy = fmaf(qh, qh, yy);
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    dot += __shfl_xor_sync(0xffffffffu, dot, o);
    xx += __shfl_xor_sync(0xffffffffu, xx, o);
    yy += __shfl_xor_sync(0xffffffffu, yy, o);
  }
  return (xx > 0.f && yy > 0.f) ? dot * (1.0f / sqrtf(xx)) * (1.0f / sqrtf(yy)) : 0.f;
}

// The outside candidate (stamp >= 0) with the largest bound, ties to the lower index, into
// (*s_o, *s_od); -1 when there is none. All threads call it.
__device__ void fps_outside_best(const float* ub, const int* stamp, int n, int* s_wi, float* s_wd, int* s_o,
                                 float* s_od) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  float bd = 0.f;
  int bi = -1;
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    if (stamp[i] >= 0) {
      const float u = ub[i];
      if (bi < 0 || fps_before(u, i, bd, bi)) { bd = u; bi = i; }
    }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float d2 = __shfl_xor_sync(0xffffffffu, bd, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
    if (i2 >= 0 && (bi < 0 || fps_before(d2, i2, bd, bi))) { bd = d2; bi = i2; }
  }
  if (lane == 0) { s_wi[warp] = bi; s_wd[warp] = bd; }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < nwarps; ++w)
      if (s_wi[w] >= 0 && (bi < 0 || fps_before(s_wd[w], s_wi[w], bd, bi))) { bd = s_wd[w]; bi = s_wi[w]; }
    *s_o = bi;
    *s_od = bd;
  }
  __syncthreads();
}

// Pool = the W candidates of largest distance to the pivots (ties to the lower index),
// ascending, with the keys in registers (n <= E * blockDim.x).
template <int E>
__device__ void fps_pool_reg(int n, const uint8_t* flags, const float* mc, bool seeded, int W, int* pool,
                             RegSelShared& rs) {
  uint32_t key[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = e * blockDim.x + threadIdx.x;
    key[e] = (i < n && flags[i] == 0) ? score_key(seeded ? 1.f - __ldcg(mc + i) : INFINITY) : 0u;
  }
  uint32_t tau;
  int need;
  block_reg_topk(key, W, rs, tau, need);
  block_reg_emit(key, 0u, tau, need, pool, rs);
}

__global__ void __launch_bounds__(kFpsThreads, 1) fps_kernel(const __grid_constant__ FpsMeta meta, const FpsArgs a) {
  extern __shared__ uint8_t fps_smem_raw[];
  __shared__ SelScratch sh;
  __shared__ int s_wi[32];
  __shared__ float s_wd[32];
  __shared__ int s_g, s_o, s_n;
  __shared__ float s_gd, s_od;
  pdl_launch_dependents();
  const FpsReq& r = meta.r[blockIdx.x];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nthr = blockDim.x;
  const int n = r.n, kd = r.kd, d = a.d;
  uint8_t* stage = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(fps_smem_raw) + 127) & ~uintptr_t(127));
  float* gram = reinterpret_cast<float*>(stage + kFpsRingBytes);
  int* pool = reinterpret_cast<int*>(gram + kFpsMaxPool * kFpsGramLd);
  float* pdist = reinterpret_cast<float*>(pool + kFpsMaxPool);
  float* prinv = pdist + kFpsMaxPool;
  int* ppick = reinterpret_cast<int*>(prinv + kFpsMaxPool);
  const int phase = a.phase;
  const int cap = phase == 0 ? kFpsMaxPool : min(kFpsMaxPoolBig, r.gram_ld);
  const float* ggram = phase == 2 ? a.gram + r.gram_off : nullptr;   // pool dot products (phase 2)
  if (phase == 1) {
    pool = a.pool_idx + r.pool_off;          // the pool goes to the workspace
  } else if (phase == 2) {
    // the staging ring is not used: the pool's arrays take its place
    pool = reinterpret_cast<int*>(stage);
    pdist = reinterpret_cast<float*>(pool + kFpsMaxPoolBig);
    prinv = pdist + kFpsMaxPoolBig;
    ppick = reinterpret_cast<int*>(prinv + kFpsMaxPoolBig);
  }
  pdl_wait();   // the pivots and their cosines come from the preceding grids
  if (kd <= 0 || n <= 0) return;
  const __nv_bfloat16* Zb = a.Z + (long long)r.n_off * a.z_stride;
  uint8_t* flags = a.flags + r.n_off;
  float* ub = a.ub + r.n_off;
  int* stamp = a.stamp + r.n_off;
  const float* mc = a.maxcos + r.n_off;
  const bool seeded = r.kr > 0;
  int* picks = a.picks + r.pick_off;

  // ---- candidates: every row that is not a pivot (an index outside [0, n) marks nothing)
  for (int i = tid; i < n; i += nthr) flags[i] = 0;
  __syncthreads();
  for (int j = tid; j < r.kr; j += nthr) {
    const int p = a.piv[r.piv_off + j];
    if (p >= 0 && p < n) flags[p] = 1;
  }
  if (tid == 0) s_n = 0;
  __syncthreads();
  {
    int c = 0;
    for (int i = tid; i < n; i += nthr) c += flags[i] == 0;
#pragma unroll
    for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0) atomicAdd(&s_n, c);
  }
  __syncthreads();
  const int ncand = s_n;
  const int t0 = r.lead;       // draws made before the loop
  int W = a.pool > 0 ? a.pool : fps_auto_pool(kd);
  W = min(W, min(ncand, cap));   // 0 only when the lead draw is the only one
  if (ncand < kd - t0) {   // the host checks K_d <= N - K_r; nothing to draw from otherwise
    if (tid == 0 && phase != 2) atomicOr(a.err, 2u);
    return;
  }

  // ---- the pool
  if (phase == 2) {
    for (int p = tid; p < W; p += nthr) pool[p] = __ldcg(a.pool_idx + r.pool_off + p);
  } else if (n <= 512) fps_pool_reg<1>(n, flags, mc, seeded, W, pool, sh.rs);
  else if (n <= 1024) fps_pool_reg<2>(n, flags, mc, seeded, W, pool, sh.rs);
  else if (n <= kRegSelMaxN) fps_pool_reg<8>(n, flags, mc, seeded, W, pool, sh.rs);
  else {
    uint32_t* keys = a.keys + (((size_t)r.n_off + 4 * (size_t)blockIdx.x + 3) & ~(size_t)3);
    uint32_t lo, hi, tau;
    int need, n_eq;
    block_fill_keys(keys, mc, n, [&](float x, int i) {
      return flags[i] == 0 ? score_key(seeded ? 1.f - x : INFINITY) : 0u;
    }, sh.ss, lo, hi);
    block_kth_largest(keys, n, W, sh.ss, lo, hi, tau, need, n_eq);
    block_emit_selected(keys, n, tau, need, sh.ss, [&](int i, int pos, bool sel) { if (sel) pool[pos] = i; });
  }
  __syncthreads();

  // ---- bounds of the candidates outside the pool (exact for the pivots and the lead draw)
  if (phase != 2) {
    if (t0 && tid == 0) {
      picks[0] = 0;
      if (a.pick_dist) a.pick_dist[r.pick_off] = INFINITY;
    }
    for (int i = tid; i < n; i += nthr) {
      const bool cand = flags[i] == 0;
      stamp[i] = cand ? t0 : -1;
      ub[i] = cand ? (seeded ? 1.f - __ldcg(mc + i) : INFINITY) : 0.f;
    }
    __syncthreads();
  }
  if (phase == 1) {   // the pool's own stamps; the cosines and draws follow in later grids
    for (int p = tid; p < W; p += nthr) stamp[pool[p]] = -1;
    if (tid == 0) a.pool_n[blockIdx.x] = W;
    return;
  }
  for (int p = tid; p < W; p += nthr) {
    const int i = pool[p];
    if (phase == 0) stamp[i] = -1;
    pdist[p] = seeded ? 1.f - __ldcg(mc + i) : INFINITY;
    ppick[p] = 0;
  }

  // ---- phase 2: 1 / ||z|| of the pool rows from the diagonal of their dot products
  if (phase == 2) {
    __syncthreads();
    for (int p = tid; p < W; p += nthr) {
      const float gpp = __ldcg(ggram + (long long)p * r.gram_ld + p);
      prinv[p] = gpp > 0.f ? 1.0f / sqrtf(gpp) : 0.f;
    }
  }

  // ---- cosines within the pool: G = Z_pool Z_pool^T (bf16 mma.sync, fp32), then normalised.
  // The pool rows stream through a ring of S chunks of 256 columns (S = 2..4 as W allows),
  // so that 64-96 KB are in flight while the block computes.
  if (phase == 0 && W > 0) {
    const int W16 = (W + 15) & ~15, nmt = W16 >> 4, nblk = nmt * nmt;
    const int slice_bytes = W16 * 128, chunk_bytes = kFpsSlices * slice_bytes;
    const int S = min(4, kFpsRingBytes / chunk_bytes);
    const int nch = (d + 64 * kFpsSlices - 1) / (64 * kFpsSlices);
    const uint32_t sbase = smem_u32(stage);
    auto load_chunk = [&](int ch, int slot) {
      for (int idx = tid; idx < W16 * 8 * kFpsSlices; idx += nthr) {
        const int row = idx >> 5, q = idx & 31, sl = q >> 3, c = q & 7;
        const int col = ch * 64 * kFpsSlices + q * 8;
        const bool ok = row < W && col < d;
        const void* src = ok ? (const void*)(Zb + (long long)pool[row] * a.z_stride + col) : (const void*)a.Z;
        cp_async16(sbase + slot * chunk_bytes + sl * slice_bytes + row * 128 + (swz(row, c) << 4), src, ok ? 16 : 0);
      }
    };
    float acc[4][2][4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int x = 0; x < 2; ++x)
#pragma unroll
        for (int y = 0; y < 4; ++y) acc[j][x][y] = 0.f;
    __syncthreads();   // pool[] is read by every thread's copies
    for (int c = 0; c < S - 1; ++c) {
      if (c < nch) load_chunk(c, c);
      cp_async_commit();
    }
    for (int ch = 0; ch < nch; ++ch) {
      // chunk ch is the oldest of the S - 1 groups in flight
      if (S == 4) cp_async_wait<2>();
      else if (S == 3) cp_async_wait<1>();
      else cp_async_wait<0>();
      __syncthreads();   // chunk ch is visible to all; slot (ch - 1) % S is free again
      if (ch + S - 1 < nch) load_chunk(ch + S - 1, (ch + S - 1) % S);
      cp_async_commit();
      const uint32_t B0 = sbase + (ch % S) * chunk_bytes;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int bi = warp + 16 * j;   // 16 x 16 output block (mt, pr)
        if (bi < nblk) {
          const int mt = bi / nmt, pr = bi - mt * nmt;
#pragma unroll
          for (int sl = 0; sl < kFpsSlices; ++sl) {
            const uint32_t Bs = B0 + sl * slice_bytes;
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
              uint32_t af[4];
              const int ar = mt * 16 + (lane & 15), ac = 2 * ks + (lane >> 4);
              ldmatrix_x4(Bs + ar * 128 + (swz(ar, ac) << 4), af[0], af[1], af[2], af[3]);
              const int mi = lane >> 3;
              const int br = pr * 16 + 8 * (mi >> 1) + (lane & 7), bc = 2 * ks + (mi & 1);
              uint32_t b0, b1, b2, b3;
              ldmatrix_x4(Bs + br * 128 + (swz(br, bc) << 4), b0, b1, b2, b3);
              mma_bf16_16816(acc[j][0], af, b0, b1);
              mma_bf16_16816(acc[j][1], af, b2, b3);
            }
          }
        }
      }
    }
    cp_async_wait<0>();
    const int g = lane >> 2, t4 = lane & 3;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int bi = warp + 16 * j;
      if (bi < nblk) {
        const int mt = bi / nmt, pr = bi - mt * nmt;
#pragma unroll
        for (int x = 0; x < 2; ++x) {
          const int col = pr * 16 + 8 * x + 2 * t4, r0 = mt * 16 + g;
          gram[r0 * kFpsGramLd + col] = acc[j][x][0];
          gram[r0 * kFpsGramLd + col + 1] = acc[j][x][1];
          gram[(r0 + 8) * kFpsGramLd + col] = acc[j][x][2];
          gram[(r0 + 8) * kFpsGramLd + col + 1] = acc[j][x][3];
        }
      }
    }
    __syncthreads();
    for (int p = tid; p < W; p += nthr) {
      const float gpp = gram[p * kFpsGramLd + p];
      prinv[p] = gpp > 0.f ? 1.0f / sqrtf(gpp) : 0.f;
    }
    __syncthreads();
    for (int x = tid; x < W * W; x += nthr) {
      const int p = x / W, q = x - p * W;
      gram[p * kFpsGramLd + q] = gram[p * kFpsGramLd + q] * prinv[p] * prinv[q];
    }
  }
  __syncthreads();

  fps_outside_best(ub, stamp, n, s_wi, s_wd, &s_o, &s_od);

  // ---- the K_d steps
  for (int t = t0; t < kd; ++t) {
    for (int round = 0;; ++round) {
      if (warp == 0) {
        float bd = 0.f;
        int bp = -1;
        for (int p = lane; p < W; p += 32)
          if (!ppick[p] && (bp < 0 || fps_before(pdist[p], p, bd, bp))) { bd = pdist[p]; bp = p; }
#pragma unroll
        for (int o = 16; o; o >>= 1) {   // pool positions are in index order
          const float d2 = __shfl_xor_sync(0xffffffffu, bd, o);
          const int p2 = __shfl_xor_sync(0xffffffffu, bp, o);
          if (p2 >= 0 && (bp < 0 || fps_before(d2, p2, bd, bp))) { bd = d2; bp = p2; }
        }
        if (lane == 0) { s_g = bp; s_gd = bd; }
      }
      __syncthreads();
      const int gp = s_g, o = s_o;
      const float gd = s_gd, od = s_od;
      const int gi = gp >= 0 ? pool[gp] : -1;
      int act;   // 0: draw from the pool; 1: draw the outside candidate; 2: refresh it; 3: none left
      if (gp >= 0 && (o < 0 || fps_before(gd, gi, od, o))) act = 0;
      else if (o < 0 || round > n) act = 3;
      else act = stamp[o] == t ? 1 : 2;
      __syncthreads();   // s_g / s_o are rewritten below
      if (act == 3) {
        if (tid == 0) atomicOr(a.err, 2u);
        return;
      }
      if (act == 0) {
        if (tid == 0) {
          picks[t] = gi;
          if (a.pick_dist) a.pick_dist[r.pick_off + t] = gd;
          ppick[gp] = 1;
          flags[gi] = 2;
        }
        if (phase == 0) {
          for (int p = tid; p < W; p += nthr) pdist[p] = fminf(pdist[p], 1.f - gram[gp * kFpsGramLd + p]);
        } else {
          const float* grow = ggram + (long long)gp * r.gram_ld;
          const float rg = prinv[gp];
          for (int p = tid; p < W; p += nthr) pdist[p] = fminf(pdist[p], 1.f - __ldcg(grow + p) * rg * prinv[p]);
        }
        __syncthreads();
        break;
      }
      if (act == 1) {
        if (tid == 0) {
          picks[t] = o;
          if (a.pick_dist) a.pick_dist[r.pick_off + t] = od;
          stamp[o] = -1;
          flags[o] = 2;
        }
        const __nv_bfloat16* zo = Zb + (long long)o * a.z_stride;
        for (int p = warp; p < W; p += nthr >> 5) {
          if (ppick[p]) continue;
          const float c = warp_row_cos(Zb + (long long)pool[p] * a.z_stride, zo, d, lane);
          if (lane == 0) pdist[p] = fminf(pdist[p], 1.f - c);
        }
        __syncthreads();
        fps_outside_best(ub, stamp, n, s_wi, s_wd, &s_o, &s_od);
        break;
      }
      // act == 2: the bound of o against the picks it has not seen
      const int s0 = stamp[o];
      const __nv_bfloat16* zo = Zb + (long long)o * a.z_stride;
      float m = INFINITY;
      for (int k = s0 + warp; k < t; k += nthr >> 5)
        m = fminf(m, 1.f - warp_row_cos(zo, Zb + (long long)picks[k] * a.z_stride, d, lane));
      if (lane == 0) s_wd[warp] = m;
      __syncthreads();
      if (tid == 0) {
        for (int w = 0; w < (nthr >> 5); ++w) m = fminf(m, s_wd[w]);
        ub[o] = fminf(ub[o], m);
        stamp[o] = t;
      }
      __syncthreads();
      fps_outside_best(ub, stamp, n, s_wi, s_wd, &s_o, &s_od);
    }
  }

  // ---- S_r and S_d together, ascending
  if (a.kept) {
    __syncthreads();
    block_compact_flags(flags, n, a.kept + r.kept_off, sh.ss);
  }
}

// Dot products of the pool rows of the requests drawing from pools above kFpsMaxPool, for
// phase 2: one block of four warps per 64 x 64 tile of a request's W x W matrix. The two row
// sets stream through shared memory in 64-column chunks (cp.async, two stages, 128-byte
// swizzled rows); each warp takes 16 rows x 64 columns with mma.sync (bf16 in, fp32 out).
constexpr int kGramThreads = 128;
constexpr int kGramChunk = 64;                                  // columns per staged chunk
constexpr int kGramStage = 2 * kFpsGramTile * kGramChunk * 2;   // rows of both sets: 16 KB

__global__ void __launch_bounds__(kGramThreads) fps_gram_kernel(const __grid_constant__ FpsMeta meta,
                                                                const FpsArgs a) {
  __shared__ __align__(128) uint8_t stage[2 * kGramStage];
  pdl_wait();   // the pools come from the preceding grid
  const int b = find_request(meta.B, blockIdx.x, [&](int i) { return meta.r[i].gt_off; });
  const FpsReq& r = meta.r[b];
  const int nt = r.gram_ld / kFpsGramTile;
  const int t = blockIdx.x - r.gt_off;
  const int ti = t / nt, tj = t - ti * nt;
  const int W = __ldcg(a.pool_n + b);
  if (ti * kFpsGramTile >= W || tj * kFpsGramTile >= W) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int* pool = a.pool_idx + r.pool_off;
  const __nv_bfloat16* Zb = a.Z + (long long)r.n_off * a.z_stride;
  const int d = a.d, nch = (d + kGramChunk - 1) / kGramChunk;
  const uint32_t sbase = smem_u32(stage);
  // row x of a chunk: set 0 (rows ti), set 1 (rows tj); 8 pieces of 16 bytes each
  auto load_chunk = [&](int ch, int slot) {
    for (int idx = tid; idx < 2 * kFpsGramTile * 8; idx += kGramThreads) {
      const int row = idx >> 3, c = idx & 7, set = row / kFpsGramTile, rr = row - set * kFpsGramTile;
      const int p = (set ? tj : ti) * kFpsGramTile + rr;
      const int col = ch * kGramChunk + c * 8;
      const bool ok = p < W && col < d;
      const void* src = ok ? (const void*)(Zb + (long long)__ldcg(pool + p) * a.z_stride + col) : (const void*)a.Z;
      cp_async16(sbase + slot * kGramStage + row * 128 + (swz(row, c) << 4), src, ok ? 16 : 0);
    }
  };
  float acc[4][2][4];
#pragma unroll
  for (int j = 0; j < 4; ++j)
#pragma unroll
    for (int x = 0; x < 2; ++x)
#pragma unroll
      for (int y = 0; y < 4; ++y) acc[j][x][y] = 0.f;
  load_chunk(0, 0);
  cp_async_commit();
  for (int ch = 0; ch < nch; ++ch) {
    if (ch + 1 < nch) load_chunk(ch + 1, (ch + 1) & 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const uint32_t A = sbase + (ch & 1) * kGramStage, B = A + kFpsGramTile * 128;
#pragma unroll
    for (int ks = 0; ks < kGramChunk / 16; ++ks) {
      uint32_t af[4];
      const int ar = warp * 16 + (lane & 15), ac = 2 * ks + (lane >> 4);
      ldmatrix_x4(A + ar * 128 + (swz(ar, ac) << 4), af[0], af[1], af[2], af[3]);
#pragma unroll
      for (int j = 0; j < 4; ++j) {   // 16-column block j of the tile
        const int mi = lane >> 3;
        const int br = j * 16 + 8 * (mi >> 1) + (lane & 7), bc = 2 * ks + (mi & 1);
        uint32_t b0, b1, b2, b3;
        ldmatrix_x4(B + br * 128 + (swz(br + kFpsGramTile, bc) << 4), b0, b1, b2, b3);
        mma_bf16_16816(acc[j][0], af, b0, b1);
        mma_bf16_16816(acc[j][1], af, b2, b3);
      }
    }
    __syncthreads();   // the slot is refilled next
  }
  cp_async_wait<0>();
  const int g = lane >> 2, t4 = lane & 3;
  float* out = a.gram + r.gram_off;
#pragma unroll
  for (int j = 0; j < 4; ++j)
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      const int col = tj * kFpsGramTile + j * 16 + 8 * x + 2 * t4;
      const int r0 = ti * kFpsGramTile + warp * 16 + g;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int row = r0 + 8 * h;
        if (row < W) {
          if (col < W) out[(long long)row * r.gram_ld + col] = acc[j][x][2 * h];
          if (col + 1 < W) out[(long long)row * r.gram_ld + col + 1] = acc[j][x][2 * h + 1];
        }
      }
    }
}

cudaError_t launch_fps(const FpsMeta& meta, const FpsArgs& a, cudaStream_t st, bool pdl) {
  if (meta.B == 0) return cudaSuccess;
  return launch_kernel(fps_kernel, dim3(meta.B), dim3(kFpsThreads), kFpsSmem + 128, st, pdl, meta, a);
}

cudaError_t launch_fps_gram(const FpsMeta& meta, const FpsArgs& a, int tiles, cudaStream_t st) {
  if (meta.B == 0 || tiles == 0) return cudaSuccess;
  return launch_kernel(fps_gram_kernel, dim3(tiles), dim3(kGramThreads), 0, st, true, meta, a);
}

}  // namespace trevs
