// Stage 1 (pre-LLM, Sec. 4.1): textual-relevance scores (Eq. 4-5), selection (Sec. 3.1 ratio
// split or Eq. 6-7 fused score) and gather of the kept feature rows.
#include <cmath>

#include "pre_llm.cuh"
#include "sm100.cuh"

namespace trevs {

// ------------------------------------------------------------------ scoring contraction
//
// A persistent grid, one CTA per SM, scores the visual rows of every request against the M
// text rows of that request. Each request is cut into tiles of 128 rows (its last tile may
// be shorter), and each tile into Z stages of 256 columns. Work is counted in (tile, stage)
// units, tile by tile; CTA c takes the contiguous units [W c / P, W (c + 1) / P), so that
// every CTA streams the same number of stages. A tile whose stages are split between CTAs
// leaves partial sums of G and ||z||^2 in the workspace (at most two per CTA: where its
// range starts and where it ends), and pre_finish_kernel adds them up in stage order.
//
// For each sub-tile the 5th-generation tensor cores compute G = Z_sub . T^T (UMMA M = 128,
// N = M_b rounded up to 16) into one of two TMEM accumulators, while eight warps sum the
// squares ||z_i||^2 from the same shared-memory stages. Four epilogue warps read a finished
// accumulator while the next sub-tile streams into the other, and form
// m_ji = max(G_ji / (||t_j|| ||z_i||), 0) and s^t_i = sqrt(sum_j m_ji^2 / M) with 1 / ||t_j||
// from the pre-pass; the [M, N] similarity never reaches memory. Selection runs in the next
// grid of the stream.
//
// Operands. Z arrives in stages of 128 rows x 256 columns: one 3D TMA box per 8 rows covers
// four 64-column slices (512 contiguous bytes of each row, 4 KB per copy), which streams HBM
// at full rate; in shared memory the 1 KB swizzle atoms of one slice lie 4 KB apart, which
// the UMMA descriptor states as its stride between 8-row groups. The SM's TMA engine is
// left to Z alone: T (hot in L2) is copied by two warps with cp.async into its own ring, in
// the same 128-byte swizzled layout, each slot holding 1, 2 or 4 consecutive slices (as many
// as fit), so that the MMA issuer synchronises once per slot rather than once per slice.
//
// Warp roles: 0 = TMA producer (Z), 1 = TMEM owner and MMA issuer, 2..3 = T copies,
// 4..7 = epilogue (warp w reads TMEM lanes 32*(w%4) .. +31), 8..15 = Z norms (two threads
// per row, two slices each). When every request has more than 112 text rows (kTHeavy), a
// stage brings in as much T as Z and the MMA issuer waits on T: warps 8..11 copy T as well,
// and warps 12..15 take the Z norms, one thread per row. (Measured on GB300: the 2 x 16,384
// batch with 128 text rows drops from 111.9 to 105.6 us per call; batches with at most 64
// text rows lose 5-8 us the same way, as their norms, not T, hold the stages.)

constexpr int kTileRows = kScoreTileRows;
constexpr int kChunk = 64;                     // d' columns per slice (one 128-byte swizzle row)
constexpr int kZSlices = 4;                    // slices per Z stage
constexpr int kZBoxRows = 8;                   // rows per Z copy (one swizzle atom per slice)
constexpr int kZBoxBytes = kZBoxRows * kZSlices * 128;
constexpr int kZStageBytes = kTileRows * kZSlices * 128;
constexpr int kMaxZStages = 4;
constexpr int kMaxTSlots = 8;
constexpr int kScoreThreads = 512;
template <bool kTHeavy> constexpr int kZNormWarps = kTHeavy ? 4 : 8;
template <bool kTHeavy> constexpr int kTCopyThreads = kTHeavy ? 192 : 64;
constexpr int kRingBudget = 200 * 1024;

struct ScoreLaunch {
  int z_stages;
  int t_slots;
  int t_slot_slices;  // 64-column slices per T slot (1, 2 or 4)
  int t_slice_bytes;  // bytes of one slice of T in a slot (M rounded up to 16 rows x 128)
  int acc_cols;       // TMEM columns of one accumulator (power of two >= 32)
  int mld;            // row length of a partial G (max M rounded up to 4)
  int bound[kMaxScoreCtas + 1];   // CTA c takes stage units [bound[c], bound[c + 1])
};

// Floats of one partial-sum slot: G [128][mld], then ||z||^2 [128].
__host__ __device__ inline long long score_slot_floats(int mld) { return (long long)kTileRows * mld + kTileRows; }

struct SubTile {
  int b, row0, h;   // request, its first row, rows (1..128)
  int tile;         // tile index over the launch
  int zs0, zs1;     // Z stages [zs0, zs1) of the tile
  int slot;         // -1: the whole tile; 0 / 1: partial sums of the range's first / last tile
};

// Scoring CTA whose stage units [bound[c], bound[c + 1]) contain unit u.
inline int score_cta_of(int u, const int* bound, int P) {
  int lo = 0, hi = P - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (bound[mid] <= u) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Calls f(segment) for the tiles of stage units [u0, u1) in order; f returns false to stop.
template <class F>
__device__ __forceinline__ void for_each_subtile(const PreMeta& meta, int nzs, long long u0, long long u1, F f) {
  if (u0 >= u1) return;
  int b = find_request(meta.B, (int)(u0 / nzs), [&](int i) { return meta.r[i].tile_off; });
  for (long long u = u0; u < u1;) {
    const int t = (int)(u / nzs);
    const int zs0 = (int)(u - (long long)t * nzs);
    const int zs1 = (int)min((long long)nzs, zs0 + (u1 - u));
    while (b + 1 < meta.B && meta.r[b + 1].tile_off <= t) ++b;
    const PreReq& r = meta.r[b];
    const int row0 = (t - r.tile_off) * kTileRows;
    const int slot = (zs0 == 0 && zs1 == nzs) ? -1 : (u == u0 ? 0 : 1);
    if (!f(SubTile{b, row0, min(kTileRows, r.n - row0), t, zs0, zs1, slot})) return;
    u += zs1 - zs0;
  }
}

// kSeed: the "text" rows are the pivot rows of Z (gathered beforehand) and each row's output
// is the largest cosine to them, unrectified (the distances of farthest point sampling, Sec. 3.1).
template <bool kSeed, bool kTHeavy>
__global__ void __launch_bounds__(kScoreThreads, 1)
    pre_score_kernel(const __grid_constant__ CUtensorMap tmZ3, const __grid_constant__ CUtensorMap tmZ2,
                     const __grid_constant__ PreMeta meta, const PreArgs a, const ScoreLaunch L) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t zfull[kMaxZStages], zempty[kMaxZStages];
  __shared__ __align__(8) uint64_t tfull[kMaxTSlots], tempty[kMaxTSlots];
  __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2], norm_full[2], norm_empty[2], mma_drain;
  __shared__ uint32_t tmem_base_s;
  __shared__ float rinv_s[4][256];   // one row per epilogue warp (no cross-warp barrier)
  __shared__ float zsq_s[2][2][kTileRows];   // [buffer][half of the columns][row]
  __shared__ volatile int s_abort;
  __shared__ volatile int s_zissued;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t zbase = smem_u32(smem);
  const uint32_t tbase = zbase + L.z_stages * kZStageBytes;   // after the Z stages
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = a.d;
  const int nk = (d + kChunk - 1) / kChunk;                 // 64-column slices
  const int nzs = (nk + kZSlices - 1) / kZSlices;           // Z stages per tile
  const long long u0 = L.bound[blockIdx.x], u1 = L.bound[blockIdx.x + 1];
  const bool ragged = (d % (kChunk * kZSlices)) != 0;       // last Z stage copied slice by slice
  // word 1 of the workspace header, when set, replaces the 2 s limit of every wait (microseconds)
  const uint32_t lim_us = __ldcg(a.err + 1);
  const uint64_t lim = lim_us ? (uint64_t)lim_us * 1000ull : 2000000000ull;
  const int SZ = L.z_stages, ST = L.t_slots, TS = L.t_slot_slices;
  const int t_slot_bytes = TS * L.t_slice_bytes;

  if (tid == 0) {
    for (int s = 0; s < SZ; ++s) {
      mbar_init(smem_u32(&zfull[s]), 1);
      mbar_init(smem_u32(&zempty[s]), 1 + kZNormWarps<kTHeavy>);   // MMA commit + the Z-norm warps
    }
    for (int s = 0; s < ST; ++s) {
      mbar_init(smem_u32(&tfull[s]), kTCopyThreads<kTHeavy>);      // the copy lanes, once their copies land
      mbar_init(smem_u32(&tempty[s]), 1);                 // MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&acc_full[i]), 1);
      mbar_init(smem_u32(&acc_empty[i]), 4);              // the epilogue warps
      mbar_init(smem_u32(&norm_full[i]), kZNormWarps<kTHeavy>);
      mbar_init(smem_u32(&norm_empty[i]), 4);
    }
    mbar_init(smem_u32(&mma_drain), 1);
    s_abort = 0;
    s_zissued = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), (uint32_t)(2 * L.acc_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  pdl_launch_dependents();   // the selection grid may start launching

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmZ3);
      tma_prefetch_desc(&tmZ2);
      const uint64_t pz = l2_policy_evict_first();   // Z is streamed once
      int gz = 0;
      for_each_subtile(meta, nzs, u0, u1, [&](const SubTile& t) {
        const PreReq& r = meta.r[t.b];
        const int nzb = (t.h + kZBoxRows - 1) / kZBoxRows;
        const int y0 = r.n_off + t.row0;
        for (int zs = t.zs0; zs < t.zs1; ++zs, ++gz) {
          const int s = gz % SZ, it = gz / SZ;
          if (gz >= SZ && !mbar_wait(smem_u32(&zempty[s]), (it - 1) & 1, &s_abort, lim)) {
            s_abort = 1;
            return false;
          }
          const uint32_t A = zbase + s * kZStageBytes;
          const uint32_t fb = smem_u32(&zfull[s]);
          const int k0 = zs * kZSlices;
          const int ns = min(kZSlices, nk - k0);
          if (!(ragged && zs == nzs - 1)) {
            mbar_arrive_expect_tx(fb, (uint32_t)(nzb * kZBoxBytes));
            for (int zb = 0; zb < nzb; ++zb) tma_load_3d(A + zb * kZBoxBytes, &tmZ3, 0, y0 + zb * kZBoxRows, k0, fb, pz);
          } else {
            // last, partial stage: slice by slice from the 2D map (zero fill beyond d')
            mbar_arrive_expect_tx(fb, (uint32_t)(nzb * ns * kZBoxRows * 128));
            for (int zb = 0; zb < nzb; ++zb)
              for (int c = 0; c < ns; ++c)
                tma_load_2d(A + zb * kZBoxBytes + c * 1024, &tmZ2, (k0 + c) * kChunk, y0 + zb * kZBoxRows, fb, pz);
          }
          s_zissued = gz + 1;
        }
        return true;
      });
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int gz = 0, gt = 0, j = 0;
      for_each_subtile(meta, nzs, u0, u1, [&](const SubTile& t) {
        const int buf = j & 1, use = j >> 1;
        if (j >= 2 && !mbar_wait(smem_u32(&acc_empty[buf]), (use - 1) & 1, &s_abort, lim)) {
          s_abort = 1;
          return false;
        }
        tc_fence_after();
        const uint32_t dg = tmem + (uint32_t)(buf * L.acc_cols);
        const uint32_t idesc = umma_idesc_bf16(kTileRows, (meta.r[t.b].m + 15) & ~15);
        int kc = 0;   // slice index within the sub-tile
        for (int zs = t.zs0; zs < t.zs1; ++zs, ++gz) {
          const int s = gz % SZ, it = gz / SZ;
          if (!mbar_wait(smem_u32(&zfull[s]), it & 1, &s_abort, lim)) {
            s_abort = 1;
            return false;
          }
          const uint32_t A = zbase + s * kZStageBytes;
          const int ns = min(kZSlices, nk - zs * kZSlices);
          for (int c0 = 0; c0 < ns; c0 += TS, ++gt) {
            const int ts = gt % ST, tit = gt / ST;
            if (!mbar_wait(smem_u32(&tfull[ts]), tit & 1, &s_abort, lim)) {
              s_abort = 1;
              return false;
            }
            fence_proxy_async_smem();   // the slot was written by cp.async (generic proxy)
            tc_fence_after();
            const uint32_t B = tbase + ts * t_slot_bytes;
            const int nsl = min(TS, ns - c0);
            for (int c = 0; c < nsl; ++c, ++kc) {
#pragma unroll
              for (int k = 0; k < kChunk / 16; ++k)
                umma_bf16(dg, umma_desc_sw128(A + (c0 + c) * 1024 + 32 * k, kZSlices * 1024),
                          umma_desc_sw128(B + c * L.t_slice_bytes + 32 * k), idesc, (kc | k) != 0);
            }
            umma_commit(smem_u32(&tempty[ts]));   // frees the T slot once these MMAs have read it
          }
          umma_commit(smem_u32(&zempty[s]));      // and the Z stage
        }
        umma_commit(smem_u32(&acc_full[buf]));    // this sub-tile's accumulator is complete
        ++j;
        return true;
      });
      if (s_abort) {
        // no MMA may still write TMEM when it is released: wait for every one issued
        const volatile int no_abort = 0;
        umma_commit(smem_u32(&mma_drain));
        mbar_wait(smem_u32(&mma_drain), 0, &no_abort, 500000000ull);
      }
    }
  } else if (warp < 4 || (kTHeavy && warp >= 8 && warp < 12)) {
    // T copies: the slices of the next slot from the request's M text rows, piece p = 16
    // bytes (row p / 8, 16-byte column p % 8 of a slice), swizzled like a TMA
    // 128-byte-swizzle box; slice c of a slot lies t_slice_bytes after slice c - 1
    const int ct = warp < 4 ? tid - 64 : 64 + (tid - 256);
    int gt = 0;
    for_each_subtile(meta, nzs, u0, u1, [&](const SubTile& st) {
      const PreReq& r = meta.r[st.b];
      const int pieces = r.m * 8;
      const uint8_t* tsrc = reinterpret_cast<const uint8_t*>(a.T + (long long)r.m_off * a.t_stride);
      for (int zs = st.zs0; zs < st.zs1; ++zs) {
        const int ns = min(kZSlices, nk - zs * kZSlices);
        for (int c0 = 0; c0 < ns; c0 += TS, ++gt) {
          const int ts = gt % ST, tit = gt / ST;
          if (gt >= ST && !mbar_wait(smem_u32(&tempty[ts]), (tit - 1) & 1, &s_abort, lim)) {
            s_abort = 1;
            return false;
          }
          const uint32_t B = tbase + ts * t_slot_bytes;
          const int nsl = min(TS, ns - c0);
          for (int c = 0; c < nsl; ++c) {
            const int kc = zs * kZSlices + c0 + c;
            const uint32_t Bc = B + c * L.t_slice_bytes;
            for (int p = ct; p < pieces; p += kTCopyThreads<kTHeavy>) {
              const int row = p >> 3, q = p & 7;
              const int col = kc * kChunk + q * 8;
              const uint8_t* src = tsrc + ((long long)row * a.t_stride + (col < d ? col : 0)) * 2;
              cp_async16(Bc + row * 128 + (swz(row, q) << 4), src, col < d ? 16 : 0);   // zero past d'
            }
          }
          cp_async_arrive_noinc(smem_u32(&tfull[ts]));
        }
      }
      return true;
    });
    cp_async_wait_all();
  } else if (warp >= (kTHeavy ? 12 : 8)) {
    // Z norms: thread zt owns row zt % 128 of every sub-tile, slices 2 (zt / 128) and + 1 of
    // every stage (with kTHeavy, all four slices)
    const int zt = tid - (kTHeavy ? 384 : 256);
    const int row = zt & (kTileRows - 1), half = kTHeavy ? 0 : zt >> 7;
    constexpr int kSl = kTHeavy ? kZSlices : 2;   // slices of a stage per thread
    int gz = 0, j = 0;
    for_each_subtile(meta, nzs, u0, u1, [&](const SubTile& st) {
      const int buf = j & 1, use = j >> 1;
      float2 acc2[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
      const bool mine = row < st.h;
      for (int zs = st.zs0; zs < st.zs1; ++zs, ++gz) {
        const int s = gz % SZ, it = gz / SZ;
        if (!mbar_wait(smem_u32(&zfull[s]), it & 1, &s_abort, lim)) {
          s_abort = 1;
          return false;
        }
        if (mine) {
          const uint8_t* rowp = smem + s * kZStageBytes + (row >> 3) * kZBoxBytes + (row & 7) * 128;
          const int ncols = min(kZSlices * kChunk, d - zs * kZSlices * kChunk);   // columns of this stage
#pragma unroll
          for (int c = kSl * half; c < kSl * half + kSl; ++c) {
#pragma unroll
            for (int qq = 0; qq < 8; ++qq) {
              if (c * kChunk + qq * 8 < ncols)   // d' is a multiple of 8: whole 16-byte pieces
                bf16_sq_acc8x2(*reinterpret_cast<const uint4*>(rowp + c * 1024 + (swz(row, qq) << 4)), acc2);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&zempty[s]));
      }
      if (j >= 2 && !mbar_wait(smem_u32(&norm_empty[buf]), (use - 1) & 1, &s_abort, lim)) {
        s_abort = 1;
        return false;
      }
      zsq_s[buf][half][row] = ((acc2[0].x + acc2[0].y) + (acc2[1].x + acc2[1].y)) + ((acc2[2].x + acc2[2].y) + (acc2[3].x + acc2[3].y));
      if (kTHeavy) zsq_s[buf][1][row] = 0.f;
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&norm_full[buf]));
      ++j;
      return true;
    });
  } else {
    const int q = warp & 3;             // TMEM lane quarter of this warp
    const int row = 32 * q + lane;      // sub-tile row owned by this thread
    float* rt = rinv_s[q];
    pdl_wait();                         // 1 / ||t|| come from the pre-pass
    int j = 0;
    for_each_subtile(meta, nzs, u0, u1, [&](const SubTile& st) {
      const PreReq& r = meta.r[st.b];
      const int m = r.m;
      const int buf = j & 1, use = j >> 1;
      __syncwarp();
      for (int c = lane; c < m; c += 32) rt[c] = __ldcg(a.t_rinv + r.m_off + c);
      __syncwarp();
      bool ok = mbar_wait(smem_u32(&acc_full[buf]), use & 1, &s_abort, lim);
      ok = ok && mbar_wait(smem_u32(&norm_full[buf]), use & 1, &s_abort, lim);
      ok = __all_sync(0xffffffffu, ok && !s_abort);
      if (!ok) {
        s_abort = 1;
        return false;
      }
      tc_fence_after();
      const uint32_t lane_base = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * L.acc_cols);
      const float zsq = zsq_s[buf][0][row] + zsq_s[buf][1][row];
      const float rz = zsq > 0.f ? 1.0f / sqrtf(zsq) : 0.f;
      float sum = 0.f, mx = -INFINITY;
      if (st.slot < 0) {
        for (int c0 = 0; c0 < m; c0 += 32) {
          float v[32];
          tmem_ld_32x32b_x32(lane_base + (uint32_t)c0, v);
#pragma unroll
          for (int jj = 0; jj < 32; ++jj) {
            if (c0 + jj < m) {
              if constexpr (kSeed) {
                mx = fmaxf(mx, v[jj] * rt[c0 + jj] * rz);
              } else {
                const float x = fmaxf(v[jj] * rt[c0 + jj] * rz, 0.f);
                sum = fmaf(x, x, sum);
              }
            }
          }
        }
      } else {
        // A tile split between CTAs: leave this CTA's partial sums (G row, columns
        // 0 .. round_up(m, 4), and ||z||^2) in its slot for pre_finish_kernel.
        const long long sf = score_slot_floats(L.mld);
        float* own = a.part + (2 * (long long)blockIdx.x + st.slot) * sf;
        float* g = own + (long long)row * L.mld;
        for (int c0 = 0; c0 < m; c0 += 32) {
          float v[32];
          tmem_ld_32x32b_x32(lane_base + (uint32_t)c0, v);
#pragma unroll
          for (int jj = 0; jj < 32; jj += 4)
            if (c0 + jj < m) *reinterpret_cast<float4*>(g + c0 + jj) = make_float4(v[jj], v[jj + 1], v[jj + 2], v[jj + 3]);
        }
        own[(long long)kTileRows * L.mld + row] = zsq;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_u32(&acc_empty[buf]));
        mbar_arrive(smem_u32(&norm_empty[buf]));
      }
      if (st.slot < 0 && row < st.h) {
        float* out = a.s_t + r.n_off + st.row0 + row;
        if constexpr (kSeed) *out = a.seed_merge ? fmaxf(mx, __ldcg(out)) : mx;
        else *out = sqrtf(sum / (float)m);
      }
      ++j;
      return true;
    });
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)(2 * L.acc_cols));
  }
  if (s_abort) {
    // let the copies already issued land before the block's shared memory is released
    if (tid == 0) {
      const volatile int no_abort = 0;
      const int zi = s_zissued;
      for (int g = zi - SZ > 0 ? zi - SZ : 0; g < zi; ++g)
        mbar_wait(smem_u32(&zfull[g % SZ]), (g / SZ) & 1, &no_abort, 500000000ull);
      atomicOr(a.err, 1u);
    }
    return;
  }
}

// Finishing grid of stage 1, one CTA per job. A job with tile >= 0 is a tile split between
// scoring CTAs: s^t of its rows from the partial sums its contributors left, added in stage
// order, with whole rows per load instruction (an SM takes in only about 45 GB/s from L2,
// so half-used sectors would double the time). The host lists the jobs (tile, request, first
// contributor, contributor count, slot of the first contributor, jobs of the request);
// requests without a split tile get one job with tile = -1. The last job of a request to
// finish (a ticket per request, reset by that job) goes on with the request's selection
// (Sec. 3.1) or fused scores (Eq. 6-7).
constexpr int kFinishThreads = 4 * kTileRows;
struct FinJob {
  int tile, b, c0, nc, slot0, count;
};
struct FinMeta {
  int njobs, mld;
  FinJob job[kMaxScoreCtas + kMaxChunk];
};

template <bool kSeed>
__device__ inline void fixup_tile(const FinJob& jb, const PreReq& r, int mld, const PreArgs& a) {
  // Warp w owns rows 8w .. 8w + 7 of the tile. A row's partial sums are mld contiguous floats:
  // P lanes (a power of two, 4..32) read it as consecutive 16-byte groups, so each load
  // instruction covers whole rows; lane gl of a segment owns groups gl, gl + P.
  const int row0 = (jb.tile - r.tile_off) * kTileRows;
  const int h = min(kTileRows, r.n - row0);
  const int m = r.m;
  const long long sf = score_slot_floats(mld);
  const int gpr = mld >> 2;
  int P = 4;
  while (P < gpr && P < 32) P <<= 1;
  const int RPW = 32 / P;                             // rows per warp pass (<= 8)
  const int ng = (gpr + P - 1) / P;                   // groups per lane (<= 2 for M <= 256)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int sub = lane / P, gl = lane % P;
  const float* p0 = a.part + (2 * (long long)jb.c0 + jb.slot0) * sf;
  float rt[2][4];
#pragma unroll
  for (int k = 0; k < 2; ++k)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int col = 4 * (gl + P * k) + e;
      rt[k][e] = (k < ng && col < m) ? __ldcg(a.t_rinv + r.m_off + col) : 0.f;
    }
  for (int pr = 0; pr < 8; pr += RPW) {
    const int row = 8 * warp + pr + sub;
    float4 acc[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
    float zsq = 0.f;
    for (int x0 = 0; x0 < jb.nc; x0 += 4) {           // four contributors' loads in flight
      float4 v[4][2];
      float zv[4];
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const bool live = x0 + x < jb.nc;
        const float* base = x0 + x == 0 ? p0 : a.part + 2 * (long long)(jb.c0 + x0 + x) * sf;
        zv[x] = (live && gl == 0) ? __ldcg(base + (long long)kTileRows * mld + row) : 0.f;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int g = gl + P * k;
          v[x][k] = (live && k < ng && g < gpr)
                        ? __ldcg(reinterpret_cast<const float4*>(base + (long long)row * mld + 4 * g))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
#pragma unroll
      for (int x = 0; x < 4; ++x) {                   // stage order: contributor c0 first
        zsq += zv[x];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          acc[k].x += v[x][k].x; acc[k].y += v[x][k].y; acc[k].z += v[x][k].z; acc[k].w += v[x][k].w;
        }
      }
    }
    const float zrow = __shfl_sync(0xffffffffu, zsq, lane - gl);
    const float rz = zrow > 0.f ? 1.0f / sqrtf(zrow) : 0.f;
    float sum = 0.f, mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const float gv[4] = {acc[k].x, acc[k].y, acc[k].z, acc[k].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (k < ng && 4 * (gl + P * k) + e < m) {
          if constexpr (kSeed) {
            mx = fmaxf(mx, gv[e] * rt[k][e] * rz);
          } else {
            const float xx = fmaxf(gv[e] * rt[k][e] * rz, 0.f);
            sum = fmaf(xx, xx, sum);
          }
        }
      }
    }
    if constexpr (kSeed) {
      for (int o = P >> 1; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (gl == 0 && row < h) {
        float* out = a.s_t + r.n_off + row0 + row;
        *out = a.seed_merge ? fmaxf(mx, __ldcg(out)) : mx;
      }
    } else {
      for (int o = P >> 1; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      if (gl == 0 && row < h) a.s_t[r.n_off + row0 + row] = sqrtf(sum / (float)m);
    }
  }
}

__global__ void __launch_bounds__(kFinishThreads, 1) pre_finish_kernel(const __grid_constant__ PreMeta meta,
                                                                       const __grid_constant__ FinMeta fm,
                                                                       const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelScratch sh;
  __shared__ int s_last;
  pdl_launch_dependents();   // the next grid (the gather) waits for this one to complete
  const FinJob& jb = fm.job[blockIdx.x];
  const PreReq& r = meta.r[jb.b];
  pdl_wait();   // partial sums and s^t come from the scoring grid (1 / ||t|| and rules from before it)
  if (a.action == kActFpsSeed) {   // pivot cosines: the split tiles only
    if (jb.tile >= 0) fixup_tile<true>(jb, r, fm.mld, a);
    return;
  }
  if (jb.tile >= 0) fixup_tile<false>(jb, r, fm.mld, a);
  if (jb.count > 1) {
    __threadfence();   // this job's s^t rows before its ticket
    __syncthreads();
    if (threadIdx.x == 0) {
      const uint32_t done = atomicAdd(a.counters + jb.b, 1u) + 1u;
      s_last = done == (uint32_t)jb.count;
      if (s_last) a.counters[jb.b] = 0u;   // ready for the next launch
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();   // the other jobs' rows, read through L2
  } else {
    __syncthreads();
  }
  if (a.big_sel && r.n > kRegSelMaxN) return;   // pre_select_big_kernel selects it
  select_request_512(a, r, jb.b, smem, smem_bytes, sh);
}

// Selection of the requests above kRegSelMaxN tokens, after the finishing grid: one block of
// 1,024 threads per request, keys and flags in shared memory (in global memory past its size),
// so that each pass over the keys takes half as long as with the finishing grid's 512.
constexpr int kBigSelThreads = 1024;
struct BigSel {
  int n;
  int b[kMaxChunk];
};

__global__ void __launch_bounds__(kBigSelThreads, 1) pre_select_big_kernel(const __grid_constant__ PreMeta meta,
                                                                           const __grid_constant__ BigSel bs,
                                                                           const PreArgs a, int smem_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelShared ss;
  pdl_wait();   // the finishing grid's s^t rows
  const int b = bs.b[blockIdx.x];
  select_request(a, meta.r[b], b, smem, smem_bytes, ss, a.mode == kModeFused && !a.s_fused_given,
                 a.action == kActSelect);
}

// Pre-pass, run ahead of the scoring grid. Blocks [0, n_sal): the saliency side of the
// selection of request b = blockIdx.x (inputs only), so that the finishing grid only ranks
// textual relevance. Remaining blocks: 1 / ||t_j|| of the text rows, one warp per row with
// all of a row's loads (up to d = 4096) in flight.
__global__ void __launch_bounds__(512) pre_saliency_kernel(const __grid_constant__ PreMeta meta,
                                                           const PreArgs a, int smem_bytes, int n_sal) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SelScratch sh;
  pdl_launch_dependents();
  if ((int)blockIdx.x >= n_sal) {
    const long long row = (long long)(blockIdx.x - n_sal) * 16 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= a.total_m) return;
    const uint4* t = reinterpret_cast<const uint4*>(a.T + row * a.t_stride);
    const int nv = a.d / 8;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int p0 = 0; p0 < nv; p0 += 16 * 32) {
      uint4 v[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int p = p0 + 32 * q + lane;
        v[q] = p < nv ? __ldg(t + p) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int q = 0; q < 16; ++q) bf16_sq_acc8(v[q], acc);
    }
    float sq = (acc[0] + acc[1]) + (acc[2] + acc[3]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (lane == 0) a.t_rinv[row] = sq > 0.f ? 1.0f / sqrtf(sq) : 0.f;
    return;
  }
  const int b = blockIdx.x;
  const PreReq r = meta.r[b];
  const bool in_smem = (size_t)r.n * 4 + 16 <= (size_t)smem_bytes;
  const size_t gbase = ((size_t)r.n_off + 4 * (size_t)b + 3) & ~(size_t)3;
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + gbase;
  const int4 rule = saliency_rule_512(a, r, keys, sh);
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

// The same matrix seen as [cols / 64][rows][64] (only whole 64-column slices): a box of
// box_rows rows x `slices` consecutive slices lands as `slices` swizzle atoms, 1 KB apart.
static cudaError_t make_tmap_sliced(CUtensorMap* tm, const void* base, long long rows, int cols, long long stride,
                                    int box_rows, int slices) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return cudaErrorNotSupported;
  const int full = cols / kChunk;
  const cuuint64_t dims[3] = {(cuuint64_t)kChunk, (cuuint64_t)(rows > 0 ? rows : 1), (cuuint64_t)(full > 0 ? full : 1)};
  const cuuint64_t strides[2] = {(cuuint64_t)stride * 2, (cuuint64_t)kChunk * 2};
  const cuuint32_t box[3] = {(cuuint32_t)kChunk, (cuuint32_t)box_rows, (cuuint32_t)slices};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult res = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Tensor map of a [rows][heads][128] bf16 tensor with element strides tok_stride (rows) and
// head_stride (heads): boxes of box_rows rows x 64 dims of one head, 128-byte swizzle, zero
// fill past the last row. A head count of 1 ignores head_stride.
cudaError_t make_tmap_heads(CUtensorMap* tm, const void* base, long long rows, int heads, long long tok_stride,
                            long long head_stride, int box_rows) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return cudaErrorNotSupported;
  if (tok_stride <= 0 || (heads > 1 && head_stride <= 0)) return cudaErrorInvalidValue;
  const cuuint64_t dims[3] = {128, (cuuint64_t)(rows > 0 ? rows : 1), (cuuint64_t)(heads > 0 ? heads : 1)};
  const cuuint64_t strides[2] = {(cuuint64_t)tok_stride * 2,
                                 (cuuint64_t)(heads > 1 ? head_stride : tok_stride) * 2};
  const cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult res = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

static int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    cached[dev] = n;
  }
  return cached[dev];
}

// Persistent scoring grid: one CTA per SM (less `reserve` SMs left to concurrent work), but
// at least four stage units per CTA.
static int score_grid(const PreMeta& meta, int d, int reserve) {
  const long long nzs = ((d + kChunk - 1) / kChunk + kZSlices - 1) / kZSlices;
  const long long W = (long long)meta.total_tiles * nzs;
  long long P = sm_count() - (reserve > 0 ? reserve : 0);
  if (P > kMaxScoreCtas) P = kMaxScoreCtas;
  if (P > W / 4) P = W / 4;
  return P < 1 ? 1 : (int)P;
}

// Unit boundaries of a scoring grid of P CTAs: every CTA takes about the same time. On GB300
// a stage costs the same up to 64 text rows and then grows with the MMA's N = M rounded up to
// 16: per-CTA times of a ragged batch (M from 8 to 256, all CTAs streaming at once) give 2.4 us
// per stage at N <= 64, 2.8 us at N = 128 and 4.0 us at N = 256. A 64-column slice is weighted
// 256 + 0.8 max(N - 64, 0) + 0.3 max(N - 128, 0), so that batches with N <= 64 throughout split
// evenly.
static void score_bounds(const PreMeta& meta, int d, int P, int* bound) {
  const int nk = (d + kChunk - 1) / kChunk;
  const int nzs = (nk + kZSlices - 1) / kZSlices;
  const int W = meta.total_tiles * nzs;
  double total = 0.0;
  for (int b = 0; b < meta.B; ++b) {
    const PreReq& r = meta.r[b];
    const int tn = (r.m + 15) & ~15;
    const double slice = 256.0 + 0.8 * (tn > 64 ? tn - 64 : 0) + 0.3 * (tn > 128 ? tn - 128 : 0);
    total += slice * nk * ((r.n + kTileRows - 1) / kTileRows);
  }
  bound[0] = 0;
  bound[P] = W;
  int c = 1;
  double acc = 0.0;   // cost of the tiles before tile t
  for (int b = 0, t = 0; b < meta.B && c < P; ++b) {
    const PreReq& r = meta.r[b];
    const int tn = (r.m + 15) & ~15;
    const double slice = 256.0 + 0.8 * (tn > 64 ? tn - 64 : 0) + 0.3 * (tn > 128 ? tn - 128 : 0), tile = slice * nk;
    for (int row0 = 0; row0 < r.n && c < P; row0 += kTileRows, ++t) {
      while (c < P && total * c / P <= acc + tile) {
        // the first stage boundary of the tile at or past CTA c's share
        int j = (int)std::ceil((total * c / P - acc) / (slice * kZSlices) - 1e-9);
        j = j < 0 ? 0 : (j > nzs ? nzs : j);
        bound[c++] = t * nzs + j;
      }
      acc += tile;
    }
  }
  for (; c < P; ++c) bound[c] = W;
  // every CTA at least one unit
  for (c = 1; c < P; ++c) bound[c] = bound[c] > bound[c - 1] + 1 ? bound[c] : bound[c - 1] + 1;
  for (c = P - 1; c >= 1; --c) bound[c] = bound[c] < bound[c + 1] - 1 ? bound[c] : bound[c + 1] - 1;
}

// pdl: the preceding grid of the stream is the pre-pass, which this grid may overlap.
cudaError_t launch_pre_score(const PreMeta& meta, const PreArgs& a, int max_m, long long z_rows, cudaStream_t st,
                             bool pdl) {
  if (meta.total_tiles == 0) return cudaSuccess;
  ScoreLaunch L;
  const int tn = (max_m + 15) & ~15;                 // the MMA reads M rounded up to 16 rows
  L.t_slice_bytes = tn * 128;
  L.t_slot_slices = tn <= 64 ? 4 : (tn <= 128 ? 2 : 1);
  L.z_stages = 2;
  const int slot_bytes = L.t_slot_slices * L.t_slice_bytes;
  const int slots = (kRingBudget - L.z_stages * kZStageBytes) / slot_bytes;
  L.t_slots = slots > kMaxTSlots ? kMaxTSlots : slots;   // >= 2 for every M <= 256
  int cols = 32;
  while (cols < tn) cols <<= 1;
  L.acc_cols = cols;
  L.mld = (max_m + 3) & ~3;
  const int smem = L.z_stages * kZStageBytes + L.t_slots * slot_bytes + 1024;
  CUtensorMap tmZ3, tmZ2;
  cudaError_t e = make_tmap_sliced(&tmZ3, a.Z, z_rows, a.d, a.z_stride, kZBoxRows, kZSlices);
  if (e != cudaSuccess) return e;
  e = make_tmap(&tmZ2, a.Z, z_rows, a.d, a.z_stride, kZBoxRows);
  if (e != cudaSuccess) return e;
  bool heavy = true;   // every request has more than 112 text rows
  for (int b = 0; b < meta.B; ++b)
    if (meta.r[b].n > 0 && meta.r[b].m <= 112) heavy = false;
  auto kernel = a.action == kActFpsSeed ? (heavy ? pre_score_kernel<true, true> : pre_score_kernel<true, false>)
                                        : (heavy ? pre_score_kernel<false, true> : pre_score_kernel<false, false>);
  e = ensure_dynamic_smem(kernel, smem);
  if (e != cudaSuccess) return e;
  const int P = score_grid(meta, a.d, a.score_reserve);
  score_bounds(meta, a.d, P, L.bound);
  return launch_kernel(kernel, dim3(P), dim3(kScoreThreads), smem, st, pdl, tmZ3,
                       tmZ2, meta, a, L);
}

// Finishing grid after the scoring grid launched just before it (same meta, d' and max M;
// `scored` false: no scoring grid, selection only). The split tiles are listed here, on the
// host, from the same partition the scoring grid uses.
cudaError_t launch_pre_finish(const PreMeta& meta, const PreArgs& a, int max_m, int max_n, bool scored,
                              cudaStream_t st, bool pdl) {
  static thread_local FinMeta fm;
  static thread_local int jobs_of[kMaxChunk];
  fm.njobs = 0;
  fm.mld = (max_m + 3) & ~3;
  for (int b = 0; b < meta.B; ++b) jobs_of[b] = 0;
  if (scored && meta.total_tiles > 0) {
    const int nzs = ((a.d + kChunk - 1) / kChunk + kZSlices - 1) / kZSlices;
    const int P = score_grid(meta, a.d, a.score_reserve);
    static thread_local int bound[kMaxScoreCtas + 1];
    score_bounds(meta, a.d, P, bound);
    int b = 0;
    for (int c = 1; c < P; ++c) {
      const int bc = bound[c];
      if (bc % nzs == 0) continue;
      const int t = bc / nzs, t_start = t * nzs;
      const int c0 = score_cta_of(t_start, bound, P);
      if (c0 != c - 1) continue;                     // the tile's first boundary lists it
      while (b + 1 < meta.B && meta.r[b + 1].tile_off <= t) ++b;
      FinJob& j = fm.job[fm.njobs++];
      j.tile = t;
      j.b = b;
      j.c0 = c0;
      j.nc = score_cta_of(t_start + nzs - 1, bound, P) - c0 + 1;
      j.slot0 = bound[c0] < t_start ? 1 : 0;
      ++jobs_of[b];
    }
  }
  const bool per_request = a.action != kActScores && a.action != kActFpsSeed;
  if (per_request)
    for (int b = 0; b < meta.B; ++b)
      if (jobs_of[b] == 0 && meta.r[b].n > 0) {
        FinJob& j = fm.job[fm.njobs++];
        j.tile = -1; j.b = b; j.c0 = 0; j.nc = 0; j.slot0 = 0;
        jobs_of[b] = 1;
      }
  if (fm.njobs == 0) return cudaSuccess;
  for (int i = 0; i < fm.njobs; ++i) fm.job[i].count = per_request ? jobs_of[fm.job[i].b] : 1;
  int smem = 0;   // keys and flags of the block-wide selection, for requests above kRegSelMaxN
  const bool big = per_request && a.big_sel && max_n > kRegSelMaxN;
  if (per_request && !big && max_n > kRegSelMaxN && (size_t)max_n * 5 + 16 <= (size_t)160 * 1024)
    smem = max_n * 5 + 16;
  cudaError_t e = launch_kernel(pre_finish_kernel, dim3(fm.njobs), dim3(kFinishThreads), smem, st, pdl, meta, fm, a,
                                smem);
  if (e != cudaSuccess || !big) return e;
  static thread_local BigSel bs;
  bs.n = 0;
  for (int b = 0; b < meta.B; ++b)
    if (meta.r[b].n > kRegSelMaxN) bs.b[bs.n++] = b;
  const int sbig = (size_t)max_n * 5 + 16 <= (size_t)200 * 1024 ? max_n * 5 + 16 : 0;
  return launch_kernel(pre_select_big_kernel, dim3(bs.n), dim3(kBigSelThreads), sbig, st, true, meta, bs, a, sbig);
}

// Workspace bytes of the partial sums for up to max_m text rows.
size_t pre_score_part_bytes(int max_m) {
  return (size_t)2 * kMaxScoreCtas * (size_t)score_slot_floats((max_m + 3) & ~3) * sizeof(float);
}

// Pre-pass: the saliency rules of the B requests (when `saliency`) and 1 / ||t_j|| of the
// launch's text rows.
cudaError_t launch_pre_saliency(const PreMeta& meta, const PreArgs& a, int max_n, bool saliency, cudaStream_t st) {
  const int n_sal = saliency ? meta.B : 0;
  const long long tn_blocks = (a.total_m + 15) / 16;
  if (n_sal + tn_blocks == 0) return cudaSuccess;
  (void)max_n;   // requests above kRegSelMaxN keep their keys in the global scratch
  cudaError_t e = ensure_dynamic_smem(pre_saliency_kernel, 0);   // the scoring grid's carveout
  if (e != cudaSuccess) return e;
  if (launch_fault_injected()) return cudaErrorLaunchFailure;
  pre_saliency_kernel<<<(unsigned)(n_sal + tn_blocks), 512, 0, st>>>(meta, a, 0, n_sal);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherMeta& gm, cudaStream_t st, bool pdl) {
  int rows = 0;
  for (int i = 0; i < gm.njobs; ++i) rows = rows > gm.job[i].rows ? rows : gm.job[i].rows;
  if (rows == 0 || gm.njobs == 0) return cudaSuccess;
  return launch_kernel(gather_rows_kernel, dim3((rows + 7) / 8, gm.njobs), dim3(256), 0, st, pdl, gm);
}

}  // namespace trevs
