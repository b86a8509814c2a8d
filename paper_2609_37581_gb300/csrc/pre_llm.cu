// Stage 1 (pre-LLM, Sec. 4.1): textual-relevance scores (Eq. 4-5), selection (Sec. 3.1 ratio
// split or Eq. 6-7 fused score) and gather of the kept feature rows.
#include "pre_llm.cuh"
#include "sm100.cuh"

namespace trevs {

// ------------------------------------------------------------------ scoring contraction
//
// A persistent grid, one CTA per SM, scores the visual rows of every request against the M
// text rows of that request. Each request is cut into tiles of 128 rows (its last tile may
// be shorter) and the tiles into groups of G consecutive tiles (G = 1 or 2 per launch; a
// request's last group may hold fewer). A group stage covers S = 4 / G slices of 64 columns
// of its tiles (64 KB of Z), so a group takes nst = ceil(slices / S) stages. Work is counted
// in tile-stages: the stage of a group of g' tiles weighs g', the launch weighs W = tiles *
// nst, and CTA c owns the stages whose start falls in [W c / P, W (c + 1) / P), so every CTA
// streams the same number of Z bytes (stream-K). A group whose stages are split between
// CTAs leaves partial sums of G and ||z||^2 in the workspace (at most two segments per CTA:
// where its range starts and where it ends), and pre_finish_kernel adds them up in stage
// order.
//
// Z arrives in sub-stages of 32 KB: one tile's 128 rows over a pair of slices (256
// contiguous bytes of each row), each with its own barriers, in a ring of four to six. The
// tensor cores start on a sub-stage as soon as it lands and release it about 0.25 us later,
// so the SM keeps well over 100 KB of Z in flight (with 64 KB stages, two in a ring, the
// wait for their MMAs held the rate far below the HBM share). The slices of T for a pair
// serve the G tiles of the group: the SM takes in T once per G tiles (its intake, about
// 55 GB/s, is shared by Z from HBM and T from L2, and with M = 128 text rows T is as large
// as Z per tile).
//
// For each group the 5th-generation tensor cores compute G = Z_tile . T^T per tile (UMMA
// M = 128, N = M_b rounded up to 16) into G TMEM accumulators (two buffers of G), while eight
// warps sum the squares ||z_i||^2 from the same shared-memory sub-stages. Four epilogue warps
// read a finished group's accumulators while the next group streams into the other buffer,
// and form m_ji = max(G_ji / (||t_j|| ||z_i||), 0) and s^t_i = sqrt(sum_j m_ji^2 / M) with
// 1 / ||t_j|| from the pre-pass; the [M, N] similarity never reaches memory. Selection runs
// in the next grid.
//
// Operands, all by TMA in 128-byte swizzled rows. Z: boxes of 32 rows x two slices from a 4D
// map over 8-row groups when every request starts on an 8-row boundary, else of 8 rows from
// a 3D map; either way slice c of a sub-stage lies at c KB within each 8-row group of 2 KB,
// which the UMMA descriptor states as its stride between 8-row groups. A partial last slice
// (d' not a multiple of 64) comes slice by slice from a 2D map that fills zeros beyond d'.
// T: its own ring of slots of one or two slices; each slice is the request's M rounded up to
// 16 rows, as boxes of 256, 128, 64, 32 and 16 rows from 2D maps (zeros beyond d').
//
// Warp roles: 0 = Z producer, 1 = TMEM owner and MMA issuer, 2 = T producer, 4..7 =
// epilogue (warp w reads TMEM lanes 32*(w%4) .. +31), 8..15 = Z norms (a thread per row and
// slice of each sub-stage).

constexpr int kTileRows = kScoreTileRows;
constexpr int kChunk = 64;                     // d' columns per slice (one 128-byte swizzle row)
constexpr int kSubBytes = 32 * 1024;           // one Z sub-stage: a tile's 128 rows x two slices
constexpr int kMaxZSubs = 6;
constexpr int kMaxTSlots = 8;
constexpr int kScoreThreads = 512;
constexpr int kZNormWarps = 8;
constexpr int kRingBudget = 208 * 1024;        // the Z and T rings (dynamic shared memory)
constexpr int kZ4Rows = 32;                    // rows per Z box from the 4D map

constexpr int kTMaps = 5;   // T boxes of 16, 32, 64, 128 or 256 rows by one slice

// The tensor maps of T, one per box height; a request's slices come from the lowest box that
// holds its M rounded up to 16 rows.
struct TMaps {
  CUtensorMap m[kTMaps];
};

struct ScoreLaunch {
  int G;              // tiles per group (1 or 2)
  int S;              // 64-column slices per group stage (4 / G): G * S / 2 sub-stages of 32 KB
  int nst;            // stages per group: ceil(slices / S)
  int z_subs;         // Z ring depth in sub-stages
  int t_slots;        // T ring depth
  int t_slot_slices;  // slices per T slot (2, or 1 for tall T)
  int tn;             // T rows per slot slice: the largest M of the launch rounded up to a power of two
  int acc_cols;       // TMEM columns of one tile's accumulator (power of two >= 32 and >= tn)
  int mld;            // row length of a partial G (max M rounded up to 4)
  int z4;             // Z from the 4D map in boxes of 32 rows (every request on 8-row boundaries)
};

// Floats of one tile's partial sums: G [128][mld], then ||z||^2 [128]; a slot holds G tiles.
__host__ __device__ inline long long score_tile_floats(int mld) { return (long long)kTileRows * mld + kTileRows; }

// Scoring CTA whose weight range [W c / P, W (c + 1) / P) contains weight w.
__host__ __device__ inline int score_cta_of(long long w, long long W, int P) {
  return (int)(((w + 1) * P - 1) / W);
}

// The stages of one group that a CTA streams.
struct Segment {
  int b;          // request (slot in the launch)
  int tile0;      // the group's first tile over the launch
  int row0;       // the group's first row within its request
  int gp;         // tiles in the group (1..G)
  int h[2];       // rows of each tile of the group (0 past gp)
  int s0, s1;     // stages [s0, s1) of the group
  int slot;       // -1: the whole group; 0 / 1: partial sums of the range's first / last segment
};

// Walks the segments of weight range [w0, w1) in order (the same arithmetic on host and device).
struct SegWalk {
  long long w, w1;
  int b;
  bool first;
  __host__ __device__ SegWalk(const PreMeta& meta, int nst, long long w0, long long w1_)
      : w(w0), w1(w1_), b(0), first(true) {
    int lo = 0, hi = meta.B - 1;   // the last request whose first tile-stage is <= w0
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((long long)meta.r[mid].tile_off * nst <= w0) lo = mid; else hi = mid - 1;
    }
    b = lo;
  }
  __host__ __device__ bool next(const PreMeta& meta, const ScoreLaunch& L, Segment& sg) {
    while (w < w1) {
      while (b + 1 < meta.B && (long long)meta.r[b + 1].tile_off * L.nst <= w) ++b;
      const PreReq& r = meta.r[b];
      const int tiles = (r.n + kTileRows - 1) / kTileRows;
      const long long rstart = (long long)r.tile_off * L.nst;
      const int j = (int)((w - rstart) / ((long long)L.G * L.nst));
      const int gp = tiles - j * L.G < L.G ? tiles - j * L.G : L.G;
      const long long gstart = rstart + (long long)j * L.G * L.nst;
      const long long s0 = (w - gstart + gp - 1) / gp;
      long long s1 = (w1 - gstart + gp - 1) / gp;
      if (s1 > L.nst) s1 = L.nst;
      w = gstart + (long long)gp * L.nst;   // the next group
      if (s0 >= s1) continue;               // no stage of this group starts in the range
      sg.b = b;
      sg.tile0 = r.tile_off + j * L.G;
      sg.row0 = j * L.G * kTileRows;
      sg.gp = gp;
      for (int g = 0; g < 2; ++g) {
        const int left = r.n - sg.row0 - g * kTileRows;
        sg.h[g] = g < gp ? (left < kTileRows ? left : kTileRows) : 0;
      }
      sg.s0 = (int)s0;
      sg.s1 = (int)s1;
      sg.slot = (s0 == 0 && s1 == L.nst) ? -1 : (first ? 0 : 1);
      first = false;
      return true;
    }
    return false;
  }
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const void* tmap, int x, int y, int z, int w, uint32_t bar,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(bar), "l"(policy)
      : "memory");
}

// kSeed: the "text" rows are the pivot rows of Z (gathered beforehand) and each row's output
// is the largest cosine to them, unrectified (the distances of farthest point sampling, Sec. 3.1).
template <bool kSeed>
__global__ void __launch_bounds__(kScoreThreads, 1)
    pre_score_kernel(const __grid_constant__ CUtensorMap tmZ3, const __grid_constant__ CUtensorMap tmZ2,
                     const __grid_constant__ CUtensorMap tmZ4, const __grid_constant__ TMaps tmT,
                     const __grid_constant__ PreMeta meta, const PreArgs a, const ScoreLaunch L) {
  using namespace sm100;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t zfull[kMaxZSubs], zempty[kMaxZSubs];
  __shared__ __align__(8) uint64_t tfull[kMaxTSlots], tempty[kMaxTSlots];
  __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2], norm_full[2], norm_empty[2];
  __shared__ uint32_t tmem_base_s;
  __shared__ float rinv_s[4][256];              // one row per epilogue warp (no cross-warp barrier)
  __shared__ float zsq_s[2][2][2][kTileRows];   // [buffer][tile][slice of the pair][row]
  __shared__ volatile int s_abort;
  __shared__ volatile int s_zissued, s_tissued;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t zbase = smem_u32(smem);
  const int NZ = L.z_subs, ST = L.t_slots, TS = L.t_slot_slices, G = L.G, S = L.S;
  const int t_slice_bytes = L.tn * 128;
  const int t_slot_bytes = TS * t_slice_bytes;
  const uint32_t tbase = zbase + NZ * kSubBytes;      // after the Z sub-stages
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = a.d;
  const int nk = (d + kChunk - 1) / kChunk;           // 64-column slices
  const int full_slices = d / kChunk;                 // slices the 3D and 4D Z maps cover
  const long long W = (long long)meta.total_tiles * L.nst, P = gridDim.x;
  const long long w0 = W * blockIdx.x / P, w1 = W * (blockIdx.x + 1) / P;
  const long long tf = score_tile_floats(L.mld);

  if (tid == 0) {
    for (int s = 0; s < NZ; ++s) {
      mbar_init(smem_u32(&zfull[s]), 1);
      mbar_init(smem_u32(&zempty[s]), 1 + kZNormWarps);   // MMA commit + the Z-norm warps
    }
    for (int s = 0; s < ST; ++s) {
      mbar_init(smem_u32(&tfull[s]), 1);
      mbar_init(smem_u32(&tempty[s]), 1);                 // MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&acc_full[i]), 1);
      mbar_init(smem_u32(&acc_empty[i]), 4);              // the epilogue warps
      mbar_init(smem_u32(&norm_full[i]), kZNormWarps);
      mbar_init(smem_u32(&norm_empty[i]), 4);
    }
    s_abort = 0;
    s_zissued = 0;
    s_tissued = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), (uint32_t)(2 * G * L.acc_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  pdl_launch_dependents();   // the selection grid may start launching

  // A group's stage s covers slices [s S, s S + ns); its sub-stages, in order, are the slice
  // pairs h of the stage and, within a pair, the tiles g of the group: one tile x two slices.
  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(L.z4 ? &tmZ4 : &tmZ3);
      tma_prefetch_desc(&tmZ2);
      const uint64_t pz = l2_policy_evict_first();   // Z is streamed once
      int gz = 0;
      SegWalk walk(meta, L.nst, w0, w1);
      Segment sg;
      bool ok = true;
      while (ok && walk.next(meta, L, sg)) {
        const PreReq& r = meta.r[sg.b];
        for (int s = sg.s0; ok && s < sg.s1; ++s) {
          const int k0 = s * S, ns = min(S, nk - k0);
          for (int hp = 0; ok && 2 * hp < ns; ++hp) {
            const int kc = k0 + 2 * hp, nps = min(2, ns - 2 * hp);
            const bool ragged = kc + nps > full_slices;   // a partial slice: slice by slice from the 2D map
            for (int g = 0; g < sg.gp; ++g, ++gz) {
              const int st = gz % NZ, ph = gz / NZ;
              if (gz >= NZ && !mbar_wait(smem_u32(&zempty[st]), (ph - 1) & 1, &s_abort)) {
                s_abort = 1;
                ok = false;
                break;
              }
              const uint32_t A = zbase + st * kSubBytes;
              const uint32_t fb = smem_u32(&zfull[st]);
              const int h = sg.h[g];
              const int y0 = r.n_off + sg.row0 + g * kTileRows;
              if (ragged) {
                mbar_arrive_expect_tx(fb, (uint32_t)(((h + 7) / 8) * nps * 1024));
                for (int zb = 0; zb < (h + 7) / 8; ++zb)
                  for (int c = 0; c < nps; ++c)
                    tma_load_2d(A + zb * 2048 + c * 1024, &tmZ2, (kc + c) * kChunk, y0 + zb * 8, fb, pz);
              } else if (L.z4) {
                const int nb = (h + kZ4Rows - 1) / kZ4Rows;
                mbar_arrive_expect_tx(fb, (uint32_t)(nb * kZ4Rows * 2 * 128));
                for (int i = 0; i < nb; ++i)
                  tma_load_4d(A + i * kZ4Rows * 2 * 128, &tmZ4, 0, 0, kc, (y0 >> 3) + i * (kZ4Rows / 8), fb, pz);
              } else {
                mbar_arrive_expect_tx(fb, (uint32_t)(((h + 7) / 8) * 2048));
                for (int zb = 0; zb < (h + 7) / 8; ++zb) tma_load_3d(A + zb * 2048, &tmZ3, 0, y0 + zb * 8, kc, fb, pz);
              }
              s_zissued = gz + 1;
            }
          }
        }
      }
    }
  } else if (warp == 2) {
    if (lane == 0) {
      for (int i = 0; i < kTMaps; ++i) tma_prefetch_desc(&tmT.m[i]);
      const uint64_t pt = l2_policy_evict_last();   // T is read again by every tile of its request
      int gt = 0;
      SegWalk walk(meta, L.nst, w0, w1);
      Segment sg;
      bool ok = true;
      while (ok && walk.next(meta, L, sg)) {
        const PreReq& r = meta.r[sg.b];
        const int np16 = (r.m + 15) & ~15;           // the rows of T the request's MMAs read
        for (int s = sg.s0; ok && s < sg.s1; ++s) {
          const int k0 = s * S, ns = min(S, nk - k0);
          for (int hp = 0; ok && 2 * hp < ns; ++hp) {
            const int kc = k0 + 2 * hp, nps = min(2, ns - 2 * hp);
            const int nslots = TS == 2 ? 1 : nps;
            for (int q = 0; q < nslots; ++q, ++gt) {
              const int ts = gt % ST, ph = gt / ST;
              if (gt >= ST && !mbar_wait(smem_u32(&tempty[ts]), (ph - 1) & 1, &s_abort)) {
                s_abort = 1;
                ok = false;
                break;
              }
              const uint32_t B = tbase + ts * t_slot_bytes;
              const uint32_t fb = smem_u32(&tfull[ts]);
              const int c0 = TS == 2 ? 0 : q, c1 = TS == 2 ? nps : q + 1;
              mbar_arrive_expect_tx(fb, (uint32_t)((c1 - c0) * np16 * 128));
              for (int c = c0; c < c1; ++c) {
                // np16 rows as boxes of 256, 128, 64, 32 and 16 rows, one after the other
                for (int rr = 0, mi = kTMaps - 1; rr < np16; --mi) {
                  if ((16 << mi) > np16 - rr) continue;
                  tma_load_2d(B + (c - c0) * t_slice_bytes + rr * 128, &tmT.m[mi], (kc + c) * kChunk, r.m_off + rr, fb,
                              pt);
                  rr += 16 << mi;
                }
              }
              s_tissued = gt + 1;
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int gz = 0, gt = 0, j = 0;
      SegWalk walk(meta, L.nst, w0, w1);
      Segment sg;
      bool ok = true;
      while (ok && walk.next(meta, L, sg)) {
        const int buf = j & 1, use = j >> 1;
        if (j >= 2 && !mbar_wait(smem_u32(&acc_empty[buf]), (use - 1) & 1, &s_abort)) {
          s_abort = 1;
          break;
        }
        tc_fence_after();
        const uint32_t dg = tmem + (uint32_t)(buf * G * L.acc_cols);
        const uint32_t idesc = umma_idesc_bf16(kTileRows, (meta.r[sg.b].m + 15) & ~15);
        for (int s = sg.s0; ok && s < sg.s1; ++s) {
          const int k0 = s * S, ns = min(S, nk - k0);
          for (int hp = 0; ok && 2 * hp < ns; ++hp) {
            const int nps = min(2, ns - 2 * hp);
            const int nslots = TS == 2 ? 1 : nps;
            for (int q = 0; ok && q < nslots; ++q)
              if (!mbar_wait(smem_u32(&tfull[(gt + q) % ST]), ((gt + q) / ST) & 1, &s_abort)) ok = false;
            if (!ok) {
              s_abort = 1;
              break;
            }
            for (int g = 0; g < sg.gp; ++g, ++gz) {
              const int st = gz % NZ, ph = gz / NZ;
              if (!mbar_wait(smem_u32(&zfull[st]), ph & 1, &s_abort)) {
                s_abort = 1;
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t A = zbase + st * kSubBytes;
              const uint32_t dt = dg + (uint32_t)(g * L.acc_cols);
              for (int c = 0; c < nps; ++c) {
                const uint32_t B = TS == 2 ? tbase + (gt % ST) * t_slot_bytes + c * t_slice_bytes
                                           : tbase + ((gt + c) % ST) * t_slot_bytes;
#pragma unroll
                for (int k = 0; k < kChunk / 16; ++k)
                  umma_bf16(dt, umma_desc_sw128(A + c * 1024 + 32 * k, 2048), umma_desc_sw128(B + 32 * k), idesc,
                            (s != sg.s0 || hp != 0 || c != 0 || k != 0) ? 1u : 0u);
              }
              umma_commit(smem_u32(&zempty[st]));   // frees the Z sub-stage once these MMAs have read it
            }
            if (!ok) break;
            for (int q = 0; q < nslots; ++q) umma_commit(smem_u32(&tempty[(gt + q) % ST]));   // and the T slots
            gt += nslots;
          }
        }
        if (!ok) break;
        umma_commit(smem_u32(&acc_full[buf]));    // this group's accumulators are complete
        ++j;
      }
    }
  } else if (warp >= 8) {
    // Z norms: thread zt owns row zt % 128 and slice zt / 128 of every sub-stage's pair
    const int zt = tid - 256;
    const int row = zt & (kTileRows - 1), cs = zt >> 7;
    int gz = 0, j = 0;
    SegWalk walk(meta, L.nst, w0, w1);
    Segment sg;
    bool ok = true;
    while (ok && walk.next(meta, L, sg)) {
      const int buf = j & 1, use = j >> 1;
      float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};   // tiles 0 and 1 of the group
      for (int s = sg.s0; ok && s < sg.s1; ++s) {
        const int k0 = s * S, ns = min(S, nk - k0);
        for (int hp = 0; ok && 2 * hp < ns; ++hp) {
          const int kc = k0 + 2 * hp, nps = min(2, ns - 2 * hp);
          const int ncols = min(kChunk, d - (kc + cs) * kChunk);   // columns of this thread's slice
          for (int g = 0; g < sg.gp; ++g, ++gz) {
            const int st = gz % NZ, ph = gz / NZ;
            if (!mbar_wait(smem_u32(&zfull[st]), ph & 1, &s_abort)) {
              s_abort = 1;
              ok = false;
              break;
            }
            if (cs < nps && row < sg.h[g]) {
              const uint8_t* rowp = smem + st * kSubBytes + (row >> 3) * 2048 + cs * 1024 + (row & 7) * 128;
#pragma unroll
              for (int qq = 0; qq < 8; ++qq)
                if (qq * 8 < ncols) {   // d' is a multiple of 8: whole 16-byte pieces
                  const uint4 v = *reinterpret_cast<const uint4*>(rowp + (swz(row, qq) << 4));
                  if (g == 0) bf16_sq_acc8(v, acc0); else bf16_sq_acc8(v, acc1);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&zempty[st]));
          }
        }
      }
      if (!ok) break;
      if (j >= 2 && !mbar_wait(smem_u32(&norm_empty[buf]), (use - 1) & 1, &s_abort)) {
        s_abort = 1;
        break;
      }
      zsq_s[buf][0][cs][row] = (acc0[0] + acc0[1]) + (acc0[2] + acc0[3]);
      zsq_s[buf][1][cs][row] = (acc1[0] + acc1[1]) + (acc1[2] + acc1[3]);
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&norm_full[buf]));
      ++j;
    }
  } else if (warp >= 4) {
    const int q = warp & 3;             // TMEM lane quarter of this warp
    const int row = 32 * q + lane;      // tile row owned by this thread
    float* rt = rinv_s[q];
    pdl_wait();                         // 1 / ||t|| come from the pre-pass
    int j = 0;
    SegWalk walk(meta, L.nst, w0, w1);
    Segment sg;
    while (walk.next(meta, L, sg)) {
      const PreReq& r = meta.r[sg.b];
      const int m = r.m;
      const int buf = j & 1, use = j >> 1;
      __syncwarp();
      for (int c = lane; c < m; c += 32) rt[c] = __ldcg(a.t_rinv + r.m_off + c);
      __syncwarp();
      bool ok = mbar_wait(smem_u32(&acc_full[buf]), use & 1, &s_abort);
      ok = ok && mbar_wait(smem_u32(&norm_full[buf]), use & 1, &s_abort);
      ok = __all_sync(0xffffffffu, ok && !s_abort);
      if (!ok) {
        s_abort = 1;
        break;
      }
      tc_fence_after();
      float out0 = 0.f, out1 = 0.f;
      for (int g = 0; g < sg.gp; ++g) {
        const uint32_t lane_base =
            tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * G * L.acc_cols) + (uint32_t)(g * L.acc_cols);
        const float zsq = zsq_s[buf][g][0][row] + zsq_s[buf][g][1][row];
        const float rz = zsq > 0.f ? 1.0f / sqrtf(zsq) : 0.f;
        float sum = 0.f, mx = -INFINITY;
        if (sg.slot < 0) {
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
          const float o = kSeed ? mx : sqrtf(sum / (float)m);
          if (g == 0) out0 = o; else out1 = o;
        } else {
          // a group split between CTAs: leave this CTA's partial sums (G row, columns
          // 0 .. round_up(m, 4), and ||z||^2) of tile g in its slot for pre_finish_kernel
          float* own = a.part + ((2 * (long long)blockIdx.x + sg.slot) * G + g) * tf;
          float* gr = own + (long long)row * L.mld;
          for (int c0 = 0; c0 < m; c0 += 32) {
            float v[32];
            tmem_ld_32x32b_x32(lane_base + (uint32_t)c0, v);
#pragma unroll
            for (int jj = 0; jj < 32; jj += 4)
              if (c0 + jj < m) *reinterpret_cast<float4*>(gr + c0 + jj) = make_float4(v[jj], v[jj + 1], v[jj + 2], v[jj + 3]);
          }
          own[(long long)kTileRows * L.mld + row] = zsq;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_u32(&acc_empty[buf]));
        mbar_arrive(smem_u32(&norm_empty[buf]));
      }
      if (sg.slot < 0) {
        float* out = a.s_t + r.n_off + sg.row0 + row;
        if (row < sg.h[0]) out[0] = out0;
        if (sg.gp > 1 && row < sg.h[1]) out[kTileRows] = out1;
      }
      ++j;
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)(2 * G * L.acc_cols));
  }
  if (s_abort) {
    // let the copies already issued land before the block's shared memory is released
    if (tid == 0) {
      const volatile int no_abort = 0;
      const int zi = s_zissued, ti = s_tissued;
      for (int x = zi - NZ > 0 ? zi - NZ : 0; x < zi; ++x)
        mbar_wait(smem_u32(&zfull[x % NZ]), (x / NZ) & 1, &no_abort, 500000000ull);
      for (int x = ti - ST > 0 ? ti - ST : 0; x < ti; ++x)
        mbar_wait(smem_u32(&tfull[x % ST]), (x / ST) & 1, &no_abort, 500000000ull);
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
  int tile, b, c0, nc, slot0, count, gidx;   // gidx: the tile's place in its group's slot
};
struct FinMeta {
  int njobs, mld, G;
  FinJob job[2 * kMaxScoreCtas + kMaxChunk];
};

template <bool kSeed>
__device__ inline void fixup_tile(const FinJob& jb, const PreReq& r, int mld, int G, const PreArgs& a) {
  // Warp w owns rows 8w .. 8w + 7 of the tile. A row's partial sums are mld contiguous floats:
  // P lanes (a power of two, 4..32) read it as consecutive 16-byte groups, so each load
  // instruction covers whole rows; lane gl of a segment owns groups gl, gl + P.
  const int row0 = (jb.tile - r.tile_off) * kTileRows;
  const int h = min(kTileRows, r.n - row0);
  const int m = r.m;
  const long long tf = score_tile_floats(mld);
  const int gpr = mld >> 2;
  int P = 4;
  while (P < gpr && P < 32) P <<= 1;
  const int RPW = 32 / P;                             // rows per warp pass (<= 8)
  const int ng = (gpr + P - 1) / P;                   // groups per lane (<= 2 for M <= 256)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int sub = lane / P, gl = lane % P;
  const float* p0 = a.part + ((2 * (long long)jb.c0 + jb.slot0) * G + jb.gidx) * tf;
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
        const float* base = x0 + x == 0 ? p0 : a.part + (2 * (long long)(jb.c0 + x0 + x) * G + jb.gidx) * tf;
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
      if (gl == 0 && row < h) a.s_t[r.n_off + row0 + row] = mx;
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
    if (jb.tile >= 0) fixup_tile<true>(jb, r, fm.mld, fm.G, a);
    return;
  }
  if (jb.tile >= 0) fixup_tile<false>(jb, r, fm.mld, fm.G, a);
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
  select_request_512(a, r, jb.b, smem, smem_bytes, sh);
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

// Plan of a scoring launch: grid size, group width G, stage and ring shapes. Every launch of
// the scoring grid and of the finishing grid that follows it derives the same plan.
struct ScorePlan {
  ScoreLaunch L;
  int P;
  int smem;
};

static ScorePlan score_plan(const PreMeta& meta, const PreArgs& a, int max_m) {
  ScorePlan p;
  ScoreLaunch& L = p.L;
  const int nk = (a.d + kChunk - 1) / kChunk;
  // T rows per slot slice: the tallest box a request of the launch takes (its M rounded up to
  // a power of two, at least 16), which the MMA's N (M rounded up to 16) never exceeds
  L.tn = 16;
  while (L.tn < max_m) L.tn <<= 1;
  L.acc_cols = L.tn < 32 ? 32 : L.tn;
  L.mld = (max_m + 3) & ~3;
  bool rows8 = true;                          // every request's rows start on an 8-row boundary
  for (int b = 0; b < meta.B; ++b) rows8 = rows8 && (meta.r[b].n % 8 == 0);
  // grid: one CTA per SM (less the SMs left to concurrent work), at least four G = 1 stages each
  const long long W1 = (long long)meta.total_tiles * ((nk + 3) / 4);
  long long P = sm_count() - (a.score_reserve > 0 ? a.score_reserve : 0);
  if (P > kMaxScoreCtas) P = kMaxScoreCtas;
  if (P > W1 / 4) P = W1 / 4;
  p.P = P < 1 ? 1 : (int)P;
  // Two tiles per stage halve the T bytes an SM takes in per Z byte. They need the two
  // tiles' accumulators double-buffered in TMEM (4 x acc_cols <= 512), rows on 8-row
  // boundaries (4D boxes of 32 rows: narrower rows stream well only in larger boxes), and
  // about two tiles per CTA, so that groups are rarely split between CTAs.
  L.G = (4 * L.acc_cols <= 512 && rows8 && meta.total_tiles >= (7 * p.P) / 4) ? 2 : 1;
  L.S = 4 / L.G;
  L.nst = (nk + L.S - 1) / L.S;
  L.z4 = rows8 ? 1 : 0;
  // rings: the deepest Z ring (in 32 KB sub-stages) beside a T ring of at least two slots
  // and three slices (T comes from L2 and runs ahead by a pair or more), with T slots of two
  // slices when that costs no Z depth, else of one
  const int slice = L.tn * 128;
  L.z_subs = 0;
  for (int ts = 2; ts >= 1; --ts)
    for (int nz = kMaxZSubs; nz >= 2; --nz) {
      const int slots = (kRingBudget - nz * kSubBytes) / (ts * slice);
      if (slots >= 2 && slots * ts >= 3) {
        if (nz > L.z_subs) {
          L.z_subs = nz;
          L.t_slot_slices = ts;
          L.t_slots = slots > kMaxTSlots ? kMaxTSlots : slots;
        }
        break;
      }
    }
  p.smem = L.z_subs * kSubBytes + L.t_slots * L.t_slot_slices * slice + 1024;
  return p;
}

// The same matrix seen as [row groups of 8][slices][8 rows][64] (whole slices and whole row
// groups only): a box of `groups` row groups x `slices` slices lands as `groups` runs of
// `slices` swizzle atoms.
static cudaError_t make_tmap_rowgroups(CUtensorMap* tm, const void* base, long long rows, int cols, long long stride,
                                       int slices, int groups) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return cudaErrorNotSupported;
  const int full = cols / kChunk;
  const long long ng = rows / 8;
  const cuuint64_t dims[4] = {(cuuint64_t)kChunk, 8, (cuuint64_t)(full > 0 ? full : 1), (cuuint64_t)(ng > 0 ? ng : 1)};
  const cuuint64_t strides[3] = {(cuuint64_t)stride * 2, (cuuint64_t)kChunk * 2, (cuuint64_t)stride * 16};
  const cuuint32_t box[4] = {(cuuint32_t)kChunk, 8, (cuuint32_t)slices, (cuuint32_t)groups};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult res = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// pdl: the preceding grid of the stream is the pre-pass, which this grid may overlap.
cudaError_t launch_pre_score(const PreMeta& meta, const PreArgs& a, int max_m, long long z_rows, cudaStream_t st,
                             bool pdl) {
  if (meta.total_tiles == 0) return cudaSuccess;
  const ScorePlan p = score_plan(meta, a, max_m);
  const ScoreLaunch& L = p.L;
  CUtensorMap tmZ3, tmZ2, tmZ4;
  TMaps tmT;
  cudaError_t e = make_tmap_sliced(&tmZ3, a.Z, z_rows, a.d, a.z_stride, 8, 2);
  if (e == cudaSuccess) e = make_tmap(&tmZ2, a.Z, z_rows, a.d, a.z_stride, 8);
  if (e == cudaSuccess && L.z4) e = make_tmap_rowgroups(&tmZ4, a.Z, z_rows, a.d, a.z_stride, 2, kZ4Rows / 8);
  if (e == cudaSuccess && !L.z4) tmZ4 = tmZ3;   // not read
  for (int i = 0; i < kTMaps && e == cudaSuccess; ++i) e = make_tmap(&tmT.m[i], a.T, a.total_m, a.d, a.t_stride, 16 << i);
  if (e != cudaSuccess) return e;
  auto kernel = a.action == kActFpsSeed ? pre_score_kernel<true> : pre_score_kernel<false>;
  e = ensure_dynamic_smem(kernel, p.smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(kernel, dim3(p.P), dim3(kScoreThreads), p.smem, st, pdl, tmZ3, tmZ2, tmZ4, tmT, meta, a, L);
}

// Finishing grid after the scoring grid launched just before it (same meta, d' and max M;
// `scored` false: no scoring grid, selection only). The split tiles are listed here, on the
// host, from the same partition the scoring grid walks.
cudaError_t launch_pre_finish(const PreMeta& meta, const PreArgs& a, int max_m, int max_n, bool scored,
                              cudaStream_t st, bool pdl) {
  static thread_local FinMeta fm;
  static thread_local int jobs_of[kMaxChunk];
  fm.njobs = 0;
  fm.mld = (max_m + 3) & ~3;
  fm.G = 1;
  for (int b = 0; b < meta.B; ++b) jobs_of[b] = 0;
  if (scored && meta.total_tiles > 0) {
    const ScorePlan p = score_plan(meta, a, max_m);
    const ScoreLaunch& L = p.L;
    fm.G = L.G;
    const long long W = (long long)meta.total_tiles * L.nst;
    // the partial segments of every CTA, in CTA order: a group split between CTAs shows up
    // as the last partial segment of its first contributor and the first of the others
    int open_tile = -1, open_gp = 0, open_b = 0, open_c0 = 0, open_slot0 = 0, open_nc = 0;
    auto flush = [&]() {
      if (open_tile >= 0 && open_nc >= 2)
        for (int g = 0; g < open_gp; ++g) {
          FinJob& j = fm.job[fm.njobs++];
          j.tile = open_tile + g; j.b = open_b; j.c0 = open_c0; j.nc = open_nc; j.slot0 = open_slot0; j.gidx = g;
          ++jobs_of[open_b];
        }
      open_tile = -1;
    };
    for (int c = 0; c < p.P; ++c) {
      SegWalk walk(meta, L.nst, W * c / p.P, W * (c + 1) / p.P);
      Segment sg;
      while (walk.next(meta, L, sg)) {
        if (sg.slot < 0) continue;
        if (sg.tile0 == open_tile) {
          ++open_nc;
        } else {
          flush();
          open_tile = sg.tile0; open_gp = sg.gp; open_b = sg.b; open_c0 = c; open_slot0 = sg.slot; open_nc = 1;
        }
      }
    }
    flush();
  }
  const bool per_request = a.action != kActScores && a.action != kActFpsSeed;
  if (per_request)
    for (int b = 0; b < meta.B; ++b)
      if (jobs_of[b] == 0 && meta.r[b].n > 0) {
        FinJob& j = fm.job[fm.njobs++];
        j.tile = -1; j.b = b; j.c0 = 0; j.nc = 0; j.slot0 = 0; j.gidx = 0;
        jobs_of[b] = 1;
      }
  if (fm.njobs == 0) return cudaSuccess;
  for (int i = 0; i < fm.njobs; ++i) fm.job[i].count = per_request ? jobs_of[fm.job[i].b] : 1;
  int smem = 0;   // keys and flags of the block-wide selection, for requests above kRegSelMaxN
  if (per_request && max_n > kRegSelMaxN && (size_t)max_n * 5 + 16 <= (size_t)160 * 1024) smem = max_n * 5 + 16;
  return launch_kernel(pre_finish_kernel, dim3(fm.njobs), dim3(kFinishThreads), smem, st, pdl, meta, fm, a, smem);
}

// Workspace bytes of the partial sums for up to max_m text rows: two slots per scoring CTA,
// each of up to two tiles.
size_t pre_score_part_bytes(int max_m) {
  return (size_t)2 * kMaxScoreCtas * 2 * (size_t)score_tile_floats((max_m + 3) & ~3) * sizeof(float);
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
