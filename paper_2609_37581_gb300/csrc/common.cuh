// Device helpers shared by the TReVS kernels: order-preserving score keys, a
// block-wide radix select with index tie-break, ordered compaction, and thin
// wrappers over the sm_103a instructions the kernels use (cp.async, ldmatrix,
// mma.sync for the small stage-2 contractions).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace trevs {

constexpr int kMaxChunk = 256;   // requests per launch (metadata travels as kernel parameters)

// ------------------------------------------------------------------ metadata

struct PreReq {
  int n_off, n;     // visual rows [n_off, n_off + n) of Z, s_v, s_t
  int m_off, m;     // text rows of T
  int k1_off, k1;   // kept rows of kept_idx / Z_out
  int kt;           // textual share K_t of the keep budget (Sec. 3.1)
  int tile_off;     // first 128-row scoring tile of this request
};

struct PreMeta {
  int B;
  int total_tiles;  // 128-row scoring tiles over all requests (the last of a request may be short)
  PreReq r[kMaxChunk];
};

struct InReq {
  long long attn_off;  // first attention probability of this request ([Hq][l][k1] fp32)
  int l_off, l;        // text rows of Q and of the row variances
  int k1_off, k1;      // visual rows of K, V, hidden, p
  int k2_off, k2;      // kept rows of kept_local and of the compacted outputs
  int hs_off;          // first head-statistics block
  int ts_off;          // first token-score block
};

struct InMeta {
  int B;
  int total_hs;
  int total_ts;
  InReq r[kMaxChunk];
};

// Finds the request whose block range [off(b), off(b+1)) holds `x` (offsets ascending).
template <class F>
__device__ __forceinline__ int find_request(int B, int x, F off) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (off(mid) <= x) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ------------------------------------------------------------------ score keys

// Maps a float to a uint32 whose unsigned order is the float order; -0 maps like +0.
__device__ __forceinline__ uint32_t score_key(float f) {
  uint32_t b = __float_as_uint(f);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float key_to_score(uint32_t k) {
  uint32_t b = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  return __uint_as_float(b);
}

// ------------------------------------------------------------------ block selection

struct SelShared {
  uint32_t hist[2048];
  uint32_t cand[64];
  uint32_t warp_gt[32];
  uint32_t warp_eq[32];
  uint32_t bcast[4];
};

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm volatile("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// One radix pass of the block selection: histogram of digit ((w >> sh) & (nb - 1)) over the
// entries whose offset w = key - lo satisfies (w & pmask) == pval, then the digit holding
// the kk-th largest of them. Writes (digit, rank within the digit) to s.bcast[0..1].
// keys must be 16-byte aligned.
__device__ inline void radix_pass(const uint32_t* keys, int n, uint32_t lo, uint32_t pmask, uint32_t pval,
                                  int sh, uint32_t nb, int kk, SelShared& s) {
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < (int)nb; i += nthr) s.hist[i] = 0u;
  __syncthreads();
  auto count = [&](uint32_t v) {
    const uint32_t w = v - lo;
    if (v != 0u && (w & pmask) == pval) atomicAdd(&s.hist[(w >> sh) & (nb - 1u)], 1u);
  };
  const int n4 = n >> 2;
  const uint4* k4 = reinterpret_cast<const uint4*>(keys);
  for (int j = tid; j < n4; j += nthr) {
    const uint4 v = k4[j];
    count(v.x);
    count(v.y);
    count(v.z);
    count(v.w);
  }
  for (int i = 4 * n4 + tid; i < n; i += nthr) count(keys[i]);
  __syncthreads();
  // bin scan from the top: thread t < nscan owns bins [nb - (t+1)*per, nb - t*per)
  int nscan = 1;   // a power of two <= min(threads, bins, 256)
  while (nscan * 2 <= nthr && nscan * 2 <= (int)nb && nscan < 256) nscan *= 2;
  const int per = (int)nb / nscan;
  uint32_t tot = 0;
  if (tid < nscan)
    for (int j = 0; j < per; ++j) tot += s.hist[nb - 1 - (uint32_t)(tid * per + j)];
  uint32_t incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (tid < nscan && lane == 31) s.warp_gt[warp] = incl;
  __syncthreads();
  if (tid < nscan) {
    uint32_t off = 0;
    for (int w = 0; w < warp; ++w) off += s.warp_gt[w];
    incl += off;
    const uint32_t excl = incl - tot;
    if (excl < (uint32_t)kk && incl >= (uint32_t)kk) {
      uint32_t cum = excl;
      int j = 0;
      for (; j < per - 1; ++j) {
        const uint32_t c = s.hist[nb - 1 - (uint32_t)(tid * per + j)];
        if (cum + c >= (uint32_t)kk) break;
        cum += c;
      }
      s.bcast[0] = nb - 1 - (uint32_t)(tid * per + j);
      s.bcast[1] = (uint32_t)kk - cum;
    }
  }
  __syncthreads();
}

// K-th largest key (1 <= k <= number of non-zero keys) of keys[0..n); a key of 0 marks an
// excluded entry (no float maps to it). Returns the key value tau, `need`, the
// number of entries equal to tau that belong to the top k when ties go to the lower index,
// and `n_eq`, the number of entries equal to tau (need == n_eq: the top k are exactly the
// entries >= tau). [lo, hi] is the key range from block_fill_keys; keys 16-byte aligned.
// Radix select on the offsets w = key - min(keys): the first digit is the
// top 11 bits of the occupied range, so scores clustered in a narrow band still spread
// over the bins; when the chosen bin holds at most 64 entries one warp finishes by ranking
// them, otherwise further 11-bit passes count only the entries still in the running.
// All threads of the block (a multiple of 32) must call it; keys may live in shared or
// global memory.
__device__ inline void block_kth_largest(const uint32_t* keys, int n, int k, SelShared& s, uint32_t lo,
                                         uint32_t hi, uint32_t& tau, int& need, int& n_eq) {
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  if (lo >= hi) {   // every candidate key equal (or none): the first k of them
    tau = lo == hi ? lo : 0xFFFFFFFFu;
    need = k;
    n_eq = n;
    return;
  }
  const uint32_t range = hi - lo;
  const int bits = 32 - __clz(range);            // bits of the largest offset
  int sh = bits > 11 ? bits - 11 : 0;            // first digit: offset bits [sh, bits)
  uint32_t nb = 1u << (bits - sh);
  uint32_t pmask = 0u, pval = 0u;
  int kk = k;
  while (true) {
    radix_pass(keys, n, lo, pmask, pval, sh, nb, kk, s);
    const uint32_t dig = s.bcast[0];
    const uint32_t cnt = s.hist[dig];            // entries still in the running
    kk = (int)s.bcast[1];
    pval |= dig << sh;
    pmask |= (nb - 1u) << sh;
    __syncthreads();
    if (sh == 0) {                               // every remaining entry equals tau
      tau = lo + pval;
      need = kk;
      n_eq = (int)cnt;
      return;
    }
    if (cnt <= 64u) {
      // gather the candidates; one warp ranks them pairwise
      if (tid == 0) s.bcast[2] = 0u;
      __syncthreads();
      auto gather = [&](uint32_t v, bool valid) {
        const bool in = valid && v != 0u && ((v - lo) & pmask) == pval;
        const uint32_t bal = __ballot_sync(0xffffffffu, in);
        if (bal) {
          uint32_t at = 0;
          if (lane == 0) at = atomicAdd(&s.bcast[2], (uint32_t)__popc(bal));
          at = __shfl_sync(0xffffffffu, at, 0);
          if (in) s.cand[at + __popc(bal & lanemask_lt())] = v;
        }
      };
      const int n4 = n >> 2;
      const uint4* k4 = reinterpret_cast<const uint4*>(keys);
      for (int base = 0; base < n4; base += nthr) {
        const int j = base + tid;
        const uint4 v = j < n4 ? k4[j] : make_uint4(0u, 0u, 0u, 0u);
        gather(v.x, j < n4);
        gather(v.y, j < n4);
        gather(v.z, j < n4);
        gather(v.w, j < n4);
      }
      {
        const int i = 4 * n4 + tid;
        gather(i < n ? keys[i] : 0u, i < n);
      }
      __syncthreads();
      if (warp == 0) {
        for (int c = lane; c < (int)cnt; c += 32) {
          const uint32_t mine = s.cand[c];
          int gt = 0, eq = 0;
          for (int j = 0; j < (int)cnt; ++j) {
            const uint32_t o = s.cand[j];
            gt += o > mine;
            eq += o == mine;
          }
          if (gt < kk && kk <= gt + eq) {        // equal candidates write equal values
            s.bcast[0] = mine;
            s.bcast[1] = (uint32_t)(kk - gt);
            s.bcast[3] = (uint32_t)eq;
          }
        }
      }
      __syncthreads();
      tau = s.bcast[0];
      need = (int)s.bcast[1];
      n_eq = (int)s.bcast[3];
      __syncthreads();
      return;
    }
    const int nbits = sh > 11 ? 11 : sh;
    sh -= nbits;
    nb = 1u << nbits;
  }
}

// flags[i] = 1 (other flags untouched) for the k largest non-zero keys of keys[0..n) (ties to
// the lower index), for n <= blockDim.x: thread i ranks key i against every key
// (shared-memory broadcast reads).
__device__ inline void block_mark_topk_small(const uint32_t* keys, int n, int k, uint8_t* flags) {
  const int i = threadIdx.x;
  if (i < n) {
    const uint32_t mine = keys[i];
    int rank = 0;
#pragma unroll 4
    for (int j = 0; j < n; ++j) {
      const uint32_t o = keys[j];
      rank += (o > mine) || (o == mine && j < i);
    }
    if (mine != 0u && rank < k) flags[i] = 1;
  }
  __syncthreads();
}

// flags[i] |= 1 for the entries of the top k described by (tau, need, n_eq). When every
// entry equal to tau belongs (need == n_eq) this is element-wise; otherwise the ties go to
// the lower indices by an ordered pass.
__device__ inline void block_mark_selected(const uint32_t* keys, int n, uint32_t tau, int need, int n_eq,
                                           uint8_t* flags, SelShared& s);

// Visits, in ascending index order, every i selected by (tau, need):
// keys[i] > tau, or keys[i] == tau among the first `need` such indices.
// emit(i, pos, selected) is called for EVERY i < n (pos = output slot when selected).
template <class Emit>
__device__ inline void block_emit_selected(const uint32_t* keys, int n, uint32_t tau, int need,
                                           SelShared& s, Emit emit) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  int seg = (n + nwarps - 1) / nwarps;
  seg = (seg + 31) & ~31;
  const int beg = min(n, warp * seg), end = min(n, beg + seg);
  uint32_t cgt = 0, ceq = 0;
  for (int base = beg; base < end; base += 32) {
    int i = base + lane;
    uint32_t v = (i < end) ? keys[i] : 0u;
    cgt += __popc(__ballot_sync(0xffffffffu, i < end && v > tau));
    ceq += __popc(__ballot_sync(0xffffffffu, i < end && v == tau));
  }
  if (lane == 0) { s.warp_gt[warp] = cgt; s.warp_eq[warp] = ceq; }
  __syncthreads();
  uint32_t run_gt = 0, run_eq = 0;
  for (int w = 0; w < warp; ++w) { run_gt += s.warp_gt[w]; run_eq += s.warp_eq[w]; }
  const uint32_t lt = lanemask_lt();
  for (int base = beg; base < end; base += 32) {
    int i = base + lane;
    uint32_t v = (i < end) ? keys[i] : 0u;
    uint32_t bgt = __ballot_sync(0xffffffffu, i < end && v > tau);
    uint32_t beq = __ballot_sync(0xffffffffu, i < end && v == tau);
    uint32_t gt_before = run_gt + __popc(bgt & lt);
    uint32_t eq_before = run_eq + __popc(beq & lt);
    if (i < end) {
      bool sel = (v > tau) || (v == tau && eq_before < (uint32_t)need);
      uint32_t pos = gt_before + min(eq_before, (uint32_t)need);
      emit(i, (int)pos, sel);
    }
    run_gt += __popc(bgt);
    run_eq += __popc(beq);
  }
  __syncthreads();
}

// Ordered compaction of a 0/1 byte mask: out[pos] = i for every flagged i, ascending.
// Each warp owns a contiguous segment and walks it 128 entries at a time.
__device__ inline void block_compact_flags(const uint8_t* flags, int n, int* out, SelShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  int seg = (n + nwarps - 1) / nwarps;
  seg = (seg + 127) & ~127;
  const int beg = min(n, warp * seg), end = min(n, beg + seg);
  uint32_t cnt = 0;
  for (int base = beg; base < end; base += 128) {
    bool f[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = base + 32 * q + lane;
      f[q] = i < end && flags[i] != 0;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) cnt += __popc(__ballot_sync(0xffffffffu, f[q]));
  }
  if (lane == 0) s.warp_gt[warp] = cnt;
  __syncthreads();
  uint32_t run = 0;
  for (int w = 0; w < warp; ++w) run += s.warp_gt[w];
  const uint32_t lt = lanemask_lt();
  for (int base = beg; base < end; base += 128) {
    bool f[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = base + 32 * q + lane;
      f[q] = i < end && flags[i] != 0;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t b = __ballot_sync(0xffffffffu, f[q]);
      if (f[q]) out[run + __popc(b & lt)] = base + 32 * q + lane;
      run += __popc(b);
    }
  }
  __syncthreads();
}

__device__ inline void block_mark_selected(const uint32_t* keys, int n, uint32_t tau, int need, int n_eq,
                                           uint8_t* flags, SelShared& s) {
  if (need >= n_eq) {
    const int n4 = n >> 2;
    const uint4* k4 = reinterpret_cast<const uint4*>(keys);
    for (int j = threadIdx.x; j < n4; j += blockDim.x) {
      const uint4 v = k4[j];
      if (v.x >= tau) flags[4 * j] = 1;
      if (v.y >= tau) flags[4 * j + 1] = 1;
      if (v.z >= tau) flags[4 * j + 2] = 1;
      if (v.w >= tau) flags[4 * j + 3] = 1;
    }
    for (int i = 4 * n4 + threadIdx.x; i < n; i += blockDim.x)
      if (keys[i] >= tau) flags[i] = 1;
    __syncthreads();
    return;
  }
  block_emit_selected(keys, n, tau, need, s, [&](int i, int, bool sel) { if (sel) flags[i] = 1; });
}

// ------------------------------------------------------------------ register-resident selection
//
// Selection over up to E * blockDim.x entries held in registers, E per thread: thread t
// holds entries i = e * blockDim.x + t (coalesced loads). Key 0 marks an excluded entry (no
// float maps to it). The top k (ties to the lower index) are described by (tau, need):
// entry i is selected iff key > tau, or key == tau and fewer than `need` entries equal to
// tau precede it. Radix select on the offsets w = key - min(keys) with 8-bit digits, the
// first digit taking the top bits of the occupied range; it stops as soon as every
// candidate of the chosen digit belongs to the top k. Each pass costs three block
// barriers. Requires blockDim.x >= 256, a multiple of 32, and E * blockDim.x / 32 <= 512.

struct RegSelShared {
  uint32_t hist[2][256];
  uint32_t cell[512];     // per (element slot, warp) counts, then their prefix sums
  uint32_t wred[3][32];
  uint32_t res[4];
};

// Block-wide min of the non-zero keys, max of all keys and count of the non-zero keys;
// also clears hist[0] for the first radix pass.
template <int E>
__device__ inline void block_reg_stats(const uint32_t (&key)[E], RegSelShared& s, uint32_t& lo, uint32_t& hi,
                                       uint32_t& cnt) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  uint32_t l = 0xFFFFFFFFu, h = 0u, c = 0u;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (key[e] != 0u) { l = min(l, key[e]); ++c; }
    h = max(h, key[e]);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    l = min(l, __shfl_xor_sync(0xffffffffu, l, o));
    h = max(h, __shfl_xor_sync(0xffffffffu, h, o));
    c += __shfl_xor_sync(0xffffffffu, c, o);
  }
  if (lane == 0) { s.wred[0][warp] = l; s.wred[1][warp] = h; s.wred[2][warp] = c; }
  for (int i = threadIdx.x; i < 256; i += blockDim.x) s.hist[0][i] = 0u;
  __syncthreads();
  l = 0xFFFFFFFFu; h = 0u; c = 0u;
  for (int w = 0; w < nwarps; ++w) { l = min(l, s.wred[0][w]); h = max(h, s.wred[1][w]); c += s.wred[2][w]; }
  __syncthreads();   // wred is rewritten by the caller's next step
  lo = l; hi = h; cnt = c;
}

// (tau, need) of the k largest non-zero keys; `lo`, `hi`, `cnt` as from block_reg_stats.
template <int E>
__device__ inline void block_reg_topk_ranged(const uint32_t (&key)[E], int k, uint32_t lo, uint32_t hi,
                                             uint32_t cnt, RegSelShared& s, uint32_t& tau, int& need) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (k <= 0) { tau = 0xFFFFFFFFu; need = 0; return; }            // nothing
  if ((uint32_t)k >= cnt) { tau = 0u; need = 0; return; }         // every non-zero key
  if (lo == hi) { tau = lo; need = k; return; }                   // all equal: the first k
  const int bits = 32 - __clz(hi - lo);
  int sh = bits > 8 ? bits - 8 : 0;
  uint32_t nb = 1u << (bits - sh);
  uint32_t pm = 0u, pv = 0u, kk = (uint32_t)k;
  int buf = 0;
  while (true) {
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const uint32_t w = key[e] - lo;
      if (key[e] != 0u && (w & pm) == pv) atomicAdd(&s.hist[buf][(w >> sh) & (nb - 1u)], 1u);
    }
    for (int i = tid; i < 256; i += blockDim.x) s.hist[buf ^ 1][i] = 0u;
    __syncthreads();
    // thread t < nb owns digit nb - 1 - t: counts from the top digit down
    uint32_t c = 0u, incl = 0u;
    if (tid < 256) {
      c = tid < (int)nb ? s.hist[buf][nb - 1u - (uint32_t)tid] : 0u;
      incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (lane == 31) s.wred[0][warp] = incl;
    }
    __syncthreads();
    if (tid < 256 && c != 0u) {
      uint32_t off = 0u;
      for (int w = 0; w < warp; ++w) off += s.wred[0][w];
      const uint32_t ex = incl - c + off;
      if (ex < kk && kk <= ex + c) {
        s.res[0] = nb - 1u - (uint32_t)tid;
        s.res[1] = kk - ex;
        s.res[2] = c;
      }
    }
    __syncthreads();
    const uint32_t dg = s.res[0], kn = s.res[1], cn = s.res[2];
    pv |= dg << sh;
    pm |= (nb - 1u) << sh;
    buf ^= 1;
    if (kn == cn) { tau = lo + pv - 1u; need = 0; return; }      // the whole digit is in: key >= lo + pv
    if (sh == 0) { tau = lo + pv; need = (int)kn; return; }       // ties at one key value
    kk = kn;
    const int nbits = sh > 8 ? 8 : sh;
    sh -= nbits;
    nb = 1u << nbits;
  }
}

template <int E>
__device__ inline void block_reg_topk(const uint32_t (&key)[E], int k, RegSelShared& s, uint32_t& tau, int& need) {
  uint32_t lo, hi, cnt;
  block_reg_stats(key, s, lo, hi, cnt);
  block_reg_topk_ranged(key, k, lo, hi, cnt, s, tau, need);
}

// The k-th largest key (1 <= k <= number of non-zero keys).
template <int E>
__device__ inline uint32_t block_reg_kth(const uint32_t (&key)[E], int k, RegSelShared& s) {
  uint32_t tau;
  int need;
  block_reg_topk(key, k, s, tau, need);
  if (need > 0) return tau;
  // the top k are exactly the keys > tau: the k-th largest is their minimum
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  uint32_t m = 0xFFFFFFFFu;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if (key[e] > tau) m = min(m, key[e]);
#pragma unroll
  for (int o = 16; o; o >>= 1) m = min(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) s.wred[0][warp] = m;
  __syncthreads();
  m = 0xFFFFFFFFu;
  for (int w = 0; w < nwarps; ++w) m = min(m, s.wred[0][w]);
  __syncthreads();
  return m;
}

// Exclusive block-wide prefix sum of one value per thread (thread order).
__device__ inline uint32_t block_excl_scan(uint32_t v, RegSelShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) s.wred[1][warp] = incl;
  __syncthreads();
  uint32_t off = 0u;
  for (int w = 0; w < warp; ++w) off += s.wred[1][w];
  __syncthreads();
  return incl - v + off;
}

// s.cell[e * nwarps + warp] = the number of entries before the 32-entry group (e, warp), in
// index order, of each of the two per-group counts packed as lo16 | hi16 << 16.
template <int E>
__device__ inline void block_cell_offsets(const uint32_t (&packed)[E], RegSelShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  if (lane == 0) {
#pragma unroll
    for (int e = 0; e < E; ++e) s.cell[e * nwarps + warp] = packed[e];
  }
  __syncthreads();
  const int ncell = E * nwarps;
  const uint32_t v = (int)threadIdx.x < ncell ? s.cell[threadIdx.x] : 0u;
  const uint32_t ex = block_excl_scan(v, s);
  if ((int)threadIdx.x < ncell) s.cell[threadIdx.x] = ex;
  __syncthreads();
}

// Ordered output of a register-resident selection: out[pos] = i for every selected i,
// ascending, where i = e * blockDim.x + t is selected iff bit e of `force` is set or
// (tau, need) selects key[e]. Forced entries must carry key 0. Needs E * blockDim.x < 65536.
template <int E>
__device__ inline void block_reg_emit(const uint32_t (&key)[E], uint32_t force, uint32_t tau, int need, int* out,
                                      RegSelShared& s) {
  const int warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const uint32_t lt = lanemask_lt();
  uint32_t packed[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const bool def = ((force >> e) & 1u) || key[e] > tau;
    const bool eq = !def && need > 0 && key[e] == tau && key[e] != 0u;
    packed[e] = (uint32_t)__popc(__ballot_sync(0xffffffffu, def)) |
                ((uint32_t)__popc(__ballot_sync(0xffffffffu, eq)) << 16);
  }
  block_cell_offsets(packed, s);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const bool def = ((force >> e) & 1u) || key[e] > tau;
    const bool eq = !def && need > 0 && key[e] == tau && key[e] != 0u;
    const uint32_t bd = __ballot_sync(0xffffffffu, def), be = __ballot_sync(0xffffffffu, eq);
    const uint32_t base = s.cell[e * nwarps + warp];
    const uint32_t dbef = (base & 0xFFFFu) + __popc(bd & lt), ebef = (base >> 16) + __popc(be & lt);
    const int i = e * blockDim.x + threadIdx.x;
    if (def) out[dbef + min(ebef, (uint32_t)need)] = i;
    else if (eq && ebef < (uint32_t)need) out[dbef + ebef] = i;
  }
}

// Index of the need-th (1-based, index order) entry whose key equals tau; -1 if need <= 0.
template <int E>
__device__ inline int block_reg_nth_equal(const uint32_t (&key)[E], uint32_t tau, int need, RegSelShared& s) {
  if (need <= 0) return -1;
  const int warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const uint32_t lt = lanemask_lt();
  uint32_t packed[E];
#pragma unroll
  for (int e = 0; e < E; ++e) packed[e] = (uint32_t)__popc(__ballot_sync(0xffffffffu, key[e] == tau));
  block_cell_offsets(packed, s);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const uint32_t be = __ballot_sync(0xffffffffu, key[e] == tau);
    if (key[e] == tau && s.cell[e * nwarps + warp] + __popc(be & lt) + 1u == (uint32_t)need)
      s.res[3] = (uint32_t)(e * blockDim.x + threadIdx.x);
  }
  __syncthreads();
  const int cut = (int)s.res[3];
  __syncthreads();
  return cut;
}

// ------------------------------------------------------------------ launch helpers

// Raises a kernel's dynamic shared-memory limit once per (kernel, device) and size, so
// repeated launches (and launches under stream capture) make no attribute calls.
cudaError_t ensure_dynamic_smem_impl(const void* kernel, int bytes);

template <class Kernel>
inline cudaError_t ensure_dynamic_smem(Kernel kernel, int bytes) {
  return ensure_dynamic_smem_impl(reinterpret_cast<const void*>(kernel), bytes);
}

// Programmatic dependent launch: wait for the preceding grid of the stream (no-op when
// there is none), and let the next grid of the stream start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Test hook of the host-side error paths (trevs_test_fail_launch): true when this launch
// attempt of the calling thread is the one set to fail; the launch is then not made.
bool launch_fault_injected();

// Launches `kernel`, optionally allowed to start before the preceding work of the stream
// completes (it must then call pdl_wait() before it touches that work's results).
template <class... KArgs, class... Args>
inline cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                 bool pdl, Args... args) {
  if (launch_fault_injected()) return cudaErrorLaunchFailure;
  const cudaError_t e = ensure_dynamic_smem(kernel, (int)smem);   // carveout, dynamic limit
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  // a stream's priority, stated on the launch so that a captured graph keeps it
  int prio = 0;
  if (st != nullptr && cudaStreamGetPriority(st, &prio) == cudaSuccess && prio != 0) {
    attr[n].id = cudaLaunchAttributePriority;
    attr[n].val.priority = prio;
    ++n;
  }
  cfg.attrs = n ? attr : nullptr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ------------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// 16-byte async copy global -> shared; src_bytes = 0 zero-fills without reading.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                            uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D[16x8] += A[16x16] * B[16x8], bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// acc[0..3] += squares of the eight bf16 values in v (four independent chains).
__device__ __forceinline__ void bf16_sq_acc8(uint4 v, float (&acc)[4]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float lo = __uint_as_float(w[j] << 16), hi = __uint_as_float(w[j] & 0xFFFF0000u);
    acc[j] = fmaf(lo, lo, acc[j]);
    acc[j] = fmaf(hi, hi, acc[j]);
  }
}

// The same with packed fp32 FMAs (sm_100 family): eight partial sums in four pairs.
__device__ __forceinline__ void bf16_sq_acc8x2(uint4 v, float2 (&acc)[4]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 e = make_float2(__uint_as_float(w[j] << 16), __uint_as_float(w[j] & 0xFFFF0000u));
    acc[j] = __ffma2_rn(e, e, acc[j]);
  }
}

// Block-wide min of the non-zero keys and max of all keys (key 0 marks an excluded entry).
__device__ inline void block_key_range(uint32_t lo, uint32_t hi, SelShared& s, uint32_t& lo_out, uint32_t& hi_out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  if (lane == 0) { s.warp_gt[warp] = lo; s.warp_eq[warp] = hi; }
  __syncthreads();
  lo = 0xFFFFFFFFu;
  hi = 0u;
  for (int w = 0; w < nwarps; ++w) { lo = min(lo, s.warp_gt[w]); hi = max(hi, s.warp_eq[w]); }
  __syncthreads();
  lo_out = lo;
  hi_out = hi;
}

// keys[i] = f(src[i], i) for i < n by the whole block, also returning the key range
// (min over non-zero keys, max over all). 16-byte loads through L2 (the values may have
// been written by other blocks of the grid), eight in flight per thread.
template <class F>
__device__ inline void block_fill_keys(uint32_t* keys, const float* src, int n, F f, SelShared& s, uint32_t& lo,
                                       uint32_t& hi) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  uint32_t l = 0xFFFFFFFFu, h = 0u;
  auto put = [&](int i, float x) {
    const uint32_t k = f(x, i);
    keys[i] = k;
    if (k != 0u) l = min(l, k);
    h = max(h, k);
  };
  const int head = min(n, (int)(((16u - ((uint32_t)reinterpret_cast<uintptr_t>(src) & 15u)) & 15u) >> 2));
  if (tid < head) put(tid, __ldcg(src + tid));
  const float4* v = reinterpret_cast<const float4*>(src + head);
  const int nv = (n - head) >> 2;
  int j = tid;
  for (; j + 7 * nthr < nv; j += 8 * nthr) {
    float4 x[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) x[q] = __ldcg(v + j + q * nthr);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int i = head + 4 * (j + q * nthr);
      put(i, x[q].x);
      put(i + 1, x[q].y);
      put(i + 2, x[q].z);
      put(i + 3, x[q].w);
    }
  }
  for (; j < nv; j += nthr) {
    const float4 x = __ldcg(v + j);
    const int i = head + 4 * j;
    put(i, x.x);
    put(i + 1, x.y);
    put(i + 2, x.z);
    put(i + 3, x.w);
  }
  for (int i = head + 4 * nv + tid; i < n; i += nthr) put(i, __ldcg(src + i));
  block_key_range(l, h, s, lo, hi);   // synchronises: keys are complete afterwards
}

// keys[i] = f(a[i], b[i], i) for i < n by the whole block, returning the key range. Both
// sources are read with 16-byte loads when they share their alignment.
template <class F>
__device__ inline void block_fill_keys2(uint32_t* keys, const float* a, const float* b, int n, F f, SelShared& s,
                                        uint32_t& lo, uint32_t& hi) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  uint32_t l = 0xFFFFFFFFu, h = 0u;
  auto put = [&](int i, float x, float y) {
    const uint32_t k = f(x, y, i);
    keys[i] = k;
    if (k != 0u) l = min(l, k);
    h = max(h, k);
  };
  const uint32_t ma = (uint32_t)reinterpret_cast<uintptr_t>(a) & 15u, mb = (uint32_t)reinterpret_cast<uintptr_t>(b) & 15u;
  int head = n, nv = 0;
  if (ma == mb) {
    head = min(n, (int)(((16u - ma) & 15u) >> 2));
    nv = (n - head) >> 2;
  }
  for (int i = tid; i < head; i += nthr) put(i, __ldcg(a + i), __ldcg(b + i));
  const float4* va = reinterpret_cast<const float4*>(a + head);
  const float4* vb = reinterpret_cast<const float4*>(b + head);
  int j = tid;
  for (; j + 3 * nthr < nv; j += 4 * nthr) {
    float4 x[4], y[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      x[q] = __ldcg(va + j + q * nthr);
      y[q] = __ldcg(vb + j + q * nthr);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = head + 4 * (j + q * nthr);
      put(i, x[q].x, y[q].x);
      put(i + 1, x[q].y, y[q].y);
      put(i + 2, x[q].z, y[q].z);
      put(i + 3, x[q].w, y[q].w);
    }
  }
  for (; j < nv; j += nthr) {
    const float4 x = __ldcg(va + j), y = __ldcg(vb + j);
    const int i = head + 4 * j;
    put(i, x.x, y.x);
    put(i + 1, x.y, y.y);
    put(i + 2, x.z, y.z);
    put(i + 3, x.w, y.w);
  }
  for (int i = head + 4 * nv + tid; i < n; i += nthr) put(i, __ldcg(a + i), __ldcg(b + i));
  block_key_range(l, h, s, lo, hi);
}

// Physical 16-byte chunk of logical chunk c in a 128-byte row r (XOR swizzle, conflict-free
// for ldmatrix and for row-wise reads).
__device__ __forceinline__ int swz(int r, int c) { return c ^ (r & 7); }

}  // namespace trevs
