// Stage 1 (pre-LLM, Sec. 4.1) kernels: textual-relevance scoring, per-request selection
// and the gather of kept rows.
#pragma once

#include "common.cuh"

namespace trevs {

enum { kModeRatio = 0, kModeFused = 1 };

constexpr int kScoreTileRows = 128;   // visual rows per scoring tile (UMMA M)
constexpr int kMaxScoreCtas = 256;    // CTAs of the persistent scoring grid, at most
enum { kActScores = 0, kActScoresFused = 1, kActSelect = 2, kActFpsSeed = 3 };
// kActFpsSeed: the scoring contraction for farthest point sampling (Sec. 3.1). The "text"
// rows are copies of the pivot rows of Z, and s_t receives max_j cos(z_i, z_pivot_j).

struct PreArgs {
  const __nv_bfloat16* Z;
  long long z_stride;
  const __nv_bfloat16* T;
  long long t_stride;
  const float* s_v;
  float* s_t;          // [sum n]
  float* s_fused;      // [sum n] (fused mode)
  float* t_rinv;       // [sum m] 1 / ||t_j|| (0 for a zero row), from the pre-pass
  long long total_m;   // text rows of the launch
  float* part;         // [2 per scoring CTA] partial sums of tiles split between CTAs
  int* kept;           // [sum k1]
  uint8_t* flags;      // [sum n] scratch
  uint32_t* keys;      // [sum n] scratch (used when shared memory is too small)
  uint32_t* counters;  // [B] tiles finished per request (self-resetting)
  int4* sal;           // [B] saliency side of the selection (see saliency_prepare)
  int sal_ready;       // 1: sal was filled by the saliency kernel earlier in the stream
  int score_reserve;   // SMs the scoring grid leaves to work that runs beside it
  uint32_t* err;       // device status word: bit 0 = a bounded wait gave up
  int d;
  int mode;
  float tau_v, tau_t, lambda, eps;
  int action;          // kActScores / kActScoresFused / kActSelect
  int s_fused_given;   // select kernel: s_fused already holds Eq. 7 scores
  int seed_merge;      // kActFpsSeed: s_t already holds the largest cosine to earlier pivots
                       // (a pass over further pivot columns keeps the max)
  int big_sel;         // requests above kRegSelMaxN are selected by pre_select_big_kernel
};

// Saliency side of the selection, which depends on inputs only. Ratio mode: the rule for
// S_v = the K_v tokens of largest s_v, as (tau, need, n_eq, cut): token i is in S_v iff
// key(s_v[i]) > tau, or key == tau and (need >= n_eq or i <= cut). Fused mode: Med and MAD
// of s_v (Eq. 6) as float bits in .x and .y. `keys` holds n entries, 16-byte aligned.
__device__ inline int4 saliency_prepare(const PreArgs& a, const PreReq& r, uint32_t* keys, SelShared& ss) {
  const int n = r.n;
  const float* sv = a.s_v + r.n_off;
  uint32_t lo, hi, tau;
  int need, n_eq;
  if (a.mode == kModeRatio) {
    const int kv = r.k1 - r.kt;
    if (kv <= 0 || n <= 0) return make_int4(-1, 0, 1, -1);   // empty: nothing passes the rule
    block_fill_keys(keys, sv, n, [&](float x, int) { return score_key(x); }, ss, lo, hi);
    block_kth_largest(keys, n, kv, ss, lo, hi, tau, need, n_eq);
    int cut = -1;
    if (need < n_eq) {   // ties at the threshold: the need-th equal key in index order
      if (threadIdx.x == 0) ss.bcast[3] = 0u;
      __syncthreads();
      block_emit_selected(keys, n, tau, need, ss, [&](int i, int, bool sel) {
        if (sel && keys[i] == tau) atomicMax(&ss.bcast[3], (uint32_t)i);
      });
      cut = (int)ss.bcast[3];
      __syncthreads();
    }
    return make_int4((int)tau, need, n_eq, cut);
  }
  if (n <= 0) return make_int4(0, 0, 0, 0);
  const int kmed = n - (n - 1) / 2;  // lower median = kmed-th largest
  block_fill_keys(keys, sv, n, [&](float x, int) { return score_key(x); }, ss, lo, hi);
  block_kth_largest(keys, n, kmed, ss, lo, hi, tau, need, n_eq);
  const float med = key_to_score(tau);
  block_fill_keys(keys, sv, n, [&](float x, int) { return score_key(fabsf(x - med)); }, ss, lo, hi);
  block_kth_largest(keys, n, kmed, ss, lo, hi, tau, need, n_eq);
  return make_int4(__float_as_int(med), __float_as_int(key_to_score(tau)), 0, 0);
}

__device__ __forceinline__ bool in_saliency_set(float sv, int i, int4 rule) {
  const uint32_t k = score_key(sv), tau = (uint32_t)rule.x;
  return k > tau || (k == tau && (rule.y >= rule.z || i <= rule.w));
}

// Selection for one request by the whole block (any multiple of 32 threads). `b` is the
// request's slot in the launch; `sal` is its saliency rule when already prepared.
__device__ inline void select_request(const PreArgs& a, const PreReq& r, int b, uint8_t* smem, int smem_bytes,
                                      SelShared& ss, bool compute_fused, bool do_select) {
  const int n = r.n;
  if (n <= 0) return;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const float* sv = a.s_v + r.n_off;
  const float* st = a.s_t + r.n_off;
  const bool in_smem = (size_t)n * 5 + 16 <= (size_t)smem_bytes;
  // global fallback: request b's scratch starts at a 16-byte boundary inside [sum n + 4B]
  const size_t gbase = ((size_t)r.n_off + 4 * (size_t)b + 3) & ~(size_t)3;
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + gbase;
  uint8_t* flags = in_smem ? smem + (size_t)n * 4 : a.flags + gbase;
  int* out = a.kept + r.k1_off;
  uint32_t lo, hi, tau;
  int need, n_eq;
  int4 rule = make_int4(-1, 0, 1, -1);
  if (a.sal_ready) {
    pdl_wait();   // the saliency kernel precedes this grid in the stream
    rule = __ldcg(a.sal + b);
  } else if (a.mode == kModeRatio || compute_fused) {
    rule = saliency_prepare(a, r, keys, ss);
  }

  if (a.mode == kModeRatio) {
    if (!do_select) return;
    // S_v from its rule; the textual keys exclude it (key 0)
    block_fill_keys2(keys, st, sv, n, [&](float x, float v, int i) {
      const bool in_v = in_saliency_set(v, i, rule);
      flags[i] = in_v ? 1 : 0;
      return in_v ? 0u : score_key(x);
    }, ss, lo, hi);
    if (r.kt > 0 && n <= nthr) {
      block_mark_topk_small(keys, n, r.kt, flags);
    } else if (r.kt > 0) {
      block_kth_largest(keys, n, r.kt, ss, lo, hi, tau, need, n_eq);
      block_mark_selected(keys, n, tau, need, n_eq, flags, ss);
    }
    block_compact_flags(flags, n, out, ss);
    return;
  }

  // fused mode (Eq. 6-7)
  float* sf = a.s_fused + r.n_off;
  if (compute_fused) {
    const int kmed = n - (n - 1) / 2;  // lower median = kmed-th largest
    const float med_v = __int_as_float(rule.x), mad_v = __int_as_float(rule.y);
    block_fill_keys(keys, st, n, [&](float x, int) { return score_key(x); }, ss, lo, hi);
    block_kth_largest(keys, n, kmed, ss, lo, hi, tau, need, n_eq);
    const float med_t = key_to_score(tau);
    block_fill_keys(keys, st, n, [&](float x, int) { return score_key(fabsf(x - med_t)); }, ss, lo, hi);
    block_kth_largest(keys, n, kmed, ss, lo, hi, tau, need, n_eq);
    const float mad_t = key_to_score(tau);
    const float dv = mad_v + a.eps, dt = mad_t + a.eps;
    for (int i = tid; i < n; i += nthr) {
      float hv = fmaxf((__ldcg(sv + i) - med_v) / dv, 0.f) / a.tau_v;
      float ht = fmaxf((__ldcg(st + i) - med_t) / dt, 0.f) / a.tau_t;
      sf[i] = fmaxf(hv, ht) + a.lambda * sqrtf(hv * ht);
    }
    __syncthreads();
  }
  if (do_select && r.k1 > 0) {
    for (int i = tid; i < n; i += nthr) flags[i] = 0;
    block_fill_keys(keys, sf, n, [&](float x, int) { return score_key(x); }, ss, lo, hi);
    if (n <= nthr) {
      block_mark_topk_small(keys, n, r.k1, flags);
    } else {
      block_kth_largest(keys, n, r.k1, ss, lo, hi, tau, need, n_eq);
      block_mark_selected(keys, n, tau, need, n_eq, flags, ss);
    }
    block_compact_flags(flags, n, out, ss);
  }
}

// Register-resident forms of the two functions above for n <= E * blockDim.x (blockDim.x
// a multiple of 32, at least 256): thread t holds entries e * blockDim.x + t.
template <int E>
__device__ inline int4 saliency_prepare_reg(const PreArgs& a, const PreReq& r, RegSelShared& rs) {
  const int n = r.n;
  const float* sv = a.s_v + r.n_off;
  const int tid = threadIdx.x, nthr = blockDim.x;
  uint32_t key[E];
  if (a.mode == kModeRatio) {
    const int kv = r.k1 - r.kt;
    if (kv <= 0 || n <= 0) return make_int4(-1, 0, 1, -1);   // empty: nothing passes the rule
#pragma unroll
    for (int e = 0; e < E; ++e) key[e] = e * nthr + tid < n ? score_key(__ldcg(sv + e * nthr + tid)) : 0u;
    uint32_t tau;
    int need;
    block_reg_topk(key, kv, rs, tau, need);
    // ties at tau: the first `need` of them in index order, i.e. up to the need-th one
    const int cut = block_reg_nth_equal(key, tau, need, rs);
    return make_int4((int)tau, 0, 1, cut);
  }
  if (n <= 0) return make_int4(0, 0, 0, 0);
  const int kmed = n - (n - 1) / 2;  // lower median = kmed-th largest
  float v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    v[e] = e * nthr + tid < n ? __ldcg(sv + e * nthr + tid) : 0.f;
    key[e] = e * nthr + tid < n ? score_key(v[e]) : 0u;
  }
  const float med = key_to_score(block_reg_kth(key, kmed, rs));
#pragma unroll
  for (int e = 0; e < E; ++e) key[e] = e * nthr + tid < n ? score_key(fabsf(v[e] - med)) : 0u;
  const float mad = key_to_score(block_reg_kth(key, kmed, rs));
  return make_int4(__float_as_int(med), __float_as_int(mad), 0, 0);
}

template <int E>
__device__ inline void select_request_reg(const PreArgs& a, const PreReq& r, int b, RegSelShared& rs,
                                          bool compute_fused, bool do_select) {
  const int n = r.n;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const float* sv = a.s_v + r.n_off;
  const float* st = a.s_t + r.n_off;
  int4 rule = make_int4(-1, 0, 1, -1);
  if (a.sal_ready) rule = __ldcg(a.sal + b);
  else if (a.mode == kModeRatio ? do_select : compute_fused) rule = saliency_prepare_reg<E>(a, r, rs);
  uint32_t key[E];
  uint32_t tau;
  int need;
  if (a.mode == kModeRatio) {
    if (!do_select || r.k1 <= 0) return;
    // S_v from its rule (forced in); the textual keys exclude it (key 0)
    uint32_t force = 0u;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int i = e * nthr + tid;
      key[e] = 0u;
      if (i < n) {
        if (in_saliency_set(__ldcg(sv + i), i, rule)) force |= 1u << e;
        else key[e] = score_key(__ldcg(st + i));
      }
    }
    block_reg_topk(key, r.kt, rs, tau, need);
    block_reg_emit(key, force, tau, need, a.kept + r.k1_off, rs);
    return;
  }

  // fused mode (Eq. 6-7)
  float* sf = a.s_fused + r.n_off;
  float f[E];
  if (compute_fused) {
    float t[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
      t[e] = e * nthr + tid < n ? __ldcg(st + e * nthr + tid) : 0.f;
      key[e] = e * nthr + tid < n ? score_key(t[e]) : 0u;
    }
    const int kmed = n - (n - 1) / 2;  // lower median = kmed-th largest
    const float med_t = key_to_score(block_reg_kth(key, kmed, rs));
#pragma unroll
    for (int e = 0; e < E; ++e) key[e] = e * nthr + tid < n ? score_key(fabsf(t[e] - med_t)) : 0u;
    const float mad_t = key_to_score(block_reg_kth(key, kmed, rs));
    const float med_v = __int_as_float(rule.x), mad_v = __int_as_float(rule.y);
    const float dv = mad_v + a.eps, dt = mad_t + a.eps;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int i = e * nthr + tid;
      f[e] = 0.f;
      if (i < n) {
        const float hv = fmaxf((__ldcg(sv + i) - med_v) / dv, 0.f) / a.tau_v;
        const float ht = fmaxf((t[e] - med_t) / dt, 0.f) / a.tau_t;
        f[e] = fmaxf(hv, ht) + a.lambda * sqrtf(hv * ht);
        sf[i] = f[e];
      }
    }
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e) f[e] = e * nthr + tid < n ? __ldcg(sf + e * nthr + tid) : 0.f;
  }
  if (!do_select || r.k1 <= 0) return;
#pragma unroll
  for (int e = 0; e < E; ++e) key[e] = e * nthr + tid < n ? score_key(f[e]) : 0u;
  block_reg_topk(key, r.k1, rs, tau, need);
  block_reg_emit(key, 0u, tau, need, a.kept + r.k1_off, rs);
}

union SelScratch {
  SelShared ss;
  RegSelShared rs;
};

// Largest request the register-resident forms take with 512 threads (larger ones are
// faster with the keys in memory).
constexpr int kRegSelMaxN = 8 * 512;

// Saliency rule of request r by a block of 512 threads; `keys` (n entries, 16-byte
// aligned) is only touched for requests above kRegSelMaxN.
__device__ inline int4 saliency_rule_512(const PreArgs& a, const PreReq& r, uint32_t* keys, SelScratch& sh) {
  const int n = r.n;
  if (n <= 512) return saliency_prepare_reg<1>(a, r, sh.rs);
  if (n <= 1024) return saliency_prepare_reg<2>(a, r, sh.rs);
  if (n <= kRegSelMaxN) return saliency_prepare_reg<8>(a, r, sh.rs);
  return saliency_prepare(a, r, keys, sh.ss);
}

// Selection (or fused scores) of request r by a block of 512 threads.
__device__ inline void select_request_512(const PreArgs& a, const PreReq& r, int b, uint8_t* smem, int smem_bytes,
                                          SelScratch& sh) {
  const int n = r.n;
  if (n <= 0) return;
  const bool compute_fused = a.mode == kModeFused && !a.s_fused_given;
  const bool do_select = a.action == kActSelect;
  if (n <= 512) select_request_reg<1>(a, r, b, sh.rs, compute_fused, do_select);
  else if (n <= 1024) select_request_reg<2>(a, r, b, sh.rs, compute_fused, do_select);
  else if (n <= kRegSelMaxN) select_request_reg<8>(a, r, b, sh.rs, compute_fused, do_select);
  else select_request(a, r, b, smem, smem_bytes, sh.ss, compute_fused, do_select);
}

// ------------------------------------------------------------------ row gather

struct GatherJob {
  const uint8_t* src;
  uint8_t* dst;
  long long src_tok, dst_tok;    // bytes between rows
  long long src_head, dst_head;  // bytes between heads
  int heads;
  int row_bytes;                 // per (row, head), multiple of 16
  const int* idx;                // request-local source row of each destination row
  int rows;                      // destination rows (all requests)
  int tab;                       // offset table of the job's requests
};

// Per-request row offsets of one family of gathers (stage-1 rows or stage-2 rows).
struct GatherTable {
  int B;
  int dst_off[kMaxChunk + 1];
  int src_off[kMaxChunk];
  int src_rows[kMaxChunk];   // source rows of each request: out-of-range indices are skipped
};

struct GatherMeta {
  int njobs;
  GatherTable t[2];
  GatherJob job[4];
};

}  // namespace trevs
