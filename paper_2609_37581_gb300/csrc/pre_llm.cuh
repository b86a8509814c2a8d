// Stage 1 (pre-LLM, Sec. 4.1) kernels: textual-relevance scoring, per-request selection
// and the gather of kept rows.
#pragma once

#include "common.cuh"

namespace trevs {

enum { kModeRatio = 0, kModeFused = 1 };
enum { kActScores = 0, kActScoresFused = 1, kActSelect = 2 };

struct PreArgs {
  const __nv_bfloat16* Z;
  long long z_stride;
  const __nv_bfloat16* T;
  long long t_stride;
  const float* s_v;
  float* s_t;          // [sum n]
  float* s_fused;      // [sum n] (fused mode)
  int* kept;           // [sum k1]
  uint8_t* flags;      // [sum n] scratch
  uint32_t* keys;      // [sum n] scratch (used when shared memory is too small)
  uint32_t* counters;  // [B] tiles finished per request (self-resetting)
  int d;
  int mode;
  float tau_v, tau_t, lambda, eps;
  int action;          // kActScores / kActScoresFused / kActSelect
  int s_fused_given;   // select kernel: s_fused already holds Eq. 7 scores
};

// Selection for one request by the whole block (any multiple of 32 threads).
__device__ inline void select_request(const PreArgs& a, const PreReq& r, uint8_t* smem,
                                      int smem_bytes, SelShared& ss, bool compute_fused,
                                      bool do_select) {
  const int n = r.n;
  if (n <= 0) return;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const float* sv = a.s_v + r.n_off;
  const float* st = a.s_t + r.n_off;
  const bool in_smem = (size_t)n * 5 + 16 <= (size_t)smem_bytes;
  uint32_t* keys = in_smem ? reinterpret_cast<uint32_t*>(smem) : a.keys + r.n_off;
  uint8_t* flags = in_smem ? smem + (size_t)n * 4 : a.flags + r.n_off;
  int* out = a.kept + r.k1_off;
  uint32_t tau;
  int need;

  if (a.mode == kModeRatio) {
    if (!do_select) return;
    const int kv = r.k1 - r.kt, kt = r.kt;
    if (kv > 0) {
      for (int i = tid; i < n; i += nthr) keys[i] = score_key(__ldcg(sv + i));
      __syncthreads();
      block_kth_largest(keys, n, kv, ss, tau, need);
      block_emit_selected(keys, n, tau, need, ss,
                          [&](int i, int, bool sel) { flags[i] = sel ? 1 : 0; });
    } else {
      for (int i = tid; i < n; i += nthr) flags[i] = 0;
      __syncthreads();
    }
    if (kt > 0) {
      // tokens already kept by saliency get key 0, below every finite score
      for (int i = tid; i < n; i += nthr) keys[i] = flags[i] ? 0u : score_key(__ldcg(st + i));
      __syncthreads();
      block_kth_largest(keys, n, kt, ss, tau, need);
      block_emit_selected(keys, n, tau, need, ss,
                          [&](int i, int, bool sel) { if (sel) flags[i] = 1; });
    }
    block_compact_flags(flags, n, out, ss);
    return;
  }

  // fused mode (Eq. 6-7)
  float* sf = a.s_fused + r.n_off;
  if (compute_fused) {
    const int kmed = n - (n - 1) / 2;  // lower median = kmed-th largest
    // Med and MAD of one signal by two order-statistic selections
    auto med_mad = [&](const float* s, float& med, float& mad) {
      for (int i = tid; i < n; i += nthr) keys[i] = score_key(__ldcg(s + i));
      __syncthreads();
      block_kth_largest(keys, n, kmed, ss, tau, need);
      med = key_to_score(tau);
      for (int i = tid; i < n; i += nthr) keys[i] = score_key(fabsf(__ldcg(s + i) - med));
      __syncthreads();
      block_kth_largest(keys, n, kmed, ss, tau, need);
      mad = key_to_score(tau);
    };
    float med_v, mad_v, med_t, mad_t;
    med_mad(sv, med_v, mad_v);
    med_mad(st, med_t, mad_t);
    const float dv = mad_v + a.eps, dt = mad_t + a.eps;
    for (int i = tid; i < n; i += nthr) {
      float hv = fmaxf((__ldcg(sv + i) - med_v) / dv, 0.f) / a.tau_v;
      float ht = fmaxf((__ldcg(st + i) - med_t) / dt, 0.f) / a.tau_t;
      sf[i] = fmaxf(hv, ht) + a.lambda * sqrtf(hv * ht);
    }
    __syncthreads();
  }
  if (do_select && r.k1 > 0) {
    for (int i = tid; i < n; i += nthr) keys[i] = score_key(__ldcg(sf + i));
    __syncthreads();
    block_kth_largest(keys, n, r.k1, ss, tau, need);
    block_emit_selected(keys, n, tau, need, ss,
                        [&](int i, int pos, bool sel) { if (sel) out[pos] = i; });
  }
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
  int pad_;
};

struct GatherMeta {
  int B;
  int njobs;
  int dst_off[kMaxChunk + 1];
  int src_off[kMaxChunk];
  int src_rows[kMaxChunk];   // source rows of each request: out-of-range indices are skipped
  GatherJob job[4];
};

}  // namespace trevs
