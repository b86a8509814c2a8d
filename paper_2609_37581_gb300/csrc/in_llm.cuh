// Stage 2 (in-LLM, Sec. 4.2) kernel arguments.
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace trevs {

constexpr int kMaxHeads = 128;
constexpr int kKeyBlock = 64;        // visual keys per stage-2 block / shared-memory chunk
constexpr int kScoreTextRows = 16;   // text rows per token-score block

// Text rows per head-statistics block: the block keeps rows x K1 fp32 logits on chip.
inline int stats_text_rows(int max_k1) { return max_k1 <= 128 ? 64 : (max_k1 <= 512 ? 32 : 16); }

struct InArgs {
  const __nv_bfloat16* Q;
  long long q_hs, q_ts;     // head / token strides (elements)
  const __nv_bfloat16* K;
  long long k_hs, k_ts;
  int Hq, Hkv, n_keep;
  float scale;
  float* attn;              // attention probabilities, request b at attn_off: [Hq][l][k1]
  float* row_var;           // [Hq][stats_ld]: Var_i A[q, i]
  long long stats_ld;       // total text rows of the launch
  float* u;                 // [B][u_ld] head variances (Eq. 8)
  int u_ld;
  uint32_t* p_bits;         // [sum k1] Eq. 9 scores as float bits (atomicMax target)
  int* kept_local;          // [sum k2]
  int* heads_out;           // [B][n_keep] or null
  uint32_t* keys;           // [sum k1] selection scratch
  uint8_t* flags;           // [sum k1] selection scratch
  uint32_t* cnt_hs;         // [B] self-resetting tickets
  uint32_t* cnt_ts;         // [B]
  int hs_finalize;          // head-statistics blocks reduce u (ticket)
  int zero_p;               // ... and clear p for the token-score pass
  int overlap;              // head statistics need not wait for the preceding grid at start
  int independent;          // Q and K do not come from the preceding grid: the first
                            // stage-2 grid never waits for it (it may run beside it)
  const float* lse;         // full-sequence variant: log of the non-visual mass of row (h, q),
                            // at lse + h * lse_hs + (launch text row) * lse_rs; null: off
  long long lse_hs, lse_rs;
  float2* rstat;            // [Hq][stats_ld]: (T, 1 / total) of each text row, log2 units, so that
                            // A[h][q][i] = exp2(logit * scale * log2 e - T) / total
  uint32_t* err;            // device status word: bit 0 = a bounded wait gave up
};

// Tensor map of a [rows][heads][128] bf16 tensor, boxes of box_rows rows x 64 dims of one head.
cudaError_t make_tmap_heads(CUtensorMap* tm, const void* base, long long rows, int heads, long long tok_stride,
                            long long head_stride, int box_rows);

// Stage 2 on the tensor cores (in_llm_tc.cu): tensor maps of Q and K, rows per block and keys
// per token-score block (for the host's block offsets), and the two grids.
struct InQMaps {
  CUtensorMap q128, q64, q32;   // Q boxes of 128, 64 and 32 rows
};
struct InTcMaps {
  InQMaps q;
  CUtensorMap k128, k64;
};
cudaError_t make_in_tc_maps(const InArgs& a, long long q_rows, long long k_rows, InTcMaps& m);
int in_tc_text_rows();
int in_tc_score_keys();
cudaError_t launch_in_stats_tc(const InMeta& meta, const InArgs& a, const InTcMaps& m, cudaStream_t st);
cudaError_t launch_in_score_tc(const InMeta& meta, const InArgs& a, const InTcMaps& m, cudaStream_t st);

}  // namespace trevs
