// Vision-encoder saliency (Sec. 4.1, Eq. 2-3) kernel arguments.
#pragma once

#include "common.cuh"

namespace trevs {

constexpr int kClsMaxN = 16384;   // logits of one head in shared memory (64 KB)

struct ClsReq {
  int n_off, n;   // patch rows [n_off, n_off + n) of K_v and s_v
  int b;          // slot of the request in the launch (its q row and ticket)
};

struct ClsMeta {
  int B, H;
  ClsReq r[kMaxChunk];
};

struct ClsArgs {
  const __nv_bfloat16* q;   // element (b, h, c) at q + b*q_req + h*q_head + c
  long long q_req, q_head;
  const __nv_bfloat16* K;   // element (i, h, c) at K + i*k_tok + h*k_head + c
  long long k_tok, k_head;
  float scale;
  float* attn;              // [H][sum n]: A^h of every patch
  long long attn_ld;        // sum n of the launch
  float* s_v;               // [sum n]
  uint32_t* cnt;            // [B] tickets, reset by the last block of each request
};

bool cls_head_dim_supported(int dh);

}  // namespace trevs
