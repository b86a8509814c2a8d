// Stage 1 context preservation (Sec. 3.1): farthest point sampling of the K_d diversity
// tokens over the candidates C = [N] minus the pivots S_r, in cosine distance.
#pragma once

#include "pre_llm.cuh"

namespace trevs {

constexpr int kFpsThreads = 512;
constexpr int kFpsMaxPool = 128;   // candidates whose pairwise cosines are kept on chip
constexpr int kFpsMaxPoolBig = 1024;   // larger pools keep their cosines in the workspace
constexpr int kFpsGramTile = 64;       // pool cosines: rows x columns of one block of the Gram grid

// Pool size asked for K_d draws: about twice K_d, at least K_d + 32; four times K_d once
// the pool's cosines live in the workspace (K_d above 64).
__host__ __device__ inline int fps_auto_pool(int kd) {
  const int w = 2 * kd > kd + 32 ? 2 * kd : kd + 32;
  return w > kFpsMaxPool ? 4 * kd : w;
}

struct FpsReq {
  int n_off, n;       // visual rows of Z (and of maxcos, ub, stamp, flags)
  int piv_off, kr;    // pivots S_r at piv[piv_off ..], request-local rows
  int kd;             // tokens to draw
  int lead;           // 1: no pivots were given; row 0 is the first draw (distance +inf) and
                      //    stands as the single pivot of the contraction (kr = 1)
  int pick_off;       // picks / pick_dist at [pick_off ..]
  int kept_off;       // S_r and S_d together, ascending, at kept[kept_off ..] (when kept is set)
  // pools above kFpsMaxPool (phases 1 and 2): pool indices at pool_idx[pool_off ..], at most
  // gram_ld of them; their cosines at gram[gram_off ..], row stride gram_ld; Gram tiles
  // [gt_off, gt_off + (gram_ld / kFpsGramTile)^2) of the Gram grid
  int pool_off, gram_ld, gt_off;
  long long gram_off;
};

struct FpsMeta {
  int B;
  FpsReq r[kMaxChunk];
};

struct FpsArgs {
  const __nv_bfloat16* Z;
  long long z_stride;
  int d;
  const int* piv;
  const float* maxcos;   // [sum n] max over the pivots of cos(z_i, z_s); unused when kr == 0
  float* ub;             // [sum n] scratch: distance bounds of the candidates outside the pool
  int* stamp;            // [sum n] scratch: picks a bound accounts for; -1 = not outside the pool
  uint8_t* flags;        // [sum n] scratch: 1 pivot, 2 pick
  uint32_t* keys;        // [sum n + 4 per request + 4] scratch for requests above kRegSelMaxN
  int* picks;            // [sum kd] in the order they are drawn
  float* pick_dist;      // [sum kd] distance of each pick when drawn, or null
  int* kept;             // or null
  int pool;              // pool size asked for (0: automatic)
  uint32_t* err;         // device status word: bit 1 = the draw found no candidate
  // 0: pool, cosines and draws in one block (pools up to kFpsMaxPool); 1: the pool and the
  // bounds only, into pool_idx / pool_n; 2: the draws, with the pool cosines in gram
  int phase;
  int* pool_idx;         // [sum of gram_ld] pool rows of each request (phases 1, 2)
  int* pool_n;           // [B] pool size of each request (phases 1, 2)
  float* gram;           // [sum of gram_ld^2] pool dot products (phases 1, 2)
};

}  // namespace trevs
