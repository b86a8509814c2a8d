// Stage 1 context preservation (Sec. 3.1): farthest point sampling of the K_d diversity
// tokens over the candidates C = [N] minus the pivots S_r, in cosine distance.
#pragma once

#include "pre_llm.cuh"

namespace trevs {

constexpr int kFpsThreads = 512;
constexpr int kFpsMaxPool = 128;   // candidates whose pairwise cosines are kept on chip

struct FpsReq {
  int n_off, n;       // visual rows of Z (and of maxcos, ub, stamp, flags)
  int piv_off, kr;    // pivots S_r at piv[piv_off ..], request-local rows
  int kd;             // tokens to draw
  int lead;           // 1: no pivots were given; row 0 is the first draw (distance +inf) and
                      //    stands as the single pivot of the contraction (kr = 1)
  int pick_off;       // picks / pick_dist at [pick_off ..]
  int kept_off;       // S_r and S_d together, ascending, at kept[kept_off ..] (when kept is set)
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
};

}  // namespace trevs
