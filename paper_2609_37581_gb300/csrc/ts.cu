// Eq. 1 (Sec. 3.2): the textual sensitivity of every attention head. For the same image asked
// two questions, head h's attention over the K1 visual tokens, averaged over each question's
// text rows, gives two distributions s_h^(1) and s_h^(2); TS_h = 1 - cos(s_h^(1), s_h^(2)). A
// head whose visual attention hardly moves with the question has TS_h near 0.
//
// One block per (head, 128 visual keys): thread i sums column i of the head's attention over
// the text rows of each question (coalesced 128-float row segments, eight loads in flight per
// thread), scales by 1/L, and the block reduces its share of s1.s2, |s1|^2 and |s2|^2 into a
// workspace slot. The last block of a head (a self-resetting ticket) adds the slots in key
// order, so the result does not depend on which block finishes last.
#include "common.cuh"
#include "trevs.h"

namespace trevs {

trevs_status record_error(trevs_status s, const char* msg);
void record_launches(int n);

namespace {

constexpr int kTsKeys = 128;   // visual keys (and threads) per block

struct TsArgs {
  const float* a1;   // [Hq][L1][K1]
  const float* a2;   // [Hq][L2][K1]
  int L1, L2, K1, nchunk;
  float* s1;         // optional [Hq][K1] outputs: the head-mean distributions
  float* s2;
  float* part;       // [Hq][nchunk][3] block partial sums
  uint32_t* cnt;     // [Hq] tickets
  float* ts;         // [Hq]
};

// Sum over rows q < L of col[q * ld], eight loads in flight.
__device__ __forceinline__ float column_sum(const float* col, int L, long long ld) {
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int q = 0;
  for (; q + 8 <= L; q += 8) {
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] += __ldg(col + (long long)(q + j) * ld);
  }
  for (int j = 0; q < L; ++q, ++j) acc[j] += __ldg(col + (long long)q * ld);
  return ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
}

__global__ void __launch_bounds__(kTsKeys) textual_sensitivity_kernel(const TsArgs a) {
  __shared__ float red[3][kTsKeys / 32];
  __shared__ int s_last;
  const int c = blockIdx.x, h = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int i = c * kTsKeys + tid;
  float v[3] = {0.f, 0.f, 0.f};   // s1.s2, |s1|^2, |s2|^2 over this thread's key
  if (i < a.K1) {
    const float s1 = column_sum(a.a1 + (long long)h * a.L1 * a.K1 + i, a.L1, a.K1) / (float)a.L1;
    const float s2 = column_sum(a.a2 + (long long)h * a.L2 * a.K1 + i, a.L2, a.K1) / (float)a.L2;
    if (a.s1) a.s1[(long long)h * a.K1 + i] = s1;
    if (a.s2) a.s2[(long long)h * a.K1 + i] = s2;
    v[0] = s1 * s2;
    v[1] = s1 * s1;
    v[2] = s2 * s2;
  }
#pragma unroll
  for (int k = 0; k < 3; ++k) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
    if (lane == 0) red[k][warp] = v[k];
  }
  __syncthreads();
  float* slot = a.part + ((long long)h * a.nchunk + c) * 3;
  if (tid < 3) slot[tid] = (red[tid][0] + red[tid][1]) + (red[tid][2] + red[tid][3]);
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t done = atomicAdd(a.cnt + h, 1u) + 1u;
    s_last = done == (uint32_t)a.nchunk;
    if (s_last) a.cnt[h] = 0u;   // ready for the next call
  }
  __syncthreads();
  if (!s_last || tid != 0) return;
  __threadfence();
  double dot = 0.0, n1 = 0.0, n2 = 0.0;   // a few hundred slots at most: added in key order
  const float* p = a.part + (long long)h * a.nchunk * 3;
  for (int x = 0; x < a.nchunk; ++x) {
    dot += __ldcg(p + 3 * x);
    n1 += __ldcg(p + 3 * x + 1);
    n2 += __ldcg(p + 3 * x + 2);
  }
  const double den = sqrt(n1) * sqrt(n2);
  // a zero distribution has cosine 0 with everything (as for Eq. 4)
  a.ts[h] = (float)(1.0 - (den > 0.0 ? dot / den : 0.0));
}

constexpr size_t kStatusBytes = 256;
inline size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

struct TsWs {
  size_t cnt, part, end;
};

TsWs ts_ws(int Hq, int K1) {
  TsWs w;
  const int nchunk = (K1 + kTsKeys - 1) / kTsKeys;
  size_t o = kStatusBytes;
  w.cnt = o;  o = al256(o + 4 * (size_t)Hq);
  w.part = o; o = al256(o + 12 * (size_t)Hq * (size_t)nchunk);
  w.end = o;
  return w;
}

}  // namespace
}  // namespace trevs

using namespace trevs;

extern "C" {

size_t trevs_textual_sensitivity_workspace_size(int32_t Hq, int32_t K1) {
  if (Hq < 1 || K1 < 1) return 0;
  return ts_ws(Hq, K1).end;
}

trevs_status trevs_textual_sensitivity(const float* attn1, int32_t L1, const float* attn2, int32_t L2, int32_t Hq,
                                       int32_t K1, float* ts_out, float* s1_out, float* s2_out, void* workspace,
                                       size_t workspace_bytes, void* stream) {
  record_launches(0);
  if (Hq < 1 || K1 < 1 || L1 < 1 || L2 < 1)
    return record_error(TREVS_ERR_INVALID_ARGUMENT, "need Hq, K1, L1, L2 >= 1");
  if (Hq > 65535) return record_error(TREVS_ERR_UNSUPPORTED, "Hq above 65535");
  if (!attn1 || !attn2 || !ts_out)
    return record_error(TREVS_ERR_INVALID_ARGUMENT, "attn1, attn2 and ts_out must be non-NULL");
  const TsWs L = ts_ws(Hq, K1);
  if (!workspace || ((uintptr_t)workspace & 255u) != 0 || workspace_bytes < L.end)
    return record_error(TREVS_ERR_WORKSPACE, "workspace missing, not 256-byte aligned or too small");
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  TsArgs a;
  a.a1 = attn1; a.a2 = attn2;
  a.L1 = L1; a.L2 = L2; a.K1 = K1;
  a.nchunk = (K1 + kTsKeys - 1) / kTsKeys;
  a.s1 = s1_out; a.s2 = s2_out;
  a.part = reinterpret_cast<float*>(ws + L.part);
  a.cnt = reinterpret_cast<uint32_t*>(ws + L.cnt);
  a.ts = ts_out;
  if (launch_fault_injected()) return record_error(TREVS_ERR_CUDA, "injected launch failure (test hook)");
  textual_sensitivity_kernel<<<dim3((unsigned)a.nchunk, (unsigned)Hq), kTsKeys, 0,
                               static_cast<cudaStream_t>(stream)>>>(a);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return record_error(TREVS_ERR_CUDA, cudaGetErrorString(e));
  record_launches(1);
  return TREVS_OK;
}

}  // extern "C"
