// Vision-encoder saliency (Sec. 4.1, Eq. 2-3): s^v_i = (1/H) sum_h Softmax_i(q_h . k_{i,h} * scale)
// over the N patch keys of each request, scale = 1/sqrt(d_h) by default.
//
// One block per (request, head) reads the request's N keys of that head once (16-byte loads,
// d_h / 8 lanes per key row, eight rows in flight per thread), keeps the logits in shared
// memory, and writes the head's softmax row to the workspace. The last block of a request
// (a self-resetting ticket) averages the H rows in head order, so the result does not depend
// on which block finishes last. The work is a GEMV per head: K_v is read once from HBM.
#include "cls.cuh"

namespace trevs {

constexpr int kClsThreads = 256;
constexpr int kClsUnroll = 8;

template <int LPR>   // lanes per key row: d_h / 8
__global__ void __launch_bounds__(kClsThreads) cls_saliency_kernel(const __grid_constant__ ClsMeta meta,
                                                                  const ClsArgs a) {
  extern __shared__ float cls_logit[];
  __shared__ float red[kClsThreads / 32];
  __shared__ int s_last;
  const int H = meta.H;
  const ClsReq r = meta.r[blockIdx.x / H];
  const int h = blockIdx.x % H;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int sub = lane % LPR;          // 16-byte column of the row this lane reads
  const int g = tid / LPR;             // row slot of this lane group
  constexpr int kRowsPerPass = kClsThreads / LPR;
  const int n = r.n;

  float qf[8];
  {
    const uint4 qv = *reinterpret_cast<const uint4*>(a.q + r.b * a.q_req + h * a.q_head + sub * 8);
    const uint32_t w[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      qf[2 * j] = __uint_as_float(w[j] << 16);
      qf[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  }
  const __nv_bfloat16* kb = a.K + (long long)r.n_off * a.k_tok + (long long)h * a.k_head + sub * 8;
  float lmax = -INFINITY;
  for (int base = 0; base < n; base += kRowsPerPass * kClsUnroll) {   // the whole warp iterates
    uint4 kv[kClsUnroll];
#pragma unroll
    for (int u = 0; u < kClsUnroll; ++u) {
      const int i = base + u * kRowsPerPass + g;
      kv[u] = i < n ? __ldg(reinterpret_cast<const uint4*>(kb + (long long)i * a.k_tok)) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < kClsUnroll; ++u) {
      const uint32_t w[4] = {kv[u].x, kv[u].y, kv[u].z, kv[u].w};
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        dot = fmaf(qf[2 * j], __uint_as_float(w[j] << 16), dot);
        dot = fmaf(qf[2 * j + 1], __uint_as_float(w[j] & 0xFFFF0000u), dot);
      }
#pragma unroll
      for (int o = LPR >> 1; o; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      const int i = base + u * kRowsPerPass + g;
      if (i < n) {
        const float l = dot * a.scale;
        if (sub == 0) cls_logit[i] = l;
        lmax = fmaxf(lmax, l);
      }
    }
  }
  // softmax over the n patches (Eq. 2)
#pragma unroll
  for (int o = 16; o; o >>= 1) lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
  if (lane == 0) red[warp] = lmax;
  __syncthreads();
  float m = red[0];
  for (int w = 1; w < kClsThreads / 32; ++w) m = fmaxf(m, red[w]);
  __syncthreads();
  float sum = 0.f;
  for (int i = tid; i < n; i += kClsThreads) {
    const float e = expf(cls_logit[i] - m);
    cls_logit[i] = e;
    sum += e;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  if (lane == 0) red[warp] = sum;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < kClsThreads / 32; ++w) tot += red[w];
  float* arow = a.attn + (long long)h * a.attn_ld + r.n_off;
  for (int i = tid; i < n; i += kClsThreads) arow[i] = cls_logit[i] / tot;

  // Eq. 3 by the last head of the request, in head order
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t done = atomicAdd(a.cnt + r.b, 1u) + 1u;
    s_last = done == (uint32_t)H;
    if (s_last) a.cnt[r.b] = 0u;   // ready for the next launch
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int i = tid; i < n; i += kClsThreads) {
    float s = 0.f;
    for (int hh = 0; hh < H; ++hh) s += __ldcg(a.attn + (long long)hh * a.attn_ld + r.n_off + i);
    a.s_v[r.n_off + i] = s / (float)H;
  }
}

bool cls_head_dim_supported(int dh) { return dh == 32 || dh == 64 || dh == 128; }

cudaError_t launch_cls_saliency(const ClsMeta& meta, const ClsArgs& a, int dh, int max_n, cudaStream_t st) {
  if (meta.B == 0 || meta.H == 0) return cudaSuccess;
  const dim3 grid((unsigned)(meta.B * meta.H));
  const size_t smem = (size_t)max_n * sizeof(float);
  if (dh == 32) return launch_kernel(cls_saliency_kernel<4>, grid, dim3(kClsThreads), smem, st, false, meta, a);
  if (dh == 64) return launch_kernel(cls_saliency_kernel<8>, grid, dim3(kClsThreads), smem, st, false, meta, a);
  return launch_kernel(cls_saliency_kernel<16>, grid, dim3(kClsThreads), smem, st, false, meta, a);
}

}  // namespace trevs
