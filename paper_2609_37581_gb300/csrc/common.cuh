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
  int tile_off;     // first score tile of this request
};

struct PreMeta {
  int B;
  int total_tiles;
  PreReq r[kMaxChunk];
};

struct InReq {
  int l_off, l;     // text rows of Q and of the row statistics
  int k1_off, k1;   // visual rows of K, V, hidden, p
  int k2_off, k2;   // kept rows of kept_local and of the compacted outputs
  int hs_off;       // first head-statistics block (Hq * ceil(l / 16) blocks)
  int ts_off;       // first token-score block (ceil(l / 16) * ceil(k1 / 64) blocks)
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
  uint32_t hist[256];
  uint32_t warp_gt[32];
  uint32_t warp_eq[32];
  uint32_t bcast[4];
};

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm volatile("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// K-th largest key (1 <= k <= n) of keys[0..n): returns the key value tau and `need`, the
// number of entries equal to tau that belong to the top k when ties go to the lower index.
// All threads of the block must call it; keys may live in shared or global memory.
__device__ inline void block_kth_largest(const uint32_t* keys, int n, int k, SelShared& s,
                                         uint32_t& tau, int& need) {
  uint32_t prefix = 0u, mask = 0u;
  int kk = k;
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int lane = tid & 31, warp = tid >> 5;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += nthr) s.hist[i] = 0u;
    __syncthreads();
    int i = tid;
    for (; i + 3 * nthr < n; i += 4 * nthr) {
      uint32_t v0 = keys[i], v1 = keys[i + nthr], v2 = keys[i + 2 * nthr], v3 = keys[i + 3 * nthr];
      if ((v0 & mask) == prefix) atomicAdd(&s.hist[(v0 >> shift) & 255u], 1u);
      if ((v1 & mask) == prefix) atomicAdd(&s.hist[(v1 >> shift) & 255u], 1u);
      if ((v2 & mask) == prefix) atomicAdd(&s.hist[(v2 >> shift) & 255u], 1u);
      if ((v3 & mask) == prefix) atomicAdd(&s.hist[(v3 >> shift) & 255u], 1u);
    }
    for (; i < n; i += nthr) {
      uint32_t v = keys[i];
      if ((v & mask) == prefix) atomicAdd(&s.hist[(v >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      // lane l owns bins [255 - 8l - 7, 255 - 8l], scanned from the top
      uint32_t c[8];
      uint32_t tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) { c[j] = s.hist[255 - 8 * lane - j]; tot += c[j]; }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      uint32_t excl = incl - tot;
      bool here = (excl < (uint32_t)kk) && (incl >= (uint32_t)kk);
      uint32_t ballot = __ballot_sync(0xffffffffu, here);
      int owner = __ffs(ballot) - 1;
      if (lane == owner) {
        uint32_t cum = excl;
        int j = 0;
        for (; j < 7; ++j) {
          if (cum + c[j] >= (uint32_t)kk) break;
          cum += c[j];
        }
        s.bcast[0] = 255u - 8u * lane - j;
        s.bcast[1] = (uint32_t)kk - cum;
      }
    }
    __syncthreads();
    uint32_t bin = s.bcast[0];
    kk = (int)s.bcast[1];
    prefix |= bin << shift;
    mask |= 255u << shift;
    __syncthreads();
  }
  tau = prefix;
  need = kk;
}

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
__device__ inline void block_compact_flags(const uint8_t* flags, int n, int* out, SelShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  int seg = (n + nwarps - 1) / nwarps;
  seg = (seg + 31) & ~31;
  const int beg = min(n, warp * seg), end = min(n, beg + seg);
  uint32_t cnt = 0;
  for (int base = beg; base < end; base += 32) {
    int i = base + lane;
    cnt += __popc(__ballot_sync(0xffffffffu, i < end && flags[i] != 0));
  }
  if (lane == 0) s.warp_gt[warp] = cnt;
  __syncthreads();
  uint32_t run = 0;
  for (int w = 0; w < warp; ++w) run += s.warp_gt[w];
  const uint32_t lt = lanemask_lt();
  for (int base = beg; base < end; base += 32) {
    int i = base + lane;
    bool f = i < end && flags[i] != 0;
    uint32_t b = __ballot_sync(0xffffffffu, f);
    if (f) out[run + __popc(b & lt)] = i;
    run += __popc(b);
  }
  __syncthreads();
}

// ------------------------------------------------------------------ launch helpers

// Raises a kernel's dynamic shared-memory limit once per (kernel, device) and size, so
// repeated launches (and launches under stream capture) make no attribute calls.
cudaError_t ensure_dynamic_smem_impl(const void* kernel, int bytes);

template <class Kernel>
inline cudaError_t ensure_dynamic_smem(Kernel kernel, int bytes) {
  return ensure_dynamic_smem_impl(reinterpret_cast<const void*>(kernel), bytes);
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

__device__ __forceinline__ float bf16_sq_sum8(uint4 v) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    float2 f = __bfloat1622float2(h[j]);
    s = fmaf(f.x, f.x, s);
    s = fmaf(f.y, f.y, s);
  }
  return s;
}

// Physical 16-byte chunk of logical chunk c in a 128-byte row r (XOR swizzle, conflict-free
// for ldmatrix and for row-wise reads).
__device__ __forceinline__ int swz(int r, int c) { return c ^ (r & 7); }

}  // namespace trevs
