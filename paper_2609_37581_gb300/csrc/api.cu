// Host side of the C ABI declared in include/trevs.h: argument validation, workspace
// layout, per-launch request metadata and the launch sequence of each entry point.
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include "cls.cuh"
#include "fps.cuh"
#include "in_llm.cuh"
#include "pre_llm.cuh"
#include "trevs.h"

namespace trevs {
cudaError_t launch_pre_score(const PreMeta&, const PreArgs&, int max_m, long long z_rows, cudaStream_t, bool pdl);
size_t pre_score_part_bytes(int max_m);
cudaError_t launch_pre_finish(const PreMeta&, const PreArgs&, int max_m, int max_n, bool scored, cudaStream_t,
                              bool pdl);
cudaError_t launch_pre_saliency(const PreMeta&, const PreArgs&, int max_n, bool saliency, cudaStream_t);
cudaError_t launch_stream_probe(const void* Z, long long z_stride, long long rows, int d, int ctas, uint32_t* err,
                                cudaStream_t st);
cudaError_t launch_gather(const GatherMeta&, cudaStream_t, bool pdl);
cudaError_t launch_fps(const FpsMeta&, const FpsArgs&, cudaStream_t, bool pdl);
cudaError_t launch_fps_gram(const FpsMeta&, const FpsArgs&, int tiles, cudaStream_t);
cudaError_t launch_cls_saliency(const ClsMeta&, const ClsArgs&, int dh, int max_n, cudaStream_t);
cudaError_t launch_in_head_stats(const InMeta&, const InArgs&, int max_k1, cudaStream_t);
cudaError_t launch_in_token_score(const InMeta&, const InArgs&, int max_k1, cudaStream_t);
bool in_small_fits(int Hq, int max_l, int max_k1);
cudaError_t launch_in_small(const InMeta&, const InArgs&, int max_k1, cudaStream_t);
}  // namespace trevs

namespace trevs {

cudaError_t ensure_dynamic_smem_impl(const void* kernel, int bytes) {
  // Every kernel of the library prefers the largest shared-memory carveout, so that an SM
  // never has to drain and re-split L1 / shared memory between two of its grids (the scoring
  // grid needs the largest split and follows the pre-pass closely). The default dynamic limit
  // is 48 KB minus the kernel's static shared memory: opt in to what a launch asks for.
  struct Entry {
    const void* kernel;
    int device;
    int bytes;
  };
  static std::mutex mu;
  static std::vector<Entry> granted;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  Entry* x = nullptr;
  for (Entry& g : granted)
    if (g.kernel == kernel && g.device == dev) x = &g;
  if (!x) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    granted.push_back(Entry{kernel, dev, 0});
    x = &granted.back();
  }
  if (bytes > x->bytes) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    x->bytes = bytes;
  }
  return cudaSuccess;
}

// A second stream with fork / join events, created once per (host thread, device), so that
// trevs_prune_varlen can run its two independent stages as parallel branches (also under
// stream capture). Kept for the life of the thread.
struct AuxStream {
  int device = -1;
  cudaStream_t stream = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};

cudaError_t aux_stream(AuxStream*& out) {
  static thread_local AuxStream aux[8];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  for (AuxStream& x : aux)
    if (x.device == dev) {
      out = &x;
      return cudaSuccess;
    }
  for (AuxStream& x : aux)
    if (x.device < 0) {
      // the stage-1 tail runs here: at the highest priority, so that its blocks take the SMs
      // the scoring grid frees ahead of the stage-2 blocks still waiting on the caller's stream
      int least = 0, greatest = 0;
      e = cudaDeviceGetStreamPriorityRange(&least, &greatest);
      if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&x.stream, cudaStreamNonBlocking, greatest);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&x.fork, cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&x.join, cudaEventDisableTiming);
      if (e != cudaSuccess) return e;
      x.device = dev;
      out = &x;
      return cudaSuccess;
    }
  return cudaErrorInvalidDevice;
}

}  // namespace trevs

using namespace trevs;

namespace {

thread_local char g_err[512] = "";
thread_local int g_launches = 0;     // kernels enqueued by the current call
thread_local int g_fail_in = 0;      // launch attempts until the one the test hook fails (0: none)

// Counts one enqueued kernel or memset of the current call.
inline cudaError_t counted(cudaError_t e) {
  if (e == cudaSuccess) ++g_launches;
  return e;
}

trevs_status fail(trevs_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

trevs_status cuda_fail(cudaError_t e, const char* where) {
  return fail(TREVS_ERR_CUDA, "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
}
// cudaErrorLaunchFailure never comes back from an enqueue: a launch that reports it was the one
// the test hook failed (launch_fault_injected), which made no launch.

#define TREVS_TRY_CUDA(expr, where)            \
  do {                                         \
    cudaError_t e_ = (expr);                   \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

#define TREVS_CHECK(cond, ...)                                  \
  do {                                                          \
    if (!(cond)) return fail(TREVS_ERR_INVALID_ARGUMENT, __VA_ARGS__); \
  } while (0)

inline bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }
inline size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

// ---------------------------------------------------------------- workspace layouts

// Every layout starts with a 256-byte header whose first word is the device status word.
constexpr size_t kStatusBytes = 256;

struct PreWs {
  size_t counters, sal, t_rinv, part, s_t, s_fused, keys, flags;
  size_t fps_zero, fps_prow, fps_rinv, fps_maxcos, fps_ub, fps_stamp, fps_picks, fps_pooln, fps_pool, fps_gram, end;
};

// Scratch keys / flags hold sum n entries plus 16-byte alignment padding per request;
// t_rinv holds 1 / ||t_j|| of the text rows; part the partial sums of the scoring tiles
// that two or more scoring CTAs share (up to max_m text rows, or up to the pivots of the
// farthest-point contraction, min(max_k1, TREVS_MAX_TEXT_TOKENS), which reuses it). The
// fps_* regions serve farthest point sampling (Sec. 3.1) when the call asks for it: a
// 256-byte zero block, copies of the pivot rows (d columns), 1 / ||z|| of the pivots and the
// draws (all indexed like kept_idx), and the largest pivot cosine, bound and stamp of every row.
// Rows of the pool-cosine matrix a request with k1 kept tokens may need for its diversity
// draws (K_d <= K1): the automatic pool, at most kFpsMaxPoolBig, rounded up to whole tiles.
inline int fps_gram_ld(int k1) {
  if (k1 <= 0) return 0;
  const int w = fps_auto_pool(k1);
  return ((w < kFpsMaxPoolBig ? w : kFpsMaxPoolBig) + kFpsGramTile - 1) / kFpsGramTile * kFpsGramTile;
}

PreWs pre_ws(long long total_n, long long total_m, int max_m, long long total_k1 = 0, int max_k1 = 0,
             int d = 0, long long fps_pool = 0, long long fps_gram = 0) {
  PreWs w;
  const size_t padded = (size_t)total_n + 4 * (size_t)kMaxChunk + 4;
  const int max_kr = max_k1 < TREVS_MAX_TEXT_TOKENS ? max_k1 : TREVS_MAX_TEXT_TOKENS;
  const int part_rows = max_m > max_kr ? max_m : max_kr;
  const size_t k1 = (size_t)(total_k1 > 0 ? total_k1 : 0), fn = total_k1 > 0 ? (size_t)total_n : 0;
  size_t o = kStatusBytes;
  w.counters = o; o = al256(o + 4 * (size_t)kMaxChunk);
  w.sal = o;      o = al256(o + 16 * (size_t)kMaxChunk);
  w.t_rinv = o;   o = al256(o + 4 * (size_t)(total_m > 0 ? total_m : 0));
  w.part = o;     o = al256(o + (total_n > 0 ? pre_score_part_bytes(part_rows > 0 ? part_rows : 1) : 0));
  w.s_t = o;      o = al256(o + 4 * (size_t)total_n);
  w.s_fused = o;  o = al256(o + 4 * (size_t)total_n);
  w.keys = o;     o = al256(o + 4 * padded);
  w.flags = o;    o = al256(o + padded);
  w.fps_zero = o;   o = al256(o + (k1 > 0 ? 256 : 0));
  w.fps_prow = o;   o = al256(o + 2 * k1 * (size_t)(d > 0 ? d : 0));
  w.fps_rinv = o;   o = al256(o + 4 * k1);
  w.fps_picks = o;  o = al256(o + 4 * k1);
  w.fps_maxcos = o; o = al256(o + 4 * fn);
  w.fps_ub = o;     o = al256(o + 4 * fn);
  w.fps_stamp = o;  o = al256(o + 4 * fn);
  // pools above kFpsMaxPool: pool sizes, pool rows and their dot products (sum of ld^2)
  w.fps_pooln = o;  o = al256(o + (fps_gram > 0 ? 4 * (size_t)kMaxChunk : 0));
  w.fps_pool = o;   o = al256(o + 4 * (size_t)(fps_pool > 0 ? fps_pool : 0));
  w.fps_gram = o;   o = al256(o + 4 * (size_t)(fps_gram > 0 ? fps_gram : 0));
  w.end = o;
  return w;
}

struct InWs {
  size_t cnt_hs, cnt_ts, attn, row_var, rstat, u, p, keys, flags, end;
};

// total_lk1 = sum over requests of l * k1 (attention probabilities per head).
InWs in_ws(long long total_l, long long total_k1, long long total_lk1, int Hq, int B) {
  InWs w;
  size_t o = kStatusBytes;
  w.cnt_hs = o;    o = al256(o + 4 * (size_t)kMaxChunk);
  w.cnt_ts = o;    o = al256(o + 4 * (size_t)kMaxChunk);
  w.attn = o;      o = al256(o + 4 * (size_t)Hq * (size_t)total_lk1);
  w.row_var = o;   o = al256(o + 4 * (size_t)Hq * (size_t)total_l);
  w.rstat = o;     o = al256(o + 8 * (size_t)Hq * (size_t)total_l);
  w.u = o;         o = al256(o + 4 * (size_t)Hq * (size_t)(B > 0 ? B : 1));
  w.p = o;         o = al256(o + 4 * (size_t)total_k1);
  const size_t padded = (size_t)total_k1 + 4 * (size_t)kMaxChunk + 4;   // per-request 16-byte alignment
  w.keys = o;      o = al256(o + 4 * padded);
  w.flags = o;     o = al256(o + padded);
  w.end = o;
  return w;
}

// Farthest point sampling (Sec. 3.1), from byte offset `o` on: 1 / ||z_s|| of the pivots
// (piv_space entries, indexed like the pivots), the partial sums of the pivot contraction
// (up to max_kr pivots), the largest cosine of every row to its pivots, the bounds and
// stamps of the draw, and flag / key scratch for the rows.
// `zero` is 256 bytes that nothing writes: the row-0 pivot of a draw without pivots; `prow`
// holds copies of the pivot rows (d columns each), which the contraction reads as text rows.
struct FpsWs {
  size_t zero, prow, t_rinv, part, maxcos, ub, stamp, flags, keys, end;
};

FpsWs fps_ws(size_t o, long long total_n, long long piv_space, int max_kr, int d) {
  FpsWs w;
  const size_t padded = (size_t)total_n + 4 * (size_t)kMaxChunk + 4;
  if (piv_space < 1) piv_space = 1;
  if (max_kr < 1) max_kr = 1;
  o = al256(o);
  w.zero = o;    o = al256(o + 256);
  w.prow = o;    o = al256(o + 2 * (size_t)piv_space * (size_t)(d > 0 ? d : 0));
  w.t_rinv = o;  o = al256(o + 4 * (size_t)(piv_space > 0 ? piv_space : 0));
  w.part = o;    o = al256(o + (total_n > 0 && max_kr > 0
                                      ? pre_score_part_bytes(max_kr < TREVS_MAX_TEXT_TOKENS ? max_kr : TREVS_MAX_TEXT_TOKENS)
                                      : 0));
  w.maxcos = o;  o = al256(o + 4 * (size_t)total_n);
  w.ub = o;      o = al256(o + 4 * (size_t)total_n);
  w.stamp = o;   o = al256(o + 4 * (size_t)total_n);
  w.flags = o;   o = al256(o + padded);
  w.keys = o;    o = al256(o + 4 * padded);
  w.end = o;
  return w;
}

// [CLS] saliency (Eq. 2-3): per-request tickets, then the H softmax rows of every patch.
struct ClsWs {
  size_t cnt, attn, end;
};

ClsWs cls_ws(long long total_n, int H) {
  ClsWs w;
  size_t o = kStatusBytes;
  w.cnt = o;  o = al256(o + 4 * (size_t)kMaxChunk);
  w.attn = o; o = al256(o + 4 * (size_t)(H > 0 ? H : 0) * (size_t)(total_n > 0 ? total_n : 0));
  w.end = o;
  return w;
}

trevs_status check_ws(void* ws, size_t bytes, size_t need) {
  if (need == 0) return TREVS_OK;
  if (ws == nullptr) return fail(TREVS_ERR_WORKSPACE, "workspace is NULL (need %zu bytes)", need);
  if (((uintptr_t)ws & 255u) != 0) return fail(TREVS_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (bytes < need) return fail(TREVS_ERR_WORKSPACE, "workspace has %zu bytes, need %zu", bytes, need);
  return TREVS_OK;
}

int textual_count(int k1, float ratio) {
  int kt = (int)std::floor((double)ratio * (double)k1 + 0.5);
  return kt < 0 ? 0 : (kt > k1 ? k1 : kt);
}

// ---------------------------------------------------------------- stage-1 batch

struct PreTotals {
  long long n = 0, m = 0, k1 = 0;
  int max_n = 0, max_m = 0, max_k1 = 0;
  long long fps_pool = 0, fps_gram = 0;   // room for pools above kFpsMaxPool (fps_gram_ld)
};

trevs_status validate_pre_batch(const trevs_pre_batch* bt, PreTotals& t) {
  TREVS_CHECK(bt != nullptr, "pre batch is NULL");
  TREVS_CHECK(bt->B >= 0, "B = %d < 0", bt->B);
  if (bt->B == 0) return TREVS_OK;
  TREVS_CHECK(bt->reqs != nullptr, "reqs is NULL");
  TREVS_CHECK(bt->d >= 8 && bt->d % 8 == 0, "d = %d must be a positive multiple of 8", bt->d);
  for (int b = 0; b < bt->B; ++b) {
    const trevs_pre_request& r = bt->reqs[b];
    TREVS_CHECK(r.n >= 0, "request %d: n = %d < 0", b, r.n);
    TREVS_CHECK(r.k1 >= 0 && r.k1 <= r.n, "request %d: k1 = %d outside [0, n = %d]", b, r.k1, r.n);
    TREVS_CHECK(std::isfinite(r.ratio) && r.ratio >= 0.f && r.ratio <= 1.f,
                "request %d: textual ratio %g outside [0, 1]", b, (double)r.ratio);
    if (r.n > 0) {
      TREVS_CHECK(r.m >= 1, "request %d: m = %d, needs at least one text token", b, r.m);
      if (r.m > TREVS_MAX_TEXT_TOKENS)
        return fail(TREVS_ERR_UNSUPPORTED, "request %d: m = %d > %d text tokens", b, r.m, TREVS_MAX_TEXT_TOKENS);
    } else {
      TREVS_CHECK(r.m >= 0, "request %d: m = %d < 0", b, r.m);
    }
    t.n += r.n; t.m += r.m; t.k1 += r.k1;
    const long long gl = fps_gram_ld(r.k1);
    t.fps_pool += gl;
    t.fps_gram += gl * gl;
    t.max_n = r.n > t.max_n ? r.n : t.max_n;
    t.max_k1 = r.k1 > t.max_k1 ? r.k1 : t.max_k1;
    if (r.n > 0) t.max_m = r.m > t.max_m ? r.m : t.max_m;   // requests without visual rows score nothing
  }
  TREVS_CHECK(t.n < (1ll << 31) && t.m < (1ll << 31) && t.k1 < (1ll << 31), "batch too large for int32 offsets");
  if (t.n > 0) {
    TREVS_CHECK(bt->Z && bt->T && bt->s_v, "Z, T and s_v must be non-NULL");
    TREVS_CHECK(aligned16(bt->Z) && aligned16(bt->T), "Z and T must be 16-byte aligned");
    TREVS_CHECK(bt->z_row_stride >= bt->d && bt->z_row_stride % 8 == 0, "z_row_stride must be >= d and a multiple of 8");
    TREVS_CHECK(bt->t_row_stride >= bt->d && bt->t_row_stride % 8 == 0, "t_row_stride must be >= d and a multiple of 8");
  }
  if (t.k1 > 0) {
    TREVS_CHECK(bt->kept_idx != nullptr, "kept_idx is NULL");
    if (bt->Z_out) {
      TREVS_CHECK(aligned16(bt->Z_out), "Z_out must be 16-byte aligned");
      TREVS_CHECK(bt->z_out_row_stride >= bt->d && bt->z_out_row_stride % 8 == 0,
                  "z_out_row_stride must be >= d and a multiple of 8");
    }
  }
  return TREVS_OK;
}

trevs_status validate_params(const trevs_pre_params* p) {
  TREVS_CHECK(p->select_mode == TREVS_SELECT_RATIO || p->select_mode == TREVS_SELECT_FUSED,
              "select_mode %d unknown", p->select_mode);
  TREVS_CHECK(std::isfinite(p->tau_v) && p->tau_v > 0.f && std::isfinite(p->tau_t) && p->tau_t > 0.f,
              "temperatures must be positive");
  TREVS_CHECK(std::isfinite(p->lambda) && std::isfinite(p->eps) && p->eps >= 0.f, "lambda / eps invalid");
  TREVS_CHECK(std::isfinite(p->diversity) && p->diversity >= 0.f && p->diversity <= 1.f,
              "diversity share %g outside [0, 1]", (double)p->diversity);
  return TREVS_OK;
}

// K_d = floor(rho * K1 + 1/2): the tokens farthest point sampling adds to the K1 - K_d
// pivots of the selection rule (Sec. 3.1).
int diversity_count(int k1, float rho) {
  int kd = (int)std::floor((double)rho * (double)k1 + 0.5);
  return kd < 0 ? 0 : (kd > k1 ? k1 : kd);
}

// The distances of farthest point sampling take any number of pivots (in passes of at most
// TREVS_MAX_TEXT_TOKENS columns of the contraction); nothing to check beyond the batch.
trevs_status validate_diversity(const trevs_pre_batch*, const trevs_pre_params&) { return TREVS_OK; }

// The largest cosine of every row of the requests of `dm` to that request's pivot rows (the
// "text" rows of `da`, their norms already computed): the scoring contraction over at most
// TREVS_MAX_TEXT_TOKENS pivot columns per pass (its TMEM accumulator), each pass after the
// first keeping the max of what s_t holds (Sec. 3.1 distances are minima over the pivots).
trevs_status run_pivot_contraction(const PreMeta& dm, const PreArgs& da, long long z_rows, int max_n, cudaStream_t st) {
  static thread_local PreMeta pm;
  int max_kr = 0;
  for (int i = 0; i < dm.B; ++i) max_kr = dm.r[i].m > max_kr ? dm.r[i].m : max_kr;
  for (int p0 = 0; p0 < max_kr; p0 += TREVS_MAX_TEXT_TOKENS) {
    pm.B = 0;
    int tiles = 0, mm = 0;
    for (int i = 0; i < dm.B; ++i) {
      const PreReq& r = dm.r[i];
      if (r.n <= 0 || r.m <= p0) continue;   // no pivot columns left in this pass
      PreReq q = r;
      q.m_off = r.m_off + p0;
      q.m = r.m - p0 < TREVS_MAX_TEXT_TOKENS ? r.m - p0 : TREVS_MAX_TEXT_TOKENS;
      q.tile_off = tiles;
      tiles += (r.n + kScoreTileRows - 1) / kScoreTileRows;
      pm.r[pm.B++] = q;
      mm = q.m > mm ? q.m : mm;
    }
    pm.total_tiles = tiles;
    PreArgs pa = da;
    pa.seed_merge = p0 > 0 ? 1 : 0;
    TREVS_TRY_CUDA(counted(launch_pre_score(pm, pa, mm, z_rows, st, true)), "pivot contraction launch");
    TREVS_TRY_CUDA(counted(launch_pre_finish(pm, pa, mm, max_n, true, st, true)), "pivot fixup launch");
  }
  return TREVS_OK;
}

// Runs stage 1 for requests [b0, b1) of the batch; offsets are relative to the chunk. When
// `gm_out` is given the gather job is left to the caller (to share one launch with stage 2).
// after_score (may be null) is recorded on `st` right after the scoring grid is enqueued.
trevs_status run_pre_chunk(const trevs_pre_batch* bt, const trevs_pre_params& prm, int b0, int b1,
                           long long n_base, long long m_base, long long k1_base, uint8_t* ws,
                           const PreWs& L, cudaStream_t st, GatherMeta* gm_out, cudaEvent_t after_score = nullptr,
                           cudaEvent_t before_score = nullptr, cudaStream_t tail = nullptr, int reserve = 0,
                           bool* forked = nullptr) {
  static thread_local PreMeta meta;
  static thread_local GatherMeta gm;
  static thread_local int kd_of[kMaxChunk];
  meta.B = b1 - b0;
  int tiles = 0, max_n = 0, max_m = 0;
  bool draws = false;
  long long no = 0, mo = 0, ko = 0;
  for (int b = b0; b < b1; ++b) {
    const trevs_pre_request& q = bt->reqs[b];
    PreReq& r = meta.r[b - b0];
    // with a diversity share the rule picks the K_r = K1 - K_d pivots (Sec. 3.1)
    const int kd = prm.diversity > 0.f ? diversity_count(q.k1, prm.diversity) : 0;
    kd_of[b - b0] = kd;
    draws = draws || kd > 0;
    r.n_off = (int)no; r.n = q.n; r.m_off = (int)mo; r.m = q.m;
    r.k1_off = (int)ko; r.k1 = q.k1 - kd; r.kt = textual_count(q.k1 - kd, q.ratio);
    r.tile_off = tiles;
    tiles += (q.n + kScoreTileRows - 1) / kScoreTileRows;
    no += q.n; mo += q.m; ko += q.k1;
    max_n = q.n > max_n ? q.n : max_n;
    if (q.n > 0) max_m = q.m > max_m ? q.m : max_m;
  }
  meta.total_tiles = tiles;
  PreArgs a;
  memset(&a, 0, sizeof(a));
  a.Z = reinterpret_cast<const __nv_bfloat16*>(bt->Z) + n_base * bt->z_row_stride;
  a.z_stride = bt->z_row_stride;
  a.T = reinterpret_cast<const __nv_bfloat16*>(bt->T) + m_base * bt->t_row_stride;
  a.t_stride = bt->t_row_stride;
  a.s_v = bt->s_v + n_base;
  a.s_t = (bt->s_t ? bt->s_t : reinterpret_cast<float*>(ws + L.s_t)) + n_base;
  a.s_fused = (bt->s_fused ? bt->s_fused : reinterpret_cast<float*>(ws + L.s_fused)) + n_base;
  a.kept = bt->kept_idx + k1_base;
  a.flags = ws + L.flags;
  a.keys = reinterpret_cast<uint32_t*>(ws + L.keys);
  a.counters = reinterpret_cast<uint32_t*>(ws + L.counters);
  a.sal = reinterpret_cast<int4*>(ws + L.sal);
  a.sal_ready = 1;
  a.t_rinv = reinterpret_cast<float*>(ws + L.t_rinv);   // chunks run one after the other: rows from 0
  a.total_m = mo;
  a.part = reinterpret_cast<float*>(ws + L.part);
  a.err = reinterpret_cast<uint32_t*>(ws);
  a.d = bt->d;
  a.mode = prm.select_mode == TREVS_SELECT_FUSED ? kModeFused : kModeRatio;
  a.tau_v = prm.tau_v; a.tau_t = prm.tau_t; a.lambda = prm.lambda; a.eps = prm.eps;
  a.action = kActSelect;
  a.score_reserve = reserve;
  a.big_sel = 1;
  TREVS_TRY_CUDA(counted(launch_pre_saliency(meta, a, max_n, true, st)), "pre-pass launch");
  if (before_score) TREVS_TRY_CUDA(cudaEventRecord(before_score, st), "event before scoring");
  TREVS_TRY_CUDA(counted(launch_pre_score(meta, a, max_m, no, st, true)), "pre_score launch");
  if (after_score) TREVS_TRY_CUDA(cudaEventRecord(after_score, st), "event after scoring");
  // the rest of stage 1 goes on `tail` (after the scoring grid completes) when given
  if (tail) {
    TREVS_TRY_CUDA(cudaStreamWaitEvent(tail, after_score, 0), "tail after scoring");
    if (forked) *forked = true;
  }
  const cudaStream_t ts = tail ? tail : st;
  TREVS_TRY_CUDA(counted(launch_pre_finish(meta, a, max_m, max_n, true, ts, !tail)), "finishing launch");
  if (draws) {
    // Farthest point sampling of the K_d diversity tokens (Sec. 3.1) behind the pivots: the
    // scoring contraction again, over the requests that draw, with their pivots (kept_idx)
    // as the text rows; then one block per request draws and writes S_r and S_d together.
    static thread_local PreMeta dm;
    static thread_local FpsMeta fm;
    dm.B = 0;
    fm.B = 0;
    int dtiles = 0, max_kr = 0;
    // pools above kFpsMaxPool keep their cosines in the workspace: then every request of the
    // launch takes the three-grid form (pool, pool cosines, draws)
    bool big = false;
    for (int i = 0; i < meta.B; ++i) big = big || fps_auto_pool(kd_of[i]) > kFpsMaxPool;
    int pool_off = 0, gt_off = 0;
    long long gram_off = 0;
    for (int i = 0; i < meta.B; ++i) {
      const int kd = kd_of[i];
      if (kd <= 0) continue;
      const PreReq& r = meta.r[i];
      const int lead = r.k1 == 0 ? 1 : 0;   // no pivots: row 0 is the first draw and the pivot
      const int kr = r.k1 + lead;
      if (lead)
        TREVS_TRY_CUDA(counted(cudaMemsetAsync(a.kept + r.k1_off, 0, sizeof(int32_t), ts)), "row-0 pivot");
      dm.r[dm.B++] = PreReq{r.n_off, r.n, r.k1_off, kr, 0, 0, 0, dtiles};
      dtiles += (r.n + kScoreTileRows - 1) / kScoreTileRows;
      max_kr = kr > max_kr ? kr : max_kr;
      const int gl = big ? fps_gram_ld(kd) : 0;
      fm.r[fm.B++] = FpsReq{r.n_off, r.n, r.k1_off, kr, kd, lead, r.k1_off, r.k1_off, pool_off, gl, gt_off, gram_off};
      pool_off += gl;
      gt_off += (gl / kFpsGramTile) * (gl / kFpsGramTile);
      gram_off += (long long)gl * gl;
    }
    dm.total_tiles = dtiles;
    // copies of every request's kept slots (the pivots lead each request's K1 slots)
    static thread_local GatherMeta pg;
    uint16_t* prow = reinterpret_cast<uint16_t*>(ws + L.fps_prow);
    pg.njobs = 1;
    GatherTable& pt = pg.t[0];
    pt.B = meta.B;
    for (int i = 0; i < meta.B; ++i) {
      pt.dst_off[i] = meta.r[i].k1_off; pt.src_off[i] = meta.r[i].n_off; pt.src_rows[i] = meta.r[i].n;
    }
    pt.dst_off[meta.B] = (int)ko;
    GatherJob& pj = pg.job[0];
    pj.src = reinterpret_cast<const uint8_t*>(a.Z); pj.dst = reinterpret_cast<uint8_t*>(prow);
    pj.src_tok = a.z_stride * 2; pj.dst_tok = (long long)a.d * 2; pj.src_head = 0; pj.dst_head = 0;
    pj.heads = 1; pj.row_bytes = a.d * 2; pj.idx = a.kept; pj.rows = (int)ko; pj.tab = 0;
    TREVS_TRY_CUDA(counted(launch_gather(pg, ts, true)), "pivot rows launch");
    PreArgs da = a;
    da.T = reinterpret_cast<const __nv_bfloat16*>(prow);
    da.t_stride = a.d;
    da.s_t = reinterpret_cast<float*>(ws + L.fps_maxcos);
    da.t_rinv = reinterpret_cast<float*>(ws + L.fps_rinv);
    da.total_m = ko;
    da.action = kActFpsSeed;
    TREVS_TRY_CUDA(counted(launch_pre_saliency(dm, da, max_n, false, ts)), "pivot norms launch");
    const trevs_status cs = run_pivot_contraction(dm, da, no, max_n, ts);
    if (cs != TREVS_OK) return cs;
    FpsArgs f;
    memset(&f, 0, sizeof(f));
    f.Z = a.Z; f.z_stride = a.z_stride; f.d = a.d;
    f.piv = a.kept; f.maxcos = da.s_t;
    f.ub = reinterpret_cast<float*>(ws + L.fps_ub); f.stamp = reinterpret_cast<int*>(ws + L.fps_stamp);
    f.flags = a.flags; f.keys = a.keys;
    f.picks = reinterpret_cast<int*>(ws + L.fps_picks); f.pick_dist = nullptr;
    f.kept = a.kept; f.pool = 0; f.err = a.err;
    if (!big) {
      TREVS_TRY_CUDA(counted(launch_fps(fm, f, ts, true)), "farthest point sampling launch");
    } else {
      f.pool_n = reinterpret_cast<int*>(ws + L.fps_pooln);
      f.pool_idx = reinterpret_cast<int*>(ws + L.fps_pool);
      f.gram = reinterpret_cast<float*>(ws + L.fps_gram);
      f.phase = 1;
      TREVS_TRY_CUDA(counted(launch_fps(fm, f, ts, true)), "diversity pool launch");
      TREVS_TRY_CUDA(counted(launch_fps_gram(fm, f, gt_off, ts)), "pool cosines launch");
      f.phase = 2;
      TREVS_TRY_CUDA(counted(launch_fps(fm, f, ts, true)), "farthest point sampling launch");
    }
  }
  GatherMeta& g = gm_out ? *gm_out : gm;
  g.njobs = 0;
  if (bt->Z_out && ko > 0) {
    g.njobs = 1;
    GatherTable& tb = g.t[0];
    tb.B = meta.B;
    for (int i = 0; i < meta.B; ++i) {
      tb.dst_off[i] = meta.r[i].k1_off;
      tb.src_off[i] = meta.r[i].n_off;
      tb.src_rows[i] = meta.r[i].n;
    }
    tb.dst_off[meta.B] = (int)ko;
    GatherJob& j = g.job[0];
    j.src = reinterpret_cast<const uint8_t*>(a.Z);
    j.dst = reinterpret_cast<uint8_t*>(bt->Z_out + k1_base * bt->z_out_row_stride);
    j.src_tok = bt->z_row_stride * 2; j.dst_tok = bt->z_out_row_stride * 2;
    j.src_head = 0; j.dst_head = 0; j.heads = 1; j.row_bytes = bt->d * 2;
    j.idx = a.kept; j.rows = (int)ko; j.tab = 0;
    if (!gm_out) TREVS_TRY_CUDA(counted(launch_gather(g, ts, true)), "gather launch");
  }
  return TREVS_OK;
}

trevs_status run_pre_batch(const trevs_pre_batch* bt, const trevs_pre_params& prm, uint8_t* ws,
                           const PreWs& L, cudaStream_t st) {
  long long n_base = 0, m_base = 0, k1_base = 0;
  for (int b0 = 0; b0 < bt->B; b0 += kMaxChunk) {
    const int b1 = b0 + kMaxChunk < bt->B ? b0 + kMaxChunk : bt->B;
    trevs_status s = run_pre_chunk(bt, prm, b0, b1, n_base, m_base, k1_base, ws, L, st, nullptr);
    if (s != TREVS_OK) return s;
    for (int b = b0; b < b1; ++b) {
      n_base += bt->reqs[b].n; m_base += bt->reqs[b].m; k1_base += bt->reqs[b].k1;
    }
  }
  return TREVS_OK;
}

// ---------------------------------------------------------------- stage-2 batch

struct InTotals {
  long long l = 0, k1 = 0, k2 = 0, lk1 = 0;
  int max_k1 = 0;
};

trevs_status validate_in_common(int Hq, int Hkv, int d_h, int n_keep) {
  TREVS_CHECK(Hq >= 1 && Hkv >= 1 && Hq % Hkv == 0, "Hq = %d, Hkv = %d: need Hq %% Hkv == 0", Hq, Hkv);
  if (Hq > TREVS_MAX_HEADS) return fail(TREVS_ERR_UNSUPPORTED, "Hq = %d > %d", Hq, TREVS_MAX_HEADS);
  if (d_h != TREVS_HEAD_DIM) return fail(TREVS_ERR_UNSUPPORTED, "d_h = %d, only %d supported", d_h, TREVS_HEAD_DIM);
  TREVS_CHECK(n_keep >= 1 && n_keep <= Hq, "n_keep_heads = %d outside [1, Hq = %d]", n_keep, Hq);
  return TREVS_OK;
}

trevs_status validate_qk(const void* Q, long long qhs, long long qts, const void* K, long long khs,
                         long long kts) {
  TREVS_CHECK(Q && K, "Q and K must be non-NULL");
  TREVS_CHECK(aligned16(Q) && aligned16(K), "Q and K must be 16-byte aligned");
  TREVS_CHECK(qhs % 8 == 0 && qts % 8 == 0 && khs % 8 == 0 && kts % 8 == 0 && qhs >= 0 && qts >= 0 &&
                  khs >= 0 && kts >= 0,
              "Q/K strides must be non-negative multiples of 8");
  return TREVS_OK;
}

trevs_status validate_in_batch(const trevs_in_batch* bt, InTotals& t) {
  TREVS_CHECK(bt != nullptr, "in batch is NULL");
  TREVS_CHECK(bt->B >= 0, "B = %d < 0", bt->B);
  if (bt->B == 0) return TREVS_OK;
  TREVS_CHECK(bt->reqs != nullptr, "reqs is NULL");
  trevs_status s = validate_in_common(bt->Hq, bt->Hkv, bt->d_h, bt->n_keep_heads);
  if (s != TREVS_OK) return s;
  for (int b = 0; b < bt->B; ++b) {
    const trevs_in_request& r = bt->reqs[b];
    TREVS_CHECK(r.k1 >= 1, "request %d: k1 = %d < 1", b, r.k1);
    if (r.k1 > TREVS_MAX_STAGE2_TOKENS)
      return fail(TREVS_ERR_UNSUPPORTED, "request %d: k1 = %d > %d", b, r.k1, TREVS_MAX_STAGE2_TOKENS);
    TREVS_CHECK(r.l >= 1, "request %d: l = %d < 1", b, r.l);
    TREVS_CHECK(r.k2 >= 0 && r.k2 <= r.k1, "request %d: k2 = %d outside [0, k1 = %d]", b, r.k2, r.k1);
    t.l += r.l; t.k1 += r.k1; t.k2 += r.k2; t.lk1 += (long long)r.l * r.k1;
    t.max_k1 = r.k1 > t.max_k1 ? r.k1 : t.max_k1;
  }
  TREVS_CHECK(t.l < (1ll << 31) && t.k1 < (1ll << 31), "batch too large for int32 offsets");
  s = validate_qk(bt->Q, bt->q_head_stride, bt->q_tok_stride, bt->K, bt->kv_head_stride, bt->kv_tok_stride);
  if (s != TREVS_OK) return s;
  if (t.k2 > 0) TREVS_CHECK(bt->kept_local != nullptr, "kept_local is NULL");
  TREVS_CHECK((bt->hidden == nullptr) == (bt->hidden_out == nullptr), "hidden and hidden_out: both or neither");
  TREVS_CHECK((bt->V == nullptr) == (bt->V_out == nullptr), "V and V_out: both or neither");
  if (bt->hidden) {
    TREVS_CHECK(bt->d_model >= 8 && bt->d_model % 8 == 0, "d_model = %d must be a positive multiple of 8", bt->d_model);
    TREVS_CHECK(aligned16(bt->hidden) && aligned16(bt->hidden_out), "hidden tensors must be 16-byte aligned");
    TREVS_CHECK(bt->hidden_row_stride >= bt->d_model && bt->hidden_row_stride % 8 == 0 &&
                    bt->hidden_out_row_stride >= bt->d_model && bt->hidden_out_row_stride % 8 == 0,
                "hidden strides must be >= d_model and multiples of 8");
  }
  if (bt->lse_other)
    TREVS_CHECK(bt->lse_head_stride >= 0 && bt->lse_row_stride >= 0 && ((uintptr_t)bt->lse_other & 3u) == 0,
                "lse_other must be 4-byte aligned with non-negative strides");
  if (bt->K_out || bt->V_out) {
    TREVS_CHECK(bt->K_out == nullptr || aligned16(bt->K_out), "K_out must be 16-byte aligned");
    TREVS_CHECK(bt->V_out == nullptr || (aligned16(bt->V) && aligned16(bt->V_out)), "V tensors must be 16-byte aligned");
    TREVS_CHECK(bt->out_head_stride % 8 == 0 && bt->out_tok_stride % 8 == 0 && bt->out_head_stride >= 0 &&
                    bt->out_tok_stride >= 0,
                "K/V output strides must be non-negative multiples of 8");
  }
  return TREVS_OK;
}

// Appends the stage-2 compaction jobs (hidden, K, V rows) to `gm`, offsets in table 1.
void fill_compaction(GatherMeta& gm, const InMeta& meta, const uint16_t* hidden, long long hs, int d_model,
                     uint16_t* hidden_out, long long hos, const uint16_t* K, const uint16_t* V, long long khs,
                     long long kts, int Hkv, uint16_t* K_out, uint16_t* V_out, long long ohs, long long ots,
                     const int* kept, int total_k2) {
  GatherTable& tb = gm.t[1];
  tb.B = meta.B;
  for (int i = 0; i < meta.B; ++i) {
    tb.dst_off[i] = meta.r[i].k2_off;
    tb.src_off[i] = meta.r[i].k1_off;
    tb.src_rows[i] = meta.r[i].k1;
  }
  tb.dst_off[meta.B] = total_k2;
  int nj = gm.njobs;
  if (hidden) {
    GatherJob& j = gm.job[nj++];
    j.src = reinterpret_cast<const uint8_t*>(hidden); j.dst = reinterpret_cast<uint8_t*>(hidden_out);
    j.src_tok = hs * 2; j.dst_tok = hos * 2; j.src_head = 0; j.dst_head = 0;
    j.heads = 1; j.row_bytes = d_model * 2; j.idx = kept; j.rows = total_k2; j.tab = 1;
  }
  const uint16_t* srcs[2] = {K, V};
  uint16_t* dsts[2] = {K_out, V_out};
  for (int x = 0; x < 2; ++x) {
    if (!srcs[x] || !dsts[x]) continue;
    GatherJob& j = gm.job[nj++];
    j.src = reinterpret_cast<const uint8_t*>(srcs[x]); j.dst = reinterpret_cast<uint8_t*>(dsts[x]);
    j.src_tok = kts * 2; j.dst_tok = ots * 2; j.src_head = khs * 2; j.dst_head = ohs * 2;
    j.heads = Hkv; j.row_bytes = TREVS_HEAD_DIM * 2; j.idx = kept; j.rows = total_k2; j.tab = 1;
  }
  gm.njobs = nj;
}

// Runs stage 2 for requests [b0, b1). `overlap`: the preceding grid of the stream is this
// library's stage-1 work on unrelated data, so the first kernel need not wait for it.
// `merged`: gather jobs of stage 1 to launch together with the compaction.
trevs_status run_in_chunk(const trevs_in_batch* bt, int b0, int b1, long long l_base, long long k1_base,
                          long long k2_base, uint8_t* ws, const InWs& L, cudaStream_t st, bool overlap,
                          GatherMeta* merged, bool launch_gather_here = true, bool independent = false) {
  static thread_local InMeta meta;
  static thread_local GatherMeta gm_own;
  GatherMeta& gm = merged ? *merged : gm_own;
  if (!merged) gm.njobs = 0;
  meta.B = b1 - b0;
  int hs = 0, ts = 0, max_k1 = 0, max_l = 0;
  long long lo = 0, ko = 0, k2o = 0, ao = 0;
  for (int b = b0; b < b1; ++b) {
    const trevs_in_request& q = bt->reqs[b];
    InReq& r = meta.r[b - b0];
    r.attn_off = ao;
    ao += (long long)bt->Hq * q.l * q.k1;
    r.l_off = (int)lo; r.l = q.l; r.k1_off = (int)ko; r.k1 = q.k1; r.k2_off = (int)k2o; r.k2 = q.k2;
    lo += q.l; ko += q.k1; k2o += q.k2;
    max_k1 = q.k1 > max_k1 ? q.k1 : max_k1;
    max_l = q.l > max_l ? q.l : max_l;
  }
  InArgs a;
  memset(&a, 0, sizeof(a));
  a.Q = reinterpret_cast<const __nv_bfloat16*>(bt->Q) + l_base * bt->q_tok_stride;
  a.q_hs = bt->q_head_stride; a.q_ts = bt->q_tok_stride;
  a.K = reinterpret_cast<const __nv_bfloat16*>(bt->K) + k1_base * bt->kv_tok_stride;
  a.k_hs = bt->kv_head_stride; a.k_ts = bt->kv_tok_stride;
  a.Hq = bt->Hq; a.Hkv = bt->Hkv; a.n_keep = bt->n_keep_heads;
  a.scale = bt->softmax_scale > 0.f ? bt->softmax_scale : 1.0f / sqrtf((float)bt->d_h);
  a.attn = reinterpret_cast<float*>(ws + L.attn);
  a.row_var = reinterpret_cast<float*>(ws + L.row_var);
  a.rstat = reinterpret_cast<float2*>(ws + L.rstat);
  a.err = reinterpret_cast<uint32_t*>(ws);
  a.stats_ld = lo;
  a.u = (bt->u ? bt->u : reinterpret_cast<float*>(ws + L.u)) + (long long)b0 * bt->Hq;
  a.u_ld = bt->Hq;
  a.p_bits = (bt->p ? reinterpret_cast<uint32_t*>(bt->p) : reinterpret_cast<uint32_t*>(ws + L.p)) + k1_base;
  a.kept_local = bt->kept_local ? bt->kept_local + k2_base : nullptr;
  a.heads_out = bt->heads ? bt->heads + (long long)b0 * bt->n_keep_heads : nullptr;
  a.keys = reinterpret_cast<uint32_t*>(ws + L.keys);
  a.flags = ws + L.flags;
  a.cnt_hs = reinterpret_cast<uint32_t*>(ws + L.cnt_hs);
  a.cnt_ts = reinterpret_cast<uint32_t*>(ws + L.cnt_ts);
  a.hs_finalize = 1;
  a.zero_p = 1;
  if (bt->lse_other) {
    a.lse = bt->lse_other + l_base * bt->lse_row_stride;
    a.lse_hs = bt->lse_head_stride;
    a.lse_rs = bt->lse_row_stride;
  }
  a.overlap = overlap ? 1 : 0;
  a.independent = independent ? 1 : 0;
  // block counts per request: text chunks of the head-statistics and token-score grids
  static thread_local InTcMaps maps;
  const bool small = in_small_fits(bt->Hq, max_l, max_k1);
  const bool tc = !small && make_in_tc_maps(a, lo, ko, maps) == cudaSuccess;
  const int qc = tc ? in_tc_text_rows() : stats_text_rows(max_k1);
  const int sq = tc ? in_tc_text_rows() : kScoreTextRows, sk = tc ? in_tc_score_keys() : kKeyBlock;
  for (int b = b0; b < b1; ++b) {
    const trevs_in_request& q = bt->reqs[b];
    InReq& r = meta.r[b - b0];
    r.hs_off = hs;
    r.ts_off = ts;
    hs += bt->Hq * ((q.l + qc - 1) / qc);
    ts += ((q.l + sq - 1) / sq) * ((q.k1 + sk - 1) / sk);
  }
  meta.total_hs = hs;
  meta.total_ts = ts;
  if (small) {
    TREVS_TRY_CUDA(counted(launch_in_small(meta, a, max_k1, st)), "stage-2 launch");
    ++g_launches;   // two grids
  } else if (tc) {
    TREVS_TRY_CUDA(counted(launch_in_stats_tc(meta, a, maps, st)), "head statistics launch");
    TREVS_TRY_CUDA(counted(launch_in_score_tc(meta, a, maps, st)), "token scores launch");
  } else {
    TREVS_TRY_CUDA(counted(launch_in_head_stats(meta, a, max_k1, st)), "head_stats launch");
    TREVS_TRY_CUDA(counted(launch_in_token_score(meta, a, max_k1, st)), "token_score launch");
  }
  if (k2o > 0 && (bt->hidden || bt->K_out || bt->V)) {
    fill_compaction(gm, meta,
                    bt->hidden ? bt->hidden + k1_base * bt->hidden_row_stride : nullptr, bt->hidden_row_stride,
                    bt->d_model,
                    bt->hidden_out ? bt->hidden_out + k2_base * bt->hidden_out_row_stride : nullptr,
                    bt->hidden_out_row_stride, bt->K_out ? bt->K + k1_base * bt->kv_tok_stride : nullptr,
                    bt->V ? bt->V + k1_base * bt->kv_tok_stride : nullptr, bt->kv_head_stride, bt->kv_tok_stride,
                    bt->Hkv, bt->K_out ? bt->K_out + k2_base * bt->out_tok_stride : nullptr,
                    bt->V_out ? bt->V_out + k2_base * bt->out_tok_stride : nullptr, bt->out_head_stride,
                    bt->out_tok_stride, a.kept_local, (int)k2o);
  }
  if (launch_gather_here && gm.njobs > 0) TREVS_TRY_CUDA(counted(launch_gather(gm, st, true)), "compaction launch");
  return TREVS_OK;
}

// SMs the scoring grid leaves to stage 2's first grids when both stages run in one call:
// in proportion to the two stages' estimated time on the whole GPU. The scoring grid streams
// about 37 GB/s per SM. Stage 2 is weighted at 5 us per 1024 (request, head) blocks on the
// small path and at 2.5 us per million text-to-vision logits on the larger one. Sweeps on
// GB300 put these at or next to the best reserve: 24 SMs for the LLaVA-1.5 batch of 32
// (84.3 us per call against 88.2 without the overlap), 48 for LLaVA-NeXT 8 x 2,880 (112.6
// against 122.8) and for 2 x 16,384 video tokens (158.1 against 172.0).
constexpr double kScoreBytesPerUsPerSm = 37e3;    // 37 GB/s
constexpr double kSmallUsPer1024Heads = 5.0;
constexpr double kLargeUsPerMLogits = 2.5;

std::atomic<int> g_reserve_override{-1};   // trevs_set_overlap_reserve; < 0: the estimate

int overlap_reserve(const trevs_pre_batch* pre, const trevs_in_batch* in, const PreTotals& tp, bool small) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 16)
    return 0;
  const int forced = g_reserve_override.load(std::memory_order_relaxed);
  if (forced >= 0) return forced < sms / 2 ? forced : sms / 2;
  const double score_us = (double)tp.n * pre->d * 2.0 / (kScoreBytesPerUsPerSm * sms);
  double logits = 0.0;
  for (int b = 0; b < in->B; ++b) logits += (double)in->Hq * in->reqs[b].l * in->reqs[b].k1;
  const double attn_us = small ? kSmallUsPer1024Heads * in->B * in->Hq / 1024.0 : kLargeUsPerMLogits * logits * 1e-6;
  int r = (int)((double)sms * attn_us / (score_us + attn_us) + 0.5);
  const int lo = 8, hi = sms / 2;
  r = r < lo ? lo : (r > hi ? hi : r);
  // A scoring grid whose CTAs each take whole tiles leaves no tile split between CTAs, so
  // the finishing grid has no partial sums to add: take such a grid if one lies between the
  // estimate and half of it (more scoring CTAs, never fewer). On GB300 the 2 x 16,384 video
  // batch drops from 157 to 142 us per call this way (128 CTAs of 2 tiles each).
  int tiles = 0;
  for (int b = 0; b < pre->B; ++b) tiles += (pre->reqs[b].n + kScoreTileRows - 1) / kScoreTileRows;
  for (int x = r / 2 > lo ? r / 2 : lo; x <= r && tiles > 0; ++x)
    if (tiles % (sms - x) == 0) return x;
  return r;
}

trevs_status run_in_batch(const trevs_in_batch* bt, uint8_t* ws, const InWs& L, cudaStream_t st) {
  long long l_base = 0, k1_base = 0, k2_base = 0;
  for (int b0 = 0; b0 < bt->B; b0 += kMaxChunk) {
    const int b1 = b0 + kMaxChunk < bt->B ? b0 + kMaxChunk : bt->B;
    trevs_status s = run_in_chunk(bt, b0, b1, l_base, k1_base, k2_base, ws, L, st, false, nullptr);
    if (s != TREVS_OK) return s;
    for (int b = b0; b < b1; ++b) {
      l_base += bt->reqs[b].l; k1_base += bt->reqs[b].k1; k2_base += bt->reqs[b].k2;
    }
  }
  return TREVS_OK;
}

const trevs_pre_params kDefaults = {1.4f, 1.0f, 1.0f, 1e-6f, TREVS_SELECT_RATIO, 0.0f};

}  // namespace

namespace trevs {
// Lets the other translation units of the library report through trevs_last_error_string
// and trevs_last_launch_count.
trevs_status record_error(trevs_status s, const char* msg) { return fail(s, "%s", msg); }
void record_launches(int n) { g_launches = n; }
bool launch_fault_injected() { return g_fail_in > 0 && --g_fail_in == 0; }
}  // namespace trevs

// ======================================================================== C ABI

extern "C" {

void trevs_pre_params_default(trevs_pre_params* p) {
  if (p) *p = kDefaults;
}

const char* trevs_version(void) { return "0.1.0"; }

const char* trevs_last_error_string(void) { return g_err; }

int32_t trevs_last_launch_count(void) { return g_launches; }

trevs_status trevs_workspace_status(const void* workspace, size_t bytes, void* stream) {
  if (!workspace || bytes < sizeof(uint32_t)) return fail(TREVS_ERR_WORKSPACE, "workspace is NULL or too small");
  uint32_t word = 0;
  TREVS_TRY_CUDA(cudaMemcpyAsync(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost, (cudaStream_t)stream),
                 "status read");
  TREVS_TRY_CUDA(cudaStreamSynchronize((cudaStream_t)stream), "status read");
  if (word & 1u) return fail(TREVS_ERR_TIMEOUT, "a bounded device-side wait gave up (status word 0x%x)", word);
  if (word & 2u)
    return fail(TREVS_ERR_INVALID_ARGUMENT, "farthest point sampling found no candidate left (status word 0x%x)", word);
  return TREVS_OK;
}

void trevs_test_fail_launch(int32_t n) { g_fail_in = n > 0 ? n : 0; }

void trevs_set_overlap_reserve(int32_t sms) { g_reserve_override.store(sms < 0 ? -1 : sms); }

trevs_status trevs_workspace_set_wait_limit(void* workspace, size_t bytes, uint32_t microseconds, void* stream) {
  g_launches = 0;
  if (!workspace || bytes < 2 * sizeof(uint32_t)) return fail(TREVS_ERR_WORKSPACE, "workspace is NULL or too small");
  const uint32_t us = microseconds;   // pageable source: copied out before the call returns
  TREVS_TRY_CUDA(cudaMemcpyAsync(reinterpret_cast<uint32_t*>(workspace) + 1, &us, sizeof(us), cudaMemcpyHostToDevice,
                                 (cudaStream_t)stream),
                 "wait limit write");
  return TREVS_OK;
}

trevs_status trevs_workspace_init(void* workspace, size_t bytes, void* stream) {
  g_launches = 0;
  if (bytes == 0) return TREVS_OK;
  if (!workspace) return fail(TREVS_ERR_WORKSPACE, "workspace is NULL");
  TREVS_TRY_CUDA(counted(cudaMemsetAsync(workspace, 0, bytes, (cudaStream_t)stream)), "workspace memset");
  return TREVS_OK;
}

size_t trevs_pre_llm_workspace_size(int32_t N) {
  return N < 0 ? 0 : pre_ws(N, TREVS_MAX_TEXT_TOKENS, TREVS_MAX_TEXT_TOKENS).end;
}

trevs_status trevs_pre_llm_scores(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                                  const uint16_t* T, int64_t t_row_stride, int32_t M, const float* s_v,
                                  const trevs_pre_params* p, float* s_t_out, float* s_fused_out,
                                  void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  const trevs_pre_params prm = p ? *p : kDefaults;
  trevs_status s = validate_params(&prm);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(N >= 0, "N = %d < 0", N);
  if (N == 0) return TREVS_OK;
  TREVS_CHECK(s_t_out != nullptr, "s_t_out is NULL");
  TREVS_CHECK(s_fused_out == nullptr || s_v != nullptr, "s_v is needed for the fused score");
  trevs_pre_request rq = {N, M, 0, 0.f};
  trevs_pre_batch bt;
  memset(&bt, 0, sizeof(bt));
  bt.B = 1; bt.d = d; bt.reqs = &rq; bt.Z = Z; bt.z_row_stride = z_row_stride; bt.T = T;
  bt.t_row_stride = t_row_stride; bt.s_v = s_v ? s_v : s_t_out;
  PreTotals tot;
  s = validate_pre_batch(&bt, tot);
  if (s != TREVS_OK) return s;
  const PreWs L = pre_ws(N, TREVS_MAX_TEXT_TOKENS, TREVS_MAX_TEXT_TOKENS);
  s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  static thread_local PreMeta meta;
  meta.B = 1;
  meta.r[0] = PreReq{0, N, 0, M, 0, 0, 0, 0};
  meta.total_tiles = (N + kScoreTileRows - 1) / kScoreTileRows;
  PreArgs a;
  memset(&a, 0, sizeof(a));
  a.Z = reinterpret_cast<const __nv_bfloat16*>(Z); a.z_stride = z_row_stride;
  a.T = reinterpret_cast<const __nv_bfloat16*>(T); a.t_stride = t_row_stride;
  a.s_v = bt.s_v; a.s_t = s_t_out;
  a.s_fused = s_fused_out;
  a.flags = ws + L.flags; a.keys = reinterpret_cast<uint32_t*>(ws + L.keys);
  a.counters = reinterpret_cast<uint32_t*>(ws + L.counters);
  a.sal = reinterpret_cast<int4*>(ws + L.sal);
  a.t_rinv = reinterpret_cast<float*>(ws + L.t_rinv);
  a.total_m = M;
  a.part = reinterpret_cast<float*>(ws + L.part);
  a.err = reinterpret_cast<uint32_t*>(ws);
  a.d = d; a.mode = s_fused_out ? kModeFused : kModeRatio;
  a.tau_v = prm.tau_v; a.tau_t = prm.tau_t; a.lambda = prm.lambda; a.eps = prm.eps;
  a.action = s_fused_out ? kActScoresFused : kActScores;
  TREVS_TRY_CUDA(counted(launch_pre_saliency(meta, a, N, false, (cudaStream_t)stream)), "pre-pass launch");
  TREVS_TRY_CUDA(counted(launch_pre_score(meta, a, M, N, (cudaStream_t)stream, true)), "pre_score launch");
  TREVS_TRY_CUDA(counted(launch_pre_finish(meta, a, M, N, true, (cudaStream_t)stream, true)), "finishing launch");
  return TREVS_OK;
}

size_t trevs_cls_saliency_workspace_size(int32_t B, const int32_t* n, int32_t H) {
  if (B <= 0 || !n || H <= 0) return 0;
  long long total = 0;
  for (int b = 0; b < B; ++b) total += n[b] > 0 ? n[b] : 0;
  return cls_ws(total, H).end;
}

trevs_status trevs_cls_saliency_varlen(const uint16_t* q_cls, int64_t q_req_stride, int64_t q_head_stride,
                                       const uint16_t* K_v, int64_t k_tok_stride, int64_t k_head_stride,
                                       int32_t B, const int32_t* n, int32_t H, int32_t d_h, float scale,
                                       float* s_v, void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  TREVS_CHECK(B >= 0, "B = %d < 0", B);
  if (B == 0) return TREVS_OK;
  TREVS_CHECK(n != nullptr, "n is NULL");
  TREVS_CHECK(H >= 1, "H = %d < 1", H);
  if (H > TREVS_MAX_HEADS) return fail(TREVS_ERR_UNSUPPORTED, "H = %d > %d", H, TREVS_MAX_HEADS);
  if (!cls_head_dim_supported(d_h)) return fail(TREVS_ERR_UNSUPPORTED, "d_h = %d: 32, 64 or 128 supported", d_h);
  long long total = 0;
  for (int b = 0; b < B; ++b) {
    TREVS_CHECK(n[b] >= 0, "request %d: n = %d < 0", b, n[b]);
    if (n[b] > kClsMaxN) return fail(TREVS_ERR_UNSUPPORTED, "request %d: n = %d > %d patches", b, n[b], kClsMaxN);
    total += n[b];
  }
  TREVS_CHECK(total < (1ll << 31), "batch too large for int32 offsets");
  if (total == 0) return TREVS_OK;
  TREVS_CHECK(q_cls && K_v && s_v, "q_cls, K_v and s_v must be non-NULL");
  TREVS_CHECK(aligned16(q_cls) && aligned16(K_v), "q_cls and K_v must be 16-byte aligned");
  TREVS_CHECK(q_req_stride >= 0 && q_head_stride >= 0 && k_tok_stride >= 0 && k_head_stride >= 0 &&
                  q_req_stride % 8 == 0 && q_head_stride % 8 == 0 && k_tok_stride % 8 == 0 && k_head_stride % 8 == 0,
              "strides must be non-negative multiples of 8");
  TREVS_CHECK(std::isfinite(scale), "scale must be finite");
  const ClsWs L = cls_ws(total, H);
  trevs_status s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  static thread_local ClsMeta meta;
  long long n_base = 0;
  for (int b0 = 0; b0 < B; b0 += kMaxChunk) {
    const int b1 = b0 + kMaxChunk < B ? b0 + kMaxChunk : B;
    meta.B = 0;
    meta.H = H;
    long long no = 0;
    int chunk_max = 0;
    for (int b = b0; b < b1; ++b) {
      if (n[b] > 0) meta.r[meta.B++] = ClsReq{(int)no, n[b], b - b0};
      no += n[b];
      chunk_max = n[b] > chunk_max ? n[b] : chunk_max;
    }
    ClsArgs a;
    a.q = reinterpret_cast<const __nv_bfloat16*>(q_cls) + (long long)b0 * q_req_stride;
    a.q_req = q_req_stride; a.q_head = q_head_stride;
    a.K = reinterpret_cast<const __nv_bfloat16*>(K_v) + n_base * k_tok_stride;
    a.k_tok = k_tok_stride; a.k_head = k_head_stride;
    a.scale = scale > 0.f ? scale : 1.0f / std::sqrt((float)d_h);
    a.attn = reinterpret_cast<float*>(ws + L.attn);
    a.attn_ld = no;
    a.s_v = s_v + n_base;
    a.cnt = reinterpret_cast<uint32_t*>(ws + L.cnt);
    if (meta.B > 0)
      TREVS_TRY_CUDA(counted(launch_cls_saliency(meta, a, d_h, chunk_max, (cudaStream_t)stream)), "saliency launch");
    n_base += no;
  }
  return TREVS_OK;
}

size_t trevs_pre_llm_fps_workspace_size(int32_t N, int32_t K_r, int32_t d) {
  if (N < 0 || K_r < 0 || d < 0) return 0;
  return fps_ws(kStatusBytes, N, K_r, K_r, d).end;
}

trevs_status trevs_pre_llm_fps(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                               const int32_t* pivots, int32_t K_r, int32_t K_d, int32_t pool, int32_t* picks,
                               float* pick_dist, void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  TREVS_CHECK(N >= 0 && K_r >= 0 && K_d >= 0, "N = %d, K_r = %d, K_d = %d: none may be negative", N, K_r, K_d);
  TREVS_CHECK((long long)K_r + K_d <= N, "K_r + K_d = %lld exceeds N = %d", (long long)K_r + K_d, N);
  TREVS_CHECK(pool >= 0, "pool = %d < 0", pool);
  if (K_d == 0) return TREVS_OK;
  TREVS_CHECK(d >= 8 && d % 8 == 0, "d = %d must be a positive multiple of 8", d);
  TREVS_CHECK(Z != nullptr && aligned16(Z), "Z must be non-NULL and 16-byte aligned");
  TREVS_CHECK(z_row_stride >= d && z_row_stride % 8 == 0, "z_row_stride must be >= d and a multiple of 8");
  TREVS_CHECK(K_r == 0 || pivots != nullptr, "pivots is NULL");
  TREVS_CHECK(picks != nullptr, "picks is NULL");
  const FpsWs L = fps_ws(kStatusBytes, N, K_r, K_r, d);
  trevs_status s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  const cudaStream_t st = (cudaStream_t)stream;
  float* maxcos = reinterpret_cast<float*>(ws + L.maxcos);
  // without pivots row 0 is the first draw and the one pivot of the contraction
  const int lead = K_r == 0 ? 1 : 0;
  const int kr = K_r + lead;
  const int32_t* piv = lead ? reinterpret_cast<const int32_t*>(ws + L.zero) : pivots;
  {   // the largest cosine of every row to the pivots: the scoring contraction over copies of
      // the pivot rows (an index outside [0, N) leaves its zero-filled row in place)
    uint16_t* prow = reinterpret_cast<uint16_t*>(ws + L.prow);
    TREVS_TRY_CUDA(counted(cudaMemsetAsync(prow, 0, 2 * (size_t)kr * d, st)), "pivot rows clear");
    static thread_local GatherMeta pg;
    pg.njobs = 1;
    pg.t[0].B = 1;
    pg.t[0].dst_off[0] = 0; pg.t[0].dst_off[1] = kr; pg.t[0].src_off[0] = 0; pg.t[0].src_rows[0] = N;
    GatherJob& j = pg.job[0];
    j.src = reinterpret_cast<const uint8_t*>(Z); j.dst = reinterpret_cast<uint8_t*>(prow);
    j.src_tok = z_row_stride * 2; j.dst_tok = (long long)d * 2; j.src_head = 0; j.dst_head = 0;
    j.heads = 1; j.row_bytes = d * 2; j.idx = piv; j.rows = kr; j.tab = 0;
    TREVS_TRY_CUDA(counted(launch_gather(pg, st, false)), "pivot rows launch");
    static thread_local PreMeta meta;
    meta.B = 1;
    meta.r[0] = PreReq{0, N, 0, kr, 0, 0, 0, 0};
    meta.total_tiles = (N + kScoreTileRows - 1) / kScoreTileRows;
    PreArgs a;
    memset(&a, 0, sizeof(a));
    a.Z = reinterpret_cast<const __nv_bfloat16*>(Z); a.z_stride = z_row_stride;
    a.T = reinterpret_cast<const __nv_bfloat16*>(prow); a.t_stride = d;
    a.s_t = maxcos;
    a.t_rinv = reinterpret_cast<float*>(ws + L.t_rinv);
    a.total_m = kr;
    a.part = reinterpret_cast<float*>(ws + L.part);
    a.err = reinterpret_cast<uint32_t*>(ws);
    a.d = d; a.mode = kModeRatio; a.action = kActFpsSeed;
    TREVS_TRY_CUDA(counted(launch_pre_saliency(meta, a, N, false, st)), "pivot norms launch");
    const trevs_status cs = run_pivot_contraction(meta, a, N, N, st);
    if (cs != TREVS_OK) return cs;
  }
  static thread_local FpsMeta fm;
  fm.B = 1;
  fm.r[0] = FpsReq{0, N, 0, kr, K_d, lead, 0, 0};
  FpsArgs f;
  memset(&f, 0, sizeof(f));
  f.Z = reinterpret_cast<const __nv_bfloat16*>(Z); f.z_stride = z_row_stride; f.d = d;
  f.piv = piv; f.maxcos = maxcos;
  f.ub = reinterpret_cast<float*>(ws + L.ub); f.stamp = reinterpret_cast<int*>(ws + L.stamp);
  f.flags = ws + L.flags; f.keys = reinterpret_cast<uint32_t*>(ws + L.keys);
  f.picks = picks; f.pick_dist = pick_dist; f.kept = nullptr; f.pool = pool;
  f.err = reinterpret_cast<uint32_t*>(ws);
  TREVS_TRY_CUDA(counted(launch_fps(fm, f, st, true)), "farthest point sampling launch");
  return TREVS_OK;
}

trevs_status trevs_pre_llm_select(const float* s_v, const float* s_t, const float* s_fused, int32_t N,
                                  int32_t K1, float textual_ratio, const trevs_pre_params* p,
                                  int32_t* kept_idx, void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  const trevs_pre_params prm = p ? *p : kDefaults;
  trevs_status s = validate_params(&prm);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(N >= 0 && K1 >= 0 && K1 <= N, "need 0 <= K1 (%d) <= N (%d)", K1, N);
  TREVS_CHECK(std::isfinite(textual_ratio) && textual_ratio >= 0.f && textual_ratio <= 1.f,
              "textual ratio %g outside [0, 1]", (double)textual_ratio);
  if (K1 == 0) return TREVS_OK;
  TREVS_CHECK(kept_idx != nullptr, "kept_idx is NULL");
  const bool fused = prm.select_mode == TREVS_SELECT_FUSED;
  if (fused && !s_fused) TREVS_CHECK(s_v && s_t, "fused mode needs s_fused or both s_v and s_t");
  if (!fused) TREVS_CHECK(s_v && s_t, "ratio mode needs s_v and s_t");
  const PreWs L = pre_ws(N, TREVS_MAX_TEXT_TOKENS, TREVS_MAX_TEXT_TOKENS);
  s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  static thread_local PreMeta meta;
  meta.B = 1;
  meta.r[0] = PreReq{0, N, 0, 0, 0, K1, textual_count(K1, textual_ratio), 0};
  meta.total_tiles = 0;
  PreArgs a;
  memset(&a, 0, sizeof(a));
  a.s_v = s_v; a.s_t = const_cast<float*>(s_t);
  a.s_fused = s_fused ? const_cast<float*>(s_fused) : reinterpret_cast<float*>(ws + L.s_fused);
  a.s_fused_given = s_fused != nullptr;
  a.kept = kept_idx;
  a.flags = ws + L.flags; a.keys = reinterpret_cast<uint32_t*>(ws + L.keys);
  a.counters = reinterpret_cast<uint32_t*>(ws + L.counters);
  a.sal = reinterpret_cast<int4*>(ws + L.sal);
  a.err = reinterpret_cast<uint32_t*>(ws);
  a.mode = fused ? kModeFused : kModeRatio;
  a.tau_v = prm.tau_v; a.tau_t = prm.tau_t; a.lambda = prm.lambda; a.eps = prm.eps;
  a.action = kActSelect;
  TREVS_TRY_CUDA(counted(launch_pre_finish(meta, a, 0, N, false, (cudaStream_t)stream, false)), "selection launch");
  return TREVS_OK;
}

trevs_status trevs_pre_llm_gather(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                                  const int32_t* kept_idx, int32_t K1, uint16_t* Z_out,
                                  int64_t z_out_row_stride, void* stream) {
  g_launches = 0;
  TREVS_CHECK(N >= 0 && K1 >= 0 && K1 <= N, "need 0 <= K1 (%d) <= N (%d)", K1, N);
  if (K1 == 0) return TREVS_OK;
  TREVS_CHECK(d >= 8 && d % 8 == 0, "d = %d must be a positive multiple of 8", d);
  TREVS_CHECK(Z && kept_idx && Z_out, "Z, kept_idx and Z_out must be non-NULL");
  TREVS_CHECK(aligned16(Z) && aligned16(Z_out), "Z and Z_out must be 16-byte aligned");
  TREVS_CHECK(z_row_stride >= d && z_row_stride % 8 == 0 && z_out_row_stride >= d && z_out_row_stride % 8 == 0,
              "row strides must be >= d and multiples of 8");
  static thread_local GatherMeta gm;
  gm.njobs = 1;
  gm.t[0].B = 1;
  gm.t[0].dst_off[0] = 0; gm.t[0].dst_off[1] = K1; gm.t[0].src_off[0] = 0; gm.t[0].src_rows[0] = N;
  GatherJob& j = gm.job[0];
  j.src = reinterpret_cast<const uint8_t*>(Z); j.dst = reinterpret_cast<uint8_t*>(Z_out);
  j.src_tok = z_row_stride * 2; j.dst_tok = z_out_row_stride * 2; j.src_head = 0; j.dst_head = 0;
  j.heads = 1; j.row_bytes = d * 2; j.idx = kept_idx; j.rows = K1; j.tab = 0;
  TREVS_TRY_CUDA(counted(launch_gather(gm, (cudaStream_t)stream, true)), "gather launch");
  return TREVS_OK;
}

trevs_status trevs_stream_probe(const uint16_t* Z, int64_t z_row_stride, int64_t rows, int32_t d, int32_t ctas,
                                void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  TREVS_CHECK(Z != nullptr && aligned16(Z), "Z must be non-NULL and 16-byte aligned");
  TREVS_CHECK(rows >= 1 && rows <= (1LL << 31), "rows = %lld out of range", (long long)rows);
  TREVS_CHECK(d >= 256 && d % 256 == 0, "d = %d must be a positive multiple of 256", d);
  TREVS_CHECK(z_row_stride >= d && z_row_stride % 8 == 0, "z_row_stride must be >= d and a multiple of 8");
  TREVS_CHECK(ctas >= 1 && ctas <= 1024, "ctas = %d out of [1, 1024]", ctas);
  TREVS_CHECK(workspace != nullptr && workspace_bytes >= 2 * sizeof(uint32_t), "workspace (status word) missing");
  TREVS_TRY_CUDA(counted(launch_stream_probe(Z, z_row_stride, rows, d, ctas, reinterpret_cast<uint32_t*>(workspace),
                                             (cudaStream_t)stream)),
                 "streaming probe launch");
  return TREVS_OK;
}

size_t trevs_in_llm_workspace_size(int32_t Hq, int32_t L, int32_t K1) {
  if (Hq < 0 || L < 0 || K1 < 0) return 0;
  return in_ws(L, K1, 0, Hq, 1).end;   // the attention probabilities live in the caller's buffer
}

trevs_status trevs_in_llm_head_scores(const uint16_t* Q, int64_t q_head_stride, int64_t q_tok_stride,
                                      const uint16_t* K, int64_t k_head_stride, int64_t k_tok_stride,
                                      int32_t Hq, int32_t Hkv, int32_t L, int32_t K1, int32_t d_h,
                                      float softmax_scale, const float* lse_other, float* u_out, float* attn_out,
                                      void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  trevs_status s = validate_in_common(Hq, Hkv, d_h, 1);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(L >= 1, "L = %d < 1", L);
  TREVS_CHECK(K1 >= 1, "K1 = %d < 1", K1);
  if (K1 > TREVS_MAX_STAGE2_TOKENS) return fail(TREVS_ERR_UNSUPPORTED, "K1 = %d > %d", K1, TREVS_MAX_STAGE2_TOKENS);
  s = validate_qk(Q, q_head_stride, q_tok_stride, K, k_head_stride, k_tok_stride);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(u_out && attn_out, "u_out and attn_out must be non-NULL");
  const InWs W = in_ws(L, K1, 0, Hq, 1);
  s = check_ws(workspace, workspace_bytes, W.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  static thread_local InMeta meta;
  meta.B = 1;
  meta.r[0] = InReq{0, 0, L, 0, K1, 0, 0, 0, 0};
  meta.total_hs = Hq * ((L + stats_text_rows(K1) - 1) / stats_text_rows(K1));
  meta.total_ts = 0;
  InArgs a;
  memset(&a, 0, sizeof(a));
  a.Q = reinterpret_cast<const __nv_bfloat16*>(Q); a.q_hs = q_head_stride; a.q_ts = q_tok_stride;
  a.K = reinterpret_cast<const __nv_bfloat16*>(K); a.k_hs = k_head_stride; a.k_ts = k_tok_stride;
  a.Hq = Hq; a.Hkv = Hkv; a.n_keep = 1;
  a.scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)d_h);
  a.attn = attn_out;
  a.row_var = reinterpret_cast<float*>(ws + W.row_var);
  a.stats_ld = L;
  a.u = u_out; a.u_ld = Hq;
  a.cnt_hs = reinterpret_cast<uint32_t*>(ws + W.cnt_hs);
  a.cnt_ts = reinterpret_cast<uint32_t*>(ws + W.cnt_ts);
  a.hs_finalize = 1; a.zero_p = 0;
  TREVS_CHECK(lse_other == nullptr || ((uintptr_t)lse_other & 3u) == 0, "lse_other must be 4-byte aligned");
  a.lse = lse_other; a.lse_hs = L; a.lse_rs = 1;
  TREVS_TRY_CUDA(counted(launch_in_head_stats(meta, a, K1, (cudaStream_t)stream)), "head_stats launch");
  return TREVS_OK;
}

trevs_status trevs_in_llm_select(const float* u, const float* attn, int32_t Hq, int32_t L, int32_t K1,
                                 int32_t n_keep_heads, int32_t K2, int32_t* heads_out, float* p_out,
                                 int32_t* kept_local, void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  TREVS_CHECK(Hq >= 1, "Hq = %d < 1", Hq);
  if (Hq > TREVS_MAX_HEADS) return fail(TREVS_ERR_UNSUPPORTED, "Hq = %d > %d", Hq, TREVS_MAX_HEADS);
  TREVS_CHECK(n_keep_heads >= 1 && n_keep_heads <= Hq, "n_keep_heads = %d outside [1, Hq = %d]", n_keep_heads, Hq);
  TREVS_CHECK(L >= 1, "L = %d < 1", L);
  TREVS_CHECK(K1 >= 1, "K1 = %d < 1", K1);
  if (K1 > TREVS_MAX_STAGE2_TOKENS) return fail(TREVS_ERR_UNSUPPORTED, "K1 = %d > %d", K1, TREVS_MAX_STAGE2_TOKENS);
  TREVS_CHECK(K2 >= 0 && K2 <= K1, "K2 = %d outside [0, K1 = %d]", K2, K1);
  TREVS_CHECK(u && attn, "u and attn must be non-NULL");
  if (K2 > 0) TREVS_CHECK(kept_local != nullptr, "kept_local is NULL");
  const InWs W = in_ws(L, K1, 0, Hq, 1);
  trevs_status s = check_ws(workspace, workspace_bytes, W.end);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  static thread_local InMeta meta;
  meta.B = 1;
  meta.r[0] = InReq{0, 0, L, 0, K1, 0, K2, 0, 0};
  meta.total_hs = 0;
  meta.total_ts = ((L + kScoreTextRows - 1) / kScoreTextRows) * ((K1 + kKeyBlock - 1) / kKeyBlock);
  InArgs a;
  memset(&a, 0, sizeof(a));
  a.Hq = Hq; a.n_keep = n_keep_heads;
  a.attn = const_cast<float*>(attn);
  a.stats_ld = L;
  a.u = const_cast<float*>(u); a.u_ld = Hq;
  a.p_bits = p_out ? reinterpret_cast<uint32_t*>(p_out) : reinterpret_cast<uint32_t*>(ws + W.p);
  a.kept_local = kept_local; a.heads_out = heads_out;
  a.keys = reinterpret_cast<uint32_t*>(ws + W.keys);
  a.flags = ws + W.flags;
  a.cnt_hs = reinterpret_cast<uint32_t*>(ws + W.cnt_hs);
  a.cnt_ts = reinterpret_cast<uint32_t*>(ws + W.cnt_ts);
  TREVS_TRY_CUDA(counted(cudaMemsetAsync(a.p_bits, 0, 4 * (size_t)K1, (cudaStream_t)stream)), "p memset");
  TREVS_TRY_CUDA(counted(launch_in_token_score(meta, a, K1, (cudaStream_t)stream)), "token_score launch");
  return TREVS_OK;
}

trevs_status trevs_in_llm_compact(const uint16_t* hidden, int64_t hidden_row_stride, int32_t d_model,
                                  const uint16_t* Kc, const uint16_t* Vc, int64_t kv_head_stride,
                                  int64_t kv_tok_stride, int32_t Hkv, int32_t d_h, int32_t K1,
                                  const int32_t* kept_local, int32_t K2, uint16_t* hidden_out,
                                  int64_t hidden_out_row_stride, uint16_t* K_out, uint16_t* V_out,
                                  int64_t out_head_stride, int64_t out_tok_stride, void* stream) {
  g_launches = 0;
  TREVS_CHECK(K1 >= 0 && K2 >= 0 && K2 <= K1, "need 0 <= K2 (%d) <= K1 (%d)", K2, K1);
  if (K2 == 0) return TREVS_OK;
  TREVS_CHECK(kept_local != nullptr, "kept_local is NULL");
  TREVS_CHECK((hidden == nullptr) == (hidden_out == nullptr), "hidden and hidden_out: both or neither");
  TREVS_CHECK((Kc == nullptr) == (K_out == nullptr), "Kc and K_out: both or neither");
  TREVS_CHECK((Vc == nullptr) == (V_out == nullptr), "Vc and V_out: both or neither");
  if (hidden) {
    TREVS_CHECK(d_model >= 8 && d_model % 8 == 0, "d_model = %d must be a positive multiple of 8", d_model);
    TREVS_CHECK(aligned16(hidden) && aligned16(hidden_out), "hidden tensors must be 16-byte aligned");
    TREVS_CHECK(hidden_row_stride >= d_model && hidden_row_stride % 8 == 0 && hidden_out_row_stride >= d_model &&
                    hidden_out_row_stride % 8 == 0,
                "hidden strides must be >= d_model and multiples of 8");
  }
  if (Kc || Vc) {
    TREVS_CHECK(Hkv >= 1, "Hkv = %d < 1", Hkv);
    if (d_h != TREVS_HEAD_DIM) return fail(TREVS_ERR_UNSUPPORTED, "d_h = %d, only %d supported", d_h, TREVS_HEAD_DIM);
    TREVS_CHECK((!Kc || (aligned16(Kc) && aligned16(K_out))) && (!Vc || (aligned16(Vc) && aligned16(V_out))),
                "K/V tensors must be 16-byte aligned");
    TREVS_CHECK(kv_head_stride % 8 == 0 && kv_tok_stride % 8 == 0 && out_head_stride % 8 == 0 &&
                    out_tok_stride % 8 == 0 && kv_head_stride >= 0 && kv_tok_stride >= 0 && out_head_stride >= 0 &&
                    out_tok_stride >= 0,
                "K/V strides must be non-negative multiples of 8");
  }
  static thread_local InMeta meta;
  static thread_local GatherMeta gm;
  meta.B = 1;
  meta.r[0] = InReq{0, 0, 0, 0, K1, 0, K2, 0, 0};
  gm.njobs = 0;
  fill_compaction(gm, meta, hidden, hidden_row_stride, d_model, hidden_out, hidden_out_row_stride, Kc, Vc,
                  kv_head_stride, kv_tok_stride, Hkv, K_out, V_out, out_head_stride, out_tok_stride, kept_local, K2);
  TREVS_TRY_CUDA(counted(launch_gather(gm, (cudaStream_t)stream, true)), "compaction launch");
  return TREVS_OK;
}

size_t trevs_pre_llm_varlen_workspace_size(const trevs_pre_batch* batch) {
  if (!batch || batch->B <= 0 || !batch->reqs) return 0;
  long long n = 0, m = 0, k1 = 0, fpool = 0, fgram = 0;
  int max_m = 0, max_k1 = 0;
  for (int b = 0; b < batch->B; ++b) {
    const trevs_pre_request& r = batch->reqs[b];
    n += r.n > 0 ? r.n : 0;
    m += r.m > 0 ? r.m : 0;
    k1 += r.k1 > 0 ? r.k1 : 0;
    const long long gl = fps_gram_ld(r.k1);
    fpool += gl;
    fgram += gl * gl;
    if (r.n > 0 && r.m > max_m) max_m = r.m;
    if (r.k1 > max_k1) max_k1 = r.k1;
  }
  return pre_ws(n, m, max_m, k1, max_k1, batch->d, fpool, fgram).end;
}

size_t trevs_in_llm_varlen_workspace_size(const trevs_in_batch* batch) {
  if (!batch || batch->B <= 0 || !batch->reqs) return 0;
  long long l = 0, k1 = 0, lk1 = 0;
  for (int b = 0; b < batch->B; ++b) {
    const long long lb = batch->reqs[b].l > 0 ? batch->reqs[b].l : 0;
    const long long kb = batch->reqs[b].k1 > 0 ? batch->reqs[b].k1 : 0;
    l += lb; k1 += kb; lk1 += lb * kb;
  }
  return in_ws(l, k1, lk1, batch->Hq > 0 ? batch->Hq : 0, batch->B).end;
}

size_t trevs_prune_varlen_workspace_size(const trevs_pre_batch* pre, const trevs_in_batch* in) {
  return al256(trevs_pre_llm_varlen_workspace_size(pre)) + trevs_in_llm_varlen_workspace_size(in);
}

trevs_status trevs_pre_llm_varlen(const trevs_pre_batch* batch, const trevs_pre_params* p, void* workspace,
                                  size_t workspace_bytes, void* stream) {
  g_launches = 0;
  const trevs_pre_params prm = p ? *p : kDefaults;
  trevs_status s = validate_params(&prm);
  if (s != TREVS_OK) return s;
  PreTotals t;
  s = validate_pre_batch(batch, t);
  if (s != TREVS_OK || batch->B == 0) return s;
  s = validate_diversity(batch, prm);
  if (s != TREVS_OK) return s;
  const PreWs L = pre_ws(t.n, t.m, t.max_m, t.k1, t.max_k1, batch->d, t.fps_pool, t.fps_gram);
  s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  return run_pre_batch(batch, prm, reinterpret_cast<uint8_t*>(workspace), L, (cudaStream_t)stream);
}

trevs_status trevs_pre_llm_varlen_timed(const trevs_pre_batch* batch, const trevs_pre_params* p, void* workspace,
                                        size_t workspace_bytes, void* stream, void* ev_score_begin,
                                        void* ev_score_end) {
  g_launches = 0;
  const trevs_pre_params prm = p ? *p : kDefaults;
  trevs_status s = validate_params(&prm);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(ev_score_begin != nullptr && ev_score_end != nullptr, "both events must be non-NULL");
  PreTotals t;
  s = validate_pre_batch(batch, t);
  if (s != TREVS_OK) return s;
  TREVS_CHECK(batch->B >= 1, "B = 0: nothing to time");
  if (batch->B > kMaxChunk) return fail(TREVS_ERR_UNSUPPORTED, "B = %d > %d requests", batch->B, kMaxChunk);
  s = validate_diversity(batch, prm);
  if (s != TREVS_OK) return s;
  const PreWs L = pre_ws(t.n, t.m, t.max_m, t.k1, t.max_k1, batch->d, t.fps_pool, t.fps_gram);
  s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  return run_pre_chunk(batch, prm, 0, batch->B, 0, 0, 0, reinterpret_cast<uint8_t*>(workspace), L,
                       (cudaStream_t)stream, nullptr, (cudaEvent_t)ev_score_end, (cudaEvent_t)ev_score_begin);
}

trevs_status trevs_in_llm_varlen(const trevs_in_batch* batch, void* workspace, size_t workspace_bytes,
                                 void* stream) {
  g_launches = 0;
  InTotals t;
  trevs_status s = validate_in_batch(batch, t);
  if (s != TREVS_OK || batch->B == 0) return s;
  const InWs L = in_ws(t.l, t.k1, t.lk1, batch->Hq, batch->B);
  s = check_ws(workspace, workspace_bytes, L.end);
  if (s != TREVS_OK) return s;
  return run_in_batch(batch, reinterpret_cast<uint8_t*>(workspace), L, (cudaStream_t)stream);
}

trevs_status trevs_prune_varlen(const trevs_pre_batch* pre, const trevs_pre_params* p, const trevs_in_batch* in,
                                void* workspace, size_t workspace_bytes, void* stream) {
  g_launches = 0;
  const trevs_pre_params prm = p ? *p : kDefaults;
  trevs_status s = validate_params(&prm);
  if (s != TREVS_OK) return s;
  PreTotals tp;
  InTotals ti;
  s = validate_pre_batch(pre, tp);
  if (s != TREVS_OK) return s;
  s = validate_in_batch(in, ti);
  if (s != TREVS_OK) return s;
  s = validate_diversity(pre, prm);
  if (s != TREVS_OK) return s;
  const PreWs LP = pre_ws(tp.n, tp.m, tp.max_m, tp.k1, tp.max_k1, pre->d, tp.fps_pool, tp.fps_gram);
  const size_t pre_bytes = pre->B > 0 ? al256(LP.end) : 0;
  const InWs LI = in_ws(ti.l, ti.k1, ti.lk1, in->B > 0 ? in->Hq : 0, in->B);
  const size_t need = pre_bytes + (in->B > 0 ? LI.end : 0);
  s = check_ws(workspace, workspace_bytes, need);
  if (s != TREVS_OK) return s;
  uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
  const cudaStream_t st = (cudaStream_t)stream;
  if (pre->B > 0 && in->B > 0 && pre->B <= kMaxChunk && in->B <= kMaxChunk) {
    AuxStream* aux = nullptr;
    TREVS_TRY_CUDA(aux_stream(aux), "auxiliary stream");
    int max_l = 0, max_k1 = 0;
    for (int b = 0; b < in->B; ++b) {
      max_l = in->reqs[b].l > max_l ? in->reqs[b].l : max_l;
      max_k1 = in->reqs[b].k1 > max_k1 ? in->reqs[b].k1 : max_k1;
    }
    const int reserve = overlap_reserve(pre, in, tp, in_small_fits(in->Hq, max_l, max_k1));
    // Once work has forked onto the auxiliary stream it is joined back into `stream` on every
    // return, errors included, so that a stream capture never ends with an unjoined branch
    // and `stream` stays ordered after everything the call enqueued.
    bool forked = false;
    auto joined = [&](trevs_status status) -> trevs_status {
      if (!forked) return status;
      const cudaError_t e1 = cudaEventRecord(aux->join, aux->stream);
      const cudaError_t e2 = e1 == cudaSuccess ? cudaStreamWaitEvent(st, aux->join, 0) : e1;
      if (status == TREVS_OK && e2 != cudaSuccess) return cuda_fail(e2, "join");
      return status;
    };
    if (reserve > 0) {
      // One chunk each, and the stages are independent. The scoring grid leaves `reserve`
      // SMs free; stage 2 launches right behind it on the same stream (programmatic launch,
      // its attention grid never waits for the scoring grid), so its blocks take the free SMs
      // while the grid streams Z. The finishing grid and gather of stage 1 follow the scoring
      // grid's completion on the auxiliary stream, which joins back at the end.
      s = run_pre_chunk(pre, prm, 0, pre->B, 0, 0, 0, ws, LP, st, nullptr, aux->fork, nullptr, aux->stream,
                        reserve, &forked);
      if (s != TREVS_OK) return joined(s);
      s = run_in_chunk(in, 0, in->B, 0, 0, 0, ws + pre_bytes, LI, st, false, nullptr, true, true);
      return joined(s);
    }
    // One chunk each. The stages are independent, but the scoring grid fills every SM; stage
    // 2 (with its own compaction) forks once that grid is enqueued, so it waits for it to
    // finish and then runs beside the finishing grid and gather of stage 1.
    s = run_pre_chunk(pre, prm, 0, pre->B, 0, 0, 0, ws, LP, st, nullptr, aux->fork);
    if (s != TREVS_OK) return s;
    TREVS_TRY_CUDA(cudaStreamWaitEvent(aux->stream, aux->fork, 0), "fork");
    forked = true;
    s = run_in_chunk(in, 0, in->B, 0, 0, 0, ws + pre_bytes, LI, aux->stream, false, nullptr, true);
    return joined(s);
  }
  if (pre->B > 0) {
    s = run_pre_batch(pre, prm, ws, LP, st);
    if (s != TREVS_OK) return s;
  }
  if (in->B > 0) return run_in_batch(in, ws + pre_bytes, LI, st);
  return TREVS_OK;
}

}  // extern "C"
