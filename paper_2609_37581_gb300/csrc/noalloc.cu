// Stage-2 selection that allocates nothing: the scratch memory of trevs_in_llm_select lives
// in a fixed array in the library's device image instead of a caller-provided workspace.
//
// Some callers cannot obtain device memory when they call in: a serving loop whose memory
// budget is fixed at start-up and that must not grow or fragment the allocator's pool, an
// allocator that forbids cudaMalloc after warm-up (cudaMalloc and cudaFree may also
// synchronise the device, which a latency-bound loop cannot afford), or glue code in another
// language runtime that holds no device allocator at all. They can still pass their inputs
// and outputs; this entry point needs nothing else.
#include <mutex>

#include "in_llm.cuh"
#include "trevs.h"

namespace trevs {

cudaError_t launch_in_token_score(const InMeta&, const InArgs&, int max_k1, cudaStream_t);
trevs_status record_error(trevs_status s, const char* msg);
void record_launches(int n);

namespace {

// Layout of the fixed scratch, in 32-bit words: the token scores p (atomicMax target, cleared
// by every call), the per-request ticket of the selecting block, and room for the selection
// keys / flags. The token-score kernel keeps keys and flags in global memory only when its
// dynamic shared memory is smaller than 5 K1 bytes; launch_in_token_score asks for
// 5 K1 + 16 bytes, so with that sizing the keys / flags region is never touched. It stays as
// a guard: the kernel's pointers must stay valid should the shared-memory sizing change.
constexpr int kMaxK1 = TREVS_MAX_STAGE2_TOKENS;
constexpr int kOffP = 0;
constexpr int kOffTicket = kMaxK1;
constexpr int kOffKeys = kOffTicket + 64;
constexpr int kOffFlags = kOffKeys + kMaxK1 + 8;
constexpr int kWords = kOffFlags + (kMaxK1 + 8) / 4 + 8;

// Every GPU that loads the library holds this array (about 20 KB) until the process exits.
static __device__ __align__(256) uint32_t g_select_scratch[kWords];

// Device address of g_select_scratch on each device, resolved once with that device current.
uint32_t* scratch_on_device(cudaError_t& err) {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static uint32_t* addr[kMaxDevices] = {nullptr};
  int dev = 0;
  err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= kMaxDevices) {
    err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_select_scratch);
    if (err != cudaSuccess) return nullptr;
    addr[dev] = static_cast<uint32_t*>(p);
  }
  return addr[dev];
}

}  // namespace
}  // namespace trevs

using namespace trevs;

extern "C" {

trevs_status trevs_in_llm_select_noalloc(const float* u, const float* attn, int32_t Hq, int32_t L, int32_t K1,
                                         int32_t n_keep_heads, int32_t K2, int32_t* heads_out, float* p_out,
                                         int32_t* kept_local, void* stream) {
  record_launches(0);
  auto fail = [](trevs_status s, const char* msg) { return record_error(s, msg); };
  if (Hq < 1 || n_keep_heads < 1 || n_keep_heads > Hq || L < 1 || K1 < 1 || K2 < 0 || K2 > K1)
    return fail(TREVS_ERR_INVALID_ARGUMENT, "need Hq, L, K1 >= 1, 1 <= n_keep_heads <= Hq, 0 <= K2 <= K1");
  if (Hq > TREVS_MAX_HEADS) return fail(TREVS_ERR_UNSUPPORTED, "Hq above TREVS_MAX_HEADS");
  if (K1 > kMaxK1)
    return fail(TREVS_ERR_UNSUPPORTED,
                "K1 above the fixed scratch of the allocation-free entry point (TREVS_MAX_STAGE2_TOKENS)");
  if (!u || !attn || (K2 > 0 && !kept_local)) return fail(TREVS_ERR_INVALID_ARGUMENT, "u, attn and kept_local needed");
  cudaError_t e = cudaSuccess;
  uint32_t* scratch = scratch_on_device(e);
  if (!scratch) return fail(TREVS_ERR_CUDA, cudaGetErrorString(e));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  static thread_local InMeta meta;   // about 10 KB: kept off the host stack
  meta.B = 1;
  meta.r[0] = InReq{0, 0, L, 0, K1, 0, K2, 0, 0};
  meta.total_hs = 0;
  meta.total_ts = ((L + kScoreTextRows - 1) / kScoreTextRows) * ((K1 + kKeyBlock - 1) / kKeyBlock);
  InArgs a;
  memset(&a, 0, sizeof(a));
  a.Hq = Hq;
  a.n_keep = n_keep_heads;
  a.attn = const_cast<float*>(attn);
  a.stats_ld = L;
  a.u = const_cast<float*>(u);
  a.u_ld = Hq;
  a.p_bits = p_out ? reinterpret_cast<uint32_t*>(p_out) : scratch + kOffP;
  a.kept_local = kept_local;
  a.heads_out = heads_out;
  a.keys = scratch + kOffKeys;
  a.flags = reinterpret_cast<uint8_t*>(scratch + kOffFlags);
  a.cnt_ts = scratch + kOffTicket;
  a.cnt_hs = scratch + kOffTicket + 32;
  // the scores start at zero (atomicMax) and so does the ticket: clear both on every call
  e = cudaMemsetAsync(a.p_bits, 0, 4 * (size_t)K1, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(scratch + kOffTicket, 0, 4 * 64, st);
  if (e == cudaSuccess) e = launch_in_token_score(meta, a, K1, st);
  if (e != cudaSuccess) return fail(TREVS_ERR_CUDA, cudaGetErrorString(e));
  record_launches(3);
  return TREVS_OK;
}

}  // extern "C"
