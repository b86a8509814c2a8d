/*
 * trevs.h — C ABI of the GB300 (sm_103a) TReVS visual-token pruning library.
 *
 * TReVS prunes the visual tokens of a vision-language model in two stages:
 *   Stage 1 (pre-LLM, Sec. 4.1): score every projected visual token by its
 *     rectified-cosine textual relevance to the query (Eq. 4-5), combine it with
 *     the vision encoder's [CLS] saliency (Eq. 3) — by the Sec. 3.1 budget split
 *     ("textual ratio") or by the MAD-normalised fused score (Eq. 6-7) — keep the
 *     top K1 tokens and gather their feature rows in their original order.
 *   Stage 2 (in-LLM at layer l*, Sec. 4.2): compute the text-to-vision
 *     attention of every head, rank the heads by attention variance (Eq. 8),
 *     keep the high-variance heads H*, score each visual token by the max over
 *     text rows of the H*-averaged attention (Eq. 9), keep the top K2 and
 *     compact the hidden-state and K/V rows of that layer.
 *
 * Conventions for every entry point:
 *   - Tensor pointers are DEVICE memory owned by the caller. bfloat16 tensors are
 *     passed as their 16-bit patterns (uint16_t). Rows are addressed through the
 *     strides given (in elements); rows must start on 16-byte boundaries, so
 *     bf16 base pointers must be 16-byte aligned and bf16 strides multiples of 8.
 *   - The library never allocates or frees, and only trevs_workspace_status synchronises. Every call is
 *     asynchronous on `stream` (a cudaStream_t; NULL = legacy default stream).
 *     Scratch memory comes from a caller-provided workspace of at least the
 *     size the matching *_workspace_size() function returns, 256-byte aligned.
 *     A workspace must be zero-filled before its first use (trevs_workspace_init
 *     or cudaMemsetAsync); every completed call leaves its counters at zero
 *     again. After a non-OK status the workspace must be re-initialised.
 *     Calls that share a workspace must not overlap on the GPU.
 *   - All index outputs are int32, request-local, in ascending order (which is
 *     the original token order). Ties in any TopK go to the lower index.
 *   - Every argument is validated on the host before any launch; invalid
 *     arguments return TREVS_ERR_INVALID_ARGUMENT and launch nothing. Inputs must
 *     be finite. The thread-local trevs_last_error_string() explains the last
 *     non-OK status.
 *   - No exceptions cross this boundary.
 */
#ifndef TREVS_H
#define TREVS_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define TREVS_API __attribute__((visibility("default")))
#else
#define TREVS_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum trevs_status {
  TREVS_OK = 0,
  TREVS_ERR_INVALID_ARGUMENT = 1, /* bad size, null or misaligned pointer, K > N, ... */
  TREVS_ERR_WORKSPACE = 2,        /* workspace missing, misaligned or too small */
  TREVS_ERR_CUDA = 3,             /* a CUDA launch or runtime call failed */
  TREVS_ERR_UNSUPPORTED = 4,      /* valid but outside the library's limits (see below) */
  TREVS_ERR_TIMEOUT = 5           /* a bounded device-side wait gave up */
} trevs_status;

/* Selection rule of stage 1. */
enum {
  TREVS_SELECT_RATIO = 0, /* Sec. 3.1: K_t = floor(r*K1 + 1/2) tokens by textual relevance,
                             K1 - K_t by saliency; saliency top first, textual top over the
                             remaining tokens; both rank the raw scores. */
  TREVS_SELECT_FUSED = 1  /* Eq. 6-7: s = max(shat_v, shat_t) + lambda*sqrt(shat_v*shat_t),
                             shat_c = [(s_c - Med)/(MAD + eps)]_+ / tau_c, then TopK(s, K1).
                             Med is the lower median (rank floor((N-1)/2) ascending). */
};

/* Stage-1 hyper-parameters (Eq. 6-7; defaults from the paper's implementation details). */
typedef struct trevs_pre_params {
  float tau_v;         /* saliency temperature, default 1.4 */
  float tau_t;         /* textual temperature, default 1.0 */
  float lambda;        /* consistency-reward weight, default 1.0 */
  float eps;           /* MAD stabiliser, default 1e-6 (the paper leaves it unstated) */
  int32_t select_mode; /* TREVS_SELECT_RATIO (default) or TREVS_SELECT_FUSED */
  float diversity;     /* share rho of K1 drawn by farthest point sampling (Sec. 3.1 context
                          preservation): K_d = floor(rho*K1 + 1/2) tokens join the K1 - K_d
                          pivots of the rule above; the paper's K_r:K_d = 3:1 is 0.25.
                          Default 0 (no draws). Batched calls only. */
} trevs_pre_params;

/* Limits of the library (TREVS_ERR_UNSUPPORTED beyond them). */
#define TREVS_MAX_TEXT_TOKENS 256    /* M per request, stage 1 */
#define TREVS_HEAD_DIM 128           /* d_h, stage 2 */
#define TREVS_MAX_STAGE2_TOKENS 2048 /* K1 per request entering stage 2 */
#define TREVS_MAX_HEADS 128          /* Hq */

/* Fills *p with the defaults above. */
TREVS_API void trevs_pre_params_default(trevs_pre_params* p);

/* Library version string ("major.minor.patch"). */
TREVS_API const char* trevs_version(void);

/* Thread-local, human-readable reason for the last non-OK status of this thread. */
TREVS_API const char* trevs_last_error_string(void);

/* Number of kernels (and memsets) the last call on this thread enqueued. */
TREVS_API int32_t trevs_last_launch_count(void);

/* Reads the device status word at the start of a workspace and waits for `stream` to get
 * there (the one call of this library that synchronises). TREVS_OK, or TREVS_ERR_TIMEOUT
 * if a bounded device-side wait of a call that used this workspace gave up since the
 * workspace was last zero-filled, or TREVS_ERR_INVALID_ARGUMENT if farthest point sampling
 * found fewer candidates than draws (inputs that break its documented preconditions). */
TREVS_API trevs_status trevs_workspace_status(const void* workspace, size_t bytes, void* stream);

/* Zero-fills `bytes` of workspace on `stream` (cudaMemsetAsync). */
TREVS_API trevs_status trevs_workspace_init(void* workspace, size_t bytes, void* stream);

/* Test hooks of the failure paths; neither has a counterpart in the paper, and neither faults,
 * traps or hangs the GPU.
 * trevs_workspace_set_wait_limit: every bounded device-side wait of the calls that use this
 *   workspace gives up after `microseconds` instead of 2 s (0 restores 2 s); a wait that gives
 *   up makes its kernel stop, let its copies in flight land, release what it holds and set the
 *   status word (trevs_workspace_status then reports TREVS_ERR_TIMEOUT). The limit lives in the
 *   workspace header (written on `stream`), so trevs_workspace_init clears it.
 * trevs_test_fail_launch: the n-th kernel launch attempt of this host thread from now on fails
 *   without launching, as if the launch had failed (TREVS_ERR_CUDA); n <= 0 disarms it. */
TREVS_API trevs_status trevs_workspace_set_wait_limit(void* workspace, size_t bytes, uint32_t microseconds,
                                            void* stream);
TREVS_API void trevs_test_fail_launch(int32_t n);

/* ===================================================================== stage 1, one request
 *
 * Z   [N, d] bf16, row r at Z + r*z_row_stride   projected visual features z_i (Sec. 4.1)
 * T   [M, d] bf16, row j at T + j*t_row_stride   query text embeddings t_j     (Sec. 4.1)
 * s_v [N] float32                                [CLS] saliency s^v_i          (Eq. 3)
 */

/* Eq. 2-3, the vision encoder's [CLS] saliency for a batch of B requests:
 *   s_v[i] = (1/H) sum_h Softmax_i(q_h . k_{i,h} * scale) over the n[b] patch keys of request b,
 * scale = `scale` if > 0, else 1/sqrt(d_h). q_cls holds the [CLS] query of every head, element
 * (b, h, c) at q_cls + b*q_req_stride + h*q_head_stride + c; K_v the patch keys of the
 * penultimate ViT layer, packed over the requests, element (i, h, c) at
 * K_v + i*k_tok_stride + h*k_head_stride + c; s_v [sum n] float32 receives the saliency,
 * ready for the stage-1 calls. n is a host array [B]. Limits: d_h in {32, 64, 128},
 * H <= TREVS_MAX_HEADS, n[b] <= 16384. The softmax spans the patch keys only, as Eq. 2
 * writes it. */
TREVS_API size_t trevs_cls_saliency_workspace_size(int32_t B, const int32_t* n, int32_t H);
TREVS_API trevs_status trevs_cls_saliency_varlen(const uint16_t* q_cls, int64_t q_req_stride, int64_t q_head_stride,
                                       const uint16_t* K_v, int64_t k_tok_stride, int64_t k_head_stride,
                                       int32_t B, const int32_t* n, int32_t H, int32_t d_h, float scale,
                                       float* s_v, void* workspace, size_t workspace_bytes, void* stream);

/* Workspace bytes for trevs_pre_llm_scores / trevs_pre_llm_select on one request of N tokens. */
TREVS_API size_t trevs_pre_llm_workspace_size(int32_t N);

/* Eq. 4-5: s_t_out[i] = sqrt((1/M) sum_j max(cos(t_j, z_i), 0)^2) for i < N (a zero-norm
 * row has cosine 0). If s_fused_out is non-NULL, also writes the Eq. 6-7 fused score of
 * every token using s_v and *p (p may be NULL for the defaults; s_v may be NULL when
 * s_fused_out is NULL). Limits: 1 <= M <= TREVS_MAX_TEXT_TOKENS, d % 8 == 0. */
TREVS_API trevs_status trevs_pre_llm_scores(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                                  const uint16_t* T, int64_t t_row_stride, int32_t M,
                                  const float* s_v, const trevs_pre_params* p,
                                  float* s_t_out, float* s_fused_out,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* Stage-1 selection of K1 of the N tokens, written to kept_idx[0..K1) ascending.
 * Ratio mode (Sec. 3.1) reads s_v, s_t and textual_ratio in [0, 1]. Fused mode (Eq. 6-7)
 * reads s_fused when non-NULL, else computes it from s_v and s_t with *p.
 * 0 <= K1 <= N. */
TREVS_API trevs_status trevs_pre_llm_select(const float* s_v, const float* s_t, const float* s_fused,
                                  int32_t N, int32_t K1, float textual_ratio,
                                  const trevs_pre_params* p, int32_t* kept_idx,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* Z_out[k] = Z[kept_idx[k]] for k < K1 (d bf16 per row): the kept rows, in order, that are
 * passed into the LLM (Sec. 4.1). A kept_idx[k] outside [0, N) leaves row k untouched. */
TREVS_API trevs_status trevs_pre_llm_gather(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                                  const int32_t* kept_idx, int32_t K1,
                                  uint16_t* Z_out, int64_t z_out_row_stride, void* stream);

/* Workspace bytes for trevs_pre_llm_fps on one request of N tokens of width d with K_r pivots. */
TREVS_API size_t trevs_pre_llm_fps_workspace_size(int32_t N, int32_t K_r, int32_t d);

/* Sec. 3.1 context preservation: S_d = FPS({z_i | i in C}, K_d), the K_d diversity tokens
 * drawn by farthest point sampling in cosine distance from the candidates C = [N] minus the
 * pivots S_r = pivots[0..K_r) (request-local rows of Z, any order; device memory).
 * Each draw takes the candidate whose smallest distance 1 - cos(z_i, z_s) to the tokens
 * selected so far (the pivots and the earlier draws) is largest, ties to the lower index;
 * a zero row has cosine 0 with everything. With K_r = 0 the first draw is row 0.
 * picks[0..K_d) receives the draws in the order they are made (the one index output of this
 * library that is not ascending) and pick_dist[0..K_d), if non-NULL, the distance of each
 * draw when made (+inf for the first draw without pivots). `pool` is the number of
 * candidates whose pairwise cosines are kept on chip (0: automatic; at most 128); the draws
 * do not depend on it beyond rounding. A pivot outside [0, N) reads as a zero row and
 * excludes nothing. Limits: K_r + K_d <= N, d % 8 == 0 (more than TREVS_MAX_TEXT_TOKENS pivots
 * take one more pass over Z per TREVS_MAX_TEXT_TOKENS pivots). */
TREVS_API trevs_status trevs_pre_llm_fps(const uint16_t* Z, int64_t z_row_stride, int32_t N, int32_t d,
                               const int32_t* pivots, int32_t K_r, int32_t K_d, int32_t pool,
                               int32_t* picks, float* pick_dist,
                               void* workspace, size_t workspace_bytes, void* stream);

/* ===================================================================== stage 2, one request
 *
 * Q  text queries at layer l*: element (h, q, c) at Q + h*q_head_stride + q*q_tok_stride + c,
 *    h < Hq, q < L, c < d_h.
 * K  visual keys at l*: element (g, i, c) at K + g*k_head_stride + i*k_tok_stride + c,
 *    g < Hkv, i < K1. Query head h reads key head floor(h*Hkv/Hq) (grouped-query attention).
 * The attention A^h[q, i] = softmax over the K1 visual keys of (Q_h[q] . K_g[i]) * scale,
 * scale = softmax_scale if > 0 else 1/sqrt(d_h) (Sec. 4.2).
 * Full-sequence variant (optional): lse_other[h, q] is the natural log of
 * sum_j exp((Q_h[q] . k_j) * scale) over the keys of row q that are not visual (system and
 * text tokens, as the LLM's own softmax spans them). When given, the denominator of row (h, q)
 * also counts that mass, so the row sums to less than 1, and Eq. 8 takes the variance about
 * the row's own mean (its visual mass / K1). -inf means no other mass (the plain softmax).
 * attn [Hq][L][K1] float32 (dense): A^h[q, i] at attn[(h*L + q)*K1 + i].
 */

/* Workspace bytes for trevs_in_llm_head_scores / trevs_in_llm_select on one request. */
TREVS_API size_t trevs_in_llm_workspace_size(int32_t Hq, int32_t L, int32_t K1);

/* Eq. 8: u_out[h] = (1/L) sum_q Var_i A^h[q, i] (population variance over the K1 keys), and
 * the attention probabilities in attn_out (layout above). lse_other (NULL: plain softmax over
 * the visual keys) is the full-sequence variant above, [Hq][L] float32, element (h, q) at
 * lse_other[h*L + q]. Limits: d_h == TREVS_HEAD_DIM, 1 <= K1 <= TREVS_MAX_STAGE2_TOKENS,
 * 1 <= Hq <= TREVS_MAX_HEADS, Hq % Hkv == 0, L >= 1. */
TREVS_API trevs_status trevs_in_llm_head_scores(const uint16_t* Q, int64_t q_head_stride, int64_t q_tok_stride,
                                      const uint16_t* K, int64_t k_head_stride, int64_t k_tok_stride,
                                      int32_t Hq, int32_t Hkv, int32_t L, int32_t K1, int32_t d_h,
                                      float softmax_scale, const float* lse_other, float* u_out, float* attn_out,
                                      void* workspace, size_t workspace_bytes, void* stream);

/* H* = the n_keep_heads heads of largest u (ties to the lower head), written ascending to
 * heads_out (may be NULL); Eq. 9 token scores p_i = max_q (1/|H*|) sum_{h in H*} A^h[q, i]
 * (written to p_out[0..K1) when non-NULL); kept_local[0..K2) = TopK(p, K2) ascending.
 * u and attn are the outputs of trevs_in_llm_head_scores. 1 <= n_keep_heads <= Hq,
 * 0 <= K2 <= K1. */
TREVS_API trevs_status trevs_in_llm_select(const float* u, const float* attn, int32_t Hq, int32_t L, int32_t K1,
                                 int32_t n_keep_heads, int32_t K2, int32_t* heads_out,
                                 float* p_out, int32_t* kept_local,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Eq. 1 (Sec. 3.2), textual sensitivity of every head, a diagnostic of how much a head's
 * visual attention moves with the question: for two questions about the same K1 visual tokens,
 * attn1 [Hq][L1][K1] and attn2 [Hq][L2][K1] (float32, the layout trevs_in_llm_head_scores
 * writes), s_h^(x) = (1/L_x) sum_q A_x^h[q, :] and
 *   ts_out[h] = 1 - cos(s_h^(1), s_h^(2))   (a zero distribution has cosine 0).
 * s1_out / s2_out [Hq][K1] (either may be NULL) receive the head-mean distributions. Workspace:
 * trevs_textual_sensitivity_workspace_size(Hq, K1) bytes, zero-filled before first use (its
 * tickets reset themselves). Limits: Hq <= 65535. */
TREVS_API size_t trevs_textual_sensitivity_workspace_size(int32_t Hq, int32_t K1);
TREVS_API trevs_status trevs_textual_sensitivity(const float* attn1, int32_t L1, const float* attn2, int32_t L2,
                                       int32_t Hq, int32_t K1, float* ts_out, float* s1_out, float* s2_out,
                                       void* workspace, size_t workspace_bytes, void* stream);

/* Allocation-free form of trevs_in_llm_select: the same H*, Eq. 9 scores and TopK(p, K2),
 * with the same arguments except the workspace. The paper has no counterpart; this is for
 * callers that cannot hand the library device memory at the time of the call (a memory
 * budget fixed at start-up, an allocator closed after warm-up, glue code without a device
 * allocator). Its scratch is a fixed array inside the library's device image (about 20 KB
 * per GPU, held until the process exits), sized for K1 <= TREVS_MAX_STAGE2_TOKENS (2048);
 * a larger K1 returns TREVS_ERR_UNSUPPORTED and launches nothing. The call allocates no
 * device memory; it clears the part of the array that must start at zero (and p_out when
 * given) with stream-ordered memsets before its one kernel.
 * - The first call on each device resolves the array's address on the current device
 *   (cudaGetSymbolAddress; this also loads the module). Make that first call, on every
 *   device it will be used on, before capturing the call into a CUDA graph.
 * - Every call on a device shares the one array: calls that can overlap (on different
 *   streams without ordering, from several host threads, or several instances of a graph
 *   running at once) race on it and give wrong results. Order them on one stream.
 * - Errors: TREVS_ERR_INVALID_ARGUMENT / TREVS_ERR_UNSUPPORTED before any CUDA call,
 *   TREVS_ERR_CUDA when resolving the array or enqueuing fails; message in
 *   trevs_last_error_string(). */
TREVS_API trevs_status trevs_in_llm_select_noalloc(const float* u, const float* attn, int32_t Hq, int32_t L,
                                         int32_t K1, int32_t n_keep_heads, int32_t K2,
                                         int32_t* heads_out, float* p_out, int32_t* kept_local,
                                         void* stream);

/* Compaction at l* (Sec. 4.2): for k < K2 and i = kept_local[k],
 *   hidden_out[k] = hidden[i]                       (d_model bf16 per row)
 *   K_out(g, k, :) = Kc(g, i, :), V_out(g, k, :) = Vc(g, i, :) for g < Hkv (d_h bf16 each).
 * Kc/Vc use (kv_head_stride, kv_tok_stride); K_out/V_out use (out_head_stride, out_tok_stride).
 * Any of the three tensors may be skipped by passing NULL for both its input and output. */
TREVS_API trevs_status trevs_in_llm_compact(const uint16_t* hidden, int64_t hidden_row_stride, int32_t d_model,
                                  const uint16_t* Kc, const uint16_t* Vc,
                                  int64_t kv_head_stride, int64_t kv_tok_stride,
                                  int32_t Hkv, int32_t d_h, int32_t K1,
                                  const int32_t* kept_local, int32_t K2,
                                  uint16_t* hidden_out, int64_t hidden_out_row_stride,
                                  uint16_t* K_out, uint16_t* V_out,
                                  int64_t out_head_stride, int64_t out_tok_stride, void* stream);

/* ===================================================================== batched (varlen)
 *
 * A batch packs the rows of B independent requests back to back. Per-request sizes are
 * HOST arrays; row offsets are their prefix sums (request b's visual rows start at
 * sum_{b'<b} n_b', its kept rows at sum_{b'<b} k1_b', and so on). One call launches one
 * grid per step for the whole batch.
 */

typedef struct trevs_pre_request {
  int32_t n;   /* visual tokens N_b (>= 0) */
  int32_t m;   /* text tokens M_b (1..TREVS_MAX_TEXT_TOKENS when n > 0) */
  int32_t k1;  /* tokens kept by stage 1 (0..n) */
  float ratio; /* textual ratio r_b in [0, 1] (ratio mode) */
} trevs_pre_request;

typedef struct trevs_pre_batch {
  int32_t B;                       /* number of requests (>= 0) */
  int32_t d;                       /* feature width d' (% 8 == 0) */
  const trevs_pre_request* reqs;   /* host [B] */
  const uint16_t* Z;               /* [sum n, d] */
  int64_t z_row_stride;
  const uint16_t* T;               /* [sum m, d] */
  int64_t t_row_stride;
  const float* s_v;                /* [sum n] */
  float* s_t;                      /* optional output [sum n] (NULL: kept in workspace) */
  float* s_fused;                  /* optional output [sum n], fused mode only */
  int32_t* kept_idx;               /* output [sum k1], request-local, ascending per request */
  uint16_t* Z_out;                 /* output [sum k1, d] (NULL: skip the gather) */
  int64_t z_out_row_stride;
} trevs_pre_batch;

typedef struct trevs_in_request {
  int32_t k1; /* visual tokens entering stage 2 (1..TREVS_MAX_STAGE2_TOKENS) */
  int32_t l;  /* text rows at l* (>= 1) */
  int32_t k2; /* tokens kept by stage 2 (0..k1) */
} trevs_in_request;

typedef struct trevs_in_batch {
  int32_t B, Hq, Hkv, d_h, d_model, n_keep_heads;
  float softmax_scale;             /* <= 0: 1/sqrt(d_h) */
  const trevs_in_request* reqs;    /* host [B] */
  const uint16_t* Q;               /* text rows packed over requests: (h, row) at
                                      Q + h*q_head_stride + row*q_tok_stride */
  int64_t q_head_stride, q_tok_stride;
  const uint16_t* K;               /* visual rows packed: (g, row) at K + g*kv_head_stride + row*kv_tok_stride */
  const uint16_t* V;               /* same layout as K (NULL: skip V compaction) */
  int64_t kv_head_stride, kv_tok_stride;
  const uint16_t* hidden;          /* [sum k1, d_model] (NULL: skip hidden compaction) */
  int64_t hidden_row_stride;
  float* u;                        /* optional output [B, Hq] head variances (Eq. 8) */
  int32_t* heads;                  /* optional output [B, n_keep_heads] H*, ascending */
  float* p;                        /* optional output [sum k1] token scores (Eq. 9) */
  int32_t* kept_local;             /* output [sum k2], request-local, ascending */
  uint16_t* hidden_out;            /* [sum k2, d_model] */
  int64_t hidden_out_row_stride;
  uint16_t* K_out;                 /* [.., sum k2 rows] with (out_head_stride, out_tok_stride) */
  uint16_t* V_out;
  int64_t out_head_stride, out_tok_stride;
  const float* lse_other;          /* optional full-sequence variant (see stage 2 above): element
                                      (h, row) at lse_other + h*lse_head_stride + row*lse_row_stride,
                                      rows packed like Q's (NULL: plain softmax over the visual keys) */
  int64_t lse_head_stride, lse_row_stride;
} trevs_in_batch;

TREVS_API size_t trevs_pre_llm_varlen_workspace_size(const trevs_pre_batch* batch);
TREVS_API size_t trevs_in_llm_varlen_workspace_size(const trevs_in_batch* batch);
TREVS_API size_t trevs_prune_varlen_workspace_size(const trevs_pre_batch* pre, const trevs_in_batch* in);

/* Stage 1 for a batch: Eq. 4-5 scores, selection (ratio or fused, *p; NULL = defaults)
 * and gather of the kept rows. With p->diversity = rho > 0 (Sec. 3.1 context preservation)
 * the rule keeps K_r = K1 - K_d pivots (the ratio split applies to K_r), farthest point
 * sampling (as trevs_pre_llm_fps) adds K_d = floor(rho*K1 + 1/2) tokens, and kept_idx holds
 * both sets together in ascending order. The distances to the pivots take one pass over Z per
 * TREVS_MAX_TEXT_TOKENS pivots of the request with the most (the paper's K_r:K_d = 3:1 at
 * K1 = 1024 gives 768 pivots: three passes). */
TREVS_API trevs_status trevs_pre_llm_varlen(const trevs_pre_batch* batch, const trevs_pre_params* p,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* trevs_pre_llm_varlen that also times the scoring grid (Eq. 4-5) on `stream`. It has no
 * counterpart in the paper: it is a measurement hook for the kernel that dominates stage 1.
 * - ev_score_begin and ev_score_end are cudaEvent_t handles the caller created with timing
 *   enabled. The call records ev_score_begin just before the scoring grid is enqueued and
 *   ev_score_end just after it, so cudaEventElapsedTime(begin, end) spans the grid, from
 *   the completion of the pre-pass before it to the grid's own completion.
 * - Results are those of trevs_pre_llm_varlen.
 * - Limits: 1 <= B <= 256 requests (one launch chunk); a larger B returns
 *   TREVS_ERR_UNSUPPORTED, a NULL event TREVS_ERR_INVALID_ARGUMENT, before any CUDA call. */
TREVS_API trevs_status trevs_pre_llm_varlen_timed(const trevs_pre_batch* batch, const trevs_pre_params* p,
                                        void* workspace, size_t workspace_bytes, void* stream,
                                        void* ev_score_begin, void* ev_score_end);

/* Streaming probe: a measurement hook with no counterpart in the paper. One pass streams the
 * rows of Z [rows][d] (bf16, row stride z_row_stride elements) through shared memory with the
 * copies of the Eq. 4-5 scoring grid (3D TMA boxes of 8 rows x four 64-column slices, a ring
 * of two 64 KB stages per CTA, each CTA a contiguous range of 128-row x 256-column units) on
 * `ctas` CTAs of one SM each, computing nothing: each stage is released as soon as it lands.
 * Time it with events around the call on `stream`; its rate is what the scoring grid's copy
 * pattern reaches on the GPU without the grid's consumers.
 * - Z: device memory, 16-byte aligned; d a multiple of 256; z_row_stride >= d, a multiple of 8.
 * - workspace: at least 8 bytes, prepared by trevs_workspace_init; a bounded wait that gives up
 *   sets its status word (trevs_workspace_status).
 * - Invalid arguments return TREVS_ERR_INVALID_ARGUMENT before any CUDA call. */
TREVS_API trevs_status trevs_stream_probe(const uint16_t* Z, int64_t z_row_stride, int64_t rows, int32_t d,
                                          int32_t ctas, void* workspace, size_t workspace_bytes, void* stream);

/* Stage 2 for a batch: attention statistics, Eq. 8 head variances, H*, Eq. 9 token scores,
 * TopK(p, k2) and compaction of hidden, K and V rows. */
TREVS_API trevs_status trevs_in_llm_varlen(const trevs_in_batch* batch,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Both stages on independent inputs (in a model the two stages are separated by the first l*
 * LLM layers). When each stage fits one launch chunk (B <= 256), the stage-1 scoring grid
 * leaves a few SMs free and stage 2 starts beside it on `stream`; the rest of stage 1
 * runs on an internal stream forked from and joined back into `stream` with two events.
 * Larger batches run the stages one after the other. The internal stream and events are
 * created on the first call of each host thread on each device and kept for the thread's
 * life. The call stays asynchronous and can be captured into a CUDA graph. */
TREVS_API trevs_status trevs_prune_varlen(const trevs_pre_batch* pre, const trevs_pre_params* p,
                                const trevs_in_batch* in,
                                void* workspace, size_t workspace_bytes, void* stream);

/* Tuning knob of trevs_prune_varlen (no counterpart in the paper): how many SMs the scoring
 * grid leaves to stage 2 when the two stages overlap. sms < 0 (the default) restores the
 * built-in estimate, which weighs the bytes the scoring grid streams against the attention
 * work of stage 2; sms = 0 runs stage 2 after the scoring grid; larger values are clamped to
 * half the SM count. Process-wide, read at the start of each call (a captured graph keeps the
 * value of its capture). */
TREVS_API void trevs_set_overlap_reserve(int32_t sms);

#ifdef __cplusplus
}
#endif

#endif /* TREVS_H */
