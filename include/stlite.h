/*
 * stlite.h -- C ABI of libstlite.so, the GB300 (sm_103a) implementation of the
 * ST-Lite per-layer KV-cache compression pass (arXiv 2603.00188, Algorithm 1).
 *
 * One call compresses one layer of one sequence (stlite_compress_layer), a
 * batch of layers of one sequence (stlite_compress_layers), one layer of a
 * packed batch of sequences (stlite_compress_varlen), or a batch of layers of
 * a packed batch (stlite_compress_varlen_layers).  The pass has five steps:
 *   1. window scoring       A_base, Sec. 2.1 Eq. (2)
 *   2. TSG redundancy gate  rho, tau, M_time, Sec. 3.2 Eqs. (6)-(8)
 *   3. CSS saliency         Phi, Sec. 3.1 Eqs. (4)-(5)
 *   4. flat budget + top-B  S, I_keep, Sec. 2.1 and Sec. 3.3 Eq. (9)
 *   5. compaction           K' = K[I_keep], V' = V[I_keep] (Algorithm 1)
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Tensors.  Every tensor argument is a DEVICE pointer owned by the caller,
 *   16-byte aligned, densely packed in the layout given beside it:
 *     q      [w][Hq][d]        window queries (the last w query positions)
 *     k, v   [N][Hkv][d]       one layer's cached keys / values
 *     per-head outputs [Hkv][N] (float32 or uint8), idx [Hkv][B] (int32)
 *     k_out, v_out [B][Hkv][d] compacted cache
 *   Element type of q/k/v/k_out/v_out is shape->dtype (bf16 or fp32).
 *   Query head g serves KV head g / (Hq/Hkv) (grouped-query attention).
 *   Exception: v may instead be page-locked HOST memory (cudaHostAlloc,
 *   cudaMallocHost or cudaHostRegister), which kernels address directly under
 *   unified addressing.  Only the compaction reads v, and only the B kept
 *   rows per head, so values kept on the host cost B rows of host-link
 *   traffic per head instead of a copy of all N (stlite_compact,
 *   stlite_compress_layer and stlite_compress_layers).
 * Frames.  stlite_frames holds HOST arrays.  Frame f owns the contiguous
 *   visual span [offset[f], offset[f] + grid_h[f]*grid_w[f]) laid out
 *   row-major on its patch grid (u = row, v = column); frames are sorted,
 *   disjoint, inside [0, N), at most STLITE_MAX_FRAMES.  The LAST frame is the
 *   current frame; every token outside a frame is a text token.
 * Workspace.  ws is caller-allocated device memory of at least the size that
 *   stlite_workspace_size() reports for the same shape/frames/params.  It
 *   must be zero-filled before its first use (its first word is a device
 *   error word, see stlite_device_status).  Calls on one stream may share a
 *   workspace; concurrent calls on different streams need their own.
 * Streams.  `stream` is a cudaStream_t passed as void* (NULL = legacy
 *   default stream).  Every call only enqueues work: it returns after the
 *   launches, without synchronising; outputs are valid once the stream has
 *   reached that point.  No call allocates device memory.  The fused calls
 *   (stlite_compress_layer, stlite_compress_layers[_budgets],
 *   stlite_compress_varlen[_layers]) run the window score, and the last
 *   kernel of the tensor-core CSS, on a second stream beside TSG, forked from
 *   `stream` by an event and joined back into it by another before the
 *   selection, so that each call is still ordered on `stream` alone (and is
 *   captured into a graph as one fork and join).
 *   That stream (non-blocking, default priority) and its three events are
 *   created on the first fused call of each host thread on each device, and
 *   again after the device's context changed; those of the device current
 *   when the thread exits are released then (others stay until the process
 *   exits).  A call made during stream capture before them runs every stage
 *   on `stream`, as every call does while per-kernel timing is on.
 * Errors.  All arguments are validated on the host before anything is
 *   enqueued; a failed check returns STLITE_EINVAL / STLITE_EUNSUPPORTED /
 *   STLITE_EWORKSPACE and enqueues nothing.  A launch failure returns
 *   STLITE_ECUDA.  Kernels never trap: a bounded wait that runs out records
 *   STLITE_ETIMEOUT in the workspace error word, read by stlite_device_status.
 *   No call aborts the process; every call is thread-safe.
 * Numbers.  bf16 inputs are multiplied exactly and accumulated in fp32
 *   (tensor cores); fp32 inputs use fp32 FMA.  Softmax and cosines are fp32.
 */
#ifndef STLITE_H_
#define STLITE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define STLITE_API __attribute__((visibility("default")))
#else
#define STLITE_API
#endif

#define STLITE_MAX_FRAMES 256
#define STLITE_HEAD_DIM 128

typedef enum {
  STLITE_OK = 0,
  STLITE_EINVAL = 1,       /* malformed argument (null, negative, overlapping frames, ...) */
  STLITE_EUNSUPPORTED = 2, /* well-formed but outside what this build handles (d != 128, ...) */
  STLITE_EWORKSPACE = 3,   /* workspace smaller than stlite_workspace_size() */
  STLITE_ECUDA = 4,        /* a CUDA runtime call or kernel launch failed */
  STLITE_ETIMEOUT = 5      /* a kernel's bounded wait ran out (device error word) */
} stlite_status;

typedef enum { STLITE_BF16 = 0, STLITE_F32 = 1 } stlite_dtype;

typedef struct {
  int32_t n_tokens;   /* N: cached tokens of the layer, >= 1 */
  int32_t n_q_heads;  /* Hq: query heads, a multiple of n_kv_heads */
  int32_t n_kv_heads; /* Hkv: key/value heads */
  int32_t head_dim;   /* d: must be STLITE_HEAD_DIM */
  int32_t window;     /* w: observation-window queries (delta of Eq. 2), 1..256 */
  int32_t dtype;      /* stlite_dtype of q, k, v, k_out, v_out */
} stlite_shape;

typedef struct {
  int32_t n_frames;       /* F >= 0; frame F-1 is the current frame */
  const int32_t* offset;  /* host [F]: first token of each frame's visual span */
  const int32_t* grid_h;  /* host [F]: patch-grid rows (>= 1) */
  const int32_t* grid_w;  /* host [F]: patch-grid columns (>= 1) */
} stlite_frames;

/* TSG similarity (Eq. 6 uses cosine; the others are the paper's
 * similarity-metric ablation) and base scorers (Eq. 2's window score; the
 * uniform prior of the base-scoring ablation). */
typedef enum { STLITE_TSG_COSINE = 0, STLITE_TSG_DOT = 1, STLITE_TSG_NEG_L2 = 2 } stlite_tsg_metric;
typedef enum { STLITE_BASE_WINDOW = 0, STLITE_BASE_UNIFORM = 1 } stlite_base_scorer;
typedef enum { STLITE_ABASE_RAW = 0, STLITE_ABASE_MAX = 1 } stlite_abase_norm;

typedef struct {
  double beta;        /* compression ratio in (0, 1]: B = floor(beta * N) (Sec. 2.1) */
  int32_t k_override; /* > 0: use this B instead (clamped to N); 0: use beta */
  float alpha;        /* CSS weight of Eq. (9), >= 0 (paper default 1) */
  int32_t tsg_enable; /* 1: apply the TSG gate of Eq. (8); 0: M_time = 1 everywhere */
  int32_t css_enable; /* 1: add alpha * Phi (Eq. 9); 0: as alpha = 0 */
  /* Ablation variants; all zero = the method as published. */
  int32_t tsg_metric;  /* stlite_tsg_metric: rho_i = max_j of cos(k_i, k_j), k_i . k_j, or
                          -|k_i - k_j|^2 over the current frame's keys */
  int32_t tsg_fixed;   /* 0: adaptive tau of Eq. (7); 1: tau = tsg_fixed_tau for every head
                          (the fixed-threshold control: pool tokens with rho > tau are gated) */
  float tsg_fixed_tau; /* used when tsg_fixed = 1; finite */
  int32_t base_scorer; /* stlite_base_scorer: A_base of Eq. (2), or A = w/N for every token */
  int32_t abase_norm;  /* stlite_abase_norm: 0 uses A as Eq. (9) writes it; 1 divides each head's A
                          by its maximum over the N tokens first (a reading of the scale of A that
                          the paper's reported A_base values suggest) */
  int32_t css_size;    /* CSS neighbourhood k x k of Eq. (4): 0 or 3 = the 3 x 3 Moore neighbourhood;
                          5, 7 or 9 = the neighbourhood-size ablation (all in-grid cells within
                          Chebyshev distance (k-1)/2, the token itself excluded) */
} stlite_params;

/* Flat per-layer budget (Sec. 2.1, Algorithm 1 initialisation):
 * k_override > 0 ? min(k_override, N) : clamp(floor(beta * N + 1e-9), 1, N).
 * Returns -1 if N < 1 or beta is not in (0, 1] (when k_override <= 0). */
STLITE_API int32_t stlite_budget(int32_t n_tokens, double beta, int32_t k_override);

/* Bytes of workspace every call below needs for this problem. */
STLITE_API stlite_status stlite_workspace_size(const stlite_shape* shape, const stlite_frames* frames,
                                    const stlite_params* params, size_t* bytes);

/* Step 1, Eq. (2): a_base[h][j] = (1/G) sum_{g in group h} sum_{r<w}
 * softmax_j(q[r][g] . k[j][h] / sqrt(d)), all N keys, no mask.
 * a_base: device float [Hkv][N]. */
STLITE_API stlite_status stlite_score(const stlite_shape* shape, const void* q, const void* k, float* a_base,
                           void* ws, size_t ws_bytes, void* stream);

/* Step 2, Eqs. (6)-(8): for every historical visual token i (frames 0..F-2)
 * rho[h][i] = max over current-frame tokens j of cos(k_i, k_j), cos = a.b /
 * (max(|a|,1e-8) max(|b|,1e-8)); tau[h] = the min(budget, |pool|)-th smallest
 * rho; gate[h][i] = rho <= tau.  Outside the pool rho is NaN and gate is 1.
 * With F < 2 (empty pool) tau is NaN and every gate is 1.
 * rho: device float [Hkv][N]; tau: device float [Hkv]; gate: device uint8
 * [Hkv][N]; budget >= 1. */
STLITE_API stlite_status stlite_gate_frames(const stlite_shape* shape, const stlite_frames* frames,
                                 const void* k, int32_t budget, float* rho, float* tau,
                                 uint8_t* gate, void* ws, size_t ws_bytes, void* stream);

/* Step 3, Eqs. (4)-(5): for every visual token, Phi = 1 - mean cosine to its
 * in-grid 3x3 Moore neighbours in the same frame (0 when it has none); text
 * tokens get NaN.  phi: device float [Hkv][N]. */
STLITE_API stlite_status stlite_spatial_saliency(const stlite_shape* shape, const stlite_frames* frames,
                                      const void* k, float* phi, void* ws, size_t ws_bytes,
                                      void* stream);

/* Step 3 over the size x size neighbourhood (the neighbourhood-size ablation
 * of the CSS appendix): Phi = 1 - mean cosine to the in-grid cells within
 * Chebyshev distance (size-1)/2 in the same frame, the token itself
 * excluded.  size: 3, 5, 7 or 9 (3 is the method's Moore neighbourhood; this
 * entry computes it through box sums of normalised keys on the CUDA cores,
 * stlite_spatial_saliency on the tensor cores).  Any grid width.  phi as for
 * stlite_spatial_saliency; STLITE_EINVAL for another size. */
STLITE_API stlite_status stlite_spatial_saliency_size(const stlite_shape* shape, const stlite_frames* frames,
                                                      const void* k, int32_t size, float* phi, void* ws,
                                                      size_t ws_bytes, void* stream);

/* Step 4, Eq. (9) and Top_B (base_scorer = STLITE_BASE_UNIFORM replaces a_base,
 * which may then be NULL, by w/N for every token): S = a_base for text tokens, S = gate * (a_base +
 * alpha * phi) for visual tokens (phi ignored when css_enable = 0; gate may be
 * NULL = all ones); idx[h][:] = the budget tokens of largest S, equal S ranked
 * by lower index, written in ascending index order.  score_out (nullable):
 * device float [Hkv][N] receives S. */
STLITE_API stlite_status stlite_select_topk(const stlite_shape* shape, const stlite_frames* frames,
                                 const stlite_params* params, const float* a_base,
                                 const float* phi, const uint8_t* gate, int32_t budget,
                                 int32_t* idx, float* score_out, void* ws, size_t ws_bytes,
                                 void* stream);

/* Step 5: k_out[r][h][:] = k[idx[h][r]][h][:] and the same for v, bit-exact.
 * idx: device int32 [Hkv][budget].  The kernel checks every index: a row whose
 * index lies outside [0, N) is left unwritten. */
STLITE_API stlite_status stlite_compact(const stlite_shape* shape, int32_t budget, const int32_t* idx,
                             const void* k, const void* v, void* k_out, void* v_out,
                             void* stream);

/* Steps 1-5 fused for one layer (Algorithm 1).  idx_out: device int32
 * [Hkv][B] receives I_keep per head in ascending order; budget_out (nullable,
 * HOST) receives B; k_out/v_out: device [B][Hkv][d].  Runs norms, TSG (when
 * tsg_enable and F >= 2), window scoring, CSS (when css_enable), selection
 * and compaction, all on `stream`. */
STLITE_API stlite_status stlite_compress_layer(const stlite_shape* shape, const stlite_frames* frames,
                                    const stlite_params* params, const void* q, const void* k,
                                    const void* v, void* k_out, void* v_out, int32_t* idx_out,
                                    int32_t* budget_out, void* ws, size_t ws_bytes, void* stream);

/* Window score (same result as stlite_score) for callers that cannot
 * allocate device memory and so cannot provide a workspace -- for example
 * code running inside an allocator or memory-pool callback, or a process
 * whose device memory is fully reserved by another runtime.  The paper has no
 * counterpart: this is a deployment convenience.  Its scratch (an error word
 * and the per-split softmax row statistics) is one fixed 2 MiB device array
 * inside the library, which every GPU that loads the library holds until
 * exit.  A problem needs 256 + Hkv*S*w*G*8 + Hkv*w*G*4 bytes of it, where S,
 * the key splits of the first softmax pass, is at most max(4,
 * 4*ceil(304/Hkv)); a problem beyond 2 MiB is rejected with
 * STLITE_EUNSUPPORTED (checked after the shape limits of stlite_score and
 * before the pointers, so no launch is attempted).  The call allocates
 * nothing.  The array's address is resolved (cudaGetSymbolAddress) on the
 * first call on each device, and again on the first call after the current
 * context changed (cudaDeviceReset, another context made current), so make
 * that first call before any stream capture.  All calls share the array,
 * which keeps the last call's contents (each call clears its error word; the
 * statistics are fully rewritten): calls that overlap on the GPU -- issued to
 * one device on different streams, or from several threads -- race on it.
 * A bounded wait of its kernels that ran out is recorded in the array's
 * error word, which stlite_device_status(NULL, ...) reads on the current
 * device; read it before the next call clears it.
 * q, k, a_base: as for stlite_score. */
STLITE_API stlite_status stlite_score_noalloc(const stlite_shape* shape, const void* q, const void* k,
                                              float* a_base, void* stream);

/* One layer's tensors for stlite_compress_layers (all device pointers, laid
 * out as for stlite_compress_layer). */
typedef struct {
  const void* q;    /* [w][Hq][d] window queries of this layer */
  const void* k;    /* [N][Hkv][d] */
  const void* v;    /* [N][Hkv][d] */
  void* k_out;      /* [B][Hkv][d] */
  void* v_out;      /* [B][Hkv][d] */
  int32_t* idx_out; /* [Hkv][B], ascending per head */
} stlite_layer_io;

/* Algorithm 1 for n_layers layers of one sequence (one frame layout, one
 * budget), each layer compressed independently with its own window queries;
 * the result for every layer equals stlite_compress_layer's.  Each kernel
 * launch covers up to 32 layers at a time (with TSG and CSS on, eight
 * launches per batch of up to 32 layers), so small per-layer stages (the
 * selections, the compaction) fill the GPU.  layers: HOST array
 * [n_layers].  ws: n_layers times stlite_workspace_size() bytes (layer l uses
 * the l-th slice; the first word of the whole workspace is the error word).
 * budget_out (nullable, HOST) receives B. */
STLITE_API stlite_status stlite_compress_layers(const stlite_shape* shape, const stlite_frames* frames,
                                                const stlite_params* params, int32_t n_layers,
                                                const stlite_layer_io* layers, int32_t* budget_out,
                                                void* ws, size_t ws_bytes, void* stream);

/* stlite_compress_layers with a budget of its own for every layer: layer l
 * keeps budgets[l] tokens per KV head and its result equals
 * stlite_compress_layer's with k_override = budgets[l].  This is the
 * flat-versus-hierarchical ablation (appendix "CSS/TSG Interaction
 * Analysis", the budget-allocation table; Sec. 3.3 states the flat default):
 * the scoring is unchanged and only B^(l) varies across layers.  params->beta and
 * params->k_override are ignored.
 * budgets: HOST int32 [n_layers], each in [1, n_tokens]; k_out / v_out of
 *   layer l hold budgets[l] rows and idx_out [Hkv][budgets[l]].
 * Returns STLITE_EINVAL for a NULL array or an out-of-range budget, checked
 * before anything is enqueued. */
STLITE_API stlite_status stlite_compress_layers_budgets(const stlite_shape* shape, const stlite_frames* frames,
                                                        const stlite_params* params, int32_t n_layers,
                                                        const stlite_layer_io* layers, const int32_t* budgets,
                                                        void* ws, size_t ws_bytes, void* stream);

/* Hierarchical per-layer budgets from per-layer attention mass (appendix
 * "Failure Mode Derivations", F2, the noise-dominated allocation
 * proposition): B^(l) = S^(l) / sum_l' S^(l') * B_total.  The real shares
 * are made integer as the budgets in [1, n_tokens] that add up to B_total and
 * are nearest to the shares in squared distance (ties to the lower layer);
 * without clamping this is rounding by largest remainder.  Host only.
 * layer_mass: HOST [n_layers], each finite and > 0 (S^(l): e.g. the sum of a
 *   layer's window scores A_base over its heads and prefix keys).
 * total_budget: B_total in [n_layers, n_layers * n_tokens].
 * budgets: HOST int32 [n_layers] out.
 * Returns STLITE_EINVAL for invalid arguments (nothing written). */
STLITE_API stlite_status stlite_hierarchical_budgets(int32_t n_layers, const double* layer_mass, int64_t total_budget,
                                                     int32_t n_tokens, int32_t* budgets);

/* A packed batch of sequences of different lengths and frame layouts (one
 * layer): Algorithm 1 for each sequence on its own, with its own budget
 * B_s = stlite_budget(N_s, beta, k_override).
 * shape: n_tokens = the total packed length; the other fields are shared.
 * cu_seqlens: HOST int32 [n_seqs + 1], cu_seqlens[0] = 0, non-decreasing by at
 *   least 1, cu_seqlens[n_seqs] = n_tokens: sequence s owns packed tokens
 *   [cu_seqlens[s], cu_seqlens[s + 1]).
 * frames: HOST array [n_seqs]; frames[s] describes sequence s with offsets
 *   relative to the sequence's first token.
 * q: [n_seqs][w][Hq][d] (each sequence's window queries); k, v: packed
 *   [n_tokens][Hkv][d].
 * k_out, v_out: packed [sum_s B_s][Hkv][d] in sequence order; idx_out: the
 *   blocks [Hkv][B_s] of the sequences one after another (block s starts at
 *   element Hkv * sum_{r<s} B_r), indices relative to the sequence start.
 * cu_budget_out (nullable, HOST int32 [n_seqs + 1]) receives the prefix sums
 *   of B_s.  ws: at least stlite_workspace_size_varlen bytes; the sequences
 *   run one after another on `stream` and share it.  The result for each
 *   sequence equals stlite_compress_layer's on that sequence alone. */
STLITE_API stlite_status stlite_compress_varlen(const stlite_shape* shape, int32_t n_seqs,
                                                const int32_t* cu_seqlens, const stlite_frames* frames,
                                                const stlite_params* params, const void* q, const void* k,
                                                const void* v, void* k_out, void* v_out, int32_t* idx_out,
                                                int32_t* cu_budget_out, void* ws, size_t ws_bytes,
                                                void* stream);

/* stlite_compress_varlen over n_layers layers that share the packing
 * (cu_seqlens, frames): every sequence's layers run together through the
 * batched-layers path of stlite_compress_layers (each kernel launch covers up
 * to 32 layers), the sequences one after another on `stream`.  The result
 * for every layer equals stlite_compress_varlen's on that layer.
 * layers: HOST array [n_layers]; entry l holds layer l's packed tensors in
 *   the layouts of stlite_compress_varlen: q [n_seqs][w][Hq][d], k and v
 *   [n_tokens][Hkv][d], k_out and v_out [sum_s B_s][Hkv][d], idx_out the
 *   blocks [Hkv][B_s] one after another.
 * ws: n_layers times stlite_workspace_size_varlen bytes.  cu_budget_out
 *   (nullable, HOST) as for stlite_compress_varlen.
 * Every argument is checked before anything is enqueued. */
STLITE_API stlite_status stlite_compress_varlen_layers(const stlite_shape* shape, int32_t n_seqs,
                                                       const int32_t* cu_seqlens, const stlite_frames* frames,
                                                       const stlite_params* params, int32_t n_layers,
                                                       const stlite_layer_io* layers, int32_t* cu_budget_out,
                                                       void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes stlite_compress_varlen needs: the largest of the
 * sequences' stlite_workspace_size. */
STLITE_API stlite_status stlite_workspace_size_varlen(const stlite_shape* shape, int32_t n_seqs,
                                                      const int32_t* cu_seqlens, const stlite_frames* frames,
                                                      const stlite_params* params, size_t* bytes);

/* Prompt-wide base scores of the base-scoring ablation (appendix
 * "Sensitivity to the Base Attention Scoring Function"): instead of the w
 * window queries of Eq. (2), every query row of the prompt votes.  The
 * n_prompt rows q_prompt [n_prompt][Hq][d] are the queries of the last
 * n_prompt cached positions (n_prompt = N: the whole prompt); the row at
 * position p attends, as in the model's causal prefill, to the keys
 * j <= p.  With C[h][j] = (1/G) sum over the group's query heads and the
 * prompt rows of their softmax probability of key j:
 *   STLITE_PROMPT_FULL  a_base = C (the full-attention "snapshot" base);
 *   STLITE_PROMPT_MEAN  a_base = C / (number of prompt rows that attend to
 *                       j, min(n_prompt, N - j)) (Mean Attention: attention
 *                       averaged over the prompt).
 * a_base (device float [Hkv][N]) then takes the place of the window score
 * in stlite_select_topk.  bf16 caches run on the tensor cores, fp32 caches
 * on the CUDA cores; G <= 128; shape->window is not used (any valid value).
 * The work is that of the prompt's causal attention, twice (row statistics,
 * then column sums).
 * ws: at least stlite_prompt_workspace_size bytes, zero-filled before its
 * first use (its first word is the device error word of
 * stlite_device_status). */
typedef enum { STLITE_PROMPT_FULL = 0, STLITE_PROMPT_MEAN = 1 } stlite_prompt_base;
STLITE_API stlite_status stlite_prompt_score(const stlite_shape* shape, int32_t n_prompt, int32_t base,
                                             const void* q_prompt, const void* k, float* a_base, void* ws,
                                             size_t ws_bytes, void* stream);

/* Workspace bytes of stlite_prompt_score. */
STLITE_API stlite_status stlite_prompt_workspace_size(const stlite_shape* shape, int32_t n_prompt, size_t* bytes);

/* Consumer of the compressed cache: attention of query rows over a KV cache,
 * the operation a decoder runs for every generated token (the paper's
 * efficiency study compares decode latency with the full and the compressed
 * cache):  out[r][g][:] = sum_j softmax_j(q[r][g] . k[j][h] / sqrt(d)) v[j][h][:]
 * with h = g / (Hq/Hkv), over all n cached rows, no mask.
 * shape: n_tokens = cache rows n (N for the full cache, B after
 *   compaction), window = query rows w, Hq / Hkv <= 16.
 * q [w][Hq][d], k and v [n][Hkv][d] (device, shape->dtype); out: device float
 *   [w][Hq][d].  ws: at least stlite_decode_workspace_size bytes (split
 *   partials), zero-filled before its first use: its first word is the
 *   device error word that stlite_device_status reads (a bounded wait that
 *   ran out records STLITE_ETIMEOUT there). */
STLITE_API stlite_status stlite_decode_attention(const stlite_shape* shape, const void* q, const void* k,
                                                 const void* v, float* out, void* ws, size_t ws_bytes,
                                                 void* stream);

/* Workspace bytes of stlite_decode_attention for this shape. */
STLITE_API stlite_status stlite_decode_workspace_size(const stlite_shape* shape, size_t* bytes);

/* One layer's tensors for stlite_decode_attention_layers (device pointers,
 * layouts as for stlite_decode_attention). */
typedef struct {
  const void* q; /* [w][Hq][d] */
  const void* k; /* [n][Hkv][d] */
  const void* v; /* [n][Hkv][d] */
  float* out;    /* [w][Hq][d] fp32 */
} stlite_decode_io;

/* stlite_decode_attention for n_layers layers of one shape at once (the
 * decode step of a whole model over its per-layer caches): one launch of the
 * split kernel and one of the split merge per batch of up to 32 layers, the
 * splits sized so that the batch fills whole waves of the GPU.  Each layer's
 * result equals stlite_decode_attention's up to fp32 rounding (the splits
 * group the sums differently).  layers: HOST array [n_layers]; ws: at least
 * stlite_decode_layers_workspace_size bytes, zero-filled before its first
 * use (first word: the device error word). */
STLITE_API stlite_status stlite_decode_attention_layers(const stlite_shape* shape, int32_t n_layers,
                                                        const stlite_decode_io* layers, void* ws, size_t ws_bytes,
                                                        void* stream);

/* Workspace bytes of stlite_decode_attention_layers. */
STLITE_API stlite_status stlite_decode_layers_workspace_size(const stlite_shape* shape, int32_t n_layers,
                                                             size_t* bytes);

/* Reads and clears the workspace's device error word (synchronises `stream`).
 * *status receives STLITE_OK, STLITE_ETIMEOUT if a kernel's bounded wait ran
 * out since the last read, or STLITE_ECUDA if a kernel found its launch
 * configuration unusable (it then returned without touching its outputs).
 * ws = NULL reads the error word of stlite_score_noalloc's fixed scratch on
 * the current device instead. */
STLITE_API stlite_status stlite_device_status(void* ws, void* stream, stlite_status* status);

/* Diagnostic of the failure path (not part of Algorithm 1): one kernel waits,
 * through the bounded wait every tensor-core kernel of the library uses, on
 * a barrier that nothing completes.  After limit_ns (1 us .. 2 s) of
 * %globaltimer the wait gives up, records STLITE_ETIMEOUT in the workspace
 * error word and the kernel returns: stlite_device_status(ws) then reports
 * STLITE_ETIMEOUT, and the context stays usable for later calls.  Nothing
 * faults and nothing hangs.  ws: at least 16 bytes of device memory whose
 * first word is the error word (any workspace of this library qualifies). */
STLITE_API stlite_status stlite_selftest_wait_timeout(void* ws, int64_t limit_ns, void* stream);

/* Per-kernel timing (instrumentation; not part of Algorithm 1).
 * stlite_timing_enable(1) makes every later launch by this library, on a
 * stream that is not being captured into a graph, record a pair of CUDA
 * events around itself on its stream.  stlite_timing_read() waits for the
 * recorded events, writes one entry per kernel name (number of launches and
 * summed device time in ms) into `out` (up to `capacity` entries; *count
 * receives the number of distinct kernels) and clears the record.  Both are
 * process-wide and thread-safe. */
typedef struct {
  char name[32];
  int32_t launches;
  double total_ms;
} stlite_kernel_time;
STLITE_API stlite_status stlite_timing_enable(int32_t on);
STLITE_API stlite_status stlite_timing_read(stlite_kernel_time* out, int32_t capacity,
                                            int32_t* count);

/* Human-readable name of a status code (static storage). */
STLITE_API const char* stlite_status_string(stlite_status status);

#ifdef __cplusplus
}
#endif

#endif /* STLITE_H_ */
