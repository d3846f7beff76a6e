// Internal launch interface between the C ABI (api.cu) and the kernels.
// Every launcher enqueues on `st` and returns the launch status.  A launch
// covers a batch of L layers that share one frame layout (the layers of one
// model on one sequence); per-layer tensors are reached through LayerPtrs
// and per-layer workspace buffers through Strided views.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/stlite.h"
#include "common.cuh"

namespace stl {

enum DType { kBF16 = 0, kF32 = 1 };

constexpr int kMaxLayers = 32;  // layers per launch

struct Problem {
  int n;       // tokens
  int hq;      // query heads
  int hkv;     // KV heads
  int w;       // window queries
  int dtype;   // DType
  int L;       // layers in the launch
  __host__ __device__ int G() const { return hq / hkv; }
  __host__ __device__ int R() const { return w * (hq / hkv); }  // query rows per KV head
};

// Per-layer device tensors of one launch.
struct LayerPtrs {
  const void* q[kMaxLayers];
  const void* k[kMaxLayers];
  const void* v[kMaxLayers];
  void* k_out[kMaxLayers];
  void* v_out[kMaxLayers];
  int32_t* idx[kMaxLayers];
  int32_t budget[kMaxLayers];  // kept tokens per head of each layer
};

// A per-layer buffer: layer l starts `stride` bytes after layer l-1.
template <typename T>
struct Strided {
  T* base;
  size_t stride;
  __host__ __device__ T* at(int l) const {
    return reinterpret_cast<T*>(reinterpret_cast<uintptr_t>(base) + (size_t)l * stride);
  }
};
template <typename T>
inline Strided<T> strided(T* base, size_t stride) {
  Strided<T> s;
  s.base = base;
  s.stride = stride;
  return s;
}

// Shape limits shared by every entry point: STLITE_OK, or the status the
// call returns (N, heads and window within the ranges the kernels' index
// arithmetic and the selection's on-chip capacity assume).
stlite_status check_shape(const stlite_shape* s);

// ---- workspace plan (byte offsets into one layer's workspace region) ------
struct WsPlan {
  size_t err;        // uint32 error word (layer 0's is the one used)
  size_t rn;         // float [Hkv][N] inverse key norms
  size_t rn_cur;     // float [Hkv][cur_pad] inverse norms of the current frame (16-byte rows)
  size_t rowpart;    // float2 [Hkv][nsplit][R] per-split (max, sum) per query row, then float [Hkv][R]
  size_t a_base;     // float [Hkv][N]
  size_t phi;        // float [Hkv][N]
  size_t rho;        // float [Hkv][N]
  size_t rho_part;   // float [nchunk][Hkv][N]
  size_t tau;        // float [Hkv]
  size_t gate;       // uint8 [Hkv][N]
  size_t score;      // float [Hkv][N]
  size_t dots;       // float [4][Hkv][N]: E, S, SE, SW neighbour dots (tensor-core CSS)
  size_t total;      // bytes of one layer's region
  int nsplit;        // largest key-split count of the row-statistics pass
  int nchunk;        // 256-column slices of rho_part
  int cur_pad;       // current-frame length rounded up to 4
};
WsPlan plan_workspace(const Problem& p, const FrameTable& ft);

// ---- optional per-kernel timing -------------------------------------------
// While stlite_timing_enable(1) is in force, a TimingScope brackets one
// kernel launch with CUDA events recorded on the launching stream (skipped
// on a stream that is being captured into a graph).
class TimingScope {
 public:
  TimingScope(const char* name, cudaStream_t st);
  ~TimingScope();
  TimingScope(const TimingScope&) = delete;
  TimingScope& operator=(const TimingScope&) = delete;

 private:
  const char* name_;
  cudaStream_t st_;
  cudaEvent_t start_;
};

// ---- launchers ----------------------------------------------------------
// rn[l][h][j] = 1 / max(|k_l[j,h]|, 1e-8) for every token; the current
// frame's values are also written to rn_cur[l][h][j - cur_off] (row stride
// cur_pad).
cudaError_t launch_inv_norms(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> rn,
                             Strided<float> rn_cur, int cur_pad, cudaStream_t st);

// Window score (Eq. 2): row statistics then column sums.  rowpart holds, per
// layer, [Hkv][nsplit][R] float2 followed by [Hkv][R] float (row bias).
cudaError_t launch_score(const Problem& p, const LayerPtrs& io, Strided<float2> rowpart, int nsplit,
                         Strided<float> a_base, uint32_t* err, cudaStream_t st);
cudaError_t launch_score_umma(const Problem& p, const LayerPtrs& io, Strided<float2> rowpart,
                              int nsplit, Strided<float> a_base, uint32_t* err, cudaStream_t st);
// Key splits of window-score pass 1 (the partials it writes per query row);
// they depend on the shape alone, so that a layer gives the same bits alone
// or batched.  score_nsplit_max sizes the workspace.
int score_nsplit(const Problem& p);
int score_nsplit_max(const Problem& p);
// Merges pass 1's split partials into the row bias -m_r - log2(G l_r) that
// follows them in rowpart ([Hkv][R] float per layer).
void launch_row_bias(const Problem& p, int nsplit, Strided<float2> rowpart, cudaStream_t st);

// TSG partial row maxima: rho_part[l][s][h][i] = max over the current-frame
// columns of 256-column slice s of k_i.k_j * rn_j, for historical visual
// tokens i (Eq. 6 before the 1/|k_i| factor).
// metric: kTsgCosine / kTsgDot / kTsgNegL2.  The slices hold max_j of
// k_i.k_j * rn_j (cosine), k_i.k_j (dot) or 2 k_i.k_j - |k_j|^2 (negative L2);
// the selection kernel finishes rho with the row's own term.
cudaError_t launch_tsg(const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                       Strided<const float> rn, Strided<float> rho_part, int metric, uint32_t* err,
                       cudaStream_t st);
cudaError_t launch_tsg_umma(const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                            Strided<const float> rn_cur, int cur_pad, Strided<float> rho_part, int metric,
                            uint32_t* err, cudaStream_t st);

// CSS saliency Phi (Eqs. 4-5) of every visual token; also writes the inverse
// key norms of every visual token to rn (and of the current frame's to
// rn_cur, as launch_inv_norms).  Text entries are not touched.
cudaError_t launch_css(const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                       Strided<float> phi, Strided<float> rn, Strided<float> rn_cur, int cur_pad,
                       cudaStream_t st);
// Tensor-core CSS (bf16, every grid at most 127 wide): per-token squared-norm
// and E/S/SE/SW dots on the tensor cores, then Phi; writes rn and rn_cur as
// launch_css does.  with_phi = false stops after the dots (rn and rn_cur
// written), for a later launch_css_phi on the same dots.
bool css_umma_supported(const FrameTable& ft);
cudaError_t launch_css_umma(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> phi,
                            Strided<float> rn, Strided<float> rn_cur, int cur_pad, Strided<float> dE,
                            Strided<float> dS, Strided<float> dSE, Strided<float> dSW, uint32_t* err,
                            cudaStream_t st, bool with_phi = true);
// Phi of the CSS dots (the second kernel of launch_css_umma, on its own;
// the caller orders it after the dots are written).
cudaError_t launch_css_phi(const Problem& p, const FrameTable& ft, Strided<float> phi, Strided<float> rn,
                           Strided<float> rn_cur, int cur_pad, Strided<float> dE, Strided<float> dS,
                           Strided<float> dSE, Strided<float> dSW, cudaStream_t st);
// CSS over the size x size neighbourhood (size 3, 5, 7 or 9; 3 is the
// method's Moore neighbourhood) on the CUDA cores, through box sums of the
// normalised keys; any grid width.  Writes phi, rn and rn_cur as launch_css.
cudaError_t launch_css_box(const Problem& p, const FrameTable& ft, const LayerPtrs& io, int size,
                           Strided<float> phi, Strided<float> rn, Strided<float> rn_cur, int cur_pad,
                           cudaStream_t st);
// phi[h][j] = NaN for every text token j (one layer).
cudaError_t launch_fill_text_nan(const Problem& p, const FrameTable& ft, float* phi, cudaStream_t st);

// Selection: mode bit 1 = finish rho, tau and gate (Eqs. 6-8); mode bit 2 =
// integrated score and top-B (Eq. 9, Sec. 2.1).
constexpr int kSelGate = 1;
constexpr int kSelTopk = 2;
// TSG similarity (Eq. 6: cosine; dot product and negative squared L2 are the
// similarity-metric ablation).
constexpr int kTsgCosine = 0, kTsgDot = 1, kTsgNegL2 = 2;

struct SelectArgs {
  int mode;
  int budget[kMaxLayers];  // per layer
  int nchunk;
  int tsg_enable;
  int css_enable;
  float alpha;
  int tsg_metric;      // kTsgCosine / kTsgDot / kTsgNegL2: how rho is finished from the slices
  int tsg_fixed;       // 1: tau = tsg_fixed_tau instead of the adaptive select (Eq. 7)
  float tsg_fixed_tau;
  int base_uniform;    // 1: A = a_uniform for every token instead of a_base
  float a_uniform;
  int a_norm_max;      // 1: A / max_j A per head before Eq. 9
  int write_stages;    // 1: write rho, gate and score (the staged outputs); 0: only tau and the indices
  Strided<const float> rho_part;  // [nchunk][Hkv][N]
  Strided<const float> rn;        // [Hkv][N]
  Strided<float> rho;             // out [Hkv][N]
  Strided<float> tau;             // out [Hkv]
  Strided<uint8_t> gate;          // out (kSelGate) / in (kSelTopk; null base = all ones)
  Strided<const float> a_base;    // [Hkv][N]
  Strided<const float> phi;       // [Hkv][N] (null base when !css_enable)
  Strided<float> score;           // out [Hkv][N]
  int32_t* idx[kMaxLayers];       // out per layer [Hkv][budget]
};
cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a,
                          cudaStream_t st);
// Largest N the selection kernel handles.
int select_max_tokens();

// k_out[l][r][h][:] = k_l[idx[l][h][r]][h][:] and the same for v (idx, k,
// v, k_out, v_out and the budget from io).
cudaError_t launch_gather(const Problem& p, const LayerPtrs& io, cudaStream_t st);

// The identifier of the context current on this thread (0 if none is):
// caches of per-context handles compare it to tell a context re-created
// (cudaDeviceReset, another context made current) from the one they saw.
cudaError_t current_ctx_id(unsigned long long* out);

// 3-D TMA map (d, head, row) over a bf16 [n][hkv][128] tensor with boxes of
// 64 x 1 x rows and the 128-byte swizzle.
cudaError_t make_row_map(CUtensorMap* m, const void* base, int n, int hkv, int rows);

// ---- prompt-wide base scores (base-scoring ablation) -----------------------
// a_out [hkv][n] fp32 = the full-attention base (mode 0) or the Mean
// Attention base (mode 1) of the nq prompt rows q [nq][hq][128] (the last nq
// positions, causal) over k [n][hkv][128], bf16 (tensor cores) or fp32 (CUDA
// cores).  bias: prompt_bias_bytes of scratch (per-row softmax statistics).
size_t prompt_bias_bytes(int n, int nq, int hq, int hkv);
cudaError_t launch_prompt_score(DType dt, const void* q, const void* k, int n, int nq, int hq, int hkv, int mode,
                                float* a_out, float* bias, uint32_t* err, cudaStream_t st);

// ---- fixed scratch of stlite_score_noalloc ---------------------------------
// Device address of that array's error word on the current device (and
// context), resolved as stlite_score_noalloc does.
cudaError_t noalloc_error_word(uint32_t** word);

// ---- consumer: decode attention over a (compressed) cache -----------------
constexpr int kDecMaxG = 16;  // query heads per KV head
// Per-layer tensors of one decode launch (up to kMaxLayers layers).
struct DecBatch {
  const void* q[kMaxLayers];  // [w][hq][128]
  const void* k[kMaxLayers];  // [n][hkv][128]
  const void* v[kMaxLayers];
  float* out[kMaxLayers];     // [w][hq][128] fp32
};
// Cache splits per (layer, KV head, query row): one layer fills one wave;
// a batch of layers takes the count that fills whole waves best.
int decode_splits(int n, int hkv, int w, int layers);
size_t decode_workspace_bytes(int n, int hq, int hkv, int w, int layers);
// Every layer of the batch: out = attention of q over (k, v), dtype dt.
cudaError_t launch_decode(DType dt, const DecBatch& b, int layers, int n, int hq, int hkv, int w, void* ws,
                          cudaStream_t st);

}  // namespace stl
