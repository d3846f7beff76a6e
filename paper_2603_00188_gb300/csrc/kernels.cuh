// Internal launch interface between the C ABI (api.cu) and the kernels.
// Every launcher enqueues on `st` and returns the launch status.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace stl {

enum DType { kBF16 = 0, kF32 = 1 };

struct Problem {
  int n;       // tokens
  int hq;      // query heads
  int hkv;     // KV heads
  int w;       // window queries
  int dtype;   // DType
  __host__ __device__ int G() const { return hq / hkv; }
  __host__ __device__ int R() const { return w * (hq / hkv); }  // query rows per KV head
};

// ---- workspace plan (byte offsets into the caller's workspace) ----------
struct WsPlan {
  size_t err;        // uint32 error word
  size_t rn;         // float [Hkv][N] inverse key norms
  size_t rowpart;    // float2 [Hkv][nsplit][R] partial (max, sum) per query row
  size_t a_base;     // float [Hkv][N]
  size_t phi;        // float [Hkv][N]
  size_t rho;        // float [Hkv][N]
  size_t rho_part;   // float [nchunk][Hkv][N]
  size_t tau;        // float [Hkv]
  size_t gate;       // uint8 [Hkv][N]
  size_t score;      // float [Hkv][N]
  size_t total;
  int nsplit;        // key splits of the row-statistics pass
  int nchunk;        // current-frame column chunks of the TSG pass
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
cudaError_t launch_inv_norms(const Problem& p, const void* k, float* rn, cudaStream_t st);

// bias[h][r] = -m_r - log2(G l_r) from the per-split row statistics.
cudaError_t launch_row_bias(const Problem& p, const float2* part, int nsplit, float* bias,
                            cudaStream_t st);

// Window score: row statistics then column sums (Eq. 2).
cudaError_t launch_score(const Problem& p, const void* q, const void* k, float2* rowpart,
                         int nsplit, float* a_base, uint32_t* err, cudaStream_t st);

// TSG partial row maxima: rho_part[c][h][i] = max_{j in chunk c} k_i.k_j * rn_j
// for historical visual tokens i (Eq. 6 before the 1/|k_i| factor).
cudaError_t launch_tsg(const Problem& p, const FrameTable& ft, const void* k, const float* rn,
                       float* rho_part, int nchunk, uint32_t* err, cudaStream_t st);

// CSS saliency Phi (Eqs. 4-5) of every visual token; also writes the
// inverse key norms rn of every visual token.  Text entries are not touched.
cudaError_t launch_css(const Problem& p, const FrameTable& ft, const void* k, float* phi, float* rn,
                       cudaStream_t st);
// phi[h][j] = NaN for every text token j.
cudaError_t launch_fill_text_nan(const Problem& p, const FrameTable& ft, float* phi, cudaStream_t st);
// Largest N the selection kernel handles.
int select_max_tokens();

// Selection: mode bit 1 = finish rho, tau and gate (Eqs. 6-8); mode bit 2 =
// integrated score and top-B (Eq. 9, Sec. 2.1).
constexpr int kSelGate = 1;
constexpr int kSelTopk = 2;
struct SelectArgs {
  int mode;
  int budget;
  int nchunk;
  int tsg_enable;
  int css_enable;
  float alpha;
  const float* rho_part;  // [nchunk][Hkv][N]
  const float* rn;        // [Hkv][N]
  float* rho;             // out [Hkv][N]
  float* tau;             // out [Hkv]
  uint8_t* gate;          // out (kSelGate) / in (kSelTopk, nullable) [Hkv][N]
  const float* a_base;    // [Hkv][N]
  const float* phi;       // [Hkv][N] (nullable if !css_enable)
  float* score;           // out [Hkv][N]
  int32_t* idx;           // out [Hkv][budget]
};
cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a,
                          cudaStream_t st);

cudaError_t launch_gather(const Problem& p, int budget, const int32_t* idx, const void* k,
                          const void* v, void* k_out, void* v_out, cudaStream_t st);

// Tensor-core (tcgen05) paths for bf16; return cudaErrorNotSupported when the
// shape is outside what they handle.
cudaError_t launch_score_umma(const Problem& p, const void* q, const void* k, float2* rowpart,
                              int nsplit, float* a_base, uint32_t* err, cudaStream_t st);
cudaError_t launch_tsg_umma(const Problem& p, const FrameTable& ft, const void* k,
                            const float* rn, float* rho_part, int nchunk, uint32_t* err,
                            cudaStream_t st);
int umma_score_nsplit(const Problem& p);
int umma_tsg_nchunk(const FrameTable& ft);

}  // namespace stl
