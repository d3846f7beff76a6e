// CUDA-core kernels: inverse key norms, CSS saliency, and the fp32 versions
// of window scoring and TSG (fp32 inputs cannot use the bf16 tensor-core
// path without losing the exactness of the products).
#include "kernels.cuh"

namespace stl {

constexpr float kLog2e = 1.4426950408889634f;

// ---------------------------------------------------------------- norms
// rn[h][j] = 1 / max(|k_{j,h}|, 1e-8).  One warp per (token, head); lane l
// holds elements 4l..4l+3.
template <typename T>
__global__ void __launch_bounds__(256) k_inv_norms(const T* __restrict__ k, int n, int hkv,
                                                   float* __restrict__ rn) {
  int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (gw >= n * hkv) return;
  int j = gw / hkv, h = gw - j * hkv;
  float4 x = Elem<T>::load4(k + ((size_t)j * hkv + h) * kD + lane * 4);
  float s = warp_sum(dot4(x, x));
  if (lane == 0) rn[(size_t)h * n + j] = 1.0f / fmaxf(sqrtf(s), 1e-8f);
}

cudaError_t launch_inv_norms(const Problem& p, const void* k, float* rn, cudaStream_t st) {
  long long warps = (long long)p.n * p.hkv;
  int blocks = (int)((warps + 7) / 8);
  TimingScope ts("inv_norms", st);
  if (p.dtype == kBF16)
    k_inv_norms<<<blocks, 256, 0, st>>>((const __nv_bfloat16*)k, p.n, p.hkv, rn);
  else
    k_inv_norms<<<blocks, 256, 0, st>>>((const float*)k, p.n, p.hkv, rn);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- CSS
// Eqs. 4-5.  One warp per (token, head).  Text tokens get NaN; a visual token
// with no in-grid neighbour gets 0.
template <typename T>
__global__ void __launch_bounds__(256) k_css(const T* __restrict__ k, const float* __restrict__ rn,
                                             const __grid_constant__ FrameTable ft, int hkv,
                                             float* __restrict__ phi) {
  int n = ft.n_tokens;
  int gw_ = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (gw_ >= n * hkv) return;
  int j = gw_ / hkv, h = gw_ - j * hkv;
  int f = find_frame(ft, j);
  if (f < 0) {
    if (lane == 0) phi[(size_t)h * n + j] = CUDART_NAN_F;
    return;
  }
  int off = ft.off[f], gh = ft.gh[f], gw = ft.gw[f];
  int local = j - off, u = local / gw, v = local - u * gw;
  float4 c = Elem<T>::load4(k + ((size_t)j * hkv + h) * kD + lane * 4);
  float rc = rn[(size_t)h * n + j];
  float sum = 0.f;
  int cnt = 0;
#pragma unroll
  for (int du = -1; du <= 1; ++du) {
#pragma unroll
    for (int dv = -1; dv <= 1; ++dv) {
      if (du == 0 && dv == 0) continue;
      int pu = u + du, pv = v + dv;
      if (pu < 0 || pu >= gh || pv < 0 || pv >= gw) continue;
      int nb = off + pu * gw + pv;
      float4 x = Elem<T>::load4(k + ((size_t)nb * hkv + h) * kD + lane * 4);
      float dot = warp_sum(dot4(c, x));
      sum += dot * rc * rn[(size_t)h * n + nb];
      ++cnt;
    }
  }
  if (lane == 0) phi[(size_t)h * n + j] = cnt ? 1.0f - sum / (float)cnt : 0.0f;
}

cudaError_t launch_css(const Problem& p, const FrameTable& ft, const void* k, const float* rn,
                       float* phi, cudaStream_t st) {
  long long warps = (long long)p.n * p.hkv;
  int blocks = (int)((warps + 7) / 8);
  TimingScope ts("css", st);
  if (p.dtype == kBF16)
    k_css<<<blocks, 256, 0, st>>>((const __nv_bfloat16*)k, rn, ft, p.hkv, phi);
  else
    k_css<<<blocks, 256, 0, st>>>((const float*)k, rn, ft, p.hkv, phi);
  return cudaGetLastError();
}

// ------------------------------------------------------- row statistics
// Window score, first pass: for every query row r of KV head h (r = window
// row * G + group member) the running maximum m and sum l of
// 2^(x - m), x = q.k * log2(e)/sqrt(d), over the keys of one split.
constexpr int kRsRows = 256;   // query rows per block
constexpr int kRsKeys = 64;    // keys per smem tile
constexpr int kRsSmem = (kRsRows * (kD + 1) + kRsKeys * kD) * 4;

template <typename T>
__global__ void __launch_bounds__(kRsRows) k_rowstats_simt(const T* __restrict__ q,
                                                           const T* __restrict__ k, Problem p,
                                                           int nsplit, float2* __restrict__ part) {
  extern __shared__ float sm[];
  float* qs = sm;                       // [kRsRows][kD+1]
  float* ks = sm + kRsRows * (kD + 1);  // [kRsKeys][kD]
  const int s = blockIdx.x, h = blockIdx.y, r0 = blockIdx.z * kRsRows;
  const int G = p.G(), R = p.R(), tid = threadIdx.x;
  const float c = kLog2e * rsqrtf((float)kD);
  for (int e = tid; e < kRsRows * kD; e += blockDim.x) {
    int row = e / kD, t = e - row * kD, gr = r0 + row;
    float x = 0.f;
    if (gr < R) {
      int wr = gr / G, g = gr - wr * G;
      x = Elem<T>::load1(q + ((size_t)wr * p.hq + h * G + g) * kD + t);
    }
    qs[row * (kD + 1) + t] = x;
  }
  int per = (p.n + nsplit - 1) / nsplit;
  int j0 = s * per, j1 = min(p.n, j0 + per);
  float m = -CUDART_INF_F, l = 0.f;
  for (int jt = j0; jt < j1; jt += kRsKeys) {
    __syncthreads();
    for (int e = tid; e < kRsKeys * kD; e += blockDim.x) {
      int jj = e / kD, t = e - jj * kD;
      ks[e] = (jt + jj < j1) ? Elem<T>::load1(k + ((size_t)(jt + jj) * p.hkv + h) * kD + t) : 0.f;
    }
    __syncthreads();
    int nk = min(kRsKeys, j1 - jt);
    const float* qr = qs + tid * (kD + 1);
    for (int jj = 0; jj < nk; ++jj) {
      const float* kr = ks + jj * kD;
      float d0 = 0.f, d1 = 0.f;
#pragma unroll 16
      for (int t = 0; t < kD; t += 2) {
        d0 = fmaf(qr[t], kr[t], d0);
        d1 = fmaf(qr[t + 1], kr[t + 1], d1);
      }
      float x = (d0 + d1) * c;
      if (x > m) {
        l = l * exp2f(m - x) + 1.0f;
        m = x;
      } else {
        l += exp2f(x - m);
      }
    }
  }
  if (r0 + tid < R) part[((size_t)h * nsplit + s) * R + r0 + tid] = make_float2(m, l);
}

// Merge the splits: bias[h][r] = -m_r - log2(G * l_r), so that
// 2^(x + bias) = softmax probability / G.
__global__ void k_row_bias(const float2* __restrict__ part, Problem p, int nsplit,
                           float* __restrict__ bias) {
  int R = p.R();
  int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= p.hkv * R) return;
  int h = e / R, r = e - h * R;
  const float2* pp = part + (size_t)h * nsplit * R + r;
  float m = -CUDART_INF_F;
  for (int s = 0; s < nsplit; ++s) m = fmaxf(m, pp[(size_t)s * R].x);
  float l = 0.f;
  for (int s = 0; s < nsplit; ++s) {
    float2 v = pp[(size_t)s * R];
    if (v.y > 0.f) l += v.y * exp2f(v.x - m);
  }
  bias[e] = -m - log2f((float)p.G() * l);
}

// ---------------------------------------------------------- column sums
// Window score, second pass: a[h][j] = sum_r 2^(x_rj + bias_r).  One thread
// per key; the key tile is kept (padded) in shared memory.
constexpr int kCsKeys = 128;
constexpr int kCsRows = 32;
constexpr int kCsMaxR = 1024;
constexpr int kCsSmem = (kCsKeys * (kD + 1) + kCsRows * kD + kCsMaxR) * 4;

template <typename T>
__global__ void __launch_bounds__(kCsKeys) k_colsum_simt(const T* __restrict__ q,
                                                         const T* __restrict__ k, Problem p,
                                                         const float* __restrict__ bias,
                                                         float* __restrict__ a_base) {
  extern __shared__ float sm[];
  float* ks = sm;                            // [kCsKeys][kD+1]
  float* qs = ks + kCsKeys * (kD + 1);       // [kCsRows][kD]
  float* bs = qs + kCsRows * kD;             // [R]
  const int h = blockIdx.y, j0 = blockIdx.x * kCsKeys, tid = threadIdx.x;
  const int G = p.G(), R = p.R();
  const float c = kLog2e * rsqrtf((float)kD);
  for (int e = tid; e < kCsKeys * kD; e += blockDim.x) {
    int jj = e / kD, t = e - jj * kD;
    ks[jj * (kD + 1) + t] =
        (j0 + jj < p.n) ? Elem<T>::load1(k + ((size_t)(j0 + jj) * p.hkv + h) * kD + t) : 0.f;
  }
  for (int r = tid; r < R; r += blockDim.x) bs[r] = bias[(size_t)h * R + r];
  float acc = 0.f;
  const float* kr = ks + tid * (kD + 1);
  for (int rt = 0; rt < R; rt += kCsRows) {
    __syncthreads();
    for (int e = tid; e < kCsRows * kD; e += blockDim.x) {
      int row = e / kD, t = e - row * kD, gr = rt + row;
      float x = 0.f;
      if (gr < R) {
        int wr = gr / G, g = gr - wr * G;
        x = Elem<T>::load1(q + ((size_t)wr * p.hq + h * G + g) * kD + t);
      }
      qs[e] = x;
    }
    __syncthreads();
    int nr = min(kCsRows, R - rt);
    for (int row = 0; row < nr; ++row) {
      const float* qr = qs + row * kD;
      float d0 = 0.f, d1 = 0.f;
#pragma unroll 16
      for (int t = 0; t < kD; t += 2) {
        d0 = fmaf(kr[t], qr[t], d0);
        d1 = fmaf(kr[t + 1], qr[t + 1], d1);
      }
      acc += exp2f(fmaf(d0 + d1, c, bs[rt + row]));
    }
  }
  if (j0 + tid < p.n) a_base[(size_t)h * p.n + j0 + tid] = acc;
}

cudaError_t launch_row_bias(const Problem& p, const float2* part, int nsplit, float* bias,
                            cudaStream_t st) {
  int tot = p.hkv * p.R();
  TimingScope ts("row_bias", st);
  k_row_bias<<<(tot + 127) / 128, 128, 0, st>>>(part, p, nsplit, bias);
  return cudaGetLastError();
}

cudaError_t launch_score(const Problem& p, const void* q, const void* k, float2* rowpart,
                         int nsplit, float* a_base, uint32_t* err, cudaStream_t st) {
  (void)err;
  cudaFuncSetAttribute(k_rowstats_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kRsSmem);
  cudaFuncSetAttribute(k_rowstats_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kRsSmem);
  cudaFuncSetAttribute(k_colsum_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCsSmem);
  cudaFuncSetAttribute(k_colsum_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCsSmem);
  if (p.R() > kCsMaxR) return cudaErrorNotSupported;
  dim3 g1(nsplit, p.hkv, (p.R() + kRsRows - 1) / kRsRows);
  float* bias = reinterpret_cast<float*>(rowpart + (size_t)p.hkv * nsplit * p.R());
  dim3 g2((p.n + kCsKeys - 1) / kCsKeys, p.hkv);
  {
  TimingScope ts("rowstats_simt", st);
  if (p.dtype == kBF16) {
    k_rowstats_simt<<<g1, kRsRows, kRsSmem, st>>>((const __nv_bfloat16*)q, (const __nv_bfloat16*)k, p, nsplit, rowpart);
  } else {
    k_rowstats_simt<<<g1, kRsRows, kRsSmem, st>>>((const float*)q, (const float*)k, p, nsplit, rowpart);
  }
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if ((e = launch_row_bias(p, rowpart, nsplit, bias, st)) != cudaSuccess) return e;
  TimingScope ts("colsum_simt", st);
  if (p.dtype == kBF16) {
    k_colsum_simt<<<g2, kCsKeys, kCsSmem, st>>>((const __nv_bfloat16*)q, (const __nv_bfloat16*)k, p, bias, a_base);
  } else {
    k_colsum_simt<<<g2, kCsKeys, kCsSmem, st>>>((const float*)q, (const float*)k, p, bias, a_base);
  }
  return cudaGetLastError();
}

// ------------------------------------------------------------------ TSG
// fp32 path of Eq. 6: one thread per historical token, current-frame keys
// streamed through shared memory.  Writes chunk 0 of rho_part.
constexpr int kTsKeys = 64;
constexpr int kTsSmem = (kTsgTile * (kD + 1) + kTsKeys * kD + kTsKeys) * 4;

template <typename T>
__global__ void __launch_bounds__(kTsgTile) k_tsg_simt(const T* __restrict__ k,
                                                       const float* __restrict__ rn,
                                                       const __grid_constant__ FrameTable ft,
                                                       int hkv, float* __restrict__ rho_part) {
  extern __shared__ float sm[];
  float* hs = sm;                              // [128][kD+1]
  float* cs = hs + kTsgTile * (kD + 1);        // [kTsKeys][kD]
  float* cr = cs + kTsKeys * kD;               // [kTsKeys]
  const int t = blockIdx.x, h = blockIdx.y, tid = threadIdx.x, n = ft.n_tokens;
  // tile -> historical frame
  int f = 0;
  while (f + 1 < ft.n_frames - 1 && ft.tile0[f + 1] <= t) ++f;
  int fend = ft.off[f] + ft.gh[f] * ft.gw[f];
  int i0 = ft.off[f] + (t - ft.tile0[f]) * kTsgTile;
  for (int e = tid; e < kTsgTile * kD; e += blockDim.x) {
    int ii = e / kD, c = e - ii * kD;
    hs[ii * (kD + 1) + c] = (i0 + ii < fend) ? Elem<T>::load1(k + ((size_t)(i0 + ii) * hkv + h) * kD + c) : 0.f;
  }
  float best = -CUDART_INF_F;
  const float* hr = hs + tid * (kD + 1);
  for (int jt = 0; jt < ft.cur_len; jt += kTsKeys) {
    __syncthreads();
    for (int e = tid; e < kTsKeys * kD; e += blockDim.x) {
      int jj = e / kD, c = e - jj * kD;
      int j = ft.cur_off + jt + jj;
      cs[e] = (jt + jj < ft.cur_len) ? Elem<T>::load1(k + ((size_t)j * hkv + h) * kD + c) : 0.f;
    }
    for (int jj = tid; jj < kTsKeys; jj += blockDim.x)
      cr[jj] = (jt + jj < ft.cur_len) ? rn[(size_t)h * n + ft.cur_off + jt + jj] : 0.f;
    __syncthreads();
    int nk = min(kTsKeys, ft.cur_len - jt);
    for (int jj = 0; jj < nk; ++jj) {
      const float* kr = cs + jj * kD;
      float d0 = 0.f, d1 = 0.f;
#pragma unroll 16
      for (int c = 0; c < kD; c += 2) {
        d0 = fmaf(hr[c], kr[c], d0);
        d1 = fmaf(hr[c + 1], kr[c + 1], d1);
      }
      best = fmaxf(best, (d0 + d1) * cr[jj]);
    }
  }
  if (i0 + tid < fend) rho_part[(size_t)h * n + i0 + tid] = best;
}

cudaError_t launch_tsg(const Problem& p, const FrameTable& ft, const void* k, const float* rn,
                       float* rho_part, int nchunk, uint32_t* err, cudaStream_t st) {
  (void)err;
  (void)nchunk;
  cudaFuncSetAttribute(k_tsg_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTsSmem);
  cudaFuncSetAttribute(k_tsg_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTsSmem);
  int tiles = ft.n_frames >= 2 ? ft.tile0[ft.n_frames - 1] : 0;
  if (tiles == 0) return cudaSuccess;
  dim3 g(tiles, p.hkv);
  TimingScope ts("tsg_simt", st);
  if (p.dtype == kBF16)
    k_tsg_simt<<<g, kTsgTile, kTsSmem, st>>>((const __nv_bfloat16*)k, rn, ft, p.hkv, rho_part);
  else
    k_tsg_simt<<<g, kTsgTile, kTsSmem, st>>>((const float*)k, rn, ft, p.hkv, rho_part);
  return cudaGetLastError();
}

}  // namespace stl
