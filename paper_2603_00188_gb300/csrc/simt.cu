// CUDA-core kernels: inverse key norms, CSS saliency, and the fp32 versions
// of window scoring and TSG (fp32 inputs cannot use the bf16 tensor-core
// path without losing the exactness of the products).  Every kernel covers a
// batch of layers: the layer index is the high part of one grid dimension.
#include "kernels.cuh"

namespace stl {

constexpr float kLog2e = 1.4426950408889634f;

// 16 bytes of keys -> floats (8 bf16 or 4 fp32).  Shared by the norm and CSS
// kernels, so that both compute a key's norm with the same sequence of
// operations (fmaf over elements 0..127 in order) and agree bit for bit.
template <typename T>
__device__ __forceinline__ void unpack16(const uint4& w, float (&f)[16 / sizeof(T)]) {
  if constexpr (sizeof(T) == 2) {
    f[0] = __uint_as_float(w.x << 16);
    f[1] = __uint_as_float(w.x & 0xffff0000u);
    f[2] = __uint_as_float(w.y << 16);
    f[3] = __uint_as_float(w.y & 0xffff0000u);
    f[4] = __uint_as_float(w.z << 16);
    f[5] = __uint_as_float(w.z & 0xffff0000u);
    f[6] = __uint_as_float(w.w << 16);
    f[7] = __uint_as_float(w.w & 0xffff0000u);
  } else {
    f[0] = __uint_as_float(w.x);
    f[1] = __uint_as_float(w.y);
    f[2] = __uint_as_float(w.z);
    f[3] = __uint_as_float(w.w);
  }
}

// ---------------------------------------------------------------- norms
// rn[l][h][j] = 1 / max(|k_l[j,h]|, 1e-8); one thread per (token, head) row,
// grid.y = layer.
template <typename T>
__global__ void __launch_bounds__(256) k_inv_norms(const __grid_constant__ LayerPtrs io, int n, int hkv,
                                                   Strided<float> rn_all, Strided<float> rc_all, int cur_off,
                                                   int cur_len, int cur_pad) {
  constexpr int kChunks = kD * (int)sizeof(T) / 16;
  constexpr int kPer = 16 / (int)sizeof(T);
  const int l = blockIdx.y;
  const T* k = static_cast<const T*>(io.k[l]);
  float* rn = rn_all.at(l);
  const long long rows = (long long)n * hkv;
  for (long long r = (long long)blockIdx.x * blockDim.x + threadIdx.x; r < rows;
       r += (long long)gridDim.x * blockDim.x) {
    const uint4* src = reinterpret_cast<const uint4*>(k + r * kD);
    uint4 w[kChunks];
#pragma unroll
    for (int c = 0; c < kChunks; ++c) w[c] = __ldg(src + c);
    float sn = 0.f;
#pragma unroll
    for (int c = 0; c < kChunks; ++c) {
      float x[kPer];
      unpack16<T>(w[c], x);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sn = fmaf(x[t], x[t], sn);
    }
    const long long j = r / hkv, h = r - j * hkv;
    const float v = 1.0f / fmaxf(sqrtf(sn), 1e-8f);
    rn[h * n + j] = v;
    if (j >= cur_off && j < cur_off + cur_len) rc_all.at(l)[h * cur_pad + (j - cur_off)] = v;
  }
}

cudaError_t launch_inv_norms(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> rn,
                             Strided<float> rn_cur, int cur_pad, cudaStream_t st) {
  long long rows = (long long)p.n * p.hkv;
  long long blocks = (rows + 255) / 256;
  long long cap = (152 * 8 + p.L - 1) / p.L;
  if (blocks > cap) blocks = cap;
  TimingScope ts("inv_norms", st);
  dim3 grid((unsigned)blocks, p.L);
  if (p.dtype == kBF16)
    k_inv_norms<__nv_bfloat16><<<grid, 256, 0, st>>>(io, p.n, p.hkv, rn, rn_cur, ft.cur_off, ft.cur_len, cur_pad);
  else
    k_inv_norms<float><<<grid, 256, 0, st>>>(io, p.n, p.hkv, rn, rn_cur, ft.cur_off, ft.cur_len, cur_pad);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- CSS
// Eqs. 4-5 on 2-D tiles of one frame's patch grid.  A CTA (tile, frame,
// layer*Hkv + head) stages the tile's keys plus a one-cell halo in shared
// memory with asynchronous copies (key rows padded by 16 bytes, so 8 threads
// reading 8 different keys hit 8 distinct bank groups).  One thread per cell
// then computes the cell's norm and its E, S, SE, SW pair dots in one sweep,
// so every unordered neighbour pair is computed once; finally each output
// cell sums its eight directions.  The inverse norms of the output cells are
// written too (TSG uses them).
constexpr int kCssThreads = 256;
constexpr int kCssBudget = 100 * 1024;  // shared-memory bytes per CTA
constexpr int kCssMaxCols = 64;         // output columns per tile

template <typename T>
struct CssGeom {
  static constexpr int kStride = kD * (int)sizeof(T) + 16;   // padded key row
  static constexpr int kCellBytes = kStride + 5 * 4;         // key + rn + 4 pair dots
  static constexpr int kCap = kCssBudget / kCellBytes;       // cells per CTA
  // output tile of CB columns x RB rows, loaded as (RB+2) x (CB+2) cells
  __host__ __device__ static void tile(int gh, int gw, int& RB, int& CB) {
    CB = gw < kCssMaxCols ? gw : kCssMaxCols;
    RB = kCap / (CB + 2) - 2;
    if (RB < 1) RB = 1;
    if (RB > gh) RB = gh;
  }
  __host__ __device__ static int tiles(int gh, int gw) {
    int RB, CB;
    tile(gh, gw, RB, CB);
    return ((gh + RB - 1) / RB) * ((gw + CB - 1) / CB);
  }
};

template <typename T>
__global__ void __launch_bounds__(kCssThreads) k_css(const __grid_constant__ LayerPtrs io,
                                                     const __grid_constant__ FrameTable ft, int hkv,
                                                     Strided<float> phi_all, Strided<float> rn_all,
                                                     Strided<float> rc_all, int cur_pad) {
  using Gm = CssGeom<T>;
  constexpr int kChunks = kD * (int)sizeof(T) / 16;
  constexpr int kPer = 16 / (int)sizeof(T);
  extern __shared__ float4 css_smem[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(css_smem);
  const int f = blockIdx.y, l = blockIdx.z / hkv, h = blockIdx.z % hkv, n = ft.n_tokens;
  const int tid = threadIdx.x;
  if (f >= ft.n_frames) return;
  const T* k = static_cast<const T*>(io.k[l]);
  float* phi = phi_all.at(l);
  float* rn_out = rn_all.at(l);
  const int gh = ft.gh[f], gw = ft.gw[f], off = ft.off[f];
  int RB, CB;
  Gm::tile(gh, gw, RB, CB);
  const int tv = (gw + CB - 1) / CB;
  if ((int)blockIdx.x >= ((gh + RB - 1) / RB) * tv) return;
  const int u0 = ((int)blockIdx.x / tv) * RB, v0 = ((int)blockIdx.x % tv) * CB;
  const int TW = CB + 2, TH = RB + 2, cells = TW * TH;
  uint8_t* keys = sm;
  float* rn = reinterpret_cast<float*>(sm + (size_t)cells * Gm::kStride);
  float* dE = rn + cells;
  float* dS = dE + cells;
  float* dSE = dS + cells;
  float* dSW = dSE + cells;
  // stage the tile (local cell (a, b) = grid cell (u0 - 1 + a, v0 - 1 + b));
  // cells outside the grid stay unloaded and are never read
  for (int e = tid; e < cells * kChunks; e += blockDim.x) {
    const int cell = e / kChunks, ch = e - cell * kChunks;
    const int u = u0 - 1 + cell / TW, v = v0 - 1 + cell % TW;
    if (u < 0 || u >= gh || v < 0 || v >= gw) continue;
    const T* src = k + ((size_t)(off + u * gw + v) * hkv + h) * kD + ch * kPer;
    const uint32_t dst =
        static_cast<uint32_t>(__cvta_generic_to_shared(keys + (size_t)cell * Gm::kStride + 16 * ch));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
  }
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  // one thread per cell: its norm and its E, S, SE, SW pair dots in one sweep
  // (a missing partner reads the cell itself and is discarded)
  for (int cell = tid; cell < cells; cell += blockDim.x) {
    const int a = cell / TW, b = cell % TW;
    const int u = u0 - 1 + a, v = v0 - 1 + b;
    if (u < 0 || u >= gh || v < 0 || v >= gw) continue;
    const bool fwd = a <= RB && u + 1 < gh;
    const bool hasE = b + 1 < TW && v + 1 < gw;
    const bool hasSE = fwd && b + 1 < TW && v + 1 < gw;
    const bool hasSW = fwd && b >= 1 && v >= 1;
    const uint8_t* p0 = keys + (size_t)cell * Gm::kStride;
    const uint8_t* pE = hasE ? p0 + Gm::kStride : p0;
    const uint8_t* pS = fwd ? p0 + (size_t)TW * Gm::kStride : p0;
    const uint8_t* pSE = hasSE ? p0 + (size_t)(TW + 1) * Gm::kStride : p0;
    const uint8_t* pSW = hasSW ? p0 + (size_t)(TW - 1) * Gm::kStride : p0;
    float sn = 0.f, sE = 0.f, sS = 0.f, sSE = 0.f, sSW = 0.f;
#pragma unroll 4
    for (int c = 0; c < kChunks; ++c) {
      float x[kPer], y[kPer];
      unpack16<T>(*reinterpret_cast<const uint4*>(p0 + 16 * c), x);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sn = fmaf(x[t], x[t], sn);
      unpack16<T>(*reinterpret_cast<const uint4*>(pE + 16 * c), y);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sE = fmaf(x[t], y[t], sE);
      unpack16<T>(*reinterpret_cast<const uint4*>(pS + 16 * c), y);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sS = fmaf(x[t], y[t], sS);
      unpack16<T>(*reinterpret_cast<const uint4*>(pSE + 16 * c), y);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sSE = fmaf(x[t], y[t], sSE);
      unpack16<T>(*reinterpret_cast<const uint4*>(pSW + 16 * c), y);
#pragma unroll
      for (int t = 0; t < kPer; ++t) sSW = fmaf(x[t], y[t], sSW);
    }
    rn[cell] = 1.0f / fmaxf(sqrtf(sn), 1e-8f);
    dE[cell] = sE;
    dS[cell] = sS;
    dSE[cell] = sSE;
    dSW[cell] = sSW;
  }
  __syncthreads();
  for (int o = tid; o < RB * CB; o += blockDim.x) {
    const int u = u0 + o / CB, v = v0 + o % CB;
    if (u >= gh || v >= gw) continue;
    const int c = (o / CB + 1) * TW + (o % CB + 1);
    const float r0 = rn[c];
    float sum = 0.f;
    int cnt = 0;
    const bool up = u > 0, dn = u + 1 < gh, lf = v > 0, rt = v + 1 < gw;
    if (rt) { sum += dE[c] * r0 * rn[c + 1]; ++cnt; }
    if (lf) { sum += dE[c - 1] * rn[c - 1] * r0; ++cnt; }
    if (dn) { sum += dS[c] * r0 * rn[c + TW]; ++cnt; }
    if (up) { sum += dS[c - TW] * rn[c - TW] * r0; ++cnt; }
    if (dn && rt) { sum += dSE[c] * r0 * rn[c + TW + 1]; ++cnt; }
    if (up && lf) { sum += dSE[c - TW - 1] * rn[c - TW - 1] * r0; ++cnt; }
    if (dn && lf) { sum += dSW[c] * r0 * rn[c + TW - 1]; ++cnt; }
    if (up && rt) { sum += dSW[c - TW + 1] * rn[c - TW + 1] * r0; ++cnt; }
    const int j = off + u * gw + v;
    phi[(size_t)h * n + j] = cnt ? 1.0f - sum / (float)cnt : 0.0f;
    rn_out[(size_t)h * n + j] = r0;
    if (f == ft.n_frames - 1) rc_all.at(l)[(size_t)h * cur_pad + (j - off)] = r0;
  }
}

// Phi of text tokens is undefined: NaN (only the staged entry point writes it).
__global__ void k_fill_text_nan(const __grid_constant__ FrameTable ft, int hkv, float* __restrict__ phi) {
  const int n = ft.n_tokens;
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < (long long)n * hkv;
       e += (long long)gridDim.x * blockDim.x) {
    const int j = (int)(e % n);
    if (find_frame(ft, j) < 0) phi[e] = CUDART_NAN_F;
  }
}

template <typename T>
static cudaError_t css_launch_t(const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                                Strided<float> phi, Strided<float> rn, Strided<float> rn_cur, int cur_pad,
                                cudaStream_t st) {
  using Gm = CssGeom<T>;
  int tmax = 0, cmax = 0;
  for (int f = 0; f < ft.n_frames; ++f) {
    int RB, CB;
    Gm::tile(ft.gh[f], ft.gw[f], RB, CB);
    tmax = max(tmax, Gm::tiles(ft.gh[f], ft.gw[f]));
    cmax = max(cmax, (RB + 2) * (CB + 2));
  }
  if (tmax == 0) return cudaSuccess;
  const size_t smem = (size_t)cmax * Gm::kCellBytes;
  cudaError_t e = cudaFuncSetAttribute(k_css<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  TimingScope ts("css", st);
  k_css<T><<<dim3(tmax, ft.n_frames, p.L * p.hkv), kCssThreads, smem, st>>>(io, ft, p.hkv, phi, rn, rn_cur,
                                                                             cur_pad);
  return cudaGetLastError();
}

cudaError_t launch_css(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> phi,
                       Strided<float> rn, Strided<float> rn_cur, int cur_pad, cudaStream_t st) {
  if (p.dtype == kBF16) return css_launch_t<__nv_bfloat16>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
  return css_launch_t<float>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
}

// ------------------------------------------------------- CSS, k x k box
// Eqs. 4-5 over the (2R+1) x (2R+1) neighbourhood (R = 1 is the method's 3x3
// Moore neighbourhood; R = 2..4 the 5x5..9x9 kernels of the size ablation).
// With khat_j = k_j / max(|k_j|, 1e-8) the neighbour cosines add up to
//   sum_{j in N(i)} cos(k_i, k_j) = khat_i . (sum_{j in box(i)} khat_j - khat_i),
// so a cell needs one box sum of normalised keys, whatever the size, and
// the box sum separates into row sums and a sum of 2R+1 rows.  A CTA (tile,
// frame, layer*Hkv + head) stages kBoxRows x kBoxCols output cells plus an
// R-cell halo (out-of-grid cells as zero keys with rn = 0, so they add
// nothing); each 16-lane half-warp owns one output column, 8 dimensions per
// lane, walks the tile's rows once and keeps the last 2R+1 row sums in
// registers.  rn of a cell uses the same operation sequence as the norms
// kernel, so both agree bit for bit.
constexpr int kBoxRows = 8, kBoxCols = 16, kBoxThreads = 256;

template <typename T, int R>
struct BoxGeom {
  static constexpr int TH = kBoxRows + 2 * R, TW = kBoxCols + 2 * R, cells = TH * TW;
  static constexpr int stride = kD * (int)sizeof(T) + 16;  // padded key row
  static constexpr int smem = cells * stride + cells * 4;
};

template <typename T, int R>
__global__ void __launch_bounds__(kBoxThreads) k_css_box(const __grid_constant__ LayerPtrs io,
                                                         const __grid_constant__ FrameTable ft, int hkv,
                                                         Strided<float> phi_all, Strided<float> rn_all,
                                                         Strided<float> rc_all, int cur_pad) {
  using Gm = BoxGeom<T, R>;
  constexpr int kChunks = kD * (int)sizeof(T) / 16;
  constexpr int kPer = 16 / (int)sizeof(T);
  constexpr int TW = Gm::TW, TH = Gm::TH, D2 = 2 * R + 1;
  extern __shared__ float4 box_smem[];
  uint8_t* keys = reinterpret_cast<uint8_t*>(box_smem);
  float* rn = reinterpret_cast<float*>(keys + (size_t)Gm::cells * Gm::stride);
  const int f = blockIdx.y, l = blockIdx.z / hkv, h = blockIdx.z % hkv, n = ft.n_tokens;
  const int tid = threadIdx.x;
  if (f >= ft.n_frames) return;
  const int gh = ft.gh[f], gw = ft.gw[f], off = ft.off[f];
  const int tv = (gw + kBoxCols - 1) / kBoxCols;
  if ((int)blockIdx.x >= ((gh + kBoxRows - 1) / kBoxRows) * tv) return;
  const int u0 = ((int)blockIdx.x / tv) * kBoxRows, v0 = ((int)blockIdx.x % tv) * kBoxCols;
  const T* k = static_cast<const T*>(io.k[l]);
  // stage: local cell (a, b) = grid cell (u0 - R + a, v0 - R + b)
  for (int e = tid; e < Gm::cells * kChunks; e += blockDim.x) {
    const int cell = e / kChunks, ch = e - cell * kChunks;
    const int u = u0 - R + cell / TW, v = v0 - R + cell % TW;
    uint8_t* dstp = keys + (size_t)cell * Gm::stride + 16 * ch;
    if (u < 0 || u >= gh || v < 0 || v >= gw) {
      *reinterpret_cast<uint4*>(dstp) = make_uint4(0u, 0u, 0u, 0u);
      continue;
    }
    const T* src = k + ((size_t)(off + u * gw + v) * hkv + h) * kD + ch * kPer;
    const uint32_t dst = static_cast<uint32_t>(__cvta_generic_to_shared(dstp));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
  }
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  // inverse norms (0 outside the grid); the output cells' go to rn / rn_cur
  for (int cell = tid; cell < Gm::cells; cell += blockDim.x) {
    const int a = cell / TW, b = cell % TW;
    const int u = u0 - R + a, v = v0 - R + b;
    float r = 0.f;
    if (u >= 0 && u < gh && v >= 0 && v < gw) {
      const uint8_t* p0 = keys + (size_t)cell * Gm::stride;
      float sn = 0.f;
#pragma unroll 4
      for (int c = 0; c < kChunks; ++c) {
        float x[kPer];
        unpack16<T>(*reinterpret_cast<const uint4*>(p0 + 16 * c), x);
#pragma unroll
        for (int t = 0; t < kPer; ++t) sn = fmaf(x[t], x[t], sn);
      }
      r = 1.0f / fmaxf(sqrtf(sn), 1e-8f);
      if (a >= R && a < R + kBoxRows && b >= R && b < R + kBoxCols) {
        const int j = off + u * gw + v;
        rn_all.at(l)[(size_t)h * n + j] = r;
        if (f == ft.n_frames - 1) rc_all.at(l)[(size_t)h * cur_pad + (j - off)] = r;
      }
    }
    rn[cell] = r;
  }
  __syncthreads();
  // box sums: lane group (16 lanes) = output column, 8 dimensions per lane
  const int dg = tid & 15, col = tid >> 4;
  const int v = v0 + col;
  float* phi = phi_all.at(l);
  auto load8 = [&](int cell, float (&x)[8]) {
    const uint8_t* p0 = keys + (size_t)cell * Gm::stride + dg * 8 * (int)sizeof(T);
#pragma unroll
    for (int c = 0; c < 8 / kPer; ++c) {
      float y[kPer];
      unpack16<T>(*reinterpret_cast<const uint4*>(p0 + 16 * c), y);
#pragma unroll
      for (int t = 0; t < kPer; ++t) x[c * kPer + t] = y[t];
    }
  };
  float ring[D2][8];
#pragma unroll
  for (int a = 0; a < TH; ++a) {
    float hs[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) hs[e] = 0.f;
#pragma unroll
    for (int dv = 0; dv < D2; ++dv) {
      const int cell = a * TW + col + dv;
      const float r = rn[cell];
      float x[8];
      load8(cell, x);
#pragma unroll
      for (int e = 0; e < 8; ++e) hs[e] = fmaf(r, x[e], hs[e]);
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) ring[a % D2][e] = hs[e];
    if (a >= 2 * R) {
      const int o = a - 2 * R;  // output row of the tile
      const int cell = (o + R) * TW + col + R;
      const float ri = rn[cell];
      float x[8];
      load8(cell, x);
      float dot = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float s = ring[0][e];
#pragma unroll
        for (int q = 1; q < D2; ++q) s += ring[q][e];
        const float kh = ri * x[e];
        dot = fmaf(kh, s - kh, dot);
      }
#pragma unroll
      for (int m = 8; m > 0; m >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, m);
      const int u = u0 + o;
      if (dg == 0 && u < gh && v < gw) {
        const int nu = min(u + R, gh - 1) - max(u - R, 0) + 1;
        const int nv = min(v + R, gw - 1) - max(v - R, 0) + 1;
        const int cnt = nu * nv - 1;
        phi[(size_t)h * n + off + u * gw + v] = cnt ? 1.0f - dot / (float)cnt : 0.0f;
      }
    }
  }
}

template <typename T, int R>
static cudaError_t css_box_t(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> phi,
                             Strided<float> rn, Strided<float> rn_cur, int cur_pad, cudaStream_t st) {
  using Gm = BoxGeom<T, R>;
  cudaError_t e = cudaFuncSetAttribute(k_css_box<T, R>, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::smem);
  if (e != cudaSuccess) return e;
  int tiles = 1;
  for (int f = 0; f < ft.n_frames; ++f) {
    const int t = ((ft.gh[f] + kBoxRows - 1) / kBoxRows) * ((ft.gw[f] + kBoxCols - 1) / kBoxCols);
    tiles = t > tiles ? t : tiles;
  }
  TimingScope ts("css_box", st);
  dim3 grid((unsigned)tiles, (unsigned)(ft.n_frames > 0 ? ft.n_frames : 1), (unsigned)(p.L * p.hkv));
  k_css_box<T, R><<<grid, kBoxThreads, Gm::smem, st>>>(io, ft, p.hkv, phi, rn, rn_cur, cur_pad);
  return cudaGetLastError();
}

template <typename T>
static cudaError_t css_box_r(int radius, const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                             Strided<float> phi, Strided<float> rn, Strided<float> rn_cur, int cur_pad,
                             cudaStream_t st) {
  switch (radius) {
    case 1: return css_box_t<T, 1>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
    case 2: return css_box_t<T, 2>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
    case 3: return css_box_t<T, 3>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
    case 4: return css_box_t<T, 4>(p, ft, io, phi, rn, rn_cur, cur_pad, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_css_box(const Problem& p, const FrameTable& ft, const LayerPtrs& io, int size,
                           Strided<float> phi, Strided<float> rn, Strided<float> rn_cur, int cur_pad,
                           cudaStream_t st) {
  if (ft.n_frames == 0) return cudaSuccess;
  if (p.dtype == kBF16) return css_box_r<__nv_bfloat16>(size / 2, p, ft, io, phi, rn, rn_cur, cur_pad, st);
  return css_box_r<float>(size / 2, p, ft, io, phi, rn, rn_cur, cur_pad, st);
}

cudaError_t launch_fill_text_nan(const Problem& p, const FrameTable& ft, float* phi, cudaStream_t st) {
  long long tot = (long long)p.n * p.hkv;
  long long blocks = (tot + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  k_fill_text_nan<<<(int)blocks, 256, 0, st>>>(ft, p.hkv, phi);
  return cudaGetLastError();
}

// ------------------------------------------------------- row statistics
// Window score, first pass (fp32): for every query row r of KV head h (r =
// window row * G + group member) the running maximum m and sum l of
// 2^(x - m), x = q.k * log2(e)/sqrt(d), over the keys of one split.
// grid = (split, layer*Hkv + head, row chunk).
constexpr int kRsRows = 256;   // query rows per block
constexpr int kRsKeys = 64;    // keys per smem tile
constexpr int kRsSmem = (kRsRows * (kD + 1) + kRsKeys * kD) * 4;

template <typename T>
__global__ void __launch_bounds__(kRsRows) k_rowstats_simt(const __grid_constant__ LayerPtrs io, Problem p,
                                                           int nsplit, Strided<float2> part_all) {
  extern __shared__ float sm[];
  float* qs = sm;                       // [kRsRows][kD+1]
  float* ks = sm + kRsRows * (kD + 1);  // [kRsKeys][kD]
  const int s = blockIdx.x, l = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv, r0 = blockIdx.z * kRsRows;
  const T* q = static_cast<const T*>(io.q[l]);
  const T* k = static_cast<const T*>(io.k[l]);
  float2* part = part_all.at(l);
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
  float m = -CUDART_INF_F, lsum = 0.f;
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
        lsum = lsum * exp2f(m - x) + 1.0f;
        m = x;
      } else {
        lsum += exp2f(x - m);
      }
    }
  }
  if (r0 + tid < R) part[((size_t)h * nsplit + s) * R + r0 + tid] = make_float2(m, lsum);
}

// Merge the splits: bias[h][r] = -m_r - log2(G * l_r), so that
// 2^(x + bias) = softmax probability / G.  One thread per row (consecutive
// rows, coalesced loads), one pass in split order with eight partials in
// flight: (M, L) <- (max(M, m_s), L 2^(M - M') + l_s 2^(m_s - M')).
// grid.y = layer.
// Folds one split partial (m2, l2) into (m, l): the running max in log2
// units and the sum of 2^(x - max).  Symmetric in its two arguments, bit for
// bit (max and a two-term sum commute).
__device__ __forceinline__ void fold_partial(float& m, float& l, float m2, float l2) {
  if (!(l2 > 0.f)) return;
  if (!(l > 0.f)) {
    m = m2;
    l = l2;
    return;
  }
  const float mn = fmaxf(m, m2);
  l = l * exp2f(m - mn) + l2 * exp2f(m2 - mn);
  m = mn;
}

// Four lanes per query row: lane q folds splits q, q + 4, q + 8, ... (eight
// loads in flight), then the four lanes' states are folded pairwise with
// shuffles, so every lane holds the same bits and lane 0 writes the bias.
// The order depends on the split count alone.
__global__ void __launch_bounds__(128) k_row_bias(Problem p, int nsplit, Strided<float2> part_all) {
  const int R = p.R(), l = blockIdx.y;
  const float2* part = part_all.at(l);
  float* bias = reinterpret_cast<float*>(part_all.at(l) + (size_t)p.hkv * nsplit * R);
  const int e4 = blockIdx.x * blockDim.x + threadIdx.x;
  const int e = e4 >> 2, q = e4 & 3;
  const bool live = e < p.hkv * R;
  float m = -CUDART_INF_F, lsum = 0.f;
  if (live) {
    const int h = e / R, r = e - h * R;
    const float2* pp = part + (size_t)h * nsplit * R + r;
    for (int s0 = q; s0 < nsplit; s0 += 32) {
      float2 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        v[u] = s0 + 4 * u < nsplit ? pp[(size_t)(s0 + 4 * u) * R] : make_float2(-CUDART_INF_F, 0.f);
#pragma unroll
      for (int u = 0; u < 8; ++u) fold_partial(m, lsum, v[u].x, v[u].y);
    }
  }
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), l2 = __shfl_xor_sync(0xffffffffu, lsum, o);
    fold_partial(m, lsum, m2, l2);
  }
  if (live && q == 0) bias[e] = -m - log2f((float)p.G() * lsum);
}

void launch_row_bias(const Problem& p, int nsplit, Strided<float2> rowpart, cudaStream_t st) {
  const int rows = p.hkv * p.R();
  k_row_bias<<<dim3((4 * rows + 127) / 128, p.L), 128, 0, st>>>(p, nsplit, rowpart);
}

// ---------------------------------------------------------- column sums
// Window score, second pass (fp32): a[h][j] = sum_r 2^(x_rj + bias_r).  One
// thread per key; the key tile is kept (padded) in shared memory.
// grid = (key tile, layer*Hkv + head).
constexpr int kCsKeys = 128;
constexpr int kCsRows = 32;
constexpr int kCsMaxR = 1024;
constexpr int kCsSmem = (kCsKeys * (kD + 1) + kCsRows * kD + kCsMaxR) * 4;

template <typename T>
__global__ void __launch_bounds__(kCsKeys) k_colsum_simt(const __grid_constant__ LayerPtrs io, Problem p,
                                                         int nsplit, Strided<float2> part_all,
                                                         Strided<float> a_all) {
  extern __shared__ float sm[];
  float* ks = sm;                            // [kCsKeys][kD+1]
  float* qs = ks + kCsKeys * (kD + 1);       // [kCsRows][kD]
  float* bs = qs + kCsRows * kD;             // [R]
  const int l = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv, j0 = blockIdx.x * kCsKeys, tid = threadIdx.x;
  const T* q = static_cast<const T*>(io.q[l]);
  const T* k = static_cast<const T*>(io.k[l]);
  const float* bias = reinterpret_cast<const float*>(part_all.at(l) + (size_t)p.hkv * nsplit * p.R());
  float* a_base = a_all.at(l);
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

cudaError_t launch_score(const Problem& p, const LayerPtrs& io, Strided<float2> rowpart, int nsplit,
                         Strided<float> a_base, uint32_t* err, cudaStream_t st) {
  (void)err;
  if (p.R() > kCsMaxR) return cudaErrorNotSupported;
  cudaFuncSetAttribute(k_rowstats_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kRsSmem);
  cudaFuncSetAttribute(k_rowstats_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kRsSmem);
  cudaFuncSetAttribute(k_colsum_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCsSmem);
  cudaFuncSetAttribute(k_colsum_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCsSmem);
  dim3 g1(nsplit, p.L * p.hkv, (p.R() + kRsRows - 1) / kRsRows);
  dim3 g2((p.n + kCsKeys - 1) / kCsKeys, p.L * p.hkv);
  {
    TimingScope ts("rowstats_simt", st);
    if (p.dtype == kBF16)
      k_rowstats_simt<__nv_bfloat16><<<g1, kRsRows, kRsSmem, st>>>(io, p, nsplit, rowpart);
    else
      k_rowstats_simt<float><<<g1, kRsRows, kRsSmem, st>>>(io, p, nsplit, rowpart);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  {
    TimingScope ts("row_bias", st);
    launch_row_bias(p, nsplit, rowpart, st);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  TimingScope ts("colsum_simt", st);
  if (p.dtype == kBF16)
    k_colsum_simt<__nv_bfloat16><<<g2, kCsKeys, kCsSmem, st>>>(io, p, nsplit, rowpart, a_base);
  else
    k_colsum_simt<float><<<g2, kCsKeys, kCsSmem, st>>>(io, p, nsplit, rowpart, a_base);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ TSG
// fp32 path of Eq. 6: one thread per historical token, current-frame keys
// streamed through shared memory.  Writes slice 0 of rho_part (the fp32 path
// has a single slice).  grid = (row tile, layer*Hkv + head).
constexpr int kTsKeys = 64;
constexpr int kTsSmem = (kTsgTile * (kD + 1) + kTsKeys * kD + 2 * kTsKeys) * 4;

template <typename T>
__global__ void __launch_bounds__(kTsgTile) k_tsg_simt(const __grid_constant__ LayerPtrs io,
                                                       const __grid_constant__ FrameTable ft, int hkv,
                                                       Strided<const float> rn_all,
                                                       Strided<float> rho_all, int metric) {
  extern __shared__ float sm[];
  float* hs = sm;                              // [128][kD+1]
  float* cs = hs + kTsgTile * (kD + 1);        // [kTsKeys][kD]
  float* cr = cs + kTsKeys * kD;               // [kTsKeys] scale of each current key
  float* co = cr + kTsKeys;                    // [kTsKeys] offset: value = dot * scale + offset
  const int t = blockIdx.x, l = blockIdx.y / hkv, h = blockIdx.y % hkv, tid = threadIdx.x;
  const int n = ft.n_tokens;
  const T* k = static_cast<const T*>(io.k[l]);
  const float* rn = rn_all.at(l);
  float* rho_part = rho_all.at(l);
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
    for (int jj = tid; jj < kTsKeys; jj += blockDim.x) {
      // cosine: dot * rn_j; dot: dot; negative L2 (without the row's own
      // -|k_i|^2): 2 dot - |k_j|^2
      const float r = (jt + jj < ft.cur_len) ? rn[(size_t)h * n + ft.cur_off + jt + jj] : 0.f;
      cr[jj] = metric == kTsgCosine ? r : (metric == kTsgDot ? 1.f : 2.f);
      co[jj] = metric == kTsgNegL2 ? -1.f / (r * r) : 0.f;
    }
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
      best = fmaxf(best, fmaf(d0 + d1, cr[jj], co[jj]));
    }
  }
  if (i0 + tid < fend) rho_part[(size_t)h * n + i0 + tid] = best;
}

cudaError_t launch_tsg(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<const float> rn,
                       Strided<float> rho_part, int metric, uint32_t* err, cudaStream_t st) {
  (void)err;
  cudaFuncSetAttribute(k_tsg_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTsSmem);
  cudaFuncSetAttribute(k_tsg_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTsSmem);
  int tiles = ft.n_frames >= 2 ? ft.tile0[ft.n_frames - 1] : 0;
  if (tiles == 0) return cudaSuccess;
  dim3 g(tiles, p.L * p.hkv);
  TimingScope ts("tsg_simt", st);
  if (p.dtype == kBF16)
    k_tsg_simt<__nv_bfloat16><<<g, kTsgTile, kTsSmem, st>>>(io, ft, p.hkv, rn, rho_part, metric);
  else
    k_tsg_simt<float><<<g, kTsgTile, kTsSmem, st>>>(io, ft, p.hkv, rn, rho_part, metric);
  return cudaGetLastError();
}

}  // namespace stl
