// Decode attention over a KV cache -- the consumer of the compressed cache.
// A decoder attends every new query row over the cached keys and values of
// each layer; after compression the cache holds B = beta*N rows instead of N,
// and this pass reads proportionally less (the efficiency study's decode
// latency).  out[r][g] = sum_j softmax_j(q_{r,g} . k_{j,h} / sqrt(d)) v_{j,h},
// h = g / G, over every cached row.
//
// Split over the cache (flash decoding): CTA (split, h, r) owns a contiguous
// range of cached rows for the G query heads of KV head h and window row r.
// Each warp takes 32 rows at a time, one per lane: the lane computes its
// row's G scores from the shared query rows, the warp keeps an online
// (max, sum) per query head, and for the value sum every lane owns four of the
// 128 dimensions while the rows' probabilities are broadcast by shuffles.  The
// four warps merge in shared memory; a second kernel merges the splits.
#include <type_traits>

#include "kernels.cuh"

namespace stl {

constexpr int kDecThreads = 256;  // 8 warps
constexpr float kDecLog2e = 1.4426950408889634f;
constexpr int kDecWarps = kDecThreads / 32;

// Eight consecutive elements of a row as floats (16-byte aligned).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&f)[8]) {
  const uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
__device__ __forceinline__ void load8(const float* p, float (&f)[8]) {
  const float4 a = __ldg(reinterpret_cast<const float4*>(p));
  const float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// exp2(a - m) with a = -inf or m = -inf giving 0 (an empty range has weight 0).
__device__ __forceinline__ float weight(float a, float m) { return a == -CUDART_INF_F ? 0.f : exp2f(a - m); }

// Dynamic shared memory: qs[G][128] (query rows times log2(e)/sqrt(d)), then
// per warp o[G][128] and (m, l)[G].
template <typename T, int GM>
__global__ void __launch_bounds__(kDecThreads, 2) k_decode_split(const T* __restrict__ q, const T* __restrict__ k,
                                                              const T* __restrict__ v, int n, int hq, int hkv,
                                                              int per, float* part_o, float2* part_ml) {
  extern __shared__ float4 dec_smem[];
  const int split = blockIdx.x, h = blockIdx.y, r = blockIdx.z, nsplit = gridDim.x;
  const int G = hq / hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* qs = reinterpret_cast<float*>(dec_smem);
  float* wo = qs + G * kD;                               // [warp][G][128]
  float2* wml = reinterpret_cast<float2*>(wo + kDecWarps * G * kD);  // [warp][G]
  const float scale = kDecLog2e * rsqrtf((float)kD);
  for (int e = threadIdx.x; e < G * kD; e += kDecThreads) {
    const int g = e / kD, c = e % kD;
    qs[e] = Elem<T>::load1(q + ((size_t)r * hq + h * G + g) * kD + c) * scale;
  }
  __syncthreads();

  const int j0 = min(n, split * per), j1 = min(n, j0 + per);
  float m[GM], l[GM], o[GM][4];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    m[g] = -CUDART_INF_F;
    l[g] = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) o[g][e] = 0.f;
  }
  const size_t rs = (size_t)hkv * kD;  // elements between consecutive cached rows
  for (int base = j0 + warp * 32; base < j1; base += kDecWarps * 32) {
    const int t = base + lane;
    float s[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) s[g] = 0.f;
    if (t < j1) {
      const T* kr = k + (size_t)t * rs + (size_t)h * kD;
#pragma unroll 8
      for (int c = 0; c < kD; c += 8) {
        float kf[8];
        load8(kr + c, kf);
#pragma unroll
        for (int g = 0; g < GM; ++g) {
          if (g < G) {
            const float4 a = *reinterpret_cast<const float4*>(qs + g * kD + c);
            const float4 b = *reinterpret_cast<const float4*>(qs + g * kD + c + 4);
            s[g] = fmaf(kf[0], a.x, fmaf(kf[1], a.y, fmaf(kf[2], a.z, fmaf(kf[3], a.w, s[g]))));
            s[g] = fmaf(kf[4], b.x, fmaf(kf[5], b.y, fmaf(kf[6], b.z, fmaf(kf[7], b.w, s[g]))));
          }
        }
      }
    }
    // online softmax per query head over these 32 rows (log2 units)
    float p[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      if (g < G) {
        const float x = t < j1 ? s[g] : -CUDART_INF_F;
        const float mn = fmaxf(m[g], warp_max(x));
        const float a = weight(m[g], mn);
        p[g] = weight(x, mn);
        l[g] = l[g] * a + warp_sum(p[g]);
#pragma unroll
        for (int e = 0; e < 4; ++e) o[g][e] *= a;
        m[g] = mn;
      }
    }
    // value rows: lane owns dimensions 4*lane .. 4*lane + 3; eight rows'
    // loads are in flight before their products
    const int cnt = min(32, j1 - base);
    for (int t0 = 0; t0 < cnt; t0 += 8) {
      float4 vv[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (t0 + u < cnt) vv[u] = Elem<T>::load4(v + (size_t)(base + t0 + u) * rs + (size_t)h * kD + 4 * lane);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (t0 + u < cnt) {
#pragma unroll
          for (int g = 0; g < GM; ++g) {
            if (g < G) {
              const float pg = __shfl_sync(0xffffffffu, p[g], t0 + u);
              o[g][0] = fmaf(pg, vv[u].x, o[g][0]);
              o[g][1] = fmaf(pg, vv[u].y, o[g][1]);
              o[g][2] = fmaf(pg, vv[u].z, o[g][2]);
              o[g][3] = fmaf(pg, vv[u].w, o[g][3]);
            }
          }
        }
      }
    }
  }
  // merge the four warps, then write this split's partial per query head
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    if (g < G) {
      *reinterpret_cast<float4*>(wo + ((size_t)warp * G + g) * kD + 4 * lane) =
          make_float4(o[g][0], o[g][1], o[g][2], o[g][3]);
      if (lane == 0) wml[warp * G + g] = make_float2(m[g], l[g]);
    }
  }
  __syncthreads();
  // one (query head, dimension) pair per thread and step
  for (int e = threadIdx.x; e < G * kD; e += kDecThreads) {
    const int g = e / kD, c = e % kD;
    float M = -CUDART_INF_F;
    for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, wml[w * G + g].x);
    float L = 0.f, O = 0.f;
    for (int w = 0; w < kDecWarps; ++w) {
      const float a = weight(wml[w * G + g].x, M);
      L = fmaf(wml[w * G + g].y, a, L);
      O = fmaf(wo[((size_t)w * G + g) * kD + c], a, O);
    }
    const size_t slot = ((size_t)split * gridDim.z + r) * hq + h * G + g;
    part_o[slot * kD + c] = O;
    if (c == 0) part_ml[slot] = make_float2(M, L);
  }
  (void)nsplit;
}

// out[r][g][c] = merge over the splits.  grid (hq, w), one thread per
// dimension: the splits' weights exp2(m_s - M) and the normaliser are formed
// once in shared memory, then every thread sums its dimension over the splits
// with eight partial loads in flight.
constexpr int kDecMaxSplits = 1024;
__global__ void __launch_bounds__(kD) k_decode_combine(const float* part_o, const float2* part_ml, int nsplit,
                                                       int hq, int w, float* out) {
  __shared__ float wts[kDecMaxSplits];
  __shared__ float red[kD / 32];
  __shared__ float bc[2];
  const int g = blockIdx.x, r = blockIdx.y, c = threadIdx.x, lane = c & 31, wp = c >> 5;
  float mx = -CUDART_INF_F;
  for (int s = c; s < nsplit; s += kD) mx = fmaxf(mx, part_ml[((size_t)s * w + r) * hq + g].x);
  mx = warp_max(mx);
  if (lane == 0) red[wp] = mx;
  __syncthreads();
  if (c == 0) {
    float M = red[0];
    for (int i = 1; i < kD / 32; ++i) M = fmaxf(M, red[i]);
    bc[0] = M;
  }
  __syncthreads();
  const float M = bc[0];
  float ls = 0.f;
  for (int s = c; s < nsplit; s += kD) {
    const float2 ml = part_ml[((size_t)s * w + r) * hq + g];
    const float a = weight(ml.x, M);
    wts[s] = a;
    ls = fmaf(ml.y, a, ls);
  }
  ls = warp_sum(ls);
  __syncthreads();  // red is reused
  if (lane == 0) red[wp] = ls;
  __syncthreads();
  if (c == 0) {
    float L = 0.f;
    for (int i = 0; i < kD / 32; ++i) L += red[i];
    bc[1] = L;
  }
  __syncthreads();
  float O = 0.f;
  int s = 0;
  for (; s + 8 <= nsplit; s += 8) {
    float x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) x[u] = part_o[(((size_t)(s + u) * w + r) * hq + g) * kD + c];
#pragma unroll
    for (int u = 0; u < 8; ++u) O = fmaf(x[u], wts[s + u], O);
  }
  for (; s < nsplit; ++s) O = fmaf(part_o[(((size_t)s * w + r) * hq + g) * kD + c], wts[s], O);
  out[((size_t)r * hq + g) * kD + c] = O / bc[1];
}

int decode_splits(int n, int hkv, int w) {
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // about two CTAs per SM, each with at least 256 cached rows
  long long s = (2LL * sms + (long long)hkv * w - 1) / ((long long)hkv * w);
  const long long cap = (n + 255) / 256;
  if (s > cap) s = cap;
  if (s > kDecMaxSplits) s = kDecMaxSplits;
  if (s < 1) s = 1;
  return (int)s;
}

size_t decode_workspace_bytes(int n, int hq, int hkv, int w) {
  const size_t slots = (size_t)decode_splits(n, hkv, w) * w * hq;
  return slots * kD * sizeof(float) + slots * sizeof(float2) + 256;
}

cudaError_t launch_decode(DType dt, const void* q, const void* k, const void* v, int n, int hq, int hkv, int w,
                          float* out, void* ws, cudaStream_t st) {
  const int nsplit = decode_splits(n, hkv, w);
  const int per = ((n + nsplit - 1) / nsplit + 31) / 32 * 32;
  float* part_o = static_cast<float*>(ws);
  float2* part_ml = reinterpret_cast<float2*>(part_o + (size_t)nsplit * w * hq * kD);
  const int G = hq / hkv;
  const size_t smem = (size_t)G * kD * 4 + (size_t)kDecWarps * G * kD * 4 + (size_t)kDecWarps * G * 8;
  dim3 grid(nsplit, hkv, w);
  // register arrays sized for the group: G <= 4, <= 8 or <= 16 query heads
  cudaError_t fe = cudaSuccess;
  auto run = [&](auto tag, auto gm) {
    using T = decltype(tag);
    constexpr int GM = decltype(gm)::value;
    fe = cudaFuncSetAttribute(k_decode_split<T, GM>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (fe != cudaSuccess) return;
    k_decode_split<T, GM><<<grid, kDecThreads, smem, st>>>(static_cast<const T*>(q), static_cast<const T*>(k),
                                                           static_cast<const T*>(v), n, hq, hkv, per, part_o,
                                                           part_ml);
  };
  {
    TimingScope ts("decode_split", st);
    using G4 = std::integral_constant<int, 4>;
    using G8 = std::integral_constant<int, 8>;
    using G16 = std::integral_constant<int, 16>;
    if (dt == kBF16) {
      if (G <= 4) run(__nv_bfloat16(), G4());
      else if (G <= 8) run(__nv_bfloat16(), G8());
      else run(__nv_bfloat16(), G16());
    } else {
      if (G <= 4) run(float(), G4());
      else if (G <= 8) run(float(), G8());
      else run(float(), G16());
    }
  }
  if (fe != cudaSuccess) return fe;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  TimingScope ts("decode_combine", st);
  k_decode_combine<<<dim3(hq, w), kD, 0, st>>>(part_o, part_ml, nsplit, hq, w, out);
  return cudaGetLastError();
}

}  // namespace stl
