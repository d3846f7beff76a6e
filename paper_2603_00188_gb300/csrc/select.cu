// Selection kernels.  One 1024-thread CTA per KV head.
//   kSelGate: rho_i = |k_i|^-1 * max over slices of rho_part (Eq. 6), tau =
//             the min(B, |pool|)-th smallest rho (Eq. 7) by radix select,
//             gate = rho <= tau (Eq. 8).
//   kSelTopk: S from Eq. 9, then the B-th largest S by radix select and an
//             ordered stream compaction that emits the kept indices in
//             ascending order, equal scores resolved towards lower indices.
// Both selections are exact: keys are the order-preserving uint32 images of
// the fp32 values, resolved 8 bits per pass.
#include "kernels.cuh"

namespace stl {

constexpr int kSelThreads = 1024;

// Visits every token of the historical pool (visual tokens of frames
// 0..F-2), block-strided inside each frame span.
template <class Fn>
__device__ __forceinline__ void for_pool(const FrameTable& ft, Fn fn) {
  for (int f = 0; f + 1 < ft.n_frames; ++f) {
    const int b = ft.off[f], e = b + ft.gh[f] * ft.gw[f];
    for (int i = b + threadIdx.x; i < e; i += blockDim.x) fn(i);
  }
}
template <class Fn>
__device__ __forceinline__ void for_all(int n, Fn fn) {
  for (int j = threadIdx.x; j < n; j += blockDim.x) fn(j);
}

// k-th largest (1-indexed) of the keys produced by `visit`; returns the key
// T and, in *need, how many elements equal to T belong to the top k.
template <class Visit>
__device__ uint32_t radix_select_desc(Visit visit, uint32_t k, uint32_t* hist, uint32_t* sel,
                                      uint32_t* need_out) {
  uint32_t prefix = 0, mask = 0, need = k;
  const int tid = threadIdx.x, lane = tid & 31;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = tid; b < 256; b += blockDim.x) hist[b] = 0;
    __syncthreads();
    visit([&](uint32_t key) {
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    });
    __syncthreads();
    if (tid < 32) {
      uint32_t c[8], s = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        c[b] = hist[lane * 8 + b];
        s += c[b];
      }
      uint32_t incl = s;  // sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        uint32_t v = __shfl_down_sync(0xffffffffu, incl, o);
        if (lane + o < 32) incl += v;
      }
      uint32_t above = incl - s;
#pragma unroll
      for (int b = 7; b >= 0; --b) {
        if (above < need && need <= above + c[b]) {
          sel[0] = (uint32_t)(lane * 8 + b);
          sel[1] = above;
        }
        above += c[b];
      }
    }
    __syncthreads();
    const uint32_t d = sel[0];
    need -= sel[1];
    prefix |= d << shift;
    mask |= 0xffu << shift;
    __syncthreads();
  }
  *need_out = need;
  return prefix;
}

// Exclusive block-wide prefix sum of v; *total receives the block sum.
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_tot,
                                                         uint32_t* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[wid] = x;
  __syncthreads();
  if (wid == 0) {
    uint32_t t = lane < nw ? warp_tot[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint32_t y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    warp_tot[lane] = t;
  }
  __syncthreads();
  const uint32_t before = wid ? warp_tot[wid - 1] : 0u;
  *total = warp_tot[nw - 1];
  __syncthreads();
  return before + x - v;
}

__global__ void __launch_bounds__(kSelThreads) k_select(Problem p,
                                                        const __grid_constant__ FrameTable ft,
                                                        SelectArgs a) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t sel[2];
  __shared__ uint32_t warp_tot[32];
  const int h = blockIdx.x, n = p.n;
  const size_t hn = (size_t)h * n;

  if (a.mode & kSelGate) {
    float* rho = a.rho + hn;
    uint8_t* gate = a.gate + hn;
    for_all(n, [&](int j) {
      rho[j] = CUDART_NAN_F;
      gate[j] = 1;
    });
    __syncthreads();
    int pool = 0;
    for (int f = 0; f + 1 < ft.n_frames; ++f) pool += ft.gh[f] * ft.gw[f];
    if (pool > 0) {
      for_pool(ft, [&](int i) {
        float mx = -CUDART_INF_F;
        for (int c = 0; c < a.nchunk; ++c) mx = fmaxf(mx, a.rho_part[((size_t)c * p.hkv + h) * n + i]);
        rho[i] = mx * a.rn[hn + i];
      });
    }
    __syncthreads();
    if (pool > 0 && a.tsg_enable) {
      const uint32_t m = (uint32_t)min(a.budget, pool);
      uint32_t need;
      // m-th smallest rho == m-th largest of the complemented keys
      const uint32_t kt = radix_select_desc(
          [&](auto add) { for_pool(ft, [&](int i) { add(~float_key(rho[i])); }); }, m, hist, sel,
          &need);
      const float tau = key_float(~kt);
      for_pool(ft, [&](int i) { gate[i] = rho[i] <= tau ? 1 : 0; });
      if (threadIdx.x == 0) a.tau[h] = tau;
    } else if (threadIdx.x == 0) {
      a.tau[h] = CUDART_NAN_F;
    }
    __syncthreads();
  }

  if (a.mode & kSelTopk) {
    const float* ab = a.a_base + hn;
    const float* ph = a.phi ? a.phi + hn : nullptr;
    const uint8_t* gt = a.gate ? a.gate + hn : nullptr;
    float* sc = a.score + hn;
    const float alpha = a.css_enable ? a.alpha : 0.f;
    for_all(n, [&](int j) {
      float s = ab[j];
      if (find_frame(ft, j) >= 0) {
        float x = s + (alpha != 0.f ? alpha * ph[j] : 0.f);
        s = (gt == nullptr || gt[j]) ? x : 0.f;
      }
      sc[j] = s + 0.0f;
    });
    __syncthreads();
    uint32_t need;
    const uint32_t T = radix_select_desc(
        [&](auto add) { for_all(n, [&](int j) { add(float_key(sc[j])); }); },
        (uint32_t)a.budget, hist, sel, &need);
    // ordered compaction: kept = key > T, plus the first `need` keys == T
    int32_t* out = a.idx + (size_t)h * a.budget;
    uint32_t run_gt = 0, run_eq = 0;
    for (int base = 0; base < n; base += blockDim.x) {
      const int j = base + threadIdx.x;
      const uint32_t key = j < n ? float_key(sc[j]) : 0u;
      const bool g = j < n && key > T, e = j < n && key == T;
      uint32_t tot;
      const uint32_t ex = block_exclusive_scan((g ? 1u : 0u) | (e ? 0x10000u : 0u), warp_tot, &tot);
      const uint32_t gt_before = run_gt + (ex & 0xffffu), eq_before = run_eq + (ex >> 16);
      if (g || (e && eq_before < need)) out[gt_before + min(eq_before, need)] = j;
      run_gt += tot & 0xffffu;
      run_eq += tot >> 16;
    }
  }
}

cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a,
                          cudaStream_t st) {
  TimingScope ts(a.mode & kSelGate ? (a.mode & kSelTopk ? "select_gate_topk" : "select_gate") : "select_topk", st);
  k_select<<<p.hkv, kSelThreads, 0, st>>>(p, ft, a);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ gather
// k_out[r][h][:] = k[idx[h][r]][h][:] (and v): 16-byte chunks, consecutive
// threads cover consecutive chunks of one output row, so stores are fully
// coalesced and each source row is read as whole 16-byte vectors.
template <int CPR>
__global__ void __launch_bounds__(256) k_gather(const int32_t* __restrict__ idx,
                                                const uint4* __restrict__ k,
                                                const uint4* __restrict__ v, uint4* __restrict__ ko,
                                                uint4* __restrict__ vo, int n, int hkv,
                                                int budget) {
  const long long total = (long long)budget * hkv * CPR;
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(e % CPR);
    const long long rh = e / CPR;
    const int h = (int)(rh % hkv), r = (int)(rh / hkv);
    const int src = __ldg(idx + (size_t)h * budget + r);
    if (src < 0 || src >= n) continue;
    const size_t s = ((size_t)src * hkv + h) * CPR + c;
    ko[e] = __ldg(k + s);
    vo[e] = __ldg(v + s);
  }
}

cudaError_t launch_gather(const Problem& p, int budget, const int32_t* idx, const void* k,
                          const void* v, void* k_out, void* v_out, cudaStream_t st) {
  const int cpr = p.dtype == kBF16 ? kD * 2 / 16 : kD * 4 / 16;
  long long total = (long long)budget * p.hkv * cpr;
  long long blocks = (total + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  if (blocks < 1) blocks = 1;
  TimingScope ts("gather", st);
  if (cpr == 16)
    k_gather<16><<<(int)blocks, 256, 0, st>>>(idx, (const uint4*)k, (const uint4*)v, (uint4*)k_out,
                                              (uint4*)v_out, p.n, p.hkv, budget);
  else
    k_gather<32><<<(int)blocks, 256, 0, st>>>(idx, (const uint4*)k, (const uint4*)v, (uint4*)k_out,
                                              (uint4*)v_out, p.n, p.hkv, budget);
  return cudaGetLastError();
}

}  // namespace stl
