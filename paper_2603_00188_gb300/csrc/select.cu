// Selection kernel.  One cluster of CL CTAs per (layer, KV head); CTA c of a
// cluster owns the contiguous token range [c*chunk, (c+1)*chunk) and keeps
// its radix keys in shared memory for every pass.
//   kSelGate: rho_i = |k_i|^-1 * max over slices of rho_part (Eq. 6), tau =
//             the min(B, |pool|)-th smallest rho (Eq. 7), gate = rho <= tau
//             (Eq. 8).
//   kSelTopk: S from Eq. 9, then the B-th largest S and an ordered stream
//             compaction that emits the kept indices in ascending order,
//             equal scores resolved towards lower indices.
// Both selections are exact radix selects on the order-preserving uint32
// images of the fp32 values, 8 bits per pass.  Each pass builds per-warp
// histograms (warp-aggregated, no cross-warp atomics), sums them per CTA,
// then every CTA sums the cluster's histograms through distributed shared
// memory and picks the same digit; one cluster barrier per pass.
#include <cooperative_groups.h>

#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace stl {

constexpr int kSelThreads = 512;
constexpr int kSelMaxCluster = 8;
constexpr int kSelMaxChunk = 49152;  // keys per CTA held in shared memory (192 KB)

struct SelShared {
  uint32_t whist[kSelThreads / 32][256];  // per-warp histograms
  uint32_t hist[2][256];  // this CTA's histogram, double-buffered by pass parity
  uint32_t tot[256];      // cluster-wide histogram of the current pass
  uint32_t bcast[4];
  uint32_t warp_tot[32];
  uint32_t counts[2];     // (greater, equal) of this CTA for the compaction
};

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

// k-th largest (1-indexed) key over the whole cluster; key 0 marks an empty
// slot.  Returns the key T; *need_out = how many keys equal to T belong to
// the top k.
__device__ uint32_t cluster_select_desc(cg::cluster_group& cl, const uint32_t* keys, int len,
                                        uint32_t k, SelShared& sh, int& pass,
                                        uint32_t* need_out) {
  uint32_t prefix = 0, mask = 0, need = k;
  const int tid = threadIdx.x, lane = tid & 31, nw = blockDim.x >> 5, wid = tid >> 5;
  const int ncta = (int)cl.num_blocks();
  uint32_t* wh = sh.whist[wid];
  for (int shift = 24; shift >= 0; shift -= 8, ++pass) {
    uint32_t* hb = sh.hist[pass & 1];
    for (int b = lane; b < 256; b += 32) wh[b] = 0u;
    __syncwarp();
    // per-warp histogram: shared atomics on the warp's own copy (lanes of one
    // warp that hit one bin are combined by the atomic unit)
    int i = tid;
    for (; i + 3 * (int)blockDim.x < len; i += 4 * blockDim.x) {
      uint32_t k4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) k4[u] = keys[i + u * blockDim.x];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (k4[u] != 0u && (k4[u] & mask) == prefix) atomicAdd(&wh[(k4[u] >> shift) & 255u], 1u);
    }
    for (; i < len; i += blockDim.x) {
      const uint32_t key = keys[i];
      if (key != 0u && (key & mask) == prefix) atomicAdd(&wh[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    for (int b = tid; b < 256; b += blockDim.x) {
      uint32_t t = 0;
#pragma unroll 8
      for (int w = 0; w < nw; ++w) t += sh.whist[w][b];
      hb[b] = t;
    }
    cl.sync();
    for (int b = tid; b < 256; b += blockDim.x) {
      uint32_t t = 0;
      for (int r = 0; r < ncta; ++r) t += cl.map_shared_rank(hb, r)[b];
      sh.tot[b] = t;
    }
    __syncthreads();
    if (tid < 32) {
      uint32_t c[8], s = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        c[b] = sh.tot[lane * 8 + b];
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
          sh.bcast[0] = (uint32_t)(lane * 8 + b);
          sh.bcast[1] = above;
        }
        above += c[b];
      }
    }
    __syncthreads();
    need -= sh.bcast[1];
    prefix |= sh.bcast[0] << shift;
    mask |= 0xffu << shift;
    __syncthreads();
  }
  *need_out = need;
  return prefix;
}

// Calls fn(i) for the tokens of [j0, j1) inside a frame's visual span, for
// the frames [f0, f1), block-strided.  Only frames that overlap [j0, j1) are
// visited (binary search for the first; the frame loop is uniform).
template <class Fn>
__device__ __forceinline__ void for_spans(const FrameTable& ft, int f0, int f1, int j0, int j1, Fn fn) {
  int lo = f0, hi = f1 - 1, first = f1;
  while (lo <= hi) {  // first frame whose span ends after j0
    const int mid = (lo + hi) >> 1;
    if (ft.off[mid] + ft.gh[mid] * ft.gw[mid] > j0) {
      first = mid;
      hi = mid - 1;
    } else {
      lo = mid + 1;
    }
  }
  for (int f = first; f < f1 && ft.off[f] < j1; ++f) {
    const int a = max(ft.off[f], j0), b = min(ft.off[f] + ft.gh[f] * ft.gw[f], j1);
    for (int i = a + (int)threadIdx.x; i < b; i += blockDim.x) fn(i);
  }
}

// Same visiting order, four tokens per thread at a time: load(i) for all four
// is issued before use(i, value) runs for any, so their latencies overlap.
template <class Load, class Use>
__device__ __forceinline__ void for_spans4(const FrameTable& ft, int f0, int f1, int j0, int j1, Load load,
                                           Use use) {
  int lo = f0, hi = f1 - 1, first = f1;
  while (lo <= hi) {
    const int mid = (lo + hi) >> 1;
    if (ft.off[mid] + ft.gh[mid] * ft.gw[mid] > j0) {
      first = mid;
      hi = mid - 1;
    } else {
      lo = mid + 1;
    }
  }
  const int B = blockDim.x;
  for (int f = first; f < f1 && ft.off[f] < j1; ++f) {
    const int a = max(ft.off[f], j0), b = min(ft.off[f] + ft.gh[f] * ft.gw[f], j1);
    for (int i0 = a + (int)threadIdx.x; i0 < b; i0 += 4 * B) {
      decltype(load(i0)) v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u * B < b) v[u] = load(i0 + u * B);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u * B < b) use(i0 + u * B, v[u]);
    }
  }
}

__global__ void __launch_bounds__(kSelThreads) k_select(Problem p, const __grid_constant__ FrameTable ft,
                                                        SelectArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ SelShared sh;
  cg::cluster_group cl = cg::this_cluster();
  const int ncta = (int)cl.num_blocks(), c = (int)cl.block_rank();
  const int l = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv, n = p.n, tid = threadIdx.x;
  const int chunk = (n + ncta - 1) / ncta;
  const int j0 = min(n, c * chunk), j1 = min(n, j0 + chunk), len = j1 - j0;
  const size_t hn = (size_t)h * n;
  const int F = ft.n_frames;
  int pass = 0;

  if (a.mode & kSelGate) {
    float* rho = a.rho.at(l) + hn;
    uint8_t* gate = a.gate.at(l) + hn;
    const float* rp = a.rho_part.at(l);
    const float* rn = a.rn.at(l) + hn;
    for (int i = tid; i < len; i += blockDim.x) {
      rho[j0 + i] = CUDART_NAN_F;
      gate[j0 + i] = 1;
      keys[i] = 0u;
    }
    __syncthreads();
    int pool = 0;
    for (int f = 0; f + 1 < F; ++f) pool += ft.gh[f] * ft.gw[f];
    const size_t slice = (size_t)p.hkv * n;
    for_spans4(
        ft, 0, F - 1, j0, j1,
        [&](int i) {
          const float* src = rp + hn + i;
          float m0 = -CUDART_INF_F, m1 = -CUDART_INF_F;
          int s = 0;
          for (; s + 1 < a.nchunk; s += 2) {
            m0 = fmaxf(m0, __ldg(src + (size_t)s * slice));
            m1 = fmaxf(m1, __ldg(src + (size_t)(s + 1) * slice));
          }
          if (s < a.nchunk) m0 = fmaxf(m0, __ldg(src + (size_t)s * slice));
          return make_float2(fmaxf(m0, m1), __ldg(rn + i));
        },
        [&](int i, float2 v) {
          const float r = v.x * v.y;
          rho[i] = r;
          keys[i - j0] = ~float_key(r);  // m-th smallest == m-th largest complement
        });
    __syncthreads();
    if (pool > 0 && a.tsg_enable) {
      uint32_t need;
      const uint32_t kt = cluster_select_desc(cl, keys, len, (uint32_t)min(a.budget, pool), sh, pass, &need);
      const float tau = key_float(~kt);
      for_spans(ft, 0, F - 1, j0, j1, [&](int i) { gate[i] = key_float(~keys[i - j0]) <= tau ? 1 : 0; });
      if (c == 0 && tid == 0) a.tau.at(l)[h] = tau;
    } else if (c == 0 && tid == 0) {
      a.tau.at(l)[h] = CUDART_NAN_F;
    }
    __syncthreads();
  }

  if (a.mode & kSelTopk) {
    const float* ab = a.a_base.at(l) + hn;
    const float* ph = a.phi.base ? a.phi.at(l) + hn : nullptr;
    const uint8_t* gt = a.gate.base ? a.gate.at(l) + hn : nullptr;
    float* sc = a.score.at(l) + hn;
    const float alpha = a.css_enable ? a.alpha : 0.f;
    // text tokens: S = A_base; visual tokens are overwritten below
    for (int i0 = tid; i0 < len; i0 += 4 * blockDim.x) {
      float v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u * (int)blockDim.x < len) v[u] = __ldg(ab + j0 + i0 + u * blockDim.x);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * blockDim.x;
        if (i < len) {
          const float s = v[u] + 0.0f;
          sc[j0 + i] = s;
          keys[i] = float_key(s);
        }
      }
    }
    __syncthreads();
    for_spans4(
        ft, 0, F, j0, j1,
        [&](int j) {
          const float x = __ldg(ab + j) + (alpha != 0.f ? alpha * __ldg(ph + j) : 0.f);
          return (gt == nullptr || gt[j]) ? x : 0.f;
        },
        [&](int j, float x) {
          const float s = x + 0.0f;
          sc[j] = s;
          keys[j - j0] = float_key(s);
        });
    __syncthreads();
    uint32_t need;
    const uint32_t T = cluster_select_desc(cl, keys, len, (uint32_t)a.budget, sh, pass, &need);
    // this CTA's counts, then its offsets from the lower-ranked CTAs
    uint32_t g_loc = 0, e_loc = 0;
    for (int i = tid; i < len; i += blockDim.x) {
      g_loc += keys[i] > T;
      e_loc += keys[i] == T;
    }
    uint32_t tot;
    block_exclusive_scan(g_loc | (e_loc << 16), sh.warp_tot, &tot);
    if (tid == 0) {
      sh.counts[0] = tot & 0xffffu;
      sh.counts[1] = tot >> 16;
    }
    cl.sync();
    if (tid == 0) {
      uint32_t gb = 0, eb = 0;
      for (int r = 0; r < c; ++r) {
        const uint32_t* rc = cl.map_shared_rank(sh.counts, r);
        gb += rc[0];
        eb += rc[1];
      }
      sh.bcast[2] = gb;
      sh.bcast[3] = eb;
    }
    __syncthreads();
    uint32_t run_gt = sh.bcast[2], run_eq = sh.bcast[3];
    int32_t* out = a.idx[l] + (size_t)h * a.budget;
    for (int base = 0; base < len; base += blockDim.x) {
      const int i = base + tid;
      const uint32_t key = i < len ? keys[i] : 0u;
      const bool g = i < len && key > T, e = i < len && key == T;
      const uint32_t ex = block_exclusive_scan((g ? 1u : 0u) | (e ? 0x10000u : 0u), sh.warp_tot, &tot);
      const uint32_t gt_before = run_gt + (ex & 0xffffu), eq_before = run_eq + (ex >> 16);
      if (g || (e && eq_before < need)) out[gt_before + min(eq_before, need)] = j0 + i;
      run_gt += tot & 0xffffu;
      run_eq += tot >> 16;
    }
  }
  cl.sync();  // no CTA leaves while a peer may still read its shared memory
}

int select_max_tokens() { return kSelMaxCluster * kSelMaxChunk; }

cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a, cudaStream_t st) {
  // smallest cluster whose CTAs hold their keys in shared memory, grown
  // (up to 8) while the launch does not fill one wave of the SMs
  int cl = 1;
  while ((p.n + cl - 1) / cl > kSelMaxChunk) cl <<= 1;
  if (cl > kSelMaxCluster) return cudaErrorNotSupported;
  while (cl < kSelMaxCluster && p.L * p.hkv * cl * 2 <= 152) cl <<= 1;
  const int chunk = (p.n + cl - 1) / cl;
  cudaError_t e = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kSelMaxChunk * 4));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cl, p.L * p.hkv, 1);
  cfg.blockDim = dim3(kSelThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)chunk * 4;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  TimingScope ts(a.mode & kSelGate ? (a.mode & kSelTopk ? "select_gate_topk" : "select_gate") : "select_topk", st);
  e = cudaLaunchKernelEx(&cfg, k_select, p, ft, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// ------------------------------------------------------------------ gather
// k_out[l][r][h][:] = k_l[idx[l][h][r]][h][:] (and v): 16-byte chunks, four
// rows per thread in flight, consecutive threads cover consecutive chunks of
// one output row (coalesced stores, whole 16-byte source vectors).
// grid.y = layer.
template <int CPR>
__global__ void __launch_bounds__(256) k_gather(const __grid_constant__ LayerPtrs io, int n, int hkv,
                                                int budget) {
  const int l = blockIdx.y;
  const int32_t* idx = io.idx[l];
  const uint4* k = static_cast<const uint4*>(io.k[l]);
  const uint4* v = static_cast<const uint4*>(io.v[l]);
  uint4* ko = static_cast<uint4*>(io.k_out[l]);
  uint4* vo = static_cast<uint4*>(io.v_out[l]);
  const long long total = (long long)budget * hkv * CPR;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long e0 = (long long)blockIdx.x * blockDim.x + threadIdx.x; e0 < total; e0 += 4 * stride) {
    uint4 kv[4], vv[4];
    long long ee[4];
    bool ok[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const long long e = e0 + u * stride;
      ee[u] = e;
      ok[u] = false;
      if (e < total) {
        const int c = (int)(e % CPR);
        const long long rh = e / CPR;
        const int h = (int)(rh % hkv), r = (int)(rh / hkv);
        const int src = __ldg(idx + (size_t)h * budget + r);
        if (src >= 0 && src < n) {
          const size_t s = ((size_t)src * hkv + h) * CPR + c;
          kv[u] = __ldg(k + s);
          vv[u] = __ldg(v + s);
          ok[u] = true;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (ok[u]) {
        ko[ee[u]] = kv[u];
        vo[ee[u]] = vv[u];
      }
    }
  }
}

cudaError_t launch_gather(const Problem& p, int budget, const LayerPtrs& io, cudaStream_t st) {
  const int cpr = p.dtype == kBF16 ? kD * 2 / 16 : kD * 4 / 16;
  long long total = (long long)budget * p.hkv * cpr;
  long long blocks = (total + 1023) / 1024;
  long long cap = (152 * 8 + p.L - 1) / p.L;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  TimingScope ts("gather", st);
  dim3 grid((unsigned)blocks, p.L);
  if (cpr == 16)
    k_gather<16><<<grid, 256, 0, st>>>(io, p.n, p.hkv, budget);
  else
    k_gather<32><<<grid, 256, 0, st>>>(io, p.n, p.hkv, budget);
  return cudaGetLastError();
}

}  // namespace stl
