// Selection kernel.  One cluster of kSelCta CTAs per KV head; CTA c owns the
// contiguous token range [c*chunk, (c+1)*chunk) and keeps its radix keys in
// shared memory for every pass.
//   kSelGate: rho_i = |k_i|^-1 * max over slices of rho_part (Eq. 6), tau =
//             the min(B, |pool|)-th smallest rho (Eq. 7), gate = rho <= tau
//             (Eq. 8).
//   kSelTopk: S from Eq. 9, then the B-th largest S and an ordered stream
//             compaction that emits the kept indices in ascending order,
//             equal scores resolved towards lower indices.
// Both selections are exact radix selects on the order-preserving uint32
// images of the fp32 values, 8 bits per pass.  Each pass builds a per-CTA
// histogram with warp-aggregated shared atomics, then every CTA sums the
// cluster's histograms through distributed shared memory and picks the same
// digit; one cluster barrier per pass.
#include <cooperative_groups.h>

#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace stl {

constexpr int kSelCta = 8;
constexpr int kSelThreads = 1024;
constexpr int kSelMaxChunk = 46080;  // keys per CTA held in shared memory (180 KB)

struct SelShared {
  uint32_t whist[kSelThreads / 32][256];  // per-warp histograms (no cross-warp atomics)
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
  const int tid = threadIdx.x, lane = tid & 31;
  const int len_r = (len + blockDim.x - 1) / blockDim.x * blockDim.x;
  const int nw = blockDim.x >> 5, wid = tid >> 5;
  uint32_t* wh = sh.whist[wid];
  for (int shift = 24; shift >= 0; shift -= 8, ++pass) {
    uint32_t* hb = sh.hist[pass & 1];
    for (int b = lane; b < 256; b += 32) wh[b] = 0u;
    __syncwarp();
    for (int i = tid; i < len_r; i += blockDim.x) {
      const uint32_t key = i < len ? keys[i] : 0u;
      const bool valid = key != 0u && (key & mask) == prefix;
      const uint32_t bin = (key >> shift) & 255u;
      const uint32_t grp = __match_any_sync(0xffffffffu, valid ? bin : 0x100u + lane);
      if (valid && lane == __ffs(grp) - 1) wh[bin] += (uint32_t)__popc(grp);
      __syncwarp();
    }
    __syncthreads();
    for (int b = tid; b < 256; b += blockDim.x) {
      uint32_t t = 0;
      for (int w = 0; w < nw; ++w) t += sh.whist[w][b];
      hb[b] = t;
    }
    cl.sync();
    for (int b = tid; b < 256; b += blockDim.x) {
      uint32_t t = 0;
#pragma unroll
      for (int r = 0; r < kSelCta; ++r) t += cl.map_shared_rank(hb, r)[b];
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

__global__ void __cluster_dims__(kSelCta, 1, 1) __launch_bounds__(kSelThreads)
    k_select(Problem p, const __grid_constant__ FrameTable ft, SelectArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ SelShared sh;
  cg::cluster_group cl = cg::this_cluster();
  const int c = (int)cl.block_rank(), h = blockIdx.y, n = p.n, tid = threadIdx.x;
  const int chunk = (n + kSelCta - 1) / kSelCta;
  const int j0 = min(n, c * chunk), j1 = min(n, j0 + chunk), len = j1 - j0;
  const size_t hn = (size_t)h * n;
  int pass = 0;

  if (a.mode & kSelGate) {
    float* rho = a.rho + hn;
    uint8_t* gate = a.gate + hn;
    for (int i = tid; i < len; i += blockDim.x) {
      rho[j0 + i] = CUDART_NAN_F;
      gate[j0 + i] = 1;
      keys[i] = 0u;
    }
    __syncthreads();
    int pool = 0;
    for (int f = 0; f + 1 < ft.n_frames; ++f) pool += ft.gh[f] * ft.gw[f];
    for (int f = 0; f + 1 < ft.n_frames; ++f) {
      const int lo = max(ft.off[f], j0), hi = min(ft.off[f] + ft.gh[f] * ft.gw[f], j1);
      for (int i = lo + tid; i < hi; i += blockDim.x) {
        float mx = -CUDART_INF_F;
        for (int s = 0; s < a.nchunk; ++s) mx = fmaxf(mx, a.rho_part[((size_t)s * p.hkv + h) * n + i]);
        const float r = mx * a.rn[hn + i];
        rho[i] = r;
        keys[i - j0] = ~float_key(r);  // m-th smallest == m-th largest complement
      }
    }
    __syncthreads();
    if (pool > 0 && a.tsg_enable) {
      uint32_t need;
      const uint32_t kt = cluster_select_desc(cl, keys, len, (uint32_t)min(a.budget, pool), sh, pass, &need);
      const float tau = key_float(~kt);
      for (int f = 0; f + 1 < ft.n_frames; ++f) {
        const int lo = max(ft.off[f], j0), hi = min(ft.off[f] + ft.gh[f] * ft.gw[f], j1);
        for (int i = lo + tid; i < hi; i += blockDim.x) gate[i] = rho[i] <= tau ? 1 : 0;
      }
      if (c == 0 && tid == 0) a.tau[h] = tau;
    } else if (c == 0 && tid == 0) {
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
    for (int i = tid; i < len; i += blockDim.x) {
      const int j = j0 + i;
      float s = ab[j];
      if (find_frame(ft, j) >= 0) {
        const float x = s + (alpha != 0.f ? alpha * ph[j] : 0.f);
        s = (gt == nullptr || gt[j]) ? x : 0.f;
      }
      s += 0.0f;
      sc[j] = s;
      keys[i] = float_key(s);
    }
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
    int32_t* out = a.idx + (size_t)h * a.budget;
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

int select_max_tokens() { return kSelCta * kSelMaxChunk; }

cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a,
                          cudaStream_t st) {
  const int chunk = (p.n + kSelCta - 1) / kSelCta;
  if (chunk > kSelMaxChunk) return cudaErrorNotSupported;
  const size_t smem = (size_t)chunk * 4;
  cudaError_t e = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)(kSelMaxChunk * 4));
  if (e != cudaSuccess) return e;
  TimingScope ts(a.mode & kSelGate ? (a.mode & kSelTopk ? "select_gate_topk" : "select_gate") : "select_topk", st);
  k_select<<<dim3(kSelCta, p.hkv), kSelThreads, smem, st>>>(p, ft, a);
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
