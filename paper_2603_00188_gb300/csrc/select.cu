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

constexpr int kSelThreads = 512;  // two per histogram bin in the radix passes
constexpr int kSelMaxCluster = 8;
constexpr int kSelMaxChunk = 49152;  // keys per CTA held in shared memory (192 KB)

struct SelShared {
  uint32_t whist[kSelThreads / 32][256];  // per-warp histograms
  uint32_t hist[2][256];  // this CTA's histogram, double-buffered by pass parity
  uint32_t tot[256];      // cluster-wide histogram of the current pass
  uint32_t dig[2][3];     // (digit, count above it, count in it), double-buffered by pass parity
  uint32_t bcast[4];
  uint32_t warp_tot[32];
  uint32_t counts[2];     // (greater, equal) of this CTA for the compaction
  float warp_max[32];
  float cta_max;          // read by the cluster's other CTAs
  int32_t fr_off[kMaxFrames + 1];  // first token of every frame; fr_off[F] = INT_MAX
  int32_t fr_vend[kMaxFrames];     // end of every frame's visual span
};

// Maximum of v over every thread of the cluster (every CTA must call it).
__device__ float cluster_max(cg::cluster_group& cl, float v, SelShared& sh) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (lane == 0) sh.warp_max[wid] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float m = sh.warp_max[0];
    for (int w = 1; w < nw; ++w) m = fmaxf(m, sh.warp_max[w]);
    sh.cta_max = m;
  }
  cl.sync();
  float m = -CUDART_INF_F;
  for (int r = 0; r < (int)cl.num_blocks(); ++r) m = fmaxf(m, *cl.map_shared_rank(&sh.cta_max, r));
  return m;
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

// k-th largest (1-indexed) key over the whole cluster; key 0 marks an empty
// slot.  Returns the key T; *need_out = how many keys equal to T belong to
// the top k.  Per pass: per-warp histograms, one block barrier, the CTA's
// histogram (two threads per bin), one cluster barrier, the cluster's
// histogram (two threads per bin, each reading half of the CTAs), one block
// barrier, the digit found by warp 0, one block barrier.  The CTA histogram
// and the digit broadcast are double-buffered by pass parity, so that no
// barrier is needed before the next pass rewrites them: a buffer is
// rewritten two passes later, after every thread has passed the barriers
// that follow its last read.  early: the caller needs only the top-k set,
// not the k-th key itself, so the select may stop once the chosen bin holds
// exactly the keys still needed (all of them belong to the top k); it then
// returns the bin's lower bound minus one with *need_out = 0, which selects
// the same set.  Every CTA of the cluster takes that decision on the same
// cluster histogram.
__device__ uint32_t cluster_select_desc(cg::cluster_group& cl, const uint32_t* keys, int len,
                                        uint32_t k, SelShared& sh, int& pass,
                                        uint32_t* need_out, bool early) {
  uint32_t prefix = 0, mask = 0, need = k;
  const int tid = threadIdx.x, lane = tid & 31, nw = blockDim.x >> 5, wid = tid >> 5;
  const int ncta = (int)cl.num_blocks();
  uint32_t* wh = sh.whist[wid];
  const int bin = tid >> 1, half = tid & 1;  // 512 threads: two per bin
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
    {
      uint32_t t = 0;
      const int w0 = half * (nw >> 1), w1 = w0 + (nw >> 1);
#pragma unroll 8
      for (int w = w0; w < w1; ++w) t += sh.whist[w][bin];
      t += __shfl_xor_sync(0xffffffffu, t, 1);
      if (half == 0) hb[bin] = t;
    }
    cl.sync();
    {
      uint32_t t = 0;
      for (int r0 = half; r0 < ncta; r0 += 8) {  // four remote reads in flight
        uint32_t v[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) v[r] = r0 + 2 * r < ncta ? cl.map_shared_rank(hb, r0 + 2 * r)[bin] : 0u;
        t += (v[0] + v[1]) + (v[2] + v[3]);
      }
      t += __shfl_xor_sync(0xffffffffu, t, 1);
      if (half == 0) sh.tot[bin] = t;
    }
    __syncthreads();
    // warp 0: lane L holds bins 8L .. 8L+7; the digit is the bin where the
    // count of larger keys first reaches need
    uint32_t* dg = sh.dig[pass & 1];
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
          dg[0] = (uint32_t)(lane * 8 + b);
          dg[1] = above;
          dg[2] = c[b];
        }
        above += c[b];
      }
    }
    __syncthreads();
    need -= dg[1];
    prefix |= dg[0] << shift;
    mask |= 0xffu << shift;
    if (early && shift > 0 && dg[2] == need && prefix != 0u) {
      ++pass;  // the parity sequence of the double buffers goes on
      *need_out = 0u;
      return prefix - 1u;
    }
  }
  *need_out = need;
  return prefix;
}

// Warms L2 with the 128-byte lines of x[j0, j1) (one prefetch per line):
// the token loops then find their inputs in L2 instead of waiting on DRAM
// once per batch.
__device__ __forceinline__ void prefetch_l2(const void* x, size_t elem, int j0, int j1) {
  const char* b = static_cast<const char*>(x);
  const size_t lo = (size_t)j0 * elem, hi = (size_t)j1 * elem;
  for (size_t o = (lo & ~(size_t)127) + (size_t)threadIdx.x * 128; o < hi; o += (size_t)blockDim.x * 128)
    asm volatile("prefetch.global.L2 [%0];" ::"l"(b + o));
}

// Inputs of one pool token's rho: the row maxima of the TSG slices (folded
// into four) and 1/|k_i|.
struct RhoIn {
  float s[4];
  float rn;
};

// Token kinds of the flat loops.
constexpr int kTokText = 0;  // not inside any frame's visual span
constexpr int kTokPool = 1;  // visual token of a historical frame (the TSG pool)
constexpr int kTokCur = 2;   // visual token of the current (last) frame

// Last frame starting at or before token t (-1: none), on the shared copy
// of the frame table.
__device__ __forceinline__ int frame_at(const SelShared& sh, int F, int t) {
  int lo = 0, hi = F - 1, f = -1;
  while (lo <= hi) {
    const int mid = (lo + hi) >> 1;
    if (sh.fr_off[mid] <= t) {
      f = mid;
      lo = mid + 1;
    } else {
      hi = mid - 1;
    }
  }
  return f;
}

// Visits the tokens j0 + threadIdx.x + k * blockDim.x of [j0, j1) in
// batches of U per thread: load(t, kind) runs for the whole batch before
// use(t, kind, value) runs for any of it, so the batch's memory latencies
// overlap.  Each thread tracks the frame of its (increasing) tokens in the
// shared copy of the frame table (fr_off ends with INT_MAX).
template <int U, class Load, class Use>
__device__ __forceinline__ void for_tokens(const SelShared& sh, int F, int j0, int j1, Load load, Use use) {
  const int B = blockDim.x;
  int f = frame_at(sh, F, j0 + (int)threadIdx.x);
  for (int base = j0 + (int)threadIdx.x; base < j1; base += U * B) {
    int kind[U];
    decltype(load(0, 0)) v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int t = base + u * B;
      kind[u] = -1;
      if (t < j1) {
        while (sh.fr_off[f + 1] <= t) ++f;
        const bool vis = f >= 0 && t < sh.fr_vend[f];
        kind[u] = vis ? (f + 1 < F ? kTokPool : kTokCur) : kTokText;
        v[u] = load(t, kind[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (kind[u] >= 0) use(base + u * B, kind[u], v[u]);
  }
}

// The same visit in groups of four consecutive tokens t0 .. t0 + 3 (t0 =
// j0 + 4 (tid + k B)), for 128-bit loads and stores: j0, j1 and every row
// base are multiples of four tokens.  kinds[e] is the kind of t0 + e (one
// comparison for a group inside one visual span or text run).
template <class Load4, class Use4>
__device__ __forceinline__ void for_tokens4(const SelShared& sh, int F, int j0, int j1, Load4 load4, Use4 use4) {
  const int B = blockDim.x;
  int f = frame_at(sh, F, j0 + 4 * (int)threadIdx.x);
  for (int t0 = j0 + 4 * (int)threadIdx.x; t0 < j1; t0 += 4 * B) {
    int kinds[4];
    while (sh.fr_off[f + 1] <= t0) ++f;
    const int vend = f >= 0 ? sh.fr_vend[f] : -1, next = sh.fr_off[f + 1];
    if (t0 + 3 < vend || (t0 >= vend && t0 + 3 < next)) {  // one kind for the group
      const int k = t0 < vend ? (f + 1 < F ? kTokPool : kTokCur) : kTokText;
#pragma unroll
      for (int e = 0; e < 4; ++e) kinds[e] = k;
    } else {  // the group straddles a span or frame boundary
      int fe = f;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int t = t0 + e;
        while (sh.fr_off[fe + 1] <= t) ++fe;
        kinds[e] = fe >= 0 && t < sh.fr_vend[fe] ? (fe + 1 < F ? kTokPool : kTokCur) : kTokText;
      }
    }
    const auto v = load4(t0, kinds);
    use4(t0, kinds, v);
  }
}

struct RhoIn4 {
  float4 s[4];
  float4 rn;
};
struct ScoreIn4 {
  float4 A, P;
  uint32_t G;  // four gate bytes
};

__global__ void __launch_bounds__(kSelThreads, 4) k_select(Problem p, const __grid_constant__ FrameTable ft,
                                                        SelectArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ SelShared sh;
  cg::cluster_group cl = cg::this_cluster();
  const int ncta = (int)cl.num_blocks(), c = (int)cl.block_rank();
  const int l = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv, n = p.n, tid = threadIdx.x;
  const int chunk = ((n + ncta - 1) / ncta + 3) & ~3;  // four-token groups never straddle two CTAs
  const int j0 = min(n, c * chunk), j1 = min(n, j0 + chunk), len = j1 - j0;
  const bool vec = (n & 3) == 0;  // every row base [Hkv][N] is 16-byte aligned
  const size_t hn = (size_t)h * n;
  const int F = ft.n_frames;
  int pass = 0;
  int pool = 0;
  for (int f = 0; f + 1 < F; ++f) pool += ft.gh[f] * ft.gw[f];
  // the frame table in shared memory for the token loops' frame tracking
  for (int f = tid; f <= F; f += blockDim.x) {
    sh.fr_off[f] = f < F ? ft.off[f] : 0x7fffffff;
    if (f < F) sh.fr_vend[f] = ft.off[f] + ft.gh[f] * ft.gw[f];
  }
  __syncthreads();
  // tau comes from a selection only when there is a pool and TSG is on;
  // otherwise tau = NaN and every gate stays open
  const bool gate_sel = (a.mode & kSelGate) && pool > 0 && a.tsg_enable;
  float tau = CUDART_NAN_F;
  uint32_t kt_gate = 0u;  // gate: rho <= tau, i.e. key (~float_key(rho)) >= kt_gate
  uint8_t* gate = a.gate.base ? a.gate.at(l) + hn : nullptr;

  if (a.mode & kSelGate) {
    float* rho = a.rho.at(l) + hn;
    const float* rp = a.rho_part.at(l) + hn;
    const float* rn = a.rn.at(l) + hn;
    const size_t slice = (size_t)p.hkv * n;
    const int nsl = a.nchunk;
    for (int s = 0; s < nsl; ++s) prefetch_l2(rp + (size_t)s * slice, 4, j0, j1);
    prefetch_l2(rn, 4, j0, j1);
    // rho of every token: pool tokens from the TSG slices and 1/|k_i|, NaN
    // elsewhere; the selection keys are complements (m-th smallest rho ==
    // m-th largest key), 0 marks a token outside the pool.  Finish Eq. 6
    // with the row's own term: times 1/|k_i| (cosine), nothing (dot), minus
    // |k_i|^2 (negative squared L2).
    auto finish = [&](float m, float rnv) {
      return a.tsg_metric == kTsgCosine ? m * rnv : (a.tsg_metric == kTsgDot ? m : m - 1.f / (rnv * rnv));
    };
    if (vec) {
      for_tokens4(
          sh, F, j0, j1,
          [&](int t0, const int (&kinds)[4]) {
            RhoIn4 r;
            const float ninf = -CUDART_INF_F;
#pragma unroll
            for (int s = 0; s < 4; ++s) r.s[s] = make_float4(ninf, ninf, ninf, ninf);
            r.rn = make_float4(0.f, 0.f, 0.f, 0.f);
            if (kinds[0] == kTokPool || kinds[1] == kTokPool || kinds[2] == kTokPool || kinds[3] == kTokPool) {
              const float* src = rp + t0;
#pragma unroll
              for (int s = 0; s < 4; ++s)
                if (s < nsl) r.s[s] = __ldg(reinterpret_cast<const float4*>(src + (size_t)s * slice));
              for (int s = 4; s < nsl; ++s) {
                const float4 x = __ldg(reinterpret_cast<const float4*>(src + (size_t)s * slice));
                r.s[3] = make_float4(fmaxf(r.s[3].x, x.x), fmaxf(r.s[3].y, x.y), fmaxf(r.s[3].z, x.z),
                                     fmaxf(r.s[3].w, x.w));
              }
              r.rn = __ldg(reinterpret_cast<const float4*>(rn + t0));
            }
            return r;
          },
          [&](int t0, const int (&kinds)[4], const RhoIn4& v) {
            const float m0 = fmaxf(fmaxf(v.s[0].x, v.s[1].x), fmaxf(v.s[2].x, v.s[3].x));
            const float m1 = fmaxf(fmaxf(v.s[0].y, v.s[1].y), fmaxf(v.s[2].y, v.s[3].y));
            const float m2 = fmaxf(fmaxf(v.s[0].z, v.s[1].z), fmaxf(v.s[2].z, v.s[3].z));
            const float m3 = fmaxf(fmaxf(v.s[0].w, v.s[1].w), fmaxf(v.s[2].w, v.s[3].w));
            const float r0 = kinds[0] == kTokPool ? finish(m0, v.rn.x) : CUDART_NAN_F;
            const float r1 = kinds[1] == kTokPool ? finish(m1, v.rn.y) : CUDART_NAN_F;
            const float r2 = kinds[2] == kTokPool ? finish(m2, v.rn.z) : CUDART_NAN_F;
            const float r3 = kinds[3] == kTokPool ? finish(m3, v.rn.w) : CUDART_NAN_F;
            if (a.write_stages) *reinterpret_cast<float4*>(rho + t0) = make_float4(r0, r1, r2, r3);
            *reinterpret_cast<uint4*>(keys + (t0 - j0)) =
                make_uint4(kinds[0] == kTokPool ? ~float_key(r0) : 0u, kinds[1] == kTokPool ? ~float_key(r1) : 0u,
                           kinds[2] == kTokPool ? ~float_key(r2) : 0u, kinds[3] == kTokPool ? ~float_key(r3) : 0u);
          });
    } else
    for_tokens<2>(
        sh, F, j0, j1,
        [&](int t, int kind) {
          // independent loads (no max between them), so that all of a
          // batch's slices are in flight together
          RhoIn r;
#pragma unroll
          for (int s = 0; s < 4; ++s) r.s[s] = -CUDART_INF_F;
          r.rn = CUDART_NAN_F;
          if (kind == kTokPool) {
            const float* src = rp + t;
#pragma unroll
            for (int s = 0; s < 4; ++s)
              if (s < nsl) r.s[s] = __ldg(src + (size_t)s * slice);
            for (int s = 4; s < nsl; ++s) r.s[3] = fmaxf(r.s[3], __ldg(src + (size_t)s * slice));
            r.rn = __ldg(rn + t);
          }
          return r;
        },
        [&](int t, int kind, const RhoIn& v) {
          const float m = fmaxf(fmaxf(v.s[0], v.s[1]), fmaxf(v.s[2], v.s[3]));
          const float r = kind == kTokPool ? finish(m, v.rn) : CUDART_NAN_F;
          if (a.write_stages) rho[t] = r;
          keys[t - j0] = kind == kTokPool ? ~float_key(r) : 0u;
        });
    __syncthreads();
    // the score phase's inputs arrive in L2 while tau is selected
    if ((a.mode & kSelTopk) && !a.base_uniform) prefetch_l2(a.a_base.at(l) + hn, 4, j0, j1);
    if ((a.mode & kSelTopk) && a.phi.base && a.css_enable) prefetch_l2(a.phi.at(l) + hn, 4, j0, j1);
    if (gate_sel) {
      if (a.tsg_fixed) {
        tau = a.tsg_fixed_tau;  // fixed-threshold control: no selection
        kt_gate = ~float_key(tau);
      } else {
        // the fused call needs only the gated set; the staged call reports tau
        uint32_t need;
        kt_gate = cluster_select_desc(cl, keys, len, (uint32_t)min(a.budget[l], pool), sh, pass, &need,
                                      !a.write_stages);
        tau = key_float(~kt_gate);
      }
    }
    if (c == 0 && tid == 0) a.tau.at(l)[h] = tau;
    if (!(a.mode & kSelTopk)) {
      // gate only: Eq. 8 on the pool, open elsewhere
      for_tokens<2>(
          sh, F, j0, j1, [&](int, int) { return 0; },
          [&](int t, int kind, int) {
            gate[t] = (kind == kTokPool && gate_sel) ? (keys[t - j0] >= kt_gate ? 1 : 0) : 1;
          });
    }
  }

  if (a.mode & kSelTopk) {
    const float* ab = a.base_uniform ? nullptr : a.a_base.at(l) + hn;
    const float* ph = a.phi.base ? a.phi.at(l) + hn : nullptr;
    const uint8_t* gt = gate;
    float* sc = a.score.at(l) + hn;
    const float alpha = a.css_enable ? a.alpha : 0.f;
    const bool fused = (a.mode & kSelGate) != 0;  // gate decided here from the rho keys
    // optional A / max_j A (per head): the cluster-wide maximum first
    float amax = 0.f;
    if (a.a_norm_max) {
      if (ab) {
        float m = 0.f;
        for (int t = j0 + tid; t < j1; t += blockDim.x) m = fmaxf(m, __ldg(ab + t));
        amax = cluster_max(cl, m, sh);
      } else {
        amax = a.a_uniform;
      }
    }
    const bool a_div = amax > 0.f;
    // Eq. 9: S = A_base for text tokens; for visual tokens S = A_base +
    // alpha * Phi where the gate is open and 0 where it is closed
    auto score_of = [&](int t, int kind, float A, float P, float G) {
      float s;
      if (kind == kTokText) {
        s = A + 0.0f;
        if (fused && a.write_stages) gate[t] = 1;
      } else {
        bool g = G != 0.f;
        if (fused) {
          g = !(kind == kTokPool && gate_sel) || keys[t - j0] >= kt_gate;
          if (a.write_stages) gate[t] = g ? 1 : 0;
        }
        const float x = alpha != 0.f ? __fmaf_rn(alpha, P, A) : A;
        s = (g ? x : 0.f) + 0.0f;
      }
      return s;
    };
    if (vec) {
      for_tokens4(
          sh, F, j0, j1,
          [&](int t0, const int (&kinds)[4]) {
            ScoreIn4 v;
            v.A = ab ? __ldg(reinterpret_cast<const float4*>(ab + t0))
                     : make_float4(a.a_uniform, a.a_uniform, a.a_uniform, a.a_uniform);
            if (a_div)
              v.A = make_float4(__fdiv_rn(v.A.x, amax), __fdiv_rn(v.A.y, amax), __fdiv_rn(v.A.z, amax),
                                __fdiv_rn(v.A.w, amax));
            const bool vis = kinds[0] != kTokText || kinds[1] != kTokText || kinds[2] != kTokText ||
                             kinds[3] != kTokText;
            v.P = (vis && alpha != 0.f) ? __ldg(reinterpret_cast<const float4*>(ph + t0)) : make_float4(0.f, 0.f, 0.f, 0.f);
            v.G = (vis && !fused && gt != nullptr) ? __ldg(reinterpret_cast<const uint32_t*>(gt + t0)) : 0x01010101u;
            return v;
          },
          [&](int t0, const int (&kinds)[4], const ScoreIn4& v) {
            const float s0 = score_of(t0, kinds[0], v.A.x, kinds[0] != kTokText ? v.P.x : 0.f, (float)(v.G & 0xffu));
            const float s1 = score_of(t0 + 1, kinds[1], v.A.y, kinds[1] != kTokText ? v.P.y : 0.f,
                                      (float)((v.G >> 8) & 0xffu));
            const float s2 = score_of(t0 + 2, kinds[2], v.A.z, kinds[2] != kTokText ? v.P.z : 0.f,
                                      (float)((v.G >> 16) & 0xffu));
            const float s3 = score_of(t0 + 3, kinds[3], v.A.w, kinds[3] != kTokText ? v.P.w : 0.f,
                                      (float)(v.G >> 24));
            if (a.write_stages) *reinterpret_cast<float4*>(sc + t0) = make_float4(s0, s1, s2, s3);
            *reinterpret_cast<uint4*>(keys + (t0 - j0)) =
                make_uint4(float_key(s0), float_key(s1), float_key(s2), float_key(s3));
          });
    } else
    for_tokens<2>(
        sh, F, j0, j1,
        [&](int t, int kind) {
          float A = ab ? __ldg(ab + t) : a.a_uniform;
          if (a_div) A = __fdiv_rn(A, amax);
          const float P = (kind != kTokText && alpha != 0.f) ? __ldg(ph + t) : 0.f;
          const float G = (kind != kTokText && !fused && gt != nullptr) ? (float)gt[t] : 1.f;
          return make_float3(A, P, G);
        },
        [&](int t, int kind, float3 v) {
          const float s = score_of(t, kind, v.x, v.y, v.z);
          if (a.write_stages) sc[t] = s;
          keys[t - j0] = float_key(s);
        });
    __syncthreads();
    uint32_t need;
    const uint32_t T = cluster_select_desc(cl, keys, len, (uint32_t)a.budget[l], sh, pass, &need, true);
    // Ordered compaction.  Thread tid owns the contiguous run [r0, r1) of
    // this CTA's keys (odd run length: conflict-free shared reads); one
    // block scan gives its (greater, equal) counts before the run, the
    // cluster's lower ranks add theirs.
    const int per = ((len + (int)blockDim.x - 1) / (int)blockDim.x) | 1;
    const int r0 = min(len, tid * per), r1 = min(len, r0 + per);
    uint32_t g_loc = 0, e_loc = 0;
    for (int i = r0; i < r1; ++i) {
      const uint32_t k = keys[i];
      g_loc += k > T;
      e_loc += k == T;
    }
    uint32_t tot;
    const uint32_t ex = block_exclusive_scan(g_loc | (e_loc << 16), sh.warp_tot, &tot);
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
    uint32_t gt_before = sh.bcast[2] + (ex & 0xffffu), eq_before = sh.bcast[3] + (ex >> 16);
    int32_t* out = a.idx[l] + (size_t)h * a.budget[l];
    // kept: every key > T, and the first `need` keys == T in index order;
    // a kept token's slot = kept tokens before it
    for (int i = r0; i < r1; ++i) {
      const uint32_t k = keys[i];
      if (k > T) {
        out[gt_before + min(eq_before, need)] = j0 + i;
        ++gt_before;
      } else if (k == T) {
        if (eq_before < need) out[gt_before + eq_before] = j0 + i;
        ++eq_before;
      }
    }
  }
  cl.sync();  // no CTA leaves while a peer may still read its shared memory
}

int select_max_tokens() { return kSelMaxCluster * kSelMaxChunk; }

static void select_config(cudaLaunchConfig_t* cfg, cudaLaunchAttribute* attr, const Problem& p, int cl,
                          cudaStream_t st) {
  *cfg = cudaLaunchConfig_t{};
  cfg->gridDim = dim3(cl, p.L * p.hkv, 1);
  cfg->blockDim = dim3(kSelThreads, 1, 1);
  cfg->dynamicSmemBytes = (size_t)(((p.n + cl - 1) / cl + 3) & ~3) * 4;
  cfg->stream = st;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg->attrs = attr;
  cfg->numAttrs = 1;
}

cudaError_t launch_select(const Problem& p, const FrameTable& ft, const SelectArgs& a, cudaStream_t st) {
  // Cluster size: the CTAs of a cluster split one (layer, head)'s tokens.
  // Each CTA is latency-bound on its own chunk, so the estimated time is
  // (waves of co-resident clusters) x (chunk length); the smallest cluster
  // with the lowest estimate wins (fewer CTAs per cluster barrier).
  cudaError_t e = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kSelMaxChunk * 4));
  if (e != cudaSuccess) return e;
  // all of the SM's configurable memory as shared memory: the CTAs' keys
  // are what limits how many clusters are resident
  e = cudaFuncSetAttribute(k_select, cudaFuncAttributePreferredSharedMemoryCarveout,
                           (int)cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  int cl = 0, fit8 = 0;
  long long best = 0;
  const long long units = (long long)p.L * p.hkv;
  for (int c = 1; c <= kSelMaxCluster; c <<= 1) {
    const int ch = ((p.n + c - 1) / c + 3) & ~3;
    if (ch > kSelMaxChunk) continue;
    select_config(&cfg, attr, p, c, st);
    int fit = 0;
    if ((e = cudaOccupancyMaxActiveClusters(&fit, k_select, &cfg)) != cudaSuccess) return e;
    if (c == kSelMaxCluster) fit8 = fit;
    if (fit < 1) continue;
    const long long est = (units + fit - 1) / fit * ch;
    if (cl == 0 || est < best) {
      cl = c;
      best = est;
    }
  }
  // A few (layer, head) problems (one layer, a couple of layers) leave most
  // SMs idle even with clusters of 8: clusters of 16 (non-portable) halve
  // each CTA's tokens.  Only while they take at most one CTA per SM (the
  // 16-CTA barriers cost more once CTAs share SMs), so that batches keep
  // their portable shape.
  int nsm = 0, dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    nsm = 0;
  if (cl == kSelMaxCluster && units <= fit8 && units * 2 * kSelMaxCluster <= nsm &&
      cudaFuncSetAttribute(k_select, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
    const int c = 2 * kSelMaxCluster;
    select_config(&cfg, attr, p, c, st);
    int fit = 0;
    if (cudaOccupancyMaxActiveClusters(&fit, k_select, &cfg) == cudaSuccess && fit >= units) cl = c;
  }
  (void)cudaGetLastError();  // a refused non-portable query leaves no error behind
  if (cl == 0) return cudaErrorNotSupported;
  select_config(&cfg, attr, p, cl, st);
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
__global__ void __launch_bounds__(256) k_gather(const __grid_constant__ LayerPtrs io, int n, int hkv) {
  const int l = blockIdx.y;
  const int budget = io.budget[l];
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
          vv[u] = v[s];  // plain load: v may be page-locked host memory
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

cudaError_t launch_gather(const Problem& p, const LayerPtrs& io, cudaStream_t st) {
  const int cpr = p.dtype == kBF16 ? kD * 2 / 16 : kD * 4 / 16;
  int bmax = 1;
  for (int l = 0; l < p.L; ++l) bmax = io.budget[l] > bmax ? io.budget[l] : bmax;
  long long total = (long long)bmax * p.hkv * cpr;
  long long blocks = (total + 1023) / 1024;
  long long cap = (152 * 8 + p.L - 1) / p.L;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  TimingScope ts("gather", st);
  dim3 grid((unsigned)blocks, p.L);
  if (cpr == 16)
    k_gather<16><<<grid, 256, 0, st>>>(io, p.n, p.hkv);
  else
    k_gather<32><<<grid, 256, 0, st>>>(io, p.n, p.hkv);
  return cudaGetLastError();
}

}  // namespace stl
