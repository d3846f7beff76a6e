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
#include "ptx.cuh"

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
__global__ void __launch_bounds__(kDecThreads, 2) k_decode_split(const __grid_constant__ DecBatch b, int w, int n,
                                                              int hq, int hkv, int per, float* part_o_all,
                                                              float2* part_ml_all) {
  extern __shared__ float4 dec_smem[];
  const int split = blockIdx.x, h = blockIdx.y, r = blockIdx.z % w, layer = blockIdx.z / w, nsplit = gridDim.x;
  const T* __restrict__ q = static_cast<const T*>(b.q[layer]);
  const T* __restrict__ k = static_cast<const T*>(b.k[layer]);
  const T* __restrict__ v = static_cast<const T*>(b.v[layer]);
  float* part_o = part_o_all + (size_t)layer * nsplit * w * hq * kD;
  float2* part_ml = part_ml_all + (size_t)layer * nsplit * w * hq;
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
    const size_t slot = ((size_t)split * w + r) * hq + h * G + g;
    part_o[slot * kD + c] = O;
    if (c == 0) part_ml[slot] = make_float2(M, L);
  }
}

// ---------------------------------------------------------------------------
// bf16 caches: key and value tiles of 64 cached rows stream through a ring of
// shared-memory stages by TMA (128-byte swizzle, the layout of the tensor-core
// kernels).  The sixteen warps form four independent groups of four: group i
// takes tiles i, i + 4, ... (so it always uses stage i) and issues its own
// copies, the next tile's as soon as the current one is consumed.  Warp j of
// a group owns rows 16 j .. 16 j + 15 of every tile and keeps its own online
// (max, sum) per query head, so a tile needs one group barrier (the release
// of its stage).  Both products run on the warp's tensor cores (mma.sync
// m16n8k16, bf16 inputs, fp32 accumulation):
//   scores  S (16 rows x 8 heads) = K (16 x 128) Q^T, the query fragments
//           held in registers for the whole kernel, the key fragments read
//           from the swizzled stage by ldmatrix;
//   values  O^T (128 dims x 8 heads) += V^T P^T, V^T read by ldmatrix.trans,
//           P passed through shared memory as P = hi + lo, two bf16 parts
//           (about 16 bits of the fp32 probabilities).
// The sixteen warps' states merge once, after the last tile.  Every mbarrier
// wait is made by the thread that issued the copy and its outcome shared
// through shared memory after the group's barrier, so the group's warps take
// the same path and always meet there.
// Per-layer tensor maps of a batched decode launch.
struct DecMaps {
  CUtensorMap k[kMaxLayers];
  CUtensorMap v[kMaxLayers];
};

constexpr int kDecTile = 64;                         // cached rows per tile
constexpr int kDecStages = 4;
constexpr int kDecHalf = kDecTile * 128;             // one 64-dimension half of a tile: 64 rows x 128 B
constexpr int kDecStageBytes = 4 * kDecHalf;         // keys (two halves), then values (two halves)
constexpr int kDecGroups = 4;                        // consumer groups (one stage each)
constexpr int kDecGroupThreads = 128;
constexpr int kDecMmaThreads = kDecGroups * kDecGroupThreads;
constexpr int kDecMmaWarps = kDecMmaThreads / 32;
// per warp: P^T as [8 NT heads][16 rows] bf16, high and low parts
__host__ __device__ constexpr int dec_pt_bytes(int nt) { return 2 * 8 * nt * 16 * 2; }
// stages, the warps' P^T buffers, (max, sum) of every warp and head, flags
__host__ __device__ constexpr int dec_mma_smem(int nt) {
  return 1024 + kDecStages * kDecStageBytes + kDecMmaWarps * dec_pt_bytes(nt) + kDecMmaWarps * 8 * nt * 8 + 128;
}
static_assert(kDecStages == kDecGroups, "group i always uses stage i");
static_assert(kDecMmaWarps * 16 * kD * 4 <= kDecStages * kDecStageBytes, "merge buffer fits the stages");

__device__ __forceinline__ void group_sync(int gi) {
  asm volatile("bar.sync %0, 128;" ::"r"(1 + gi) : "memory");
}

// Element e (0..127) of row t of a swizzled [2][64][128 B] tile.
__device__ __forceinline__ uint32_t tile_off(int t, int e) {
  const int kb = e >> 6, c = (e >> 3) & 7;
  return (uint32_t)(kb * kDecHalf + t * 128 + ((c ^ (t & 7)) << 4) + (e & 7) * 2);
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
               : "r"(addr));
}
// d += a b (m16n8k16, bf16 in, fp32 accumulate)
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// NT: 8-head column tiles of the query group (1 for G <= 8, 2 for G <= 16).
template <int NT>
__global__ void __launch_bounds__(kDecMmaThreads, 1)
    k_decode_mma(const __grid_constant__ DecMaps maps, const __grid_constant__ DecBatch b, int w, int n, int hq,
                 int hkv, int per, float* part_o_all, float2* part_ml_all, uint32_t* err) {
  extern __shared__ uint8_t dec_raw[];
  uint8_t* sm = dec_raw + ((1024u - (smem_u32(dec_raw) & 1023u)) & 1023u);
  const int split = blockIdx.x, h = blockIdx.y, r = blockIdx.z % w, layer = blockIdx.z / w;
  const CUtensorMap& kmap = maps.k[layer];
  const CUtensorMap& vmap = maps.v[layer];
  const __nv_bfloat16* __restrict__ q = static_cast<const __nv_bfloat16*>(b.q[layer]);
  float* part_o = part_o_all + (size_t)layer * gridDim.x * w * hq * kD;
  float2* part_ml = part_ml_all + (size_t)layer * gridDim.x * w * hq;
  const int G = hq / hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gi = warp >> 2, wq = warp & 3, id = tid & (kDecGroupThreads - 1);
  const int g8 = lane >> 2, t4 = lane & 3;
  uint8_t* pt_all = sm + kDecStages * kDecStageBytes;                        // [warps][dec_pt_bytes]
  float2* wml = reinterpret_cast<float2*>(pt_all + kDecMmaWarps * dec_pt_bytes(NT));  // [warps][8 NT]
  uint64_t* bars = reinterpret_cast<uint64_t*>(wml + kDecMmaWarps * 8 * NT);
  const uint32_t b_full = smem_u32(&bars[0]);
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(&bars[kDecStages]);
  volatile uint32_t* flags = abort_flag + 1;  // one per group
  const uint32_t s0 = smem_u32(sm);
  const int j0 = min(n, split * per), j1 = min(n, j0 + per);
  const int ntiles = (j1 - j0 + kDecTile - 1) / kDecTile;

  if (tid == 0) {
    for (int i = 0; i < kDecStages; ++i) mbar_init(b_full + 8 * i, 1);
    *abort_flag = 0u;
    fence_mbar_init();
  }
  __syncthreads();
  // keys and values of tile it into stage it % kDecStages (one thread)
  auto issue = [&](int it) {
    const int s = it % kDecStages;
    const uint32_t dst = s0 + s * kDecStageBytes;
    const int row = j0 + it * kDecTile;
    mbar_arrive_expect_tx(b_full + 8 * s, (uint32_t)kDecStageBytes);
    tma_load_3d(dst, &kmap, b_full + 8 * s, 0, h, row);
    tma_load_3d(dst + kDecHalf, &kmap, b_full + 8 * s, 64, h, row);
    tma_load_3d(dst + 2 * kDecHalf, &vmap, b_full + 8 * s, 0, h, row);
    tma_load_3d(dst + 3 * kDecHalf, &vmap, b_full + 8 * s, 64, h, row);
  };
  if (id == 0 && gi < ntiles) issue(gi);

  // B fragments of the scores: query head 8 nt + g8 (zero past the group),
  // dimensions 16 ks + 2 t4 + {0, 1} and + 8
  uint32_t qb[8][NT][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int head = 8 * nt + g8;
    const uint32_t* qr = reinterpret_cast<const uint32_t*>(q + ((size_t)r * hq + h * G + (head < G ? head : 0)) * kD);
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      qb[ks][nt][0] = head < G ? __ldg(qr + 8 * ks + t4) : 0u;
      qb[ks][nt][1] = head < G ? __ldg(qr + 8 * ks + 4 + t4) : 0u;
    }
  }
  const float scale = kDecLog2e * rsqrtf((float)kD);
  // running state of heads 8 nt + 2 t4 + e; O^T fragments: o[mt][nt][j] is
  // dimension 16 mt + g8 + 8 (j >> 1), head 8 nt + 2 t4 + (j & 1)
  float m[NT][2], l[NT][2], o[8][NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    m[nt][0] = m[nt][1] = -CUDART_INF_F;
    l[nt][0] = l[nt][1] = 0.f;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][nt][0] = o[mt][nt][1] = o[mt][nt][2] = o[mt][nt][3] = 0.f;
  }
  uint8_t* pt = pt_all + warp * dec_pt_bytes(NT);  // hi at 0, lo at half
  __nv_bfloat16* pt_hi = reinterpret_cast<__nv_bfloat16*>(pt);
  __nv_bfloat16* pt_lo = pt_hi + 8 * NT * 16;
  const int r0 = 16 * wq;

  for (int it = gi; it < ntiles; it += kDecGroups) {
    const int s = it % kDecStages;
    const uint32_t par = (uint32_t)(it / kDecStages) & 1u;
    if (id == 0) {
      const bool ok = mbar_wait(b_full + 8 * s, par, err, abort_flag);
      if (!ok) mbar_wait_drain(b_full + 8 * s, par);  // the copy in flight ends before the CTA does
      flags[gi] = ok ? 1u : 0u;
    }
    group_sync(gi);
    if (flags[gi] == 0u) break;  // the same value for every thread of the group
    const uint32_t kt = s0 + s * kDecStageBytes, vt = kt + 2 * kDecHalf;
    const int base = j0 + it * kDecTile;
    // scores of rows r0 + g8 and r0 + g8 + 8, heads 8 nt + 2 t4 + {0, 1}
    float c[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) c[nt][0] = c[nt][1] = c[nt][2] = c[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint32_t a[4];
      ldsm_x4(kt + tile_off(r0 + (lane & 7) + 8 * ((lane >> 3) & 1), 16 * ks + 8 * (lane >> 4)), a);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(c[nt], a, qb[ks][nt][0], qb[ks][nt][1]);
    }
    const bool va = base + r0 + g8 < j1, vb = base + r0 + g8 + 8 < j1;
    // online softmax per head over the warp's 16 rows (log2 units)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int head = 8 * nt + 2 * t4 + e;
        const float xa = (va && head < G) ? c[nt][e] * scale : -CUDART_INF_F;
        const float xb = (vb && head < G) ? c[nt][2 + e] * scale : -CUDART_INF_F;
        float mx = fmaxf(xa, xb);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float mn = fmaxf(m[nt][e], mx);
        const float alpha = weight(m[nt][e], mn);
        const float pa = weight(xa, mn), pb = weight(xb, mn);
        float sum = pa + pb;
        sum += __shfl_xor_sync(0xffffffffu, sum, 4);
        sum += __shfl_xor_sync(0xffffffffu, sum, 8);
        sum += __shfl_xor_sync(0xffffffffu, sum, 16);
        l[nt][e] = l[nt][e] * alpha + sum;
        m[nt][e] = mn;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          o[mt][nt][e] *= alpha;
          o[mt][nt][2 + e] *= alpha;
        }
        // P^T[head][row] as hi + lo
        const __nv_bfloat16 ha = __float2bfloat16_rn(pa), hb = __float2bfloat16_rn(pb);
        pt_hi[head * 16 + g8] = ha;
        pt_hi[head * 16 + g8 + 8] = hb;
        pt_lo[head * 16 + g8] = __float2bfloat16_rn(pa - __bfloat162float(ha));
        pt_lo[head * 16 + g8 + 8] = __float2bfloat16_rn(pb - __bfloat162float(hb));
      }
    }
    __syncwarp();
    // B fragments of the values: P^T rows 2 t4 + {0, 1} (and + 8) of head 8 nt + g8
    uint32_t bh[NT][2], bl[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int head = 8 * nt + g8;
      bh[nt][0] = *reinterpret_cast<const uint32_t*>(pt_hi + head * 16 + 2 * t4);
      bh[nt][1] = *reinterpret_cast<const uint32_t*>(pt_hi + head * 16 + 2 * t4 + 8);
      bl[nt][0] = *reinterpret_cast<const uint32_t*>(pt_lo + head * 16 + 2 * t4);
      bl[nt][1] = *reinterpret_cast<const uint32_t*>(pt_lo + head * 16 + 2 * t4 + 8);
    }
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      uint32_t a[4];
      ldsm_x4_trans(vt + tile_off(r0 + (lane & 7) + 8 * ((lane >> 4) & 1), 16 * mt + 8 * ((lane >> 3) & 1)), a);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        mma_bf16_16816(o[mt][nt], a, bh[nt][0], bh[nt][1]);
        mma_bf16_16816(o[mt][nt], a, bl[nt][0], bl[nt][1]);
      }
    }
    __syncwarp();  // P^T is rewritten by the next tile
    // the group is done with this stage: its reads are ordered before the
    // next copy into it
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    group_sync(gi);
    if (id == 0 && it + kDecGroups < ntiles) issue(it + kDecGroups);
  }
  // merge the sixteen warps (through the stage buffers, idle once every
  // group has finished), then write this split's partial per query head
  __syncthreads();
  float* wo = reinterpret_cast<float*>(sm);  // [warps][8 NT heads][128]
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int head = 8 * nt + 2 * t4 + e;
      if (g8 == 0) wml[warp * 8 * NT + head] = make_float2(m[nt][e], l[nt][e]);
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        wo[((size_t)warp * 8 * NT + head) * kD + 16 * mt + g8] = o[mt][nt][e];
        wo[((size_t)warp * 8 * NT + head) * kD + 16 * mt + g8 + 8] = o[mt][nt][2 + e];
      }
    }
  }
  __syncthreads();
  for (int e = tid; e < G * kD; e += kDecMmaThreads) {
    const int g = e / kD, cc = e % kD;
    float M = -CUDART_INF_F;
    for (int w = 0; w < kDecMmaWarps; ++w) M = fmaxf(M, wml[w * 8 * NT + g].x);
    float O = 0.f, L = 0.f;
    for (int w = 0; w < kDecMmaWarps; ++w) {
      const float2 ml = wml[w * 8 * NT + g];
      const float wgt = weight(ml.x, M);
      L = fmaf(ml.y, wgt, L);
      O = fmaf(wo[((size_t)w * 8 * NT + g) * kD + cc], wgt, O);
    }
    const size_t slot = ((size_t)split * w + r) * hq + h * G + g;
    part_o[slot * kD + cc] = O;
    if (cc == 0) part_ml[slot] = make_float2(M, L);
  }
}

// out[r][g][c] = merge over the splits.  grid (hq, w), one thread per
// dimension: the splits' weights exp2(m_s - M) and the normaliser are formed
// once in shared memory, then every thread sums its dimension over the splits
// with eight partial loads in flight.
constexpr int kDecMaxSplits = 1024;
__global__ void __launch_bounds__(kD) k_decode_combine(const __grid_constant__ DecBatch b, const float* part_o_all,
                                                       const float2* part_ml_all, int nsplit, int hq, int w) {
  __shared__ float wts[kDecMaxSplits];
  __shared__ float red[kD / 32];
  __shared__ float bc[2];
  const int g = blockIdx.x, r = blockIdx.y % w, layer = blockIdx.y / w, c = threadIdx.x, lane = c & 31, wp = c >> 5;
  const float* part_o = part_o_all + (size_t)layer * nsplit * w * hq * kD;
  const float2* part_ml = part_ml_all + (size_t)layer * nsplit * w * hq;
  float* out = b.out[layer];
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

int decode_splits(int n, int hkv, int w, int layers) {
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long cap0 = (n + 255) / 256;  // at least 256 cached rows per split
  const long long cap = cap0 < kDecMaxSplits ? cap0 : kDecMaxSplits;
  if (layers <= 1) {
    // one layer: one wave of one CTA per SM
    long long s = ((long long)sms + (long long)hkv * w - 1) / ((long long)hkv * w);
    if (s > cap) s = cap;
    if (s < 1) s = 1;
    return (int)s;
  }
  // a batch of layers: the split count whose CTAs fill whole waves best
  // (among fills within 2 % the fewest CTAs)
  const long long units = (long long)layers * hkv * w;
  long long smax = 4 * ((sms + units - 1) / units);
  if (smax < 4) smax = 4;
  if (smax > cap) smax = cap;
  long long best = 1;
  double best_eff = 0.0;
  for (long long s = 1; s <= smax; ++s) {
    const long long ctas = units * s, waves = (ctas + sms - 1) / sms;
    const double eff = (double)ctas / (double)(waves * sms);
    if (eff > best_eff + 0.02) {
      best = s;
      best_eff = eff;
    }
  }
  return (int)best;
}

// Workspace: the error word (first 256 bytes), then every layer's split
// partials.
size_t decode_workspace_bytes(int n, int hq, int hkv, int w, int layers) {
  const size_t slots = (size_t)layers * decode_splits(n, hkv, w, layers) * w * hq;
  return 256 + slots * kD * sizeof(float) + slots * sizeof(float2);
}

cudaError_t launch_decode(DType dt, const DecBatch& b, int layers, int n, int hq, int hkv, int w, void* ws,
                          cudaStream_t st) {
  const int nsplit = decode_splits(n, hkv, w, layers);
  uint32_t* err = static_cast<uint32_t*>(ws);
  float* part_o = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + 256);
  float2* part_ml = reinterpret_cast<float2*>(part_o + (size_t)layers * nsplit * w * hq * kD);
  const int G = hq / hkv;
  dim3 grid(nsplit, hkv, w * layers);
  cudaError_t e = cudaSuccess;
  if (dt == kBF16) {
    const int per = ((n + nsplit - 1) / nsplit + kDecTile - 1) / kDecTile * kDecTile;
    DecMaps maps;
    for (int l = 0; l < layers; ++l) {
      if ((e = make_row_map(&maps.k[l], b.k[l], n, hkv, kDecTile)) != cudaSuccess) return e;
      if ((e = make_row_map(&maps.v[l], b.v[l], n, hkv, kDecTile)) != cudaSuccess) return e;
    }
    auto run = [&](auto nt) {
      constexpr int NT = decltype(nt)::value;
      e = cudaFuncSetAttribute(k_decode_mma<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, dec_mma_smem(NT));
      if (e != cudaSuccess) return;
      k_decode_mma<NT><<<grid, kDecMmaThreads, dec_mma_smem(NT), st>>>(maps, b, w, n, hq, hkv, per, part_o,
                                                                       part_ml, err);
    };
    TimingScope ts("decode_split", st);
    if (G <= 8)
      run(std::integral_constant<int, 1>());
    else
      run(std::integral_constant<int, 2>());
  } else {
    const int per = ((n + nsplit - 1) / nsplit + 31) / 32 * 32;
    const size_t smem = (size_t)G * kD * 4 + (size_t)kDecWarps * G * kD * 4 + (size_t)kDecWarps * G * 8;
    auto run = [&](auto gm) {
      constexpr int GM = decltype(gm)::value;
      e = cudaFuncSetAttribute(k_decode_split<float, GM>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return;
      k_decode_split<float, GM><<<grid, kDecThreads, smem, st>>>(b, w, n, hq, hkv, per, part_o, part_ml);
    };
    TimingScope ts("decode_split", st);
    if (G <= 4)
      run(std::integral_constant<int, 4>());
    else if (G <= 8)
      run(std::integral_constant<int, 8>());
    else
      run(std::integral_constant<int, 16>());
  }
  if (e != cudaSuccess) return e;
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  TimingScope ts("decode_combine", st);
  k_decode_combine<<<dim3(hq, w * layers), kD, 0, st>>>(b, part_o, part_ml, nsplit, hq, w);
  return cudaGetLastError();
}

}  // namespace stl
