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

// ---------------------------------------------------------------------------
// bf16 caches: key and value tiles of 64 cached rows stream through a ring of
// shared-memory stages by TMA (128-byte swizzle, the layout of the tensor-core
// kernels).  The sixteen warps form four independent groups of four: group i
// takes tiles i, i + 4, ... (so it always uses stage i), issues its own
// copies (the next tile's as soon as the current one is consumed), keeps its
// own online (max, sum) per query head and meets only its own named barrier,
// so the groups' copy and barrier latencies overlap one another's work.  A
// group consumes a tile in three phases:
//   1. scores: thread (row t = id % 64, half sl = id / 64) dots dimensions
//      64 sl .. 64 sl + 63 of its row's key with every query head of the
//      group (a warp's lanes share the half, so query reads are broadcasts);
//      the two halves' partial scores are summed through shared memory;
//   2. online softmax: warp w of the group updates (max, sum) of query heads
//      w, w + 4, ... and turns the tile's scores into probabilities;
//   3. values: thread (dimension pair dp = id % 64, row parity ts = id / 64)
//      accumulates p * v over rows ts, ts + 2, ... for every query head.
// Scores and probabilities are kept parity-major: entry (g, t) at
// g * 64 + (t % 2) * 32 + t / 2.  The groups and row parities are merged
// once, after the last tile.  Every mbarrier wait is made by the thread that
// issued the copy and its outcome shared through shared memory after the
// group's barrier, so the group's warps take the same path and always meet
// there.
constexpr int kDecTile = 64;                         // cached rows per tile
constexpr int kDecStages = 4;
constexpr int kDecHalf = kDecTile * 128;             // one 64-dimension half of a tile: 64 rows x 128 B
constexpr int kDecStageBytes = 4 * kDecHalf;         // keys (two halves), then values (two halves)
constexpr int kDecGroups = 4;                        // consumer groups (one stage each)
constexpr int kDecGroupThreads = 128;
constexpr int kDecConsumers = kDecGroups * kDecGroupThreads;  // warps 0-15
constexpr int kDecTmaThreads = kDecConsumers;
constexpr int kDecQPitch = kD + 4;                   // floats per staged query row
// per group: ps [GM][64], part [2][GM][64], m, l, a [GM], the wait flag (+3 pad)
__host__ __device__ constexpr int dec_group_floats(int gm) { return 3 * gm * kDecTile + 3 * gm + 4; }
constexpr int kDecTmaSmem = 1024 + kDecStages * kDecStageBytes + kDecMaxG * kDecQPitch * 4 +
                            kDecGroups * dec_group_floats(kDecMaxG) * 4 + 128;
static_assert(kDecStages == kDecGroups, "group i always uses stage i");
static_assert(kDecGroups * 2 * kDecMaxG * kD * 4 <= kDecStages * kDecStageBytes, "merge buffer fits the stages");

__device__ __forceinline__ void group_sync(int gi) {
  asm volatile("bar.sync %0, 128;" ::"r"(1 + gi) : "memory");
}
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 5, 512;" ::: "memory"); }

// Element e (0..127) of row t of a swizzled [2][64][128 B] tile.
__device__ __forceinline__ uint32_t tile_off(int t, int e) {
  const int kb = e >> 6, c = (e >> 3) & 7;
  return (uint32_t)(kb * kDecHalf + t * 128 + ((c ^ (t & 7)) << 4) + (e & 7) * 2);
}

template <int GM>
__global__ void __launch_bounds__(kDecTmaThreads, 1)
    k_decode_tma(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                 const __nv_bfloat16* __restrict__ q, int n, int hq, int hkv, int per, float* part_o,
                 float2* part_ml, uint32_t* err) {
  extern __shared__ uint8_t dec_raw[];
  uint8_t* sm = dec_raw + ((1024u - (smem_u32(dec_raw) & 1023u)) & 1023u);
  const int split = blockIdx.x, h = blockIdx.y, r = blockIdx.z;
  const int G = hq / hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int GF = dec_group_floats(GM);
  float* qs = reinterpret_cast<float*>(sm + kDecStages * kDecStageBytes);  // [GM][kDecQPitch]
  float* gscr = qs + GM * kDecQPitch;                                        // [groups][GF]
  uint64_t* bars = reinterpret_cast<uint64_t*>(gscr + kDecGroups * GF);     // 8-byte aligned
  const uint32_t b_full = smem_u32(&bars[0]);
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(&bars[kDecStages]);
  const uint32_t s0 = smem_u32(sm);
  const int j0 = min(n, split * per), j1 = min(n, j0 + per);
  const int ntiles = (j1 - j0 + kDecTile - 1) / kDecTile;

  if (tid == 0) {
    for (int i = 0; i < kDecStages; ++i) mbar_init(b_full + 8 * i, 1);
    *abort_flag = 0u;
    fence_mbar_init();
  }
  // query rows of the group, times log2(e)/sqrt(d); every group's running
  // (max, sum)
  const float scale = kDecLog2e * rsqrtf((float)kD);
  for (int e = tid; e < G * kD; e += kDecTmaThreads)
    qs[(e / kD) * kDecQPitch + e % kD] = __bfloat162float(q[((size_t)r * hq + h * G) * kD + e]) * scale;
  for (int e = tid; e < kDecGroups * GM; e += kDecTmaThreads) {
    float* st = gscr + (e / GM) * GF + 3 * GM * kDecTile;
    st[e % GM] = -CUDART_INF_F;  // m
    st[GM + e % GM] = 0.f;       // l
  }
  __syncthreads();
  (void)warp;
  (void)lane;
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

  // ---------------------------------------------------------- consumers
  const int gi = tid / kDecGroupThreads, id = tid % kDecGroupThreads, wl = id >> 5;
  if (id == 0 && gi < ntiles) issue(gi);
  float* ps = gscr + gi * GF;              // [GM][64] scores, then probabilities
  float* part = ps + GM * kDecTile;        // [2][GM][64] half-row partial scores
  float* st_m = part + 2 * GM * kDecTile;  // running max, sum, and this tile's rescale
  float* st_l = st_m + GM;
  float* st_a = st_l + GM;
  volatile uint32_t* flag = reinterpret_cast<volatile uint32_t*>(st_a + GM);
  float o[GM][2];  // dimensions 2*dp, 2*dp + 1 over this thread's row parity
#pragma unroll
  for (int g = 0; g < GM; ++g) o[g][0] = o[g][1] = 0.f;
  const int dp = id & 63, ts = id >> 6;   // phase 3 roles
  const int t1 = id & 63, sl = id >> 6;   // phase 1 roles
  for (int it = gi; it < ntiles; it += kDecGroups) {
    const int s = it % kDecStages;
    const uint32_t par = (uint32_t)(it / kDecStages) & 1u;
    if (id == 0) {
      const bool ok = mbar_wait(b_full + 8 * s, par, err, abort_flag);
      if (!ok) mbar_wait_drain(b_full + 8 * s, par);  // the copy in flight ends before the CTA does
      *flag = ok ? 1u : 0u;
    }
    group_sync(gi);
    if (*flag == 0u) break;  // the same value for every thread of the group
    const uint8_t* kt = sm + s * kDecStageBytes;
    const uint8_t* vt = kt + 2 * kDecHalf;
    const int base = j0 + it * kDecTile;
    // phase 1: row t1, dimensions 64 sl .. 64 sl + 63 in two quarters of
    // 32, every query head
    {
      float acc[GM];
#pragma unroll
      for (int g = 0; g < GM; ++g) acc[g] = 0.f;
#pragma unroll
      for (int qq = 0; qq < 2; ++qq) {
        const int d0 = 64 * sl + 32 * qq;
        float kf[32];
#pragma unroll
        for (int m = 0; m < 4; ++m) {
          const uint4 u = *reinterpret_cast<const uint4*>(kt + tile_off(t1, d0 + 8 * m));
          const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            kf[8 * m + 2 * i] = __uint_as_float(w4[i] << 16);
            kf[8 * m + 2 * i + 1] = __uint_as_float(w4[i] & 0xffff0000u);
          }
        }
#pragma unroll
        for (int g = 0; g < GM; ++g) {
          if (g < G) {
            float x0 = 0.f, x1 = 0.f;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 a = *reinterpret_cast<const float4*>(qs + g * kDecQPitch + d0 + 4 * j);
              float& x = (j & 1) ? x1 : x0;
              x = fmaf(kf[4 * j], a.x, fmaf(kf[4 * j + 1], a.y, fmaf(kf[4 * j + 2], a.z, fmaf(kf[4 * j + 3], a.w, x))));
            }
            acc[g] += x0 + x1;
          }
        }
      }
#pragma unroll
      for (int g = 0; g < GM; ++g)
        if (g < G) part[(sl * GM + g) * kDecTile + t1] = acc[g];
    }
    group_sync(gi);
    // phase 1b: sum the halves; scores of rows past the range are -inf
    for (int e = id; e < G * kDecTile; e += kDecGroupThreads) {
      const int g = e / kDecTile, t = e % kDecTile;
      const float x = part[g * kDecTile + t] + part[(GM + g) * kDecTile + t];
      ps[g * kDecTile + (t & 1) * 32 + (t >> 1)] = base + t < j1 ? x : -CUDART_INF_F;
    }
    group_sync(gi);
    // phase 2: online softmax of query head g over the tile's 64 rows (any
    // two positions per lane: the order of rows does not matter here)
    for (int g = wl; g < G; g += kDecGroupThreads / 32) {
      const float x0 = ps[g * kDecTile + lane], x1 = ps[g * kDecTile + lane + 32];
      const float mo = st_m[g];
      const float mn = fmaxf(mo, warp_max(fmaxf(x0, x1)));
      const float p0 = weight(x0, mn), p1 = weight(x1, mn);
      const float sum = warp_sum(p0 + p1);
      ps[g * kDecTile + lane] = p0;
      ps[g * kDecTile + lane + 32] = p1;
      if (lane == 0) {
        const float a = weight(mo, mn);
        st_a[g] = a;
        st_l[g] = st_l[g] * a + sum;
        st_m[g] = mn;
      }
    }
    group_sync(gi);
    // phase 3: rows ts + 2 k, dimensions 2 dp and 2 dp + 1, every query head,
    // in two halves of 16 rows
#pragma unroll
    for (int g = 0; g < GM; ++g)
      if (g < G) {
        const float a = st_a[g];
        o[g][0] *= a;
        o[g][1] *= a;
      }
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float2 vv[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const uint32_t w = *reinterpret_cast<const uint32_t*>(vt + tile_off(ts + 2 * (16 * hh + k), 2 * dp));
        vv[k] = make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
      }
#pragma unroll
      for (int g = 0; g < GM; ++g) {
        if (g < G) {
          float y0 = o[g][0], y1 = o[g][1], z0 = 0.f, z1 = 0.f;
#pragma unroll
          for (int k4 = 0; k4 < 4; ++k4) {
            const float4 pk = *reinterpret_cast<const float4*>(ps + g * kDecTile + ts * 32 + 16 * hh + 4 * k4);
            y0 = fmaf(pk.x, vv[4 * k4].x, y0);
            y1 = fmaf(pk.x, vv[4 * k4].y, y1);
            z0 = fmaf(pk.y, vv[4 * k4 + 1].x, z0);
            z1 = fmaf(pk.y, vv[4 * k4 + 1].y, z1);
            y0 = fmaf(pk.z, vv[4 * k4 + 2].x, y0);
            y1 = fmaf(pk.z, vv[4 * k4 + 2].y, y1);
            z0 = fmaf(pk.w, vv[4 * k4 + 3].x, z0);
            z1 = fmaf(pk.w, vv[4 * k4 + 3].y, z1);
          }
          o[g][0] = y0 + z0;
          o[g][1] = y1 + z1;
        }
      }
    }
    // the group is done with this stage: its reads are ordered before the
    // next copy into it
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    group_sync(gi);
    if (id == 0 && it + kDecGroups < ntiles) issue(it + kDecGroups);
  }
  // merge the groups and row parities (through the stage buffers, idle once
  // every group has finished), then write this split's partial per query head
  consumer_sync();
  float* red = reinterpret_cast<float*>(sm);  // [groups][2 parities][GM][128]
#pragma unroll
  for (int g = 0; g < GM; ++g)
    if (g < G)
      *reinterpret_cast<float2*>(red + (((size_t)gi * 2 + ts) * GM + g) * kD + 2 * dp) = make_float2(o[g][0], o[g][1]);
  consumer_sync();
  for (int e = tid; e < G * kD; e += kDecConsumers) {
    const int g = e / kD, c = e % kD;
    float M = -CUDART_INF_F;
#pragma unroll
    for (int q4 = 0; q4 < kDecGroups; ++q4) M = fmaxf(M, gscr[q4 * GF + 3 * GM * kDecTile + g]);
    float O = 0.f, L = 0.f;
#pragma unroll
    for (int q4 = 0; q4 < kDecGroups; ++q4) {
      const float* st = gscr + q4 * GF + 3 * GM * kDecTile;
      const float w = weight(st[g], M);
      L = fmaf(st[GM + g], w, L);
      O = fmaf(red[(((size_t)q4 * 2 + 0) * GM + g) * kD + c] + red[(((size_t)q4 * 2 + 1) * GM + g) * kD + c], w, O);
    }
    const size_t slot = ((size_t)split * gridDim.z + r) * hq + h * G + g;
    part_o[slot * kD + c] = O;
    if (c == 0) part_ml[slot] = make_float2(M, L);
  }
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
  // one wave of one CTA per SM, each with at least 256 cached rows
  long long s = ((long long)sms + (long long)hkv * w - 1) / ((long long)hkv * w);
  const long long cap = (n + 255) / 256;
  if (s > cap) s = cap;
  if (s > kDecMaxSplits) s = kDecMaxSplits;
  if (s < 1) s = 1;
  return (int)s;
}

// Workspace: the error word (first 256 bytes), then the split partials.
size_t decode_workspace_bytes(int n, int hq, int hkv, int w) {
  const size_t slots = (size_t)decode_splits(n, hkv, w) * w * hq;
  return 256 + slots * kD * sizeof(float) + slots * sizeof(float2);
}

cudaError_t launch_decode(DType dt, const void* q, const void* k, const void* v, int n, int hq, int hkv, int w,
                          float* out, void* ws, cudaStream_t st) {
  const int nsplit = decode_splits(n, hkv, w);
  uint32_t* err = static_cast<uint32_t*>(ws);
  float* part_o = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + 256);
  float2* part_ml = reinterpret_cast<float2*>(part_o + (size_t)nsplit * w * hq * kD);
  const int G = hq / hkv;
  dim3 grid(nsplit, hkv, w);
  cudaError_t e = cudaSuccess;
  if (dt == kBF16) {
    const int per = ((n + nsplit - 1) / nsplit + kDecTile - 1) / kDecTile * kDecTile;
    CUtensorMap km, vm;
    if ((e = make_row_map(&km, k, n, hkv, kDecTile)) != cudaSuccess) return e;
    if ((e = make_row_map(&vm, v, n, hkv, kDecTile)) != cudaSuccess) return e;
    auto run = [&](auto gm) {
      constexpr int GM = decltype(gm)::value;
      e = cudaFuncSetAttribute(k_decode_tma<GM>, cudaFuncAttributeMaxDynamicSharedMemorySize, kDecTmaSmem);
      if (e != cudaSuccess) return;
      k_decode_tma<GM><<<grid, kDecTmaThreads, kDecTmaSmem, st>>>(
          km, vm, static_cast<const __nv_bfloat16*>(q), n, hq, hkv, per, part_o, part_ml, err);
    };
    TimingScope ts("decode_split", st);
    if (G <= 4)
      run(std::integral_constant<int, 4>());
    else if (G <= 8)
      run(std::integral_constant<int, 8>());
    else
      run(std::integral_constant<int, 16>());
  } else {
    const int per = ((n + nsplit - 1) / nsplit + 31) / 32 * 32;
    const size_t smem = (size_t)G * kD * 4 + (size_t)kDecWarps * G * kD * 4 + (size_t)kDecWarps * G * 8;
    auto run = [&](auto gm) {
      constexpr int GM = decltype(gm)::value;
      e = cudaFuncSetAttribute(k_decode_split<float, GM>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return;
      k_decode_split<float, GM><<<grid, kDecThreads, smem, st>>>(static_cast<const float*>(q),
                                                                 static_cast<const float*>(k),
                                                                 static_cast<const float*>(v), n, hq, hkv, per,
                                                                 part_o, part_ml);
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
  k_decode_combine<<<dim3(hq, w), kD, 0, st>>>(part_o, part_ml, nsplit, hq, w, out);
  return cudaGetLastError();
}

}  // namespace stl
