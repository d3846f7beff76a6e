// Tensor-core (tcgen05 + TMA) kernels for bf16 caches:
//   k_tsg_umma       TSG redundancy, Eq. 6: historical keys x current-frame
//                    keys on the tensor cores, scale-and-row-max epilogue.
//   k_rowstats_umma  window score pass 1 (Eq. 2): per query row running max
//                    and sum of exponentials over a split of the keys.
//   k_colsum_umma    window score pass 2: per key sum over query rows of the
//                    softmax probabilities.
//
// All three share one structure: warp 0 issues TMA loads of 128-byte-swizzled
// key tiles, warp 1 issues tcgen05.mma into TMEM (fp32 accumulators), and
// groups of four warps (one warp per TMEM lane quarter) drain TMEM with
// tcgen05.ld and run the fp32 epilogue: two groups (warps 2-9) in TSG and
// the column sums, four (warps 2-17) in the row statistics.  Every mbarrier
// wait is bounded.
#include <cudaTypedefs.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace stl {

constexpr int kThreads = 320;  // 10 warps
constexpr float kLog2eF = 1.4426950408889634f;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  uint32_t a = smem_u32(p);
  return p + ((1024u - (a & 1023u)) & 1023u);
}

// Per-layer tensor maps of K (one launch covers up to kMaxLayers layers).
struct KMaps {
  CUtensorMap m[kMaxLayers];
};

// Q rows [r0, r0 + rows) of KV head h into shared memory in the K-major
// 128B-swizzle layout [2 K-halves][rows][128 B]; query row r = window row *
// G + group member; rows past R are zero.
__device__ __forceinline__ void load_q_sw128(uint8_t* sq, int rows, const __nv_bfloat16* q,
                                             const Problem& p, int h, int r0 = 0) {
  const int G = p.G(), R = p.R();
  for (int e = threadIdx.x; e < rows * 16; e += blockDim.x) {
    int row = e >> 4, c16 = e & 15, kb = c16 >> 3, cc = c16 & 7;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (r0 + row < R) {
      int wr = (r0 + row) / G, g = (r0 + row) - wr * G;
      val = __ldg(reinterpret_cast<const uint4*>(q + ((size_t)wr * p.hq + h * G + g) * kD + c16 * 8));
    }
    *reinterpret_cast<uint4*>(sq + (size_t)kb * rows * 128 + row * 128 + ((cc ^ (row & 7)) << 4)) = val;
  }
  fence_proxy_async_smem();
}

// First token of TSG row tile t and the end of the rows it may write: its
// frame's visual span, or the whole historical range for spanning tiles.
// For a loop whose tiles only grow: f carries the frame of the previous
// tile (start it at 0).
__device__ __forceinline__ void tsg_tile_next(const FrameTable& ft, int t, int& f, int& tok0, int& fend) {
  if (ft.tsg_span) {
    tok0 = ft.tsg_off + t * kTsgTile;
    fend = ft.tsg_end;
    return;
  }
  while (f + 1 < ft.n_frames - 1 && ft.tile0[f + 1] <= t) ++f;
  tok0 = ft.off[f] + (t - ft.tile0[f]) * kTsgTile;
  fend = ft.off[f] + ft.gh[f] * ft.gw[f];
}

// =========================================================================
// TSG.  CTA (x, chunk, h): current-frame columns [512*chunk, 512*chunk+512)
// of head h stay in shared memory (128 KB); historical row tiles of 128
// tokens stream through two 32 KB stages.  TMEM holds the 128 x 512 fp32
// product as two 256-column accumulator stages; epilogue group g owns stage g
// and writes slice 2*chunk+g of rho_part: max_j acc_ij * rn_j.  Columns past
// the current frame carry rn = NaN, which fmaxf ignores.
constexpr int kTsgB = 0;                  // [2][512][128 B]
constexpr int kTsgAStages = 3;
constexpr int kTsgA = 131072;                              // [3 stages][2][128][128 B]
constexpr int kTsgRn = kTsgA + kTsgAStages * 32768;        // float[512]
constexpr int kTsgBar = kTsgRn + 2048;                     // 12 mbarriers + slot + abort
constexpr int kTsgUsed = kTsgBar + 128;                    // bytes after 1024-alignment
constexpr int kTsgSmem = 232448;                           // the per-CTA maximum; the rest is alignment slack

// METRIC kTsgCosine: acc_ij * rn_j; kTsgDot: acc_ij; kTsgNegL2: 2 acc_ij -
// |k_j|^2 (the row's own -|k_i|^2 is added by the selection kernel).  The
// per-column term sits in rn_s (rn_j, 1, or -|k_j|^2), NaN past the frame.
template <int METRIC>
__global__ void __launch_bounds__(kThreads, 1)
    k_tsg_umma(const __grid_constant__ KMaps maps, const __grid_constant__ FrameTable ft,
               Strided<const float> rc_all, int cur_pad, Strided<float> rho_all, int hkv, uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  if ((int)(sm - smem_raw) + kTsgUsed > kTsgSmem) {  // uniform: the layout would not fit
    if (threadIdx.x == 0) record_error(err, kErrLaunch);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int chunk = blockIdx.y, l = blockIdx.z / hkv, h = blockIdx.z % hkv, n = ft.n_tokens;
  const CUtensorMap& kmap = maps.m[l];
  const float* rn_cur = rc_all.at(l) + (size_t)h * cur_pad;  // 16-byte aligned rows
  float* rho_part = rho_all.at(l);
  const int n_tiles = ft.tsg_tiles;
  const int col0 = chunk * 512;
  const int valid = min(512, ft.cur_len - col0);
  const int nst = valid > 256 ? 2 : 1;
  const uint32_t sB = smem_u32(sm + kTsgB), sA = smem_u32(sm + kTsgA);
  float* rn_s = reinterpret_cast<float*>(sm + kTsgRn);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kTsgBar);
  const uint32_t b_afull = smem_u32(&bars[0]), b_aempty = smem_u32(&bars[kTsgAStages]);
  const uint32_t b_bfull = smem_u32(&bars[2 * kTsgAStages]);
  const uint32_t b_accfull = smem_u32(&bars[2 * kTsgAStages + 1]);
  const uint32_t b_accempty = smem_u32(&bars[2 * kTsgAStages + 3]);
  const uint32_t b_done = smem_u32(&bars[2 * kTsgAStages + 5]);
  uint32_t* slot = reinterpret_cast<uint32_t*>(sm + kTsgBar + (2 * kTsgAStages + 6) * 8);
  volatile uint32_t* abort_flag = slot + 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kTsgAStages; ++i) {
      mbar_init(b_afull + 8 * i, 1);
      mbar_init(b_aempty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4);
    }
    mbar_init(b_bfull, 1);
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&kmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(slot), 512);
    tmem_relinquish();
  }
  // inverse norms of this chunk's current-frame columns (NaN past the frame)
  for (int c = (int)threadIdx.x - 64; c < 512; c += kThreads - 64) {
    if (c >= 0) {
      float v = CUDART_NAN_F;
      if (c < valid) {
        const float r = rn_cur[col0 + c];
        v = METRIC == kTsgCosine ? r : (METRIC == kTsgDot ? 1.f : -1.f / (r * r));
      }
      rn_s[c] = v;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(b_bfull, 131072);
      for (int kb = 0; kb < 2; ++kb)
        for (int rb = 0; rb < 4; ++rb)
          tma_load_3d(sB + kb * 65536 + rb * 16384, &kmap, b_bfull, kb * 64, h,
                      ft.cur_off + col0 + rb * 128);
      int it = 0, issued[kTsgAStages] = {0, 0, 0}, tf = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
        const int s = it % kTsgAStages;
        const uint32_t u = (uint32_t)(it / kTsgAStages);
        if (!mbar_wait(b_aempty + 8 * s, (u & 1u) ^ 1u, err, abort_flag)) break;
        int tok0, fend;
        tsg_tile_next(ft, t, tf, tok0, fend);
        mbar_arrive_expect_tx(b_afull + 8 * s, 32768);
        tma_load_3d(sA + s * 32768, &kmap, b_afull + 8 * s, 0, h, tok0);
        tma_load_3d(sA + s * 32768 + 16384, &kmap, b_afull + 8 * s, 64, h, tok0);
        ++issued[s];
      }
      if (*abort_flag) {  // drain copies still in flight before the CTA exits
        mbar_wait_drain(b_bfull, 0);
        for (int s = 0; s < kTsgAStages; ++s)
          if (issued[s]) mbar_wait_drain(b_afull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(b_bfull, 0, err, abort_flag);
      int it = 0;
      for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x, ++it) {
        const int s = it % kTsgAStages;
        const uint32_t u = (uint32_t)(it / kTsgAStages);
        if (!mbar_wait(b_afull + 8 * s, u & 1u, err, abort_flag)) break;
        tc_fence_after();
        for (int g = 0; g < nst && ok; ++g) {
          if (!mbar_wait(b_accempty + 8 * g, ((uint32_t)it & 1u) ^ 1u, err, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int ncols = (min(256, valid - g * 256) + 15) & ~15;
          const uint32_t idesc = idesc_bf16(128, ncols);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t kb = k >> 2, koff = (k & 3) * 32;
            uint64_t ad = desc_sw128(sA + s * 32768 + kb * 16384 + koff);
            uint64_t bd = desc_sw128(sB + kb * 65536 + g * 256 * 128 + koff);
            umma_bf16(tmem + g * 256, ad, bd, idesc, k > 0 ? 1u : 0u);
          }
          umma_commit(b_accfull + 8 * g);
        }
        if (!ok) break;
        umma_commit(b_aempty + 8 * s);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else {
    const int g = (warp - 2) >> 2, quarter = warp & 3;
    if (g < nst) {
      const int valid_g = min(256, valid - g * 256);
      const uint32_t tbase = tmem + ((uint32_t)(quarter * 32) << 16) + g * 256;
      const float* rg = rn_s + g * 256;
      int it = 0, tf = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
        if (!warp_wait(b_accfull + 8 * g, (uint32_t)it & 1u, err, abort_flag)) break;
        tc_fence_after();
        float mx = -CUDART_INF_F;
        if (valid_g == 256) {
          // full stage: no masked column, packed products and 3-input max
          // into eight independent running maxima (short dependency chains)
          float m[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) m[i] = -CUDART_INF_F;
          auto reduce = [&](const uint32_t (&v)[64], int c) {
            const float4* r4 = reinterpret_cast<const float4*>(rg + c * 64);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float4 r = r4[i];
              const float v0 = __uint_as_float(v[4 * i]), v1 = __uint_as_float(v[4 * i + 1]);
              const float v2 = __uint_as_float(v[4 * i + 2]), v3 = __uint_as_float(v[4 * i + 3]);
              float p0, p1, p2, p3;
              if (METRIC == kTsgNegL2) {
                fma2(v0, v1, 2.f, 2.f, r.x, r.y, p0, p1);
                fma2(v2, v3, 2.f, 2.f, r.z, r.w, p2, p3);
              } else {
                mul2(v0, v1, r.x, r.y, p0, p1);
                mul2(v2, v3, r.z, r.w, p2, p3);
              }
              m[(2 * i) & 7] = max3(m[(2 * i) & 7], p0, p1);
              m[(2 * i + 1) & 7] = max3(m[(2 * i + 1) & 7], p2, p3);
            }
          };
          // two register sets: chunk c + 1 loads while chunk c is reduced
          uint32_t b0[64], b1[64];
          tmem_ld64_issue(tbase, b0);
          tmem_ld64_wait(b0);
          tmem_ld64_issue(tbase + 64, b1);
          reduce(b0, 0);
          tmem_ld64_wait_after(b1, m);
          tmem_ld64_issue(tbase + 128, b0);
          reduce(b1, 1);
          tmem_ld64_wait_after(b0, m);
          tmem_ld64_issue(tbase + 192, b1);
          reduce(b0, 2);
          tmem_ld64_wait_after(b1, m);
          reduce(b1, 3);
          mx = fmaxf(fmaxf(max3(m[0], m[1], m[2]), max3(m[3], m[4], m[5])), fmaxf(m[6], m[7]));
        } else {
          // ragged stage: columns past the frame carry rn = NaN, ignored by fmaxf
          for (int c = 0; c < 8; ++c) {
            if (c * 32 >= valid_g) break;
            float v[32];
            tmem_ld32(tbase + c * 32, v);
            const float4* r4 = reinterpret_cast<const float4*>(rg + c * 32);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              float4 r = r4[i];
              if (METRIC == kTsgNegL2) {
                mx = fmaxf(mx, fmaf(v[4 * i], 2.f, r.x));
                mx = fmaxf(mx, fmaf(v[4 * i + 1], 2.f, r.y));
                mx = fmaxf(mx, fmaf(v[4 * i + 2], 2.f, r.z));
                mx = fmaxf(mx, fmaf(v[4 * i + 3], 2.f, r.w));
              } else {
                mx = fmaxf(mx, v[4 * i] * r.x);
                mx = fmaxf(mx, v[4 * i + 1] * r.y);
                mx = fmaxf(mx, v[4 * i + 2] * r.z);
                mx = fmaxf(mx, v[4 * i + 3] * r.w);
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_accempty + 8 * g);
        int tok0, fend;
        tsg_tile_next(ft, t, tf, tok0, fend);
        const int tok = tok0 + quarter * 32 + lane;
        if (tok < fend) rho_part[((size_t)(2 * chunk + g) * hkv + h) * n + tok] = mx;
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// =========================================================================
// Window score pass 1.  CTA (split * NMH + mh, h): query rows [256 mh,
// 256 mh + 128 MT) of head h (MT <= 2 m-tiles of 128) stay in shared memory
// as the A operand; key tiles of 256 keys stream as the B operand.  TMEM:
// two slots of 256 columns, one (m-tile, key tile) item each; every
// epilogue group drains a quarter of each item's keys and keeps, per query
// row, the running max m (raw dot units) and l = sum 2^((x - m) c).  The
// groups merge at the end; part[h][split][r] = (m c, l).
constexpr int kMaxKStages = 4;        // key-tile ring depth (as shared memory allows)
constexpr int kScoreSmemCap = 200 * 1024;

// barrier block of the score kernels: kfull[S], kempty[S], accfull[2],
// accempty[2], done, then the TMEM slot and the abort flag
struct ScoreBars {
  uint32_t kfull, kempty, accfull, accempty, done;
  uint32_t* slot;
  volatile uint32_t* abort_flag;
};
__device__ __forceinline__ ScoreBars score_bars(uint8_t* base) {
  ScoreBars b;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base);
  b.kfull = smem_u32(&bars[0]);
  b.kempty = smem_u32(&bars[kMaxKStages]);
  b.accfull = smem_u32(&bars[2 * kMaxKStages]);
  b.accempty = smem_u32(&bars[2 * kMaxKStages + 2]);
  b.done = smem_u32(&bars[2 * kMaxKStages + 4]);
  b.slot = reinterpret_cast<uint32_t*>(base + (2 * kMaxKStages + 5) * 8);
  b.abort_flag = b.slot + 1;
  return b;
}
constexpr int kScoreBarBytes = 128;

// Window-score passes: a TMA warp, an MMA warp and kScoreGroups epilogue
// groups of four warps.  With 18 warps, an SM sub-partition holds five of
// them, so its 64 K registers leave at most 96 per thread.
constexpr int kScoreGroups = 4;
constexpr int kScoreThreads = (2 + 4 * kScoreGroups) * 32;
constexpr int kScoreMaxReg = 96;
static_assert(kScoreGroups == 4, "the column sums add four partial sums per key");

// NMH CTAs share a key split, each holding MT m-tiles of Q (query rows
// [256 mh, 256 mh + 128 MT)): for R > 256 two CTAs read the same key tiles
// at about the same time (adjacent in the grid, so the second read mostly
// hits L2) instead of one CTA with all of Q, whose 128 KB would leave room
// only for 128-key tiles.
constexpr int kRsXBuf = 3;
struct RsLayout {
  int MT, NMH, KN, q_bytes, k_stage_bytes, kstages, off_k, off_bar, off_xch, total;
};
__host__ __device__ inline RsLayout rs_layout(int R) {
  RsLayout L;
  L.MT = R <= 128 ? 1 : 2;
  L.NMH = R <= 256 ? 1 : 2;
  L.KN = 256;  // keys per tile = MMA N of one (m-tile, key tile) item
  L.q_bytes = L.MT * 128 * 256;
  L.k_stage_bytes = L.KN * 256;
  // split-end exchange: kRsXBuf buffers of every group's (m, l) per row,
  // then kRsXBuf x 4 arrival counters
  const int xch = kRsXBuf * kScoreGroups * L.MT * 128 * 8 + kRsXBuf * 4 * 4;
  const int fixed = L.q_bytes + kScoreBarBytes + xch + 1024;
  L.kstages = (kScoreSmemCap - fixed) / L.k_stage_bytes;
  if (L.kstages > kMaxKStages) L.kstages = kMaxKStages;
  if (L.kstages < 2) L.kstages = 2;
  L.off_k = L.q_bytes;
  L.off_bar = L.off_k + L.kstages * L.k_stage_bytes;
  L.off_xch = L.off_bar + kScoreBarBytes;
  L.total = L.off_xch + xch + 1024;
  return L;
}

__device__ __forceinline__ void online_merge(float& m, float& l, float m2, float l2, float c) {
  float mn = fmaxf(m, m2);
  if (mn == -CUDART_INF_F) return;
  float a = (m == -CUDART_INF_F) ? 0.f : l * exp2f((m - mn) * c);
  float b = (m2 == -CUDART_INF_F) ? 0.f : l2 * exp2f((m2 - mn) * c);
  m = mn;
  l = a + b;
}

template <int MT>
__global__ void __maxnreg__(kScoreMaxReg)
    k_rowstats_umma(const __grid_constant__ KMaps maps, const __grid_constant__ LayerPtrs io, Problem p,
                    int nsplit, int cps, Strided<float2> part_all, uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  const RsLayout L = rs_layout(p.R());
  constexpr int KN = 256;
  constexpr int CW = KN / kScoreGroups;  // key columns per group and item
  const int R = p.R();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // this CTA's key splits [s0, s0 + cps) of `per_t` tiles each (the last
  // split of the head may be shorter)
  const int s0 = (blockIdx.x / L.NMH) * cps, r0 = (blockIdx.x % L.NMH) * 256;
  const int layer = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv, n = p.n;
  const CUtensorMap& kmap = maps.m[layer];
  const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(io.q[layer]);
  float2* part = part_all.at(layer);
  const int tiles_all = (n + KN - 1) / KN;
  const int per_t = (tiles_all + nsplit - 1) / nsplit;
  const int t0 = min(tiles_all, s0 * per_t), t1 = min(tiles_all, (s0 + cps) * per_t);
  const int j0 = t0 * KN, j1 = n;
  const int ntiles = t1 - t0;
  const int nitems = ntiles * MT;
  const uint32_t sQ = smem_u32(sm), sK = smem_u32(sm + L.off_k);
  const ScoreBars bb = score_bars(sm + L.off_bar);
  const uint32_t b_kfull = bb.kfull, b_kempty = bb.kempty, b_accfull = bb.accfull;
  const uint32_t b_accempty = bb.accempty, b_done = bb.done;
  uint32_t* slot = bb.slot;
  volatile uint32_t* abort_flag = bb.abort_flag;
  const int S = L.kstages;
  float2* xch = reinterpret_cast<float2*>(sm + L.off_xch);
  uint32_t* xcnt = reinterpret_cast<uint32_t*>(sm + L.off_xch + kRsXBuf * kScoreGroups * MT * 128 * 8);
  const float c = kLog2eF * rsqrtf((float)kD);

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(b_kfull + 8 * i, 1);
      mbar_init(b_kempty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4 * kScoreGroups);  // every epilogue warp
    }
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    for (int i = 0; i < kRsXBuf * 4; ++i) xcnt[i] = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&kmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(slot), 512);
    tmem_relinquish();
  }
  load_q_sw128(sm, MT * 128, q, p, h, r0);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;

  // Work items u = t * MT + mt: m-tile mt of Q against key tile t, into
  // TMEM slot u % 2 (KN columns).  All kScoreGroups epilogue groups drain every
  // item, group g taking key columns [g*CW, (g+1)*CW): four warps per SM
  // sub-partition hide one another's latencies, and one item drains while
  // the MMA fills the other slot.  Each group keeps a row state per m-tile,
  // (running max m in raw dot units, l = sum 2^((x - m) c)).  At the end of
  // every key split each warp parks its states in exchange buffer
  // (split index in the CTA) % kRsXBuf and counts itself in; the warp that
  // arrives last for its lane quarter merges the four groups' states in
  // group order and writes the split's partial.  Nobody waits, and the
  // partials depend on the shape alone, not on how many splits a CTA takes.
  // A buffer is rewritten kRsXBuf splits (>= 3 items) later, which the MMA
  // can only have produced once every warp has finished with it.
  float ms[MT], ls[MT];
#pragma unroll
  for (int i = 0; i < MT; ++i) {
    ms[i] = -CUDART_INF_F;
    ls[i] = 0.f;
  }
  const int g = warp >= 2 ? (warp - 2) >> 2 : 0, quarter = warp & 3;

  if (warp == 0) {
    if (lane == 0) {
      int issued[kMaxKStages] = {0, 0, 0, 0};
      int ks = 0;        // stage of tile it (it % S), counted instead of divided
      uint32_t kp = 0u;  // passes over the ring (it / S)
      for (int it = 0; it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks;
        const uint32_t u = kp;
        if (!mbar_wait(b_kempty + 8 * s, (u & 1u) ^ 1u, err, abort_flag)) break;
        const int tok = j0 + it * KN;
        mbar_arrive_expect_tx(b_kfull + 8 * s, (uint32_t)L.k_stage_bytes);
        tma_load_3d(sK + s * L.k_stage_bytes, &kmap, b_kfull + 8 * s, 0, h, tok);
        tma_load_3d(sK + s * L.k_stage_bytes + KN * 128, &kmap, b_kfull + 8 * s, 64, h, tok);
        ++issued[s];
      }
      if (*abort_flag)
        for (int s = 0; s < S; ++s)
          if (issued[s]) mbar_wait_drain(b_kfull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, KN);
      bool ok = true;
      int u = 0, ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; ok && it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks;
        if (!mbar_wait(b_kfull + 8 * s, kp & 1u, err, abort_flag)) break;
        for (int mt = 0; mt < MT; ++mt, ++u) {
          const int as = u & 1;
          if (!mbar_wait(b_accempty + 8 * as, ((uint32_t)(u >> 1) & 1u) ^ 1u, err, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t kb = k >> 2, koff = (k & 3) * 32;
            uint64_t ad = desc_sw128(sQ + kb * (MT * 128 * 128) + mt * 128 * 128 + koff);
            uint64_t bd = desc_sw128(sK + s * L.k_stage_bytes + kb * (KN * 128) + koff);
            umma_bf16(tmem + as * 256, ad, bd, idesc, k > 0 ? 1u : 0u);
          }
          umma_commit(b_accfull + 8 * as);
        }
        if (!ok) break;
        umma_commit(b_kempty + 8 * s);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else {
    const uint32_t lanebase = tmem + ((uint32_t)(quarter * 32) << 16) + g * CW;
    // Every epilogue warp runs the same item sequence and the same split
    // flushes (named barrier 1 of the 16 epilogue warps), also after a wait
    // gave up: the abort flag then makes every later wait return at once.
    bool live = true;
    int nflush = 0, tin = 0;  // splits handed over, tiles into the current split
    for (int u = 0; u < nitems; ++u) {
      const int as = u & 1;
      const int t = u / MT, mt = u % MT;
      if (live && !warp_wait(b_accfull + 8 * as, (uint32_t)(u >> 1) & 1u, err, abort_flag)) live = false;
      if (live) {
        tc_fence_after();
        uint32_t b[CW];
        tmem_ld64_issue(lanebase + as * 256, b);
        tmem_ld64_wait(b);
        // the item's TMEM columns are in registers: release the slot
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_accempty + 8 * as);
        float m = ms[0], l = ls[0];
#pragma unroll
        for (int i = 1; i < MT; ++i)
          if (mt == i) {
            m = ms[i];
            l = ls[i];
          }
        const int nv = min(CW, j1 - (j0 + t * KN + g * CW));
        if (nv == CW) {
          // chunk maximum over four independent chains: chain r starts at
          // element r and takes pairs 4 + 2r + 8i, 5 + 2r + 8i
          float cm[4];
#pragma unroll
          for (int r = 0; r < 4; ++r) cm[r] = __uint_as_float(b[r]);
#pragma unroll
          for (int i = 4; i < CW; i += 8) {
#pragma unroll
            for (int r = 0; r < 4; ++r)
              if (i + 2 * r + 1 < CW)
                cm[r] = max3(cm[r], __uint_as_float(b[i + 2 * r]), __uint_as_float(b[i + 2 * r + 1]));
          }
          const float mn = fmaxf(m, fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3])));
          const float mnc = mn * c;
          float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
          // three phases (exponent arguments, exponentials, sums) in place, so
          // that independent work separates dependent instructions
#pragma unroll
          for (int i = 0; i < CW; i += 2) {
            float x0, x1;
            fma2(__uint_as_float(b[i]), __uint_as_float(b[i + 1]), c, c, -mnc, -mnc, x0, x1);
            b[i] = __float_as_uint(x0);
            b[i + 1] = __float_as_uint(x1);
          }
#pragma unroll
          for (int i = 0; i < CW; ++i) b[i] = __float_as_uint(ex2_approx(__uint_as_float(b[i])));
#pragma unroll
          for (int i = 0; i < CW; i += 4) {
            add2(s0, s1, __uint_as_float(b[i]), __uint_as_float(b[i + 1]));
            add2(s2, s3, __uint_as_float(b[i + 2]), __uint_as_float(b[i + 3]));
          }
          l = (m == -CUDART_INF_F ? 0.f : l * ex2_approx((m - mn) * c)) + ((s0 + s1) + (s2 + s3));
          m = mn;
        } else if (nv > 0) {
          float mc = -CUDART_INF_F;
#pragma unroll
          for (int i = 0; i < CW; ++i)
            if (i < nv) mc = fmaxf(mc, __uint_as_float(b[i]));
          const float mn = fmaxf(m, mc);
          const float mnc = mn * c;
          float sacc = 0.f;
#pragma unroll
          for (int i = 0; i < CW; ++i)
            if (i < nv) sacc += ex2_approx(fmaf(__uint_as_float(b[i]), c, -mnc));
          l = (m == -CUDART_INF_F ? 0.f : l * ex2_approx((m - mn) * c)) + sacc;
          m = mn;
        }
#pragma unroll
        for (int i = 0; i < MT; ++i)
          if (mt == i) {
            ms[i] = m;
            ls[i] = l;
          }
      }
      // end of a key split: hand the states over (see above) and start over
      // (the CTA's tiles start on a split boundary)
      if (mt == MT - 1) ++tin;
      if (mt == MT - 1 && (tin == per_t || t + 1 == ntiles)) {
        const int split = s0 + nflush, xb = nflush % kRsXBuf;
        ++nflush;
        tin = 0;
        float2* xp = xch + (size_t)xb * kScoreGroups * MT * 128;
#pragma unroll
        for (int i = 0; i < MT; ++i) xp[(g * MT + i) * 128 + quarter * 32 + lane] = make_float2(ms[i], ls[i]);
        __syncwarp();
        uint32_t last = 0u;
        if (lane == 0) {
          // release the warp's states (cumulative over the __syncwarp) and
          // acquire the other groups' ones with the same atomic
          uint32_t old;
          asm volatile("atom.acq_rel.cta.shared::cta.add.u32 %0, [%1], 1;"
                       : "=r"(old) : "r"(smem_u32(&xcnt[xb * 4 + quarter])) : "memory");
          last = (old & 3u) == 3u ? 1u : 0u;
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        __syncwarp();
        if (last) {
#pragma unroll
          for (int i = 0; i < MT; ++i) {
            const int row = r0 + i * 128 + quarter * 32 + lane;
            const float2 v0 = xp[i * 128 + quarter * 32 + lane];
            float m = v0.x, l = v0.y;
            for (int o = 1; o < kScoreGroups; ++o) {
              const float2 v = xp[(o * MT + i) * 128 + quarter * 32 + lane];
              online_merge(m, l, v.x, v.y, c);
            }
            if (row < R) part[((size_t)h * nsplit + split) * R + row] = make_float2(m * c, l);
          }
        }
#pragma unroll
        for (int i = 0; i < MT; ++i) {
          ms[i] = -CUDART_INF_F;
          ls[i] = 0.f;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// =========================================================================
// Window score pass 2.  CTA (x, h): key tiles of 128 tokens are the A operand
// (M = 128, one key per TMEM lane), Q of head h (NQ = R rounded up to 32
// rows) is the B operand.  Each epilogue thread sums 2^(x_r c + bias_r) for
// its key over its group's range of at most 64 query rows; a merge warp adds
// the four groups' partial sums and stores A_base.  TMEM: two slots of W columns, so that
// one item drains while the next one is computed.  An item is a key tile
// against all NQ query columns (W = NQ <= 256), or against one of nh = 2
// column halves (NQ > 256, rounded to 64, W = NQ / 2).
struct CsLayout {
  int NQ, nh, W, nstage, kstages, tmem_cols, q_bytes, off_k, off_bias, off_bar, off_xch, total;
};
// partial sums [kCsXBuf][kScoreGroups][128 keys] fp32, then the mbarriers
// xfull[kCsXBuf] (every epilogue warp has parked its partials) and
// xfree[kCsXBuf] (the merge warp has summed them)
constexpr int kCsXBuf = 3;
constexpr int kCsXchBytes = kCsXBuf * kScoreGroups * 128 * 4 + kCsXBuf * 2 * 8;
// Column sums add a merge warp (warp 2 + 4 kScoreGroups) to the score
// passes' TMA, MMA and epilogue warps: 19 warps at 96 registers.
constexpr int kCsThreads = kScoreThreads + 32;
__host__ __device__ inline CsLayout cs_layout(int R) {
  CsLayout L;
  L.NQ = R > 256 ? (R + 63) & ~63 : (R + 31) & ~31;
  L.nh = L.NQ > 256 ? 2 : 1;
  L.W = L.NQ / L.nh;
  L.nstage = 2;
  L.tmem_cols = 32;
  while (L.tmem_cols < L.nstage * L.W) L.tmem_cols <<= 1;
  L.q_bytes = L.NQ * 256;
  const int fixed = L.q_bytes + L.NQ * 4 + kScoreBarBytes + kCsXchBytes + 1024;
  L.kstages = (kScoreSmemCap - fixed) / 32768;
  if (L.kstages > kMaxKStages) L.kstages = kMaxKStages;
  if (L.kstages < 2) L.kstages = 2;
  L.off_k = L.q_bytes;
  L.off_bias = L.off_k + L.kstages * 32768;
  L.off_bar = L.off_bias + L.NQ * 4;
  L.off_xch = L.off_bar + kScoreBarBytes;
  L.total = L.off_xch + kCsXchBytes + 1024;
  return L;
}

// NH: column halves per key tile (cs_layout's nh), a template parameter so
// that the one-half loop compiles away.
template <int NH>
__global__ void __maxnreg__(kScoreMaxReg)
    k_colsum_umma(const __grid_constant__ KMaps maps, const __grid_constant__ LayerPtrs io, Problem p,
                  Strided<float2> part_all, int nsplit, Strided<float> a_all, uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  const CsLayout L = cs_layout(p.R());
  constexpr int nh = NH;
  const int NQ = L.NQ, W = L.W, R = p.R(), n = p.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int layer = blockIdx.y / p.hkv, h = blockIdx.y % p.hkv;
  const CUtensorMap& kmap = maps.m[layer];
  const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(io.q[layer]);
  const float2* part = part_all.at(layer);
  float* a_base = a_all.at(layer);
  const int ntiles_all = (n + 127) / 128;
  const uint32_t sQ = smem_u32(sm), sK = smem_u32(sm + L.off_k);
  float* bias_s = reinterpret_cast<float*>(sm + L.off_bias);
  const ScoreBars bb = score_bars(sm + L.off_bar);
  const uint32_t b_kfull = bb.kfull, b_kempty = bb.kempty, b_accfull = bb.accfull;
  const uint32_t b_accempty = bb.accempty, b_done = bb.done;
  uint32_t* slot = bb.slot;
  volatile uint32_t* abort_flag = bb.abort_flag;
  const int S = L.kstages;
  const float c = kLog2eF * rsqrtf((float)kD);
  float* xch = reinterpret_cast<float*>(sm + L.off_xch);
  const uint32_t b_xfull = smem_u32(sm + L.off_xch + kCsXBuf * kScoreGroups * 128 * 4);
  const uint32_t b_xfree = b_xfull + 8 * kCsXBuf;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(b_kfull + 8 * i, 1);
      mbar_init(b_kempty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4 * kScoreGroups);  // every epilogue warp
    }
    for (int i = 0; i < kCsXBuf; ++i) {
      mbar_init(b_xfull + 8 * i, 4 * kScoreGroups);
      mbar_init(b_xfree + 8 * i, 1);
    }
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&kmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(slot), (uint32_t)L.tmem_cols);
    tmem_relinquish();
  }
  load_q_sw128(sm, NQ, q, p, h);
  // pass 1's merged row statistics: bias_r = -m_r - log2(G l_r), so that
  // 2^(x c + bias_r) is the softmax probability divided by G (padded rows
  // get -inf and add exact zeros)
  const float* bias_g = reinterpret_cast<const float*>(part + (size_t)p.hkv * nsplit * R) + (size_t)h * R;
  for (int r = threadIdx.x; r < NQ; r += blockDim.x) bias_s[r] = r < R ? bias_g[r] : -CUDART_INF_F;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;
  int ntiles = 0;
  for (int t = blockIdx.x; t < ntiles_all; t += gridDim.x) ++ntiles;

  if (warp == 0) {
    if (lane == 0) {
      int issued[kMaxKStages] = {0, 0, 0, 0};
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks;
        const uint32_t u = kp;
        if (!mbar_wait(b_kempty + 8 * s, (u & 1u) ^ 1u, err, abort_flag)) break;
        const int tok = (blockIdx.x + it * gridDim.x) * 128;
        mbar_arrive_expect_tx(b_kfull + 8 * s, 32768);
        tma_load_3d(sK + s * 32768, &kmap, b_kfull + 8 * s, 0, h, tok);
        tma_load_3d(sK + s * 32768 + 16384, &kmap, b_kfull + 8 * s, 64, h, tok);
        ++issued[s];
      }
      if (*abort_flag)
        for (int s = 0; s < S; ++s)
          if (issued[s]) mbar_wait_drain(b_kfull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; ok && it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks;
        const uint32_t u = kp;
        if (!mbar_wait(b_kfull + 8 * s, u & 1u, err, abort_flag)) break;
        // item it*nh + hh: query columns [hh W, hh W + W) into TMEM slot item % 2
#pragma unroll
        for (int hh = 0; hh < nh; ++hh) {
          const int item = it * nh + hh, as = item & 1;
          if (!mbar_wait(b_accempty + 8 * as, ((uint32_t)(item >> 1) & 1u) ^ 1u, err, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t idesc = idesc_bf16(128, W);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t kb = k >> 2, koff = (k & 3) * 32;
            uint64_t ad = desc_sw128(sK + s * 32768 + kb * 16384 + koff);
            uint64_t bd = desc_sw128(sQ + kb * (NQ * 128) + hh * W * 128 + koff);
            umma_bf16(tmem + as * W, ad, bd, idesc, k > 0 ? 1u : 0u);
          }
          umma_commit(b_accfull + 8 * as);
        }
        if (!ok) break;
        umma_commit(b_kempty + 8 * s);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else if (warp < 2 + 4 * kScoreGroups) {
    // Every group drains every item: group g the item's query columns
    // [c0, c1), at most 64; columns of padded rows carry bias = -inf, so
    // they add exact zeros.  A thread's sum runs over the tile's nh items.
    // The groups' partial sums of a tile go to shared buffer it % kCsXBuf
    // (once the merge warp has released that buffer's previous tile), and
    // every warp arrives on the buffer's xfull barrier; the merge warp adds
    // them.  The drain of the next item does not wait for the sum.
    const int g = (warp - 2) >> 2, quarter = warp & 3, row = quarter * 32 + lane;
    const int gwid = (((W + kScoreGroups - 1) / kScoreGroups) + 31) & ~31;
    const int c0 = min(W, g * gwid), c1 = min(W, c0 + gwid);
    const uint32_t lanebase = tmem + ((uint32_t)(quarter * 32) << 16);
    bool ok = true;
    int xb = 0;         // exchange buffer of tile it (it % kCsXBuf), counted
    uint32_t xu = 0u;   // uses of that buffer so far (it / kCsXBuf)
    for (int it = 0; ok && it < ntiles; ++it) {
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
      for (int hh = 0; hh < nh; ++hh) {
        const int item = it * nh + hh, as = item & 1;
        if (!warp_wait(b_accfull + 8 * as, (uint32_t)(item >> 1) & 1u, err, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tb = lanebase + as * W + c0;
        const float4* b4 = reinterpret_cast<const float4*>(bias_s + hh * W + c0);
        if (c1 - c0 == 64) {
          float v[64];
          tmem_ld64(tb, v);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_accempty + 8 * as);
          // three phases over the chunk (exponent arguments, exponentials,
          // sums), so that independent work separates dependent instructions
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float4 b = b4[i];
            fma2(v[4 * i], v[4 * i + 1], c, c, b.x, b.y, v[4 * i], v[4 * i + 1]);
            fma2(v[4 * i + 2], v[4 * i + 3], c, c, b.z, b.w, v[4 * i + 2], v[4 * i + 3]);
          }
#pragma unroll
          for (int i = 0; i < 64; ++i) v[i] = ex2_approx(v[i]);
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            add2(a0, a1, v[4 * i], v[4 * i + 1]);
            add2(a2, a3, v[4 * i + 2], v[4 * i + 3]);
          }
        } else if (c1 - c0 == 32) {
          float v[32];
          tmem_ld32(tb, v);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_accempty + 8 * as);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float4 b = b4[i];
            fma2(v[4 * i], v[4 * i + 1], c, c, b.x, b.y, v[4 * i], v[4 * i + 1]);
            fma2(v[4 * i + 2], v[4 * i + 3], c, c, b.z, b.w, v[4 * i + 2], v[4 * i + 3]);
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = ex2_approx(v[i]);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            add2(a0, a1, v[4 * i], v[4 * i + 1]);
            add2(a2, a3, v[4 * i + 2], v[4 * i + 3]);
          }
        } else {
          __syncwarp();
          if (lane == 0) mbar_arrive(b_accempty + 8 * as);
        }
      }
      if (!ok) break;
      if (xu > 0 && !warp_wait(b_xfree + 8 * xb, (xu - 1u) & 1u, err, abort_flag)) break;
      __syncwarp();  // every lane's store follows lane 0's acquire
      xch[xb * (kScoreGroups * 128) + g * 128 + row] = (a0 + a1) + (a2 + a3);
      __syncwarp();
      if (lane == 0) mbar_arrive(b_xfull + 8 * xb);
      if (++xb == kCsXBuf) {
        xb = 0;
        ++xu;
      }
    }
  } else {
    // Merge warp: A_base of tile it = the four groups' partials added in
    // group order, stored by lanes on consecutive keys; then the buffer is
    // released for tile it + kCsXBuf.
    int xb = 0;
    uint32_t xu = 0u;
    for (int it = 0; it < ntiles; ++it) {
      if (!warp_wait(b_xfull + 8 * xb, xu & 1u, err, abort_flag)) break;
      const float* xp = xch + xb * (kScoreGroups * 128);
      const int tok0 = (blockIdx.x + it * gridDim.x) * 128;
#pragma unroll
      for (int r = lane; r < 128; r += 32) {
        const float acc = (xp[r] + xp[128 + r]) + (xp[256 + r] + xp[384 + r]);
        if (tok0 + r < n) a_base[(size_t)h * n + tok0 + r] = acc;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(b_xfree + 8 * xb);
      if (++xb == kCsXBuf) {
        xb = 0;
        ++xu;
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)L.tmem_cols);
  }
}

// =========================================================================
// CSS on the tensor cores (bf16).  CTA (x, layer*Hkv + head) walks 128-token
// tiles of the frames' visual spans.  For a tile starting at token t0 of a
// frame with grid width gw, B = keys of tokens [t0, t0 + NB), NB =
// roundup16(128 + gw + 1) <= 256, and A = its first 128 rows; one tcgen05
// MMA gives every dot product a row needs: D[i][i] (squared norm),
// D[i][i+1] (E), D[i][i+gw-1] (SW), D[i][i+gw] (S), D[i][i+gw+1] (SE).  Each
// epilogue thread drains its TMEM row window in 32-column chunks, parks each
// chunk in its own row of a padded shared buffer and picks the five
// diagonals; k_css_phi then forms Phi from the per-token dots (Eqs. 4-5).
// B stages hold cap_rows key rows ([2 halves][cap_rows][128 B]), loaded as
// 64-row TMA boxes: the widest frame of the launch sets cap_rows =
// roundup64(roundup16(128 + gw + 1)), and as many stages as fit (2 to 4).
constexpr int kCssStgRow = 36;                           // floats per staged row (16-byte rows, no conflicts)
constexpr int kCssStgBytes = 8 * 32 * kCssStgRow * 4;    // 8 warps x [32][36] floats
constexpr int kCssBarBytes = 128;                        // kfull[4], kempty[4], accfull[2], accempty[2], done, slot, abort
constexpr int kCssSmemMax = 232448;
constexpr int kCssMaxGw = 127;                           // NB <= 256
constexpr int kCssMaxStages = 4;

struct CssGeom {
  int cap_rows;     // key rows per B stage (multiple of 64)
  int stage_bytes;  // 2 * cap_rows * 128
  int stages;       // B stages in the ring
  int smem;         // dynamic shared memory of the launch
};

struct CssDots {
  Strided<float> rn, dE, dS, dSE, dSW, rn_cur;
  int cur_pad;
};

// Frame f and first token t0 of CSS tile t (the tiles of frame f are
// ctile0[f] .. ctile0[f+1]-1), for a loop whose tiles only grow: f carries
// the frame of the previous tile (start it at 0), so a step costs a
// comparison or two instead of a search.
__device__ __forceinline__ void css_tile_next(const FrameTable& ft, int t, int& f, int& t0) {
  while (f + 1 < ft.n_frames && ft.ctile0[f + 1] <= t) ++f;
  t0 = ft.off[f] + (t - ft.ctile0[f]) * 128;
}

__global__ void __launch_bounds__(kThreads, 1)
    k_css_umma(const __grid_constant__ KMaps maps, const __grid_constant__ FrameTable ft, int hkv,
               CssDots out, CssGeom geo, uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  const int S = geo.stages, SB = geo.stage_bytes, half_bytes = geo.cap_rows * 128;
  const int off_stg = S * SB, off_bar = off_stg + kCssStgBytes;
  if ((int)(sm - smem_raw) + off_bar + kCssBarBytes > geo.smem) {  // uniform: the layout would not fit
    if (threadIdx.x == 0) record_error(err, kErrLaunch);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int l = blockIdx.y / hkv, h = blockIdx.y % hkv, n = ft.n_tokens;
  const CUtensorMap& kmap = maps.m[l];
  const int ntiles_all = ft.ctile0[ft.n_frames];
  const uint32_t sB = smem_u32(sm);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + off_bar);
  const uint32_t b_kfull = smem_u32(&bars[0]), b_kempty = smem_u32(&bars[kCssMaxStages]);
  const uint32_t b_accfull = smem_u32(&bars[2 * kCssMaxStages]);
  const uint32_t b_accempty = smem_u32(&bars[2 * kCssMaxStages + 2]);
  const uint32_t b_done = smem_u32(&bars[2 * kCssMaxStages + 4]);
  uint32_t* slot = reinterpret_cast<uint32_t*>(sm + off_bar + (2 * kCssMaxStages + 5) * 8);
  volatile uint32_t* abort_flag = slot + 1;
  int ntiles = 0;
  for (int t = blockIdx.x; t < ntiles_all; t += gridDim.x) ++ntiles;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(b_kfull + 8 * i, 1);
      mbar_init(b_kempty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4);
    }
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&kmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(slot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;

  if (warp == 0) {
    if (lane == 0) {
      int issued[kCssMaxStages] = {0, 0, 0, 0};
      int f = 0, ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks;
        const uint32_t u = kp;
        if (!mbar_wait(b_kempty + 8 * s, (u & 1u) ^ 1u, err, abort_flag)) break;
        int t0;
        css_tile_next(ft, blockIdx.x + it * gridDim.x, f, t0);
        const int nbox = (((128 + ft.gw[f] + 1 + 15) & ~15) + 63) / 64;  // 64-row boxes covering NB rows
        mbar_arrive_expect_tx(b_kfull + 8 * s, (uint32_t)(2 * nbox * 64 * 128));
        for (int kb = 0; kb < 2; ++kb)
          for (int r = 0; r < nbox; ++r)
            tma_load_3d(sB + s * SB + kb * half_bytes + r * 8192, &kmap, b_kfull + 8 * s, kb * 64, h,
                        t0 + r * 64);
        ++issued[s];
      }
      if (*abort_flag)
        for (int s = 0; s < S; ++s)
          if (issued[s]) mbar_wait_drain(b_kfull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int f = 0, ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; it < ntiles; ++it, ks = ks + 1 == S ? 0 : ks + 1, kp += ks == 0u ? 1u : 0u) {
        const int s = ks, as = it & 1;
        if (!mbar_wait(b_kfull + 8 * s, kp & 1u, err, abort_flag)) break;
        if (!mbar_wait(b_accempty + 8 * as, ((uint32_t)(it >> 1) & 1u) ^ 1u, err, abort_flag)) break;
        tc_fence_after();
        int t0;
        css_tile_next(ft, blockIdx.x + it * gridDim.x, f, t0);
        const int nb = (128 + ft.gw[f] + 1 + 15) & ~15;
        const uint32_t idesc = idesc_bf16(128, nb);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t kb = k >> 2, koff = (k & 3) * 32;
          const uint64_t d = desc_sw128(sB + s * SB + kb * half_bytes + koff);
          umma_bf16(tmem + as * 256, d, d, idesc, k > 0 ? 1u : 0u);
        }
        umma_commit(b_accfull + 8 * as);
        umma_commit(b_kempty + 8 * s);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else {
    const int g = (warp - 2) >> 2, quarter = warp & 3;
    float* stg = reinterpret_cast<float*>(sm + off_stg) + (size_t)(warp - 2) * 32 * kCssStgRow + lane * kCssStgRow;
    const uint32_t tbase = tmem + ((uint32_t)(quarter * 32) << 16) + g * 256 + quarter * 32;
    float* rn_o = out.rn.at(l) + (size_t)h * n;
    float* e_o = out.dE.at(l) + (size_t)h * n;
    float* s_o = out.dS.at(l) + (size_t)h * n;
    float* se_o = out.dSE.at(l) + (size_t)h * n;
    float* sw_o = out.dSW.at(l) + (size_t)h * n;
    float* rc_o = out.rn_cur.at(l) + (size_t)h * out.cur_pad;
    int f = 0;
    for (int it = g; it < ntiles; it += 2) {
      const uint32_t ua = (uint32_t)(it >> 1);
      if (!warp_wait(b_accfull + 8 * g, ua & 1u, err, abort_flag)) break;
      tc_fence_after();
      int t0;
      css_tile_next(ft, blockIdx.x + it * gridDim.x, f, t0);
      const int gw = ft.gw[f];
      const int dd[5] = {0, 1, gw - 1, gw, gw + 1};
      float val[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
      const int nch = (32 + gw + 1 + 31) >> 5;  // row i needs columns i .. i+gw+1
      // park a 32-column chunk in this lane's staging row and pick the
      // diagonals that fall in it
      auto pick = [&](const uint32_t (&w)[32], int c) {
#pragma unroll
        for (int k = 0; k < 8; ++k)
          *reinterpret_cast<uint4*>(stg + 4 * k) = make_uint4(w[4 * k], w[4 * k + 1], w[4 * k + 2], w[4 * k + 3]);
#pragma unroll
        for (int q = 0; q < 5; ++q) {
          const int idx = lane + dd[q] - 32 * c;
          if (idx >= 0 && idx < 32) val[q] = stg[idx];
        }
      };
      if (nch <= 3) {
        // every load of the window in flight at once (grids up to 63 wide)
        uint32_t w0[32], w1[32], w2[32];
        tmem_ld32_issue(tbase, w0);
        if (nch > 1) tmem_ld32_issue(tbase + 32, w1);
        if (nch > 2) tmem_ld32_issue(tbase + 64, w2);
        tmem_wait_regs96(w0, w1, w2);
        pick(w0, 0);
        if (nch > 1) pick(w1, 1);
        if (nch > 2) pick(w2, 2);
      } else {
        for (int c = 0; c < nch; ++c) {
          uint32_t w0[32], w1[32], w2[32];
          tmem_ld32_issue(tbase + c * 32, w0);
          tmem_wait_regs96(w0, w1, w2);
          pick(w0, c);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_accempty + 8 * g);
      const int tok = t0 + quarter * 32 + lane;
      if (tok < ft.off[f] + ft.gh[f] * gw) {
        const float r = 1.0f / fmaxf(sqrtf(val[0]), 1e-8f);
        rn_o[tok] = r;
        e_o[tok] = val[1];
        sw_o[tok] = val[2];
        s_o[tok] = val[3];
        se_o[tok] = val[4];
        if (f == ft.n_frames - 1) rc_o[tok - ft.cur_off] = r;
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Phi from the per-token dots: the eight in-grid Moore neighbours of (u, v)
// are E, W, S, N, SE, NW, SW, NE; W's dot is E of the left neighbour, N's is
// S of the upper one, NW's is SE of the upper-left one and NE's is SW of the
// upper-right one.  A thread takes kPhiRun consecutive cells of one grid
// row, so that the index arithmetic and the loads of the shared neighbours
// are done once per run.  grid = (run block, frame, layer*Hkv + head).
constexpr int kPhiRun = 4;
__global__ void __launch_bounds__(256) k_css_phi(const __grid_constant__ FrameTable ft, int hkv, CssDots d,
                                                 Strided<float> phi_all) {
  const int f = blockIdx.y, l = blockIdx.z / hkv, h = blockIdx.z % hkv, n = ft.n_tokens;
  if (f >= ft.n_frames) return;
  const int gh = ft.gh[f], gw = ft.gw[f], off = ft.off[f];
  const int runs = (gw + kPhiRun - 1) / kPhiRun;  // runs per grid row
  const int slot = blockIdx.x * blockDim.x + threadIdx.x;
  if (slot >= gh * runs) return;
  const int u = slot / runs, v0 = (slot - u * runs) * kPhiRun;
  const size_t hn = (size_t)h * n;
  const float* rn = d.rn.at(l) + hn;
  const float* e = d.dE.at(l) + hn;
  const float* s = d.dS.at(l) + hn;
  const float* se = d.dSE.at(l) + hn;
  const float* sw = d.dSW.at(l) + hn;
  const bool up = u > 0, dn = u + 1 < gh;
  const int j0 = off + u * gw + v0;  // token of cell (u, v0)
  // columns v0 - 1 .. v0 + kPhiRun of the rows above, at and below: index
  // c + 1 holds column v0 + c (loads outside the grid are skipped)
  float ra[kPhiRun + 2], rc[kPhiRun + 2], rb[kPhiRun + 2];
  float ec[kPhiRun + 1], sa[kPhiRun], sc[kPhiRun], sea[kPhiRun + 1], sec[kPhiRun], swa[kPhiRun + 1], swc[kPhiRun];
  static_assert(kPhiRun == 4, "the vector path loads a run as one float4");
  // 16-byte loads of the run's columns when every row of the arrays and the
  // frame's rows start on a 16-byte boundary (N, the frame offset and the
  // grid width multiples of four); v0 + 3 < gw then holds as well
  if ((n & 3) == 0 && (off & 3) == 0 && (gw & 3) == 0) {
    auto ld4 = [](const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); };
    auto put4 = [](float* d, float4 x) {
      d[0] = x.x;
      d[1] = x.y;
      d[2] = x.z;
      d[3] = x.w;
    };
    const bool lf0 = v0 > 0, rt4 = v0 + kPhiRun < gw;
    put4(rc + 1, ld4(rn + j0));
    rc[0] = lf0 ? __ldg(rn + j0 - 1) : 0.f;
    rc[5] = rt4 ? __ldg(rn + j0 + 4) : 0.f;
    put4(ec + 1, ld4(e + j0));
    ec[0] = lf0 ? __ldg(e + j0 - 1) : 0.f;
    if (up) {
      put4(ra + 1, ld4(rn + j0 - gw));
      ra[0] = lf0 ? __ldg(rn + j0 - gw - 1) : 0.f;
      ra[5] = rt4 ? __ldg(rn + j0 - gw + 4) : 0.f;
      put4(sea + 1, ld4(se + j0 - gw));
      sea[0] = lf0 ? __ldg(se + j0 - gw - 1) : 0.f;
      put4(sa, ld4(s + j0 - gw));
      // SW of (u - 1, v + 2) for c = -1 .. 3: columns v0 + 1 .. v0 + 5
      const float4 w0 = ld4(sw + j0 - gw);
      const float4 w1 = rt4 ? ld4(sw + j0 - gw + 4) : make_float4(0.f, 0.f, 0.f, 0.f);
      swa[0] = w0.y;
      swa[1] = w0.z;
      swa[2] = w0.w;
      swa[3] = w1.x;
      swa[4] = w1.y;
    } else {
#pragma unroll
      for (int i = 0; i < kPhiRun + 2; ++i) ra[i] = 0.f;
#pragma unroll
      for (int i = 0; i < kPhiRun + 1; ++i) sea[i] = swa[i] = 0.f;
#pragma unroll
      for (int i = 0; i < kPhiRun; ++i) sa[i] = 0.f;
    }
    if (dn) {
      put4(rb + 1, ld4(rn + j0 + gw));
      rb[0] = lf0 ? __ldg(rn + j0 + gw - 1) : 0.f;
      rb[5] = rt4 ? __ldg(rn + j0 + gw + 4) : 0.f;
      put4(sc, ld4(s + j0));
      put4(sec, ld4(se + j0));
      put4(swc, ld4(sw + j0));
    } else {
#pragma unroll
      for (int i = 0; i < kPhiRun + 2; ++i) rb[i] = 0.f;
#pragma unroll
      for (int i = 0; i < kPhiRun; ++i) sc[i] = sec[i] = swc[i] = 0.f;
    }
  } else {
#pragma unroll
    for (int c = -1; c <= kPhiRun; ++c) {
      const int v = v0 + c;
      const bool in = v >= 0 && v < gw;
      rc[c + 1] = in ? __ldg(rn + j0 + c) : 0.f;
      ra[c + 1] = in && up ? __ldg(rn + j0 + c - gw) : 0.f;
      rb[c + 1] = in && dn ? __ldg(rn + j0 + c + gw) : 0.f;
    }
#pragma unroll
    for (int c = -1; c < kPhiRun; ++c) {
      const int v = v0 + c;
      const bool in = v >= 0 && v < gw;
      ec[c + 1] = in ? __ldg(e + j0 + c) : 0.f;                    // E of (u, v)
      sea[c + 1] = in && up ? __ldg(se + j0 + c - gw) : 0.f;       // SE of (u - 1, v)
      const bool in2 = v + 2 >= 0 && v + 2 < gw;
      swa[c + 1] = in2 && up ? __ldg(sw + j0 + c + 2 - gw) : 0.f;  // SW of (u - 1, v + 2)
    }
#pragma unroll
    for (int c = 0; c < kPhiRun; ++c) {
      const bool in = v0 + c < gw;
      sa[c] = in && up ? __ldg(s + j0 + c - gw) : 0.f;
      sc[c] = in && dn ? __ldg(s + j0 + c) : 0.f;
      sec[c] = in && dn ? __ldg(se + j0 + c) : 0.f;
      swc[c] = in && dn ? __ldg(sw + j0 + c) : 0.f;
    }
  }
  float* phi = phi_all.at(l) + hn;
#pragma unroll
  for (int c = 0; c < kPhiRun; ++c) {
    const int v = v0 + c;
    if (v >= gw) break;
    const bool lf = v > 0, rt = v + 1 < gw;
    const float r0 = rc[c + 1];
    float sum = 0.f;
    int cnt = 0;
    if (rt) { sum += ec[c + 1] * r0 * rc[c + 2]; ++cnt; }
    if (lf) { sum += ec[c] * rc[c] * r0; ++cnt; }
    if (dn) { sum += sc[c] * r0 * rb[c + 1]; ++cnt; }
    if (up) { sum += sa[c] * ra[c + 1] * r0; ++cnt; }
    if (dn && rt) { sum += sec[c] * r0 * rb[c + 2]; ++cnt; }
    if (up && lf) { sum += sea[c] * ra[c] * r0; ++cnt; }
    if (dn && lf) { sum += swc[c] * r0 * rb[c]; ++cnt; }
    if (up && rt) { sum += swa[c] * ra[c + 2] * r0; ++cnt; }
    phi[j0 + c] = cnt ? 1.0f - sum / (float)cnt : 0.0f;
  }
}

// =========================================================================
// host side

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// K [N][Hkv][128] bf16 as a 3-D tensor (d, head, token); box = 64 x 1 x rows
// with the 128-byte swizzle, out-of-range tokens read as zero.
static cudaError_t make_kmap(CUtensorMap* m, const void* k, int n, int hkv, int rows) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)hkv, (cuuint64_t)n};
  cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)hkv * kD * 2};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)rows};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(k), dims, strides, box,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_row_map(CUtensorMap* m, const void* base, int n, int hkv, int rows) {
  return make_kmap(m, base, n, hkv, rows);
}

static int sm_count() {
  int dev = 0, c = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev);
  return c > 0 ? c : 148;
}

// CTAs per work unit (1..cap): one wave when the units are fewer than the
// SMs, else the split among 1..4 that fills whole waves best.
static int pick_split(int units, int cap, int slots) {
  // Splits s of each unit so that units * s CTAs (one per SM) fill whole
  // waves as nearly as possible; among equal fills the fewest CTAs win.
  if (cap < 1) cap = 1;
  const int even = (slots + units - 1) / units;
  int smax = 4 * even;
  if (smax < 4) smax = 4;
  if (smax > cap) smax = cap;
  int best = 1;
  double best_eff = 0.0;
  for (int s = 1; s <= smax; ++s) {
    const long long ctas = (long long)units * s;
    const long long waves = (ctas + slots - 1) / slots;
    const double eff = (double)ctas / (double)(waves * slots);
    if (eff > best_eff + 0.02) {
      best = s;
      best_eff = eff;
    }
  }
  return best;
}

static cudaError_t make_kmaps(KMaps* maps, const LayerPtrs& io, int L, int n, int hkv, int rows) {
  for (int l = 0; l < L; ++l) {
    cudaError_t e = make_kmap(&maps->m[l], io.k[l], n, hkv, rows);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Key splits of window-score pass 1.  They fix how the fp32 row sums are
// grouped, so they depend on the problem shape only -- not on the batch
// size or the device -- and a layer gives the same bits alone or batched:
// one wave of a nominal 152-SM GB300 for one layer, more waves for batches.
static int score_tiles(const Problem& p) {
  const int kn = p.dtype == kBF16 ? rs_layout(p.R()).KN : 64;
  return (p.n + kn - 1) / kn;
}

int score_nsplit_max(const Problem& p) {
  const int tiles = score_tiles(p);
  if (p.dtype == kBF16) {
    // bf16: enough splits that one layer alone fills one wave of a nominal
    // 152-SM GB300, every split non-empty; a batch of layers runs several
    // splits per CTA (the partials stay those of the shape)
    // (at least two tiles per split: a one-tile split hands its partial over
    // after every tile and doubles the partials the row-bias pass merges)
    const int nmh = rs_layout(p.R()).NMH;
    int target = (152 + p.hkv * nmh - 1) / (p.hkv * nmh);
    if (target > tiles) target = tiles;
    if (target < 1) target = 1;
    int per_t = (tiles + target - 1) / target;
    if (per_t < 2) per_t = 2;
    return (tiles + per_t - 1) / per_t;
  }
  int s = pick_split(p.hkv, tiles, 2 * 152);
  return s < 1 ? 1 : s;
}

int score_nsplit(const Problem& p) { return score_nsplit_max(p); }

cudaError_t launch_tsg_umma(const Problem& p, const FrameTable& ft, const LayerPtrs& io,
                            Strided<const float> rn_cur, int cur_pad, Strided<float> rho_part, int metric,
                            uint32_t* err, cudaStream_t st) {
  if (ft.n_frames < 2) return cudaSuccess;
  const int n_tiles = ft.tsg_tiles;
  if (n_tiles == 0 || ft.cur_len == 0) return cudaSuccess;
  const int nchunk = (ft.cur_len + 511) / 512;
  KMaps local;
  cudaError_t e = make_kmaps(&local, io, p.L, p.n, p.hkv, 128);
  if (e != cudaSuccess) return e;
  auto kern = metric == kTsgDot ? k_tsg_umma<kTsgDot> : (metric == kTsgNegL2 ? k_tsg_umma<kTsgNegL2> : k_tsg_umma<kTsgCosine>);
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kTsgSmem);
  if (e != cudaSuccess) return e;
  const int groups = nchunk * p.L * p.hkv;
  const int gx = pick_split(groups, n_tiles, sm_count());
  dim3 grid(gx, nchunk, p.L * p.hkv);
  TimingScope ts("tsg_umma", st);
  kern<<<grid, kThreads, kTsgSmem, st>>>(local, ft, rn_cur, cur_pad, rho_part, p.hkv, err);
  return cudaGetLastError();
}

cudaError_t launch_score_umma(const Problem& p, const LayerPtrs& io, Strided<float2> rowpart, int nsplit,
                              Strided<float> a_base, uint32_t* err, cudaStream_t st) {
  const int R = p.R();
  if (R > 512) return cudaErrorNotSupported;
  const RsLayout L1 = rs_layout(R);
  const CsLayout L2 = cs_layout(R);
  KMaps m1, m2;
  cudaError_t e = make_kmaps(&m1, io, p.L, p.n, p.hkv, L1.KN);
  if (e != cudaSuccess) return e;
  if ((e = make_kmaps(&m2, io, p.L, p.n, p.hkv, 128)) != cudaSuccess) return e;
  auto rs_kernel = L1.MT == 1 ? k_rowstats_umma<1> : k_rowstats_umma<2>;
  if ((e = cudaFuncSetAttribute(rs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, L1.total)) !=
      cudaSuccess)
    return e;
  auto cs_kernel = L2.nh == 2 ? k_colsum_umma<2> : k_colsum_umma<1>;
  if ((e = cudaFuncSetAttribute(cs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, L2.total)) != cudaSuccess)
    return e;
  {
    TimingScope ts("rowstats_umma", st);
    // CTAs per (layer, head, row half): whole waves for the batch, each
    // taking cps consecutive splits
    const int cph0 = pick_split(p.L * p.hkv * L1.NMH, nsplit, sm_count());
    const int cps = (nsplit + cph0 - 1) / cph0;
    const int cph = (nsplit + cps - 1) / cps;
    rs_kernel<<<dim3(cph * L1.NMH, p.L * p.hkv), kScoreThreads, L1.total, st>>>(m1, io, p, nsplit, cps, rowpart,
                                                                               err);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  {
    TimingScope ts("row_bias", st);
    launch_row_bias(p, nsplit, rowpart, st);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int tiles = (p.n + 127) / 128;
  const int gx = pick_split(p.L * p.hkv, tiles, sm_count());
  TimingScope ts("colsum_umma", st);
  cs_kernel<<<dim3(gx, p.L * p.hkv), kCsThreads, L2.total, st>>>(m2, io, p, rowpart, nsplit, a_base, err);
  return cudaGetLastError();
}

bool css_umma_supported(const FrameTable& ft) {
  for (int f = 0; f < ft.n_frames; ++f)
    if (ft.gw[f] > kCssMaxGw) return false;
  return true;
}

cudaError_t launch_css_umma(const Problem& p, const FrameTable& ft, const LayerPtrs& io, Strided<float> phi,
                            Strided<float> rn, Strided<float> rn_cur, int cur_pad, Strided<float> dE,
                            Strided<float> dS, Strided<float> dSE, Strided<float> dSW, uint32_t* err,
                            cudaStream_t st, bool with_phi) {
  const int tiles = ft.ctile0[ft.n_frames];
  if (tiles == 0) return cudaSuccess;
  KMaps maps;
  cudaError_t e = make_kmaps(&maps, io, p.L, p.n, p.hkv, 64);
  if (e != cudaSuccess) return e;
  CssGeom geo;
  int nb_max = 0;
  for (int f = 0; f < ft.n_frames; ++f) nb_max = max(nb_max, (128 + ft.gw[f] + 1 + 15) & ~15);
  geo.cap_rows = (nb_max + 63) / 64 * 64;
  geo.stage_bytes = 2 * geo.cap_rows * 128;
  geo.smem = kCssSmemMax;
  geo.stages = (kCssSmemMax - 1024 - kCssStgBytes - kCssBarBytes) / geo.stage_bytes;
  if (geo.stages > kCssMaxStages) geo.stages = kCssMaxStages;
  if (geo.stages < 2) return cudaErrorNotSupported;
  if ((e = cudaFuncSetAttribute(k_css_umma, cudaFuncAttributeMaxDynamicSharedMemorySize, geo.smem)) !=
      cudaSuccess)
    return e;
  CssDots d;
  d.rn = rn;
  d.dE = dE;
  d.dS = dS;
  d.dSE = dSE;
  d.dSW = dSW;
  d.rn_cur = rn_cur;
  d.cur_pad = cur_pad;
  const int gx = pick_split(p.L * p.hkv, tiles, sm_count());
  {
    TimingScope ts("css_umma", st);
    k_css_umma<<<dim3(gx, p.L * p.hkv), kThreads, geo.smem, st>>>(maps, ft, p.hkv, d, geo, err);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  return with_phi ? launch_css_phi(p, ft, phi, rn, rn_cur, cur_pad, dE, dS, dSE, dSW, st) : cudaSuccess;
}

cudaError_t launch_css_phi(const Problem& p, const FrameTable& ft, Strided<float> phi, Strided<float> rn,
                           Strided<float> rn_cur, int cur_pad, Strided<float> dE, Strided<float> dS,
                           Strided<float> dSE, Strided<float> dSW, cudaStream_t st) {
  if (ft.ctile0[ft.n_frames] == 0) return cudaSuccess;
  CssDots d;
  d.rn = rn;
  d.dE = dE;
  d.dS = dS;
  d.dSE = dSE;
  d.dSW = dSW;
  d.rn_cur = rn_cur;
  d.cur_pad = cur_pad;
  int cmax = 1;  // the most kPhiRun-cell runs of any frame
  for (int f = 0; f < ft.n_frames; ++f) cmax = max(cmax, ft.gh[f] * ((ft.gw[f] + kPhiRun - 1) / kPhiRun));
  TimingScope ts("css_phi", st);
  k_css_phi<<<dim3((cmax + 255) / 256, ft.n_frames, p.L * p.hkv), 256, 0, st>>>(ft, p.hkv, d, phi);
  return cudaGetLastError();
}

}  // namespace stl
