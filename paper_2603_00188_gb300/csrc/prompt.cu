// Prompt-wide base scores on the tensor cores (bf16): the Mean Attention and
// full-attention ("snapshot") bases of the base-scoring ablation (appendix
// "Sensitivity to the Base Attention Scoring Function").  The last nq cached
// positions are query rows; row (position p, query head g) attends causally
// to keys j <= p.  For KV head h:
//   C[j] = (1/G) sum_{g in group h} sum_{p >= j} softmax_{j' <= p}(q_{p,g} . k_{j',h} / sqrt(d))_j
// full base A = C; Mean Attention A = C / #{prompt rows that attend to j}.
//
//   k_prompt_rowstats  pass 1: one CTA per 128-row m-tile of query rows
//                      (P1 = floor(128 / G) whole positions, G rows each);
//                      key tiles of 256 stream up to the tile's last
//                      position; per row the running max and sum of
//                      exponentials under the causal mask, merged over four
//                      epilogue groups into bias_r = -m_r - log2(G l_r).
//   k_prompt_colsum    pass 2: one CTA per 128-key tile, the tile resident
//                      in shared memory as the A operand; chunks of P2 =
//                      floor(256 / G) positions (G P2 rows) stream as the
//                      B operand from the first chunk that can see the
//                      tile; each key sums 2^(x c + bias_r) over the rows
//                      that attend to it.  Every key's sum is formed in one
//                      CTA, in a fixed order: no atomics, no reduction pass.
//
// Query rows come straight from q [nq][Hq][128] through a 3-D TMA box (d,
// the group's G heads, positions): its lines land in shared memory in
// (position, head) order, which is the row order r = position * G + g.
// Same warp roles as the window-score passes: warp 0 TMA, warp 1 MMA, four
// groups of four epilogue warps; every mbarrier wait is bounded.
#include <cudaTypedefs.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace stl {

namespace {

constexpr int kPrGroups = 4;
constexpr int kPrThreads = (2 + 4 * kPrGroups) * 32;
constexpr int kPrMaxReg = 96;
constexpr float kPrLog2e = 1.4426950408889634f;

// pass 1: Q m-tile [2 halves][128 rows][128 B], two key stages of 256 keys
constexpr int kP1Q = 0;
constexpr int kP1K = 32768;
constexpr int kP1KStage = 65536;
constexpr int kP1Stages = 2;
constexpr int kP1Bar = kP1K + kP1Stages * kP1KStage;  // 8 mbarriers, slot, abort
constexpr int kP1Xch = kP1Bar + 128;                   // float2 [4 groups][128 rows]
constexpr int kP1Smem = kP1Xch + kPrGroups * 128 * 8 + 1024;

// pass 2: key tile [2 halves][128 keys][128 B], two Q stages of 256 rows,
// the stages' row biases, the groups' partial sums
constexpr int kP2K = 0;
constexpr int kP2Q = 32768;
constexpr int kP2QStage = 65536;
constexpr int kP2Stages = 2;
constexpr int kP2Bias = kP2Q + kP2Stages * kP2QStage;  // float [stages][256]
constexpr int kP2Bar = kP2Bias + kP2Stages * 1024;
constexpr int kP2Xch = kP2Bar + 128;                    // float [4 groups][128 keys]
constexpr int kP2Smem = kP2Xch + kPrGroups * 128 * 4 + 1024;

__device__ __forceinline__ uint8_t* pr_align1024(uint8_t* p) {
  uint32_t a = smem_u32(p);
  return p + ((1024u - (a & 1023u)) & 1023u);
}

// Contiguous global -> shared copy completing on `bar` (16-byte aligned
// addresses, size a multiple of 16).
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}

// Named barrier over the 16 epilogue warps (id 1).
__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, %0;" ::"n"(4 * kPrGroups * 32)); }

}  // namespace

struct PromptMaps {
  CUtensorMap q1;  // box 64 x G x P1
  CUtensorMap q2;  // box 64 x G x P2
  CUtensorMap k1;  // box 64 x 1 x 256
  CUtensorMap k2;  // box 64 x 1 x 128
};

struct PromptArgs {
  int n, nq, hq, hkv, G;
  int p1, p2;      // positions per pass-1 m-tile / pass-2 chunk
  int n_mt, n_ch;  // m-tiles and chunks per head
  int crp;         // bias floats per chunk (G P2 rounded up to 4)
  int mode;        // 0 full, 1 mean
};

// bias [Hkv][n_ch][crp]: entry of row (relative position pr, head g of the
// group) at chunk pr / P2, offset (pr % P2) G + g; every other entry -inf.
__global__ void k_prompt_bias_fill(float* bias, size_t count) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < count; i += (size_t)gridDim.x * blockDim.x)
    bias[i] = -CUDART_INF_F;
}

__global__ void __maxnreg__(kPrMaxReg)
    k_prompt_rowstats(const __grid_constant__ PromptMaps maps, PromptArgs a, float* bias, uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = pr_align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x % a.hkv;
  const int mt = a.n_mt - 1 - (int)(blockIdx.x / a.hkv);  // longest rows first
  const int p_first = a.n - a.nq;
  const int pr0 = mt * a.p1;                               // first relative position of the tile
  const int npos = min(a.p1, a.nq - pr0);
  const int rows = npos * a.G;
  const int pa = p_first + pr0;                            // first absolute position
  const int kend = pa + npos;                              // keys [0, kend) are visible to some row
  const int ntiles = (kend + 255) / 256;
  const uint32_t sQ = smem_u32(sm + kP1Q), sK = smem_u32(sm + kP1K);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kP1Bar);
  const uint32_t b_kfull = smem_u32(&bars[0]), b_kempty = smem_u32(&bars[kP1Stages]);
  const uint32_t b_accfull = smem_u32(&bars[2 * kP1Stages]), b_accempty = smem_u32(&bars[2 * kP1Stages + 2]);
  const uint32_t b_q = smem_u32(&bars[2 * kP1Stages + 4]), b_done = smem_u32(&bars[2 * kP1Stages + 5]);
  uint32_t* slot = reinterpret_cast<uint32_t*>(sm + kP1Bar + 8 * (2 * kP1Stages + 6));
  volatile uint32_t* abort_flag = slot + 1;
  float2* xch = reinterpret_cast<float2*>(sm + kP1Xch);
  const float c = kPrLog2e * rsqrtf((float)kD);

  if (threadIdx.x == 0) {
    for (int i = 0; i < kP1Stages; ++i) {
      mbar_init(b_kfull + 8 * i, 1);
      mbar_init(b_kempty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4 * kPrGroups);
    }
    mbar_init(b_q, 1);
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&maps.q1);
    tma_prefetch_desc(&maps.k1);
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
      // the m-tile's rows: positions [pr0, pr0 + P1) of the group's G heads
      const uint32_t qbytes = 2u * 128u * (uint32_t)(a.G * a.p1);
      mbar_arrive_expect_tx(b_q, qbytes);
      tma_load_3d(sQ, &maps.q1, b_q, 0, h * a.G, pr0);
      tma_load_3d(sQ + 16384, &maps.q1, b_q, 64, h * a.G, pr0);
      int issued[kP1Stages] = {0, 0};
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; it < ntiles; ++it, ks = ks + 1 == kP1Stages ? 0 : ks + 1, kp += ks == 0 ? 1u : 0u) {
        if (!mbar_wait(b_kempty + 8 * ks, (kp & 1u) ^ 1u, err, abort_flag)) break;
        mbar_arrive_expect_tx(b_kfull + 8 * ks, (uint32_t)kP1KStage);
        tma_load_3d(sK + ks * kP1KStage, &maps.k1, b_kfull + 8 * ks, 0, h, it * 256);
        tma_load_3d(sK + ks * kP1KStage + 32768, &maps.k1, b_kfull + 8 * ks, 64, h, it * 256);
        ++issued[ks];
      }
      if (*abort_flag) {
        mbar_wait_drain(b_q, 0);
        for (int s = 0; s < kP1Stages; ++s)
          if (issued[s]) mbar_wait_drain(b_kfull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, 256);
      bool ok = mbar_wait(b_q, 0, err, abort_flag);
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; ok && it < ntiles; ++it, ks = ks + 1 == kP1Stages ? 0 : ks + 1, kp += ks == 0 ? 1u : 0u) {
        if (!mbar_wait(b_kfull + 8 * ks, kp & 1u, err, abort_flag)) break;
        const int as = it & 1;
        if (!mbar_wait(b_accempty + 8 * as, ((uint32_t)(it >> 1) & 1u) ^ 1u, err, abort_flag)) break;
        tc_fence_after();
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t kb = k >> 2, koff = (k & 3) * 32;
          const uint64_t ad = desc_sw128(sQ + kb * 16384 + koff);
          const uint64_t bd = desc_sw128(sK + ks * kP1KStage + kb * 32768 + koff);
          umma_bf16(tmem + as * 256, ad, bd, idesc, k > 0 ? 1u : 0u);
        }
        umma_commit(b_accfull + 8 * as);
        umma_commit(b_kempty + 8 * ks);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else {
    // group g drains key columns [64 g, 64 g + 64) of every item; the
    // thread owns query row `row` (TMEM lane) at absolute position pos
    const int g = (warp - 2) >> 2, quarter = warp & 3, row = quarter * 32 + lane;
    const int pos = pa + row / a.G;
    const uint32_t lanebase = tmem + ((uint32_t)(quarter * 32) << 16) + g * 64;
    float m = -CUDART_INF_F, l = 0.f;
    for (int it = 0; it < ntiles; ++it) {
      const int as = it & 1;
      if (!warp_wait(b_accfull + 8 * as, (uint32_t)(it >> 1) & 1u, err, abort_flag)) break;
      tc_fence_after();
      float v[64];
      tmem_ld64(lanebase + as * 256, v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_accempty + 8 * as);
      const int key0 = it * 256 + g * 64;
      if (key0 + 63 <= pa) {
        // every row of the tile sees all 64 keys.  The maximum over four
        // independent max3 chains (exact in any order); then exponent
        // arguments, exponentials and sums in three phases with packed
        // fp32x2 operations (each lane of a pair rounds as the scalar op)
        float cm[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) cm[r] = v[r];
#pragma unroll
        for (int i = 4; i < 64; i += 8) {
#pragma unroll
          for (int r = 0; r < 4; ++r)
            if (i + 2 * r + 1 < 64) cm[r] = max3(cm[r], v[i + 2 * r], v[i + 2 * r + 1]);
        }
        const float mx = fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3]));
        const float mn = fmaxf(m, mx), mnc = mn * c;
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
        for (int i = 0; i < 64; i += 2) fma2(v[i], v[i + 1], c, c, -mnc, -mnc, v[i], v[i + 1]);
#pragma unroll
        for (int i = 0; i < 64; ++i) v[i] = ex2_approx(v[i]);
#pragma unroll
        for (int i = 0; i < 64; i += 4) {
          add2(s0, s1, v[i], v[i + 1]);
          add2(s2, s3, v[i + 2], v[i + 3]);
        }
        l = (m == -CUDART_INF_F ? 0.f : l * ex2_approx((m - mn) * c)) + ((s0 + s1) + (s2 + s3));
        m = mn;
      } else {
        // causal edge: keys key0 + i <= pos only
        const int nv = max(0, min(64, pos - key0 + 1));
        if (nv > 0) {
          float mx = -CUDART_INF_F;
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (i < nv) mx = fmaxf(mx, v[i]);
          const float mn = fmaxf(m, mx), mnc = mn * c;
          float sacc = 0.f;
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (i < nv) sacc += ex2_approx(fmaf(v[i], c, -mnc));
          l = (m == -CUDART_INF_F ? 0.f : l * ex2_approx((m - mn) * c)) + sacc;
          m = mn;
        }
      }
    }
    // merge the four groups' states per row in group order
    xch[g * 128 + row] = make_float2(m, l);
    epilogue_sync();
    if (g == 0 && row < rows && !*abort_flag) {
      float mm = xch[row].x, ll = xch[row].y;
      for (int o = 1; o < kPrGroups; ++o) {
        const float2 s = xch[o * 128 + row];
        const float mn = fmaxf(mm, s.x);
        if (mn == -CUDART_INF_F) continue;
        const float x = mm == -CUDART_INF_F ? 0.f : ll * exp2f((mm - mn) * c);
        const float y = s.x == -CUDART_INF_F ? 0.f : s.y * exp2f((s.x - mn) * c);
        mm = mn;
        ll = x + y;
      }
      const int prel = pr0 + row / a.G, gq = row - (row / a.G) * a.G;
      const size_t at = ((size_t)h * a.n_ch + prel / a.p2) * a.crp + (size_t)(prel % a.p2) * a.G + gq;
      bias[at] = -mm * c - log2f((float)a.G * ll);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

__global__ void __maxnreg__(kPrMaxReg)
    k_prompt_colsum(const __grid_constant__ PromptMaps maps, PromptArgs a, const float* bias, float* a_out,
                    uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = pr_align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x % a.hkv, kt = blockIdx.x / a.hkv;  // keys seen by the most rows first
  const int j0 = kt * 128;
  const int p_first = a.n - a.nq;
  const int cstart = j0 <= p_first ? 0 : (j0 - p_first) / a.p2;
  const int nitems = a.n_ch - cstart;
  const uint32_t sK = smem_u32(sm + kP2K), sQ = smem_u32(sm + kP2Q);
  float* bias_s = reinterpret_cast<float*>(sm + kP2Bias);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kP2Bar);
  const uint32_t b_qfull = smem_u32(&bars[0]), b_qempty = smem_u32(&bars[kP2Stages]);
  const uint32_t b_accfull = smem_u32(&bars[2 * kP2Stages]), b_accempty = smem_u32(&bars[2 * kP2Stages + 2]);
  const uint32_t b_k = smem_u32(&bars[2 * kP2Stages + 4]), b_done = smem_u32(&bars[2 * kP2Stages + 5]);
  uint32_t* slot = reinterpret_cast<uint32_t*>(sm + kP2Bar + 8 * (2 * kP2Stages + 6));
  volatile uint32_t* abort_flag = slot + 1;
  float* xch = reinterpret_cast<float*>(sm + kP2Xch);
  const float c = kPrLog2e * rsqrtf((float)kD);
  const int qrows = a.G * a.p2;  // real lines of a chunk; lines up to 256 stay zero

  // zero the lines of every Q stage that no copy writes, and the bias
  // columns past the copied ones (-inf: they add exact zeros)
  for (int e = threadIdx.x; e < kP2Stages * 2 * (256 - qrows) * 8; e += blockDim.x) {
    const int per_half = (256 - qrows) * 8;
    const int s = e / (2 * per_half), rem = e % (2 * per_half), kb = rem / per_half, w = rem % per_half;
    *reinterpret_cast<uint4*>(sm + kP2Q + s * kP2QStage + kb * 32768 + qrows * 128 + w * 16) = make_uint4(0, 0, 0, 0);
  }
  for (int e = threadIdx.x; e < kP2Stages * 256; e += blockDim.x)
    if ((e & 255) >= a.crp) bias_s[e] = -CUDART_INF_F;
  fence_proxy_async_smem();
  if (threadIdx.x == 0) {
    for (int i = 0; i < kP2Stages; ++i) {
      mbar_init(b_qfull + 8 * i, 1);
      mbar_init(b_qempty + 8 * i, 1 + 4 * kPrGroups);  // the MMA's commit and every epilogue warp (bias)
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_accfull + 8 * i, 1);
      mbar_init(b_accempty + 8 * i, 4 * kPrGroups);
    }
    mbar_init(b_k, 1);
    mbar_init(b_done, 1);
    *abort_flag = 0u;
    fence_mbar_init();
    tma_prefetch_desc(&maps.q2);
    tma_prefetch_desc(&maps.k2);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(slot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;
  const float* bias_h = bias + (size_t)h * a.n_ch * a.crp;

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(b_k, 32768u);
      tma_load_3d(sK, &maps.k2, b_k, 0, h, j0);
      tma_load_3d(sK + 16384, &maps.k2, b_k, 64, h, j0);
      const uint32_t qbytes = 2u * 128u * (uint32_t)qrows + 4u * (uint32_t)a.crp;
      int issued[kP2Stages] = {0, 0};
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; it < nitems; ++it, ks = ks + 1 == kP2Stages ? 0 : ks + 1, kp += ks == 0 ? 1u : 0u) {
        if (!mbar_wait(b_qempty + 8 * ks, (kp & 1u) ^ 1u, err, abort_flag)) break;
        const int ch = cstart + it;
        mbar_arrive_expect_tx(b_qfull + 8 * ks, qbytes);
        tma_load_3d(sQ + ks * kP2QStage, &maps.q2, b_qfull + 8 * ks, 0, h * a.G, ch * a.p2);
        tma_load_3d(sQ + ks * kP2QStage + 32768, &maps.q2, b_qfull + 8 * ks, 64, h * a.G, ch * a.p2);
        bulk_g2s(smem_u32(bias_s + ks * 256), bias_h + (size_t)ch * a.crp, 4u * (uint32_t)a.crp,
                 b_qfull + 8 * ks);
        ++issued[ks];
      }
      if (*abort_flag) {
        mbar_wait_drain(b_k, 0);
        for (int s = 0; s < kP2Stages; ++s)
          if (issued[s]) mbar_wait_drain(b_qfull + 8 * s, (uint32_t)(issued[s] - 1) & 1u);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, 256);
      bool ok = mbar_wait(b_k, 0, err, abort_flag);
      int ks = 0;
      uint32_t kp = 0u;
      for (int it = 0; ok && it < nitems; ++it, ks = ks + 1 == kP2Stages ? 0 : ks + 1, kp += ks == 0 ? 1u : 0u) {
        if (!mbar_wait(b_qfull + 8 * ks, kp & 1u, err, abort_flag)) break;
        const int as = it & 1;
        if (!mbar_wait(b_accempty + 8 * as, ((uint32_t)(it >> 1) & 1u) ^ 1u, err, abort_flag)) break;
        tc_fence_after();
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t kb = k >> 2, koff = (k & 3) * 32;
          const uint64_t ad = desc_sw128(sK + kb * 16384 + koff);
          const uint64_t bd = desc_sw128(sQ + ks * kP2QStage + kb * 32768 + koff);
          umma_bf16(tmem + as * 256, ad, bd, idesc, k > 0 ? 1u : 0u);
        }
        umma_commit(b_accfull + 8 * as);
        umma_commit(b_qempty + 8 * ks);
      }
      umma_commit(b_done);
      mbar_wait_drain(b_done, 0);
    }
  } else {
    // group g drains query columns [64 g, 64 g + 64) of every item; the
    // thread owns key j (TMEM lane `row`).  Chunk ch's column col is the row
    // at position p_first + ch P2 + col / G, which attends to j iff
    // col >= (j - chunk's first position) G.
    const int g = (warp - 2) >> 2, quarter = warp & 3, row = quarter * 32 + lane;
    const int j = j0 + row;
    const uint32_t lanebase = tmem + ((uint32_t)(quarter * 32) << 16) + g * 64;
    float sum = 0.f, comp = 0.f;  // compensated running total over the items
    int ks = 0;
    for (int it = 0; it < nitems; ++it, ks = ks + 1 == kP2Stages ? 0 : ks + 1) {
      const int as = it & 1;
      if (!warp_wait(b_accfull + 8 * as, (uint32_t)(it >> 1) & 1u, err, abort_flag)) break;
      tc_fence_after();
      float v[64];
      tmem_ld64(lanebase + as * 256, v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_accempty + 8 * as);
      const float4* b4 = reinterpret_cast<const float4*>(bias_s + ks * 256 + g * 64);
      const int p0 = p_first + (cstart + it) * a.p2;
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
      if (p0 >= j0 + 127) {
        // every row of the chunk sees every key of the tile: exponent
        // arguments, exponentials and sums in three phases, packed fp32x2
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
          add2(s0, s1, v[4 * i], v[4 * i + 1]);
          add2(s2, s3, v[4 * i + 2], v[4 * i + 3]);
        }
      } else {
        const int colmin = max(0, (j - p0) * a.G) - g * 64;  // first visible column of the group's 64
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float4 b = b4[i];
          s0 += 4 * i >= colmin ? ex2_approx(fmaf(v[4 * i], c, b.x)) : 0.f;
          s1 += 4 * i + 1 >= colmin ? ex2_approx(fmaf(v[4 * i + 1], c, b.y)) : 0.f;
          s2 += 4 * i + 2 >= colmin ? ex2_approx(fmaf(v[4 * i + 2], c, b.z)) : 0.f;
          s3 += 4 * i + 3 >= colmin ? ex2_approx(fmaf(v[4 * i + 3], c, b.w)) : 0.f;
        }
      }
      // this stage's biases are read: count the warp out of the stage
      __syncwarp();
      if (lane == 0) mbar_arrive(b_qempty + 8 * ks);
      const float y = ((s0 + s1) + (s2 + s3)) - comp;
      const float t = sum + y;
      comp = (t - sum) - y;
      sum = t;
    }
    xch[g * 128 + row] = sum;
    epilogue_sync();
    if (g == 0 && j < a.n && !*abort_flag) {
      float acc = (xch[row] + xch[128 + row]) + (xch[256 + row] + xch[384 + row]);
      if (a.mode == 1) acc /= (float)min(a.nq, a.n - j);
      a_out[(size_t)h * a.n + j] = acc;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ---- fp32 caches: the same two passes on the CUDA cores --------------------
// Pass 1: one CTA of 128 threads per (query row, KV head); each thread keeps
// an online (max, sum of 2^(x c - max c)) over its strided keys j <= pos, and
// the block merges the threads' states in a fixed order.
constexpr int kPrSimtRows = 128;
__global__ void __launch_bounds__(kPrSimtRows) k_prompt_rowstats_simt(const float* __restrict__ q,
                                                                     const float* __restrict__ k, PromptArgs a,
                                                                     float* bias) {
  __shared__ float qs[kD];
  __shared__ float2 st[kPrSimtRows];
  const int row = blockIdx.x, h = blockIdx.y, tid = threadIdx.x;
  const int prel = row / a.G, gq = row - prel * a.G;
  const int pos = a.n - a.nq + prel;
  const float c = kPrLog2e * rsqrtf((float)kD);
  qs[tid] = q[((size_t)prel * a.hq + h * a.G + gq) * kD + tid];
  __syncthreads();
  float m = -CUDART_INF_F, l = 0.f;
  for (int j = tid; j <= pos; j += kPrSimtRows) {
    const float4* kr = reinterpret_cast<const float4*>(k + ((size_t)j * a.hkv + h) * kD);
    float d = 0.f;
#pragma unroll 8
    for (int e = 0; e < kD / 4; ++e) {
      const float4 kv = __ldg(kr + e);
      d = fmaf(kv.x, qs[4 * e], d);
      d = fmaf(kv.y, qs[4 * e + 1], d);
      d = fmaf(kv.z, qs[4 * e + 2], d);
      d = fmaf(kv.w, qs[4 * e + 3], d);
    }
    const float x = d * c;
    if (x > m) {
      l = (m == -CUDART_INF_F ? 0.f : l * exp2f(m - x)) + 1.f;
      m = x;
    } else {
      l += exp2f(x - m);
    }
  }
  st[tid] = make_float2(m, l);
  __syncthreads();
  if (tid == 0) {
    float mm = -CUDART_INF_F, ll = 0.f;
    for (int t = 0; t < kPrSimtRows; ++t) {
      const float2 s = st[t];
      const float mn = fmaxf(mm, s.x);
      if (mn == -CUDART_INF_F) continue;
      ll = (mm == -CUDART_INF_F ? 0.f : ll * exp2f(mm - mn)) + (s.x == -CUDART_INF_F ? 0.f : s.y * exp2f(s.x - mn));
      mm = mn;
    }
    const size_t at = ((size_t)h * a.n_ch + prel / a.p2) * a.crp + (size_t)(prel % a.p2) * a.G + gq;
    bias[at] = -mm - log2f((float)a.G * ll);
  }
}

// Pass 2: one CTA of 256 threads per (32-key tile, KV head).  The tile's keys
// and, in turn, tiles of query rows (with their biases) sit in shared
// memory (32-row tiles); thread t sums 2^(x c + bias_r) for key t % 32 over rows t / 32 + 8 i
// that attend to it, and the eight partial sums of a key are added in a
// fixed order.
constexpr int kPrSimtKeys = 32, kPrSimtRowTile = 32, kPrSimtThreads = 256;
__global__ void __launch_bounds__(kPrSimtThreads) k_prompt_colsum_simt(const float* __restrict__ q,
                                                                      const float* __restrict__ k, PromptArgs a,
                                                                      const float* bias, float* a_out) {
  __shared__ float ks[kPrSimtKeys][kD + 1];
  __shared__ float qs[kPrSimtRowTile][kD + 1];
  __shared__ float bs[kPrSimtRowTile];
  __shared__ float part[kPrSimtThreads];
  const int h = blockIdx.y, tid = threadIdx.x, j0 = blockIdx.x * kPrSimtKeys;
  const int kk = tid % kPrSimtKeys, rsub = tid / kPrSimtKeys;
  const int j = j0 + kk;
  const int p_first = a.n - a.nq;
  const float c = kPrLog2e * rsqrtf((float)kD);
  for (int e = tid; e < kPrSimtKeys * kD; e += kPrSimtThreads) {
    const int r = e / kD, d = e % kD;
    ks[r][d] = j0 + r < a.n ? k[((size_t)(j0 + r) * a.hkv + h) * kD + d] : 0.f;
  }
  const int rows = a.nq * a.G;
  const int r_start = j0 <= p_first ? 0 : (j0 - p_first) * a.G;  // rows before it see no key of the tile
  float acc = 0.f;
  for (int r0 = r_start; r0 < rows; r0 += kPrSimtRowTile) {
    __syncthreads();
    for (int e = tid; e < kPrSimtRowTile * kD; e += kPrSimtThreads) {
      const int r = e / kD, d = e % kD, row = r0 + r;
      float v = 0.f;
      if (row < rows) {
        const int prel = row / a.G, gq = row - prel * a.G;
        v = q[((size_t)prel * a.hq + h * a.G + gq) * kD + d];
      }
      qs[r][d] = v;
    }
    for (int r = tid; r < kPrSimtRowTile; r += kPrSimtThreads) {
      const int row = r0 + r;
      float b = -CUDART_INF_F;
      if (row < rows) {
        const int prel = row / a.G, gq = row - prel * a.G;
        b = bias[((size_t)h * a.n_ch + prel / a.p2) * a.crp + (size_t)(prel % a.p2) * a.G + gq];
      }
      bs[r] = b;
    }
    __syncthreads();
    for (int r = rsub; r < kPrSimtRowTile; r += kPrSimtThreads / kPrSimtKeys) {
      const int row = r0 + r;
      if (row >= rows || p_first + row / a.G < j) continue;  // past the rows, or before key j
      float d = 0.f;
#pragma unroll 8
      for (int e = 0; e < kD; ++e) d = fmaf(ks[kk][e], qs[r][e], d);
      acc += exp2f(fmaf(d, c, bs[r]));
    }
  }
  part[tid] = acc;
  __syncthreads();
  if (rsub == 0 && j < a.n) {
    float s = 0.f;
    for (int t = 0; t < kPrSimtThreads / kPrSimtKeys; ++t) s += part[t * kPrSimtKeys + kk];
    if (a.mode == 1) s /= (float)min(a.nq, a.n - j);
    a_out[(size_t)h * a.n + j] = s;
  }
}

// ---- host --------------------------------------------------------------

namespace {

PFN_cuTensorMapEncodeTiled_v12000 prompt_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &qr) ==
            cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// q [nq][hq][128] bf16 as a 3-D tensor (d, query head, position); box 64 x
// G x P with the 128-byte swizzle; positions past nq read as zero.
cudaError_t make_prompt_qmap(CUtensorMap* m, const void* q, int nq, int hq, int G, int P) {
  auto fn = prompt_encode_fn();
  if (!fn) return cudaErrorNotSupported;
  cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)hq, (cuuint64_t)nq};
  cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)hq * kD * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)P};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

PromptArgs prompt_args(int n, int nq, int hq, int hkv, int mode) {
  PromptArgs a;
  a.n = n;
  a.nq = nq;
  a.hq = hq;
  a.hkv = hkv;
  a.G = hq / hkv;
  a.p1 = 128 / a.G;
  a.p2 = 256 / a.G;
  a.n_mt = (nq + a.p1 - 1) / a.p1;
  a.n_ch = (nq + a.p2 - 1) / a.p2;
  a.crp = (a.G * a.p2 + 3) / 4 * 4;
  a.mode = mode;
  return a;
}

}  // namespace

size_t prompt_bias_bytes(int n, int nq, int hq, int hkv) {
  const PromptArgs a = prompt_args(n, nq, hq, hkv, 0);
  return (size_t)hkv * a.n_ch * a.crp * 4;
}

cudaError_t launch_prompt_score(DType dt, const void* q, const void* k, int n, int nq, int hq, int hkv, int mode,
                                float* a_out, float* bias, uint32_t* err, cudaStream_t st) {
  const PromptArgs a = prompt_args(n, nq, hq, hkv, mode);
  if (a.p1 < 1) return cudaErrorNotSupported;
  if (dt == kF32) {
    const size_t nbias = (size_t)hkv * a.n_ch * a.crp;
    const size_t blocks = (nbias + 255) / 256;
    cudaError_t e;
    {
      TimingScope ts("prompt_bias_fill", st);
      k_prompt_bias_fill<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0, st>>>(bias, nbias);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const float* qf = static_cast<const float*>(q);
    const float* kf = static_cast<const float*>(k);
    {
      TimingScope ts("prompt_rowstats_simt", st);
      k_prompt_rowstats_simt<<<dim3((unsigned)(nq * a.G), hkv), kPrSimtRows, 0, st>>>(qf, kf, a, bias);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    TimingScope ts("prompt_colsum_simt", st);
    k_prompt_colsum_simt<<<dim3((unsigned)((n + kPrSimtKeys - 1) / kPrSimtKeys), hkv), kPrSimtThreads, 0, st>>>(
        qf, kf, a, bias, a_out);
    (void)err;
    return cudaGetLastError();
  }
  PromptMaps maps;
  cudaError_t e = make_prompt_qmap(&maps.q1, q, nq, hq, a.G, a.p1);
  if (e == cudaSuccess) e = make_prompt_qmap(&maps.q2, q, nq, hq, a.G, a.p2);
  if (e == cudaSuccess) e = make_row_map(&maps.k1, k, n, hkv, 256);
  if (e == cudaSuccess) e = make_row_map(&maps.k2, k, n, hkv, 128);
  if (e != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(k_prompt_rowstats, cudaFuncAttributeMaxDynamicSharedMemorySize, kP1Smem)) !=
      cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(k_prompt_colsum, cudaFuncAttributeMaxDynamicSharedMemorySize, kP2Smem)) !=
      cudaSuccess)
    return e;
  const size_t nbias = (size_t)hkv * a.n_ch * a.crp;
  {
    TimingScope ts("prompt_bias_fill", st);
    const size_t blocks = (nbias + 255) / 256;
    k_prompt_bias_fill<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0, st>>>(bias, nbias);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  {
    TimingScope ts("prompt_rowstats", st);
    k_prompt_rowstats<<<(unsigned)(a.n_mt * hkv), kPrThreads, kP1Smem, st>>>(maps, a, bias, err);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  TimingScope ts("prompt_colsum", st);
  k_prompt_colsum<<<(unsigned)(((n + 127) / 128) * hkv), kPrThreads, kP2Smem, st>>>(maps, a, bias, a_out, err);
  return cudaGetLastError();
}

}  // namespace stl
