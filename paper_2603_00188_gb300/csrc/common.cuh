// Device-side helpers shared by every ST-Lite kernel (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>

namespace stl {

constexpr int kD = 128;            // head dimension handled by every kernel
constexpr int kMaxFrames = 256;    // frames per sequence
constexpr int kTsgTile = 128;      // historical tokens per TSG row tile

// Device error word bits (first 32-bit word of the workspace).
constexpr uint32_t kErrTimeout = 1u;  // a bounded wait ran out
constexpr uint32_t kErrLaunch = 2u;   // a kernel found its launch configuration unusable

// Bounded waits give up after this many nanoseconds of %globaltimer.
constexpr uint64_t kWaitLimitNs = 1000000000ull;

// Frame layout of one sequence, passed by value (__grid_constant__) so that
// no host-to-device copy is needed.  Frame f owns tokens
// [off[f], off[f] + gh[f]*gw[f]); the last frame is the current frame.
// tile0[f] is the index of the first 128-token TSG row tile of historical
// frame f (tile0[F-1] = total tiles over frames 0..F-2).
struct FrameTable {
  int32_t n_frames;
  int32_t n_tokens;
  int32_t cur_off;   // first token of the current frame (0 if F == 0)
  int32_t cur_len;   // its visual token count (0 if F == 0)
  int32_t off[kMaxFrames];
  int32_t gh[kMaxFrames];
  int32_t gw[kMaxFrames];
  int32_t tile0[kMaxFrames + 1];
  int32_t ctile0[kMaxFrames + 1];  // first 128-token CSS tile of every frame (all frames)
  // Row tiles of the tensor-core TSG pass: per historical frame (tile0), or,
  // when that takes more tiles, 128-token tiles spanning the whole range
  // [tsg_off, tsg_end) of the historical frames, text tokens included (their
  // rho slices are never read).
  int32_t tsg_tiles;
  int32_t tsg_span;  // 1: spanning tiles
  int32_t tsg_off, tsg_end;
};

// Frame holding token j, or -1 for a text token (binary search on offsets).
__device__ __forceinline__ int find_frame(const FrameTable& ft, int j) {
  int lo = 0, hi = ft.n_frames - 1, f = -1;
  while (lo <= hi) {
    int mid = (lo + hi) >> 1;
    if (ft.off[mid] <= j) {
      f = mid;
      lo = mid + 1;
    } else {
      hi = mid - 1;
    }
  }
  if (f >= 0 && j < ft.off[f] + ft.gh[f] * ft.gw[f]) return f;
  return -1;
}

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  // 4 consecutive elements starting at p (16-byte aligned)
  static __device__ __forceinline__ float4 load4(const float* p) {
    return __ldg(reinterpret_cast<const float4*>(p));
  }
  static __device__ __forceinline__ float load1(const float* p) { return __ldg(p); }
};
template <>
struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float4 load4(const __nv_bfloat16* p) {
    uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
    float4 r;
    r.x = __uint_as_float(u.x << 16);
    r.y = __uint_as_float(u.x & 0xffff0000u);
    r.z = __uint_as_float(u.y << 16);
    r.w = __uint_as_float(u.y & 0xffff0000u);
    return r;
  }
  static __device__ __forceinline__ float load1(const __nv_bfloat16* p) {
    return __bfloat162float(p[0]);
  }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float dot4(float4 a, float4 b) {
  return fmaf(a.x, b.x, fmaf(a.y, b.y, fmaf(a.z, b.z, a.w * b.w)));
}

// Order-preserving map float -> uint32 (ascending keys = ascending floats).
// -0.0 is folded onto +0.0 first so that the two compare equal, as they do
// as numbers.
__device__ __forceinline__ uint32_t float_key(float x) {
  uint32_t u = __float_as_uint(x + 0.0f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t k) {
  uint32_t u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
  return __uint_as_float(u);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void record_error(uint32_t* err, uint32_t bits) {
  if (err) atomicOr(err, bits);
}

}  // namespace stl
