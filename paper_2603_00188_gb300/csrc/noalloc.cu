// stlite_score_noalloc: the window-score call (same kernels as stlite_score)
// for callers that cannot allocate device memory -- e.g. code running inside
// an allocator or memory-pool callback, a host with a fixed, fully reserved
// device budget, or a runtime that forbids cudaMalloc while it owns the
// device -- and therefore cannot provide the usual workspace.  Its scratch
// (the device error word and the per-split row statistics of the two-pass
// softmax) lives in one file-scope device array instead.
#include <mutex>

#include "../../include/stlite.h"
#include "kernels.cuh"

using namespace stl;

namespace {

constexpr size_t kScratchBytes = 2u << 20;  // 2 MiB, held by every device that loads the library
constexpr size_t kErrBytes = 256;           // error word, then the row statistics
constexpr int kMaxDevices = 64;

// Device-side scratch.  In host code this name is only a stand-in for the
// symbol: the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// The resolved address of each device's array, with the context it belongs
// to: the array is part of the library's module, which is loaded into each
// context anew (after cudaDeviceReset, or when another context is current),
// possibly at another address.  A call whose current context differs from
// the cached one resolves the address again.
struct ScratchSlot {
  unsigned long long ctx_id;
  void* addr;
};
std::mutex g_setup_mu;
ScratchSlot g_slot[kMaxDevices] = {};

// Set-up, with the device current: resolve the array's address once per
// device and context (cudaGetSymbolAddress, return code checked).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  unsigned long long ctx = 0;
  if ((e = stl::current_ctx_id(&ctx)) != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(g_setup_mu);
  if (ctx == 0 || !g_slot[dev].addr || g_slot[dev].ctx_id != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // makes the device's primary context current if none was
    if (e != cudaSuccess) return e;
    if ((e = stl::current_ctx_id(&ctx)) != cudaSuccess) return e;
    if (ctx == 0) return cudaErrorDeviceUninitialized;
    g_slot[dev].ctx_id = ctx;
    g_slot[dev].addr = p;
  }
  *out = g_slot[dev].addr;
  return cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace stl {

cudaError_t noalloc_error_word(uint32_t** word) {
  void* base = nullptr;
  cudaError_t e = scratch_address(&base);
  if (e == cudaSuccess) *word = static_cast<uint32_t*>(base);
  return e;
}

}  // namespace stl

extern "C" stlite_status stlite_score_noalloc(const stlite_shape* s, const void* q, const void* k,
                                              float* a_base, void* stream) {
  // the shape limits of stlite_score, then the fixed scratch's capacity, then
  // the pointers: a problem too large for the array is refused whatever the
  // pointers are
  stlite_status status = check_shape(s);
  if (status != STLITE_OK) return status;
  Problem p;
  p.n = s->n_tokens;
  p.hq = s->n_q_heads;
  p.hkv = s->n_kv_heads;
  p.w = s->window;
  p.dtype = s->dtype == STLITE_BF16 ? kBF16 : kF32;
  p.L = 1;
  FrameTable ft = {};
  ft.n_tokens = p.n;
  const WsPlan plan = plan_workspace(p, ft);
  const size_t stats = (size_t)p.hkv * plan.nsplit * p.R() * 8 + (size_t)p.hkv * p.R() * 4;
  if (kErrBytes + stats > kScratchBytes) return STLITE_EUNSUPPORTED;  // beyond the fixed scratch
  if (!q || !k || !a_base) return STLITE_EINVAL;
  if (!aligned16(q) || !aligned16(k) || !aligned16(a_base)) return STLITE_EINVAL;
  void* base = nullptr;
  if (scratch_address(&base) != cudaSuccess) return STLITE_ECUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t* err = static_cast<uint32_t*>(base);
  float2* rowpart = reinterpret_cast<float2*>(static_cast<unsigned char*>(base) + kErrBytes);
  if (cudaMemsetAsync(err, 0, sizeof(uint32_t), st) != cudaSuccess) return STLITE_ECUDA;
  LayerPtrs io = {};
  io.q[0] = q;
  io.k[0] = k;
  const int nsplit = score_nsplit(p);
  const Strided<float2> parts = strided(rowpart, 0);
  const Strided<float> out = strided(a_base, 0);
  cudaError_t e = p.dtype == kBF16 ? launch_score_umma(p, io, parts, nsplit, out, err, st)
                                   : launch_score(p, io, parts, nsplit, out, err, st);
  return e == cudaSuccess ? STLITE_OK : STLITE_ECUDA;
}
