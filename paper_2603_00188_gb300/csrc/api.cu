// C ABI of libstlite.so: argument validation, workspace planning and the
// launch sequence of each entry point.  Declarations and the contract of
// every call are in include/stlite.h.
#include <math.h>
#include <string.h>

#include <atomic>
#include <cmath>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/stlite.h"
#include "kernels.cuh"

using namespace stl;

namespace {

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

stlite_status build_frames(const stlite_shape* s, const stlite_frames* fr, FrameTable* ft) {
  memset(ft, 0, sizeof(*ft));
  ft->n_tokens = s->n_tokens;
  if (!fr) return STLITE_EINVAL;
  const int F = fr->n_frames;
  if (F < 0) return STLITE_EINVAL;
  if (F > STLITE_MAX_FRAMES) return STLITE_EUNSUPPORTED;
  if (F > 0 && (!fr->offset || !fr->grid_h || !fr->grid_w)) return STLITE_EINVAL;
  long long prev_end = 0;
  for (int f = 0; f < F; ++f) {
    const long long off = fr->offset[f], gh = fr->grid_h[f], gw = fr->grid_w[f];
    if (off < 0 || gh < 1 || gw < 1) return STLITE_EINVAL;
    if (off < prev_end) return STLITE_EINVAL;  // sorted and disjoint
    if (off + gh * gw > s->n_tokens) return STLITE_EINVAL;
    prev_end = off + gh * gw;
    ft->off[f] = (int32_t)off;
    ft->gh[f] = (int32_t)gh;
    ft->gw[f] = (int32_t)gw;
  }
  ft->n_frames = F;
  ft->tile0[0] = 0;
  for (int f = 0; f + 1 < F; ++f)
    ft->tile0[f + 1] = ft->tile0[f] + (ft->gh[f] * ft->gw[f] + kTsgTile - 1) / kTsgTile;
  ft->ctile0[0] = 0;
  for (int f = 0; f < F; ++f)
    ft->ctile0[f + 1] = ft->ctile0[f] + (ft->gh[f] * ft->gw[f] + kTsgTile - 1) / kTsgTile;
  if (F > 0) {
    ft->cur_off = ft->off[F - 1];
    ft->cur_len = ft->gh[F - 1] * ft->gw[F - 1];
  }
  if (F >= 2) {
    // ragged frames waste the rows of each frame's last tile; spanning tiles
    // waste the text rows between frames instead: take the fewer tiles
    ft->tsg_off = ft->off[0];
    ft->tsg_end = ft->off[F - 2] + ft->gh[F - 2] * ft->gw[F - 2];
    const int span = (ft->tsg_end - ft->tsg_off + kTsgTile - 1) / kTsgTile;
    ft->tsg_span = span < ft->tile0[F - 1] ? 1 : 0;
    ft->tsg_tiles = ft->tsg_span ? span : ft->tile0[F - 1];
  }
  return STLITE_OK;
}

stlite_status check_params(const stlite_params* pr) {
  if (!pr) return STLITE_EINVAL;
  if (pr->k_override < 0) return STLITE_EINVAL;
  if (pr->k_override == 0 && !(pr->beta > 0.0 && pr->beta <= 1.0)) return STLITE_EINVAL;
  if (!(pr->alpha >= 0.f) || !isfinite(pr->alpha)) return STLITE_EINVAL;
  if (pr->tsg_metric < STLITE_TSG_COSINE || pr->tsg_metric > STLITE_TSG_NEG_L2) return STLITE_EINVAL;
  if (pr->tsg_fixed != 0 && pr->tsg_fixed != 1) return STLITE_EINVAL;
  if (pr->tsg_fixed && !isfinite(pr->tsg_fixed_tau)) return STLITE_EINVAL;
  if (pr->base_scorer != STLITE_BASE_WINDOW && pr->base_scorer != STLITE_BASE_UNIFORM) return STLITE_EINVAL;
  if (pr->abase_norm != STLITE_ABASE_RAW && pr->abase_norm != STLITE_ABASE_MAX) return STLITE_EINVAL;
  if (pr->css_size != 0 && pr->css_size != 3 && pr->css_size != 5 && pr->css_size != 7 && pr->css_size != 9)
    return STLITE_EINVAL;
  return STLITE_OK;
}

Problem to_problem(const stlite_shape* s, int L) {
  Problem p;
  p.n = s->n_tokens;
  p.hq = s->n_q_heads;
  p.hkv = s->n_kv_heads;
  p.w = s->window;
  p.dtype = s->dtype == STLITE_BF16 ? kBF16 : kF32;
  p.L = L;
  return p;
}

bool use_tensor_cores(const Problem& p) { return p.dtype == kBF16; }

stlite_status cuda_status(cudaError_t e) { return e == cudaSuccess ? STLITE_OK : STLITE_ECUDA; }

}  // namespace

namespace stl {

// Shape checks shared by every entry point (the kernels' index arithmetic
// relies on these limits).
stlite_status check_shape(const stlite_shape* s) {
  if (!s) return STLITE_EINVAL;
  if (s->n_tokens < 1 || s->n_q_heads < 1 || s->n_kv_heads < 1 || s->window < 1 ||
      s->head_dim < 1)
    return STLITE_EINVAL;
  if (s->n_q_heads % s->n_kv_heads != 0) return STLITE_EINVAL;
  if (s->dtype != STLITE_BF16 && s->dtype != STLITE_F32) return STLITE_EINVAL;
  if (s->head_dim != STLITE_HEAD_DIM) return STLITE_EUNSUPPORTED;
  if (s->window > 256) return STLITE_EUNSUPPORTED;
  const long long R = (long long)s->window * (s->n_q_heads / s->n_kv_heads);
  if (R > 512) return STLITE_EUNSUPPORTED;
  if ((long long)s->n_tokens * s->n_kv_heads > (1LL << 30)) return STLITE_EUNSUPPORTED;
  if (s->n_tokens > select_max_tokens()) return STLITE_EUNSUPPORTED;
  if (s->n_kv_heads > 4096) return STLITE_EUNSUPPORTED;
  return STLITE_OK;
}

// One layer's workspace region; regions of consecutive layers follow each
// other.  Every buffer is 256-byte aligned.
WsPlan plan_workspace(const Problem& p, const FrameTable& ft) {
  WsPlan w;
  const size_t hn = (size_t)p.hkv * p.n;
  w.nsplit = score_nsplit_max(p);
  w.nchunk = use_tensor_cores(p) && ft.n_frames >= 2 ? (ft.cur_len + 255) / 256 : 1;
  if (w.nchunk < 1) w.nchunk = 1;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  w.cur_pad = ft.n_frames > 0 ? (ft.cur_len + 3) / 4 * 4 : 4;
  w.err = take(4);
  w.rn = take(hn * 4);
  w.rn_cur = take((size_t)p.hkv * w.cur_pad * 4);
  w.rowpart = take((size_t)p.hkv * w.nsplit * p.R() * 8 + (size_t)p.hkv * p.R() * 4);
  w.a_base = take(hn * 4);
  w.phi = take(hn * 4);
  w.rho = take(hn * 4);
  w.rho_part = take((size_t)w.nchunk * hn * 4);
  w.tau = take((size_t)p.hkv * 4);
  w.gate = take(hn);
  w.score = take(hn * 4);
  w.dots = take(4 * hn * 4);
  w.total = o;
  return w;
}

// The second stream of a call and its events: fork, join, CSS dots done
// (see aux_stream).
struct AuxStream {
  unsigned long long ctx_id;
  cudaStream_t s;
  cudaEvent_t ev[3];
};
AuxStream* aux_stream(cudaStream_t st);

// ---- per-kernel timing ----------------------------------------------------
namespace {
struct TimingRecord {
  const char* name;
  cudaEvent_t start, stop;
};
std::atomic<int> g_timing_on{0};
std::mutex g_timing_mu;
std::vector<TimingRecord> g_records;
std::vector<cudaEvent_t> g_event_pool;

cudaEvent_t take_event() {
  {
    std::lock_guard<std::mutex> lk(g_timing_mu);
    if (!g_event_pool.empty()) {
      cudaEvent_t e = g_event_pool.back();
      g_event_pool.pop_back();
      return e;
    }
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

bool stream_capturing(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  return cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs != cudaStreamCaptureStatusNone;
}
}  // namespace

TimingScope::TimingScope(const char* name, cudaStream_t st) : name_(name), st_(st), start_(nullptr) {
  if (!g_timing_on.load(std::memory_order_relaxed) || stream_capturing(st)) return;
  start_ = take_event();
  if (start_ && cudaEventRecord(start_, st_) != cudaSuccess) start_ = nullptr;
}

TimingScope::~TimingScope() {
  if (!start_) return;
  cudaEvent_t stop = take_event();
  if (!stop || cudaEventRecord(stop, st_) != cudaSuccess) return;
  std::lock_guard<std::mutex> lk(g_timing_mu);
  g_records.push_back({name_, start_, stop});
}

namespace {
// cuCtxGetCurrent and cuCtxGetId through the runtime's driver entry points
// (no link against the driver library).
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

bool driver_fns(CtxGetCurrentFn* get_current, CtxGetIdFn* get_id) {
  static CtxGetCurrentFn cur = nullptr;
  static CtxGetIdFn id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      cur = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      id = reinterpret_cast<CtxGetIdFn>(p);
  });
  *get_current = cur;
  *get_id = id;
  return cur && id;
}
}  // namespace

cudaError_t current_ctx_id(unsigned long long* out) {
  CtxGetCurrentFn get_current;
  CtxGetIdFn get_id;
  if (!driver_fns(&get_current, &get_id)) return cudaErrorNotSupported;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  *out = 0;
  if (ctx && get_id(ctx, out) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  return cudaSuccess;
}

// ---- a second stream for the independent stages of one call ----------------
// The window score (step 1) does not depend on CSS and TSG (steps 2-3), nor
// TSG on CSS's Phi: a call runs the score and Phi on a second stream, forked
// from and joined back into the caller's with events, so that SMs that one
// chain's last wave leaves idle take the other chain's work.  The second
// stream and its events belong to the calling host thread and device (a
// thread enqueues its calls in order, so one set of events serves them all);
// they are made outside graph capture only, and again when the device's
// context has changed (the old handles went with the old context).  While
// per-kernel timing is on, every launch stays on the caller's stream, so
// that each kernel is timed alone.
namespace {
constexpr int kMaxAuxDevices = 64;
// The calling thread's second streams, one per device.  When the thread
// exits, the one of the device then current is released if the context it
// was made in is still current there (a stream with work still queued is
// released by CUDA once that work is done).  Nothing here makes a device or
// context current: after a reset that would create a context only to find
// the handles gone.
struct AuxSlots {
  AuxStream slot[kMaxAuxDevices] = {};
  ~AuxSlots() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxAuxDevices) return;
    AuxStream& x = slot[dev];
    unsigned long long ctx = 0;
    if (!x.s || current_ctx_id(&ctx) != cudaSuccess || ctx != x.ctx_id) return;
    for (cudaEvent_t e : x.ev)
      if (e) cudaEventDestroy(e);
    cudaStreamDestroy(x.s);
    (void)cudaGetLastError();
  }
};
thread_local AuxSlots t_aux;
}  // namespace

AuxStream* aux_stream(cudaStream_t st) {
  if (g_timing_on.load(std::memory_order_relaxed)) return nullptr;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxAuxDevices) return nullptr;
  unsigned long long ctx = 0;
  if (current_ctx_id(&ctx) != cudaSuccess || ctx == 0) return nullptr;
  AuxStream& x = t_aux.slot[dev];
  if (x.s && x.ctx_id == ctx) return &x;
  if (stream_capturing(st)) return nullptr;
  AuxStream n = {};
  n.ctx_id = ctx;
  bool ok = cudaStreamCreateWithFlags(&n.s, cudaStreamNonBlocking) == cudaSuccess;
  for (int i = 0; ok && i < 3; ++i) ok = cudaEventCreateWithFlags(&n.ev[i], cudaEventDisableTiming) == cudaSuccess;
  if (!ok) {
    for (int i = 0; i < 3; ++i)
      if (n.ev[i]) cudaEventDestroy(n.ev[i]);
    if (n.s) cudaStreamDestroy(n.s);
    (void)cudaGetLastError();
    return nullptr;
  }
  x = n;
  return &x;
}

}  // namespace stl

namespace {

// One launch context: a batch of L (<= kMaxLayers) layers whose workspace
// regions start at `ws`.
struct Ctx {
  Problem p;
  FrameTable ft;
  WsPlan plan;
  uint8_t* ws;
  uint32_t* err;
  cudaStream_t st;
  template <typename T>
  Strided<T> view(size_t off) const {
    return strided(reinterpret_cast<T*>(ws + off), plan.total);
  }
};

stlite_status prepare(const stlite_shape* shape, const stlite_frames* frames, void* ws, size_t ws_bytes,
                      int n_layers, void* stream, Ctx* c) {
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  stlite_frames none = {0, nullptr, nullptr, nullptr};
  if ((s = build_frames(shape, frames ? frames : &none, &c->ft)) != STLITE_OK) return s;
  c->p = to_problem(shape, 1);
  c->plan = plan_workspace(c->p, c->ft);
  if (!ws || !aligned16(ws)) return STLITE_EINVAL;
  if (ws_bytes / (size_t)n_layers < c->plan.total) return STLITE_EWORKSPACE;
  c->ws = static_cast<uint8_t*>(ws);
  c->err = reinterpret_cast<uint32_t*>(c->ws + c->plan.err);
  c->st = static_cast<cudaStream_t>(stream);
  return STLITE_OK;
}

LayerPtrs single_layer(const void* q, const void* k, const void* v, void* ko, void* vo, int32_t* idx) {
  LayerPtrs io;
  memset(&io, 0, sizeof(io));
  io.q[0] = q;
  io.k[0] = k;
  io.v[0] = v;
  io.k_out[0] = ko;
  io.v_out[0] = vo;
  io.idx[0] = idx;
  return io;
}

template <typename T>
Strided<T> one(T* p) {
  return strided(p, 0);
}

// CSS (Eqs. 4-5) into phi, plus the inverse key norms rn / rn_cur that TSG
// uses.  bf16 caches whose grids are at most 127 wide take the tensor-core
// kernel; otherwise the CUDA-core one.
// size: the CSS neighbourhood (0 or 3 = the method's 3x3; 5, 7, 9 = the
// size ablation, on the box-sum kernel).
// defer_phi: the tensor-core CSS leaves Phi to a later run_css_phi and sets
// *deferred (the other kernels produce Phi themselves).
cudaError_t run_css(const Ctx& c, const LayerPtrs& io, Strided<float> phi, int size = 3, bool defer_phi = false,
                    bool* deferred = nullptr) {
  Strided<float> rn = c.view<float>(c.plan.rn), rc = c.view<float>(c.plan.rn_cur);
  if (deferred) *deferred = false;
  if (size > 3) return launch_css_box(c.p, c.ft, io, size, phi, rn, rc, c.plan.cur_pad, c.st);
  if (use_tensor_cores(c.p) && css_umma_supported(c.ft)) {
    if (defer_phi && deferred) *deferred = true;
    const size_t hn4 = (size_t)c.p.hkv * c.p.n * 4;
    Strided<float> dE = c.view<float>(c.plan.dots), dS = c.view<float>(c.plan.dots + hn4);
    Strided<float> dSE = c.view<float>(c.plan.dots + 2 * hn4), dSW = c.view<float>(c.plan.dots + 3 * hn4);
    return launch_css_umma(c.p, c.ft, io, phi, rn, rc, c.plan.cur_pad, dE, dS, dSE, dSW, c.err, c.st,
                           !(defer_phi && deferred));
  }
  return launch_css(c.p, c.ft, io, phi, rn, rc, c.plan.cur_pad, c.st);
}

// Phi of a deferred tensor-core CSS (its dots written), on stream st.
cudaError_t run_css_phi(const Ctx& c, Strided<float> phi, cudaStream_t st) {
  const size_t hn4 = (size_t)c.p.hkv * c.p.n * 4;
  return launch_css_phi(c.p, c.ft, phi, c.view<float>(c.plan.rn), c.view<float>(c.plan.rn_cur), c.plan.cur_pad,
                        c.view<float>(c.plan.dots), c.view<float>(c.plan.dots + hn4),
                        c.view<float>(c.plan.dots + 2 * hn4), c.view<float>(c.plan.dots + 3 * hn4), st);
}

// The inverse norms alone: from the CSS kernel when that is the tensor-core
// one (so that every path sees the same bits), else from the norms kernel
// (whose arithmetic matches the CUDA-core CSS kernel's).
cudaError_t run_norms(const Ctx& c, const LayerPtrs& io) {
  if (use_tensor_cores(c.p) && css_umma_supported(c.ft)) return run_css(c, io, c.view<float>(c.plan.phi));
  return launch_inv_norms(c.p, c.ft, io, c.view<float>(c.plan.rn), c.view<float>(c.plan.rn_cur), c.plan.cur_pad,
                          c.st);
}

cudaError_t run_score(const Ctx& c, const LayerPtrs& io, Strided<float> a_base) {
  Strided<float2> rp = c.view<float2>(c.plan.rowpart);
  const int ns = score_nsplit(c.p);
  if (use_tensor_cores(c.p)) return launch_score_umma(c.p, io, rp, ns, a_base, c.err, c.st);
  return launch_score(c.p, io, rp, ns, a_base, c.err, c.st);
}

cudaError_t run_tsg(const Ctx& c, const LayerPtrs& io, int metric) {
  Strided<const float> rn = c.view<const float>(c.plan.rn);
  Strided<float> rp = c.view<float>(c.plan.rho_part);
  if (use_tensor_cores(c.p))
    return launch_tsg_umma(c.p, c.ft, io, c.view<const float>(c.plan.rn_cur), c.plan.cur_pad, rp, metric, c.err,
                           c.st);
  return launch_tsg(c.p, c.ft, io, rn, rp, metric, c.err, c.st);
}

// The ablation fields of the parameters, for the selection kernel.
void select_variants(SelectArgs& a, const stlite_params* params, const Problem& p) {
  a.tsg_metric = params->tsg_metric;
  a.tsg_fixed = params->tsg_fixed;
  a.tsg_fixed_tau = params->tsg_fixed_tau;
  a.base_uniform = params->base_scorer == STLITE_BASE_UNIFORM ? 1 : 0;
  a.a_uniform = (float)p.w / (float)p.n;  // the window score's total, spread evenly
  a.a_norm_max = params->abase_norm == STLITE_ABASE_MAX ? 1 : 0;
}

// Algorithm 1 for a batch of layers (steps 1-5), every stage one launch.
// Layer l keeps io.budget[l] tokens per KV head.  With a second stream
// (aux_stream), step 1 runs on it beside steps 2-3: CSS and TSG are enqueued
// first, so that they take the SMs first and the window score fills those
// their last waves leave idle (the other order measured slower).  TSG needs
// CSS's inverse norms but not Phi, so with the tensor-core CSS its second
// kernel (Phi from the dots) goes last on the second stream, after an event
// that marks the dots done: TSG starts as soon as the dots are written.
stlite_status compress_batch(const Ctx& c, const stlite_params* params, const LayerPtrs& io) {
  const bool tsg = params->tsg_enable && c.ft.n_frames >= 2;
  const bool window = params->base_scorer == STLITE_BASE_WINDOW;
  Strided<float> a_base = c.view<float>(c.plan.a_base);
  Strided<float> phi = c.view<float>(c.plan.phi);
  AuxStream* x = window && (params->css_enable || tsg) ? aux_stream(c.st) : nullptr;
  cudaError_t e = cudaSuccess;
  if (x) {
    e = cudaEventRecord(x->ev[0], c.st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(x->s, x->ev[0], 0);
  }
  // CSS also produces the inverse key norms TSG needs; without CSS a plain
  // norms pass provides them.
  bool late_phi = false;
  if (e == cudaSuccess && params->css_enable) {
    e = run_css(c, io, phi, params->css_size, x != nullptr, &late_phi);
    if (e == cudaSuccess && late_phi) e = cudaEventRecord(x->ev[2], c.st);
  } else if (e == cudaSuccess && tsg) {
    e = run_norms(c, io);
  }
  if (e == cudaSuccess && tsg) e = run_tsg(c, io, params->tsg_metric);
  if (e == cudaSuccess && window) {
    Ctx cs = c;
    if (x) cs.st = x->s;
    e = run_score(cs, io, a_base);
  }
  if (e == cudaSuccess && late_phi) {
    e = cudaStreamWaitEvent(x->s, x->ev[2], 0);
    if (e == cudaSuccess) e = run_css_phi(c, phi, x->s);
  }
  if (e == cudaSuccess && x) e = cudaEventRecord(x->ev[1], x->s);
  if (e == cudaSuccess && x) e = cudaStreamWaitEvent(c.st, x->ev[1], 0);
  if (e != cudaSuccess) return STLITE_ECUDA;
  SelectArgs a = {};
  a.mode = (tsg ? kSelGate : 0) | kSelTopk;
  for (int l = 0; l < c.p.L; ++l) a.budget[l] = io.budget[l];
  a.nchunk = c.plan.nchunk;
  a.tsg_enable = tsg ? 1 : 0;
  a.css_enable = params->css_enable ? 1 : 0;
  a.alpha = params->alpha;
  select_variants(a, params, c.p);
  a.rho_part = c.view<const float>(c.plan.rho_part);
  a.rn = c.view<const float>(c.plan.rn);
  a.rho = c.view<float>(c.plan.rho);
  a.tau = c.view<float>(c.plan.tau);
  a.gate = tsg ? c.view<uint8_t>(c.plan.gate) : strided<uint8_t>(nullptr, 0);
  a.a_base = c.view<const float>(c.plan.a_base);
  a.phi = params->css_enable ? c.view<const float>(c.plan.phi) : strided<const float>(nullptr, 0);
  a.score = c.view<float>(c.plan.score);
  a.write_stages = 0;  // rho, gate and S stay on chip: only the indices leave
  for (int l = 0; l < c.p.L; ++l) a.idx[l] = io.idx[l];
  if ((e = launch_select(c.p, c.ft, a, c.st)) != cudaSuccess) return STLITE_ECUDA;
  return cuda_status(launch_gather(c.p, io, c.st));
}

}  // namespace

extern "C" {

int32_t stlite_budget(int32_t n_tokens, double beta, int32_t k_override) {
  if (n_tokens < 1) return -1;
  if (k_override > 0) return k_override < n_tokens ? k_override : n_tokens;
  if (!(beta > 0.0 && beta <= 1.0)) return -1;
  long long b = (long long)floor(beta * (double)n_tokens + 1e-9);
  if (b < 1) b = 1;
  if (b > n_tokens) b = n_tokens;
  return (int32_t)b;
}

stlite_status stlite_workspace_size(const stlite_shape* shape, const stlite_frames* frames,
                                    const stlite_params* params, size_t* bytes) {
  if (!bytes) return STLITE_EINVAL;
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  if (params && (s = check_params(params)) != STLITE_OK) return s;
  stlite_frames none = {0, nullptr, nullptr, nullptr};
  FrameTable ft;
  if ((s = build_frames(shape, frames ? frames : &none, &ft)) != STLITE_OK) return s;
  *bytes = plan_workspace(to_problem(shape, 1), ft).total;
  return STLITE_OK;
}

stlite_status stlite_score(const stlite_shape* shape, const void* q, const void* k, float* a_base,
                           void* ws, size_t ws_bytes, void* stream) {
  Ctx c;
  stlite_status s = prepare(shape, nullptr, ws, ws_bytes, 1, stream, &c);
  if (s != STLITE_OK) return s;
  if (!q || !k || !a_base || !aligned16(q) || !aligned16(k) || !aligned16(a_base)) return STLITE_EINVAL;
  return cuda_status(run_score(c, single_layer(q, k, nullptr, nullptr, nullptr, nullptr), one(a_base)));
}

stlite_status stlite_gate_frames(const stlite_shape* shape, const stlite_frames* frames,
                                 const void* k, int32_t budget, float* rho, float* tau,
                                 uint8_t* gate, void* ws, size_t ws_bytes, void* stream) {
  Ctx c;
  stlite_status s = prepare(shape, frames, ws, ws_bytes, 1, stream, &c);
  if (s != STLITE_OK) return s;
  if (!k || !rho || !tau || !gate || !aligned16(k) || !aligned16(rho) || !aligned16(tau) ||
      !aligned16(gate))
    return STLITE_EINVAL;
  if (budget < 1 || budget > c.p.n) return STLITE_EINVAL;
  const LayerPtrs io = single_layer(nullptr, k, nullptr, nullptr, nullptr, nullptr);
  cudaError_t e = run_norms(c, io);
  if (e == cudaSuccess) e = run_tsg(c, io, kTsgCosine);
  if (e != cudaSuccess) return STLITE_ECUDA;
  SelectArgs a = {};
  a.mode = kSelGate;
  a.budget[0] = budget;
  a.nchunk = c.plan.nchunk;
  a.tsg_enable = 1;
  a.rho_part = c.view<const float>(c.plan.rho_part);
  a.rn = c.view<const float>(c.plan.rn);
  a.rho = one(rho);
  a.tau = one(tau);
  a.gate = one(gate);
  a.write_stages = 1;
  return cuda_status(launch_select(c.p, c.ft, a, c.st));
}

stlite_status stlite_spatial_saliency(const stlite_shape* shape, const stlite_frames* frames,
                                      const void* k, float* phi, void* ws, size_t ws_bytes,
                                      void* stream) {
  Ctx c;
  stlite_status s = prepare(shape, frames, ws, ws_bytes, 1, stream, &c);
  if (s != STLITE_OK) return s;
  if (!k || !phi || !aligned16(k) || !aligned16(phi)) return STLITE_EINVAL;
  const LayerPtrs io = single_layer(nullptr, k, nullptr, nullptr, nullptr, nullptr);
  cudaError_t e = run_css(c, io, one(phi));
  if (e == cudaSuccess) e = launch_fill_text_nan(c.p, c.ft, phi, c.st);
  return cuda_status(e);
}

stlite_status stlite_spatial_saliency_size(const stlite_shape* shape, const stlite_frames* frames,
                                           const void* k, int32_t size, float* phi, void* ws, size_t ws_bytes,
                                           void* stream) {
  if (size != 3 && size != 5 && size != 7 && size != 9) return STLITE_EINVAL;
  Ctx c;
  stlite_status s = prepare(shape, frames, ws, ws_bytes, 1, stream, &c);
  if (s != STLITE_OK) return s;
  if (!k || !phi || !aligned16(k) || !aligned16(phi)) return STLITE_EINVAL;
  const LayerPtrs io = single_layer(nullptr, k, nullptr, nullptr, nullptr, nullptr);
  cudaError_t e = launch_css_box(c.p, c.ft, io, size, one(phi), c.view<float>(c.plan.rn),
                                 c.view<float>(c.plan.rn_cur), c.plan.cur_pad, c.st);
  if (e == cudaSuccess) e = launch_fill_text_nan(c.p, c.ft, phi, c.st);
  return cuda_status(e);
}

stlite_status stlite_select_topk(const stlite_shape* shape, const stlite_frames* frames,
                                 const stlite_params* params, const float* a_base,
                                 const float* phi, const uint8_t* gate, int32_t budget,
                                 int32_t* idx, float* score_out, void* ws, size_t ws_bytes,
                                 void* stream) {
  Ctx c;
  stlite_status s = prepare(shape, frames, ws, ws_bytes, 1, stream, &c);
  if (s != STLITE_OK) return s;
  if ((s = check_params(params)) != STLITE_OK) return s;
  const bool uniform = params->base_scorer == STLITE_BASE_UNIFORM;
  if ((!uniform && !a_base) || (a_base && !aligned16(a_base)) || !idx || !aligned16(idx)) return STLITE_EINVAL;
  if (params->css_enable && (!phi || !aligned16(phi))) return STLITE_EINVAL;
  if ((gate && !aligned16(gate)) || (score_out && !aligned16(score_out))) return STLITE_EINVAL;
  if (budget < 1 || budget > c.p.n) return STLITE_EINVAL;
  SelectArgs a = {};
  a.mode = kSelTopk;
  a.budget[0] = budget;
  a.css_enable = params->css_enable ? 1 : 0;
  a.alpha = params->alpha;
  select_variants(a, params, c.p);
  a.a_base = one(a_base);
  a.phi = params->css_enable ? one(phi) : strided<const float>(nullptr, 0);
  a.gate = one(const_cast<uint8_t*>(gate));
  a.score = score_out ? one(score_out) : c.view<float>(c.plan.score);
  a.idx[0] = idx;
  a.write_stages = 1;
  return cuda_status(launch_select(c.p, c.ft, a, c.st));
}

stlite_status stlite_compact(const stlite_shape* shape, int32_t budget, const int32_t* idx,
                             const void* k, const void* v, void* k_out, void* v_out,
                             void* stream) {
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  if (!idx || !k || !v || !k_out || !v_out) return STLITE_EINVAL;
  if (!aligned16(idx) || !aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out))
    return STLITE_EINVAL;
  if (budget < 1 || budget > shape->n_tokens) return STLITE_EINVAL;
  const Problem p = to_problem(shape, 1);
  LayerPtrs io = single_layer(nullptr, k, v, k_out, v_out, const_cast<int32_t*>(idx));
  io.budget[0] = budget;
  return cuda_status(launch_gather(p, io, static_cast<cudaStream_t>(stream)));
}

stlite_status stlite_compress_layer(const stlite_shape* shape, const stlite_frames* frames,
                                    const stlite_params* params, const void* q, const void* k,
                                    const void* v, void* k_out, void* v_out, int32_t* idx_out,
                                    int32_t* budget_out, void* ws, size_t ws_bytes,
                                    void* stream) {
  stlite_layer_io io = {q, k, v, k_out, v_out, idx_out};
  return stlite_compress_layers(shape, frames, params, 1, &io, budget_out, ws, ws_bytes, stream);
}

}  // extern "C"

namespace {

// Algorithm 1 over n_layers layers, layer l keeping budgets[l] tokens per
// KV head; every budget is checked before anything is enqueued.  The pointer
// checks are skipped for a packed batch's per-sequence offsets (their bases
// were checked; an index block there starts on a 4-byte boundary, which the
// kernels' scalar index accesses need).
stlite_status compress_layers_impl(const stlite_shape* shape, const stlite_frames* frames,
                                   const stlite_params* params, int32_t n_layers,
                                   const stlite_layer_io* layers, const int32_t* budgets, void* ws,
                                   size_t ws_bytes, void* stream, bool check_pointers = true) {
  Ctx c;
  stlite_status s = prepare(shape, frames, ws, ws_bytes, n_layers, stream, &c);
  if (s != STLITE_OK) return s;
  for (int l = 0; l < n_layers; ++l) {
    const stlite_layer_io& x = layers[l];
    if (check_pointers) {
      if (!x.q || !x.k || !x.v || !x.k_out || !x.v_out || !x.idx_out) return STLITE_EINVAL;
      if (!aligned16(x.q) || !aligned16(x.k) || !aligned16(x.v) || !aligned16(x.k_out) ||
          !aligned16(x.v_out) || !aligned16(x.idx_out))
        return STLITE_EINVAL;
    }
    if (budgets[l] < 1 || budgets[l] > c.p.n) return STLITE_EINVAL;
  }
  // one launch per stage for up to kMaxLayers layers at a time
  for (int l0 = 0; l0 < n_layers; l0 += kMaxLayers) {
    const int L = n_layers - l0 < kMaxLayers ? n_layers - l0 : kMaxLayers;
    Ctx cb = c;
    cb.p.L = L;
    cb.ws = c.ws + (size_t)l0 * c.plan.total;
    LayerPtrs io;
    memset(&io, 0, sizeof(io));
    for (int l = 0; l < L; ++l) {
      const stlite_layer_io& x = layers[l0 + l];
      io.q[l] = x.q;
      io.k[l] = x.k;
      io.v[l] = x.v;
      io.k_out[l] = x.k_out;
      io.v_out[l] = x.v_out;
      io.idx[l] = x.idx_out;
      io.budget[l] = budgets[l0 + l];
    }
    if ((s = compress_batch(cb, params, io)) != STLITE_OK) return s;
  }
  return STLITE_OK;
}

}  // namespace

extern "C" {

stlite_status stlite_compress_layers(const stlite_shape* shape, const stlite_frames* frames,
                                     const stlite_params* params, int32_t n_layers,
                                     const stlite_layer_io* layers, int32_t* budget_out, void* ws,
                                     size_t ws_bytes, void* stream) {
  if (n_layers < 1 || !layers || !shape) return STLITE_EINVAL;
  stlite_status s = check_params(params);
  if (s != STLITE_OK) return s;
  const int32_t budget = stlite_budget(shape->n_tokens, params->beta, params->k_override);
  if (budget < 1) return STLITE_EINVAL;
  std::vector<int32_t> budgets((size_t)n_layers, budget);
  s = compress_layers_impl(shape, frames, params, n_layers, layers, budgets.data(), ws, ws_bytes, stream);
  if (s == STLITE_OK && budget_out) *budget_out = budget;
  return s;
}

stlite_status stlite_compress_layers_budgets(const stlite_shape* shape, const stlite_frames* frames,
                                             const stlite_params* params, int32_t n_layers,
                                             const stlite_layer_io* layers, const int32_t* budgets,
                                             void* ws, size_t ws_bytes, void* stream) {
  if (n_layers < 1 || !layers || !budgets || !shape) return STLITE_EINVAL;
  stlite_status s = check_params(params);
  if (s != STLITE_OK) return s;
  return compress_layers_impl(shape, frames, params, n_layers, layers, budgets, ws, ws_bytes, stream);
}

stlite_status stlite_hierarchical_budgets(int32_t n_layers, const double* layer_mass, int64_t total_budget,
                                          int32_t n_tokens, int32_t* budgets) {
  if (n_layers < 1 || !layer_mass || !budgets || n_tokens < 1) return STLITE_EINVAL;
  if (total_budget < n_layers || total_budget > (int64_t)n_layers * n_tokens) return STLITE_EINVAL;
  double sum = 0.0;
  for (int l = 0; l < n_layers; ++l) {
    if (!(layer_mass[l] > 0.0) || !std::isfinite(layer_mass[l])) return STLITE_EINVAL;
    sum += layer_mass[l];
  }
  if (!std::isfinite(sum)) return STLITE_EINVAL;
  // B(l) = S(l) / sum S * B_total made integer: the budgets in [1, N] adding
  // up to B_total nearest to the real shares in squared distance.  The
  // problem is separable and convex, so one-token greedy steps from
  // clamp(floor(share)) reach the minimiser: add where share - b is largest
  // (room left), or take where b - share is largest (b > 1); ties go to the
  // lower layer.
  std::vector<double> share((size_t)n_layers);
  std::vector<int64_t> b((size_t)n_layers);
  int64_t given = 0;
  for (int l = 0; l < n_layers; ++l) {
    share[l] = layer_mass[l] / sum * (double)total_budget;
    const double f = floor(share[l]);
    b[l] = f < 1.0 ? 1 : f > (double)n_tokens ? n_tokens : (int64_t)f;
    given += b[l];
  }
  for (; given < total_budget; ++given) {
    int best = -1;
    for (int l = 0; l < n_layers; ++l)
      if (b[l] < n_tokens && (best < 0 || share[l] - (double)b[l] > share[best] - (double)b[best])) best = l;
    ++b[best];
  }
  for (; given > total_budget; --given) {
    int best = -1;
    for (int l = 0; l < n_layers; ++l)
      if (b[l] > 1 && (best < 0 || (double)b[l] - share[l] > (double)b[best] - share[best])) best = l;
    --b[best];
  }
  for (int l = 0; l < n_layers; ++l) budgets[l] = (int32_t)b[l];
  return STLITE_OK;
}

// Packed batches (stlite_compress_varlen): per-sequence shapes.
static stlite_status varlen_shapes(const stlite_shape* shape, int32_t n_seqs, const int32_t* cu,
                                   const stlite_frames* frames, size_t* ws_max) {
  if (!shape || n_seqs < 1 || !cu || !frames) return STLITE_EINVAL;
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  if (cu[0] != 0 || cu[n_seqs] != shape->n_tokens) return STLITE_EINVAL;
  size_t mx = 0;
  for (int i = 0; i < n_seqs; ++i) {
    if (cu[i + 1] <= cu[i]) return STLITE_EINVAL;
    stlite_shape ss = *shape;
    ss.n_tokens = cu[i + 1] - cu[i];
    if ((s = check_shape(&ss)) != STLITE_OK) return s;
    FrameTable ft;
    if ((s = build_frames(&ss, &frames[i], &ft)) != STLITE_OK) return s;
    const size_t b = plan_workspace(to_problem(&ss, 1), ft).total;
    if (b > mx) mx = b;
  }
  *ws_max = mx;
  return STLITE_OK;
}

stlite_status stlite_workspace_size_varlen(const stlite_shape* shape, int32_t n_seqs, const int32_t* cu_seqlens,
                                           const stlite_frames* frames, const stlite_params* params,
                                           size_t* bytes) {
  if (!bytes) return STLITE_EINVAL;
  stlite_status s;
  if (params && (s = check_params(params)) != STLITE_OK) return s;
  return varlen_shapes(shape, n_seqs, cu_seqlens, frames, bytes);
}

stlite_status stlite_compress_varlen(const stlite_shape* shape, int32_t n_seqs, const int32_t* cu_seqlens,
                                     const stlite_frames* frames, const stlite_params* params, const void* q,
                                     const void* k, const void* v, void* k_out, void* v_out, int32_t* idx_out,
                                     int32_t* cu_budget_out, void* ws, size_t ws_bytes, void* stream) {
  size_t ws_need = 0;
  stlite_status s = varlen_shapes(shape, n_seqs, cu_seqlens, frames, &ws_need);
  if (s != STLITE_OK) return s;
  if ((s = check_params(params)) != STLITE_OK) return s;
  if (!q || !k || !v || !k_out || !v_out || !idx_out) return STLITE_EINVAL;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out) ||
      !aligned16(idx_out))
    return STLITE_EINVAL;
  if (!ws || !aligned16(ws)) return STLITE_EINVAL;
  if (ws_bytes < ws_need) return STLITE_EWORKSPACE;
  // every budget is checked before anything is enqueued
  for (int i = 0; i < n_seqs; ++i)
    if (stlite_budget(cu_seqlens[i + 1] - cu_seqlens[i], params->beta, params->k_override) < 1)
      return STLITE_EINVAL;
  const size_t e = shape->dtype == STLITE_BF16 ? 2 : 4;
  const size_t row = (size_t)shape->n_kv_heads * shape->head_dim * e;  // one token of k / v
  const size_t qseq = (size_t)shape->window * shape->n_q_heads * shape->head_dim * e;
  size_t cum = 0;
  if (cu_budget_out) cu_budget_out[0] = 0;
  for (int i = 0; i < n_seqs; ++i) {
    stlite_shape ss = *shape;
    ss.n_tokens = cu_seqlens[i + 1] - cu_seqlens[i];
    Ctx c;
    if ((s = prepare(&ss, &frames[i], ws, ws_bytes, 1, stream, &c)) != STLITE_OK) return s;
    const int32_t b = stlite_budget(ss.n_tokens, params->beta, params->k_override);
    const size_t t0 = (size_t)cu_seqlens[i];
    LayerPtrs io =
        single_layer(static_cast<const uint8_t*>(q) + i * qseq, static_cast<const uint8_t*>(k) + t0 * row,
                     static_cast<const uint8_t*>(v) + t0 * row, static_cast<uint8_t*>(k_out) + cum * row,
                     static_cast<uint8_t*>(v_out) + cum * row, idx_out + (size_t)shape->n_kv_heads * cum);
    io.budget[0] = b;
    if ((s = compress_batch(c, params, io)) != STLITE_OK) return s;
    cum += (size_t)b;
    if (cu_budget_out) cu_budget_out[i + 1] = (int32_t)cum;
  }
  return STLITE_OK;
}

stlite_status stlite_compress_varlen_layers(const stlite_shape* shape, int32_t n_seqs, const int32_t* cu_seqlens,
                                            const stlite_frames* frames, const stlite_params* params,
                                            int32_t n_layers, const stlite_layer_io* layers,
                                            int32_t* cu_budget_out, void* ws, size_t ws_bytes, void* stream) {
  size_t ws_need = 0;
  stlite_status s = varlen_shapes(shape, n_seqs, cu_seqlens, frames, &ws_need);
  if (s != STLITE_OK) return s;
  if ((s = check_params(params)) != STLITE_OK) return s;
  if (n_layers < 1 || !layers) return STLITE_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    const stlite_layer_io& x = layers[l];
    if (!x.q || !x.k || !x.v || !x.k_out || !x.v_out || !x.idx_out) return STLITE_EINVAL;
    if (!aligned16(x.q) || !aligned16(x.k) || !aligned16(x.v) || !aligned16(x.k_out) || !aligned16(x.v_out) ||
        !aligned16(x.idx_out))
      return STLITE_EINVAL;
  }
  if (!ws || !aligned16(ws)) return STLITE_EINVAL;
  if (ws_bytes / (size_t)n_layers < ws_need) return STLITE_EWORKSPACE;
  for (int i = 0; i < n_seqs; ++i)
    if (stlite_budget(cu_seqlens[i + 1] - cu_seqlens[i], params->beta, params->k_override) < 1)
      return STLITE_EINVAL;
  const size_t e = shape->dtype == STLITE_BF16 ? 2 : 4;
  const size_t row = (size_t)shape->n_kv_heads * shape->head_dim * e;  // one token of k / v
  const size_t qseq = (size_t)shape->window * shape->n_q_heads * shape->head_dim * e;
  std::vector<stlite_layer_io> io((size_t)n_layers);
  size_t cum = 0;
  if (cu_budget_out) cu_budget_out[0] = 0;
  for (int i = 0; i < n_seqs; ++i) {
    stlite_shape ss = *shape;
    ss.n_tokens = cu_seqlens[i + 1] - cu_seqlens[i];
    const int32_t b = stlite_budget(ss.n_tokens, params->beta, params->k_override);
    const size_t t0 = (size_t)cu_seqlens[i];
    for (int l = 0; l < n_layers; ++l) {
      const stlite_layer_io& x = layers[l];
      io[l].q = static_cast<const uint8_t*>(x.q) + i * qseq;
      io[l].k = static_cast<const uint8_t*>(x.k) + t0 * row;
      io[l].v = static_cast<const uint8_t*>(x.v) + t0 * row;
      io[l].k_out = static_cast<uint8_t*>(x.k_out) + cum * row;
      io[l].v_out = static_cast<uint8_t*>(x.v_out) + cum * row;
      io[l].idx_out = x.idx_out + (size_t)shape->n_kv_heads * cum;
    }
    std::vector<int32_t> budgets((size_t)n_layers, b);
    if ((s = compress_layers_impl(&ss, &frames[i], params, n_layers, io.data(), budgets.data(), ws, ws_bytes,
                                  stream, false)) != STLITE_OK)
      return s;
    cum += (size_t)b;
    if (cu_budget_out) cu_budget_out[i + 1] = (int32_t)cum;
  }
  return STLITE_OK;
}

// Prompt-wide base scores (Mean Attention / full-attention bases).
static stlite_status check_prompt(const stlite_shape* shape, int32_t n_prompt, int32_t base) {
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  if (n_prompt < 1 || n_prompt > shape->n_tokens) return STLITE_EINVAL;
  if (base != STLITE_PROMPT_FULL && base != STLITE_PROMPT_MEAN) return STLITE_EINVAL;
  if (shape->n_q_heads / shape->n_kv_heads > 128) return STLITE_EUNSUPPORTED;
  return STLITE_OK;
}

static size_t prompt_ws_bytes(const stlite_shape* shape, int32_t n_prompt) {
  return 256 + prompt_bias_bytes(shape->n_tokens, n_prompt, shape->n_q_heads, shape->n_kv_heads);
}

stlite_status stlite_prompt_workspace_size(const stlite_shape* shape, int32_t n_prompt, size_t* bytes) {
  if (!bytes) return STLITE_EINVAL;
  stlite_status s = check_prompt(shape, n_prompt, STLITE_PROMPT_FULL);
  if (s != STLITE_OK) return s;
  *bytes = prompt_ws_bytes(shape, n_prompt);
  return STLITE_OK;
}

stlite_status stlite_prompt_score(const stlite_shape* shape, int32_t n_prompt, int32_t base, const void* q_prompt,
                                  const void* k, float* a_base, void* ws, size_t ws_bytes, void* stream) {
  stlite_status s = check_prompt(shape, n_prompt, base);
  if (s != STLITE_OK) return s;
  if (!q_prompt || !k || !a_base || !ws) return STLITE_EINVAL;
  if (!aligned16(q_prompt) || !aligned16(k) || !aligned16(a_base) || !aligned16(ws)) return STLITE_EINVAL;
  if (ws_bytes < prompt_ws_bytes(shape, n_prompt)) return STLITE_EWORKSPACE;
  uint8_t* w = static_cast<uint8_t*>(ws);
  return cuda_status(launch_prompt_score(shape->dtype == STLITE_BF16 ? kBF16 : kF32, q_prompt, k, shape->n_tokens,
                                         n_prompt, shape->n_q_heads,
                                         shape->n_kv_heads, base, a_base, reinterpret_cast<float*>(w + 256),
                                         reinterpret_cast<uint32_t*>(w), static_cast<cudaStream_t>(stream)));
}

// Decode attention over a (compressed) cache.
static stlite_status check_decode(const stlite_shape* shape) {
  stlite_status s = check_shape(shape);
  if (s != STLITE_OK) return s;
  if (shape->n_q_heads / shape->n_kv_heads > kDecMaxG) return STLITE_EUNSUPPORTED;
  return STLITE_OK;
}

stlite_status stlite_decode_workspace_size(const stlite_shape* shape, size_t* bytes) {
  if (!bytes) return STLITE_EINVAL;
  stlite_status s = check_decode(shape);
  if (s != STLITE_OK) return s;
  *bytes = decode_workspace_bytes(shape->n_tokens, shape->n_q_heads, shape->n_kv_heads, shape->window, 1);
  return STLITE_OK;
}

stlite_status stlite_decode_attention(const stlite_shape* shape, const void* q, const void* k, const void* v,
                                      float* out, void* ws, size_t ws_bytes, void* stream) {
  stlite_status s = check_decode(shape);
  if (s != STLITE_OK) return s;
  if (!q || !k || !v || !out || !ws) return STLITE_EINVAL;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(ws)) return STLITE_EINVAL;
  if (ws_bytes < decode_workspace_bytes(shape->n_tokens, shape->n_q_heads, shape->n_kv_heads, shape->window, 1))
    return STLITE_EWORKSPACE;
  DecBatch b;
  memset(&b, 0, sizeof(b));
  b.q[0] = q;
  b.k[0] = k;
  b.v[0] = v;
  b.out[0] = out;
  return cuda_status(launch_decode(shape->dtype == STLITE_BF16 ? kBF16 : kF32, b, 1, shape->n_tokens,
                                   shape->n_q_heads, shape->n_kv_heads, shape->window, ws,
                                   static_cast<cudaStream_t>(stream)));
}

// The launches of a call run batches of kMaxLayers layers and then the rest;
// the batch size sets the splits, so the workspace is the larger need.
static size_t decode_layers_bytes(const stlite_shape* shape, int32_t n_layers) {
  size_t need = 0;
  const int full = n_layers >= kMaxLayers ? kMaxLayers : 0, rest = n_layers % kMaxLayers;
  for (int L : {full, rest})
    if (L > 0) {
      const size_t b =
          decode_workspace_bytes(shape->n_tokens, shape->n_q_heads, shape->n_kv_heads, shape->window, L);
      if (b > need) need = b;
    }
  return need;
}

stlite_status stlite_decode_layers_workspace_size(const stlite_shape* shape, int32_t n_layers, size_t* bytes) {
  if (!bytes || n_layers < 1) return STLITE_EINVAL;
  stlite_status s = check_decode(shape);
  if (s != STLITE_OK) return s;
  *bytes = decode_layers_bytes(shape, n_layers);
  return STLITE_OK;
}

stlite_status stlite_decode_attention_layers(const stlite_shape* shape, int32_t n_layers,
                                             const stlite_decode_io* layers, void* ws, size_t ws_bytes,
                                             void* stream) {
  stlite_status s = check_decode(shape);
  if (s != STLITE_OK) return s;
  if (n_layers < 1 || !layers || !ws || !aligned16(ws)) return STLITE_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    const stlite_decode_io& x = layers[l];
    if (!x.q || !x.k || !x.v || !x.out) return STLITE_EINVAL;
    if (!aligned16(x.q) || !aligned16(x.k) || !aligned16(x.v) || !aligned16(x.out)) return STLITE_EINVAL;
  }
  if (ws_bytes < decode_layers_bytes(shape, n_layers)) return STLITE_EWORKSPACE;
  // up to kMaxLayers layers per launch; the batches share the workspace
  for (int l0 = 0; l0 < n_layers; l0 += kMaxLayers) {
    const int L = n_layers - l0 < kMaxLayers ? n_layers - l0 : kMaxLayers;
    DecBatch b;
    memset(&b, 0, sizeof(b));
    for (int l = 0; l < L; ++l) {
      b.q[l] = layers[l0 + l].q;
      b.k[l] = layers[l0 + l].k;
      b.v[l] = layers[l0 + l].v;
      b.out[l] = layers[l0 + l].out;
    }
    if ((s = cuda_status(launch_decode(shape->dtype == STLITE_BF16 ? kBF16 : kF32, b, L, shape->n_tokens,
                                       shape->n_q_heads, shape->n_kv_heads, shape->window, ws,
                                       static_cast<cudaStream_t>(stream)))) != STLITE_OK)
      return s;
  }
  return STLITE_OK;
}

stlite_status stlite_device_status(void* ws, void* stream, stlite_status* status) {
  if (!status || (ws && !aligned16(ws))) return STLITE_EINVAL;
  if (!ws) {  // the error word of stlite_score_noalloc's fixed scratch on the current device
    uint32_t* word = nullptr;
    if (noalloc_error_word(&word) != cudaSuccess) return STLITE_ECUDA;
    ws = word;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t word = 0;
  if (cudaMemcpyAsync(&word, ws, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess) return STLITE_ECUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return STLITE_ECUDA;
  if (cudaMemsetAsync(ws, 0, 4, st) != cudaSuccess) return STLITE_ECUDA;
  *status = (word & kErrTimeout) ? STLITE_ETIMEOUT : (word ? STLITE_ECUDA : STLITE_OK);
  return STLITE_OK;
}

stlite_status stlite_timing_enable(int32_t on) {
  g_timing_on.store(on ? 1 : 0);
  return STLITE_OK;
}

stlite_status stlite_timing_read(stlite_kernel_time* out, int32_t capacity, int32_t* count) {
  if (!count || capacity < 0 || (capacity > 0 && !out)) return STLITE_EINVAL;
  std::vector<TimingRecord> recs;
  {
    std::lock_guard<std::mutex> lk(g_timing_mu);
    recs.swap(g_records);
  }
  std::map<std::string, std::pair<int, double>> agg;
  bool ok = true;
  for (auto& r : recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.stop) != cudaSuccess || cudaEventElapsedTime(&ms, r.start, r.stop) != cudaSuccess)
      ok = false;
    auto& a = agg[r.name];
    a.first += 1;
    a.second += ms;
  }
  {
    std::lock_guard<std::mutex> lk(g_timing_mu);
    for (auto& r : recs) {
      g_event_pool.push_back(r.start);
      g_event_pool.push_back(r.stop);
    }
  }
  int i = 0;
  for (auto& kv : agg) {
    if (i < capacity) {
      memset(out[i].name, 0, sizeof(out[i].name));
      strncpy(out[i].name, kv.first.c_str(), sizeof(out[i].name) - 1);
      out[i].launches = kv.second.first;
      out[i].total_ms = kv.second.second;
    }
    ++i;
  }
  *count = i;
  return ok ? STLITE_OK : STLITE_ECUDA;
}

const char* stlite_status_string(stlite_status status) {
  switch (status) {
    case STLITE_OK: return "ok";
    case STLITE_EINVAL: return "invalid argument";
    case STLITE_EUNSUPPORTED: return "unsupported shape or layout";
    case STLITE_EWORKSPACE: return "workspace too small";
    case STLITE_ECUDA: return "CUDA launch or runtime error";
    case STLITE_ETIMEOUT: return "a kernel wait timed out";
  }
  return "unknown status";
}

}  // extern "C"
