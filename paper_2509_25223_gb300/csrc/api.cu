// api.cu -- the C ABI declared in include/rdn.h: argument validation, error
// reporting and dispatch to the kernel launchers.  No exception or abort
// crosses this boundary; every entry point returns an rdn_status_t.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "status.cuh"

namespace rdn {
namespace prof {
namespace {
struct Rec {
  const char *name;
  cudaEvent_t ev[2];
};
std::atomic<bool> g_active{false};
std::mutex g_mu;
std::vector<Rec> g_recs;
size_t g_next = 0;   // next record to fill
size_t g_seen = 0;   // launches seen while active
thread_local long g_open = -1;  // record opened by begin() on this thread
}  // namespace

bool active() { return g_active.load(std::memory_order_relaxed); }

void begin(const char *name, cudaStream_t s) {
  std::lock_guard<std::mutex> lk(g_mu);
  ++g_seen;
  g_open = -1;
  if (g_next < g_recs.size()) {
    g_open = (long)g_next++;
    g_recs[g_open].name = name;
    cudaEventRecord(g_recs[g_open].ev[0], s);
  }
}

void end(cudaStream_t s) {
  if (g_open < 0) return;
  std::lock_guard<std::mutex> lk(g_mu);
  cudaEventRecord(g_recs[g_open].ev[1], s);
  g_open = -1;
}
}  // namespace prof
}  // namespace rdn

namespace {

thread_local char g_err[512] = "";

rdn_status_t fail(rdn_status_t st, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof g_err, fmt, ap);
  va_end(ap);
  return st;
}

rdn_status_t ok() {
  g_err[0] = '\0';
  return RDN_OK;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

#define REQUIRE_PTR(p)                                                        \
  do {                                                                        \
    if (!(p)) return fail(RDN_ERR_INVALID_ARG, "%s: " #p " is NULL", fn);     \
    if (!aligned16(p))                                                        \
      return fail(RDN_ERR_MISALIGNED, "%s: " #p " is not 16-byte aligned", fn); \
  } while (0)
#define OPTIONAL_PTR(p)                                                       \
  do {                                                                        \
    if ((p) && !aligned16(p))                                                 \
      return fail(RDN_ERR_MISALIGNED, "%s: " #p " is not 16-byte aligned", fn); \
  } while (0)

rdn_status_t check_clip(const char *fn, float c) {
  if (isnan(c) || c < 0.f) return fail(RDN_ERR_INVALID_ARG, "%s: clip must be >= 0 (got %g)", fn, c);
  return RDN_OK;
}

rdn_status_t check_fwd_shapes(const char *fn, const rdn_fwd_args *a) {
  if (!a) return fail(RDN_ERR_INVALID_ARG, "%s: args is NULL", fn);
  if (a->B < 1 || a->H < 1 || a->T < 0)
    return fail(RDN_ERR_INVALID_ARG, "%s: need B >= 1, H >= 1, T >= 0 (got B=%d T=%d H=%d)", fn,
                a->B, a->T, a->H);
  if (a->dtype != RDN_F32 && a->dtype != RDN_BF16)
    return fail(RDN_ERR_UNSUPPORTED, "%s: dtype %d unsupported", fn, a->dtype);
  if (!((a->Dk == 64 || a->Dk == 128) && a->Dv == a->Dk))
    return fail(RDN_ERR_UNSUPPORTED, "%s: supported head dims are Dk = Dv in {64, 128} (got %d, %d)",
                fn, a->Dk, a->Dv);
  if ((long long)a->B * a->T * a->H > (1ll << 31) / 128)
    return fail(RDN_ERR_UNSUPPORTED, "%s: B*T*H = %lld too large", fn,
                (long long)a->B * a->T * a->H);
  if (a->cu_seqlens) {  // packed sequences: one row of T tokens split by the table
    if (a->B != 1)
      return fail(RDN_ERR_INVALID_ARG, "%s: cu_seqlens needs B = 1 (got B=%d)", fn, a->B);
    if (a->num_seqs < 1 || (long long)a->num_seqs * a->H > (1ll << 24))
      return fail(RDN_ERR_INVALID_ARG, "%s: need 1 <= num_seqs, num_seqs*H <= 2^24 (got %d)", fn,
                  a->num_seqs);
    if (!aligned16(a->cu_seqlens))
      return fail(RDN_ERR_MISALIGNED, "%s: cu_seqlens is not 16-byte aligned", fn);
  }
  if (a->flags & ~(RDN_FLAG_SAVE_FOR_BWD | RDN_FLAG_TIED_GAMMA | RDN_FLAG_VARIANTS |
                   RDN_FLAG_F32_OUT | RDN_FLAG_QK_NORM))
    return fail(RDN_ERR_UNSUPPORTED, "%s: flags 0x%x unsupported", fn, a->flags);
  if ((a->flags & RDN_FLAG_QK_NORM) && !(a->qk_eps > 0.f && !isinf(a->qk_eps)))
    return fail(RDN_ERR_INVALID_ARG, "%s: RDN_FLAG_QK_NORM needs qk_eps > 0 and finite (got %g)",
                fn, a->qk_eps);
  if ((a->flags & RDN_FLAG_F32_OUT) && a->dtype == RDN_BF16 && a->Dk != 128)
    return fail(RDN_ERR_UNSUPPORTED,
                "%s: RDN_FLAG_F32_OUT with bf16 inputs needs Dk = 128 (the tensor-core path)", fn);
  if (isnan(a->scale) || isinf(a->scale))
    return fail(RDN_ERR_INVALID_ARG, "%s: scale must be finite", fn);
  return check_clip(fn, a->clip);
}

rdn_status_t check_fwd_ptrs(const char *fn, const rdn_fwd_args *a) {
  if (a->T > 0) {
    REQUIRE_PTR(a->q);
    REQUIRE_PTR(a->k);
    REQUIRE_PTR(a->v);
    REQUIRE_PTR(a->g);
    REQUIRE_PTR(a->beta);
    REQUIRE_PTR(a->gamma);
    REQUIRE_PTR(a->o);
  }
  OPTIONAL_PTR(a->S0);
  OPTIONAL_PTR(a->R0);
  OPTIONAL_PTR(a->ST);
  OPTIONAL_PTR(a->RT);
  OPTIONAL_PTR(a->S_chunks);
  OPTIONAL_PTR(a->R_chunks);
  if ((a->S_chunks == nullptr) != (a->R_chunks == nullptr))
    return fail(RDN_ERR_INVALID_ARG, "%s: S_chunks and R_chunks must be both set or both NULL", fn);
  if ((a->flags & RDN_FLAG_SAVE_FOR_BWD) && !a->S_chunks && a->T > 0)
    return fail(RDN_ERR_INVALID_ARG, "%s: RDN_FLAG_SAVE_FOR_BWD needs S_chunks and R_chunks", fn);
  return RDN_OK;
}

// The arguments with the tied-gate flag resolved: gamma is beta.
rdn_fwd_args untied(const rdn_fwd_args &a) {
  rdn_fwd_args u = a;
  if (a.flags & RDN_FLAG_TIED_GAMMA) u.gamma = a.beta;
  return u;
}

// The failures RDN_FAULT_INJECT asks for (rdn::fault_injection), after validation.
rdn_status_t injected(const char *fn) {
  switch (rdn::fault_injection()) {
    case 1: return fail(RDN_ERR_WORKSPACE, "%s: workspace check failed (injected)", fn);
    case 2: return fail(RDN_ERR_CUDA, "%s: launch failed (injected)", fn);
    default: return RDN_OK;
  }
}

rdn_status_t cuda_status(const char *fn, cudaError_t e) {
  if (e == cudaSuccess) return ok();
  return fail(RDN_ERR_CUDA, "%s: CUDA error %d (%s)", fn, (int)e, cudaGetErrorString(e));
}

// An NVTX range named after the entry point for the duration of the call
// (host side: validation and enqueueing), seen by profilers and free without one.
struct CallRange {
  explicit CallRange(const char *fn) { nvtxRangePushA(fn); }
  ~CallRange() { nvtxRangePop(); }
};

rdn_status_t fwd_common(const char *fn, const rdn_fwd_args *a0, int variant, cudaStream_t s) {
  CallRange range(fn);
  rdn_status_t st = check_fwd_shapes(fn, a0);
  if (st != RDN_OK) return st;
  const rdn_fwd_args ua = untied(*a0);
  const rdn_fwd_args *a = &ua;
  if ((st = check_fwd_ptrs(fn, a)) != RDN_OK) return st;
  const rdn::FwdPlan plan = rdn::plan_fwd(*a, variant);
  if (plan.total_bytes > 0) {
    if (!a->workspace || a->workspace_bytes < plan.total_bytes)
      return fail(RDN_ERR_WORKSPACE, "%s: workspace of %zu bytes required (got %zu)", fn,
                  plan.total_bytes, a->workspace ? a->workspace_bytes : (size_t)0);
    if (!aligned16(a->workspace))
      return fail(RDN_ERR_WORKSPACE, "%s: workspace is not 16-byte aligned", fn);
  }
  if ((st = injected(fn)) != RDN_OK) return st;
  return cuda_status(fn, rdn::launch_fwd(*a, variant, s));
}

}  // namespace

extern "C" {

const char *rdn_last_error(void) { return g_err; }

const char *rdn_version(void) { return "rdn-gb300 0.1 (sm_103a)"; }

rdn_status_t rdn_prof_start(int capacity) {
  using namespace rdn::prof;
  if (capacity < 0 || capacity > (1 << 20))
    return fail(RDN_ERR_INVALID_ARG, "rdn_prof_start: capacity %d out of range", capacity);
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_active.load()) return fail(RDN_ERR_INVALID_ARG, "rdn_prof_start: already recording");
  g_recs.assign((size_t)capacity, Rec{"", {nullptr, nullptr}});
  for (auto &r : g_recs)
    for (auto &e : r.ev) {
      cudaError_t err = cudaEventCreate(&e);
      if (err != cudaSuccess) {
        for (auto &r2 : g_recs)
          for (auto &e2 : r2.ev)
            if (e2) cudaEventDestroy(e2);
        g_recs.clear();
        return fail(RDN_ERR_CUDA, "rdn_prof_start: cudaEventCreate: %s", cudaGetErrorString(err));
      }
    }
  g_next = 0;
  g_seen = 0;
  g_active.store(true);
  return ok();
}

rdn_status_t rdn_prof_stop(rdn_prof_record *out, int cap, int *n) {
  using namespace rdn::prof;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_active.load()) return fail(RDN_ERR_INVALID_ARG, "rdn_prof_stop: not recording");
  g_active.store(false);
  rdn_status_t st = RDN_OK;
  for (size_t i = 0; i < g_next; ++i) {
    cudaError_t err = cudaEventSynchronize(g_recs[i].ev[1]);
    float ms = -1.f;
    if (err == cudaSuccess) err = cudaEventElapsedTime(&ms, g_recs[i].ev[0], g_recs[i].ev[1]);
    if (err != cudaSuccess && st == RDN_OK)
      st = fail(RDN_ERR_CUDA, "rdn_prof_stop: %s", cudaGetErrorString(err));
    if (out && (int)i < cap) {
      snprintf(out[i].name, sizeof out[i].name, "%s", g_recs[i].name);
      out[i].ms = ms;
    }
  }
  if (n) *n = (int)g_seen;
  for (auto &r : g_recs)
    for (auto &e : r.ev)
      if (e) cudaEventDestroy(e);
  g_recs.clear();
  g_next = g_seen = 0;
  return st == RDN_OK ? ok() : st;
}

// ---- rdn_fwd_noalloc: the forward with a built-in scratch array.
//
// For callers that own only their inputs and outputs and may not allocate
// device memory (see rdn.h).  The scratch is this file-scope device array; in
// host code its name is only a host-side stand-in, so its device address is
// looked up with cudaGetSymbolAddress once per device (with that device
// current) and passed to the kernels like a caller workspace.
static __device__ __align__(256) unsigned char g_noalloc_scratch[RDN_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void *g_noalloc_ptr[kMaxDevices] = {};
}  // namespace

// The status word (status.cuh): one per device, looked up like the scratch.
static __device__ int g_status;
namespace {
std::mutex g_status_mu;
void *g_status_ptr[kMaxDevices] = {};
}  // namespace

}  // extern "C"

namespace rdn {
int fault_injection() {
  const char *e = getenv("RDN_FAULT_INJECT");
  if (!e) return 0;
  if (!strcmp(e, "workspace")) return 1;
  if (!strcmp(e, "launch")) return 2;
  if (!strcmp(e, "device_wait")) return 3;
  if (!strcmp(e, "device_wait_bwd")) return 4;
  return 0;
}

int *status_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_status_mu);
  if (!g_status_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
    g_status_ptr[dev] = p;
  }
  return static_cast<int *>(g_status_ptr[dev]);
}
}  // namespace rdn

extern "C" {

rdn_status_t rdn_device_status(rdn_stream_t stream, int *status) {
  const char *fn = "rdn_device_status";
  if (!status) return fail(RDN_ERR_INVALID_ARG, "%s: status is NULL", fn);
  int *w = rdn::status_word();
  if (!w) return fail(RDN_ERR_CUDA, "%s: the status word of this device is not available", fn);
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  int v = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&v, w, sizeof v, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && v != 0) {
    const int zero = 0;
    e = cudaMemcpy(w, &zero, sizeof zero, cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) return cuda_status(fn, e);
  *status = v;
  return ok();
}

rdn_status_t rdn_fwd_noalloc(const rdn_fwd_args *a0, rdn_stream_t stream) {
  const char *fn = "rdn_fwd_noalloc";
  CallRange range(fn);
  rdn_status_t st = check_fwd_shapes(fn, a0);
  if (st != RDN_OK) return st;
  const rdn_fwd_args ua = untied(*a0);
  const rdn_fwd_args *a = &ua;
  if (a->flags & RDN_FLAG_SAVE_FOR_BWD)  // what it saves would stay in the built-in scratch
    return fail(RDN_ERR_UNSUPPORTED,
                "%s: RDN_FLAG_SAVE_FOR_BWD needs a caller workspace (use rdn_fwd)", fn);
  if ((st = check_fwd_ptrs(fn, a)) != RDN_OK) return st;
  const size_t need = rdn::plan_fwd(*a, 1).total_bytes;
  if (need > (size_t)RDN_NOALLOC_SCRATCH_BYTES) {
    // per-chunk record size and fixed overhead, from the workspace plan
    rdn_fwd_args one = *a, two = *a;
    one.B = one.H = two.B = two.H = 1;
    one.cu_seqlens = two.cu_seqlens = nullptr;
    one.T = rdn::kChunk;
    two.T = 2 * rdn::kChunk;
    const size_t per_chunk = rdn::plan_fwd(two, 1).total_bytes - rdn::plan_fwd(one, 1).total_bytes;
    const size_t fixed = rdn::plan_fwd(one, 1).total_bytes - per_chunk;
    return fail(RDN_ERR_WORKSPACE,
                "%s: this problem needs %zu bytes of scratch (%lld chunk records) but "
                "the built-in scratch holds %zu bytes (at most %zu chunks); use rdn_fwd with a "
                "caller workspace",
                fn, need, rdn::call_records(*a),
                (size_t)RDN_NOALLOC_SCRATCH_BYTES,
                ((size_t)RDN_NOALLOC_SCRATCH_BYTES - fixed) / per_chunk);
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_status(fn, e);
  if (dev < 0 || dev >= kMaxDevices)
    return fail(RDN_ERR_UNSUPPORTED, "%s: device ordinal %d beyond %d", fn, dev, kMaxDevices);
  void *scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void *p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess) return cuda_status(fn, e);
      g_noalloc_ptr[dev] = p;
    }
    scratch = g_noalloc_ptr[dev];
  }
  rdn_fwd_args b = *a;
  b.workspace = scratch;
  b.workspace_bytes = RDN_NOALLOC_SCRATCH_BYTES;
  return cuda_status(fn, rdn::launch_fwd(b, 1, (cudaStream_t)stream));
}

rdn_status_t rla_fwd_workspace_size(const rdn_fwd_args *a, size_t *bytes) {
  rdn_status_t st = check_fwd_shapes("rla_fwd_workspace_size", a);
  if (st != RDN_OK) return st;
  if (!bytes) return fail(RDN_ERR_INVALID_ARG, "rla_fwd_workspace_size: bytes is NULL");
  *bytes = rdn::plan_fwd(*a, 0).total_bytes;
  return ok();
}

rdn_status_t rdn_fwd_workspace_size(const rdn_fwd_args *a, size_t *bytes) {
  rdn_status_t st = check_fwd_shapes("rdn_fwd_workspace_size", a);
  if (st != RDN_OK) return st;
  if (!bytes) return fail(RDN_ERR_INVALID_ARG, "rdn_fwd_workspace_size: bytes is NULL");
  *bytes = rdn::plan_fwd(*a, 1).total_bytes;
  return ok();
}

rdn_status_t rdn_chunk_slots(const rdn_fwd_args *a, long long *slots) {
  rdn_status_t st = check_fwd_shapes("rdn_chunk_slots", a);
  if (st != RDN_OK) return st;
  if (!slots) return fail(RDN_ERR_INVALID_ARG, "rdn_chunk_slots: slots is NULL");
  *slots = rdn::call_records(*a);
  return ok();
}

rdn_status_t rla_fwd(const rdn_fwd_args *a, rdn_stream_t stream) {
  return fwd_common("rla_fwd", a, 0, (cudaStream_t)stream);
}

rdn_status_t rdn_fwd(const rdn_fwd_args *a, rdn_stream_t stream) {
  return fwd_common("rdn_fwd", a, 1, (cudaStream_t)stream);
}

namespace {
rdn_status_t bwd_workspace_common(const char *fn, const rdn_bwd_args *a, int variant,
                                  size_t *bytes) {
  if (!a) return fail(RDN_ERR_INVALID_ARG, "%s: args is NULL", fn);
  rdn_status_t st = check_fwd_shapes(fn, &a->fwd);
  if (st != RDN_OK) return st;
  if (!bytes) return fail(RDN_ERR_INVALID_ARG, "%s: bytes is NULL", fn);
  *bytes = rdn::plan_bwd(*a, variant).total_bytes;
  return ok();
}

rdn_status_t bwd_common(const char *fn, const rdn_bwd_args *a0, int variant, cudaStream_t stream) {
  CallRange range(fn);
  if (!a0) return fail(RDN_ERR_INVALID_ARG, "%s: args is NULL", fn);
  rdn_status_t st = check_fwd_shapes(fn, &a0->fwd);
  if (st != RDN_OK) return st;
  rdn_bwd_args ua = *a0;
  ua.fwd = untied(a0->fwd);
  const rdn_bwd_args *a = &ua;
  const rdn_fwd_args *f = &a->fwd;
  if (f->T > 0) {
    REQUIRE_PTR(f->q);
    REQUIRE_PTR(f->k);
    REQUIRE_PTR(f->v);
    REQUIRE_PTR(f->g);
    REQUIRE_PTR(f->beta);
    REQUIRE_PTR(f->gamma);
    REQUIRE_PTR(a->dO);
    REQUIRE_PTR(a->dq);
    REQUIRE_PTR(a->dk);
    REQUIRE_PTR(a->dv);
    REQUIRE_PTR(a->dg);
    REQUIRE_PTR(a->dbeta);
    if (!(f->flags & RDN_FLAG_TIED_GAMMA)) REQUIRE_PTR(a->dgamma);
  }
  OPTIONAL_PTR(a->dgamma);
  OPTIONAL_PTR(f->S0);
  OPTIONAL_PTR(f->R0);
  OPTIONAL_PTR(f->S_chunks);
  OPTIONAL_PTR(f->R_chunks);
  if ((f->S_chunks == nullptr) != (f->R_chunks == nullptr))
    return fail(RDN_ERR_INVALID_ARG, "%s: S_chunks and R_chunks must be both set or both NULL", fn);
  if ((f->flags & RDN_FLAG_SAVE_FOR_BWD) && !f->workspace && f->T > 0)
    return fail(RDN_ERR_INVALID_ARG,
                "%s: RDN_FLAG_SAVE_FOR_BWD in fwd.flags needs the forward's fwd.workspace", fn);
  if (f->workspace && f->T > 0) {  // the forward's records, reused
    if (!f->S_chunks)
      return fail(RDN_ERR_INVALID_ARG,
                  "%s: fwd.workspace is reused only together with fwd.S_chunks/R_chunks", fn);
    if (!aligned16(f->workspace))
      return fail(RDN_ERR_WORKSPACE, "%s: fwd.workspace is not 16-byte aligned", fn);
    const size_t fneed = rdn::plan_fwd(*f, variant).total_bytes;
    if (f->workspace_bytes < fneed)
      return fail(RDN_ERR_WORKSPACE, "%s: fwd.workspace of %zu bytes required (got %zu)", fn, fneed,
                  f->workspace_bytes);
  }
  OPTIONAL_PTR(a->dST);
  OPTIONAL_PTR(a->dRT);
  OPTIONAL_PTR(a->dS0);
  OPTIONAL_PTR(a->dR0);
  const rdn::BwdPlan plan = rdn::plan_bwd(*a, variant);
  if (plan.total_bytes > 0) {
    if (!a->workspace || a->workspace_bytes < plan.total_bytes)
      return fail(RDN_ERR_WORKSPACE, "%s: workspace of %zu bytes required (got %zu)", fn,
                  plan.total_bytes, a->workspace ? a->workspace_bytes : (size_t)0);
    if (!aligned16(a->workspace))
      return fail(RDN_ERR_WORKSPACE, "%s: workspace is not 16-byte aligned", fn);
  }
  if ((st = injected(fn)) != RDN_OK) return st;
  return cuda_status(fn, rdn::launch_bwd(*a, variant, stream));
}
}  // namespace

rdn_status_t rla_bwd_workspace_size(const rdn_bwd_args *a, size_t *bytes) {
  return bwd_workspace_common("rla_bwd_workspace_size", a, 0, bytes);
}

rdn_status_t rdn_bwd_workspace_size(const rdn_bwd_args *a, size_t *bytes) {
  return bwd_workspace_common("rdn_bwd_workspace_size", a, 1, bytes);
}

rdn_status_t rla_bwd(const rdn_bwd_args *a, rdn_stream_t stream) {
  return bwd_common("rla_bwd", a, 0, (cudaStream_t)stream);
}

rdn_status_t rdn_bwd(const rdn_bwd_args *a, rdn_stream_t stream) {
  return bwd_common("rdn_bwd", a, 1, (cudaStream_t)stream);
}

namespace {
rdn_status_t prologue_common(const char *fn, const rdn_prologue_args *a, bool bwd,
                             cudaStream_t stream) {
  CallRange range(fn);
  if (!a) return fail(RDN_ERR_INVALID_ARG, "%s: args is NULL", fn);
  if (a->rows < 1 || a->rows > (1ll << 40))
    return fail(RDN_ERR_INVALID_ARG, "%s: rows must be in [1, 2^40] (got %lld)", fn, a->rows);
  if (a->D != 64 && a->D != 128)
    return fail(RDN_ERR_UNSUPPORTED, "%s: supported row lengths are D in {64, 128}", fn);
  if (a->dtype != RDN_F32 && a->dtype != RDN_BF16)
    return fail(RDN_ERR_UNSUPPORTED, "%s: dtype %d unsupported", fn, a->dtype);
  if (!(a->eps > 0.f) || isinf(a->eps))
    return fail(RDN_ERR_INVALID_ARG, "%s: eps must be positive and finite", fn);
  for (int i = 0; i < 2; ++i) {
    if (i == 1 && !a->x[1]) break;
    REQUIRE_PTR(a->x[i]);
    if (!bwd) {
      REQUIRE_PTR(a->y[i]);
      if (a->y[i] == a->x[i]) return fail(RDN_ERR_INVALID_ARG, "%s: y aliases x", fn);
    } else {
      REQUIRE_PTR(a->dy[i]);
      REQUIRE_PTR(a->dx[i]);
    }
  }
  return cuda_status(fn, rdn::launch_prologue(*a, bwd, stream));
}
}  // namespace

rdn_status_t rdn_qk_prologue(const rdn_prologue_args *a, rdn_stream_t stream) {
  return prologue_common("rdn_qk_prologue", a, false, (cudaStream_t)stream);
}

rdn_status_t rdn_qk_prologue_bwd(const rdn_prologue_args *a, rdn_stream_t stream) {
  return prologue_common("rdn_qk_prologue_bwd", a, true, (cudaStream_t)stream);
}

rdn_status_t rdn_decode_step(const rdn_decode_args *a, rdn_stream_t stream) {
  const char *fn = "rdn_decode_step";
  CallRange range(fn);
  if (!a) return fail(RDN_ERR_INVALID_ARG, "%s: args is NULL", fn);
  if (a->N < 1 || a->H < 1)
    return fail(RDN_ERR_INVALID_ARG, "%s: need N >= 1, H >= 1 (got N=%d H=%d)", fn, a->N, a->H);
  if (!((a->Dk == 64 || a->Dk == 128) && a->Dv == a->Dk))
    return fail(RDN_ERR_UNSUPPORTED, "%s: supported head dims are Dk = Dv in {64, 128}", fn);
  if (a->dtype != RDN_F32 && a->dtype != RDN_BF16)
    return fail(RDN_ERR_UNSUPPORTED, "%s: dtype %d unsupported", fn, a->dtype);
  if (a->variant != 0 && a->variant != 1)
    return fail(RDN_ERR_INVALID_ARG, "%s: variant must be 0 (RLA) or 1 (RDN)", fn);
  if ((long long)a->N * a->H > (1ll << 31) / 4)
    return fail(RDN_ERR_UNSUPPORTED, "%s: N*H too large", fn);
  rdn_status_t st = check_clip(fn, a->clip);
  if (st != RDN_OK) return st;
  if (isnan(a->scale) || isinf(a->scale)) return fail(RDN_ERR_INVALID_ARG, "%s: scale must be finite", fn);
  if (a->flags & ~(RDN_FLAG_TIED_GAMMA | RDN_FLAG_VARIANTS | RDN_FLAG_QK_NORM))
    return fail(RDN_ERR_UNSUPPORTED, "%s: flags 0x%x unsupported", fn, a->flags);
  if ((a->flags & RDN_FLAG_QK_NORM) && !(a->qk_eps > 0.f && !isinf(a->qk_eps)))
    return fail(RDN_ERR_INVALID_ARG, "%s: RDN_FLAG_QK_NORM needs qk_eps > 0 and finite (got %g)",
                fn, a->qk_eps);
  REQUIRE_PTR(a->q);
  REQUIRE_PTR(a->k);
  REQUIRE_PTR(a->v);
  REQUIRE_PTR(a->g);
  REQUIRE_PTR(a->beta);
  if (!(a->flags & RDN_FLAG_TIED_GAMMA)) REQUIRE_PTR(a->gamma);
  REQUIRE_PTR(a->S);
  REQUIRE_PTR(a->R);
  REQUIRE_PTR(a->o);
  if (a->S == a->R) return fail(RDN_ERR_INVALID_ARG, "%s: S and R alias", fn);
  rdn_decode_args b = *a;
  if (a->flags & RDN_FLAG_TIED_GAMMA) b.gamma = a->beta;
  return cuda_status(fn, rdn::launch_decode(b, (cudaStream_t)stream));
}

}  // extern "C"
