// common.cuh -- small device helpers shared by the RLA/RDN kernels.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "rdn.h"

namespace rdn {

// Chunk length of the chunkwise-parallel forms (tokens per chunk).
constexpr int kChunk = 64;
// the variant flags of rdn.h, which the fp32 chunk kernels implement
#define RDN_FLAG_VARIANTS                                                             \
  (RDN_FLAG_DECAYED_RESIDUAL | RDN_FLAG_PLAIN_COMBINE | RDN_FLAG_TANH_RESIDUAL | \
   RDN_FLAG_STATELESS_AUX)

template <typename T> __device__ __forceinline__ float to_f32(T x);
template <> __device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float clampf(float x, float c) { return fminf(fmaxf(x, -c), c); }

// The residual map of Section 3.3 (clip to [-c, c]) or, with tnh, the
// log-cosh residual c tanh(x / c) of Appendix B; and their derivatives (the
// clip's taken as 1 on |x| <= c).
__device__ __forceinline__ float resid_map(float x, float c, bool tnh) {
  if (!tnh) return clampf(x, c);
  if (isinf(c)) return x;
  if (c == 0.f) return 0.f;
  return c * tanhf(x / c);
}
// The residual map's derivative (in [0, 1]) as 16-bit fixed point, d * 65535
// rounded: an absolute error of at most 7.7e-6 over the whole range, where a
// bf16 copy would be off by up to 2^-9 of d (the product d dX2 of the backward
// can be large against the gradients it lands in).
__device__ __forceinline__ uint32_t grad_q16(float d) { return __float2uint_rn(d * 65535.f); }
__device__ __forceinline__ float grad_uq16(uint32_t q) { return (float)q * (1.f / 65535.f); }
__device__ __forceinline__ float resid_grad(float x, float c, bool tnh) {
  if (!tnh) return fabsf(x) <= c ? 1.f : 0.f;
  if (isinf(c)) return 1.f;
  if (c == 0.f) return 0.f;
  const float t = tanhf(x / c);
  return 1.f - t * t;
}

}  // namespace rdn

// Per-launch timing of the library's kernels (rdn_prof_start / _stop).
namespace rdn {
namespace prof {
bool active();
void begin(const char *name, cudaStream_t s);
void end(cudaStream_t s);
}  // namespace prof
}  // namespace rdn

// Wraps one kernel launch statement with the timing events when recording.
#define RDN_LAUNCH(name, stream, ...)                      \
  do {                                                     \
    const bool rdn_prof_on_ = ::rdn::prof::active();       \
    if (rdn_prof_on_) ::rdn::prof::begin(name, stream);    \
    __VA_ARGS__;                                           \
    if (rdn_prof_on_) ::rdn::prof::end(stream);            \
  } while (0)

// Internal launchers (defined in the kernel translation units, called by
// api.cu after argument validation).  Each returns cudaGetLastError() of its
// launches.
namespace rdn {
cudaError_t launch_decode(const rdn_decode_args &a, cudaStream_t s);
cudaError_t launch_prologue(const rdn_prologue_args &a, bool bwd, cudaStream_t s);
// The prologue's backward with dy in fp32 whatever a.dtype (x in a.dtype; dx
// in a.dtype, or fp32 when f32dx).
cudaError_t launch_prologue_bwd_f32dy(const rdn_prologue_args &a, bool f32dx, cudaStream_t s);

// Sequences and record slots of a call: B sequences of T tokens with B * H *
// ceil(T/64) records, or num_seqs packed sequences whose sum over s of
// ceil(len_s/64) <= num_seqs + ceil(T/64) chunks bounds the records per head.
inline int call_seqs(const rdn_fwd_args &a) { return a.cu_seqlens ? a.num_seqs : a.B; }
inline long long call_records(const rdn_fwd_args &a) {
  const long long nc = (a.T + kChunk - 1) / kChunk;
  return a.cu_seqlens ? (long long)a.H * (a.num_seqs + nc) : (long long)a.B * a.H * nc;
}
// bytes of the device sequence table (FwdParams::seq) in a workspace
inline size_t seq_table_bytes(const rdn_fwd_args &a) {
  return a.cu_seqlens ? ((sizeof(long long) * 2 * ((size_t)a.num_seqs + 1) + 255) & ~(size_t)255) : 0;
}
// Fill seq (seq_table_bytes) from the caller's cu_seqlens, clamping it into a
// valid table; one small kernel on s.
cudaError_t launch_seq_table(const rdn_fwd_args &a, long long *seq, cudaStream_t s);

struct FwdPlan {
  int NC;                // chunks per sequence
  size_t prep_bytes;     // per-chunk precomputed matrices
  size_t total_bytes;    // workspace the forward needs
};
FwdPlan plan_fwd(const rdn_fwd_args &a, int variant);
cudaError_t launch_fwd(const rdn_fwd_args &a, int variant, cudaStream_t s);

struct BwdPlan {
  size_t total_bytes;
};
BwdPlan plan_bwd(const rdn_bwd_args &a, int variant);
cudaError_t launch_bwd(const rdn_bwd_args &a, int variant, cudaStream_t s);
}  // namespace rdn
