// prologue.cu -- the query / key activation and normalisation that precede the
// recurrence (Section 3.4 omits them from its equations): per row of D
//     u = SiLU(x) = x sigmoid(x),   y = u / max(||u||_2, eps)
// and its backward
//     du = (dy - y <y, dy>) / ||u||   (||u|| > eps;  du = dy / eps otherwise)
//     dx = du * sigmoid(x) (1 + x (1 - sigmoid(x))).
//
// Memory-bound (read x, write y; the backward reads x and dy and writes dx,
// recomputing u and the norm instead of saving them).  In the forward each
// lane holds 16 consecutive bytes of a row (one 16-byte access, kept packed
// in registers until used), so a row takes D * size / 16 lanes and a warp has
// 2 to 8 rows per access; the backward, which holds x and dy, gives a row a
// whole warp (D / 32 elements per lane, fewer registers, more warps).  Four
// accesses are in flight per warp; the row's norm and <y, dy> are reduced
// with shuffles within its lanes; q and k are the two rows of the grid
// (blockIdx.y), each a grid-stride range.  Loads and stores are streaming
// (every element is touched once).
#include "common.cuh"

namespace rdn {
namespace {

constexpr int kProThreads = 256;
constexpr int kRowsInFlight = 4;  // rows whose loads a warp issues together
constexpr int kWaves = 2;         // resident CTAs per SM x kWaves in the grid

template <typename T, int E>
struct Vec;
template <>
struct Vec<float, 4> {
  using Raw = float4;
  __device__ static Raw ldr(const float *p) { return __ldcs(reinterpret_cast<const float4 *>(p)); }
  __device__ static void unpack(const Raw &a, float (&v)[4]) {
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  }
  __device__ static void st(float *p, const float (&v)[4]) {
    __stcs(reinterpret_cast<float4 *>(p), make_float4(v[0], v[1], v[2], v[3]));
  }
};
template <>
struct Vec<float, 2> {
  using Raw = float2;
  __device__ static Raw ldr(const float *p) { return __ldcs(reinterpret_cast<const float2 *>(p)); }
  __device__ static void unpack(const Raw &a, float (&v)[2]) {
    v[0] = a.x; v[1] = a.y;
  }
  __device__ static void st(float *p, const float (&v)[2]) {
    __stcs(reinterpret_cast<float2 *>(p), make_float2(v[0], v[1]));
  }
};
template <>
struct Vec<__nv_bfloat16, 4> {
  using Raw = uint2;
  __device__ static Raw ldr(const __nv_bfloat16 *p) { return __ldcs(reinterpret_cast<const uint2 *>(p)); }
  __device__ static void unpack(const Raw &a, float (&v)[4]) {
    const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162 *>(&a.x);
    const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162 *>(&a.y);
    v[0] = __low2float(lo); v[1] = __high2float(lo); v[2] = __low2float(hi); v[3] = __high2float(hi);
  }
  __device__ static void st(__nv_bfloat16 *p, const float (&v)[4]) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(v[0], v[1]), hi = __floats2bfloat162_rn(v[2], v[3]);
    uint2 a;
    a.x = *reinterpret_cast<const uint32_t *>(&lo);
    a.y = *reinterpret_cast<const uint32_t *>(&hi);
    __stcs(reinterpret_cast<uint2 *>(p), a);
  }
};
template <>
struct Vec<__nv_bfloat16, 8> {
  using Raw = uint4;
  __device__ static Raw ldr(const __nv_bfloat16 *p) { return __ldcs(reinterpret_cast<const uint4 *>(p)); }
  __device__ static void unpack(const Raw &a, float (&v)[8]) {
    const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&w[i]);
      v[2 * i] = __low2float(b);
      v[2 * i + 1] = __high2float(b);
    }
  }
  __device__ static void st(__nv_bfloat16 *p, const float (&v)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 b = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
      w[i] = *reinterpret_cast<const uint32_t *>(&b);
    }
    __stcs(reinterpret_cast<uint4 *>(p), make_uint4(w[0], w[1], w[2], w[3]));
  }
};
template <>
struct Vec<__nv_bfloat16, 2> {
  using Raw = unsigned;
  __device__ static Raw ldr(const __nv_bfloat16 *p) { return __ldcs(reinterpret_cast<const unsigned *>(p)); }
  __device__ static void unpack(const Raw &a, float (&v)[2]) {
    const __nv_bfloat162 x = *reinterpret_cast<const __nv_bfloat162 *>(&a);
    v[0] = __low2float(x); v[1] = __high2float(x);
  }
  __device__ static void st(__nv_bfloat16 *p, const float (&v)[2]) {
    const __nv_bfloat162 x = __floats2bfloat162_rn(v[0], v[1]);
    __stcs(reinterpret_cast<unsigned *>(p), *reinterpret_cast<const unsigned *>(&x));
  }
};

// sum over the LPR lanes of a row (aligned groups of LPR lanes)
template <int LPR>
__device__ __forceinline__ float row_sum(float v) {
#pragma unroll
  for (int off = LPR / 2; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

struct ProP {
  long long rows;  // rows per tensor (blockIdx.y picks the tensor: q, then k)
  float eps;
  const void *x[2], *dy[2];
  void *o[2];  // y (forward) or dx (backward)
};

// GT, OT: the element types of dy and of dx (InT, or fp32 for gradients the
// library keeps in fp32 before this step, and for fp32 results)
template <typename InT, int D, bool BWD, typename GT = InT, typename OT = InT>
__global__ void __launch_bounds__(kProThreads) prologue_kernel(ProP p) {
  // elements per lane: one 16-byte access (the backward, which holds x and
  // dy, one warp per row: D / 32 elements per lane, fewer registers)
  constexpr int E = BWD ? D / 32 : 16 / (int)sizeof(InT);
  constexpr int LPR = D / E;                 // lanes per row
  constexpr int RPW = 32 / LPR;              // rows per warp access
  constexpr int ROWS = kRowsInFlight * RPW;  // rows a warp has in flight
  using V = Vec<InT, E>;
  using VG = Vec<GT, E>;
  using VO = Vec<OT, E>;
  const int lane = threadIdx.x & 31, sub = lane / LPR, li = lane % LPR;
  const long long warp = ((long long)blockIdx.x * kProThreads + threadIdx.x) >> 5;
  const long long nwarps = ((long long)gridDim.x * kProThreads) >> 5;
  const InT *X = reinterpret_cast<const InT *>(p.x[blockIdx.y]);
  const GT *DY = reinterpret_cast<const GT *>(p.dy[blockIdx.y]);
  OT *O = reinterpret_cast<OT *>(p.o[blockIdx.y]);
  for (long long base = warp * ROWS; base < p.rows; base += nwarps * ROWS) {
    typename V::Raw xr[kRowsInFlight];  // packed until used
    typename VG::Raw gr[kRowsInFlight];
    // the loads of all rows first
#pragma unroll
    for (int u = 0; u < kRowsInFlight; ++u) {
      const long long r = base + u * RPW + sub;
      xr[u] = typename V::Raw{};
      gr[u] = typename VG::Raw{};
      if (r < p.rows) {
        const size_t off = (size_t)r * D + li * E;
        xr[u] = V::ldr(X + off);
        if (BWD) gr[u] = VG::ldr(DY + off);
      }
    }
#pragma unroll
    for (int u = 0; u < kRowsInFlight; ++u) {
      const long long r = base + u * RPW + sub;  // (rows past the end: computed, not stored)
      float x[E], g[E], s[E], uu[E], ss = 0.f;
      V::unpack(xr[u], x);
      if (BWD) VG::unpack(gr[u], g);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        s[e] = __fdividef(1.f, 1.f + __expf(-x[e]));  // (2-ulp divide: issue-bound loop)
        uu[e] = x[e] * s[e];
        ss = fmaf(uu[e], uu[e], ss);
      }
      const float n = sqrtf(row_sum<LPR>(ss));
      const float m = fmaxf(n, p.eps), inv = 1.f / m;
      float out[E];
      if (!BWD) {
#pragma unroll
        for (int e = 0; e < E; ++e) out[e] = uu[e] * inv;
      } else {
        float dot = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e) dot = fmaf(uu[e] * inv, g[e], dot);
        dot = row_sum<LPR>(dot);
        const bool big = n > p.eps;
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const float du = big ? (g[e] - uu[e] * inv * dot) * inv : g[e] * inv;
          out[e] = du * s[e] * (1.f + x[e] * (1.f - s[e]));
        }
      }
      if (r < p.rows) VO::st(O + (size_t)r * D + li * E, out);
    }
  }
}

template <typename InT, int D, typename GT = InT, typename OT = InT>
cudaError_t launch_t(const ProP &p, bool bwd, cudaStream_t s) {
  int dev = 0, nsm = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  const int rows_per_warp = bwd ? kRowsInFlight : kRowsInFlight * 32 / (D * (int)sizeof(InT) / 16);
  const int nt = p.x[1] ? 2 : 1;  // tensors: grid.y
  const long long warps = (p.rows + rows_per_warp - 1) / rows_per_warp;
  const long long want = (warps + kProThreads / 32 - 1) / (kProThreads / 32);
  int occ = 0;  // a few waves of resident CTAs, grid-stride beyond
  e = bwd ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, prologue_kernel<InT, D, true, GT, OT>, kProThreads, 0)
          : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, prologue_kernel<InT, D, false>, kProThreads, 0);
  if (e != cudaSuccess) return e;
  const long long cap = ((long long)nsm * (occ > 0 ? occ : 1) * kWaves + nt - 1) / nt;
  const dim3 grid((unsigned)(want < cap ? want : cap), nt);
  if (bwd)
    RDN_LAUNCH("qk_prologue_bwd", s, prologue_kernel<InT, D, true, GT, OT><<<grid, kProThreads, 0, s>>>(p));
  else
    RDN_LAUNCH("qk_prologue", s, prologue_kernel<InT, D, false><<<grid, kProThreads, 0, s>>>(p));
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prologue(const rdn_prologue_args &a, bool bwd, cudaStream_t s) {
  ProP p;
  p.rows = a.rows;
  p.eps = a.eps;
  for (int i = 0; i < 2; ++i) {
    p.x[i] = a.x[i];
    p.dy[i] = bwd ? a.dy[i] : nullptr;
    p.o[i] = bwd ? a.dx[i] : a.y[i];
  }
  if (a.dtype == RDN_BF16)
    return a.D == 128 ? launch_t<__nv_bfloat16, 128>(p, bwd, s) : launch_t<__nv_bfloat16, 64>(p, bwd, s);
  return a.D == 128 ? launch_t<float, 128>(p, bwd, s) : launch_t<float, 64>(p, bwd, s);
}

cudaError_t launch_prologue_bwd_f32dy(const rdn_prologue_args &a, bool f32dx, cudaStream_t s) {
  ProP p;
  p.rows = a.rows;
  p.eps = a.eps;
  for (int i = 0; i < 2; ++i) {
    p.x[i] = a.x[i];
    p.dy[i] = a.dy[i];
    p.o[i] = a.dx[i];
  }
  if (a.dtype == RDN_BF16) {
    if (f32dx)
      return a.D == 128 ? launch_t<__nv_bfloat16, 128, float, float>(p, true, s)
                        : launch_t<__nv_bfloat16, 64, float, float>(p, true, s);
    return a.D == 128 ? launch_t<__nv_bfloat16, 128, float>(p, true, s)
                      : launch_t<__nv_bfloat16, 64, float>(p, true, s);
  }
  return a.D == 128 ? launch_t<float, 128>(p, true, s) : launch_t<float, 64>(p, true, s);
}

}  // namespace rdn
