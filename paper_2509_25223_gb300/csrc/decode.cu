// decode.cu -- single-token recurrent step of RLA / RDN (Section 3.4 at one t),
// states updated in place.
//
// Memory-bound: each step reads S and R [Dk][Dv] fp32 once and writes them
// once (4*Dk*Dv*4 bytes per (n,h)); everything else is < 1 KB.  One CTA
// handles one (n, h) and a 64-column slice of d_v.  Thread (rg, cg) owns
// rows rg*RPT .. rg*RPT+RPT-1 and columns 4cg .. 4cg+3 of the slice, keeps
// them in registers between the read and the write (128-bit, coalesced,
// evict-first), and the four read-outs
//     p = S^T k,  sq = S^T q,  rk = R^T k,  rq = R^T q
// are reduced over d_k with a shuffle (two row groups per warp) and a
// shared-memory pass over the eight warps.  Per column j then
//     r  = clip(v - p)                                   (Section 3.3)
//     e  = v - a p   (RDN) | v (RLA)      S' = a S + beta k e^T
//     e2 = r - a rk  (RDN) | r (RLA)      R' = a R + gam  k e2^T
//     o  = a sq + gam (q^T R') = a sq + gam (a rq + gam (k.q) e2)
// which is the right (RDN) / left (RLA) formulation of Section 3.4 with the
// delta-rule product expanded: a S (I - b k k^T) + b k v^T = a S + b k (v - a S^T k)^T.
// With RDN_FLAG_QK_NORM the rows of q and k are the raw x, turned into
// y = SiLU(x) / max(||SiLU(x)||, eps) here (held in the input dtype, as the
// forward holds them) before the step.
// The variant flags change the step as in the chunk kernels: r = resid(v - a p)
// (decayed residual), c tanh(x / c) (tanh residual), R' = k r^T without
// reading R (stateless correction, o's correction term gam (k.q) r), and
// o = sq + q^T R' (plain combine).
#include "common.cuh"

namespace rdn {
namespace {

constexpr int kDecThreads = 256;
constexpr int kSliceCols = 64;  // columns of d_v per CTA

template <int D, bool RDN_VARIANT, typename InT>
__global__ void __launch_bounds__(kDecThreads, 2)
decode_kernel(int H, const InT *__restrict__ q, const InT *__restrict__ k,
              const InT *__restrict__ v, const float *__restrict__ g,
              const float *__restrict__ beta, const float *__restrict__ gam,
              float clip, float scale, float *__restrict__ S, float *__restrict__ R,
              InT *__restrict__ o, unsigned mods, bool qkn, float qk_eps) {
  constexpr int RPT = D / 16;             // rows per thread (16 row groups)
  constexpr int NSLICE = D / kSliceCols;  // column slices per (n,h)
  __shared__ float q_s[D], k_s[D];
  __shared__ float red[8][4][kSliceCols];  // per-warp partial read-outs
  __shared__ float tot[4][kSliceCols];
  __shared__ float kq_s;
  __shared__ float nrm_s[2];

  const int nh = blockIdx.x / NSLICE;
  const int slice = blockIdx.x % NSLICE;
  const int tid = threadIdx.x;
  const int cg = tid & 15, rg = tid >> 4;
  const int warp = tid >> 5;
  const size_t sbase = (size_t)nh * D * D + (size_t)slice * kSliceCols + 4 * cg;
  const bool dec_res = mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = mods & RDN_FLAG_PLAIN_COMBINE;
  const bool tnh = mods & RDN_FLAG_TANH_RESIDUAL;
  const bool stl = mods & RDN_FLAG_STATELESS_AUX;

  // issue the state loads first: they are the whole cost of the step
  float4 s_reg[RPT], r_reg[RPT];
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const size_t off = sbase + (size_t)(rg * RPT + i) * D;
    s_reg[i] = __ldcs(reinterpret_cast<const float4 *>(S + off));
    r_reg[i] = stl ? make_float4(0.f, 0.f, 0.f, 0.f)  // (the stateless R is not read)
                   : __ldcs(reinterpret_cast<const float4 *>(R + off));
  }
  if (!qkn) {
    for (int i = tid; i < D; i += kDecThreads) {
      q_s[i] = scale * to_f32(q[(size_t)nh * D + i]);
      k_s[i] = to_f32(k[(size_t)nh * D + i]);
    }
  } else {  // warp 0: q's row, warp 1: k's row
    if (warp < 2) {
      const InT *x = (warp == 0 ? q : k) + (size_t)nh * D;
      float u[D / 32], ss = 0.f;
#pragma unroll
      for (int i = 0; i < D / 32; ++i) {
        const float xi = to_f32(x[(tid & 31) + 32 * i]);
        u[i] = xi * __fdividef(1.f, 1.f + __expf(-xi));
        ss = fmaf(u[i], u[i], ss);
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
      const float inv = 1.f / fmaxf(sqrtf(ss), qk_eps);
      float *dst = warp == 0 ? q_s : k_s;
      const float f = warp == 0 ? scale : 1.f;
#pragma unroll
      for (int i = 0; i < D / 32; ++i) dst[(tid & 31) + 32 * i] = f * to_f32(from_f32<InT>(u[i] * inv));
    }
  }
  __syncthreads();
  if (warp == 0) {
    float s = 0.f;
    for (int i = tid; i < D; i += 32) s += q_s[i] * k_s[i];
#pragma unroll
    for (int off = 16; off; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (tid == 0) kq_s = s;
  }

  float acc[4][4];  // [p, sq, rk, rq][column]
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[a][c] = 0.f;
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const float ki = k_s[rg * RPT + i], qi = q_s[rg * RPT + i];
    const float sv[4] = {s_reg[i].x, s_reg[i].y, s_reg[i].z, s_reg[i].w};
    const float rv[4] = {r_reg[i].x, r_reg[i].y, r_reg[i].z, r_reg[i].w};
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      acc[0][c] = fmaf(ki, sv[c], acc[0][c]);
      acc[1][c] = fmaf(qi, sv[c], acc[1][c]);
      acc[2][c] = fmaf(ki, rv[c], acc[2][c]);
      acc[3][c] = fmaf(qi, rv[c], acc[3][c]);
    }
  }
  // the two row groups of a warp share cg: fold them with one shuffle
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[a][c] += __shfl_xor_sync(0xffffffffu, acc[a][c], 16);
  if ((tid & 31) < 16) {
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int c = 0; c < 4; ++c) red[warp][a][4 * cg + c] = acc[a][c];
  }
  __syncthreads();
  {  // 256 threads = 4 quantities x 64 columns: each sums the eight warps
    const int a = tid >> 6, col = tid & 63;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += red[w][a][col];
    tot[a][col] = s;
  }
  __syncthreads();

  const float alpha = __expf(g[nh]);
  const float b = beta[nh], gm = gam[nh];
  const float kq = kq_s;
  float e[4], e2[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    const int col = 4 * cg + c;
    const float vj = to_f32(v[(size_t)nh * D + slice * kSliceCols + col]);
    const float p = tot[0][col], rk = tot[2][col];
    const float r = resid_map(vj - (dec_res ? alpha * p : p), clip, tnh);
    e[c] = RDN_VARIANT ? vj - alpha * p : vj;
    e2[c] = stl ? r : RDN_VARIANT ? r - alpha * rk : r;
    if (rg == 0) {
      // q^T R' = a rq + gam (k.q) e2, or (k.q) r for the stateless R' = k r^T
      const float qr = stl ? kq * r : alpha * tot[3][col] + gm * kq * e2[c];
      const float oj = plain ? tot[1][col] + qr : alpha * tot[1][col] + gm * qr;
      o[(size_t)nh * D + slice * kSliceCols + col] = from_f32<InT>(oj);
    }
  }
  // R' = a R + gam k e2^T, or k r^T for the stateless correction
  const float ra = stl ? 0.f : alpha, rgm = stl ? 1.f : gm;
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const float ki = k_s[rg * RPT + i];
    const float bk = b * ki, gk = rgm * ki;
    float4 sn, rn;
    sn.x = fmaf(alpha, s_reg[i].x, bk * e[0]);
    sn.y = fmaf(alpha, s_reg[i].y, bk * e[1]);
    sn.z = fmaf(alpha, s_reg[i].z, bk * e[2]);
    sn.w = fmaf(alpha, s_reg[i].w, bk * e[3]);
    rn.x = fmaf(ra, r_reg[i].x, gk * e2[0]);
    rn.y = fmaf(ra, r_reg[i].y, gk * e2[1]);
    rn.z = fmaf(ra, r_reg[i].z, gk * e2[2]);
    rn.w = fmaf(ra, r_reg[i].w, gk * e2[3]);
    const size_t off = sbase + (size_t)(rg * RPT + i) * D;
    __stcs(reinterpret_cast<float4 *>(S + off), sn);
    __stcs(reinterpret_cast<float4 *>(R + off), rn);
  }
}

template <int D, typename InT>
cudaError_t launch_decode_t(const rdn_decode_args &a, cudaStream_t s) {
  const int grid = a.N * a.H * (D / kSliceCols);
  if (a.variant == 1)
    RDN_LAUNCH("decode", s,
               decode_kernel<D, true, InT><<<grid, kDecThreads, 0, s>>>(
                   a.H, (const InT *)a.q, (const InT *)a.k, (const InT *)a.v, a.g, a.beta,
                   a.gamma, a.clip, a.scale, a.S, a.R, (InT *)a.o, a.flags & RDN_FLAG_VARIANTS,
                   (a.flags & RDN_FLAG_QK_NORM) != 0, a.qk_eps));
  else
    RDN_LAUNCH("decode", s,
               decode_kernel<D, false, InT><<<grid, kDecThreads, 0, s>>>(
                   a.H, (const InT *)a.q, (const InT *)a.k, (const InT *)a.v, a.g, a.beta,
                   a.gamma, a.clip, a.scale, a.S, a.R, (InT *)a.o, a.flags & RDN_FLAG_VARIANTS,
                   (a.flags & RDN_FLAG_QK_NORM) != 0, a.qk_eps));
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode(const rdn_decode_args &a, cudaStream_t s) {
  if (a.dtype == RDN_BF16)
    return a.Dk == 128 ? launch_decode_t<128, __nv_bfloat16>(a, s)
                       : launch_decode_t<64, __nv_bfloat16>(a, s);
  return a.Dk == 128 ? launch_decode_t<128, float>(a, s) : launch_decode_t<64, float>(a, s);
}

}  // namespace rdn
