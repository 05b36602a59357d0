// chunk_fwd.cu -- chunkwise-parallel forward of RLA / RDN (Section 3.4),
// fp32 SIMT path.
//
// Chunk algebra (C = 64 tokens; b_t = in-chunk cumulative log-decay,
// Gam_t = exp(b_t), Gprev_t = exp(b_{t-1}), b_0 = 0; states stored [d_k][d_v]):
//
//   RDN writes the delta rule as S_t = a_t S_{t-1} + beta_t k_t e_t^T with the
//   delta error e_t = v_t - a_t S_{t-1}^T k_t (Section 2.2).  Unrolling the
//   chunk gives (I + A) E = V - diag(Gam) K S0 with the strictly lower
//   A[t,i] = exp(b_t - b_i) beta_i (k_t.k_i), so E = T (V - diag(Gam) K S0),
//   T = (I + A)^-1 (the UT form of the WY representation).  RLA: E = V.
//
//   P   = diag(Gprev) K S0 + Ap E,   Ap[t,i] = exp(b_{t-1}-b_i) beta_i (k_t.k_i), i<t
//         (P_t = S_{t-1}^T k_t, the undecayed prediction of Section 3.3)
//   Ob  = diag(Gam) Q S0 + Mq E,     Mq[t,i] = exp(b_t-b_i) beta_i (q_t.k_i), i<t
//         (Ob_t = a_t S_{t-1}^T q_t, the base prediction)
//   S_C = Gam_C S0 + K^T diag(beta_i exp(b_C - b_i)) E
//   r   = clip(V - P, -c, c)                                   (Section 3.3)
//   the auxiliary pass repeats this with values r, rate gamma, state R; its
//   read-out includes token t:  Oa = diag(Gam) Q R0 + M2 E2,
//         M2[t,i] = exp(b_t-b_i) gamma_i (q_t.k_i), i<=t
//   o   = Ob + diag(gamma) Oa.
//
// Kernel 1 (chunk_prep): one CTA per chunk -- everything that does not depend
// on the state: the Gram matrices, the masked/decayed matrices Ap, Mq, M2 and
// (RDN) the two unit-lower inverses T_beta, T_gamma by forward substitution.
// Kernel 2 (chunk_scan): one CTA per (b, h, 32-column slice of d_v) -- the
// sequential pass over chunks carrying S and R slices in shared memory.  Each
// value column is independent (the clip is elementwise), so slicing d_v is
// exact; only the prep work is shared between slices.
#include <type_traits>

#include "chunk_common.cuh"
#include "status.cuh"

namespace rdn {
namespace {

// ---------------------------------------------------------------- kernel 1
// Image writer: element (r, c) of a 64-column chunk matrix, value x, into a
// K-major 128B-swizzled bf16 hi / lo pair (lo tile `lo_off` bytes after hi).
__device__ __forceinline__ void img_put(uint8_t *tile, uint32_t lo_off, int r, int c, float x) {
  const uint32_t o = (uint32_t)(r * 128 + ((((c >> 3) ^ (r & 7)) & 7) << 4) + (c & 7) * 2);
  const __nv_bfloat16 hi = __float2bfloat16_rn(x);
  *reinterpret_cast<__nv_bfloat16 *>(tile + o) = hi;
  *reinterpret_cast<__nv_bfloat16 *>(tile + lo_off + o) = __float2bfloat16_rn(x - __bfloat162float(hi));
}

template <int DK, bool RDNV, typename InT, bool IMG>
__global__ void __launch_bounds__(kThreads, 1) chunk_prep_kernel(FwdParams p) {
  constexpr int LDK = DK + 1;
  constexpr int LDC = C + 1;
  extern __shared__ float sm[];
  float *Ks = sm;                 // [C][LDK]
  float *Qs = Ks + C * LDK;       // [C][LDK]
  float *KK = Qs + C * LDK;       // [C][LDC]
  float *QK = KK + C * LDC;       // [C][LDC]
  float *Ab = QK + C * LDC;       // [C][LDC]
  float *Ag = Ab + C * LDC;       // [C][LDC]
  float *Tb = Ag + C * LDC;       // [C][LDC]
  float *Tg = Tb + C * LDC;       // [C][LDC]
  float *cum = Tg + C * LDC;      // [C]
  float *cprev = cum + C;         // [C]
  float *bet = cprev + C;         // [C]
  float *gam = bet + C;           // [C]
  float *gg = gam + C;            // [C]
  float *Wsc = gg + C;            // [2][3*256] scratch of the blocked inverse

  const long long chunk = blockIdx.x;
  if (chunk >= total_records(p)) return;  // (packed sequences: the grid covers the bound)
  int sq, h, c;
  rec_decode(p, chunk, sq, h, c);
  const SeqSpan sp = seq_span(p, sq, h);
  const int t0 = c * C;
  const int n = min(C, sp.len - t0);
  const int tid = threadIdx.x;
  const InT *q = (const InT *)p.q;
  const InT *k = (const InT *)p.k;

  for (int e = tid; e < C * DK; e += kThreads) {
    const int t = e / DK, d = e % DK;
    float kv = 0.f, qv = 0.f;
    if (t < n) {
      const size_t off = ((size_t)(sp.tok0 + t0 + t) * p.H + h) * DK + d;
      kv = to_f32(k[off]);
      qv = p.scale * to_f32(q[off]);
    }
    Ks[t * LDK + d] = kv;
    Qs[t * LDK + d] = qv;
  }
  if (tid < C) {
    const int t = tid;
    float gv = 0.f, bv = 0.f, mv = 0.f;
    if (t < n) {
      const size_t off = (size_t)(sp.tok0 + t0 + t) * p.H + h;
      gv = p.g[off];
      bv = p.beta[off];
      mv = p.gamma[off];
    }
    gg[t] = gv;
    bet[t] = bv;
    gam[t] = mv;
  }
  __syncthreads();
  if (tid == 0) {
    float s = 0.f;
    for (int t = 0; t < C; ++t) {
      cprev[t] = s;
      s += gg[t];
      cum[t] = s;
    }
  }
  // Gram matrices K K^T and Q K^T
  {
    using MM = BlockMM<C, C, DK>;
    float acc[MM::RPT];
    MM::run(Ks, LDK, 1, Ks, 1, LDK, acc);
#pragma unroll
    for (int i = 0; i < MM::RPT; ++i) KK[MM::row(i) * LDC + MM::col()] = acc[i];
    MM::run(Qs, LDK, 1, Ks, 1, LDK, acc);
#pragma unroll
    for (int i = 0; i < MM::RPT; ++i) QK[MM::row(i) * LDC + MM::col()] = acc[i];
  }
  __syncthreads();
  float *rec = p.ws + (size_t)chunk * kRecFloats;
  // variants: the decayed residual predicts with a_t S_{t-1} k_t, so Ap takes
  // the decay to t (not t-1); the plain combine reads S_{t-1} q_t, so Mq takes
  // the decay to t-1; the stateless correction reads r_t (q_t.k_t) alone
  const bool dec_res = p.mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = p.mods & RDN_FLAG_PLAIN_COMBINE;
  const bool stl = p.mods & RDN_FLAG_STATELESS_AUX;
  for (int e = tid; e < C * C; e += kThreads) {
    const int t = e / C, i = e % C;
    float ap = 0.f, mq = 0.f, m2 = 0.f, ab = 0.f, ag = 0.f;
    if (i <= t) {
      const float dec = expf(cum[t] - cum[i]);
      m2 = stl ? (i == t ? QK[t * LDC + i] : 0.f) : dec * gam[i] * QK[t * LDC + i];
      if (i < t) {
        const float decp = expf(cprev[t] - cum[i]);
        ap = (dec_res ? dec : decp) * bet[i] * KK[t * LDC + i];
        mq = (plain ? decp : dec) * bet[i] * QK[t * LDC + i];
        ab = dec * bet[i] * KK[t * LDC + i];
        ag = dec * gam[i] * KK[t * LDC + i];
      }
    }
    if (IMG) {
      uint8_t *img = reinterpret_cast<uint8_t *>(rec);
      img_put(img + IMG_APMQ, 16384, t, i, ap);
      img_put(img + IMG_APMQ, 16384, 64 + t, i, mq);
      img_put(img + IMG_M2, 8192, t, i, gam[t] * m2);  // the image holds diag(gamma) M2
    } else {
      rec[OFF_AP + e] = ap;
      rec[OFF_MQ + e] = mq;
      rec[OFF_M2 + e] = m2;
    }
    if (RDNV) {
      Ab[t * LDC + i] = ab;
      Ag[t * LDC + i] = ag;
    }
  }
  if (tid < C) {
    const int t = tid;
    const float cC = cum[C - 1];
    rec[OFF_VEC + V_GAM + t] = expf(cum[t]);
    rec[OFF_VEC + V_GPREV + t] = expf(cprev[t]);
    rec[OFF_VEC + V_ALPHA + t] = expf(gg[t]);
    rec[OFF_VEC + V_WS + t] = bet[t] * expf(cC - cum[t]);
    // (stateless correction: R at the chunk end is k r^T of its last token)
    rec[OFF_VEC + V_WR + t] = stl ? (t == n - 1 ? 1.f : 0.f) : gam[t] * expf(cC - cum[t]);
    if (t == 0) rec[OFF_VEC + V_GAMC] = expf(cC);
  }
  if (RDNV) {
    __syncthreads();
    // (I + A)^-1 by 16 x 16 blocks: threads 0..127 invert I + A_beta,
    // threads 128..255 invert I + A_gamma.
    {
      const int g = tid & 127;
      const float *A = tid < 128 ? Ab : Ag;
      float *Tm = tid < 128 ? Tb : Tg;
      float *W = Wsc + (tid < 128 ? 0 : 768);
      inv_diag_blocks(A, Tm, LDC, g);
      for (int i = 1; i < 4; ++i) {
        __syncthreads();
        inv_block_row_w(A, Tm, W, LDC, i, g);
        __syncthreads();
        inv_block_row_t(Tm, W, LDC, i, g);
      }
    }
    __syncthreads();
    for (int e = tid; e < C * C; e += kThreads) {
      const int t = e / C, i = e % C;
      if (IMG) {
        uint8_t *img = reinterpret_cast<uint8_t *>(rec);
        img_put(img + IMG_TB, 8192, t, i, Tb[t * LDC + i]);
        img_put(img + IMG_TG, 8192, t, i, Tg[t * LDC + i]);
      } else {
        rec[OFF_TB + e] = Tb[t * LDC + i];
        rec[OFF_TG + e] = Tg[t * LDC + i];
      }
    }
  } else if (IMG) {
    // RLA has no delta rule: T_beta = T_gamma = I, which the tensor-core
    // backward reads in their place
    for (int e = tid; e < C * C; e += kThreads) {
      const int t = e / C, i = e % C;
      uint8_t *img = reinterpret_cast<uint8_t *>(rec);
      img_put(img + IMG_TB, 8192, t, i, t == i ? 1.f : 0.f);
      img_put(img + IMG_TG, 8192, t, i, t == i ? 1.f : 0.f);
    }
  }
}

// ---------------------------------------------------------------- kernel 2
constexpr int kScanThreads = 512;  // threads of a scan CTA (latency bound: 16 warps)

template <int DK, bool RDNV, typename InT>
__global__ void __launch_bounds__(kScanThreads, 1) chunk_scan_kernel(FwdParams p) {
  constexpr int DV = DK;
  extern __shared__ float sm[];
  float *Ks = sm;                 // [C][DK]
  float *Qs = Ks + C * DK;        // [C][DK]
  float *Ss = Qs + C * DK;        // [DK][kDVS]
  float *Rs = Ss + DK * kDVS;     // [DK][kDVS]
  float *Vs = Rs + DK * kDVS;     // [C][kDVS]
  float *CC = Vs + C * kDVS;      // [C][C]
  float *KS = CC + C * C;         // [C][kDVS]
  float *QS = KS + C * kDVS;
  float *Es = QS + C * kDVS;
  float *Ps = Es + C * kDVS;
  float *Ob = Ps + C * kDVS;
  float *Ws = Ob + C * kDVS;
  float *vec = Ws + C * kDVS;     // [6*C]

  const int bh = blockIdx.x;
  const int h = bh % p.H;
  const SeqSpan sp = seq_span(p, bh / p.H, h);
  const int j0 = blockIdx.y * kDVS;
  const int tid = threadIdx.x;
  const InT *q = (const InT *)p.q;
  const InT *k = (const InT *)p.k;
  const InT *v = (const InT *)p.v;
  InT *o = (InT *)p.o;
  const float clip = p.clip;
  const bool dec_res = p.mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = p.mods & RDN_FLAG_PLAIN_COMBINE;
  const bool tnh = p.mods & RDN_FLAG_TANH_RESIDUAL;
  const bool stl = p.mods & RDN_FLAG_STATELESS_AUX;
  const bool rdn_aux = RDNV && !stl;  // the auxiliary pass runs the delta rule

  const size_t sbase = (size_t)bh * DK * DV;
  for (int e = tid; e < DK * kDVS; e += kScanThreads) {
    const int i = e / kDVS, jj = e % kDVS;
    Ss[e] = p.S0 ? p.S0[sbase + (size_t)i * DV + j0 + jj] : 0.f;
    Rs[e] = p.R0 ? p.R0[sbase + (size_t)i * DV + j0 + jj] : 0.f;
  }

  for (int c = 0; c < sp.nc; ++c) {
    const int t0 = c * C;
    const int n = min(C, sp.len - t0);
    const float *rec = p.ws + (size_t)(sp.rbase + c) * kRecFloats;
    __syncthreads();  // previous chunk done with every buffer
    if (p.S_chunks) {
      float *sc = p.S_chunks + (size_t)(sp.rbase + c) * DK * DV;
      float *rc = p.R_chunks + (size_t)(sp.rbase + c) * DK * DV;
      for (int e = tid; e < DK * kDVS; e += kScanThreads) {
        const int i = e / kDVS, jj = e % kDVS;
        sc[(size_t)i * DV + j0 + jj] = Ss[e];
        rc[(size_t)i * DV + j0 + jj] = Rs[e];
      }
    }
    for (int e = tid; e < C * DK; e += kScanThreads) {
      const int t = e / DK, d = e % DK;
      float kv = 0.f, qv = 0.f;
      if (t < n) {
        const size_t off = ((size_t)(sp.tok0 + t0 + t) * p.H + h) * DK + d;
        kv = to_f32(k[off]);
        qv = p.scale * to_f32(q[off]);
      }
      Ks[e] = kv;
      Qs[e] = qv;
    }
    for (int e = tid; e < C * kDVS; e += kScanThreads) {
      const int t = e / kDVS, jj = e % kDVS;
      Vs[e] = t < n ? to_f32(v[((size_t)(sp.tok0 + t0 + t) * p.H + h) * DV + j0 + jj]) : 0.f;
    }
    for (int e = tid; e < 6 * C; e += kScanThreads) vec[e] = rec[OFF_VEC + e];
    __syncthreads();
    const float *Gam = vec + V_GAM, *Gprev = vec + V_GPREV;
    const float *wS = vec + V_WS, *wR = vec + V_WR;
    const float GamC = vec[V_GAMC];

    using MMk = BlockMM<C, kDVS, DK, kScanThreads>;  // [C x DK] @ [DK x DVS]
    using MMc = BlockMM<C, kDVS, C, kScanThreads>;   // [C x C] @ [C x DVS]
    using MMu = BlockMM<DK, kDVS, C, kScanThreads>;  // [DK x C] @ [C x DVS]
    const int col = MMk::col();
    {
      float a1[MMk::RPT], a2[MMk::RPT];
      MMk::run(Ks, DK, 1, Ss, kDVS, 1, a1);
      MMk::run(Qs, DK, 1, Ss, kDVS, 1, a2);
#pragma unroll
      for (int i = 0; i < MMk::RPT; ++i) {
        const int t = MMk::row(i);
        KS[t * kDVS + col] = a1[i];
        QS[t * kDVS + col] = a2[i];
        if (RDNV) Ws[t * kDVS + col] = Vs[t * kDVS + col] - Gam[t] * a1[i];
      }
    }
    const float *E = Vs;
    if (RDNV) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TB + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, Ws, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) Es[MMc::row(i) * kDVS + col] = a1[i];
      E = Es;
    }
    __syncthreads();
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_AP + e];
    __syncthreads();
    {
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, E, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        // P_t = S_{t-1}^T k_t (decayed residual: a_t S_{t-1}^T k_t)
        const float pt = (dec_res ? Gam[t] : Gprev[t]) * KS[t * kDVS + col] + a1[i];
        Ps[t * kDVS + col] = resid_map(Vs[t * kDVS + col] - pt, clip, tnh);  // r, Section 3.3
      }
    }
    __syncthreads();
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_MQ + e];
    __syncthreads();
    {
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, E, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        Ob[t * kDVS + col] = (plain ? Gprev[t] : Gam[t]) * QS[t * kDVS + col] + a1[i];
      }
    }
    // S_C = Gam_C S0 + K^T diag(wS) E   (W = wS * E)
    for (int e = tid; e < C * kDVS; e += kScanThreads) Ws[e] = wS[e / kDVS] * E[e];
    __syncthreads();
    {
      float a1[MMu::RPT];
      MMu::run(Ks, 1, DK, Ws, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMu::RPT; ++i) {
        const int r = MMu::row(i);
        Ss[r * kDVS + col] = GamC * Ss[r * kDVS + col] + a1[i];
      }
    }
    // auxiliary pass: values r (in Ps), rate gamma, state R
    {
      float a1[MMk::RPT], a2[MMk::RPT];
      MMk::run(Ks, DK, 1, Rs, kDVS, 1, a1);
      MMk::run(Qs, DK, 1, Rs, kDVS, 1, a2);
      __syncthreads();  // every thread done reading Ws / CC of the S pass
#pragma unroll
      for (int i = 0; i < MMk::RPT; ++i) {
        const int t = MMk::row(i);
        QS[t * kDVS + col] = stl ? 0.f : a2[i];  // Q R0 (the stateless R carries nothing)
        if (rdn_aux) Ws[t * kDVS + col] = Ps[t * kDVS + col] - Gam[t] * a1[i];
      }
    }
    const float *E2 = Ps;
    if (rdn_aux) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TG + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, Ws, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) Es[MMc::row(i) * kDVS + col] = a1[i];
      E2 = Es;
    }
    __syncthreads();
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_M2 + e];
    __syncthreads();
    {
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, E2, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        if (t < n) {
          const float gm = plain ? 1.f : p.gamma[(size_t)(sp.tok0 + t0 + t) * p.H + h];
          const float oa = Gam[t] * QS[t * kDVS + col] + a1[i];
          o[((size_t)(sp.tok0 + t0 + t) * p.H + h) * DV + j0 + col] =
              from_f32<InT>(Ob[t * kDVS + col] + gm * oa);
        }
      }
    }
    // R_C = Gam_C R0 + K^T diag(wR) E2
    for (int e = tid; e < C * kDVS; e += kScanThreads) Ws[e] = wR[e / kDVS] * E2[e];
    __syncthreads();
    {
      float a1[MMu::RPT];
      MMu::run(Ks, 1, DK, Ws, kDVS, 1, a1);
#pragma unroll
      for (int i = 0; i < MMu::RPT; ++i) {
        const int r = MMu::row(i);
        Rs[r * kDVS + col] = (stl ? 0.f : GamC) * Rs[r * kDVS + col] + a1[i];
      }
    }
  }
  __syncthreads();
  for (int e = tid; e < DK * kDVS; e += kScanThreads) {
    const int i = e / kDVS, jj = e % kDVS;
    if (p.ST) p.ST[sbase + (size_t)i * DV + j0 + jj] = Ss[e];
    if (p.RT) p.RT[sbase + (size_t)i * DV + j0 + jj] = Rs[e];
  }
}

template <int DK>
constexpr size_t prep_smem() {
  return sizeof(float) * (2 * C * (DK + 1) + 6 * C * (C + 1) + 5 * C + 2 * 768);
}
template <int DK>
constexpr size_t scan_smem() {
  return sizeof(float) * (2 * C * DK + 2 * DK * kDVS + C * kDVS + C * C + 6 * C * kDVS + 6 * C);
}

template <int DK, bool RDNV, typename InT>
cudaError_t launch_t(const FwdParams &p, cudaStream_t s, bool do_prep, bool do_scan,
                     bool img = false) {
  auto prep = img ? chunk_prep_kernel<DK, RDNV, InT, true> : chunk_prep_kernel<DK, RDNV, InT, false>;
  auto scan = chunk_scan_kernel<DK, RDNV, InT>;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(prep, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)prep_smem<DK>())) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(scan, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)scan_smem<DK>())) != cudaSuccess)
    return e;
  if (do_prep) {
    // the images for bf16 inputs and d = 128 come from the tensor-core prep,
    // which also normalises q and k (RDN_FLAG_QK_NORM) as it loads them; for
    // the other preps the prologue kernel writes the normalised copies first
    constexpr bool tc_prep = DK == 128 && std::is_same<InT, __nv_bfloat16>::value;
    const bool use_tc_prep = tc_prep && img && (p.mods & ~kTcVariants) == 0;
    if (p.qk_norm && !use_tc_prep) {
      rdn_prologue_args pa{};
      pa.rows = (long long)p.B * p.T * p.H;
      pa.D = DK;
      pa.dtype = std::is_same<InT, __nv_bfloat16>::value ? RDN_BF16 : RDN_F32;
      pa.eps = p.qk_eps;
      pa.x[0] = p.qraw;
      pa.x[1] = p.kraw;
      pa.y[0] = const_cast<void *>(p.q);
      pa.y[1] = const_cast<void *>(p.k);
      if ((e = launch_prologue(pa, false, s)) != cudaSuccess) return e;
    }
    if (use_tc_prep) {
      if ((e = launch_prep_tc(p, !RDNV, s)) != cudaSuccess) return e;
    } else {
      RDN_LAUNCH("chunk_prep", s, prep<<<(unsigned)p.nrec, kThreads, prep_smem<DK>(), s>>>(p));
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  if (do_scan)
    RDN_LAUNCH("chunk_scan", s, scan<<<dim3(p.nseq * p.H, DK / kDVS), kScanThreads, scan_smem<DK>(), s>>>(p));
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_fwd_parts(const FwdParams &p, int DK, bool rdnv, bool bf16, bool do_prep,
                             bool do_scan, cudaStream_t s) {
  // bf16 inputs with d = 128 (RDN, and RLA with a hi + lo copy of S for its
  // read-outs) run the tensor-core scan; everything else, and the variants,
  // the fp32 SIMT one
  const bool tc_scan = do_scan && fwd_uses_tc(p, DK, bf16);
  cudaError_t e = cudaSuccess;
  // (the tensor-core scan reads the records as shared-memory images)
  if (DK == 128) {
    if (rdnv) e = bf16 ? launch_t<128, true, __nv_bfloat16>(p, s, do_prep, do_scan && !tc_scan, tc_scan)
                       : launch_t<128, true, float>(p, s, do_prep, do_scan);
    else e = bf16 ? launch_t<128, false, __nv_bfloat16>(p, s, do_prep, do_scan && !tc_scan, tc_scan)
                  : launch_t<128, false, float>(p, s, do_prep, do_scan);
  } else {
    if (rdnv) e = bf16 ? launch_t<64, true, __nv_bfloat16>(p, s, do_prep, do_scan)
                       : launch_t<64, true, float>(p, s, do_prep, do_scan);
    else e = bf16 ? launch_t<64, false, __nv_bfloat16>(p, s, do_prep, do_scan)
                  : launch_t<64, false, float>(p, s, do_prep, do_scan);
  }
  if (e != cudaSuccess || !tc_scan) return e;
  return launch_fwd_tc(p, rdnv, s);
}

cudaError_t launch_prep(const FwdParams &p, int DK, bool rdnv, bool bf16, bool img, cudaStream_t s) {
  if (DK == 128) {
    if (rdnv) return bf16 ? launch_t<128, true, __nv_bfloat16>(p, s, true, false, img)
                          : launch_t<128, true, float>(p, s, true, false, img);
    return bf16 ? launch_t<128, false, __nv_bfloat16>(p, s, true, false, img)
                : launch_t<128, false, float>(p, s, true, false, img);
  }
  if (rdnv) return bf16 ? launch_t<64, true, __nv_bfloat16>(p, s, true, false, img)
                        : launch_t<64, true, float>(p, s, true, false, img);
  return bf16 ? launch_t<64, false, __nv_bfloat16>(p, s, true, false, img)
              : launch_t<64, false, float>(p, s, true, false, img);
}

// Block-wide inclusive scan of one value per thread (blockDim.x = 1024).
template <typename Op>
__device__ long long block_incl_scan(long long x, Op op, long long *wsum) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, x, d);
    if (lane >= d) x = op(x, y);
  }
  if (lane == 31) wsum[wid] = x;
  __syncthreads();
  if (wid == 0) {
    long long w = wsum[lane];
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, w, d);
      if (lane >= d) w = op(w, y);
    }
    wsum[lane] = w;
  }
  __syncthreads();
  if (wid > 0) x = op(x, wsum[wid - 1]);
  __syncthreads();  // (wsum is reused by the next call)
  return x;
}

// The packed-sequence table FwdParams::seq from cu_seqlens[0 .. N]: first
// tokens are the running maximum of the entries clamped into [0, T] (with
// entry 0 read as 0 and entry N as T, so the table always covers [0, T) in
// order), first chunks the exclusive prefix sum of ceil(len_s / 64).  One CTA.
__global__ void __launch_bounds__(1024) seq_table_kernel(const int *__restrict__ cu, int N, int T,
                                                         long long *__restrict__ seq) {
  __shared__ long long wsum[32];
  __shared__ long long carry;
  const int tid = threadIdx.x;
  if (tid == 0) carry = 0;
  __syncthreads();
  auto mx = [](long long a, long long b) { return a > b ? a : b; };
  auto add = [](long long a, long long b) { return a + b; };
  for (int base = 0; base <= N; base += 1024) {
    const int s = base + tid;
    long long x = 0;
    if (s <= N) x = s == 0 ? 0 : s == N ? T : min(max(cu[s], 0), T);
    x = mx(block_incl_scan(x, mx, wsum), carry);
    if (s <= N) seq[2 * s] = x;
    if (tid == 1023) carry = x;  // (padding reads 0 and leaves the maximum alone)
    __syncthreads();
  }
  if (tid == 0) carry = 0;
  __syncthreads();  // (also orders the token offsets before they are read back)
  for (int base = 0; base <= N; base += 1024) {
    const int s = base + tid;
    const long long nc = s < N ? (seq[2 * s + 2] - seq[2 * s] + C - 1) / C : 0;
    const long long incl = block_incl_scan(nc, add, wsum) + carry;
    if (s <= N) seq[2 * s + 1] = incl - nc;  // entry N: the total
    if (tid == 1023) carry = incl;
    __syncthreads();
  }
}

cudaError_t launch_seq_table(const rdn_fwd_args &a, long long *seq, cudaStream_t s) {
  RDN_LAUNCH("seq_table", s, seq_table_kernel<<<1, 1024, 0, s>>>(a.cu_seqlens, a.num_seqs, a.T, seq));
  return cudaGetLastError();
}

FwdPlan plan_fwd(const rdn_fwd_args &a, int variant) {
  FwdPlan pl;
  pl.NC = (a.T + C - 1) / C;
  pl.prep_bytes = sizeof(float) * (size_t)kRecFloats;
  const size_t nrec = (size_t)call_records(a);
  // per-chunk records, the saved intermediates if asked for, the normalised
  // q, k (RDN_FLAG_QK_NORM), the packed-sequence table, then a 256-byte tail
  pl.total_bytes = pl.prep_bytes * nrec + seq_table_bytes(a) + 256;
  if (a.flags & RDN_FLAG_SAVE_FOR_BWD)
    pl.total_bytes += saved_layout(nrec, a.Dv, a.flags & RDN_FLAG_TANH_RESIDUAL).bytes;
  pl.total_bytes += qk_norm_bytes(a);  // (after those: qk_norm_offset)
  return pl;
}

cudaError_t launch_fwd(const rdn_fwd_args &a, int variant, cudaStream_t s) {
  const size_t sbytes = sizeof(float) * (size_t)call_seqs(a) * a.H * a.Dk * a.Dv;
  if (a.T == 0) {  // no tokens: the final states are the initial ones
    cudaError_t e = cudaSuccess;
    if (a.ST) e = a.S0 ? cudaMemcpyAsync(a.ST, a.S0, sbytes, cudaMemcpyDeviceToDevice, s)
                       : cudaMemsetAsync(a.ST, 0, sbytes, s);
    if (e == cudaSuccess && a.RT)
      e = a.R0 ? cudaMemcpyAsync(a.RT, a.R0, sbytes, cudaMemcpyDeviceToDevice, s)
               : cudaMemsetAsync(a.RT, 0, sbytes, s);
    return e;
  }
  FwdParams p = make_fwd_params(a);
  p.ws = (float *)a.workspace;
  const size_t total = plan_fwd(a, variant).total_bytes;
  p.err = status_word();
  p.inject = fault_injection() == 3 ? 1 : 0;
  if (a.cu_seqlens) {
    long long *seq = (long long *)((char *)a.workspace + total - 256 - seq_table_bytes(a));
    const cudaError_t e = launch_seq_table(a, seq, s);
    if (e != cudaSuccess) return e;
    p.seq = seq;
  }
  if (a.flags & RDN_FLAG_SAVE_FOR_BWD) {
    const SavedLayout l = saved_layout((size_t)p.nrec, a.Dv, a.flags & RDN_FLAG_TANH_RESIDUAL);
    p.sv_E = (uint8_t *)a.workspace + l.e;
    p.sv_E2 = (uint8_t *)a.workspace + l.e2;
    p.sv_mask = (unsigned long long *)((char *)a.workspace + l.mask);
  }
  if (p.qk_norm) set_qk_norm_copies(p, a, (char *)a.workspace + qk_norm_offset(a));
  return launch_fwd_parts(p, a.Dk, variant == 1, a.dtype == RDN_BF16, true, true, s);
}

}  // namespace rdn
