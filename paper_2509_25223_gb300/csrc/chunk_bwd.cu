// chunk_bwd.cu -- backward of the chunkwise RLA / RDN forward (fp32 SIMT:
// fp32 inputs, d = 64, the tanh residual and the stateless correction), and
// the dispatcher of both backward paths.
//
// Reverse mode of the chunk algebra in chunk_fwd.cu (the paper gives no
// backward; this is the adjoint of the forward as computed).  Per chunk,
// given the carried dS, dR (gradients w.r.t. the chunk-end states) and dO:
//
//   auxiliary pass  dOa = diag(gam) dO;  dgam += rowsum(dO * Oa)
//                   dM2 = incl(dOa E2^T);  dE2 = M2^T dOa + diag(wR) K dR
//                   RDN: dX2 = Tg^T dE2, dAg = -strict(dX2 E2^T), dRv = dX2,
//                        dKR = -diag(Gam) dX2;   RLA: dRv = dE2
//                   dR0 = Gam_C dR + K^T dKR + Q^T diag(Gam) dOa
//   clip            dV = dRv * [|v - P| <= c],  dP = -dV
//   base pass       dMq = strict(dO E^T);  dAp = strict(dP E^T)
//                   dE = Mq^T dO + Ap^T dP + diag(wS) K dS
//                   RDN: dX = Tb^T dE, dAb = -strict(dX E^T), dV += dX,
//                        dKS = diag(Gprev) dP - diag(Gam) dX;   RLA: dV += dE
//                   dS0 = Gam_C dS + K^T dKS + Q^T diag(Gam) dO
//   dK, dQ collect the state products (E dS^T, dKS S0^T, ...); the C x C
//   gradients dAp, dMq, dM2, dAb, dAg and the per-row factors then give
//   d(KK^T), d(QK^T), dbeta, dgamma and the gradient of the in-chunk
//   cumulative log-decay, whose reverse cumulative sum is dg.
//
// Kernel bwd_scan: one CTA per (b, h, 16-column slice of d_v), chunks in
// reverse, recomputing the chunk's forward pieces from the chunk-start
// states.  Value columns are independent in the forward, so each slice owns
// its dv, dS, dR columns; its contributions to dK, dQ and to the C x C and
// per-row gradients (sums over d_v) are added into a per-chunk accumulator.
// Kernel bwd_finish: one CTA per chunk, folds the accumulator into dq, dk,
// dg, dbeta, dgamma.
#include "chunk_common.cuh"
#include "status.cuh"

namespace rdn {
namespace {

constexpr int kBDVS = 16;       // value columns per backward scan CTA
constexpr int kScanThreads = 512;  // threads of a backward scan CTA (latency bound: 16 warps)
constexpr int LDV = kBDVS + 1;  // padded row stride of the [C][kBDVS] tiles

template <int DK>
struct Acc {  // per-chunk accumulator record (floats)
  static constexpr int DKo = 0, DQo = C * DK;
  static constexpr int DAP = 2 * C * DK, DMQ = DAP + kCC, DM2 = DMQ + kCC, DAB = DM2 + kCC,
                       DAG = DAB + kCC, VEC = DAG + kCC;
  // per-row vectors: d(gamma) from the read-out, dGam, dGprev, dwS, dwR; then dGamC
  static constexpr int V_DGAM_OUT = 0, V_DGAM = C, V_DGPREV = 2 * C, V_DWS = 3 * C, V_DWR = 4 * C,
                       V_DGAMC = 5 * C;
  static constexpr int FLOATS = VEC + 6 * C;
};

struct BwdParams {
  FwdParams f;  // forward inputs; f.ws = prep records
  const void *dO;
  const float *dST, *dRT;
  const float *Sc, *Rc;  // chunk-start states [B,H,NC,DK,DV]
  void *dq, *dk, *dv;
  float *dg, *dbeta, *dgamma, *dS0, *dR0;
  float *acc;  // [B*H*NC] accumulator records
  // RDN_FLAG_QK_NORM with bf16 inputs: dq, dk (w.r.t. the normalised q, k)
  // stored here in fp32 for the normalisation's backward; else NULL
  float *gq32, *gk32;
};

// ---------------------------------------------------------------- kernel 1
template <int DK, bool RDNV, typename InT>
__global__ void __launch_bounds__(kScanThreads, 1) bwd_scan_kernel(BwdParams p) {
  constexpr int DV = DK;
  constexpr int LDK = DK + 1;
  using L = Acc<DK>;
  extern __shared__ float sm[];
  float *Ks = sm;                // [C][LDK]
  float *Qs = Ks + C * LDK;      // [C][LDK] (scaled q)
  float *S0 = Qs + C * LDK;      // [DK][LDV] chunk-start states (slice)
  float *R0 = S0 + DK * LDV;
  float *dS = R0 + DK * LDV;     // carried gradients w.r.t. the chunk-end states
  float *dR = dS + DK * LDV;
  float *CC = dR + DK * LDV;     // [C][C] staging of one chunk matrix
  float *Vs = CC + C * C;        // [C][LDV] tiles
  float *dOs = Vs + C * LDV;
  float *KS = dOs + C * LDV;
  float *QS = KS + C * LDV;
  float *KR = QS + C * LDV;
  float *QR = KR + C * LDV;
  float *Es = QR + C * LDV;
  float *E2 = Es + C * LDV;
  float *XR = E2 + C * LDV;      // v - P, the residual before the clip
  float *T1 = XR + C * LDV;
  float *T2 = T1 + C * LDV;
  float *T3 = T2 + C * LDV;
  float *vec = T3 + C * LDV;     // [6*C] Gam, Gprev, alpha, wS, wR, GamC
  float *gmv = vec + 6 * C;      // [C] gamma per token
  float *red = gmv + C;          // [6*C] per-row sums of this slice

  const int bh = blockIdx.x;
  const int H = p.f.H, h = bh % H;
  const SeqSpan sp = seq_span(p.f, bh / H, h);  // this (sequence, head)'s tokens and records
  const long long tok0 = sp.tok0;
  const int NC = sp.nc, T = sp.len;
  const int j0 = blockIdx.y * kBDVS;
  const int tid = threadIdx.x;
  const InT *q = (const InT *)p.f.q;
  const InT *k = (const InT *)p.f.k;
  const InT *v = (const InT *)p.f.v;
  const InT *dO = (const InT *)p.dO;
  InT *dv = (InT *)p.dv;
  const float clip = p.f.clip;
  const size_t sbase = (size_t)bh * DK * DV;
  const bool dec_res = p.f.mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = p.f.mods & RDN_FLAG_PLAIN_COMBINE;
  const bool tnh = p.f.mods & RDN_FLAG_TANH_RESIDUAL;
  const bool stl = p.f.mods & RDN_FLAG_STATELESS_AUX;
  const bool rdn_aux = RDNV && !stl;  // the auxiliary pass runs the delta rule

  using MMk = BlockMM<C, kBDVS, DK, kScanThreads>;   // [C x DK] @ [DK x DVS]
  using MMc = BlockMM<C, kBDVS, C, kScanThreads>;    // [C x C] @ [C x DVS]
  using MMg = BlockMM<C, C, kBDVS, kScanThreads>;    // [C x DVS] @ [DVS x C]
  using MMd = BlockMM<C, DK, kBDVS, kScanThreads>;   // [C x DVS] @ [DVS x DK]
  using MMu = BlockMM<DK, kBDVS, C, kScanThreads>;   // [DK x C] @ [C x DVS]
  const int col = MMk::col();

  for (int e = tid; e < DK * kBDVS; e += kScanThreads) {
    const int i = e / kBDVS, jj = e % kBDVS;
    dS[i * LDV + jj] = p.dST ? p.dST[sbase + (size_t)i * DV + j0 + jj] : 0.f;
    dR[i * LDV + jj] = p.dRT ? p.dRT[sbase + (size_t)i * DV + j0 + jj] : 0.f;
  }

  for (int c = NC - 1; c >= 0; --c) {
    const int t0 = c * C;
    const int n = min(C, T - t0);
    const size_t chunk = (size_t)(sp.rbase + c);
    const float *rec = p.f.ws + chunk * kRecFloats;
    float *acc = p.acc + chunk * L::FLOATS;
    __syncthreads();
    for (int e = tid; e < C * DK; e += kScanThreads) {
      const int t = e / DK, d = e % DK;
      float kv = 0.f, qv = 0.f;
      if (t < n) {
        const size_t off = ((size_t)(tok0 + t0 + t) * H + h) * DK + d;
        kv = to_f32(k[off]);
        qv = p.f.scale * to_f32(q[off]);
      }
      Ks[t * LDK + d] = kv;
      Qs[t * LDK + d] = qv;
    }
    for (int e = tid; e < C * kBDVS; e += kScanThreads) {
      const int t = e / kBDVS, jj = e % kBDVS;
      float vv = 0.f, dd = 0.f;
      if (t < n) {
        const size_t off = ((size_t)(tok0 + t0 + t) * H + h) * DV + j0 + jj;
        vv = to_f32(v[off]);
        dd = to_f32(dO[off]);
      }
      Vs[t * LDV + jj] = vv;
      dOs[t * LDV + jj] = dd;
    }
    for (int e = tid; e < DK * kBDVS; e += kScanThreads) {
      const int i = e / kBDVS, jj = e % kBDVS;
      const size_t off = chunk * DK * DV + (size_t)i * DV + j0 + jj;
      S0[i * LDV + jj] = p.Sc[off];
      R0[i * LDV + jj] = p.Rc[off];
    }
    for (int e = tid; e < 6 * C; e += kScanThreads) {
      vec[e] = rec[OFF_VEC + e];
      red[e] = 0.f;
    }
    if (tid < C) gmv[tid] = tid < n ? p.f.gamma[(size_t)(tok0 + t0 + tid) * H + h] : 0.f;
    __syncthreads();
    const float *Gam = vec + V_GAM, *Gprev = vec + V_GPREV, *wS = vec + V_WS, *wR = vec + V_WR;
    const float GamC = vec[V_GAMC];

    // ---- recompute the chunk's forward pieces
    {
      float a1[MMk::RPT], a2[MMk::RPT], a3[MMk::RPT], a4[MMk::RPT];
      MMk::run(Ks, LDK, 1, S0, LDV, 1, a1);
      MMk::run(Qs, LDK, 1, S0, LDV, 1, a2);
      MMk::run(Ks, LDK, 1, R0, LDV, 1, a3);
      MMk::run(Qs, LDK, 1, R0, LDV, 1, a4);
#pragma unroll
      for (int i = 0; i < MMk::RPT; ++i) {
        const int t = MMk::row(i);
        KS[t * LDV + col] = a1[i];
        QS[t * LDV + col] = a2[i];
        KR[t * LDV + col] = stl ? 0.f : a3[i];  // (the stateless R carries nothing)
        QR[t * LDV + col] = stl ? 0.f : a4[i];
        if (RDNV) T1[t * LDV + col] = Vs[t * LDV + col] - Gam[t] * a1[i];
      }
    }
    const float *E = Vs;
    if (RDNV) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TB + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, T1, LDV, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) Es[MMc::row(i) * LDV + col] = a1[i];
      E = Es;
    }
    __syncthreads();
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_AP + e];
    __syncthreads();
    {
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, E, LDV, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        const float x =
            Vs[t * LDV + col] - ((dec_res ? Gam[t] : Gprev[t]) * KS[t * LDV + col] + a1[i]);
        XR[t * LDV + col] = x;
        if (rdn_aux) T1[t * LDV + col] = resid_map(x, clip, tnh) - Gam[t] * KR[t * LDV + col];
        else E2[t * LDV + col] = resid_map(x, clip, tnh);
      }
    }
    __syncthreads();
    if (rdn_aux) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TG + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, T1, LDV, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) E2[MMc::row(i) * LDV + col] = a1[i];
      __syncthreads();
    }
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_M2 + e];
    __syncthreads();
    {  // Oa -> T2, dOa -> T3, row sums d(gamma)_out and dGam
      float a1[MMc::RPT];
      MMc::run(CC, C, 1, E2, LDV, 1, a1);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        const float oa = Gam[t] * QR[t * LDV + col] + a1[i];
        const float dOv = dOs[t * LDV + col];
        const float doa = plain ? dOv : gmv[t] * dOv;
        T3[t * LDV + col] = doa;
        if (!plain) atomicAdd(&red[L::V_DGAM_OUT + t], dOv * oa);
        atomicAdd(&red[L::V_DGAM + t], doa * QR[t * LDV + col]);
      }
    }
    __syncthreads();

    // ---- adjoint of the auxiliary pass
    {
      float kd[MMk::RPT], a1[MMc::RPT];
      MMk::run(Ks, LDK, 1, dR, LDV, 1, kd);
      MMc::run(CC, 1, C, T3, LDV, 1, a1);  // M2^T dOa
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        T1[t * LDV + col] = a1[i] + wR[t] * kd[i];  // dE2
        if (!stl) {  // (stateless: wR is a constant and R0 does not enter)
          atomicAdd(&red[L::V_DWR + t], kd[i] * E2[t * LDV + col]);
          QR[t * LDV + col] = Gam[t] * T3[t * LDV + col];  // dQR
        }
      }
      float g1[MMg::RPT];
      MMg::run(T3, LDV, 1, E2, 1, LDV, g1);  // dM2 = dOa E2^T (inclusive)
#pragma unroll
      for (int i = 0; i < MMg::RPT; ++i) {
        const int t = MMg::row(i), ii = MMg::col();
        if (ii <= t) atomicAdd(&acc[L::DM2 + t * C + ii], g1[i]);
      }
    }
    __syncthreads();
    const float *dRv = T1;
    if (rdn_aux) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TG + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, 1, C, T1, LDV, 1, a1);  // dX2 = Tg^T dE2
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) T2[MMc::row(i) * LDV + col] = a1[i];
      __syncthreads();
      float g1[MMg::RPT];
      MMg::run(T2, LDV, 1, E2, 1, LDV, g1);  // dAg = -strict(dX2 E2^T)
#pragma unroll
      for (int i = 0; i < MMg::RPT; ++i) {
        const int t = MMg::row(i), ii = MMg::col();
        if (ii < t) atomicAdd(&acc[L::DAG + t * C + ii], -g1[i]);
      }
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        T1[t * LDV + col] = -Gam[t] * a1[i];  // dKR
        atomicAdd(&red[L::V_DGAM + t], -a1[i] * KR[t * LDV + col]);
      }
      dRv = T2;
    }
    // T3 <- diag(wR) E2 for dK += diag(wR) E2 dR^T
    for (int e = tid; e < C * kBDVS; e += kScanThreads) {
      const int t = e / kBDVS, jj = e % kBDVS;
      T3[t * LDV + jj] = wR[t] * E2[t * LDV + jj];
    }
    __syncthreads();
    float dKacc[MMd::RPT], dQacc[MMd::RPT];
    {
      float g1[MMd::RPT];
      MMd::run(T3, LDV, 1, dR, 1, LDV, dKacc);
      if (rdn_aux) {
        MMd::run(T1, LDV, 1, R0, 1, LDV, g1);
#pragma unroll
        for (int i = 0; i < MMd::RPT; ++i) dKacc[i] += g1[i];
      }
      MMd::run(QR, LDV, 1, R0, 1, LDV, dQacc);
      float s = 0.f;
      if (!stl)
        for (int e = tid; e < DK * kBDVS; e += kScanThreads) {
          const int i = e / kBDVS, jj = e % kBDVS;
          s += dR[i * LDV + jj] * R0[i * LDV + jj];
        }
      atomicAdd(&red[L::V_DGAMC], s);
    }
    __syncthreads();
    {  // dR0 = Gam_C dR + K^T dKR + Q^T dQR (stateless: 0)
      float u1[MMu::RPT], u2[MMu::RPT];
      MMu::run(Qs, 1, LDK, QR, LDV, 1, u2);
      if (rdn_aux) MMu::run(Ks, 1, LDK, T1, LDV, 1, u1);
#pragma unroll
      for (int i = 0; i < MMu::RPT; ++i) {
        const int r = MMu::row(i);
        dR[r * LDV + col] =
            stl ? 0.f : GamC * dR[r * LDV + col] + u2[i] + (rdn_aux ? u1[i] : 0.f);
      }
    }
    // clip: dV = dRv * [|x| <= c] into T3 (dP = -dV; tanh: times 1 - (r/c)^2)
    for (int e = tid; e < C * kBDVS; e += kScanThreads) {
      const int t = e / kBDVS, jj = e % kBDVS;
      T3[t * LDV + jj] = dRv[t * LDV + jj] * resid_grad(XR[t * LDV + jj], clip, tnh);
    }
    __syncthreads();

    // ---- adjoint of the base pass
    {
      float g1[MMg::RPT], g2[MMg::RPT];
      MMg::run(dOs, LDV, 1, E, 1, LDV, g1);  // dMq = strict(dO E^T)
      MMg::run(T3, LDV, 1, E, 1, LDV, g2);   // dAp = strict(dP E^T) = -strict(dV E^T)
#pragma unroll
      for (int i = 0; i < MMg::RPT; ++i) {
        const int t = MMg::row(i), ii = MMg::col();
        if (ii < t) {
          atomicAdd(&acc[L::DMQ + t * C + ii], g1[i]);
          atomicAdd(&acc[L::DAP + t * C + ii], -g2[i]);
        }
      }
    }
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_MQ + e];
    __syncthreads();
    float de[MMc::RPT];
    MMc::run(CC, 1, C, dOs, LDV, 1, de);  // Mq^T dO
    __syncthreads();
    for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_AP + e];
    __syncthreads();
    {
      float a1[MMc::RPT], kd[MMk::RPT];
      MMc::run(CC, 1, C, T3, LDV, 1, a1);  // Ap^T dV  (= -Ap^T dP)
      MMk::run(Ks, LDK, 1, dS, LDV, 1, kd);
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        const float dv_ = T3[t * LDV + col];
        T1[t * LDV + col] = de[i] - a1[i] + wS[t] * kd[i];  // dE
        atomicAdd(&red[L::V_DWS + t], kd[i] * E[t * LDV + col]);
        // the prediction's state term: Gprev KS (decayed residual: Gam KS)
        atomicAdd(&red[(dec_res ? L::V_DGAM : L::V_DGPREV) + t], -dv_ * KS[t * LDV + col]);
        T2[t * LDV + col] = -(dec_res ? Gam[t] : Gprev[t]) * dv_;  // dKS (base part)
        const float dOv = dOs[t * LDV + col];
        // the base read-out Gam QS (plain combine: Gprev QS)
        atomicAdd(&red[(plain ? L::V_DGPREV : L::V_DGAM) + t], dOv * QS[t * LDV + col]);
        QS[t * LDV + col] = (plain ? Gprev[t] : Gam[t]) * dOv;  // dQS
      }
    }
    __syncthreads();
    if (RDNV) {
      for (int e = tid; e < C * C; e += kScanThreads) CC[e] = rec[OFF_TB + e];
      __syncthreads();
      float a1[MMc::RPT];
      MMc::run(CC, 1, C, T1, LDV, 1, a1);  // dX = Tb^T dE
      __syncthreads();
#pragma unroll
      for (int i = 0; i < MMc::RPT; ++i) {
        const int t = MMc::row(i);
        T1[t * LDV + col] = a1[i];
        T3[t * LDV + col] += a1[i];                  // dV += dX
        T2[t * LDV + col] -= Gam[t] * a1[i];         // dKS -= Gam dX
        atomicAdd(&red[L::V_DGAM + t], -a1[i] * KS[t * LDV + col]);
      }
      __syncthreads();
      float g1[MMg::RPT];
      MMg::run(T1, LDV, 1, E, 1, LDV, g1);  // dAb = -strict(dX E^T)
#pragma unroll
      for (int i = 0; i < MMg::RPT; ++i) {
        const int t = MMg::row(i), ii = MMg::col();
        if (ii < t) atomicAdd(&acc[L::DAB + t * C + ii], -g1[i]);
      }
    } else {
      for (int e = tid; e < C * kBDVS; e += kScanThreads) {
        const int t = e / kBDVS, jj = e % kBDVS;
        T3[t * LDV + jj] += T1[t * LDV + jj];  // dV += dE
      }
    }
    // XR <- diag(wS) E for dK += diag(wS) E dS^T
    for (int e = tid; e < C * kBDVS; e += kScanThreads) {
      const int t = e / kBDVS, jj = e % kBDVS;
      XR[t * LDV + jj] = wS[t] * E[t * LDV + jj];
    }
    __syncthreads();
    {
      float g1[MMd::RPT];
      MMd::run(XR, LDV, 1, dS, 1, LDV, g1);
#pragma unroll
      for (int i = 0; i < MMd::RPT; ++i) dKacc[i] += g1[i];
      MMd::run(T2, LDV, 1, S0, 1, LDV, g1);
#pragma unroll
      for (int i = 0; i < MMd::RPT; ++i) dKacc[i] += g1[i];
      MMd::run(QS, LDV, 1, S0, 1, LDV, g1);
#pragma unroll
      for (int i = 0; i < MMd::RPT; ++i) dQacc[i] += g1[i];
      float s = 0.f;
      for (int e = tid; e < DK * kBDVS; e += kScanThreads) {
        const int i = e / kBDVS, jj = e % kBDVS;
        s += dS[i * LDV + jj] * S0[i * LDV + jj];
      }
      atomicAdd(&red[L::V_DGAMC], s);
    }
    __syncthreads();
    {  // dS0 = Gam_C dS + K^T dKS + Q^T dQS
      float u1[MMu::RPT], u2[MMu::RPT];
      MMu::run(Ks, 1, LDK, T2, LDV, 1, u1);
      MMu::run(Qs, 1, LDK, QS, LDV, 1, u2);
#pragma unroll
      for (int i = 0; i < MMu::RPT; ++i) {
        const int r = MMu::row(i);
        dS[r * LDV + col] = GamC * dS[r * LDV + col] + u1[i] + u2[i];
      }
    }
    // ---- outputs of this slice
#pragma unroll
    for (int i = 0; i < MMd::RPT; ++i) {
      const int t = MMd::row(i), d = MMd::col();
      atomicAdd(&acc[L::DKo + t * DK + d], dKacc[i]);
      atomicAdd(&acc[L::DQo + t * DK + d], dQacc[i]);
    }
    for (int e = tid; e < C * kBDVS; e += kScanThreads) {
      const int t = e / kBDVS, jj = e % kBDVS;
      if (t < n) dv[((size_t)(tok0 + t0 + t) * H + h) * DV + j0 + jj] = from_f32<InT>(T3[t * LDV + jj]);
    }
    __syncthreads();
    for (int e = tid; e < 5 * C + 1; e += kScanThreads) atomicAdd(&acc[L::VEC + e], red[e]);
  }
  __syncthreads();
  for (int e = tid; e < DK * kBDVS; e += kScanThreads) {
    const int i = e / kBDVS, jj = e % kBDVS;
    if (p.dS0) p.dS0[sbase + (size_t)i * DV + j0 + jj] = dS[i * LDV + jj];
    if (p.dR0) p.dR0[sbase + (size_t)i * DV + j0 + jj] = dR[i * LDV + jj];
  }
}

// ---------------------------------------------------------------- kernel 2
// One CTA per chunk.  Each warp owns 4 rows t of the C x C gradients; lane l
// handles columns l and l + 32.  Row sums (d cum_t, d cprev_t) are reduced
// with shuffles; column sums (d cum_i, dbeta_i, dgamma_i) go through
// shared-memory tiles and a column pass, so no shared-memory atomics are
// contended.
template <int DK, bool RDNV, typename InT>
__global__ void __launch_bounds__(kScanThreads, 1) bwd_finish_kernel(BwdParams p) {
  constexpr int LDK = DK + 1;
  constexpr int LDC = C + 1;
  using L = Acc<DK>;
  extern __shared__ float sm[];
  float *Ks = sm;               // [C][LDK]
  float *Qs = Ks + C * LDK;     // [C][LDK]
  float *KK = Qs + C * LDK;     // [C][LDC]
  float *QK = KK + C * LDC;     // [C][LDC]
  float *dKK = QK + C * LDC;    // [C][LDC] symmetrised before use
  float *dQK = dKK + C * LDC;   // [C][LDC]
  float *colG = dQK + C * LDC;  // [C][LDC] column contributions to d cum
  float *colB = colG + C * LDC; // [C][LDC] ... to dbeta
  float *colM = colB + C * LDC; // [C][LDC] ... to dgamma
  float *cum = colM + C * LDC;  // [C]
  float *cprev = cum + C;
  float *bet = cprev + C;
  float *gam = bet + C;
  float *gg = gam + C;
  float *dcum = gg + C;
  float *dcprev = dcum + C;
  float *dbet = dcprev + C;
  float *dgam = dbet + C;

  const long long chunk = blockIdx.x;
  if (chunk >= total_records(p.f)) return;  // (packed sequences: the grid is a bound)
  const int H = p.f.H;
  int sq, h, c;
  rec_decode(p.f, chunk, sq, h, c);
  const SeqSpan sp = seq_span(p.f, sq, h);
  const long long tok0 = sp.tok0;
  const int t0 = c * C;
  const int n = min(C, sp.len - t0);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const InT *q = (const InT *)p.f.q;
  const InT *k = (const InT *)p.f.k;
  const float *acc = p.acc + (size_t)chunk * L::FLOATS;
  const bool dec_res = p.f.mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = p.f.mods & RDN_FLAG_PLAIN_COMBINE;
  const bool stl = p.f.mods & RDN_FLAG_STATELESS_AUX;

  for (int e = tid; e < C * DK; e += kScanThreads) {
    const int t = e / DK, d = e % DK;
    float kv = 0.f, qv = 0.f;
    if (t < n) {
      const size_t off = ((size_t)(tok0 + t0 + t) * H + h) * DK + d;
      kv = to_f32(k[off]);
      qv = p.f.scale * to_f32(q[off]);
    }
    Ks[t * LDK + d] = kv;
    Qs[t * LDK + d] = qv;
  }
  if (tid < C) {
    const int t = tid;
    float gv = 0.f, bv = 0.f, mv = 0.f;
    if (t < n) {
      const size_t off = (size_t)(tok0 + t0 + t) * H + h;
      gv = p.f.g[off];
      bv = p.f.beta[off];
      mv = p.f.gamma[off];
    }
    gg[t] = gv;
    bet[t] = bv;
    gam[t] = mv;
  }
  __syncthreads();
  if (warp == 0) {  // in-chunk cumulative log-decay (two 32-wide shuffle scans)
    float a = gg[lane], b2 = gg[32 + lane];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float ua = __shfl_up_sync(0xffffffffu, a, off);
      const float ub = __shfl_up_sync(0xffffffffu, b2, off);
      if (lane >= off) {
        a += ua;
        b2 += ub;
      }
    }
    b2 += __shfl_sync(0xffffffffu, a, 31);
    cum[lane] = a;
    cum[32 + lane] = b2;
    cprev[lane] = a - gg[lane];
    cprev[32 + lane] = b2 - gg[32 + lane];
  }
  {
    using MM = BlockMM<C, C, DK, kScanThreads>;
    float a[MM::RPT];
    MM::run(Ks, LDK, 1, Ks, 1, LDK, a);
#pragma unroll
    for (int i = 0; i < MM::RPT; ++i) KK[MM::row(i) * LDC + MM::col()] = a[i];
    MM::run(Qs, LDK, 1, Ks, 1, LDK, a);
#pragma unroll
    for (int i = 0; i < MM::RPT; ++i) QK[MM::row(i) * LDC + MM::col()] = a[i];
  }
  __syncthreads();
  // ---- row pass over the C x C gradients
  constexpr int kRowsPerWarp = C / (kScanThreads / 32);
  for (int rr = 0; rr < kRowsPerWarp; ++rr) {
    const int t = warp * kRowsPerWarp + rr;
    float rowc = 0.f, rowp = 0.f;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int i = lane + 32 * half;
      const int e = t * C + i;
      float dkk = 0.f, dqk = 0.f, cg = 0.f, cb = 0.f, cm = 0.f;
      if (i <= t) {
        const float dec = expf(cum[t] - cum[i]);
        const float kk = KK[t * LDC + i], qk = QK[t * LDC + i];
        const float bi = bet[i], gi = gam[i];
        if (stl) {  // M2 = diag(QK): no decay, no rate
          if (i == t) dqk += acc[L::DM2 + e];
        } else {  // M2: inclusive, gamma, QK
          const float dm = acc[L::DM2 + e];
          const float G = dm * dec * gi * qk;
          rowc += G;
          cg += G;
          cm += dm * dec * qk;
          dqk += dm * dec * gi;
        }
        if (i < t) {
          const float decp = expf(cprev[t] - cum[i]);
          {  // Ap: strict, beta, KK, previous-token decay (decayed residual: to t)
            const float dA = dec_res ? dec : decp;
            const float dm = acc[L::DAP + e];
            const float G = dm * dA * bi * kk;
            if (dec_res) rowc += G; else rowp += G;
            cg += G;
            cb += dm * dA * kk;
            dkk += dm * dA * bi;
          }
          {  // Mq: strict, beta, QK (plain combine: decay to t-1)
            const float dA = plain ? decp : dec;
            const float dm = acc[L::DMQ + e];
            const float G = dm * dA * bi * qk;
            if (plain) rowp += G; else rowc += G;
            cg += G;
            cb += dm * dA * qk;
            dqk += dm * dA * bi;
          }
          if (RDNV) {
            const float da = acc[L::DAB + e], dg2 = acc[L::DAG + e];
            const float Gb = da * dec * bi * kk, Gg = dg2 * dec * gi * kk;
            rowc += Gb + Gg;
            cg += Gb + Gg;
            cb += da * dec * kk;
            cm += dg2 * dec * kk;
            dkk += da * dec * bi + dg2 * dec * gi;
          }
        }
      }
      dKK[t * LDC + i] = dkk;
      dQK[t * LDC + i] = dqk;
      colG[t * LDC + i] = cg;
      colB[t * LDC + i] = cb;
      colM[t * LDC + i] = cm;
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      rowc += __shfl_xor_sync(0xffffffffu, rowc, off);
      rowp += __shfl_xor_sync(0xffffffffu, rowp, off);
    }
    if (lane == 0) {
      dcum[t] = rowc;
      dcprev[t] = rowp;
    }
  }
  __syncthreads();
  // ---- column pass and per-row factors
  if (tid < C) {
    const int i = tid;
    float sg = 0.f, sb = 0.f, sm2 = 0.f;
    for (int t = i; t < C; ++t) {
      sg += colG[t * LDC + i];
      sb += colB[t * LDC + i];
      sm2 += colM[t * LDC + i];
    }
    const float cC = cum[C - 1];
    const float eC = expf(cC - cum[i]);
    const float dwS = acc[L::VEC + L::V_DWS + i], dwR = acc[L::VEC + L::V_DWR + i];
    dbet[i] = sb + dwS * eC;
    dgam[i] = sm2 + acc[L::VEC + L::V_DGAM_OUT + i] + dwR * eC;
    // d cum_i: - column sums - (dwS wS + dwR wR) + dGam * Gam
    dcum[i] += -sg - (dwS * bet[i] + dwR * gam[i]) * eC + acc[L::VEC + L::V_DGAM + i] * expf(cum[i]);
    dcprev[i] += acc[L::VEC + L::V_DGPREV + i] * expf(cprev[i]);
  }
  __syncthreads();
  if (warp == 0) {  // chunk-end terms land on cum_C = cum[C-1] (padding has g = 0)
    const float cC = cum[C - 1];
    float s = 0.f;
    for (int t = lane; t < C; t += 32)
      s += (acc[L::VEC + L::V_DWS + t] * bet[t] + acc[L::VEC + L::V_DWR + t] * gam[t]) *
           expf(cC - cum[t]);
#pragma unroll
    for (int off = 16; off; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) dcum[C - 1] += s + acc[L::VEC + L::V_DGAMC] * expf(cC);
  }
  // symmetrise: dK gets (dKK + dKK^T) K
  for (int e = tid; e < C * C; e += kScanThreads) {
    const int t = e / C, i = e % C;
    if (i < t) {
      const float s2 = dKK[t * LDC + i] + dKK[i * LDC + t];
      dKK[t * LDC + i] = s2;
      dKK[i * LDC + t] = s2;
    } else if (i == t) {
      dKK[t * LDC + i] *= 2.f;
    }
  }
  __syncthreads();
  {
    using MM = BlockMM<C, DK, C, kScanThreads>;
    float a1[MM::RPT], a2[MM::RPT], a3[MM::RPT];
    MM::run(dKK, LDC, 1, Ks, LDK, 1, a1);   // (dKK + dKK^T) K
    MM::run(dQK, 1, LDC, Qs, LDK, 1, a2);   // dQK^T Q
    MM::run(dQK, LDC, 1, Ks, LDK, 1, a3);   // dQK K
    InT *dk = (InT *)p.dk;
    InT *dq = (InT *)p.dq;
#pragma unroll
    for (int i = 0; i < MM::RPT; ++i) {
      const int t = MM::row(i), d = MM::col();
      if (t < n) {
        const size_t off = ((size_t)(tok0 + t0 + t) * H + h) * DK + d;
        const float gk = acc[L::DKo + t * DK + d] + a1[i] + a2[i];
        const float gq = p.f.scale * (acc[L::DQo + t * DK + d] + a3[i]);
        if (p.gq32) {
          p.gk32[off] = gk;
          p.gq32[off] = gq;
        } else {
          dk[off] = from_f32<InT>(gk);
          dq[off] = from_f32<InT>(gq);
        }
      }
    }
  }
  if (warp == 0) {  // dg_s = sum_{t>=s} dcum_t + sum_{t>s} dcprev_t (reverse scans)
    float a = dcum[C - 1 - lane], b2 = dcum[31 - lane];
    float pa = dcprev[C - 1 - lane], pb = dcprev[31 - lane];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float ua = __shfl_up_sync(0xffffffffu, a, off), ub = __shfl_up_sync(0xffffffffu, b2, off);
      const float upa = __shfl_up_sync(0xffffffffu, pa, off), upb = __shfl_up_sync(0xffffffffu, pb, off);
      if (lane >= off) {
        a += ua;
        b2 += ub;
        pa += upa;
        pb += upb;
      }
    }
    // a: suffix sums over t in [C-1-lane, C) ; b2 over [31-lane, 32) plus the upper half
    const float topc = __shfl_sync(0xffffffffu, a, 31), topp = __shfl_sync(0xffffffffu, pa, 31);
    b2 += topc;
    pb += topp;
    // sum_{t>s} dcprev_t = (suffix including s) - dcprev_s
    gg[C - 1 - lane] = a + (pa - dcprev[C - 1 - lane]);
    gg[31 - lane] = b2 + (pb - dcprev[31 - lane]);
  }
  __syncthreads();
  if (tid < n) {
    const size_t off = (size_t)(tok0 + t0 + tid) * H + h;
    p.dg[off] = gg[tid];
    p.dbeta[off] = dbet[tid];
    p.dgamma[off] = dgam[tid];
  }
}

template <int DK>
constexpr size_t scan_smem() {
  return sizeof(float) * (2 * C * (DK + 1) + 4 * DK * LDV + C * C + 13 * C * LDV + 6 * C + C + 6 * C);
}
template <int DK>
constexpr size_t finish_smem() {
  return sizeof(float) * (2 * C * (DK + 1) + 7 * C * (C + 1) + 9 * C);
}

template <int DK, bool RDNV, typename InT>
cudaError_t launch_t(const BwdParams &p, cudaStream_t s) {
  auto scan = bwd_scan_kernel<DK, RDNV, InT>;
  auto fin = bwd_finish_kernel<DK, RDNV, InT>;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(scan, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)scan_smem<DK>())) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(fin, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)finish_smem<DK>())) != cudaSuccess)
    return e;
  RDN_LAUNCH("bwd_scan", s, scan<<<dim3(p.f.nseq * p.f.H, DK / kBDVS), kScanThreads, scan_smem<DK>(), s>>>(p));
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  RDN_LAUNCH("bwd_finish", s, fin<<<(unsigned)p.f.nrec, kScanThreads, finish_smem<DK>(), s>>>(p));
  return cudaGetLastError();
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct BwdLayout {
  size_t prep, acc, states, o, tc, qk, g32, tied, seq, total;
};

// bf16 inputs with d = 128 take the tensor-core backward (RDN, and RLA with
// identity T matrices in its records), the variants the fp32 one
bool use_tc_bwd(const rdn_fwd_args &f, int variant) {
  (void)variant;
  return f.dtype == RDN_BF16 && f.Dk == 128 && !(f.flags & RDN_FLAG_VARIANTS & ~kTcVariants);
}

// The forward's per-chunk records are valid input when the caller passes the
// forward's workspace with its chunk-start states and they are in the format
// this backward reads: shared-memory images where the forward ran the
// tensor-core scan, read by the tensor-core backward; fp32 otherwise (the
// two choices agree for every argument set, so the check only guards them).
bool reuse_fwd_records(const rdn_fwd_args &f, int variant) {
  const FwdParams fp = make_fwd_params(f);
  return f.workspace && f.S_chunks &&
         fwd_uses_tc(fp, f.Dk, f.dtype == RDN_BF16) == use_tc_bwd(f, variant);
}

BwdLayout layout(const rdn_bwd_args &a, int variant) {
  const rdn_fwd_args &f = a.fwd;
  const bool tc = use_tc_bwd(f, variant);
  const long long nrec = call_records(f);  // record slots
  const size_t accf = f.Dk == 128 ? Acc<128>::FLOATS : Acc<64>::FLOATS;
  BwdLayout l;
  // the forward's records are read from its workspace when it is passed
  l.prep = reuse_fwd_records(f, variant) ? 0 : align256(sizeof(float) * nrec * kRecFloats);
  // (the tensor-core kernels keep their per-chunk sums in shared memory)
  l.acc = tc ? 0 : align256(sizeof(float) * nrec * accf);
  const bool need_states = f.S_chunks == nullptr;
  l.states = need_states ? align256(sizeof(float) * nrec * f.Dk * f.Dv) : 0;  // each of S, R
  const size_t esz = f.dtype == RDN_BF16 ? 2 : 4;
  l.o = need_states ? align256(esz * (size_t)f.B * f.T * f.H * f.Dv) : 0;
  l.tc = tc ? align256(bwd_tc_extra_bytes(nrec, f.flags & RDN_FLAG_TANH_RESIDUAL)) : 0;
  // normalised q, k (RDN_FLAG_QK_NORM), unless the forward's workspace has them
  l.qk = reuse_fwd_records(f, variant) ? 0 : align256(qk_norm_bytes(f));
  // and, with bf16 inputs, dq, dk (w.r.t. the normalised q, k) in fp32 for
  // the normalisation's backward: its projection (dy - y <y, dy>) would
  // otherwise start from bf16-rounded dy
  l.g32 = (f.flags & RDN_FLAG_QK_NORM) && f.dtype == RDN_BF16
              ? align256(2 * sizeof(float) * (size_t)f.B * f.T * f.H * f.Dk)
              : 0;
  l.seq = seq_table_bytes(f);
  // tied gates without a dgamma buffer: the gamma part is made here, then added
  l.tied = (f.flags & RDN_FLAG_TIED_GAMMA) && !a.dgamma
               ? align256(sizeof(float) * (size_t)f.B * f.T * f.H)
               : 0;
  // + the packed-sequence table and a 256-byte tail
  l.total = l.prep + l.acc + 2 * l.states + l.o + l.tc + l.qk + l.g32 + l.tied + l.seq + 256;
  return l;
}

}  // namespace

BwdPlan plan_bwd(const rdn_bwd_args &a, int variant) {
  if (a.fwd.T == 0) return BwdPlan{0};
  return BwdPlan{layout(a, variant).total};
}

static __global__ void add_inplace_kernel(float *__restrict__ a, const float *__restrict__ b,
                                          size_t n) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    a[i] += b[i];
}

static cudaError_t launch_bwd_impl(const rdn_bwd_args &a, int variant, cudaStream_t s);

cudaError_t launch_bwd(const rdn_bwd_args &a0, int variant, cudaStream_t s) {
  const rdn_fwd_args &f = a0.fwd;
  if (!(f.flags & RDN_FLAG_TIED_GAMMA) || f.T == 0) return launch_bwd_impl(a0, variant, s);
  // tied gates (gamma is beta): the untied gradients, then dbeta += dgamma
  rdn_bwd_args a = a0;
  const BwdLayout l = layout(a0, variant);
  // (after what the untied backward uses: its own plan is l.total - l.tied bytes)
  if (!a.dgamma) a.dgamma = (float *)((char *)a.workspace + l.total - l.tied);
  cudaError_t e = launch_bwd_impl(a, variant, s);
  if (e != cudaSuccess) return e;
  const size_t n = (size_t)f.B * f.T * f.H;
  const unsigned grid = (unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  RDN_LAUNCH("tied_gate_grad", s, add_inplace_kernel<<<grid, 256, 0, s>>>(a.dbeta, a.dgamma, n));
  return cudaGetLastError();
}

static cudaError_t launch_bwd_impl(const rdn_bwd_args &a, int variant, cudaStream_t s) {
  const rdn_fwd_args &f = a.fwd;
  const size_t sbytes = sizeof(float) * (size_t)call_seqs(f) * f.H * f.Dk * f.Dv;
  if (f.T == 0) {  // no tokens: the initial-state gradients are the upstream ones
    cudaError_t e = cudaSuccess;
    if (a.dS0) e = a.dST ? cudaMemcpyAsync(a.dS0, a.dST, sbytes, cudaMemcpyDeviceToDevice, s)
                         : cudaMemsetAsync(a.dS0, 0, sbytes, s);
    if (e == cudaSuccess && a.dR0)
      e = a.dRT ? cudaMemcpyAsync(a.dR0, a.dRT, sbytes, cudaMemcpyDeviceToDevice, s)
                : cudaMemsetAsync(a.dR0, 0, sbytes, s);
    return e;
  }
  const BwdLayout l = layout(a, variant);
  char *ws = (char *)a.workspace;
  BwdParams p;
  p.f = make_fwd_params(f);
  // fp32 results (RDN_FLAG_F32_OUT in fwd.flags) are the backward's dq, dk, dv;
  // a forward recomputed here keeps its o in fwd.dtype
  const bool grad_f32 = p.f.f32out != 0;
  p.f.f32out = 0;
  p.f.inject = fault_injection() == 4 ? 2 : 0;
  const bool reuse = reuse_fwd_records(f, variant);
  p.f.ws = reuse ? (float *)f.workspace : (float *)ws;
  p.f.err = status_word();
  if (f.cu_seqlens) {  // this call's own copy of the packed-sequence table
    long long *seq = (long long *)(ws + l.total - 256 - l.seq);
    cudaError_t e = launch_seq_table(f, seq, s);
    if (e != cudaSuccess) return e;
    p.f.seq = seq;
  }
  if (p.f.qk_norm)  // the normalised q, k: the forward's, or made with this call's records
    set_qk_norm_copies(p.f, f, reuse ? (char *)f.workspace + qk_norm_offset(f)
                                     : ws + l.prep + l.acc + 2 * l.states + l.o + l.tc);
  if (reuse && (f.flags & RDN_FLAG_SAVE_FOR_BWD)) {  // E, E2 and the mask kept by the forward
    const SavedLayout sl = saved_layout((size_t)p.f.nrec, f.Dv, f.flags & RDN_FLAG_TANH_RESIDUAL);
    p.f.sv_E = (uint8_t *)f.workspace + sl.e;
    p.f.sv_E2 = (uint8_t *)f.workspace + sl.e2;
    p.f.sv_mask = (unsigned long long *)((char *)f.workspace + sl.mask);
  }
  p.f.ST = p.f.RT = nullptr;
  const bool bf = f.dtype == RDN_BF16;
  const bool rdnv = variant == 1;
  const bool tc = use_tc_bwd(f, variant);
  cudaError_t e = cudaSuccess;  // (nothing to launch first when both the states and records are reused)
  if (f.S_chunks == nullptr) {  // recompute the chunk-start states
    p.f.S_chunks = (float *)(ws + l.prep + l.acc);
    p.f.R_chunks = (float *)(ws + l.prep + l.acc + l.states);
    p.f.o = ws + l.prep + l.acc + 2 * l.states;
    e = launch_fwd_parts(p.f, f.Dk, rdnv, bf, true, true, s);
    // the tensor-core forward leaves its records as shared-memory images,
    // which the tensor-core backward reads too; the SIMT backward needs fp32
    if (e == cudaSuccess && fwd_uses_tc(p.f, f.Dk, bf) && !tc)
      e = launch_prep(p.f, f.Dk, rdnv, bf, false, s);
  } else if (!reuse) {
    e = launch_prep(p.f, f.Dk, rdnv, bf, tc, s);
  }
  if (e != cudaSuccess) return e;
  p.Sc = p.f.S_chunks;
  p.Rc = p.f.R_chunks;
  p.acc = (float *)(ws + l.prep);
  p.dO = a.dO;
  p.dST = a.dST;
  p.dRT = a.dRT;
  p.dq = a.dq;
  p.dk = a.dk;
  p.dv = a.dv;
  p.dg = a.dg;
  p.dbeta = a.dbeta;
  p.dgamma = a.dgamma;
  p.dS0 = a.dS0;
  p.dR0 = a.dR0;
  p.gq32 = p.gk32 = nullptr;
  if (l.g32) {
    p.gq32 = (float *)(ws + l.prep + l.acc + 2 * l.states + l.o + l.tc + l.qk);
    p.gk32 = p.gq32 + (size_t)f.B * f.T * f.H * f.Dk;
  }
  if (tc) {  // (with the normalisation: dq, dk into the fp32 copies, as fp32 results)
    e = launch_bwd_tc(p.f, a.dO, a.dST, a.dRT, p.Sc, p.Rc, p.gq32 ? p.gq32 : a.dq,
                      p.gk32 ? p.gk32 : a.dk, a.dv, a.dg, a.dbeta, a.dgamma, a.dS0, a.dR0,
                      ws + l.prep + l.acc + 2 * l.states + l.o, !rdnv, grad_f32,
                      p.gq32 != nullptr, s);
  } else {
    if ((e = cudaMemsetAsync(p.acc, 0, l.acc, s)) != cudaSuccess) return e;
    if (rdnv) {
      if (f.Dk == 128) e = bf ? launch_t<128, true, __nv_bfloat16>(p, s) : launch_t<128, true, float>(p, s);
      else e = bf ? launch_t<64, true, __nv_bfloat16>(p, s) : launch_t<64, true, float>(p, s);
    } else {
      if (f.Dk == 128) e = bf ? launch_t<128, false, __nv_bfloat16>(p, s) : launch_t<128, false, float>(p, s);
      else e = bf ? launch_t<64, false, __nv_bfloat16>(p, s) : launch_t<64, false, float>(p, s);
    }
  }
  if (e != cudaSuccess || !p.f.qk_norm) return e;
  // dq, dk w.r.t. the caller's x: the normalisation's transposed Jacobian, in place
  rdn_prologue_args pa{};
  pa.rows = (long long)f.B * f.T * f.H;
  pa.D = f.Dk;
  pa.dtype = f.dtype;
  pa.eps = f.qk_eps;
  pa.x[0] = f.q;
  pa.x[1] = f.k;
  pa.dx[0] = a.dq;
  pa.dx[1] = a.dk;
  if (p.gq32) {  // from the fp32 copies
    pa.dy[0] = p.gq32;
    pa.dy[1] = p.gk32;
    return launch_prologue_bwd_f32dy(pa, grad_f32, s);
  }
  pa.dy[0] = a.dq;
  pa.dy[1] = a.dk;
  return launch_prologue(pa, true, s);
}

}  // namespace rdn
