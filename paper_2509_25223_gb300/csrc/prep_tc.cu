// prep_tc.cu -- chunk_prep on the tensor cores for RDN and RLA with bf16
// inputs and d_k = 128: the state-independent matrices of one 64-token chunk (the UT
// form of the delta rule over a chunk of Section 3.4's recurrence; algebra
// in chunk_fwd.cu's header), written as the shared-memory images the
// tensor-core scans copy into their operand slots.
//
// Two persistent CTAs of 256 threads per SM, each walking chunks (the next
// chunk's K, Q and gates are fetched while the current one finishes):
//   1. the Gram matrices [K ; Q] K^T in one tcgen05 product (bf16 inputs are
//      exact, fp32 accumulation; the query scale is applied to the result);
//   2. thread (row, half) turns its TMEM row into the decayed, gated matrices
//      Ap, Mq, diag(gamma) M2 (written straight to the record as bf16 hi + lo
//      image rows) and A_beta, A_gamma (fp32, shared memory);
//   3. T_beta = (I + A_beta)^-1 and T_gamma = (I + A_gamma)^-1, 128 threads
//      each, in fp32, as a recursive 2 x 2 block inverse of the unit-lower
//      matrix: diagonal 16 x 16 blocks by forward substitution, then
//      T_ij = -T_ii A_ij T_jj for the 16-row blocks (1,0), (3,2) and the
//      32-row block (1,0), the products register-tiled;
//   4. their image rows and the gate vectors.
#include "chunk_common.cuh"
#include "tc_common.cuh"

namespace rdn {
namespace {

using namespace tc;

constexpr int D = 128;
constexpr int NTH = 256;
constexpr int LDA = C + 1;  // A_beta, A_gamma: rows written by the row pass, read as scalars
constexpr int LDT = C + 4;  // T_beta, T_gamma: rows read as 16-byte vectors
constexpr int LDW = 36;     // product scratch W, 32 x 32

namespace pp {
constexpr uint32_t KQ = 0;                   // K rows 0..63, Q rows 64..127, 2 x 16 KB
constexpr uint32_t AB = 32768;               // fp32 A_beta, A_gamma [64][LDA]
constexpr uint32_t AG = AB + 64 * LDA * 4;
constexpr uint32_t TB = AG + 64 * LDA * 4;   // fp32 T_beta, T_gamma [64][LDT]
constexpr uint32_t TG = TB + 64 * LDT * 4;
constexpr uint32_t WS = TG + 64 * LDT * 4;   // product scratch, 2 x [32][LDW]
// cum, cprev, beta, gamma, g, and cum, cprev times log2(e) (7 x 64)
constexpr uint32_t VEC = WS + 2 * 32 * LDW * 4;
static_assert(TB % 16 == 0 && TG % 16 == 0 && WS % 16 == 0 && VEC % 16 == 0, "16-byte rows");
constexpr uint32_t CTL = VEC + 7 * 64 * 4;   // mbarrier, flag, drain mbarrier
constexpr uint32_t SLOT = CTL + 24;          // TMEM base
constexpr size_t SMEM = SLOT + 16;
static_assert(2 * (SMEM + 1024) <= 233472, "two CTAs per SM");
}  // namespace pp

// Row r, columns c0 .. c0+15 (c0 a multiple of 16 below 64) of a 64-column
// image in global memory: bf16 hi part at `hi`, lo part `lo_off` bytes later.
__device__ __forceinline__ void img_row16(uint8_t *hi, uint32_t lo_off, int r, int c0,
                                          const float (&v)[16]) {
  uint32_t h[8], l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) split_pack_bf16(v[2 * i], v[2 * i + 1], h[i], l[i]);
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const uint32_t off = sw128(r, c0 + 8 * half);
    *reinterpret_cast<uint4 *>(hi + off) =
        make_uint4(h[4 * half], h[4 * half + 1], h[4 * half + 2], h[4 * half + 3]);
    *reinterpret_cast<uint4 *>(hi + lo_off + off) =
        make_uint4(l[4 * half], l[4 * half + 1], l[4 * half + 2], l[4 * half + 3]);
  }
}

// T = (I + A)^-1 for a strictly lower 64 x 64 A, by 128 threads (g = thread
// index in the group); W is 32 x LDW scratch.  The caller synchronises the
// block between the stages (0: diagonal blocks; 1, 2: the 16-row blocks; 3, 4:
// the 32-row block), all groups of the block running the same stage.  The
// 16 x 16 blocks above the diagonal are never written: the caller zeroes them
// once.
__device__ __forceinline__ void inv64_stage(int stage, const float *A, float *Tm, float *W, int g) {
  if (stage == 0) {
    // diagonal 16 x 16 blocks: thread (block, column) forward-substitutes its
    // column, x[r] = delta(r, col) - sum_{m < r} A[r][m] x[m], the terms added
    // in the order of m; the updates of the rows below m are independent, so
    // they are made as soon as x[m] is final (a 16-step chain instead of 120)
    if (g < 64) {
      const int b0 = (g >> 4) * 16, col = g & 15;
      float x[16];
#pragma unroll
      for (int r = 0; r < 16; ++r) x[r] = (r == col) ? 1.f : 0.f;
#pragma unroll
      for (int m = 0; m < 16; ++m) {
        if (m < col) x[m] = 0.f;  // (above the diagonal)
#pragma unroll
        for (int r = m + 1; r < 16; ++r) x[r] = fmaf(-A[(b0 + r) * LDA + b0 + m], x[m], x[r]);
      }
#pragma unroll
      for (int r = 0; r < 16; ++r) Tm[(b0 + r) * LDT + b0 + col] = x[r];
    }
  } else if (stage <= 2) {
    // 16-row blocks (i, j) = (1, 0) and (3, 2): W = A_ij T_jj, then
    // T_ij = -T_ii W; thread (block, row r, columns 4q .. 4q + 3)
    const int bi = 2 * (g >> 6) + 1, bj = bi - 1, r = (g >> 2) & 15, q = g & 3;
    float *w = W + (g >> 6) * 16 * LDW;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    if (stage == 1) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const float a = A[(16 * bi + r) * LDA + 16 * bj + k];
        const float4 t = *reinterpret_cast<const float4 *>(Tm + (16 * bj + k) * LDT + 16 * bj + 4 * q);
        acc[0] = fmaf(a, t.x, acc[0]); acc[1] = fmaf(a, t.y, acc[1]);
        acc[2] = fmaf(a, t.z, acc[2]); acc[3] = fmaf(a, t.w, acc[3]);
      }
      *reinterpret_cast<float4 *>(w + r * LDW + 4 * q) = make_float4(acc[0], acc[1], acc[2], acc[3]);
    } else {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const float a = Tm[(16 * bi + r) * LDT + 16 * bi + k];
        const float4 t = *reinterpret_cast<const float4 *>(w + k * LDW + 4 * q);
        acc[0] = fmaf(a, t.x, acc[0]); acc[1] = fmaf(a, t.y, acc[1]);
        acc[2] = fmaf(a, t.z, acc[2]); acc[3] = fmaf(a, t.w, acc[3]);
      }
      *reinterpret_cast<float4 *>(Tm + (16 * bi + r) * LDT + 16 * bj + 4 * q) =
          make_float4(-acc[0], -acc[1], -acc[2], -acc[3]);
    }
  } else {
    // the 32-row block: W = A[32:64, 0:32] T[0:32, 0:32], then
    // T[32:64, 0:32] = -T[32:64, 32:64] W; thread (rows rp, rp + 16, columns 4q .. 4q + 3)
    const int q = g & 7, rp = g >> 3;
    float a0[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f};
    if (stage == 3) {
#pragma unroll 8
      for (int k = 0; k < 32; ++k) {
        const float x0 = A[(32 + rp) * LDA + k], x1 = A[(48 + rp) * LDA + k];
        const float4 t = *reinterpret_cast<const float4 *>(Tm + k * LDT + 4 * q);
        a0[0] = fmaf(x0, t.x, a0[0]); a0[1] = fmaf(x0, t.y, a0[1]);
        a0[2] = fmaf(x0, t.z, a0[2]); a0[3] = fmaf(x0, t.w, a0[3]);
        a1[0] = fmaf(x1, t.x, a1[0]); a1[1] = fmaf(x1, t.y, a1[1]);
        a1[2] = fmaf(x1, t.z, a1[2]); a1[3] = fmaf(x1, t.w, a1[3]);
      }
      *reinterpret_cast<float4 *>(W + rp * LDW + 4 * q) = make_float4(a0[0], a0[1], a0[2], a0[3]);
      *reinterpret_cast<float4 *>(W + (rp + 16) * LDW + 4 * q) = make_float4(a1[0], a1[1], a1[2], a1[3]);
    } else {
#pragma unroll 8
      for (int k = 0; k < 32; ++k) {
        const float x0 = Tm[(32 + rp) * LDT + 32 + k], x1 = Tm[(48 + rp) * LDT + 32 + k];
        const float4 t = *reinterpret_cast<const float4 *>(W + k * LDW + 4 * q);
        a0[0] = fmaf(x0, t.x, a0[0]); a0[1] = fmaf(x0, t.y, a0[1]);
        a0[2] = fmaf(x0, t.z, a0[2]); a0[3] = fmaf(x0, t.w, a0[3]);
        a1[0] = fmaf(x1, t.x, a1[0]); a1[1] = fmaf(x1, t.y, a1[1]);
        a1[2] = fmaf(x1, t.z, a1[2]); a1[3] = fmaf(x1, t.w, a1[3]);
      }
      *reinterpret_cast<float4 *>(Tm + (32 + rp) * LDT + 4 * q) =
          make_float4(-a0[0], -a0[1], -a0[2], -a0[3]);
      *reinterpret_cast<float4 *>(Tm + (48 + rp) * LDT + 4 * q) =
          make_float4(-a1[0], -a1[1], -a1[2], -a1[3]);
    }
  }
}

// rla: RLA's records (no delta rule: T_beta = T_gamma = I, written as such
// for the tensor-core backward; Ap, Mq, M2 and the vectors are RDN's)
__global__ void __launch_bounds__(NTH, 2) prep_tc_kernel(FwdParams p, bool rla) {
  using namespace pp;
  extern __shared__ __align__(1024) uint8_t sm[];
  const uint32_t sb = smem_u32(sm);
  if (sb & 1023u) {
    if (threadIdx.x == 0 && p.err) atomicExch(p.err, RDN_ERR_CUDA);
    return;
  }
  float *cum = reinterpret_cast<float *>(sm + VEC), *cprev = cum + 64, *bet = cum + 128,
        *gam = cum + 192, *gg = cum + 256, *cum2 = cum + 320, *cprev2 = cum + 384;
  float *Ab = reinterpret_cast<float *>(sm + AB), *Ag = reinterpret_cast<float *>(sm + AG);
  float *Tb = reinterpret_cast<float *>(sm + TB), *Tg = reinterpret_cast<float *>(sm + TG);
  float *Wsc = reinterpret_cast<float *>(sm + WS);
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm + CTL);
  volatile int *flag = reinterpret_cast<volatile int *>(sm + CTL + 8);
  uint64_t *barD = reinterpret_cast<uint64_t *>(sm + CTL + 16);  // the drain after a wait gave up
  uint32_t *slot = reinterpret_cast<uint32_t *>(sm + SLOT);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = p.H;
  const size_t nct = (size_t)total_records(p);
  // the rows loaded: the caller's q, k, or with RDN_FLAG_QK_NORM their raw x,
  // normalised here (and the results stored to the copies p.q, p.k)
  const bool qkn = p.qk_norm != 0;
  const __nv_bfloat16 *q = (const __nv_bfloat16 *)(qkn ? p.qraw : p.q);
  const __nv_bfloat16 *k = (const __nv_bfloat16 *)(qkn ? p.kraw : p.k);
  constexpr float kLog2e = 1.4426950408889634f;
  const bool dec_res = p.mods & RDN_FLAG_DECAYED_RESIDUAL;
  const bool plain = p.mods & RDN_FLAG_PLAIN_COMBINE;
  // the stateless correction R_t = r_t k_t^T: the auxiliary pass has no delta
  // rule (identity T_gamma), its in-chunk product is diag(gamma_t q_t.k_t)
  // (no decay), and the chunk-end R is the last valid token's k r^T (wR one-hot)
  const bool stl = p.mods & RDN_FLAG_STATELESS_AUX;

  if (tid == 0) {
    mbar_init(bar, 1);
    mbar_init(barD, 1);
    fence_mbar_init();
    *flag = 0;
  }
  if (warp == 0) tmem_alloc(slot, 64);
  // a chunk's K, Q (exact bf16, rows t, zero past the end), asynchronous, and
  // its gates into registers (threads 0..63); fetched while the previous chunk
  // of this CTA finishes
  auto fetch_kq = [&](size_t ck) {
    int s_, h_, cc_;
    rec_decode(p, (long long)ck, s_, h_, cc_);
    const SeqSpan sp_ = seq_span(p, s_, h_);
    const long long tok0_ = sp_.tok0;
    const int t0_ = cc_ * C, n_ = min(C, sp_.len - t0_);
    for (int e = tid; e < 64 * 16; e += NTH) {
      const int t = e >> 4, chn = e & 15;
      const bool vld = t < n_;
      const size_t off = ((size_t)(tok0_ + t0_ + (vld ? t : 0)) * H + h_) * D + chn * 8;
      const int blk = chn >> 3, cc = (chn & 7) * 8;
      cp_async16(sm + KQ + blk * 16384 + sw128(t, cc), k + off, vld);
      cp_async16(sm + KQ + blk * 16384 + sw128(64 + t, cc), q + off, vld);
    }
  };
  struct Gates {
    float g, b, m;
  };
  auto fetch_gates = [&](size_t ck) {
    int s_, h_, cc_;
    rec_decode(p, (long long)ck, s_, h_, cc_);
    const SeqSpan sp_ = seq_span(p, s_, h_);
    const long long tok0_ = sp_.tok0;
    const int t0_ = cc_ * C, n_ = min(C, sp_.len - t0_);
    Gates x{0.f, 0.f, 0.f};
    if (tid < C && tid < n_) {
      const size_t off = (size_t)(tok0_ + t0_ + tid) * H + h_;
      x.g = p.g[off];
      x.b = p.beta[off];
      x.m = p.gamma[off];
    }
    return x;
  };
  // RDN_FLAG_QK_NORM: y = SiLU(x) / max(||SiLU(x)||, eps) for the 128 rows of
  // the [K ; Q] tile in place (thread (row, half): 64 of a row's 128
  // elements in registers, the pair's sums of squares combined by a
  // shuffle; zero rows past the end stay zero).  The sigmoid is the prologue
  // kernel's, so that both paths give the same y up to the order of the sum.
  auto normalize_rows = [&]() {
    const int r = tid >> 1, hh = tid & 1;  // row (K rows 0..63, Q rows 64..127), column half
    uint8_t *blk = sm + KQ + hh * 16384;
    float u[64];  // SiLU(x), this thread's half row
    float ss = 0.f;
#pragma unroll
    for (int c8 = 0; c8 < 8; ++c8) {
      const uint4 w = *reinterpret_cast<const uint4 *>(blk + sw128(r, 8 * c8));
      const __nv_bfloat16 *b = reinterpret_cast<const __nv_bfloat16 *>(&w);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float x = __bfloat162float(b[e]);
        u[8 * c8 + e] = x * __fdividef(1.f, 1.f + __expf(-x));
        ss = fmaf(u[8 * c8 + e], u[8 * c8 + e], ss);
      }
    }
    ss += __shfl_xor_sync(0xffffffffu, ss, 1);
    const float inv = 1.f / fmaxf(sqrtf(ss), p.qk_eps);
#pragma unroll
    for (int c8 = 0; c8 < 8; ++c8) {
      uint4 w;
      uint32_t *wv = reinterpret_cast<uint32_t *>(&w);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 o2 =
            __floats2bfloat162_rn(u[8 * c8 + 2 * e] * inv, u[8 * c8 + 2 * e + 1] * inv);
        wv[e] = *reinterpret_cast<const uint32_t *>(&o2);
      }
      *reinterpret_cast<uint4 *>(blk + sw128(r, 8 * c8)) = w;
    }
  };
  // ... and the valid rows of y from the tile to the normalised copies, 16
  // bytes a thread, whole rows per half warp (after a barrier; while the Gram
  // product reads the same tile)
  auto store_rows = [&](size_t ck) {
    int s_, h_, cc_;
    rec_decode(p, (long long)ck, s_, h_, cc_);
    const SeqSpan sp_ = seq_span(p, s_, h_);
    const int t0_ = cc_ * C, n_ = min(C, sp_.len - t0_);
    for (int e = tid; e < 128 * 16; e += NTH) {
      const int r = e >> 4, chn = e & 15, t = r & 63;
      if (t >= n_) continue;
      const uint4 w = *reinterpret_cast<const uint4 *>(sm + KQ + (chn >> 3) * 16384 +
                                                       sw128(r, (chn & 7) * 8));
      __nv_bfloat16 *dst = (__nv_bfloat16 *)(r < 64 ? p.k : p.q) +
                           ((size_t)(sp_.tok0 + t0_ + t) * H + h_) * D + chn * 8;
      *reinterpret_cast<uint4 *>(dst) = w;
    }
  };
  // the inverses' 16 x 16 blocks above the diagonal: zero throughout
  for (int e = tid; e < 2 * 64 * 64; e += NTH) {
    const int m = e >> 12, r = (e >> 6) & 63, c = e & 63;
    if ((c >> 4) > (r >> 4)) (m ? Tg : Tb)[r * LDT + c] = 0.f;
  }
  Gates gt{0.f, 0.f, 0.f};
  if (blockIdx.x < nct) {
    fetch_kq(blockIdx.x);
    gt = fetch_gates(blockIdx.x);
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tm = *slot;

  bool ok = true;
  uint32_t it = 0;  // chunks done by this CTA: the MMA barrier's parity
  for (size_t chunk = blockIdx.x; chunk < nct && ok; chunk += gridDim.x, ++it) {
    const size_t next = chunk + gridDim.x;
    if (tid < C) {
      gg[tid] = gt.g;
      bet[tid] = gt.b;
      gam[tid] = gt.m;
    }
    cp_async_wait_all();  // this chunk's K, Q
    if (qkn) {
      __syncthreads();  // (every thread's copies landed)
      normalize_rows();
    }
    fence_async_smem();
    fence_before_sync();
    __syncthreads();  // (also: every thread is done with the previous chunk)
    fence_after_sync();
    if (tid == 0) {  // [K ; Q] K^T: lanes 0..63 K K^T, lanes 64..127 Q K^T (unscaled)
      mma_tile(tm, sb + KQ, 16384, sb + KQ, 16384, 8, idesc_bf16(128, 64), false);
      mma_commit(bar);
    }
    if (qkn) store_rows(chunk);  // (while the product runs)
    if (warp == 0) {  // in-chunk cumulative log-decay, while the product runs
      float a = gg[lane], a2 = gg[32 + lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float ua = __shfl_up_sync(0xffffffffu, a, off);
        const float ub = __shfl_up_sync(0xffffffffu, a2, off);
        if (lane >= off) {
          a += ua;
          a2 += ub;
        }
      }
      a2 += __shfl_sync(0xffffffffu, a, 31);
      const float p1 = a - gg[lane], p2 = a2 - gg[32 + lane];
      cum[lane] = a;
      cum[32 + lane] = a2;
      cprev[lane] = p1;
      cprev[32 + lane] = p2;
      cum2[lane] = a * kLog2e;
      cum2[32 + lane] = a2 * kLog2e;
      cprev2[lane] = p1 * kLog2e;
      cprev2[32 + lane] = p2 * kLog2e;
    }
    if (!mbar_wait(bar, it & 1u)) *flag = 1;
    __syncthreads();
    fence_after_sync();
    ok = *flag == 0;
    if (!ok) break;
    if (next < nct) {  // K, Q are done with: the next chunk's, during this one
      fetch_kq(next);
      gt = fetch_gates(next);
    }
    uint8_t *img = reinterpret_cast<uint8_t *>(p.ws + chunk * kRecFloats);
    {  // thread (row r, half hf) of the Gram read-out: columns i in [32 hf, 32 hf + 32)
      const int r = tid & 127, hf = tid >> 7;
      float gv[32];
      {
        const uint32_t ta = tm + ((uint32_t)((warp & 3) * 32) << 16) + 32 * hf;
        float x0[16], x1[16];
        tmem_ld16x2(ta, x0, ta + 16, x1);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          gv[i] = x0[i];
          gv[16 + i] = x1[i];
        }
      }
      if (r < 64) {  // K K^T row t: Ap (previous-token decay), A_beta, A_gamma (strict);
                     // e^{b_t - b_i} = e^{b_{t-1} - b_i} e^{g_t}, both factors <= 1
        const int t = r;
        const float cp2 = cprev2[t], al = exp2f(cum2[t] - cp2);
#pragma unroll
        for (int c0 = 0; c0 < 32; c0 += 16) {
          const int i0 = 32 * hf + c0;
          float c2[16], bt[16], gm[16], ap[16];
          lds16(cum2 + i0, c2);
          lds16(bet + i0, bt);
          lds16(gam + i0, gm);
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int i = i0 + u;
            float a_p = 0.f, a_b = 0.f, a_g = 0.f;
            if (i < t) {
              const float dk = exp2f(cp2 - c2[u]) * gv[c0 + u];
              a_p = dk * bt[u];
              a_b = a_p * al;
              a_g = dk * al * gm[u];
            }
            ap[u] = dec_res ? a_b : a_p;  // (decayed residual: Ap decays to t)
            Ab[t * LDA + i] = a_b;
            Ag[t * LDA + i] = a_g;
          }
          img_row16(img + IMG_APMQ, 16384, t, i0, ap);
        }
      } else {  // Q K^T row t: Mq (strict), diag(gamma) M2 (inclusive)
        const int t = r - 64;
        // (plain combine: S_{t-1} q_t reads Mq decayed to t-1, and the output
        // has no gamma_t, so the image is M2 itself)
        const float ct2 = cum2[t], gtt = plain ? 1.f : gam[t], cq2 = plain ? cprev2[t] : ct2;
#pragma unroll
        for (int c0 = 0; c0 < 32; c0 += 16) {
          const int i0 = 32 * hf + c0;
          float c2[16], bt[16], gm[16], mq[16], m2[16];
          lds16(cum2 + i0, c2);
          lds16(bet + i0, bt);
          lds16(gam + i0, gm);
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int i = i0 + u;
            const float qk = p.scale * gv[c0 + u];
            const float dec = i <= t ? exp2f(ct2 - c2[u]) * qk : 0.f;
            mq[u] = i < t ? (plain ? exp2f(cq2 - c2[u]) * qk : dec) * bt[u] : 0.f;
            m2[u] = stl ? (i == t ? gtt * qk : 0.f) : gtt * dec * gm[u];
          }
          img_row16(img + IMG_APMQ, 16384, 64 + t, i0, mq);
          img_row16(img + IMG_M2, 8192, t, i0, m2);
        }
      }
    }
    __syncthreads();
    if (!rla) {  // T_beta (threads 0..127) and T_gamma (128..255)
      const int g = tid & 127;
      const float *A = tid < 128 ? Ab : Ag;
      float *Tm = tid < 128 ? Tb : Tg;
      float *W = Wsc + (tid < 128 ? 0 : 32 * LDW);
#pragma unroll 1
      for (int stage = 0; stage < 5; ++stage) {
        if (stage) __syncthreads();
        inv64_stage(stage, A, Tm, W, g);
      }
    }
    __syncthreads();
    {  // image rows of T: thread (row r, matrix m, half hf)
      const int r = tid & 63, m = (tid >> 6) & 1, hf = tid >> 7;
      const float *Tm = m ? Tg : Tb;
      uint8_t *dst = img + (m ? IMG_TG : IMG_TB);
#pragma unroll
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        if (rla || (m && stl)) {
#pragma unroll
          for (int u = 0; u < 16; ++u) v[u] = r == 32 * hf + c0 + u ? 1.f : 0.f;
        } else {
          lds16(Tm + r * LDT + 32 * hf + c0, v);
        }
        img_row16(dst, 8192, r, 32 * hf + c0, v);
      }
    }
    if (tid < C) {
      float *rec = p.ws + chunk * kRecFloats;
      const int t = tid;
      int s_, h_, cc_;
      rec_decode(p, (long long)chunk, s_, h_, cc_);
      const int n_ = min(C, seq_span(p, s_, h_).len - cc_ * C);  // valid tokens
      const float cC = cum[C - 1];
      rec[OFF_VEC + V_GAM + t] = __expf(cum[t]);
      rec[OFF_VEC + V_GPREV + t] = __expf(cprev[t]);
      rec[OFF_VEC + V_ALPHA + t] = __expf(gg[t]);
      rec[OFF_VEC + V_WS + t] = bet[t] * __expf(cC - cum[t]);
      rec[OFF_VEC + V_WR + t] = stl ? (t == n_ - 1 ? 1.f : 0.f) : gam[t] * __expf(cC - cum[t]);
      if (t == 0) rec[OFF_VEC + V_GAMC] = __expf(cC);
    }
  }
  if (!ok && tid == 0) {
    if (p.err) atomicExch(p.err, RDN_ERR_TIMEOUT);
    mma_commit(barD);  // the Gram product still in flight, before TMEM is freed
    mbar_wait(barD, 0);
  }
  cp_async_wait_all();  // no copy of this CTA outlives it (a fetch for a chunk not reached)
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, 64);
}

}  // namespace

cudaError_t launch_prep_tc(const FwdParams &p, bool rla, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(prep_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)pp::SMEM);
  if (e != cudaSuccess) return e;
  int dev = 0, nsm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  const size_t nct = (size_t)p.nrec;  // (packed sequences: a bound; the kernel reads the count)
  const unsigned grid = (unsigned)(nct < 2 * (size_t)nsm ? nct : 2 * (size_t)nsm);  // two per SM
  RDN_LAUNCH("chunk_prep", s, prep_tc_kernel<<<grid, NTH, pp::SMEM, s>>>(p, rla));
  return cudaGetLastError();
}

}  // namespace rdn
