// chunk_common.cuh -- layout of the per-chunk records shared by the
// chunkwise forward and backward, and a block-level fp32 product helper.
#pragma once
#include "common.cuh"

namespace rdn {

constexpr int C = kChunk;
constexpr int kThreads = 256;
constexpr int kDVS = 32;  // value columns per scan CTA

// Per-chunk workspace record written by chunk_prep (floats).
constexpr int kCC = C * C;
constexpr int OFF_TB = 0, OFF_TG = kCC, OFF_AP = 2 * kCC, OFF_MQ = 3 * kCC, OFF_M2 = 4 * kCC;
constexpr int OFF_VEC = 5 * kCC;
// vectors: Gam, Gprev, alpha, wS, wR, then GamC at [5*C]
constexpr int V_GAM = 0, V_GPREV = C, V_ALPHA = 2 * C, V_WS = 3 * C, V_WR = 4 * C, V_GAMC = 5 * C;
constexpr int kRecFloats = OFF_VEC + 6 * C;

// The tensor-core scan reads the same record in a second format: the chunk
// matrices as shared-memory images (bf16 hi + lo parts, K-major, 128-byte
// swizzled), copied to shared memory with bulk copies.  Byte offsets:
//   T_beta  hi | lo  (64 rows each)      [IMG_TB,   IMG_TB + 16 KB)
//   [Ap ; Mq] hi | lo (128 rows each)    [IMG_APMQ, IMG_APMQ + 32 KB)
//   T_gamma hi | lo                      [IMG_TG,   ...)
//   diag(gamma) M2 hi | lo               [IMG_M2,   ...)  (rows t scaled by gamma_t)
//   the gate vectors at the same place as in the fp32 record (OFF_VEC).
constexpr int IMG_TB = 0, IMG_APMQ = 16384, IMG_TG = 49152, IMG_M2 = 65536;
static_assert(IMG_M2 + 16384 == OFF_VEC * 4, "image fills the matrix part of the record");

// Block-level fp32 product over shared memory (NT threads): the calling thread
// gets acc[i] = sum_k A(m_i, k) B(k, n) for n = tid % N and m_i = tid / N + i * (NT / N).
// A(m,k) = A[m*a_m + k*a_k], B(k,n) = B[k*b_k + n*b_n].  With N >= 32 the lanes
// of a warp share m, so A reads are broadcasts.
template <int M, int N, int K, int NT = kThreads>
struct BlockMM {
  static constexpr int RG = NT / N;
  static constexpr int RPT = M / RG;
  static_assert(NT % N == 0 && M % RG == 0, "tile");
  __device__ static __forceinline__ void run(const float *A, int a_m, int a_k, const float *B,
                                             int b_k, int b_n, float (&acc)[RPT]) {
    const int n = threadIdx.x % N, rg = threadIdx.x / N;
#pragma unroll
    for (int i = 0; i < RPT; ++i) acc[i] = 0.f;
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
      const float bv = B[k * b_k + n * b_n];
#pragma unroll
      for (int i = 0; i < RPT; ++i) acc[i] = fmaf(A[(rg + i * RG) * a_m + k * a_k], bv, acc[i]);
    }
  }
  __device__ static __forceinline__ int row(int i) { return threadIdx.x / N + i * RG; }
  __device__ static __forceinline__ int col() { return threadIdx.x % N; }
};

// (I + A)^-1 for a 64 x 64 strictly lower A (row stride ld), by 16 x 16
// blocks, with 128 threads (g = thread index within the group):
//   diagonal blocks  T_ii = (I + A_ii)^-1 by forward substitution (one thread
//                    per block column, the column kept in registers);
//   block row i      W_j = sum_{k=j}^{i-1} A_ik T_kj,  T_ij = -T_ii W_j.
// W is scratch of 3 x 256 floats.  The caller synchronises the block between
// the calls of the 4 stages (stage 0: diagonal; stage i: block row i).
__device__ __forceinline__ void inv_diag_blocks(const float *A, float *Tm, int ld, int g) {
  if (g < 64) {
    const int blk = g >> 4, col = g & 15, b0 = blk * 16;
    float x[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      float s = (r == col) ? 1.f : 0.f;
#pragma unroll
      for (int m = 0; m < r; ++m) s = fmaf(-A[(b0 + r) * ld + b0 + m], x[m], s);
      x[r] = (r < col) ? 0.f : s;
    }
#pragma unroll
    for (int r = 0; r < 16; ++r) Tm[(b0 + r) * ld + b0 + col] = x[r];
  }
  // zero the strictly upper blocks once
  for (int e = g; e < 64 * 64; e += 128) {
    const int r = e >> 6, c = e & 63;
    if ((c >> 4) > (r >> 4)) Tm[r * ld + c] = 0.f;
  }
}
__device__ __forceinline__ void inv_block_row_w(const float *A, const float *Tm, float *W, int ld,
                                                int i, int g) {
  for (int e = g; e < i * 256; e += 128) {
    const int j = e >> 8, r = (e >> 4) & 15, cc = e & 15;
    float s = 0.f;
    for (int k = j; k < i; ++k)
#pragma unroll
      for (int m = 0; m < 16; ++m)
        s = fmaf(A[(16 * i + r) * ld + 16 * k + m], Tm[(16 * k + m) * ld + 16 * j + cc], s);
    W[e] = s;
  }
}
__device__ __forceinline__ void inv_block_row_t(float *Tm, const float *W, int ld, int i, int g) {
  for (int e = g; e < i * 256; e += 128) {
    const int j = e >> 8, r = (e >> 4) & 15, cc = e & 15;
    float s = 0.f;
#pragma unroll
    for (int m = 0; m < 16; ++m) s = fmaf(Tm[(16 * i + r) * ld + 16 * i + m], W[j * 256 + m * 16 + cc], s);
    Tm[(16 * i + r) * ld + 16 * j + cc] = -s;
  }
}

struct FwdParams {
  int B, T, H, NC;
  const void *q, *k, *v;
  const float *g, *beta, *gamma;
  float clip, scale;
  const float *S0, *R0;
  void *o;
  float *ST, *RT, *S_chunks, *R_chunks;
  float *ws;  // NC*B*H records of kRecFloats
  int *err;   // device status word (RDN_ERR_TIMEOUT if a bounded wait gave up) or NULL
  // forward intermediates kept for the backward (RDN_FLAG_SAVE_FOR_BWD) or NULL:
  // E, E2 per chunk as a 32 KB shared-memory image of E^T (rows j, columns t;
  // bf16 hi 16 KB | lo 16 KB, K-major, 128-byte swizzled), the clip mask as
  // [chunk][j] (bit t = |x| <= c)
  uint8_t *sv_E, *sv_E2;
  unsigned long long *sv_mask;
  // Packed variable-length sequences (rdn_fwd_args.cu_seqlens), or NULL for B
  // sequences of T tokens each: for s = 0 .. nseq, {first token, first chunk}
  // of sequence s (entry nseq closes the list: {T, total chunks}).
  const long long *seq;
  int nseq;        // sequences: B, or the number of packed sequences
  long long nrec;  // record slots: B * H * NC, or a bound on H * (total chunks)
  unsigned mods;   // the variant flags (RDN_FLAG_VARIANTS bits of rdn_fwd_args.flags)
  int f32out;      // o stored in fp32 (RDN_FLAG_F32_OUT on the tensor-core forward)
  int inject;      // 1: the tensor-core scan, 2: the backward chain skips its first MMA
                   // completion signal and waits ~5 ms for it (tests)
  // RDN_FLAG_QK_NORM: q and k above are then the normalised copies
  // SiLU(x) / max(||SiLU(x)||, qk_eps), written by the pass that makes the
  // chunk records (launch_t in chunk_fwd.cu), and qraw, kraw the caller's x
  const void *qraw, *kraw;
  float qk_eps;
  int qk_norm;
};

// Where sequence s's tokens and (s, h)'s chunk records are.  Token t of the
// sequence is row (tok0 + t) * H + h of the [tokens][H] inputs; chunk c of
// (s, h) is record rbase + c (also the index of its chunk-start states and
// saved intermediates).  With packed sequences the records of sequence s
// start at (its first chunk) * H, heads one after the other.
struct SeqSpan {
  long long tok0, rbase;
  int len, nc;
};
__host__ __device__ __forceinline__ SeqSpan seq_span(const FwdParams &p, int s, int h) {
  SeqSpan q;
  if (p.seq) {
    q.tok0 = p.seq[2 * s];
    q.len = (int)(p.seq[2 * s + 2] - q.tok0);
    q.nc = (q.len + C - 1) / C;
    q.rbase = p.seq[2 * s + 1] * p.H + (long long)h * q.nc;
  } else {
    q.tok0 = (long long)s * p.T;
    q.len = p.T;
    q.nc = p.NC;
    q.rbase = ((long long)s * p.H + h) * p.NC;
  }
  return q;
}
// chunk records in use (at most nseq * H * NC slots)
__device__ __forceinline__ long long total_records(const FwdParams &p) {
  return p.seq ? p.seq[2 * p.nseq + 1] * p.H : (long long)p.nseq * p.H * p.NC;
}
// record r -> (sequence s, head h, chunk c); r < total_records(p)
__device__ __forceinline__ void rec_decode(const FwdParams &p, long long r, int &s, int &h, int &c) {
  if (!p.seq) {
    if (r <= 0x7fffffffll) {  // (32-bit divisions: a 64-bit one is a long software routine)
      const unsigned ru = (unsigned)r, nc = (unsigned)p.NC, hn = (unsigned)p.H;
      const unsigned bh = ru / nc;
      c = (int)(ru - bh * nc);
      s = (int)(bh / hn);
      h = (int)(bh - (unsigned)s * hn);
      return;
    }
    const long long bh = r / p.NC;
    c = (int)(r - bh * p.NC);
    s = (int)(bh / p.H);
    h = (int)(bh - (long long)s * p.H);
    return;
  }
  int lo = 0, hi = p.nseq - 1;  // the last sequence whose records start at or before r
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.seq[2 * mid + 1] * p.H <= r) lo = mid; else hi = mid - 1;
  }
  s = lo;
  const int nc = (int)((p.seq[2 * s + 2] - p.seq[2 * s] + C - 1) / C);
  const long long off = r - p.seq[2 * s + 1] * p.H;  // < H * nc
  h = (int)((unsigned)off / (unsigned)nc);
  c = (int)(off - (long long)h * nc);
}

// Where the forward keeps those intermediates: after the nrec record slots.
// With the tanh residual (deriv) the clip mask's place holds the residual
// map's derivative instead, [chunk][j][t] as 16-bit fixed point (grad_q16).
struct SavedLayout {
  size_t e, e2, mask, bytes;  // byte offsets from the workspace base; region size
};
inline size_t mask_bytes_per_chunk(int Dv, bool deriv) {
  return deriv ? (size_t)Dv * C * 2 : (size_t)Dv * sizeof(unsigned long long);
}
inline SavedLayout saved_layout(size_t nct, int Dv, bool deriv) {
  SavedLayout l;
  l.e = nct * sizeof(float) * (size_t)kRecFloats;
  l.e2 = l.e + nct * sizeof(float) * C * Dv;
  l.mask = l.e2 + nct * sizeof(float) * C * Dv;
  l.bytes = l.mask + nct * mask_bytes_per_chunk(Dv, deriv) - l.e;
  return l;
}


inline FwdParams make_fwd_params(const rdn_fwd_args &a) {
  FwdParams p;
  p.B = a.B; p.T = a.T; p.H = a.H;
  p.NC = (a.T + C - 1) / C;
  p.q = a.q; p.k = a.k; p.v = a.v;
  p.g = a.g; p.beta = a.beta; p.gamma = a.gamma;
  p.clip = a.clip; p.scale = a.scale;
  p.S0 = a.S0; p.R0 = a.R0;
  p.o = a.o;
  p.ST = a.ST; p.RT = a.RT; p.S_chunks = a.S_chunks; p.R_chunks = a.R_chunks;
  p.ws = nullptr;
  p.err = nullptr;
  p.sv_E = p.sv_E2 = nullptr;
  p.sv_mask = nullptr;
  p.seq = nullptr;  // set by the launcher once the table is in its workspace
  p.nseq = call_seqs(a);
  p.nrec = call_records(a);
  p.mods = a.flags & RDN_FLAG_VARIANTS;
  p.f32out = (a.flags & RDN_FLAG_F32_OUT) && a.dtype == RDN_BF16;
  p.inject = 0;
  p.qraw = a.q;
  p.kraw = a.k;
  p.qk_eps = a.qk_eps;
  p.qk_norm = (a.flags & RDN_FLAG_QK_NORM) ? 1 : 0;
  return p;
}

// RDN_FLAG_QK_NORM: the normalised q, then k, [tokens][H][Dk] in dtype, at
// qk_norm_offset bytes into the forward's workspace (after the records and
// the saved intermediates) and in the backward's when it makes its own records.
inline size_t qk_norm_bytes(const rdn_fwd_args &a) {
  if (!(a.flags & RDN_FLAG_QK_NORM)) return 0;
  const size_t esz = a.dtype == RDN_BF16 ? 2 : 4;
  return 2 * esz * (size_t)a.B * a.T * a.H * a.Dk;  // (a multiple of 256)
}
inline size_t qk_norm_offset(const rdn_fwd_args &a) {
  const size_t nrec = (size_t)call_records(a);
  size_t off = sizeof(float) * (size_t)kRecFloats * nrec;
  if (a.flags & RDN_FLAG_SAVE_FOR_BWD)
    off += saved_layout(nrec, a.Dv, a.flags & RDN_FLAG_TANH_RESIDUAL).bytes;
  return off;
}
// Points p.q, p.k at the normalised copies starting at `base`.
inline void set_qk_norm_copies(FwdParams &p, const rdn_fwd_args &a, char *base) {
  const size_t half = qk_norm_bytes(a) / 2;
  p.q = base;
  p.k = base + half;
}

// The variant flags the tensor-core kernels implement: all four (the decayed
// residual, the plain combine, the tanh residual, the stateless correction).
constexpr unsigned kTcVariants = RDN_FLAG_DECAYED_RESIDUAL | RDN_FLAG_PLAIN_COMBINE |
                                 RDN_FLAG_TANH_RESIDUAL | RDN_FLAG_STATELESS_AUX;
// Whether the forward runs the tensor-core scan (and its records are
// shared-memory images): bf16 inputs, d = 128, no variant flag outside
// kTcVariants, for RDN and RLA alike.
inline bool fwd_uses_tc(const FwdParams &p, int DK, bool bf16) {
  return bf16 && DK == 128 && (p.mods & ~kTcVariants) == 0;
}

// Tensor-core scan (fwd_tc.cu): bf16 inputs with d_k = d_v = 128.
cudaError_t launch_fwd_tc(const FwdParams &p, bool rdnv, cudaStream_t s);

// Prep kernel alone; img selects the shared-memory-image record format read
// by the tensor-core kernels (else the fp32 format of the SIMT kernels).
cudaError_t launch_prep(const FwdParams &p, int DK, bool rdnv, bool bf16, bool img, cudaStream_t s);

// Tensor-core backward (bwd_tc.cu): recompute, chain and post kernels.
cudaError_t launch_prep_tc(const FwdParams &p, bool rla, cudaStream_t s);
size_t bwd_tc_extra_bytes(long long nrec, bool deriv);  // (deriv: the tanh residual's)
cudaError_t launch_bwd_tc(const FwdParams &f, const void *dO, const float *dST, const float *dRT,
                          const float *Sc, const float *Rc, void *dq, void *dk, void *dv, float *dg,
                          float *dbeta, float *dgamma, float *dS0, float *dR0, char *extra,
                          bool rla, bool grad_f32, bool dqk_f32, cudaStream_t s);

// Launch the forward's prep kernel (per-chunk records into p.ws) and/or its
// scan kernel (outputs, optional chunk-start states).
cudaError_t launch_fwd_parts(const FwdParams &p, int DK, bool rdnv, bool bf16, bool do_prep,
                             bool do_scan, cudaStream_t s);

}  // namespace rdn
