// fwd_tc.cu -- tensor-core (tcgen05 / TMEM) scan of the chunkwise RLA / RDN
// forward, bf16 inputs, d_k = d_v = 128.
//
// Same chunk algebra as chunk_fwd.cu (see its header), computed in the
// transposed orientation so that every product has the value dimension
// d_v = 128 as its M dimension: TMEM lane j holds value column j.  The CTA's
// 16 warps form 4 groups of 128 threads; thread j of group g owns value
// column j for the token columns t in [16g, 16g + 16) of the chunk (and the
// state columns [16g, 16g + 16) and [64 + 16g, 80 + 16g)), so that the four
// warps sharing a TMEM lane quadrant hide one another's latencies.  Per chunk of 64
// tokens, with KQ = [K ; Q] (128 x d_k, exact bf16, unscaled):
//
//   MMA1  D1   = S^T  KQ^T          -> [KS | QS]                  (N=128, K=128)
//   MMA5  D3   = R^T  KQ^T          -> [KR | QR] (chunk-start R, issued with MMA1)
//         X    = V - Gam*KS         (= V - alpha * Gprev*KS); QS rescaled in TMEM
//                                      to Gam*scale*QS
//   MMA2  E^T  = X^T  T_beta^T      (over KS; Gprev*KS back in its place after)
//   MMA3  D1  += E^T  [Ap ; Mq]^T   -> [P | Ob]                   (N=128, K=64)
//   MMA4  S   += (wS E)^T K         onto S scaled by Gam_C in TMEM while MMA1
//                                      ran: S_C = Gam_C S + U       (N=128, K=64)
//         r    = clip(V - P)        (Section 3.3; kept in registers)
//         X2   = r - Gam*KR
//   MMA6  E2^T = X2^T T_gamma^T
//   MMA7  D1[:, Ob half] += E2^T (diag(gamma) M2)^T
//   MMA8  R   += (wR E2)^T K        onto R scaled by Gam_C during MMA1: R_C
//         o    = D1[:, Ob half] + gamma * Gam*scale*QR   (= Ob + gamma * Oa)
//
// RLA skips MMA2 and MMA6 (E = V, E2 = r).  X, E, wS E and their auxiliary
// counterparts (magnitude ~ |v|) enter the MMAs as bf16 hi + lo pairs, which
// keeps their rounding well below the state's own scale; so does S in MMA1
// (hi + lo copies); R and the chunk's K, Q are single bf16 (K, Q exactly).
// The states S, R live in TMEM in fp32 for the whole sequence; their bf16
// copies (the A operands of MMA1 and MMA5) are rewritten in shared memory
// after each update.  The chunk's V
// and [K ; Q] tiles are fetched by cp.async while the previous chunk
// finishes.  One thread issues the MMAs; every wait is an mbarrier wait with
// a time limit.  The state-independent chunk matrices (T_beta, T_gamma, Ap,
// Mq, diag(gamma) M2) come from chunk_prep's records as bf16 hi + lo
// shared-memory images; they are streamed into two slots by bulk copies one
// phase ahead of their use (slot A: T_beta then T_gamma; slot B: [Ap;Mq] then
// M2) and enter the MMAs as three products (hi*hi + hi*lo + lo*hi).
//
// TMEM (512 columns): [0,128) S   [128,256) R   [256,384) D1   [384,512) D3
// (D1 holds KS|QS, then E | Ob, Gprev KS + Ap E = P | Ob, then E2 | Ob + gamma M2 E2).
#include <cuda.h>
#include <cudaTypedefs.h>

#include "chunk_common.cuh"
#include "tc_common.cuh"

namespace rdn {
namespace {

using namespace tc;

constexpr int D = 128;
constexpr int kTcThreads = 512;
constexpr int kGroups = kTcThreads / 128;  // threads sharing a value column
static_assert(kGroups == 4, "each group owns 16 of a chunk's 64 token columns");

// shared-memory carve-up (bytes from the 1024-aligned dynamic base)
constexpr uint32_t SM_SA = 0;          // S^T bf16, 128 x 128, two 64-col blocks
constexpr uint32_t SM_RA = 32768;      // R^T bf16
constexpr uint32_t SM_KQ = 65536;      // [K ; Q] unscaled, 128 rows x 128, two 64-col blocks
                                       // (K rows also serve as the MN-major B of the updates)
constexpr uint32_t SM_V = 98304;       // V, 64 rows t x 128 columns j, two 8 KB blocks
constexpr uint32_t SM_SLOTA = 114688;  // T_beta then T_gamma image (hi | lo), 16 KB
constexpr uint32_t SM_SLOTB = 131072;  // [Ap;Mq] then M2 image (hi | lo), 32 KB
// value-like operands are split into bf16 hi + lo parts (two MMAs each):
constexpr uint32_t SM_XE = 163840;     // X^T then E^T (X2^T then E2^T), hi part, 128 x 64
constexpr uint32_t SM_XE_LO = 180224;  //   lo part
constexpr uint32_t SM_W = 196608;      // (wS E)^T / (wR E2)^T, hi part
constexpr uint32_t SM_W_LO = 212992;   //   lo part
constexpr uint32_t SM_VEC = 229376;    // 7 x 64 fp32: Gam Gprev (unused) wS wR gamma, GamC
// 5 mbarriers: MMA, slot A, slot B, drain, tile copies
constexpr uint32_t SM_BAR = SM_VEC + 7 * 64 * 4;
constexpr uint32_t SM_SLOT = SM_BAR + 40;
constexpr uint32_t SM_FLAG = SM_SLOT + 4;
constexpr uint32_t SM_BYTES = SM_FLAG + 4;
constexpr size_t kTcSmem = SM_BYTES;
static_assert(kTcSmem <= 232448, "shared memory");

constexpr uint32_t T_S = 0, T_R = 128, T_D1 = 256, T_X = 384;  // T_X: D3

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Write 16 consecutive values (columns c0..c0+15 of row r) of a K-major SW128
// tile whose 64-column blocks are blk_bytes apart.
__device__ __forceinline__ void st_row16(uint8_t *tile, uint32_t blk_bytes, int r, int c0,
                                         const float (&v)[16]) {
  uint8_t *blk = tile + (c0 >> 6) * blk_bytes;
  const int cc = c0 & 63;
  uint4 a, b;
  a.x = pack_bf16(v[0], v[1]);
  a.y = pack_bf16(v[2], v[3]);
  a.z = pack_bf16(v[4], v[5]);
  a.w = pack_bf16(v[6], v[7]);
  b.x = pack_bf16(v[8], v[9]);
  b.y = pack_bf16(v[10], v[11]);
  b.z = pack_bf16(v[12], v[13]);
  b.w = pack_bf16(v[14], v[15]);
  *reinterpret_cast<uint4 *>(blk + sw128(r, cc)) = a;
  *reinterpret_cast<uint4 *>(blk + sw128(r, cc + 8)) = b;
}

// Same, split into bf16 hi + lo parts (split_pack_bf16) in two tiles.
__device__ __forceinline__ void st_row16_split(uint8_t *hi, uint8_t *lo, int r, int c0,
                                               const float (&v)[16]) {
  uint32_t h[8], l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) split_pack_bf16(v[2 * i], v[2 * i + 1], h[i], l[i]);
  const int cc = c0 & 63;
  *reinterpret_cast<uint4 *>(hi + sw128(r, cc)) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4 *>(hi + sw128(r, cc + 8)) = make_uint4(h[4], h[5], h[6], h[7]);
  *reinterpret_cast<uint4 *>(lo + sw128(r, cc)) = make_uint4(l[0], l[1], l[2], l[3]);
  *reinterpret_cast<uint4 *>(lo + sw128(r, cc + 8)) = make_uint4(l[4], l[5], l[6], l[7]);
}

// D (+)= (A_hi + A_lo)(B_hi + B_lo)^T without the lo*lo term: three MMAs
// over K = 64 for K-major 128B-swizzled tiles.
__device__ __forceinline__ void mma_split3(uint32_t d, uint32_t a_hi, uint32_t a_lo,
                                           uint32_t b_hi, uint32_t b_lo, uint32_t idesc,
                                           bool accumulate_first) {
  mma_tile(d, a_hi, 0, b_hi, 0, 4, idesc, accumulate_first);
  mma_tile(d, a_hi, 0, b_lo, 0, 4, idesc, true);
  mma_tile(d, a_lo, 0, b_hi, 0, 4, idesc, true);
}

// kGeneric: the variant flags (FwdParams::mods) are read; the method's
// instances have them folded away
// Tensor maps (CUtensorMap, 64-byte aligned) over v, k, q as [tokens][H][D]
// with a 64-token x 64-column box (make_tile_map); ok: they are valid.
struct FwdMaps {
  alignas(64) unsigned char v[128];
  alignas(64) unsigned char k[128];
  alignas(64) unsigned char q[128];
  bool ok;
};

template <bool RDNV, bool kGeneric>
__global__ void __launch_bounds__(kTcThreads, 1)
    fwd_tc_kernel(FwdParams p, const __grid_constant__ FwdMaps maps) {
  extern __shared__ __align__(1024) uint8_t sm[];
  const uint32_t sbase = smem_u32(sm);
  if (sbase & 1023u) {  // the swizzled tiles need a 1024-byte aligned base
    if (threadIdx.x == 0 && p.err) atomicExch(p.err, RDN_ERR_CUDA);
    return;
  }
  float *vec = reinterpret_cast<float *>(sm + SM_VEC);
  float *Gam = vec, *Gprev = vec + 64, *wS = vec + 192, *wR = vec + 256,
        *gamv = vec + 320;
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm + SM_BAR);
  uint64_t *barA = bar + 1, *barB = bar + 2;  // slot A / slot B bulk copies
  uint64_t *barD = bar + 3;  // the drain after a wait that gave up
  uint64_t *barE = bar + 4;  // a whole chunk's V, K, Q tiles by tensor-map copies
  uint32_t *slot = reinterpret_cast<uint32_t *>(sm + SM_SLOT);
  volatile int *flag = reinterpret_cast<volatile int *>(sm + SM_FLAG);

  const int tid = threadIdx.x, warp = tid >> 5;
  const int j = tid & 127;       // value column == TMEM lane
  const int g16 = (warp >> 2) * 16;  // this thread's token (and state) columns start
  const int bh = blockIdx.x;
  const int h = bh % p.H;
  const SeqSpan sp = seq_span(p, bh / p.H, h);  // this (sequence, head)'s tokens and records
  const long long tok0 = sp.tok0;
  const int T = sp.len, H = p.H, NC = sp.nc;
  const __nv_bfloat16 *q = (const __nv_bfloat16 *)p.q;
  const __nv_bfloat16 *k = (const __nv_bfloat16 *)p.k;
  const __nv_bfloat16 *v = (const __nv_bfloat16 *)p.v;
  __nv_bfloat16 *o = (__nv_bfloat16 *)p.o;
  const float clip = p.clip;
  const bool dec_res = kGeneric && (p.mods & RDN_FLAG_DECAYED_RESIDUAL);
  const bool plain = kGeneric && (p.mods & RDN_FLAG_PLAIN_COMBINE);  // o = S_{t-1} q + R_t q
  // the log-cosh residual r = c tanh(x / c); the backward then reads the
  // derivative 1 - (r / c)^2 of each element (16-bit fixed point) where the
  // clip mask goes
  const bool tnh = kGeneric && (p.mods & RDN_FLAG_TANH_RESIDUAL);
  // the stateless correction R_t = r_t k_t^T: no read-out of the carried R
  // (X2 = r, no gamma Gam Q R term in o), R not carried over a chunk (scaled
  // by 0); the records hold the identity T_gamma, diag(gamma qk) and the
  // one-hot wR that make the rest of the pass compute it
  const bool stl = kGeneric && (p.mods & RDN_FLAG_STATELESS_AUX);
  const size_t st_base = (size_t)bh * D * D;

  if (tid == 0) {
    mbar_init(bar, 1);
    mbar_init(barA, 1);
    mbar_init(barB, 1);
    mbar_init(barD, 1);
    mbar_init(barE, 1);
    fence_mbar_init();
    *flag = 0;
  }
  if (warp == 0) tmem_alloc(slot, 512);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tm = *slot;
  const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
  uint32_t phase = 0, phA = 0, phB = 0;  // phA/phB: tracked by thread 0 only
  bool pendA = false, pendB = false;      // (thread 0) a slot copy armed and not yet waited for
  // the waits on the MMAs: normally about a second; a test (p.inject) skips the
  // first phase's completion signal and waits about 5 ms for it instead
  const long long mma_limit = p.inject == 1 ? 10000000ll : 2000000000ll;
  bool skip_commit = p.inject == 1;
  // S - bf16(S) as a second bf16 image (rows j), so that the read-outs K S,
  // Q S use S to ~16 bits.  RLA's state is not contracted by a delta term and
  // its prediction S k is a large sum the residual v - S k cancels against;
  // RDN's single-bf16 read-outs put the output error of the long-context
  // workload (T = 16384) at the 2e-2 RMS bound.  The image lives in tiles that
  // are free from the end of a chunk to the next one's MMA1 / MMA3: RDN the
  // X/E^T pair (key blocks 0 | 1), RLA (no T matrices) slot A and the E^T lo tile.
  constexpr uint32_t kSloBase = RDNV ? SM_XE : SM_SLOTA;
  constexpr uint32_t kSloBlk = RDNV ? SM_XE_LO - SM_XE : SM_XE_LO - SM_SLOTA;
  auto store_state_lo = [&](int c0, const float (&s)[16]) {
    float lo[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) lo[i] = s[i] - __bfloat162float(__float2bfloat16_rn(s[i]));
    st_row16(sm + kSloBase, kSloBlk, j, c0, lo);
  };
  auto rec_of = [&](int c) {
    return reinterpret_cast<const uint8_t *>(p.ws + (size_t)(sp.rbase + c) * kRecFloats);
  };
  // thread 0: start the bulk copy of a chunk-matrix image into a slot
  auto load_slot = [&](uint8_t *dst, uint64_t *b, const uint8_t *src, uint32_t bytes) {
    mbar_expect_tx(b, bytes);
    bulk_g2s(dst, src, bytes, b);
    (b == barA ? pendA : pendB) = true;
  };
  if (tid == 0 && NC > 0) {  // (a packed sequence may be empty)
    if (RDNV) load_slot(sm + SM_SLOTA, barA, rec_of(0) + IMG_TB, 16384);
    load_slot(sm + SM_SLOTB, barB, rec_of(0) + IMG_APMQ, 32768);
  }
  // chunk tiles (rows t, exact bf16, zero past the sequence end), asynchronous;
  // the next chunk's are fetched while the current one finishes
  auto fetch_v = [&](int c) {
    const int t0 = c * 64, n = min(64, T - t0);
    for (int e = tid; e < 64 * 16; e += kTcThreads) {
      const int t = e >> 4, ch = e & 15;
      const bool vld = t < n;
      const size_t off = ((size_t)(tok0 + t0 + (vld ? t : 0)) * H + h) * D + ch * 8;
      cp_async16(sm + SM_V + (ch >> 3) * 8192 + sw128(t, (ch & 7) * 8), v + off, vld);
    }
  };
  auto fetch_kq = [&](int c) {
    const int t0 = c * 64, n = min(64, T - t0);
    for (int e = tid; e < 64 * 16; e += kTcThreads) {
      const int t = e >> 4, ch = e & 15;
      const bool vld = t < n;
      const size_t off = ((size_t)(tok0 + t0 + (vld ? t : 0)) * H + h) * D + ch * 8;
      const int blk = ch >> 3, cc = (ch & 7) * 8;
      cp_async16(sm + SM_KQ + blk * 16384 + sw128(t, cc), k + off, vld);
      cp_async16(sm + SM_KQ + blk * 16384 + sw128(64 + t, cc), q + off, vld);
    }
  };
  // v[t, j] of the current chunk from its tile
  auto vs = [&](int t) {
    return __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(
        sm + SM_V + (j >> 6) * 8192 + sw128(t, j & 63)));
  };
  if (NC > 0) {
    fetch_v(0);
    fetch_kq(0);
  }
  // Chunks between the first and the last are whole: with tensor maps thread 0
  // brings their V (after step (e)) and K, Q (after step (g)) tiles by tiled
  // bulk copies on one phase of barrier E, and no cp.async wait is needed for
  // them.  The first chunk is fetched above and the last one, which may be
  // ragged, by cp.async with zero fill.
  const bool tma = maps.ok;
  auto by_tma = [&](int cc) { return tma && cc > 0 && cc < NC - 1; };
  uint32_t phE = 0;    // phases of barrier E waited for
  bool pendE = false;  // (thread 0) a phase armed and not yet waited for
  auto tma_v = [&](int cc) {  // (thread 0) arms barrier E for the chunk's three tiles
    const int row = (int)(tok0 + (long long)cc * 64);
    mbar_expect_tx(barE, 49152);
    pendE = true;
    for (int kb = 0; kb < 2; ++kb) tma_load_3d(sm + SM_V + kb * 8192, maps.v, 64 * kb, h, row, barE);
  };
  auto tma_kq = [&](int cc) {
    const int row = (int)(tok0 + (long long)cc * 64);
    for (int kb = 0; kb < 2; ++kb) {
      tma_load_3d(sm + SM_KQ + kb * 16384, maps.k, 64 * kb, h, row, barE);
      tma_load_3d(sm + SM_KQ + kb * 16384 + 8192, maps.q, 64 * kb, h, row, barE);
    }
  };

  // initial states -> TMEM (fp32) and bf16 A operands
  for (int c0 = g16; c0 < D; c0 += 64) {
    float s[16], r[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      s[i] = p.S0 ? p.S0[st_base + (size_t)(c0 + i) * D + j] : 0.f;
      r[i] = p.R0 ? p.R0[st_base + (size_t)(c0 + i) * D + j] : 0.f;
    }
    tmem_st16(tm + lane + T_S + c0, s);
    tmem_st16(tm + lane + T_R + c0, r);
    st_row16(sm + SM_SA, 16384, j, c0, s);
    st_row16(sm + SM_RA, 16384, j, c0, r);
    store_state_lo(c0, s);
    if (p.S_chunks && NC > 0) {  // the first chunk's start states, for the backward
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        p.S_chunks[(size_t)sp.rbase * D * D + (size_t)(c0 + i) * D + j] = s[i];
        p.R_chunks[(size_t)sp.rbase * D * D + (size_t)(c0 + i) * D + j] = r[i];
      }
    }
  }

  // one MMA phase: make smem writes visible, issue, run `during` (work that
  // the MMAs do not touch), wait.  Returns false on timeout (the caller aborts).
  auto run_phase = [&](auto issue, auto during) -> bool {
    fence_async_smem();
    fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      fence_after_sync();
      if (!issue()) *flag = 1;  // a slot's bulk copy did not arrive in time
      if (!skip_commit) mma_commit(bar);
      skip_commit = false;
    }
    during();
    const bool ok = mbar_wait(bar, phase, mma_limit);
    phase ^= 1u;
    if (!ok) *flag = 1;
    __syncthreads();
    fence_after_sync();
    return *flag == 0;
  };

  // L2 prefetch of a chunk's record and V, K, Q rows and gammas, one chunk
  // ahead of the cp.async and bulk copies that read them
  auto prefetch_chunk = [&](int c) {
    const int t0_ = c * 64, n_ = min(64, T - t0_);
    if (tid == 0) {
      const uint8_t *r = rec_of(c);
      static_assert((kRecFloats * 4) % 16 == 0 && kRecFloats * 4 > 65536, "record");
      prefetch_l2_bulk(r, 65536);
      prefetch_l2_bulk(r + 65536, kRecFloats * 4 - 65536);
    }
    if (tid < 384) {
      const int rr = tid >> 1, t = rr & 63, w = rr >> 6;
      const __nv_bfloat16 *src = w == 0 ? v : (w == 1 ? k : q);
      if (t < n_) prefetch_l2_line(src + ((size_t)(tok0 + t0_ + t) * H + h) * D + (tid & 1) * 64);
    } else if (tid < 416) {
      const int t = 2 * (tid - 384);
      if (t < n_) prefetch_l2_line(p.gamma + (size_t)(tok0 + t0_ + t) * H + h);
    }
  };

  auto nothing = [] {};
  // a state's TMEM copy times the chunk's total decay, in place (its updates
  // accumulate onto it); this thread's columns.  The values it reads are the
  // chunk-start state, which goes to `start` ([i][j], fp32; NULL = not kept)
  // here, while MMA1 runs: stores on the path between the chunks cost the
  // scan 18 % (0.13 of 0.73 ms on the bench workload).
  auto scale_state = [&](uint32_t col, float f, float *start) {
    float x[16], y[16];
    tmem_ld16x2(tm + lane + col + g16, x, tm + lane + col + g16 + 64, y);
    if (start) {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        start[(size_t)(g16 + i) * D + j] = x[i];
        start[(size_t)(g16 + 64 + i) * D + j] = y[i];
      }
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      x[i] *= f;
      y[i] *= f;
    }
    tmem_st16(tm + lane + col + g16, x);
    tmem_st16(tm + lane + col + g16 + 64, y);
  };

  // a chunk's gate values (threads 0..63, one token each) and its total decay,
  // loaded into registers one chunk ahead of their use
  struct Pre {
    float gm, gp, ws, wr, g, gc;
  };
  auto fetch_pre = [&](int c) {
    const float *rc = p.ws + (size_t)(sp.rbase + c) * kRecFloats;
    const int t0_ = c * 64, n_ = min(64, T - t0_);
    Pre x;
    x.gm = x.gp = x.ws = x.wr = x.g = 0.f;
    if (tid < 64) {
      x.gm = rc[OFF_VEC + V_GAM + tid];
      x.gp = rc[OFF_VEC + V_GPREV + tid];
      x.ws = rc[OFF_VEC + V_WS + tid];
      x.wr = rc[OFF_VEC + V_WR + tid];
      x.g = tid < n_ ? p.gamma[(size_t)(tok0 + t0_ + tid) * H + h] : 0.f;
    }
    x.gc = rc[OFF_VEC + V_GAMC];
    return x;
  };
  Pre pre{};
  if (NC > 0) pre = fetch_pre(0);

  float rres[16];  // clipped residual r[t] of column j, t in [g16, g16 + 16)
  bool alive = true;
  for (int c = 0; c < NC && alive; ++c) {
    const int t0 = c * 64;
    const int n = min(64, T - t0);
    if (c + 1 < NC) prefetch_chunk(c + 1);
    // this chunk's V, K, Q tiles (fetched during the previous chunk)
    if (by_tma(c)) {
      if (!mbar_wait(barE, phE & 1u)) *flag = 1;
      ++phE;
      if (tid == 0) pendE = false;
    } else {
      cp_async_wait_all();
    }
    __syncthreads();  // every thread is done with the previous chunk's tiles and vectors
    if (*flag) {
      alive = false;
      break;
    }

    // ---- (a) chunk inputs -> shared memory (the chunk-start states for the
    // backward are stored while MMA1 runs; the first chunk's with the initial
    // states)
    float *sc_cur = (p.S_chunks && c > 0) ? p.S_chunks + (size_t)(sp.rbase + c) * D * D : nullptr;
    float *rc_cur = sc_cur ? p.R_chunks + (size_t)(sp.rbase + c) * D * D : nullptr;
    if (tid < 64) {
      Gam[tid] = pre.gm;
      Gprev[tid] = pre.gp;
      wS[tid] = pre.ws;
      wR[tid] = pre.wr;
      gamv[tid] = pre.g;
    }
    const float GamC = pre.gc;
    if (c + 1 < NC) pre = fetch_pre(c + 1);  // in flight during this chunk
    __syncthreads();

    // ---- (b) MMA1: D1 = S^T [K ; Q]^T and MMA5: X = R^T [K ; Q]^T (unscaled
    // read-outs K S | Q S and K R | Q R; both from the chunk-start states);
    // meanwhile the TMEM states are scaled by Gam_C, for MMA4 and MMA8 to
    // accumulate onto (the MMAs read the states' bf16 copies)
    alive = run_phase([&] {
      if (p.sv_E2) bulk_wait_read();  // the E2^T tiles of the previous chunk are rewritten next
      mma_tile(tm + T_D1, sbase + SM_SA, 16384, sbase + SM_KQ, 16384, 8, idesc_bf16(128, 128),
               false);
      // + the state's lo part
      mma_tile(tm + T_D1, sbase + kSloBase, kSloBlk, sbase + SM_KQ, 16384, 8,
               idesc_bf16(128, 128), true);
      mma_tile(tm + T_X, sbase + SM_RA, 16384, sbase + SM_KQ, 16384, 8, idesc_bf16(128, 128),
               false);
      return true;
    }, [&] {
      scale_state(T_S, GamC, sc_cur);
      scale_state(T_R, stl ? 0.f : GamC, rc_cur);
    });
    if (!alive) break;
    // Ob accumulates onto Gam * scale * QS
    float gks[16], vv[16];  // gks: K S, then Gprev K S; vv: this thread's V entries, until (e)
    {
      const int c0 = g16;
      float x[16], gm[16];
      tmem_ld16x2(tm + lane + T_D1 + 64 + c0, x, tm + lane + T_D1 + c0, gks);
      lds16(plain ? Gprev + c0 : Gam + c0, gm);
#pragma unroll
      for (int i = 0; i < 16; ++i) x[i] *= gm[i] * p.scale;
      tmem_st16(tm + lane + T_D1 + 64 + c0, x);
    }

    // ---- (c) X = V - Gam KS (= V - alpha Gprev KS)  ->  MMA2: E^T = X^T T_beta^T into
    // D1[0,64) (over KS); P accumulates onto Gprev KS, kept in registers until then
    {
      const int c0 = g16;
      float x[16], gm[16], gp[16];
      lds16(Gam + c0, gm);
      lds16(Gprev + c0, gp);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        vv[i] = vs(c0 + i);
        x[i] = vv[i] - gm[i] * gks[i];
        gks[i] *= dec_res ? gm[i] : gp[i];  // (decayed residual: P = a S_{t-1} k)
      }
      if (RDNV)
        st_row16_split(sm + SM_XE, sm + SM_XE_LO, j, c0, x);
      else
        tmem_st16(tm + lane + T_D1 + c0, gks);
    }
    if (RDNV) {
      alive = run_phase([&] {
        if (!mbar_wait(barA, phA)) return false;
        phA ^= 1u;
        pendA = false;
        mma_split3(tm + T_D1, sbase + SM_XE, sbase + SM_XE_LO, sbase + SM_SLOTA,
                   sbase + SM_SLOTA + 8192, idesc_bf16(128, 64), false);
        return true;
      }, nothing);
      if (!alive) break;
      if (tid == 0) load_slot(sm + SM_SLOTA, barA, rec_of(c) + IMG_TG, 16384);
    }

    // ---- (d) E -> EA, wS*E -> WA, Gprev KS -> D1[0,64);  MMA3: D1 += E^T [Ap;Mq]^T,
    // MMA4: S += (wS E)^T K
    const size_t ci = (size_t)(sp.rbase + c);  // chunk index of the saved intermediates
    {
      const int c0 = g16;
      float e[16], w[16];
      if (RDNV) {
        tmem_ld16(tm + lane + T_D1 + c0, e);
        tmem_st16(tm + lane + T_D1 + c0, gks);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) e[i] = vv[i];
      }
      lds16(wS + c0, w);
#pragma unroll
      for (int i = 0; i < 16; ++i) w[i] *= e[i];
      st_row16_split(sm + SM_XE, sm + SM_XE_LO, j, c0, e);
      st_row16_split(sm + SM_W, sm + SM_W_LO, j, c0, w);
    }
    alive = run_phase([&] {
      if (!mbar_wait(barB, phB)) return false;
      phB ^= 1u;
      pendB = false;
      mma_split3(tm + T_D1, sbase + SM_XE, sbase + SM_XE_LO, sbase + SM_SLOTB,
                 sbase + SM_SLOTB + 16384, idesc_bf16(128, 128), true);
      if (p.sv_E) {  // keep the E^T image (hi | lo) for the backward
        static_assert(SM_XE_LO == SM_XE + 16384, "contiguous");
        bulk_s2g(p.sv_E + ci * 32768, sm + SM_XE, 32768);
        bulk_commit();
      }
      mma_tile_kmn(tm + T_S, sbase + SM_W, 0, sbase + SM_KQ, 16384, 4, idesc_bf16(128, 128),
                   true);
      mma_tile_kmn(tm + T_S, sbase + SM_W_LO, 0, sbase + SM_KQ, 16384, 4, idesc_bf16(128, 128),
                   true);
      return true;
    }, nothing);
    if (!alive) break;
    if (tid == 0) load_slot(sm + SM_SLOTB, barB, rec_of(c) + IMG_M2, 16384);

    // ---- (e) r = clip(V - P); S (= Gam_C S + U, fp32 in TMEM) -> bf16 copy in SA
    {
      const int c0 = g16;
      unsigned msk = 0u;  // bit i: |x| <= c at t = c0 + i (the clip passes the gradient)
      float pp[16];
      tmem_ld16(tm + lane + T_D1 + c0, pp);
      if (!tnh) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float x = vv[i] - pp[i];
          if (fabsf(x) <= clip) msk |= 1u << i;
          rres[i] = clampf(x, clip);
        }
        // bits [c0, c0 + 16) of the column's 64-bit mask word (little-endian)
        if (p.sv_mask) reinterpret_cast<uint16_t *>(p.sv_mask + ci * D + j)[c0 >> 4] = (uint16_t)msk;
      } else {
        uint32_t dg[8];  // the derivative at t = c0 .. c0 + 15, pairs of 16-bit words
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          const float x0 = vv[i] - pp[i], x1 = vv[i + 1] - pp[i + 1];
          rres[i] = resid_map(x0, clip, true);
          rres[i + 1] = resid_map(x1, clip, true);
          dg[i / 2] = grad_q16(resid_grad(x0, clip, true)) |
                      (grad_q16(resid_grad(x1, clip, true)) << 16);
        }
        if (p.sv_mask) {
          uint4 *dst = reinterpret_cast<uint4 *>(reinterpret_cast<uint16_t *>(p.sv_mask) +
                                                 (ci * D + j) * 64 + c0);
          dst[0] = make_uint4(dg[0], dg[1], dg[2], dg[3]);
          dst[1] = make_uint4(dg[4], dg[5], dg[6], dg[7]);
        }
      }
    }
    {
      float s0[16], s1[16];
      tmem_ld16x2(tm + lane + T_S + g16, s0, tm + lane + T_S + g16 + 64, s1);
      st_row16(sm + SM_SA, 16384, j, g16, s0);
      st_row16(sm + SM_SA, 16384, j, g16 + 64, s1);
    }
    if (tid == 0 && p.sv_E) bulk_wait_read();  // the E^T tiles are rewritten next
    __syncthreads();
    if (c + 1 < NC) {  // every thread is past its last read of V
      if (!by_tma(c + 1))
        fetch_v(c + 1);
      else if (tid == 0)
        tma_v(c + 1);
    }

    // ---- (f) X2 = r - Gam KR;  MMA6: E2^T = X2^T T_gamma^T (into D1[0,64))
    if (RDNV) {
      {
        const int c0 = g16;
        float x[16], gm[16];
        tmem_ld16(tm + lane + T_X + c0, x);
        lds16(Gam + c0, gm);
#pragma unroll
        for (int i = 0; i < 16; ++i) x[i] = stl ? rres[i] : rres[i] - gm[i] * x[i];
        st_row16_split(sm + SM_XE, sm + SM_XE_LO, j, c0, x);
      }
      alive = run_phase([&] {
        if (!mbar_wait(barA, phA)) return false;
        phA ^= 1u;
        pendA = false;
        mma_split3(tm + T_D1, sbase + SM_XE, sbase + SM_XE_LO, sbase + SM_SLOTA,
                   sbase + SM_SLOTA + 8192, idesc_bf16(128, 64), false);
        return true;
      }, nothing);
      if (!alive) break;
      if (tid == 0 && c + 1 < NC) load_slot(sm + SM_SLOTA, barA, rec_of(c + 1) + IMG_TB, 16384);
    }

    // ---- (g) E2 -> EA, wR*E2 -> WA;  MMA7: Ob += E2^T (gamma M2)^T;  MMA8: U2 = (wR E2)^T K
    {
      const int c0 = g16;
      float e[16], w[16];
      if (RDNV) {
        tmem_ld16(tm + lane + T_D1 + c0, e);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) e[i] = rres[i];
      }
      lds16(wR + c0, w);
#pragma unroll
      for (int i = 0; i < 16; ++i) w[i] *= e[i];
      st_row16_split(sm + SM_XE, sm + SM_XE_LO, j, c0, e);
      st_row16_split(sm + SM_W, sm + SM_W_LO, j, c0, w);
    }
    alive = run_phase([&] {
      const uint32_t i64 = idesc_bf16(128, 64);
      if (!mbar_wait(barB, phB)) return false;
      phB ^= 1u;
      pendB = false;
      // the image is diag(gamma) M2: its product lands on Ob directly
      mma_split3(tm + T_D1 + 64, sbase + SM_XE, sbase + SM_XE_LO, sbase + SM_SLOTB,
                 sbase + SM_SLOTB + 8192, i64, true);
      if (p.sv_E2) {  // and the E2^T image
        bulk_s2g(p.sv_E2 + ci * 32768, sm + SM_XE, 32768);
        bulk_commit();
      }
      mma_tile_kmn(tm + T_R, sbase + SM_W, 0, sbase + SM_KQ, 16384, 4, idesc_bf16(128, 128), true);
      mma_tile_kmn(tm + T_R, sbase + SM_W_LO, 0, sbase + SM_KQ, 16384, 4, idesc_bf16(128, 128),
                   true);
      return true;
    }, nothing);
    if (!alive) break;
    if (tid == 0 && c + 1 < NC) load_slot(sm + SM_SLOTB, barB, rec_of(c + 1) + IMG_APMQ, 32768);
    if (c + 1 < NC) {  // K, Q are done with
      if (!by_tma(c + 1))
        fetch_kq(c + 1);
      else if (tid == 0)
        tma_kq(c + 1);
    }

    // ---- (h) o = (Ob + diag(gamma) M2 E2) + gamma * Gam QR;  R (= Gam_C R + U2) -> RA
    // o is staged as a [t][j] tile in W's place (free after MMA8; bf16, or fp32
    // over W and its lo part) and stored 16 bytes at a time
    __nv_bfloat16 *ostg = reinterpret_cast<__nv_bfloat16 *>(sm + SM_W);
    float *ostg32 = reinterpret_cast<float *>(sm + SM_W);
    static_assert(SM_W_LO == SM_W + 16384, "fp32 o staging spans W and its lo part");
    {
      const int c0 = g16;
      float ob[16], oa[16], gm[16], gv[16];
      tmem_ld16x2(tm + lane + T_D1 + 64 + c0, ob, tm + lane + T_X + 64 + c0, oa);
      lds16(Gam + c0, gm);
      lds16(gamv + c0, gv);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int t = c0 + i;
        const float gg = plain ? 1.f : gv[i];
        const float ov = stl ? ob[i] : fmaf(gg * gm[i] * p.scale, oa[i], ob[i]);
        if (p.f32out)
          ostg32[t * D + j] = ov;
        else
          ostg[t * D + j] = __float2bfloat16_rn(ov);
      }
    }
    {
      float r0[16], r1[16];
      tmem_ld16x2(tm + lane + T_R + g16, r0, tm + lane + T_R + g16 + 64, r1);
      st_row16(sm + SM_RA, 16384, j, g16, r0);
      st_row16(sm + SM_RA, 16384, j, g16 + 64, r1);
    }
    // the state's lo part below goes over the E2^T tiles: their bulk store to
    // the saved E2 must have read them
    if (p.sv_E2 && tid == 0) bulk_wait_read();
    __syncthreads();  // the o tile, and the E2^T tiles
    {  // the updated state's lo part, for the next chunk's read-outs
      float s0[16], s1[16];
      tmem_ld16x2(tm + lane + T_S + g16, s0, tm + lane + T_S + g16 + 64, s1);
      store_state_lo(g16, s0);
      store_state_lo(g16 + 64, s1);
    }
    if (p.f32out) {
      float *of = (float *)p.o;
      for (int e = tid; e < 64 * 32; e += kTcThreads) {
        const int t = e >> 5, ch = e & 31;
        if (t < n)
          *reinterpret_cast<uint4 *>(of + ((size_t)(tok0 + t0 + t) * H + h) * D + ch * 4) =
              *reinterpret_cast<const uint4 *>(sm + SM_W + t * 512 + ch * 16);
      }
    } else {
      for (int e = tid; e < 64 * 16; e += kTcThreads) {
        const int t = e >> 4, ch = e & 15;
        if (t < n)
          *reinterpret_cast<uint4 *>(o + ((size_t)(tok0 + t0 + t) * H + h) * D + ch * 8) =
              *reinterpret_cast<const uint4 *>(sm + SM_W + t * 256 + ch * 16);
      }
    }
  }

  if (tid == 0 && p.sv_E) bulk_wait_all();
  if (alive) {  // final states
    for (int c0 = g16; c0 < D; c0 += 64) {
      float s[16], r[16];
      tmem_ld16(tm + lane + T_S + c0, s);
      tmem_ld16(tm + lane + T_R + c0, r);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (p.ST) p.ST[st_base + (size_t)(c0 + i) * D + j] = s[i];
        if (p.RT) p.RT[st_base + (size_t)(c0 + i) * D + j] = r[i];
      }
    }
  } else {
    // a bounded wait gave up: record it, then let every operation of this CTA
    // still in flight finish (again with bounded waits) before its shared
    // memory and TMEM are released -- the MMAs this thread issued (one commit
    // covers them all), the slot copies armed and not waited for, the
    // cp.async tile copies and the bulk stores
    if (tid == 0) {
      if (p.err) atomicExch(p.err, RDN_ERR_TIMEOUT);
      mma_commit(barD);
      mbar_wait(barD, 0);
      if (pendA) mbar_wait(barA, phA);
      if (pendB) mbar_wait(barB, phB);
      if (pendE) mbar_wait(barE, phE & 1u);
      bulk_wait_all();
    }
    cp_async_wait_all();
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, 512);
}

}  // namespace

namespace {
// the driver's tensor-map encoder, looked up once through the runtime (no
// link against the driver library)
PFN_cuTensorMapEncodeTiled_v12000 tile_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      f = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }();
  return fn;
}
}  // namespace

bool make_tile_map(void *map128, const void *base, int D, int H, long long rows) {
  static_assert(sizeof(CUtensorMap) == 128, "tensor map size");
  const auto enc = tile_map_encoder();
  if (!enc || !base || rows < 1) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)rows};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2};  // bytes, dims 1, 2
  const cuuint32_t box[3] = {64, 1, 64};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(reinterpret_cast<CUtensorMap *>(map128), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
             const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t launch_fwd_tc(const FwdParams &p, bool rdnv, cudaStream_t s) {
  FwdMaps maps;
  const long long rows = (long long)p.B * p.T;
  maps.ok = make_tile_map(maps.v, p.v, D, p.H, rows) && make_tile_map(maps.k, p.k, D, p.H, rows) &&
            make_tile_map(maps.q, p.q, D, p.H, rows);
  const bool generic = p.mods != 0;
  auto kern = rdnv ? (generic ? fwd_tc_kernel<true, true> : fwd_tc_kernel<true, false>)
                   : (generic ? fwd_tc_kernel<false, true> : fwd_tc_kernel<false, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kTcSmem);
  if (e != cudaSuccess) return e;
  RDN_LAUNCH("fwd_tc_scan", s, kern<<<p.nseq * p.H, kTcThreads, kTcSmem, s>>>(p, maps));
  return cudaGetLastError();
}

}  // namespace rdn
