// bwd_tc.cu -- tensor-core (tcgen05 / TMEM) backward of the chunkwise RDN
// forward, bf16 inputs, d_k = d_v = 128; RLA (TcBwdParams::rla) and two of
// the variant flags are runtime modes of separate kernel instances.
//
// Reverse mode of the chunk algebra of chunk_fwd.cu (the same steps as
// chunk_bwd.cu, whose header lists them), split by what depends on the
// gradients carried between chunks:
//
//  1. bwd_recompute (parallel, one CTA per chunk): from the chunk-start
//     states rebuild E, E2 and the clip mask (the forward's pieces for one
//     chunk).  It does not run when the forward saved them.
//  2. bwd_chain (sequential over chunks, one CTA per (b,h)): the carried
//     gradients.  With dR, dS the gradients w.r.t. a chunk's end states,
//        dE2 = M2^T dOa + diag(wR) K dR        dX2 = T_gamma^T dE2
//        dP  = -mask * dX2                     dKR = -diag(Gam) dX2
//        dR_prev = Gam_C dR + K^T dKR + Q^T diag(Gam gamma) dO
//        dE  = Mq^T dO + Ap^T dP + diag(wS) K dS     dX = T_beta^T dE
//        dKS = diag(Gprev) dP - diag(Gam) dX
//        dS_prev = Gam_C dS + K^T dKS + Q^T diag(Gam) dO
//        dv  = -dP + dX
//     No forward quantity other than the clip mask enters this chain.
//  3. bwd_post (parallel, one CTA per chunk): every product that reduces over
//     the value dimension -- the state terms of dK, dQ, the five C x C
//     gradients, the per-row gate terms -- and then the gradients of the chunk
//     matrices' entries turned into dq, dk, dg, dbeta, dgamma (the work that
//     bwd_finish of chunk_bwd.cu does on the SIMT path).
//
// Orientation: value column j = TMEM lane j, owned by thread j of a group of
// 128 threads (bwd_chain: 4 groups, group g taking the token and key columns
// [16g, 16g + 16) and [64 + 16g, 80 + 16g); bwd_post: 2 groups), for every
// column quantity (X, E, dO, dX2, ...), which is kept as a bf16 hi + lo tile
// [j][t] (K-major for products over t).  Products over j use the same tiles
// as MN-major operands.  The chunk matrices come from chunk_prep's images
// (bf16 hi + lo); products with them are three MMAs (hi*hi + hi*lo + lo*hi).
// States and carried gradients enter their products as bf16 hi + lo as well.
#include "chunk_common.cuh"
#include "tc_common.cuh"

namespace rdn {
namespace {

using namespace tc;

constexpr int D = 128;
constexpr int NT = 128;   // threads per CTA of bwd_recompute
constexpr int NTC = 512;  // threads per CTA of bwd_chain (4 warps per TMEM lane quadrant)

// bwd_post's per-token sums kept in shared memory from where they are formed
// to the gate pass (floats): the read-out part of d gamma, dwS, dwR (C each).
struct A8 {
  static constexpr int V_DGAM_OUT = 0, V_DWS = C, V_DWR = 2 * C;
  static constexpr int FLOATS = 3 * C;
};

struct TcBwdParams {
  FwdParams f;          // inputs; f.ws = prep records (shared-memory images)
  const void *dO;
  const float *dST, *dRT;
  const float *Sc, *Rc;  // chunk-start states [B,H,NC,D,D]
  void *dv;
  float *dS0, *dR0;
  uint8_t *Ebuf, *E2buf; // [B*H*NC][32 KB]: images of E^T, E2^T (rows j, columns t; hi | lo)
  float *dX2buf, *dXbuf; // [B*H*NC][64][128]
  uint8_t *gimg;         // [B*H*NC][128 KB]: gradients w.r.t. each chunk's end states as
                         // bf16 images (rows j): dS hi | dR hi | dS lo | dR lo, 32 KB each
  unsigned long long *mask;  // [B*H*NC][128]: bit t = clip inactive (|x| <= c)
  void *dq, *dk;             // outputs of bwd_post
  float *dg, *dbeta, *dgamma;
  // RLA: the records carry T_beta = T_gamma = I and the deltas are absent
  // (E = V, E2 = r), so the terms through -Gam K S0, -Gam K R0 and the
  // gradients of A_beta, A_gamma drop out; the chunk-start state enters the
  // recomputed prediction with a lo part (RLA's S is not contracted)
  bool rla;
  bool f32g;    // dq, dk, dv stored in fp32 (RDN_FLAG_F32_OUT), else bf16
  bool f32qk;   // dq, dk stored in fp32 whatever f32g (for a step that follows)
  // tensor maps (CUtensorMap, 64-byte aligned) over k, q, dO as [tokens][H][D]
  // with a 64-token x 64-column box (make_tile_map); tma: they are valid
  alignas(64) unsigned char map_k[128];
  alignas(64) unsigned char map_q[128];
  alignas(64) unsigned char map_do[128];
  bool tma;
};

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Row r, columns c0..c0+15 of a K-major SW128 tile (64-col blocks blk apart).
__device__ __forceinline__ void put16(uint8_t *tile, uint32_t blk, int r, int c0,
                                      const float (&v)[16]) {
  uint8_t *b = tile + (c0 >> 6) * blk;
  const int cc = c0 & 63;
  uint4 x, y;
  x.x = pack2(v[0], v[1]); x.y = pack2(v[2], v[3]); x.z = pack2(v[4], v[5]); x.w = pack2(v[6], v[7]);
  y.x = pack2(v[8], v[9]); y.y = pack2(v[10], v[11]); y.z = pack2(v[12], v[13]); y.w = pack2(v[14], v[15]);
  *reinterpret_cast<uint4 *>(b + sw128(r, cc)) = x;
  *reinterpret_cast<uint4 *>(b + sw128(r, cc + 8)) = y;
}
// hi / lo split (split_pack_bf16) of 16 values into two single-block tiles
__device__ __forceinline__ void put16s(uint8_t *hi, uint8_t *lo, int r, int c0,
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
// the same for 8 values (one 16-byte chunk of each tile)
__device__ __forceinline__ void put8s(uint8_t *hi, uint8_t *lo, int r, int c0,
                                      const float (&v)[8]) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) split_pack_bf16(v[2 * i], v[2 * i + 1], h[i], l[i]);
  *reinterpret_cast<uint4 *>(hi + sw128(r, c0)) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4 *>(lo + sw128(r, c0)) = make_uint4(l[0], l[1], l[2], l[3]);
}
// K-major A (single block, K = 64) times MN-major B, split both: 3 products
__device__ __forceinline__ void mma_s3_kmn(uint32_t d, uint32_t a_hi, uint32_t a_lo,
                                           uint32_t b_hi, uint32_t b_lo, uint32_t b_lbo,
                                           uint32_t idesc, bool acc_first) {
  mma_tile_kmn(d, a_hi, 0, b_hi, b_lbo, 4, idesc, acc_first);
  mma_tile_kmn(d, a_hi, 0, b_lo, b_lbo, 4, idesc, true);
  mma_tile_kmn(d, a_lo, 0, b_hi, b_lbo, 4, idesc, true);
}
// K-major A and B (single block, K = 64), split both
__device__ __forceinline__ void mma_s3_kk(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint32_t b_hi,
                                          uint32_t b_lo, uint32_t idesc, bool acc_first) {
  mma_tile(d, a_hi, 0, b_hi, 0, 4, idesc, acc_first);
  mma_tile(d, a_hi, 0, b_lo, 0, 4, idesc, true);
  mma_tile(d, a_lo, 0, b_hi, 0, 4, idesc, true);
}

// Common per-CTA machinery: mbarriers (MMA, copies A, B, C, and D for the
// drain), TMEM, phases.  Thread 0 counts the copy phases it arms on A, B, C
// and the ones it has seen complete, so that a CTA whose bounded wait gave up
// can wait (again with a limit) for every copy and MMA still in flight before
// it releases its shared memory and TMEM (ctl_drain).
struct Ctl {
  uint64_t *bar, *barA, *barB, *barC, *barD;
  volatile int *flag;
  uint32_t phase, phA, phB;
  uint32_t armA, armB, armC, seenA, seenB, seenC;  // (thread 0) copy phases on A, B, C
  long long limit;             // the MMA waits' limit in cycles
  bool skip;                   // (thread 0) the next phase skips its completion signal (tests)
};

__device__ __forceinline__ void ctl_init(Ctl &k, uint8_t *base, int tid) {
  k.bar = reinterpret_cast<uint64_t *>(base);
  k.barA = k.bar + 1;
  k.barB = k.bar + 2;
  k.barC = k.bar + 3;
  k.flag = reinterpret_cast<volatile int *>(base + 32);
  k.barD = reinterpret_cast<uint64_t *>(base + 40);
  k.phase = k.phA = k.phB = 0;
  k.armA = k.armB = k.armC = k.seenA = k.seenB = k.seenC = 0;
  k.limit = 2000000000ll;
  k.skip = false;
  if (tid == 0) {
    mbar_init(k.bar, 1);
    mbar_init(k.barA, 1);
    mbar_init(k.barB, 1);
    mbar_init(k.barC, 1);
    mbar_init(k.barD, 1);
    fence_mbar_init();
    *k.flag = 0;
  }
}

// the barrier and counters of copy barrier W (0: A, 1: B, 2: C)
template <int W>
__device__ __forceinline__ uint64_t *ctl_bar(Ctl &k) {
  return W == 0 ? k.barA : (W == 1 ? k.barB : k.barC);
}
template <int W>
__device__ __forceinline__ uint32_t &ctl_armed(Ctl &k) {
  return W == 0 ? k.armA : (W == 1 ? k.armB : k.armC);
}
template <int W>
__device__ __forceinline__ uint32_t &ctl_seen(Ctl &k) {
  return W == 0 ? k.seenA : (W == 1 ? k.seenB : k.seenC);
}
// (thread 0) arm a copy phase of barrier W for `bytes`
template <int W>
__device__ __forceinline__ void ctl_arm(Ctl &k, uint32_t bytes) {
  mbar_expect_tx(ctl_bar<W>(k), bytes);
  ++ctl_armed<W>(k);
}
// wait for a copy phase of barrier W (thread 0 counts it)
template <int W>
__device__ __forceinline__ bool ctl_wait(Ctl &k, uint32_t parity, int tid) {
  const bool ok = mbar_wait(ctl_bar<W>(k), parity);
  if (ok && tid == 0) ++ctl_seen<W>(k);
  return ok;
}
template <int W>
__device__ __forceinline__ void ctl_drain_copies(Ctl &k) {
  for (; ctl_seen<W>(k) < ctl_armed<W>(k); ++ctl_seen<W>(k))
    mbar_wait(ctl_bar<W>(k), ctl_seen<W>(k) & 1u);
}
// (thread 0, after a wait gave up) every MMA this thread issued (one commit
// covers them) and every armed copy phase, with bounded waits
__device__ __forceinline__ void ctl_drain(Ctl &k) {
  mma_commit(k.barD);
  mbar_wait(k.barD, 0);
  ctl_drain_copies<0>(k);
  ctl_drain_copies<1>(k);
  ctl_drain_copies<2>(k);
}

template <int W>
__device__ __forceinline__ void load_slot(Ctl &k, uint8_t *dst, const void *src, uint32_t bytes) {
  ctl_arm<W>(k, bytes);
  bulk_g2s(dst, src, bytes, ctl_bar<W>(k));
}

// One MMA phase: publish shared-memory writes, issue (thread 0), wait.
template <typename F>
__device__ __forceinline__ bool phase_run(Ctl &k, int tid, F issue) {
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  if (tid == 0) {
    fence_after_sync();
    if (!issue()) *k.flag = 1;
    if (!k.skip) mma_commit(k.bar);
    k.skip = false;
  }
  const bool ok = mbar_wait(k.bar, k.phase, k.limit);
  k.phase ^= 1u;
  if (!ok) *k.flag = 1;
  __syncthreads();
  fence_after_sync();
  return *k.flag == 0;
}

// The same, running `during` (work the MMAs do not touch) between the issue
// and the wait.
template <typename F, typename G>
__device__ __forceinline__ bool phase_run_with(Ctl &k, int tid, F issue, G during) {
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  if (tid == 0) {
    fence_after_sync();
    if (!issue()) *k.flag = 1;
    if (!k.skip) mma_commit(k.bar);
    k.skip = false;
  }
  during();
  const bool ok = mbar_wait(k.bar, k.phase, k.limit);
  k.phase ^= 1u;
  if (!ok) *k.flag = 1;
  __syncthreads();
  fence_after_sync();
  return *k.flag == 0;
}

// The same phase in two halves, for work that overlaps the MMAs: publish and
// issue ...
template <typename F>
__device__ __forceinline__ void phase_issue(Ctl &k, int tid, F issue) {
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  if (tid == 0) {
    fence_after_sync();
    if (!issue()) *k.flag = 1;
    if (!k.skip) mma_commit(k.bar);
    k.skip = false;
  }
}
// ... then wait for them (every thread).
__device__ __forceinline__ bool phase_wait(Ctl &k) {
  const bool ok = mbar_wait(k.bar, k.phase, k.limit);
  k.phase ^= 1u;
  if (!ok) *k.flag = 1;
  __syncthreads();
  fence_after_sync();
  return *k.flag == 0;
}

// thread 0: wait for a slot's bulk copy
template <int W>
__device__ __forceinline__ bool slot_wait(Ctl &k, uint32_t &ph) {
  const bool ok = ctl_wait<W>(k, ph, 0);
  ph ^= 1u;
  return ok;
}

__device__ __forceinline__ const uint8_t *rec_bytes(const FwdParams &p, size_t chunk) {
  return reinterpret_cast<const uint8_t *>(p.ws + chunk * kRecFloats);
}

// ======================================================================== 1
// bwd_recompute: the forward pieces of one chunk from its start states.
namespace rc {
constexpr uint32_t SA = 0, RA = 32768, B1 = 65536, SLOTA = 98304, SLOTB = 114688;
constexpr uint32_t XE = 147456, XE_LO = 163840, VEC = 180224;
constexpr uint32_t CTL = VEC + 7 * 64 * 4;
constexpr uint32_t SLOT = CTL + 48;
constexpr uint32_t SA_LO = 183296;  // S0 - bf16(S0), two 16 KB blocks
static_assert(SA_LO >= SLOT + 16 && SA_LO % 1024 == 0, "layout");
constexpr size_t SMEM = SA_LO + 32768;
constexpr uint32_t T_D1 = 0, T_D3 = 128, T_X = 256;
}  // namespace rc

__global__ void __launch_bounds__(NT, 1) bwd_recompute_kernel(TcBwdParams P) {
  using namespace rc;
  extern __shared__ __align__(1024) uint8_t sm[];
  const uint32_t sb = smem_u32(sm);
  const FwdParams &p = P.f;
  if (sb & 1023u) {
    if (threadIdx.x == 0 && p.err) atomicExch(p.err, RDN_ERR_CUDA);
    return;
  }
  float *vec = reinterpret_cast<float *>(sm + VEC);
  float *Gam = vec, *Gprev = vec + 64, *gamv = vec + 320;
  uint32_t *slot = reinterpret_cast<uint32_t *>(sm + SLOT);
  const int tid = threadIdx.x, warp = tid >> 5, j = tid;
  const size_t chunk = blockIdx.x;
  if ((long long)chunk >= total_records(p)) return;  // (packed sequences: the grid is a bound)
  const int H = p.H;
  int sq, h, c;
  rec_decode(p, (long long)chunk, sq, h, c);
  const SeqSpan sp = seq_span(p, sq, h);
  const long long tok0 = sp.tok0;
  const int T = sp.len;
  const int t0 = c * 64, n = min(64, T - t0);
  const __nv_bfloat16 *k = (const __nv_bfloat16 *)p.k, *v = (const __nv_bfloat16 *)p.v;
  const uint8_t *rec = rec_bytes(p, chunk);
  const float clip = p.clip;

  Ctl K;
  ctl_init(K, sm + CTL, tid);
  if (warp == 0) tmem_alloc(slot, 512);
  if (tid == 0) {
    load_slot<0>(K, sm + SLOTA, rec + IMG_TB, 16384);
    load_slot<1>(K, sm + SLOTB, rec + IMG_APMQ, 32768);
  }
  if (tid < 64) {
    Gam[tid] = reinterpret_cast<const float *>(rec)[OFF_VEC + V_GAM + tid];
    Gprev[tid] = reinterpret_cast<const float *>(rec)[OFF_VEC + V_GPREV + tid];
    gamv[tid] = tid < n ? p.gamma[(size_t)(tok0 + t0 + tid) * H + h] : 0.f;
  }
  // chunk-start states -> bf16 A operands (row j = column j of [i][j])
  {
    const float *S0 = P.Sc + chunk * D * D, *R0 = P.Rc + chunk * D * D;
    for (int c0 = 0; c0 < D; c0 += 16) {
      float s[16], r[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        s[i] = S0[(size_t)(c0 + i) * D + j];
        r[i] = R0[(size_t)(c0 + i) * D + j];
      }
      put16(sm + SA, 16384, j, c0, s);
      put16(sm + RA, 16384, j, c0, r);
      {  // S0 - bf16(S0), as the forward scan's read-outs use it
#pragma unroll
        for (int i = 0; i < 16; ++i) s[i] -= __bfloat162float(__float2bfloat16_rn(s[i]));
        put16(sm + SA_LO, 16384, j, c0, s);
      }
    }
  }
  __syncthreads();
  // B1 = K (64 rows, exact bf16); the forward scan's arithmetic: unscaled
  // read-outs, gates applied in fp32
  for (int e = tid; e < 64 * 16; e += NT) {
    const int t = e >> 4, ch = e & 15;
    const bool vld = t < n;
    const size_t off = ((size_t)(tok0 + t0 + (vld ? t : 0)) * H + h) * D + ch * 8;
    cp_async16(sm + B1 + (ch >> 3) * 16384 + sw128(t, (ch & 7) * 8), k + off, vld);
  }
  cp_async_wait_all();
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tm = *slot;
  const uint32_t lane = (uint32_t)(warp * 32) << 16;
  auto vval = [&](int t) -> float {
    return t < n ? __bfloat162float(v[((size_t)(tok0 + t0 + t) * H + h) * D + j]) : 0.f;
  };

  bool ok = phase_run(K, tid, [&] {  // KS, KR
    mma_tile(tm + T_D1, sb + SA, 16384, sb + B1, 16384, 8, idesc_bf16(128, 64), false);
    mma_tile(tm + T_D1, sb + SA_LO, 16384, sb + B1, 16384, 8, idesc_bf16(128, 64), true);
    mma_tile(tm + T_D3, sb + RA, 16384, sb + B1, 16384, 8, idesc_bf16(128, 64), false);
    return true;
  });
  float r[64];
  if (ok) {  // X = V - Gam KS -> E = T_beta X; D1 <- Gprev KS (P accumulates onto it)
#pragma unroll
    for (int c0 = 0; c0 < 64; c0 += 16) {
      float ks[16], x[16];
      tmem_ld16(tm + lane + T_D1 + c0, ks);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        x[i] = vval(c0 + i) - (P.rla ? 0.f : Gam[c0 + i] * ks[i]);
        ks[i] *= (p.mods & RDN_FLAG_DECAYED_RESIDUAL) ? Gam[c0 + i] : Gprev[c0 + i];
      }
      tmem_st16(tm + lane + T_D1 + c0, ks);
      put16s(sm + XE, sm + XE_LO, j, c0, x);
    }
    ok = phase_run(K, tid, [&] {
      if (!slot_wait<0>(K, K.phA)) return false;
      mma_s3_kk(tm + T_X, sb + XE, sb + XE_LO, sb + SLOTA, sb + SLOTA + 8192, idesc_bf16(128, 64),
                 false);
      return true;
    });
  }
  if (ok) {
    if (tid == 0) load_slot<0>(K, sm + SLOTA, rec + IMG_TG, 16384);
#pragma unroll
    for (int c0 = 0; c0 < 64; c0 += 16) {
      float e[16];
      tmem_ld16(tm + lane + T_X + c0, e);
      put16s(sm + XE, sm + XE_LO, j, c0, e);
    }
    ok = phase_run(K, tid, [&] {  // D1 += E Ap^T -> P (the Ap rows of the [Ap ; Mq] image)
      if (!slot_wait<1>(K, K.phB)) return false;
      mma_s3_kk(tm + T_D1, sb + XE, sb + XE_LO, sb + SLOTB, sb + SLOTB + 16384,
                 idesc_bf16(128, 64), true);
      static_assert(XE_LO == XE + 16384, "contiguous");
      bulk_s2g(P.Ebuf + chunk * 32768, sm + XE, 32768);  // the E^T image, for bwd_post
      bulk_commit();
      bulk_wait_read();
      return true;
    });
  }
  if (ok) {
    // the clip mask, or with the tanh residual its derivative ([j][t], grad_q16)
    const bool tnh = p.mods & RDN_FLAG_TANH_RESIDUAL;
    uint16_t *drow = reinterpret_cast<uint16_t *>(P.mask) + (chunk * D + j) * 64;
    unsigned long long m = 0ull;
#pragma unroll
    for (int c0 = 0; c0 < 64; c0 += 16) {
      float pp[16], kr[16];
      tmem_ld16(tm + lane + T_D1 + c0, pp);
      tmem_ld16(tm + lane + T_D3 + c0, kr);
      float x2[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int t = c0 + i;
        const float x = vval(t) - pp[i];
        if (fabsf(x) <= clip) m |= 1ull << t;
        r[t] = resid_map(x, clip, tnh);
        if (tnh) drow[t] = (uint16_t)grad_q16(resid_grad(x, clip, true));
        x2[i] = r[t] - ((P.rla || (p.mods & RDN_FLAG_STATELESS_AUX)) ? 0.f : Gam[t] * kr[i]);
      }
      put16s(sm + XE, sm + XE_LO, j, c0, x2);
    }
    if (!tnh) P.mask[chunk * D + j] = m;
    ok = phase_run(K, tid, [&] {  // E2 = T_gamma X2
      if (!slot_wait<0>(K, K.phA)) return false;
      mma_s3_kk(tm + T_X, sb + XE, sb + XE_LO, sb + SLOTA, sb + SLOTA + 8192, idesc_bf16(128, 64),
                 false);
      return true;
    });
  }
  if (ok) {  // the E2^T image, for bwd_post
#pragma unroll
    for (int c0 = 0; c0 < 64; c0 += 16) {
      float e[16];
      tmem_ld16(tm + lane + T_X + c0, e);
      put16s(sm + XE, sm + XE_LO, j, c0, e);
    }
    fence_async_smem();
    __syncthreads();
    if (tid == 0) {
      bulk_s2g(P.E2buf + chunk * 32768, sm + XE, 32768);
      bulk_commit();
      bulk_wait_all();
    }
  } else if (tid == 0) {
    if (p.err) atomicExch(p.err, RDN_ERR_TIMEOUT);
    ctl_drain(K);  // no copy or MMA of this CTA outlives it
  }
  if (tid == 0) bulk_wait_all();
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, 512);
}

// ======================================================================== 2
// bwd_chain: the gradients carried between chunks, chunks in reverse.
namespace ch {
// K, Q | carried gradients dS, dR as bf16 hi + lo A operands (phase A) | slots
// | dO.  After phase A the 128 KB of gradient tiles serve as scratch for the
// split column tiles; the gradient tiles are rewritten at the chunk end.
constexpr uint32_t KQ = 0;
constexpr uint32_t DSH = 32768, DRH = 65536, DSL = 98304, DRL = 131072;
constexpr uint32_t SLOTA = 163840;   // diag(gamma) M2 -> T_gamma -> T_beta (16 KB)
constexpr uint32_t SLOTB = 180224;   // Mq -> Ap (hi 8 KB | lo 8 KB)
constexpr uint32_t DOT = 196608;     // dO, exact bf16, rows t (two 8 KB column blocks)
// scratch column tiles (hi, lo) inside the gradient-tile region
constexpr uint32_t S0H = 32768, S0L = 49152, S1H = 65536, S1L = 81920;
constexpr uint32_t S2H = 98304, S2L = 114688, S3H = 131072, S3L = 147456;
constexpr uint32_t VEC = 212992;                 // Gam Gprev wS wR gamma (5 x 64)
constexpr uint32_t CTL = VEC + 5 * 64 * 4;
constexpr uint32_t SLOT = CTL + 48;
constexpr size_t SMEM = SLOT + 16;
static_assert(SMEM <= 232448, "shared memory");
constexpr uint32_t T_DS = 0, T_DR = 128, T_R1 = 256, T_R2 = 320, T_R3 = 384, T_R4 = 448;
}  // namespace ch

// kGeneric: the RLA mode and the variant flags (TcBwdParams::rla, FwdParams::mods)
// are read; the RDN method's instance has them folded away
template <bool kGeneric>
__global__ void __launch_bounds__(NTC, 1) bwd_chain_kernel(const __grid_constant__ TcBwdParams P) {
  using namespace ch;
  extern __shared__ __align__(1024) uint8_t sm[];
  const uint32_t sb = smem_u32(sm);
  const FwdParams &p = P.f;
  const bool rla = kGeneric && P.rla;
  const unsigned mods = kGeneric ? p.mods : 0u;
  if (sb & 1023u) {
    if (threadIdx.x == 0 && p.err) atomicExch(p.err, RDN_ERR_CUDA);
    return;
  }
  float *vec = reinterpret_cast<float *>(sm + VEC);
  float *Gam = vec, *Gprev = vec + 64, *wS = vec + 128, *wR = vec + 192, *gamv = vec + 256;
  uint32_t *slot = reinterpret_cast<uint32_t *>(sm + SLOT);
  const int tid = threadIdx.x, warp = tid >> 5, j = tid & 127;
  const int g16 = (warp >> 2) * 16;  // this thread's token (and key) columns start
  const int bh = blockIdx.x;
  const int H = p.H, h = bh % H;
  const SeqSpan sp = seq_span(p, bh / H, h);  // this (sequence, head)'s tokens and records
  const long long tok0 = sp.tok0;
  const int NC = sp.nc, T = sp.len;
  const __nv_bfloat16 *q = (const __nv_bfloat16 *)p.q, *k = (const __nv_bfloat16 *)p.k,
                      *dOp = (const __nv_bfloat16 *)P.dO;
  __nv_bfloat16 *dv = (__nv_bfloat16 *)P.dv;
  const size_t st_base = (size_t)bh * D * D;

  Ctl K;
  ctl_init(K, sm + CTL, tid);
  if (p.inject == 2) {  // (a test: the first phase's signal is skipped, the wait gives up)
    K.limit = 10000000ll;
    K.skip = true;
  }
  if (warp == 0) tmem_alloc(slot, 512);
  // slot loads: A holds diag(gamma) M2, then T_gamma, then T_beta; B holds
  // Mq (hi | lo), then Ap (hi | lo) -- each 8 KB half copied from the
  // [Ap ; Mq] image
  auto load_mq = [&](size_t ck) {
    const uint8_t *r = rec_bytes(p, ck);
    ctl_arm<1>(K, 16384);
    bulk_g2s(sm + SLOTB, r + IMG_APMQ + 8192, 8192, K.barB);
    bulk_g2s(sm + SLOTB + 8192, r + IMG_APMQ + 16384 + 8192, 8192, K.barB);
  };
  auto load_ap = [&](size_t ck) {
    const uint8_t *r = rec_bytes(p, ck);
    ctl_arm<1>(K, 16384);
    bulk_g2s(sm + SLOTB, r + IMG_APMQ, 8192, K.barB);
    bulk_g2s(sm + SLOTB + 8192, r + IMG_APMQ + 16384, 8192, K.barB);
  };
  if (tid == 0 && NC > 0) {  // (a packed sequence may be empty)
    const size_t last = (size_t)(sp.rbase + NC - 1);
    load_slot<0>(K, sm + SLOTA, rec_bytes(p, last) + IMG_M2, 16384);
    load_mq(last);
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tm = *slot;
  const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
  // a carried gradient's bf16 hi + lo tiles (rows j), 16 of its key rows
  auto put_grad16 = [&](uint32_t hi, uint32_t lo, int c0, const float (&g)[16]) {
    put16s(sm + hi + (c0 >> 6) * 16384, sm + lo + (c0 >> 6) * 16384, j, c0, g);
  };
  // both carried gradients' tiles from their fp32 TMEM copies
  auto write_grad_tiles = [&]() {
#pragma unroll 1
    for (int c0 = g16; c0 < D; c0 += 64) {
      float s[16], r[16];
      tmem_ld16x2(tm + lane + T_DS + c0, s, tm + lane + T_DR + c0, r);
      put_grad16(DSH, DSL, c0, s);
      put_grad16(DRH, DRL, c0, r);
    }
    fence_async_smem();  // the tiles are read by the MMAs and by a bulk copy
  };
  // a carried gradient's TMEM copy times the chunk's total decay, in place
  // (this chunk's products accumulate onto it); this thread's columns
  auto scale_grad = [&](uint32_t col, float f) {
    float x[16], y[16];
    tmem_ld16x2(tm + lane + col + g16, x, tm + lane + col + g16 + 64, y);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      x[i] *= f;
      y[i] *= f;
    }
    tmem_st16(tm + lane + col + g16, x);
    tmem_st16(tm + lane + col + g16 + 64, y);
  };
  for (int c0 = g16; c0 < D; c0 += 64) {  // upstream gradients of the final states
    float s[16], r[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      s[i] = P.dST ? P.dST[st_base + (size_t)(c0 + i) * D + j] : 0.f;
      r[i] = P.dRT ? P.dRT[st_base + (size_t)(c0 + i) * D + j] : 0.f;
    }
    tmem_st16(tm + lane + T_DS + c0, s);
    tmem_st16(tm + lane + T_DR + c0, r);
  }
  write_grad_tiles();

  // a chunk's K, Q, dO tiles (rows t, exact bf16, zero past the end), asynchronous
  auto fetch_kq = [&](int c) {
    const int t0 = c * 64, n = min(64, T - t0);
    for (int e = tid; e < 64 * 16; e += NTC) {
      const int t = e >> 4, chn = e & 15;
      const bool vld = t < n;
      const size_t off = ((size_t)(tok0 + t0 + (vld ? t : 0)) * H + h) * D + chn * 8;
      const int blk = chn >> 3, cc = (chn & 7) * 8;
      cp_async16(sm + KQ + blk * 16384 + sw128(t, cc), k + off, vld);
      cp_async16(sm + KQ + blk * 16384 + sw128(64 + t, cc), q + off, vld);
    }
  };
  auto fetch_do = [&](int c) {
    const int t0 = c * 64, n = min(64, T - t0);
    for (int e = tid; e < 64 * 16; e += NTC) {
      const int t = e >> 4, chn = e & 15;
      const bool vld = t < n;
      const size_t off = ((size_t)(tok0 + t0 + (vld ? t : 0)) * H + h) * D + chn * 8;
      cp_async16(sm + DOT + (chn >> 3) * 8192 + sw128(t, (chn & 7) * 8), dOp + off, vld);
    }
  };
  // a chunk's gate vectors (threads 0..63, one token each) and this thread's
  // 16 bits of the clip-mask word, into registers
  struct Pre {
    float gam_, gprev, ws_, wr_, g_, gamc;
    unsigned m;
    uint4 d0, d1;  // the tanh residual's derivative at this thread's 16 tokens (grad_q16)
  };
  const bool tnh = kGeneric && (mods & RDN_FLAG_TANH_RESIDUAL);
  // the stateless correction: the chunk-end R is not carried into the next
  // chunk nor read out there, so the gradient carried back to it is zero
  // (dR_prev = 0; a chunk's own dR is the upstream dRT for the last chunk)
  const bool stl = kGeneric && (mods & RDN_FLAG_STATELESS_AUX);
  auto fetch_pre = [&](int c) {
    const size_t ck = (size_t)(sp.rbase + c);
    const int t0 = c * 64, n = min(64, T - t0);
    const float *rf = p.ws + ck * kRecFloats;
    Pre x;
    x.gam_ = x.gprev = x.ws_ = x.wr_ = x.g_ = 0.f;
    if (tid < 64) {
      const int t = tid;
      x.gam_ = rf[OFF_VEC + V_GAM + t];
      x.gprev = rf[OFF_VEC + V_GPREV + t];
      x.ws_ = rf[OFF_VEC + V_WS + t];
      x.wr_ = rf[OFF_VEC + V_WR + t];
      x.g_ = t < n ? p.gamma[(size_t)(tok0 + t0 + t) * H + h] : 0.f;
    }
    x.gamc = rf[OFF_VEC + V_GAMC];
    // bits [g16, g16 + 16) of the column's 64-bit word (little-endian)
    if (!tnh) {
      x.m = reinterpret_cast<const uint16_t *>(P.mask + ck * D + j)[g16 >> 4];
    } else {
      const uint4 *dp_ = reinterpret_cast<const uint4 *>(
          reinterpret_cast<const uint16_t *>(P.mask) + (ck * D + j) * 64 + g16);
      x.d0 = dp_[0];
      x.d1 = dp_[1];
    }
    return x;
  };
  Pre pre{};
  if (NC > 0) {
    fetch_kq(NC - 1);
    fetch_do(NC - 1);
    pre = fetch_pre(NC - 1);
  }
  // Chunks before the last are whole 64-token chunks: with tensor maps, thread 0
  // brings their dO (after phase D) and K, Q (after phase E) tiles by tiled bulk
  // copies, all on one phase of barrier C; the last chunk, which may be ragged,
  // is fetched above by cp.async with zero fill.
  const bool tma = P.tma;
  uint32_t tma_ph = 0;    // phases of barrier C waited for
  uint32_t tma_arms = 0;  // (thread 0) phases armed, and of those seen complete
  uint32_t tma_seen = 0;
  auto tma_do = [&](int cc) {  // (thread 0) arms barrier C for the whole chunk
    const int row = (int)(tok0 + (long long)cc * 64);
    ++tma_arms;
    mbar_expect_tx(K.barC, 49152);
    for (int kb = 0; kb < 2; ++kb) tma_load_3d(sm + DOT + kb * 8192, P.map_do, 64 * kb, h, row, K.barC);
  };
  auto tma_kq = [&](int cc) {
    const int row = (int)(tok0 + (long long)cc * 64);
    for (int kb = 0; kb < 2; ++kb) {
      tma_load_3d(sm + KQ + kb * 16384, P.map_k, 64 * kb, h, row, K.barC);
      tma_load_3d(sm + KQ + kb * 16384 + 8192, P.map_q, 64 * kb, h, row, K.barC);
    }
  };

  bool ok = true;
  for (int c = NC - 1; c >= 0 && ok; --c) {
    const size_t chunk = (size_t)(sp.rbase + c);
    const int t0 = c * 64, n = min(64, T - t0);
    __syncthreads();
    if (tid == 0) {  // gradients w.r.t. this chunk's end states, for bwd_post: the tile
      // images, as two groups: the hi tiles (rewritten after phase A), then the
      // lo tiles (rewritten after phase B)
      static_assert(DRH == DSH + 32768 && DSL == DRH + 32768 && DRL == DSL + 32768, "contiguous");
      bulk_s2g(P.gimg + chunk * 131072, sm + DSH, 65536);
      bulk_commit();
      bulk_s2g(P.gimg + chunk * 131072 + 65536, sm + DSL, 65536);
      bulk_commit();
    }
    if (tid < 64) {
      Gam[tid] = pre.gam_;
      Gprev[tid] = pre.gprev;
      wS[tid] = pre.ws_;
      wR[tid] = pre.wr_;
      gamv[tid] = pre.g_;
    }
    const float GamC = pre.gamc;
    const unsigned m = pre.m;  // bit i: clip inactive at t = g16 + i
    const uint4 dd0 = pre.d0, dd1 = pre.d1;  // (tanh residual)
    // this chunk's tiles: by cp.async (waited for here) only for the first, ragged
    // chunk or without tensor maps -- a cp.async wait with none in flight still
    // cost about 3.6k cycles a chunk (clock64 marks)
    if (!tma || c == NC - 1) cp_async_wait_all();
    if (tma && c < NC - 1) {  // (by tiled bulk copies)
      if (mbar_wait(K.barC, tma_ph & 1u))
        tma_seen = tma_ph + 1;
      else
        *K.flag = 1;
      ++tma_ph;
    }
    __syncthreads();
    if (*K.flag) {
      ok = false;
      break;
    }
    auto dO = [&](int t) {  // dO[t, j] from the tile
      return __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(
          sm + DOT + (j >> 6) * 8192 + sw128(t, j & 63)));
    };
    // ---- phase A: K dR, K dS (gradients hi + lo), M2^T (gamma dO), Mq^T dO; meanwhile
    // dR, dS (TMEM) times Gam_C, onto which the products of phases B .. E accumulate
    // (the MMAs read their shared-memory tiles)
    ok = phase_run_with(K, tid, [&] {
      if (!slot_wait<0>(K, K.phA)) return false;
      if (!slot_wait<1>(K, K.phB)) return false;
      const uint32_t i64 = idesc_bf16(128, 64);
      mma_tile(tm + T_R1, sb + DRH, 16384, sb + KQ, 16384, 8, i64, false);
      mma_tile(tm + T_R1, sb + DRL, 16384, sb + KQ, 16384, 8, i64, true);
      mma_tile(tm + T_R2, sb + DSH, 16384, sb + KQ, 16384, 8, i64, false);
      mma_tile(tm + T_R2, sb + DSL, 16384, sb + KQ, 16384, 8, i64, true);
      // dO enters as the MN-major A operand (rows t, value-column atoms 8 KB apart)
      mma_tile_mnmn(tm + T_R3, sb + DOT, 8192, sb + SLOTA, 16384, 4, i64, false);
      mma_tile_mnmn(tm + T_R3, sb + DOT, 8192, sb + SLOTA + 8192, 16384, 4, i64, true);
      mma_tile_mnmn(tm + T_R4, sb + DOT, 8192, sb + SLOTB, 16384, 4, i64, false);
      mma_tile_mnmn(tm + T_R4, sb + DOT, 8192, sb + SLOTB + 8192, 16384, 4, i64, true);
      bulk_wait_read_all_but_last();  // the hi tiles become scratch after this phase
      return true;
    }, [&] {
      scale_grad(T_DR, stl ? 0.f : GamC);
      scale_grad(T_DS, GamC);
    });
    if (!ok) break;
    if (tid == 0) {
      load_slot<0>(K, sm + SLOTA, rec_bytes(p, chunk) + IMG_TG, 16384);
      load_ap(chunk);
    }
    // dE2 = M2^T dOa + wR K dR ; dE (partial) = Mq^T dO + wS K dS ; dQR = Gam gamma dO
    {
      const int c0 = g16;
      float x[16], y[16], w[16];
      tmem_ld16x2(tm + lane + T_R1 + c0, x, tm + lane + T_R3 + c0, y);
      lds16(wR + c0, w);
#pragma unroll
      for (int i = 0; i < 16; ++i) y[i] += w[i] * x[i];
      put16s(sm + S0H, sm + S0L, j, c0, y);
      tmem_ld16x2(tm + lane + T_R2 + c0, x, tm + lane + T_R4 + c0, y);
      lds16(wS + c0, w);
#pragma unroll
      for (int i = 0; i < 16; ++i) y[i] += w[i] * x[i];
      tmem_st16(tm + lane + T_R4 + c0, y);
      lds16(Gam + c0, x);
      lds16(gamv + c0, w);
      const bool plain = mods & RDN_FLAG_PLAIN_COMBINE;  // (no gamma_t in the output)
#pragma unroll
      for (int i = 0; i < 16; ++i)  // dQR (Q unscaled)
        x[i] = stl ? 0.f : p.scale * x[i] * (plain ? 1.f : w[i]) * dO(c0 + i);
      put16s(sm + S1H, sm + S1L, j, c0, x);
    }
    // ---- phase B: dX2 = T_gamma^T dE2 ; U_R = Q^T dQR
    ok = phase_run(K, tid, [&] {
      if (!slot_wait<0>(K, K.phA)) return false;
      mma_s3_kmn(tm + T_R3, sb + S0H, sb + S0L, sb + SLOTA, sb + SLOTA + 8192, 16384,
                 idesc_bf16(128, 64), false);
      const uint32_t i128 = idesc_bf16(128, 128);
      mma_tile_kmn(tm + T_DR, sb + S1H, 0, sb + KQ + 8192, 16384, 4, i128, true);
      mma_tile_kmn(tm + T_DR, sb + S1L, 0, sb + KQ + 8192, 16384, 4, i128, true);
      bulk_wait_read();  // and the lo tiles after this one
      return true;
    });
    if (!ok) break;
    if (tid == 0) load_slot<0>(K, sm + SLOTA, rec_bytes(p, chunk) + IMG_TB, 16384);
    float dP[16];  // t in [g16, g16 + 16)
    {  // dX2 -> dP = -mask dX2, dKR = -Gam dX2; dX2 itself (fp32 [t][j]) for bwd_post,
       // staged in the free scratch tiles and bulk-copied
      float *stg = reinterpret_cast<float *>(sm + S0H);
      {
        const int c0 = g16;
        float x[16], dkr[16], dp[16];
        tmem_ld16(tm + lane + T_R3 + c0, x);
        lds16(Gam + c0, dkr);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int t = c0 + i;
          stg[t * D + j] = x[i];
          if (tnh) {  // the derivative of c tanh(x / c) instead of the mask
            const uint32_t w = (i < 8 ? reinterpret_cast<const uint32_t *>(&dd0)
                                      : reinterpret_cast<const uint32_t *>(&dd1))[(i & 7) >> 1];
            dp[i] = -grad_uq16((i & 1) ? w >> 16 : w & 0xffffu) * x[i];
          } else {
            dp[i] = ((m >> i) & 1u) ? -x[i] : 0.f;
          }
          dP[i] = dp[i];
          dkr[i] = (rla || stl) ? 0.f : -dkr[i] * x[i];
        }
        put16s(sm + S2H, sm + S2L, j, c0, dkr);
        put16s(sm + S3H, sm + S3L, j, c0, dp);
      }
    }
    // ---- phase C: U_R += K^T dKR ; Ap^T dP
    ok = phase_run(K, tid, [&] {
      static_assert(S0L == S0H + 16384, "contiguous");
      bulk_s2g(P.dX2buf + chunk * 64 * D, sm + S0H, 32768);  // (published by this barrier)
      bulk_commit();
      if (!slot_wait<1>(K, K.phB)) return false;
      const uint32_t i128 = idesc_bf16(128, 128);
      mma_tile_kmn(tm + T_DR, sb + S2H, 0, sb + KQ, 16384, 4, i128, true);
      mma_tile_kmn(tm + T_DR, sb + S2L, 0, sb + KQ, 16384, 4, i128, true);
      mma_s3_kmn(tm + T_R3, sb + S3H, sb + S3L, sb + SLOTB, sb + SLOTB + 8192, 16384,
                 idesc_bf16(128, 64), false);
      bulk_wait_read();  // the staging is rewritten next
      return true;
    });
    if (!ok) break;
    if (tid == 0 && c > 0) load_mq(chunk - 1);
    {  // dE = dE_partial + Ap^T dP; dQS = Gam dO (dR is complete in TMEM)
      {
        const int c0 = g16;
        float a[16], e[16], dqs[16];
        tmem_ld16x2(tm + lane + T_R4 + c0, a, tm + lane + T_R3 + c0, e);
        // the base read-out Gam Q S0 (plain combine: Gprev Q S0)
        lds16((mods & RDN_FLAG_PLAIN_COMBINE) ? Gprev + c0 : Gam + c0, dqs);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          a[i] += e[i];
          dqs[i] = p.scale * dqs[i] * dO(c0 + i);
        }
        put16s(sm + S0H, sm + S0L, j, c0, a);
        put16s(sm + S1H, sm + S1L, j, c0, dqs);
      }
    }
    // ---- phase D: dX = T_beta^T dE ; U_S = Q^T dQS
    ok = phase_run(K, tid, [&] {
      if (!slot_wait<0>(K, K.phA)) return false;
      mma_s3_kmn(tm + T_R3, sb + S0H, sb + S0L, sb + SLOTA, sb + SLOTA + 8192, 16384,
                 idesc_bf16(128, 64), false);
      const uint32_t i128 = idesc_bf16(128, 128);
      mma_tile_kmn(tm + T_DS, sb + S1H, 0, sb + KQ + 8192, 16384, 4, i128, true);
      mma_tile_kmn(tm + T_DS, sb + S1L, 0, sb + KQ + 8192, 16384, 4, i128, true);
      return true;
    });
    if (!ok) break;
    if (tid == 0 && c > 0) load_slot<0>(K, sm + SLOTA, rec_bytes(p, chunk - 1) + IMG_M2, 16384);
    if (c > 0) {  // every thread is past its last read of this chunk's dO
      if (!tma)
        fetch_do(c - 1);
      else if (tid == 0)
        tma_do(c - 1);
    }
    {  // dX -> dv = -dP + dX ; dKS = Gprev dP - Gam dX; dX (fp32 [t][j]) and dv
       // (bf16 [t][j]) staged in the free scratch tiles
      float *stg = reinterpret_cast<float *>(sm + S0H);
      __nv_bfloat16 *dvs = reinterpret_cast<__nv_bfloat16 *>(sm + S1H);
      float *dvs32 = reinterpret_cast<float *>(sm + S1H);  // (fp32 dv: over S1H and S1L)
      static_assert(S1L == S1H + 16384, "fp32 dv staging spans the pair");
      {
        const int c0 = g16;
        float x[16], dks[16], gm[16];
        tmem_ld16(tm + lane + T_R3 + c0, x);
        // the prediction's state term: Gprev K S0 (decayed residual: Gam K S0)
        lds16((mods & RDN_FLAG_DECAYED_RESIDUAL) ? Gam + c0 : Gprev + c0, dks);
        lds16(Gam + c0, gm);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int t = c0 + i;
          stg[t * D + j] = x[i];
          if (P.f32g)
            dvs32[t * D + j] = x[i] - dP[i];
          else
            dvs[t * D + j] = __float2bfloat16_rn(x[i] - dP[i]);
          dks[i] = dks[i] * dP[i] - (rla ? 0.f : gm[i] * x[i]);
        }
        put16s(sm + S2H, sm + S2L, j, c0, dks);
      }
      fence_async_smem();
      __syncthreads();
      if (tid == 0) {
        bulk_s2g(P.dXbuf + chunk * 64 * D, sm + S0H, 32768);
        bulk_commit();
      }
      if (P.f32g) {  // dv rows, 16 bytes at a time
        float *dvf = (float *)P.dv;
        for (int e = tid; e < 64 * 32; e += NTC) {
          const int t = e >> 5, chn = e & 31;
          if (t < n)
            *reinterpret_cast<uint4 *>(dvf + ((size_t)(tok0 + t0 + t) * H + h) * D + chn * 4) =
                *reinterpret_cast<const uint4 *>(sm + S1H + t * 512 + chn * 16);
        }
      } else {
        for (int e = tid; e < 64 * 16; e += NTC) {
          const int t = e >> 4, chn = e & 15;
          if (t < n)
            *reinterpret_cast<uint4 *>(dv + ((size_t)(tok0 + t0 + t) * H + h) * D + chn * 8) =
                *reinterpret_cast<const uint4 *>(sm + S1H + t * 256 + chn * 16);
        }
      }
    }
    // ---- phase E: U_S += K^T dKS
    ok = phase_run(K, tid, [&] {
      const uint32_t i128 = idesc_bf16(128, 128);
      mma_tile_kmn(tm + T_DS, sb + S2H, 0, sb + KQ, 16384, 4, i128, true);
      mma_tile_kmn(tm + T_DS, sb + S2L, 0, sb + KQ, 16384, 4, i128, true);
      bulk_wait_read();  // the staging is rewritten next (the gradient tiles)
      return true;
    });
    if (!ok) break;
    if (c > 0) {  // the next chunk's inputs, while this one finishes
      if (!tma)
        fetch_kq(c - 1);
      else if (tid == 0)
        tma_kq(c - 1);
      pre = fetch_pre(c - 1);
    }
    // the carried gradients' tiles (dS, dR complete in TMEM): the A operands of
    // the next chunk's phase A (the scratch tiles in their place are done with)
#pragma unroll 1
    for (int c0 = g16; c0 < D; c0 += 64) {
      float s[16], r[16];
      tmem_ld16x2(tm + lane + T_DS + c0, s, tm + lane + T_DR + c0, r);
      put_grad16(DSH, DSL, c0, s);
      put_grad16(DRH, DRL, c0, r);
    }
    fence_async_smem();  // the tiles are read by the MMAs and by a bulk copy
  }
  if (ok) {
    for (int c0 = g16; c0 < D; c0 += 64) {
      float s[16], r[16];
      tmem_ld16(tm + lane + T_DS + c0, s);
      tmem_ld16(tm + lane + T_DR + c0, r);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (P.dS0) P.dS0[st_base + (size_t)(c0 + i) * D + j] = s[i];
        if (P.dR0) P.dR0[st_base + (size_t)(c0 + i) * D + j] = r[i];
      }
    }
  } else if (tid == 0) {
    if (p.err) atomicExch(p.err, RDN_ERR_TIMEOUT);
    // no copy into this CTA's shared memory or MMA outlives it (bounded waits)
    ctl_drain(K);
    for (; tma_seen < tma_arms; ++tma_seen) mbar_wait(K.barC, tma_seen & 1u);
  }
  cp_async_wait_all();
  if (tid == 0) bulk_wait_all();
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, 512);
}

// ======================================================================== 3
// bwd_post: everything that reduces over the value dimension, followed by the
// chunk-matrix part of the gradients (the work bwd_finish of chunk_bwd.cu does
// for the SIMT path), one persistent CTA of 512 threads per SM walking the
// chunks.  Thread (j, qd) owns value column j = TMEM lane j and quarter qd of
// the chunk's tokens (or of the key rows of a state).
//
// dK and dQ are accumulated transposed in TMEM (lane = key dimension d,
// column t for dK_t, 64 + t for dQ_t):
//   P2  R0 [dKR ; dQR]^T        P3  S0 [dKS ; dQS]^T
//   P4  dR (diag(wR) E2)^T + dS (diag(wS) E)^T        (dK columns only)
//   P7  K^T [dKK + dKK^T ; dQK]^T, and Q^T dQK kept apart (scaled at read-out)
// The C x C gradients (P5) and the Gram matrices K K^T, Q K^T go through
// shared memory for the element-wise pass over (t, i) of Eqs. for T, M2, Mq, Ap.
// Q enters the tensor-core products unscaled; the scale is applied to the
// fp32 results.
namespace po {
constexpr int NTP = 512;
constexpr uint32_t SA = 0, SB = 65536;  // state images: hi 2 x 16 KB | lo 2 x 16 KB, rows j
constexpr uint32_t XH = 131072, XL = 147456, YH = 163840, YL = 180224;  // [j][t] atoms
constexpr uint32_t KQ = 196608;         // K rows 0..63, Q rows 64..127, 2 x 16 KB
constexpr uint32_t VEC = 229376;        // Gam Gprev wS wR gamma dGam dGprev (7 x 64), dGamC
constexpr uint32_t RED = VEC + 7 * 64 * 4 + 16;  // the 16 warps' <dS, S0> + <dR, R0> parts
constexpr uint32_t PARK = RED + 16 * 4;           // per-token sums kept to the gate pass (A8)
constexpr uint32_t CTL = PARK + A8::FLOATS * 4;
constexpr uint32_t SLOT = CTL + 48;
constexpr size_t SMEM = SLOT + 16;
static_assert(SMEM <= 232448, "shared memory");
// element-wise pass: fp32 C x C tiles (row stride 65) over the state images
constexpr int LDC = 65, TILE = 64 * LDC;
constexpr int F_DM2 = 0, F_DMQ = TILE, F_DAB = 2 * TILE, F_KK = 3 * TILE, F_DAG = 4 * TILE,
              F_DAP = 5 * TILE, F_QK = 6 * TILE, F_VEC = 7 * TILE;
static_assert((F_VEC + 9 * 64 + 6 * 8 * 64) * 4 <= (int)XH, "finish scratch");
// TMEM columns
constexpr uint32_t T_KS = 0, T_KR = 128, T_DKQ = 256, T_D2 = 384;
constexpr uint32_t T_KDR = 0, T_KDS = 64, T_U1 = 128, T_U2 = 192;  // P4, after the read-outs
// P5 (after the read-outs and P4): two 128-column products and the Gram one
// (past the dK, dQ accumulators)
constexpr uint32_t T_P5A = 0, T_P5B = 128, T_GR = 448;
}  // namespace po

// Sums over the 128 value columns: thread (j, qd) holds v[t - 16 qd] for the
// tokens t of its quarter.  Warp 4 qd + w covers columns [32 w, 32 w + 32);
// after the warp's transposed reduction lane 2 i holds its sum for token
// 16 qd + i.  Each warp leaves its part (16 floats) at part[16 warp, +16), so
// that several sums share the barriers ...
__device__ __forceinline__ void warp_row_part(const float (&v)[16], float *part, int tid) {
  const float o = warp_transpose_reduce16(v);
  const int warp = tid >> 5, lane = tid & 31;
  if (!(lane & 1)) part[warp * 16 + (lane >> 1)] = o;
}
// ... and, after a barrier, token t's total is the sum of its four warps' parts.
__device__ __forceinline__ float row_total(const float *part, int t) {
  const int g = t >> 4, i = t & 15;
  return part[(4 * g) * 16 + i] + part[(4 * g + 1) * 16 + i] + part[(4 * g + 2) * 16 + i] +
         part[(4 * g + 3) * 16 + i];
}

template <bool kGeneric>  // (as bwd_chain_kernel's)
__global__ void __launch_bounds__(po::NTP, 1) bwd_post_kernel(TcBwdParams P) {
  using namespace po;
  extern __shared__ __align__(1024) uint8_t sm[];
  const uint32_t sb = smem_u32(sm);
  const FwdParams &p = P.f;
  if (sb & 1023u) {
    if (threadIdx.x == 0 && p.err) atomicExch(p.err, RDN_ERR_CUDA);
    return;
  }
  float *vec = reinterpret_cast<float *>(sm + VEC);
  float *Gam = vec, *Gprev = vec + 64, *wS = vec + 128, *wR = vec + 192, *gamv = vec + 256;
  float *dGamS = vec + 320, *dGprevS = vec + 384, *dGamC = vec + 448;
  float *red = reinterpret_cast<float *>(sm + RED);
  float *park = reinterpret_cast<float *>(sm + PARK);
  uint32_t *slot = reinterpret_cast<uint32_t *>(sm + SLOT);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j = tid & 127, qd = tid >> 7, tb = 16 * qd;
  const int H = p.H;
  const size_t nct = (size_t)total_records(p);
  const float scale = p.scale;
  const bool rla = kGeneric && P.rla;
  // residual against a_t S_{t-1} k_t; o = S_{t-1} q_t + R_t q_t
  const bool dec_res = kGeneric && (p.mods & RDN_FLAG_DECAYED_RESIDUAL);
  const bool plain = kGeneric && (p.mods & RDN_FLAG_PLAIN_COMBINE);
  // the tanh residual: dP = -(1 - (r/c)^2) dX2 from the stored derivative
  const bool tnh = kGeneric && (p.mods & RDN_FLAG_TANH_RESIDUAL);
  // the stateless correction: R0 enters nothing (its read-outs, its P2 and
  // <dR, R0> terms are zero), wR is a constant one-hot (no gate gradient
  // through it) and M2 is diag(q_t . k_t) (no decay, no rate)
  const bool stl = kGeneric && (p.mods & RDN_FLAG_STATELESS_AUX);
  const __nv_bfloat16 *q = (const __nv_bfloat16 *)p.q, *k = (const __nv_bfloat16 *)p.k,
                      *dOp = (const __nv_bfloat16 *)P.dO;
  Ctl K;
  ctl_init(K, sm + CTL, tid);
  if (warp == 0) tmem_alloc(slot, 512);
  fence_before_sync();
  __syncthreads();  // barriers initialised, TMEM allocated
  fence_after_sync();
  const uint32_t tm = *slot;
  // A chunk's inputs are fetched in two parts, each during the previous chunk
  // (this CTA loops over chunks): the chunk-start states, fp32, staged where
  // their images go; then dX2, dX (fp32 [t][j], staged in the pair's place
  // until P2) and the K, Q tile.
  auto fetch_states = [&](size_t ck) {
    if (tid == 0) {
      ctl_arm<0>(K, 131072);
      bulk_g2s(sm + SA, P.Sc + ck * D * D, 65536, K.barA);
      bulk_g2s(sm + SB, P.Rc + ck * D * D, 65536, K.barA);
    }
  };
  auto fetch_rest = [&](size_t ck) {
    if (tid == 0) {
      ctl_arm<2>(K, 65536);
      bulk_g2s(sm + XH, P.dX2buf + ck * 64 * D, 32768, K.barC);
      bulk_g2s(sm + YH, P.dXbuf + ck * 64 * D, 32768, K.barC);
    }
    int s_, h_, cc_;
    rec_decode(p, (long long)ck, s_, h_, cc_);
    const SeqSpan sp_ = seq_span(p, s_, h_);
    const long long tok0_ = sp_.tok0;
    const int t0_ = cc_ * 64, n_ = min(64, sp_.len - t0_);
    for (int e = tid; e < 64 * 16; e += NTP) {  // K, Q (exact bf16), asynchronous
      const int t = e >> 4, chn = e & 15;
      const bool vld = t < n_;
      const size_t off = ((size_t)(tok0_ + t0_ + (vld ? t : 0)) * H + h_) * D + chn * 8;
      const int blk = chn >> 3, cc = (chn & 7) * 8;
      cp_async16(sm + KQ + blk * 16384 + sw128(t, cc), k + off, vld);
      cp_async16(sm + KQ + blk * 16384 + sw128(64 + t, cc), q + off, vld);
    }
  };
  if (blockIdx.x < nct) {
    fetch_states(blockIdx.x);
    fetch_rest(blockIdx.x);
  }
  // the previous chunk's dq, dk from TMEM to HBM (row = its first token row *
  // H + h; n = its valid tokens, -1 = none pending)
  long long dkq_row = 0;
  int dkq_n = -1;
  auto store_dkq = [&]() {
    __nv_bfloat16 *dk = (__nv_bfloat16 *)P.dk, *dq = (__nv_bfloat16 *)P.dq;
    const uint32_t tl = (uint32_t)((warp & 3) * 32) << 16;
    float a[16], d2[16], qv[16];
    tmem_ld16x2(tm + tl + T_DKQ + tb, a, tm + tl + T_D2 + tb, d2);
    tmem_ld16(tm + tl + T_DKQ + 64 + tb, qv);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int t = tb + i;
      if (t < dkq_n) {
        const size_t off = (size_t)(dkq_row + (long long)t * H) * D + j;
        if (P.f32qk) {
          ((float *)P.dk)[off] = a[i] + scale * d2[i];
          ((float *)P.dq)[off] = scale * qv[i];
        } else {
          dk[off] = __float2bfloat16_rn(a[i] + scale * d2[i]);
          dq[off] = __float2bfloat16_rn(scale * qv[i]);
        }
      }
    }
    dkq_n = -1;
  };
  bool ok = true;
  uint32_t it = 0;  // chunks done by this CTA: the parity of barrier B
  for (size_t chunk = blockIdx.x; chunk < nct && ok; chunk += gridDim.x, ++it) {
  const size_t next = chunk + gridDim.x;
  int sq, h, c;
  rec_decode(p, (long long)chunk, sq, h, c);
  const SeqSpan sp = seq_span(p, sq, h);
  const long long tok0 = sp.tok0;
  const int t0 = c * 64, n = min(64, sp.len - t0);
  const float *recf = p.ws + chunk * kRecFloats;
  const float *S0 = P.Sc + chunk * D * D, *R0 = P.Rc + chunk * D * D;
  const uint8_t *gimg = P.gimg + chunk * 131072;  // dS hi | dR hi | dS lo | dR lo
  // this thread's tokens of dX2, dX (from the staging) and dO: read after P1 is
  // issued, so that the MMA issue does not wait behind them
  float x2v[16], xv[16], dov[16];
  // this thread's key rows of a state: [32 qd, 32 qd + 32), the columns
  // [32 (qd & 1), +32) of 64-row block qd >> 1 of the image
  const uint32_t kblk = (uint32_t)(qd >> 1) * 16384u;
  const int kc0 = 32 * (qd & 1);
  // fp32 [i][j] state staged at `base` -> rows j of its (hi | lo) image at
  // `base` (every thread reads its values before any writes)
  auto stage_to_image = [&](uint32_t base) {
    const float *st = reinterpret_cast<const float *>(sm + base);
    float v[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = st[(32 * qd + i) * D + j];
    __syncthreads();
#pragma unroll
    for (int c0 = 0; c0 < 32; c0 += 16) {
      float w[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) w[i] = v[c0 + i];
      put16s(sm + base + kblk, sm + base + 32768 + kblk, j, kc0 + c0, w);
    }
  };
  // sum over this thread's entries of (image at base, hi + lo) * x[i][j]
  auto dot_image = [&](uint32_t base, const float (&x)[32]) {
    float s = 0.f;
#pragma unroll
    for (int k8 = 0; k8 < 4; ++k8) {
      const int c8 = (kc0 >> 3) + k8;
      const uint32_t o = base + kblk + j * 128 + (((c8 ^ (j & 7)) & 7) << 4);
      const uint4 hv = *reinterpret_cast<const uint4 *>(sm + o);
      const uint4 lv = *reinterpret_cast<const uint4 *>(sm + o + 32768);
      const __nv_bfloat16 *hb = reinterpret_cast<const __nv_bfloat16 *>(&hv);
      const __nv_bfloat16 *lb = reinterpret_cast<const __nv_bfloat16 *>(&lv);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        s += (__bfloat162float(hb[e]) + __bfloat162float(lb[e])) * x[k8 * 8 + e];
    }
    return s;
  };
  // this thread's 16 tokens of a [j][t] atom pair (hi, lo)
  auto put_tok = [&](const float (&x)[16], uint32_t hi, uint32_t lo) {
    put16s(sm + hi, sm + lo, j, tb, x);
  };
  const uint32_t tm_lane = (uint32_t)((warp & 3) * 32) << 16;
  const uint32_t i128 = idesc_bf16(128, 128), i64 = idesc_bf16(128, 64);

  cp_async_wait_all();  // K, Q tile (published by the barriers below)
  if (!ctl_wait<0>(K, 0, tid)) *K.flag = 1;  // phase_run below reports it to every thread
#pragma unroll 1
  for (int s2 = 0; s2 < 2; ++s2) stage_to_image(s2 ? SB : SA);  // images of S0, R0
  // ---- P1: read-outs [K S0 | Q S0] and [K R0 | Q R0] (lanes j, columns t')
  phase_issue(K, tid, [&] {
    const uint32_t t_ = *slot;
    mma_tile<true>(t_ + T_KS, sb + SA, 16384, sb + KQ, 16384, 8, i128, false);
    mma_tile<true>(t_ + T_KS, sb + SA + 32768, 16384, sb + KQ, 16384, 8, i128, true);
    mma_tile<true>(t_ + T_KR, sb + SB, 16384, sb + KQ, 16384, 8, i128, false);
    mma_tile<true>(t_ + T_KR, sb + SB + 32768, 16384, sb + KQ, 16384, 8, i128, true);
    return true;
  });
  // while P1 runs: this thread's dO and the gate vectors (loads first, their
  // latency under the stores), the previous chunk's dq, dk, then dX2 and dX
  // from their staging
  const unsigned long long m = tnh ? 0ull : P.mask[chunk * D + j] >> tb;
  const uint16_t *drow = reinterpret_cast<const uint16_t *>(P.mask) + (chunk * D + j) * 64 + tb;
  __nv_bfloat16 dob[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int t = tb + i;
    dob[i] = t < n ? dOp[((size_t)(tok0 + t0 + t) * H + h) * D + j] : __float2bfloat16(0.f);
  }
  float gvv[5];
  if (tid < 64) {
    gvv[0] = recf[OFF_VEC + V_GAM + tid];
    gvv[1] = recf[OFF_VEC + V_GPREV + tid];
    gvv[2] = recf[OFF_VEC + V_WS + tid];
    gvv[3] = recf[OFF_VEC + V_WR + tid];
    gvv[4] = tid < n ? p.gamma[(size_t)(tok0 + t0 + tid) * H + h] : 0.f;
  }
  if (dkq_n >= 0) store_dkq();
#pragma unroll
  for (int i = 0; i < 16; ++i) dov[i] = __bfloat162float(dob[i]);
  if (tid < 64) {
    Gam[tid] = gvv[0];
    Gprev[tid] = gvv[1];
    wS[tid] = gvv[2];
    wR[tid] = gvv[3];
    gamv[tid] = gvv[4];
  }
  if (!ctl_wait<2>(K, 0, tid)) *K.flag = 1;
  {
    const float *x2s = reinterpret_cast<const float *>(sm + XH);
    const float *xs = reinterpret_cast<const float *>(sm + YH);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      x2v[i] = x2s[(tb + i) * D + j];
      xv[i] = xs[(tb + i) * D + j];
    }
  }
  ok = phase_wait(K);  // (its barrier also publishes the gate vectors)
  auto dp_of = [&](int i) {
    if (tnh) return -grad_uq16(drow[i]) * x2v[i];
    return ((m >> i) & 1ull) ? -x2v[i] : 0.f;
  };
  if (ok) {  // per-token gate terms: dGam, dGprev, and <dR,R0> + <dS,S0>
    // the three sums' warp parts go where dX2 was staged (read into x2v above)
    float *part = reinterpret_cast<float *>(sm + XH);
    float rv[16];
    {
      float qs[16], qr[16];
      tmem_ld16x2(tm + tm_lane + T_KS + 64 + tb, qs, tm + tm_lane + T_KR + 64 + tb, qr);
      if (stl) {
#pragma unroll
        for (int i = 0; i < 16; ++i) qr[i] = 0.f;
      }
      // d gamma_t from the read-out: dO_t . (Gam_t Q R0)_t (the rest of Oa_t in P6)
      lds16(Gam + tb, rv);
#pragma unroll
      for (int i = 0; i < 16; ++i) rv[i] = plain ? 0.f : scale * rv[i] * dov[i] * qr[i];
      warp_row_part(rv, part, tid);
      lds16(gamv + tb, rv);
#pragma unroll
      for (int i = 0; i < 16; ++i)  // (plain combine: Gprev Q S0 and no gamma_t)
        rv[i] = plain ? scale * dov[i] * qr[i] : scale * dov[i] * (qs[i] + rv[i] * qr[i]);
    }
    {
      float ks[16], kr[16];
      tmem_ld16x2(tm + tm_lane + T_KS + tb, ks, tm + tm_lane + T_KR + tb, kr);
      if (stl) {
#pragma unroll
        for (int i = 0; i < 16; ++i) kr[i] = 0.f;
      }
      if (!rla) {
#pragma unroll
        for (int i = 0; i < 16; ++i) rv[i] -= x2v[i] * kr[i] + xv[i] * ks[i];
      }
      // the prediction's state term: Gprev K S0 (decayed residual: Gam K S0)
      if (dec_res) {
#pragma unroll
        for (int i = 0; i < 16; ++i) rv[i] += dp_of(i) * ks[i];
      }
      warp_row_part(rv, part + 256, tid);
#pragma unroll
      for (int i = 0; i < 16; ++i) rv[i] = dec_res ? 0.f : dp_of(i) * ks[i];
      if (plain) {  // the base read-out's gate is Gprev
        float qs[16];
        tmem_ld16(tm + tm_lane + T_KS + 64 + tb, qs);
#pragma unroll
        for (int i = 0; i < 16; ++i) rv[i] += scale * dov[i] * qs[i];
      }
    }
    warp_row_part(rv, part + 512, tid);
    __syncthreads();
    if (tid < 192) {
      const int w = tid >> 6, t = tid & 63;
      const float tot = row_total(part + 256 * w, t);
      if (w == 0)
        park[A8::V_DGAM_OUT + t] = tot;
      else
        (w == 1 ? dGamS : dGprevS)[t] = tot;
    }
    __syncthreads();  // (P2's operands go where the parts are)
    // ---- P2: dK, dQ += R0 [dKR ; dQR]^T, dKR = -Gam dX2, dQR = Gam gamma dO
    float x[16], y[16];
    lds16(Gam + tb, x);
    lds16(gamv + tb, y);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      y[i] = stl ? 0.f : (plain ? 1.f : y[i]) * x[i] * dov[i];
      x[i] = (rla || stl) ? 0.f : -x[i] * x2v[i];
    }
    put_tok(x, XH, XL);
    put_tok(y, YH, YL);
    ok = phase_run(K, tid, [&] {
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SB, 16384, sb + XH, 32768, 8, i128, false);
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SB, 16384, sb + XL, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SB + 32768, 16384, sb + XH, 32768, 8, i128, true);
      return true;
    });
  }
  if (ok && tid == 0) {  // R0's image is done with: dR's image into its place
    ctl_arm<1>(K, 65536);
    bulk_g2s(sm + SB, gimg + 32768, 32768, K.barB);
    bulk_g2s(sm + SB + 32768, gimg + 98304, 32768, K.barB);
  }
  // <dR, R0> + <dS, S0> into dGamC, each computed while MMAs run: the states
  // are re-read from L2 (not through L1, which holds the prefetched dO rows),
  // the gradients' images are in the states' places
  float gdot = 0.f;
  auto dot_state = [&](const float *st, uint32_t img) {
    float x[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] = __ldcg(st + (size_t)(32 * qd + i) * D + j);
    return dot_image(img, x);
  };
  if (ok) {  // ---- P3: dK, dQ += S0 [dKS ; dQS]^T, dKS = Gprev dP - Gam dX, dQS = Gam dO;
             // meanwhile <dR, R0>
    float x[16], y[16];
    lds16(dec_res ? Gam + tb : Gprev + tb, x);
    lds16(Gam + tb, y);
    float gq[16];  // the base read-out's gate: Gam (plain combine: Gprev)
    lds16(plain ? Gprev + tb : Gam + tb, gq);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      x[i] = x[i] * dp_of(i) - (rla ? 0.f : y[i] * xv[i]);
      y[i] = gq[i] * dov[i];
    }
    put_tok(x, XH, XL);
    put_tok(y, YH, YL);
    ok = phase_run_with(K, tid, [&] {
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SA, 16384, sb + XH, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SA, 16384, sb + XL, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_DKQ, sb + SA + 32768, 16384, sb + XH, 32768, 8, i128, true);
      return true;
    }, [&] {
      if (!ctl_wait<1>(K, it & 1u, tid)) *K.flag = 1;  // dR's image
      gdot = stl ? 0.f : dot_state(R0, SB);
    });
  }
  if (ok && tid == 0) {  // and dS's image into S0's; the E2^T, E^T images into the pair's
    ctl_arm<0>(K, 65536);
    bulk_g2s(sm + SA, gimg, 32768, K.barA);
    bulk_g2s(sm + SA + 32768, gimg + 65536, 32768, K.barA);
    ctl_arm<2>(K, 65536);
    bulk_g2s(sm + XH, P.E2buf + chunk * 32768, 32768, K.barC);  // hi at XH, lo at XL
    bulk_g2s(sm + YH, P.Ebuf + chunk * 32768, 32768, K.barC);   // hi at YH, lo at YL
  }
  // this thread's 16 tokens of row j of a (hi | lo) image of a [j][t] matrix
  auto image_row = [&](uint32_t base, float (&out)[16]) {
#pragma unroll
    for (int k8 = 0; k8 < 2; ++k8) {
      const int c8 = (tb >> 3) + k8;
      const uint32_t o = base + j * 128 + (((c8 ^ (j & 7)) & 7) << 4);
      const uint4 hv = *reinterpret_cast<const uint4 *>(sm + o);
      const uint4 lv = *reinterpret_cast<const uint4 *>(sm + o + 16384);
      const __nv_bfloat16 *hb = reinterpret_cast<const __nv_bfloat16 *>(&hv);
      const __nv_bfloat16 *lb = reinterpret_cast<const __nv_bfloat16 *>(&lv);
#pragma unroll
      for (int e = 0; e < 8; ++e) out[k8 * 8 + e] = __bfloat162float(hb[e]) + __bfloat162float(lb[e]);
    }
  };
  if (ok) {  // ---- P4: dR E2^T, dS E^T (scaled by wR, wS per token below); K dR, K dS read-outs;
             // meanwhile <dS, S0> and the dGamC reduction
    if (!ctl_wait<2>(K, 1, tid)) *K.flag = 1;  // the E images, for every thread
    if (!ctl_wait<0>(K, 1, tid)) *K.flag = 1;  // dS's image
    phase_issue(K, tid, [&] {
      mma_tile_mnmn<true>(tm + T_U1, sb + SB, 16384, sb + XH, 16384, 8, i64, false);
      mma_tile_mnmn<true>(tm + T_U1, sb + SB, 16384, sb + XL, 16384, 8, i64, true);
      mma_tile_mnmn<true>(tm + T_U1, sb + SB + 32768, 16384, sb + XH, 16384, 8, i64, true);
      mma_tile_mnmn<true>(tm + T_U2, sb + SA, 16384, sb + YH, 16384, 8, i64, false);
      mma_tile_mnmn<true>(tm + T_U2, sb + SA, 16384, sb + YL, 16384, 8, i64, true);
      mma_tile_mnmn<true>(tm + T_U2, sb + SA + 32768, 16384, sb + YH, 16384, 8, i64, true);
      // (K dR)^T, (K dS)^T (lanes j, columns t; K exact)
      mma_tile<true>(tm + T_KDR, sb + SB, 16384, sb + KQ, 16384, 8, i64, false);
      mma_tile<true>(tm + T_KDR, sb + SB + 32768, 16384, sb + KQ, 16384, 8, i64, true);
      mma_tile<true>(tm + T_KDS, sb + SA, 16384, sb + KQ, 16384, 8, i64, false);
      mma_tile<true>(tm + T_KDS, sb + SA + 32768, 16384, sb + KQ, 16384, 8, i64, true);
      return true;
    });
    gdot += dot_state(S0, SA);
#pragma unroll
    for (int off = 16; off; off >>= 1) gdot += __shfl_xor_sync(0xffffffffu, gdot, off);
    if (lane == 0) red[warp] = gdot;
    ok = phase_wait(K);  // (its barrier publishes the parts)
    if (ok && tid == 0) {
      float s = 0.f;
      for (int w = 0; w < NTP / 32; ++w) s += red[w];
      *dGamC = s;
    }
  }
  if (ok) {
    // dK += diag(wR) E2 dR^T + diag(wS) E dS^T  (lanes i, columns t of this half)
    {
      float a[16], u1[16], u2[16], wr[16], ws[16];
      tmem_ld16x2(tm + tm_lane + T_DKQ + tb, a, tm + tm_lane + T_U1 + tb, u1);
      tmem_ld16(tm + tm_lane + T_U2 + tb, u2);
      lds16(wR + tb, wr);
      lds16(wS + tb, ws);
#pragma unroll
      for (int i = 0; i < 16; ++i) a[i] = fmaf(wr[i], u1[i], fmaf(ws[i], u2[i], a[i]));
      tmem_st16(tm + tm_lane + T_DKQ + tb, a);
    }
    // dwR_t = sum_j (K dR)[t,j] E2[t,j], dwS_t = sum_j (K dS)[t,j] E[t,j]; the
    // warp parts where dS's image was
    float *part = reinterpret_cast<float *>(sm + SA);
#pragma unroll 1
    for (int w = 0; w < 2; ++w) {
      float ev[16], rv[16];
      image_row(w == 0 ? XH : YH, ev);
      tmem_ld16(tm + tm_lane + (w == 0 ? T_KDR : T_KDS) + tb, rv);
#pragma unroll
      for (int i = 0; i < 16; ++i) rv[i] = (w == 0 && stl) ? 0.f : rv[i] * ev[i];
      warp_row_part(rv, part + 256 * w, tid);
    }
    __syncthreads();
    if (tid < 128) {  // read in the gate pass
      const int w = tid >> 6, t = tid & 63;
      park[(w == 0 ? A8::V_DWR : A8::V_DWS) + t] = row_total(part + 256 * w, t);
    }
    __syncthreads();  // (P5's operands go where the parts are)
  }
  // ---- P5: C x C gradients (lanes t' of a stacked pair, columns s of [E2 ; E])
  //   [dO ; dX2] [E2 ; E]^T -> dO E2^T | dO E^T ; dX2 E2^T | (unused)
  //   [dX ; dP] [E2 ; E]^T  -> (unused) | dX E^T ; (unused) | dP E^T
  //   and the Gram matrices [K ; Q] K^T, all in one phase: 128-column
  //   products take about the issue time of 64-column ones
  // images: E2 at XH (hi | lo), E at YH (hi | lo), 32 KB apart; the pair
  // [dO ; dX2] at SA (dO atom hi SA, lo SA + 16 KB; dX2 atom hi SA + 32 KB, lo
  // SA + 48 KB) and [dX ; dP] at SB the same way (dR's image is done with)
  // token tid's g and beta for the element-wise pass, loaded while P5 runs
  float g_t = 0.f, beta_t = 0.f;
  if (ok) {
    if (tid < n) {
      const size_t off = (size_t)(tok0 + t0 + tid) * H + h;
      g_t = p.g[off];
      beta_t = p.beta[off];
    }
    float y[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) y[i] = dp_of(i);
    put_tok(xv, SB, SB + 16384);
    put_tok(y, SB + 32768, SB + 49152);
    put_tok(dov, SA, SA + 16384);  // gamma_t enters in the element-wise pass
    put_tok(x2v, SA + 32768, SA + 49152);
    static_assert(YH - XH == 32768 && YL - XL == 32768, "the [E2 ; E] atoms");
    ok = phase_run(K, tid, [&] {
      mma_tile_mnmn<true>(tm + T_P5A, sb + SA, 32768, sb + XH, 32768, 8, i128, false);
      mma_tile_mnmn<true>(tm + T_P5A, sb + SA, 32768, sb + XL, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_P5A, sb + SA + 16384, 32768, sb + XH, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_P5B, sb + SB, 32768, sb + XH, 32768, 8, i128, false);
      mma_tile_mnmn<true>(tm + T_P5B, sb + SB, 32768, sb + XL, 32768, 8, i128, true);
      mma_tile_mnmn<true>(tm + T_P5B, sb + SB + 16384, 32768, sb + XH, 32768, 8, i128, true);
      mma_tile<true>(tm + T_GR, sb + KQ, 16384, sb + KQ, 16384, 8, i64, false);
      return true;
    });
  }
  // the next chunk's states into L2 while the element-wise pass and P7 run
  // (their copies into shared memory start once the element-wise pass is done
  // with the region, while P7 runs)
  if (ok && tid == 0 && next < nct) {
    prefetch_l2_bulk(P.Sc + next * D * D, 65536);
    prefetch_l2_bulk(P.Rc + next * D * D, 65536);
  }
  // ---- element-wise pass over (t, i): the gradients of the chunk matrices'
  // entries turned into gradients of K K^T, Q K^T and of the gates
  float *F = reinterpret_cast<float *>(sm);
  float *cum = F + F_VEC, *cprev = cum + 64, *bet = cum + 128, *gam = cum + 192, *gg = cum + 256,
        *dcum = cum + 320, *dcprev = cum + 384, *dbet = cum + 448, *dgam = cum + 512;
  float *prt = cum + 576;  // [6][8][64] partial sums
  float o_dg = 0.f, o_dbeta = 0.f, o_dgamma = 0.f;  // this thread's token's gate gradients
  if (ok) {
    {
      const int r = j & 63;
      {
        float g1[16], g2[16], g3[16], gr[16];
        // g1: dO E2^T (rows t < 64) | dX2 E2^T; g2: dO E^T | dP E^T; g3: dX E^T
        tmem_ld16x2(tm + tm_lane + T_P5A + tb, g1,
                    tm + tm_lane + (j < 64 ? T_P5A : T_P5B) + 64 + tb, g2);
        tmem_ld16x2(tm + tm_lane + T_P5B + 64 + tb, g3, tm + tm_lane + T_GR + tb, gr);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int e = r * LDC + tb + i;
          if (j < 64) {
            F[F_DM2 + e] = g1[i];
            F[F_DMQ + e] = g2[i];
            F[F_DAB + e] = rla ? 0.f : -g3[i];
            F[F_KK + e] = gr[i];
          } else {
            F[F_DAG + e] = (rla || stl) ? 0.f : -g1[i];  // (no T_gamma to differentiate)
            F[F_DAP + e] = g2[i];
            F[F_QK + e] = scale * gr[i];
          }
        }
      }
    }
    if (tid < 64) {
      gg[tid] = g_t;
      bet[tid] = beta_t;
      gam[tid] = gamv[tid];
    }
    __syncthreads();
    if (warp == 0) {  // in-chunk cumulative log-decay
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
      cum[lane] = a;
      cum[32 + lane] = a2;
      cprev[lane] = a - gg[lane];
      cprev[32 + lane] = a2 - gg[32 + lane];
    }
    __syncthreads();
    {  // row pass: thread (t, eighth) over i in [8 q8, 8 q8 + 8)
      const int t = tid & 63, q8 = tid >> 6;
      const float ct = cum[t], cpt = cprev[t];
      const float gt = gam[t];
      float rowc = 0.f, rowp = 0.f, dgo = 0.f;
#pragma unroll
      for (int ii = 0; ii < 8; ++ii) {
        const int i = 8 * q8 + ii, e = t * LDC + i;
        float dkk = 0.f, dqk = 0.f, cg = 0.f, cb = 0.f, cm = 0.f;
        if (i <= t) {
          const float dec = __expf(ct - cum[i]);
          const float kk = F[F_KK + e], qk = F[F_QK + e], bi = bet[i], gi = gam[i];
          if (stl) {  // M2 = diag(Q K^T): the diagonal only, no decay, no rate
            if (i == t) {
              const float g1 = F[F_DM2 + e];
              if (!plain) dgo += qk * g1;
              dqk += plain ? g1 : gt * g1;
            }
          } else {  // M2: inclusive, gamma, Q K^T; G1 holds dO E2^T, dM2 = gamma_t dO E2^T
            const float g1 = F[F_DM2 + e];
            if (!plain) dgo += dec * gi * qk * g1;  // d gamma_t += (M2 E2)_t . dO_t
            const float dm = plain ? g1 : gt * g1;
            const float G = dm * dec * gi * qk;
            rowc += G;
            cg += G;
            cm += dm * dec * qk;
            dqk += dm * dec * gi;
          }
          if (i < t) {
            const float decp = __expf(cpt - cum[i]);
            {  // Ap: strict, beta, K K^T, previous-token decay (decayed residual: to t)
              const float dA = dec_res ? dec : decp;
              const float dm = F[F_DAP + e];
              const float G = dm * dA * bi * kk;
              if (dec_res) rowc += G; else rowp += G;
              cg += G;
              cb += dm * dA * kk;
              dkk += dm * dA * bi;
            }
            {  // Mq: strict, beta, Q K^T (plain combine: decay to t-1)
              const float dA = plain ? decp : dec;
              const float dm = F[F_DMQ + e];
              const float G = dm * dA * bi * qk;
              if (plain) rowp += G; else rowc += G;
              cg += G;
              cb += dm * dA * qk;
              dqk += dm * dA * bi;
            }
            {  // A_beta, A_gamma: strict, K K^T
              const float da = F[F_DAB + e], dg2 = F[F_DAG + e];
              const float Gb = da * dec * bi * kk, Gg = dg2 * dec * gi * kk;
              rowc += Gb + Gg;
              cg += Gb + Gg;
              cb += da * dec * kk;
              cm += dg2 * dec * kk;
              dkk += da * dec * bi + dg2 * dec * gi;
            }
          }
        }
        F[F_KK + e] = dkk;
        F[F_QK + e] = dqk;
        F[F_DM2 + e] = cg;
        F[F_DMQ + e] = cb;
        F[F_DAB + e] = cm;
      }
      prt[0 * 512 + q8 * 64 + t] = rowc;
      prt[1 * 512 + q8 * 64 + t] = rowp;
      prt[5 * 512 + q8 * 64 + t] = dgo;
    }
    __syncthreads();
    {  // column pass: thread (i, eighth) over t in [8 q8, 8 q8 + 8)
      const int i = tid & 63, q8 = tid >> 6;
      float sg = 0.f, sbv = 0.f, smv = 0.f;
#pragma unroll
      for (int tt = 0; tt < 8; ++tt) {
        const int e = (8 * q8 + tt) * LDC + i;
        sg += F[F_DM2 + e];
        sbv += F[F_DMQ + e];
        smv += F[F_DAB + e];
      }
      prt[2 * 512 + q8 * 64 + i] = sg;
      prt[3 * 512 + q8 * 64 + i] = sbv;
      prt[4 * 512 + q8 * 64 + i] = smv;
    }
    __syncthreads();
    if (tid < 64) {
      const int i = tid;
      float s5[6];
#pragma unroll
      for (int w = 0; w < 6; ++w) {
        float a = 0.f;
#pragma unroll
        for (int q8 = 0; q8 < 8; ++q8) a += prt[w * 512 + q8 * 64 + i];
        s5[w] = a;
      }
      const float cC = cum[63];
      const float eC = __expf(cC - cum[i]);
      const float dwS = park[A8::V_DWS + i], dwR = park[A8::V_DWR + i];
      dbet[i] = s5[3] + dwS * eC;
      dgam[i] = s5[4] + s5[5] + park[A8::V_DGAM_OUT + i] + dwR * eC;
      dcum[i] = s5[0] - s5[2] - (dwS * bet[i] + dwR * gam[i]) * eC + dGamS[i] * __expf(cum[i]);
      dcprev[i] = s5[1] + dGprevS[i] * __expf(cprev[i]);
    }
    __syncthreads();
    if (warp == 0) {  // chunk-end terms land on cum_C = cum[63] (padding has g = 0)
      const float cC = cum[63];
      float s = 0.f;
      for (int t = lane; t < 64; t += 32)
        s += (park[A8::V_DWS + t] * bet[t] + park[A8::V_DWR + t] * gam[t]) *
             __expf(cC - cum[t]);
#pragma unroll
      for (int off = 16; off; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (lane == 0) dcum[63] += s + *dGamC * __expf(cC);
      __syncwarp();
      // dg_s = sum_{t >= s} dcum_t + sum_{t > s} dcprev_t (reverse scans)
      float a = dcum[63 - lane], a2 = dcum[31 - lane];
      float pa = dcprev[63 - lane], pb = dcprev[31 - lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float ua = __shfl_up_sync(0xffffffffu, a, off), ub = __shfl_up_sync(0xffffffffu, a2, off);
        const float upa = __shfl_up_sync(0xffffffffu, pa, off), upb = __shfl_up_sync(0xffffffffu, pb, off);
        if (lane >= off) {
          a += ua;
          a2 += ub;
          pa += upa;
          pb += upb;
        }
      }
      a2 += __shfl_sync(0xffffffffu, a, 31);
      pb += __shfl_sync(0xffffffffu, pa, 31);
      gg[63 - lane] = a + (pa - dcprev[63 - lane]);
      gg[31 - lane] = a2 + (pb - dcprev[31 - lane]);
    }
    {  // B operand [dKK + dKK^T ; dQK] (rows t, columns i), hi | lo
      const int t = tid & 63, q8 = tid >> 6;
      float v[8], w[8];
#pragma unroll
      for (int ii = 0; ii < 8; ++ii) {
        const int i = 8 * q8 + ii;
        v[ii] = i == t ? 2.f * F[F_KK + t * LDC + t] : F[F_KK + t * LDC + i] + F[F_KK + i * LDC + t];
        w[ii] = F[F_QK + t * LDC + i];
      }
      put8s(sm + XH, sm + XL, t, 8 * q8, v);
      put8s(sm + XH, sm + XL, 64 + t, 8 * q8, w);
    }
    // ---- P7: dK, dQ += K^T [dKK + dKK^T ; dQK]^T ; D2 = Q^T dQK
    phase_issue(K, tid, [&] {
      mma_tile_mnk<true>(tm + T_DKQ, sb + KQ, 16384, sb + XH, 4, i128, true);
      mma_tile_mnk<true>(tm + T_DKQ, sb + KQ, 16384, sb + XL, 4, i128, true);
      mma_tile_mnmn<true>(tm + T_D2, sb + KQ + 8192, 16384, sb + XH + 8192, 16384, 4, i64, false);
      mma_tile_mnmn<true>(tm + T_D2, sb + KQ + 8192, 16384, sb + XL + 8192, 16384, 4, i64, true);
      return true;
    });
    if (tid < n) {  // the vectors live where the next chunk's states are staged
      o_dg = gg[tid];
      o_dbeta = dbet[tid];
      o_dgamma = dgam[tid];
    }
    __syncthreads();
    if (next < nct) fetch_states(next);  // the state images and the fp32 tiles are done with
    if (next < nct) {  // the next chunk's dO rows, mask words and gate vectors into L1
      int s_, h_, cc_;
      rec_decode(p, (long long)next, s_, h_, cc_);
      const SeqSpan sp_ = seq_span(p, s_, h_);
      const long long tok0_ = sp_.tok0;
      const int t0_ = cc_ * 64, n_ = min(64, sp_.len - t0_);
      if (tid < 128) {  // 64 rows of 256 bytes
        const int t = tid >> 1;
        if (t < n_) prefetch_l1_line(dOp + ((size_t)(tok0_ + t0_ + t) * H + h_) * D + (tid & 1) * 64);
      } else if (tid < 136) {  // 128 mask words
        if (!tnh) prefetch_l1_line(P.mask + next * D + (tid - 128) * 16);
      } else if (tid < 148) {  // the record's 6 x 64 gate floats
        prefetch_l1_line(p.ws + next * kRecFloats + OFF_VEC + (tid - 136) * 32);
      } else if (tid < 180) {  // gamma, one line per two tokens
        const int t = 2 * (tid - 148);
        if (t < n_) prefetch_l1_line(p.gamma + (size_t)(tok0_ + t0_ + t) * H + h_);
      }
    }
    ok = phase_wait(K);
    if (ok && next < nct) fetch_rest(next);  // K, Q and the pair region are done with
  }
  if (ok) {
    if (tid < n) {
      const size_t off = (size_t)(tok0 + t0 + tid) * H + h;
      P.dg[off] = o_dg;
      P.dbeta[off] = o_dbeta;
      P.dgamma[off] = o_dgamma;
    }
    // dq, dk of this chunk: read out and stored during the next chunk's P1
    // (T_DKQ, T_D2 keep them until its P2), or after the last chunk
    dkq_row = (tok0 + t0) * H + h;
    dkq_n = n;
  }
  }  // chunks
  if (ok && dkq_n >= 0) store_dkq();
  if (!ok && tid == 0) {
    if (p.err) atomicExch(p.err, RDN_ERR_TIMEOUT);
    ctl_drain(K);  // no bulk copy or MMA of this CTA outlives it
  }
  cp_async_wait_all();  // (nor a cp.async of a chunk not reached)
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, 512);
}

}  // namespace


size_t bwd_tc_extra_bytes(long long nrec, bool deriv) {
  const size_t nct = (size_t)nrec;
  return nct * (4 * 64 * D * sizeof(float) + 2 * (size_t)D * D * sizeof(float) +
                mask_bytes_per_chunk(D, deriv));
}

cudaError_t launch_bwd_tc(const FwdParams &f, const void *dO, const float *dST, const float *dRT,
                          const float *Sc, const float *Rc, void *dq, void *dk, void *dv, float *dg,
                          float *dbeta, float *dgamma, float *dS0, float *dR0, char *extra,
                          bool rla, bool grad_f32, bool dqk_f32, cudaStream_t s) {
  TcBwdParams P;
  P.rla = rla;
  P.f32g = grad_f32;
  P.f32qk = grad_f32 || dqk_f32;
  P.dq = dq;
  P.dk = dk;
  P.dg = dg;
  P.dbeta = dbeta;
  P.dgamma = dgamma;
  P.f = f;
  P.dO = dO;
  P.dST = dST;
  P.dRT = dRT;
  P.Sc = Sc;
  P.Rc = Rc;
  P.dv = dv;
  P.dS0 = dS0;
  P.dR0 = dR0;
  const size_t nct = (size_t)f.nrec;  // record slots (packed sequences: a bound)
  float *x = reinterpret_cast<float *>(extra);
  P.Ebuf = reinterpret_cast<uint8_t *>(x);
  P.E2buf = reinterpret_cast<uint8_t *>(x + nct * 64 * D);
  P.dX2buf = x + 2 * nct * 64 * D;
  P.dXbuf = x + 3 * nct * 64 * D;
  P.gimg = reinterpret_cast<uint8_t *>(x + 4 * nct * 64 * D);
  P.mask = reinterpret_cast<unsigned long long *>(P.gimg + nct * 131072);
  // the chain's tiles of whole chunks by tensor-map copies (else cp.async)
  const long long rows = (long long)f.B * f.T;
  P.tma = make_tile_map(P.map_k, f.k, D, f.H, rows) && make_tile_map(P.map_q, f.q, D, f.H, rows) &&
          make_tile_map(P.map_do, dO, D, f.H, rows);
  const bool saved = f.sv_E && f.sv_E2 && f.sv_mask;  // E, E2, mask kept by the forward
  if (saved) {
    P.Ebuf = f.sv_E;
    P.E2buf = f.sv_E2;
    P.mask = f.sv_mask;
  }
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(bwd_recompute_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)rc::SMEM)) != cudaSuccess)
    return e;
  const bool generic = rla || f.mods != 0;
  auto chain = generic ? bwd_chain_kernel<true> : bwd_chain_kernel<false>;
  auto post = generic ? bwd_post_kernel<true> : bwd_post_kernel<false>;
  if ((e = cudaFuncSetAttribute(chain, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)ch::SMEM)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(post, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)po::SMEM)) != cudaSuccess)
    return e;
  if (!saved) {
    RDN_LAUNCH("bwd_recompute", s, bwd_recompute_kernel<<<(unsigned)nct, NT, rc::SMEM, s>>>(P));
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  RDN_LAUNCH("bwd_chain", s, chain<<<f.nseq * f.H, NTC, ch::SMEM, s>>>(P));
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  int dev = 0, nsm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  const unsigned post_grid = (unsigned)(nct < (size_t)nsm ? nct : (size_t)nsm);  // one CTA per SM
  RDN_LAUNCH("bwd_post", s, post<<<post_grid, po::NTP, po::SMEM, s>>>(P));
  return cudaGetLastError();
}

}  // namespace rdn
