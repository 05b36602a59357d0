/*
 * rdn.h -- C ABI of the GB300 (sm_103a) library for the layer hot path of
 * Residual Linear Attention (RLA) and Residual Delta Net (RDN),
 * "Enhancing Linear Attention with Residual Learning", arXiv 2509.25223.
 *
 * The operation (Section 3.4, "Final Formulations"; residual clipping
 * Section 3.3; gates Section 3.2), per batch element b and head h, token t:
 *
 *   r_t = Clip_[-c,c](v_t - S_{t-1} k_t)                (elementwise in d_v)
 *   RLA: R_t = a_t R_{t-1} + gam_t r_t k_t^T
 *        S_t = a_t S_{t-1} + beta_t v_t k_t^T
 *   RDN: R_t = a_t R_{t-1} (I - gam_t k_t k_t^T) + gam_t r_t k_t^T
 *        S_t = a_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T
 *   o_t = a_t S_{t-1} (scale q_t) + gam_t R_t (scale q_t)
 *
 * with a_t = exp(g_t).  The gates are passed as the log-decay g = log(a) <= 0
 * and the rates beta, gam in [0,1]; the model-side gate projections, the SiLU
 * and the L2 normalisation of q and k (Section 3.4, paragraph after the
 * formulations) happen before these calls.
 *
 * Conventions shared by every entry point:
 *  - Pointers are DEVICE pointers owned by the caller.  The library never
 *    frees them and keeps none of them after the call returns.
 *  - Layouts are contiguous row-major:
 *      q, k          [B,T,H,Dk]        v, o, dO      [B,T,H,Dv]
 *      g, beta, gam  [B,T,H]  fp32
 *      S0,R0,ST,RT   [B,H,Dk,Dv] fp32  (the paper's d_v x d_k state,
 *                                        stored transposed: row i is key dim i)
 *      S_chunks, R_chunks [B,H,NC,Dk,Dv] fp32, NC = ceil(T/64): the states at
 *                    the start of each 64-token chunk.
 *    (packed variable-length sequences change the B axis: rdn_fwd_args
 *    .cu_seqlens.)
 *  - Every pointer must be 16-byte aligned.
 *  - All work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream) and is asynchronous.  Argument errors are reported before
 *    anything is enqueued; launch errors are checked right after the launch;
 *    faults inside a kernel surface at the caller's next synchronisation.
 *  - Scratch memory is the caller's: each entry point that needs it states
 *    the size through its *_workspace_size function, and the caller passes a
 *    device buffer of at least that size (16-byte aligned).  The library
 *    makes no allocation of its own on these paths.
 *  - No C++ exception or abort crosses this boundary.  Every function
 *    returns an rdn_status_t; rdn_last_error() gives a message for the last
 *    failure on the calling thread.
 *  - Calls are reentrant: the library keeps no per-call state outside the
 *    caller's buffers.
 */
#ifndef RDN_H_
#define RDN_H_

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *rdn_stream_t; /* same type as cudaStream_t */

typedef enum {
  RDN_OK = 0,
  RDN_ERR_INVALID_ARG = 1, /* bad shape, NULL where required, c < 0 or NaN */
  RDN_ERR_UNSUPPORTED = 2, /* valid but not implemented (dtype, Dk/Dv, flags) */
  RDN_ERR_CUDA = 3,        /* a CUDA runtime call or launch failed */
  RDN_ERR_TIMEOUT = 4,     /* a bounded device-side wait gave up */
  RDN_ERR_WORKSPACE = 5,   /* workspace missing, too small or misaligned */
  RDN_ERR_MISALIGNED = 6   /* a pointer is not 16-byte aligned */
} rdn_status_t;

typedef enum { RDN_F32 = 0, RDN_BF16 = 1 } rdn_dtype_t;

/* rdn_fwd_args.flags.  RDN_FLAG_SAVE_FOR_BWD (rla_fwd / rdn_fwd; needs
 * S_chunks and R_chunks): the forward also keeps, in its workspace after the
 * per-chunk matrices, the delta errors E and E2 of both passes (RLA: V and r)
 * and the clip mask of every chunk (the intermediates of the residual pass);
 * ask *_fwd_workspace_size with the flag set.  rla_bwd / rdn_bwd given that
 * workspace (fwd.workspace) and the same flag in fwd.flags reads them instead
 * of recomputing them.  On the bf16, Dk = 128 path this removes a pass of the
 * backward; on the others the flag only reserves the space. */
#define RDN_FLAG_SAVE_FOR_BWD 0x1u

/* RDN_FLAG_TIED_GAMMA (all four entry points): the residual rate is tied to
 * the base rate, gamma_t = beta_t (the paper's tied-gate ablation): `gamma`
 * is ignored (may be NULL) and `beta` serves as both.  rla_bwd / rdn_bwd then
 * return in dbeta the gradient w.r.t. the shared gate (the sum of the two
 * gates' gradients of the untied computation); dgamma may be NULL, and if
 * given receives the gamma part alone.  The backward's fwd.flags carries it. */
#define RDN_FLAG_TIED_GAMMA 0x2u

/* The paper's variants of the method (all four entry points; any
 * combination; the backward's fwd.flags carries them):
 *   RDN_FLAG_DECAYED_RESIDUAL  the residual against the decayed prediction,
 *       r_t = Clip(v_t - a_t S_{t-1} k_t) (the gated-delta error);
 *   RDN_FLAG_PLAIN_COMBINE     the ungated output o_t = S_{t-1} q_t + R_t q_t
 *       (output-combination ablation, Section 4.3);
 *   RDN_FLAG_TANH_RESIDUAL     the log-cosh residual of Appendix B with the
 *       threshold as its scale, r_t = c tanh((v_t - S_{t-1} k_t) / c)
 *       (c = 1 is the paper's tanh; c = INFINITY no limit; c = 0 gives 0);
 *   RDN_FLAG_STATELESS_AUX     the stateless correction of the residual-
 *       fitting ablation (Section 4.3): R_t = r_t k_t^T replaces the
 *       recurrence for R, so R0 is ignored (dR0 = 0 unless T = 0) and RT =
 *       r_T k_T^T.
 * Every variant runs on the tensor-core kernels for bf16 inputs with Dk = 128
 * (the tanh residual's backward reads the map's derivative per element, 16-bit
 * fixed point, where the clip mask goes) and on the fp32 chunk kernels for
 * every other dtype and head dimension. */
#define RDN_FLAG_DECAYED_RESIDUAL 0x4u
#define RDN_FLAG_PLAIN_COMBINE 0x8u
#define RDN_FLAG_TANH_RESIDUAL 0x10u
#define RDN_FLAG_STATELESS_AUX 0x20u

/* RDN_FLAG_F32_OUT: results in fp32 for bf16 inputs -- the forward's o
 * (rla_fwd / rdn_fwd) and, given in the backward's fwd.flags, dq, dk, dv
 * (rla_bwd / rdn_bwd; dO stays in fwd.dtype).  Every accumulation is fp32 in
 * either case; the flag only skips the final rounding to bf16, so a caller
 * can compare the computation itself against a reference without the bf16
 * storage rounding of the results (half a bf16 ulp, 2^-9 relative).
 * Supported where the tensor-core kernels run (RDN_BF16, Dk = Dv = 128)
 * and, as a no-op, for RDN_F32; otherwise RDN_ERR_UNSUPPORTED. */
#define RDN_FLAG_F32_OUT 0x40u

/* RDN_FLAG_QK_NORM (rla_fwd / rdn_fwd, rdn_decode_step, and in the
 * backward's fwd.flags): q and k are the raw projections x, and the library
 * applies the activation and normalisation of rdn_qk_prologue to them itself,
 * per row of Dk elements
 *     y = SiLU(x) / max(||SiLU(x)||_2, qk_eps),
 * before the recurrence, holding y in `dtype` (as a caller's own prologue
 * pass would); the backward returns dq and dk with respect to x (the map's
 * transposed Jacobian applied to the gradients w.r.t. y).  On the tensor-core
 * path (RDN_BF16, Dk = Dv = 128) the forward's per-chunk pass normalises the
 * rows as it loads them and keeps y in the workspace for the scan and the
 * backward; elsewhere the prologue kernel writes y first.  The backward keeps
 * the gradients w.r.t. y in fp32 (for bf16 inputs) and applies the Jacobian
 * in one streaming pass.  Needs qk_eps > 0 and finite (else
 * RDN_ERR_INVALID_ARG); *_fwd_workspace_size and *_bwd_workspace_size grow by
 * the normalised copies (2 B T H Dk elements of dtype) and the fp32 gradients
 * (2 B T H Dk floats, bf16 inputs). */
#define RDN_FLAG_QK_NORM 0x80u

/* Arguments of rla_fwd / rdn_fwd.
 *   B, T, H           batch, tokens, heads; B, H >= 1, T >= 0 (T = 0 copies
 *                     S0/R0 to ST/RT).
 *   Dk, Dv            head dimensions.  RDN_BF16 supports Dk = Dv = 128 and
 *                     Dk = Dv = 64; RDN_F32 supports Dk, Dv in {64, 128}.
 *   dtype             element type of q, k, v and o.  Gates and states are
 *                     always fp32 and every accumulation is fp32.
 *   q, k, v           inputs (q, k expected L2-normalised; not checked).
 *   g, beta, gamma    per-token, per-head log-decay g = log(alpha) and rates.
 *   clip              the threshold c of Section 3.3; INFINITY = no clip;
 *                     c < 0 or NaN -> RDN_ERR_INVALID_ARG.
 *   S0, R0            initial states or NULL (= zero).
 *   o                 output [B,T,H,Dv] in `dtype` (fp32 with RDN_FLAG_F32_OUT).
 *   ST, RT            final states or NULL (= not returned).
 *   S_chunks,R_chunks optional chunk-start states (outputs; NULL = not
 *                     stored).  rdn_bwd can consume them instead of
 *                     recomputing.
 *   scale             multiplies q (the paper uses 1).
 *   flags             0, or RDN_FLAG_SAVE_FOR_BWD and / or
 *                     RDN_FLAG_TIED_GAMMA, the variant flags,
 *                     RDN_FLAG_F32_OUT, RDN_FLAG_QK_NORM (above).
 *   qk_eps            (last field) norm floor for RDN_FLAG_QK_NORM.
 *   workspace         device scratch of *_fwd_workspace_size() bytes.
 *   cu_seqlens        NULL, or packed variable-length sequences: a device
 *                     int32 array of num_seqs + 1 token offsets, 0 =
 *                     cu_seqlens[0] <= cu_seqlens[1] <= ... <=
 *                     cu_seqlens[num_seqs] = T.  Then B must be 1 and
 *                     sequence s is tokens cu_seqlens[s] .. cu_seqlens[s+1]-1
 *                     of the [1,T,H,.] inputs, each with its own recurrence
 *                     (states restart at S0[s], R0[s]; empty sequences are
 *                     allowed).  S0, R0, ST, RT (and the backward's dST,
 *                     dRT, dS0, dR0) are [num_seqs,H,Dk,Dv]; S_chunks and
 *                     R_chunks hold rdn_chunk_slots() blocks of Dk x Dv fp32,
 *                     block (first chunk of s) * H + h * nc_s + c for chunk c
 *                     of sequence s, head h (nc_s = ceil(len_s / 64)).  The
 *                     table is read on the device only: a table that breaks
 *                     the ordering above is clamped into it (no fault, the
 *                     result is unspecified).  Sequences are independent,
 *                     exactly as B separate calls would run them.
 *   num_seqs          number of packed sequences (>= 1) when cu_seqlens is
 *                     set; ignored otherwise.                             */
typedef struct {
  int B, T, H, Dk, Dv;
  int dtype; /* rdn_dtype_t */
  const void *q, *k, *v;
  const float *g, *beta, *gamma;
  float clip;
  const float *S0, *R0;
  void *o;
  float *ST, *RT;
  float *S_chunks, *R_chunks;
  float scale;
  unsigned flags;
  void *workspace;
  size_t workspace_bytes;
  const int *cu_seqlens;
  int num_seqs;
  float qk_eps; /* the norm floor of RDN_FLAG_QK_NORM; ignored without it */
} rdn_fwd_args;

/* Arguments of rdn_bwd.  `fwd` holds the forward's inputs (its o, ST, RT,
 * S_chunks and R_chunks outputs are ignored except as noted).
 *   fwd.S_chunks/R_chunks  if both non-NULL they are READ as the forward's
 *                     chunk-start states (as written by rdn_fwd on the same
 *                     inputs); if NULL the backward recomputes them into its
 *                     workspace.
 *   fwd.workspace     NULL, or (only together with S_chunks/R_chunks) the
 *                     workspace of the rdn_fwd call that wrote them, READ
 *                     as that forward left it: its per-chunk matrices
 *                     (the chunk form's T, A and M blocks) are reused instead of
 *                     recomputed.  fwd.workspace_bytes must be at least
 *                     rdn_fwd_workspace_size(&fwd); the same q, k, g, beta,
 *                     gamma, scale and clip as in that call are the caller's
 *                     responsibility (not checked).  It is only read.
 *   fwd.flags         RDN_FLAG_SAVE_FOR_BWD if that forward ran with it
 *                     (then fwd.workspace is required), and
 *                     RDN_FLAG_TIED_GAMMA for tied gates, the variant
 *                     flags, RDN_FLAG_F32_OUT and RDN_FLAG_QK_NORM (with
 *                     fwd.qk_eps) as the forward had them; else 0.
 *   dO                upstream gradient of o, [B,T,H,Dv] in fwd.dtype.
 *   dST, dRT          upstream gradients of ST, RT, or NULL (= 0).
 *   dq, dk            [B,T,H,Dk] in fwd.dtype;  dv [B,T,H,Dv] in fwd.dtype
 *                     (all three fp32 with RDN_FLAG_F32_OUT in fwd.flags).
 *   dg, dbeta, dgamma [B,T,H] fp32.  dg is the gradient w.r.t. the
 *                     log-decay g; the gradient w.r.t. alpha is dg / alpha.
 *   dS0, dR0          [B,H,Dk,Dv] fp32, or NULL (= not returned).
 * At |v - S_{t-1}k| == c the clip passes the gradient (inclusive mask).    */
typedef struct {
  rdn_fwd_args fwd;
  const void *dO;
  const float *dST, *dRT;
  void *dq, *dk, *dv;
  float *dg, *dbeta, *dgamma;
  float *dS0, *dR0;
  void *workspace;
  size_t workspace_bytes;
} rdn_bwd_args;

/* Arguments of rdn_decode_step: one token for N independent sequences.
 *   N, H, Dk, Dv      Dk = Dv = 128 or 64.
 *   dtype             element type of q, k, v, o (RDN_BF16 or RDN_F32).
 *   q, k [N,H,Dk]; v, o [N,H,Dv]; g, beta, gamma [N,H] fp32.
 *   S, R [N,H,Dk,Dv] fp32, read and updated IN PLACE (must not alias any
 *   other argument).
 *   variant           0 = RLA, 1 = RDN.
 *   flags             0, or RDN_FLAG_TIED_GAMMA (gamma ignored, beta serves
 *                     as both rates), the variant flags and / or
 *                     RDN_FLAG_QK_NORM (q, k raw x, normalised in the step
 *                     with qk_eps and held in dtype, as the forward does):
 *                     the same token step as the forward with those flags. */
typedef struct {
  int N, H, Dk, Dv;
  int dtype;
  int variant;
  const void *q, *k, *v;
  const float *g, *beta, *gamma;
  float clip;
  float scale;
  float *S, *R;
  void *o;
  unsigned flags;
  float qk_eps; /* the norm floor of RDN_FLAG_QK_NORM; ignored without it */
} rdn_decode_args;

/* Arguments of rdn_qk_prologue / rdn_qk_prologue_bwd: the activation and
 * normalisation the model applies to queries and keys before the recurrence
 * (Section 3.4 leaves them out of its equations): per row of D elements
 *     u = SiLU(x) = x * sigmoid(x),   y = u / max(||u||_2, eps).
 *   rows              number of rows of each tensor (B*T*H for q or k), >= 1.
 *   D                 row length, 64 or 128.
 *   dtype             RDN_BF16 or RDN_F32 for every tensor below.
 *   eps               norm floor, > 0 and finite (1e-12 matches common
 *                     normalisation defaults).
 *   x[i]              pre-activation rows [rows][D] (q in x[0], k in x[1];
 *                     x[1] may be NULL for one tensor).  Read only.
 *   y[i]              (prologue) outputs [rows][D], may not alias x.
 *   dy[i], dx[i]      (backward) upstream gradients of y and the gradients
 *                     w.r.t. x [rows][D]; the backward recomputes y from x.
 * Every pointer is a caller-owned 16-byte aligned device pointer; unused
 * fields are ignored.  Errors: RDN_ERR_INVALID_ARG (rows < 1, eps, NULL
 * pointers), RDN_ERR_UNSUPPORTED (D, dtype), RDN_ERR_MISALIGNED. */
typedef struct {
  long long rows;
  int D;
  int dtype; /* rdn_dtype_t */
  float eps;
  const void *x[2];
  void *y[2];
  const void *dy[2];
  void *dx[2];
} rdn_prologue_args;

/* y = SiLU(x) / max(||SiLU(x)||, eps) row-wise for one or two tensors. */
rdn_status_t rdn_qk_prologue(const rdn_prologue_args *args, rdn_stream_t stream);
/* dx = d<dy, y>/dx of the same map. */
rdn_status_t rdn_qk_prologue_bwd(const rdn_prologue_args *args, rdn_stream_t stream);

/* RLA forward, Section 3.4 (left formulation).  Chunkwise-parallel form:
 * additive base state, no triangular solves. */
rdn_status_t rla_fwd(const rdn_fwd_args *args, rdn_stream_t stream);

/* RDN forward, Section 3.4 (right formulation).  Gated delta rule on S and
 * on R, chunkwise (64 tokens) with the UT/WY triangular form of the delta
 * rule; the clipped residual is formed and consumed on chip. */
rdn_status_t rdn_fwd(const rdn_fwd_args *args, rdn_stream_t stream);

/* RDN forward for callers that cannot allocate device memory.  The paper has
 * no counterpart; this is a deployment convenience.  Some callers own only
 * their input and output buffers: an inference-engine plugin that is handed
 * fixed tensors, or a serving loop that forbids device allocation after
 * start-up (cudaMalloc can synchronise the device and can fail under
 * fragmentation).  This entry point computes exactly what rdn_fwd computes,
 * from the same arguments, but its scratch is a fixed array compiled into the
 * library (RDN_NOALLOC_SCRATCH_BYTES, held on every GPU that loads the
 * library until the process exits) instead of args->workspace, which is
 * ignored.  It allocates nothing.
 *   - RDN_FLAG_SAVE_FOR_BWD is rejected (RDN_ERR_UNSUPPORTED): what it saves
 *     would stay in the built-in scratch, out of rdn_bwd's reach.
 *   - Size limit: the scratch holds one 83,456-byte record per 64-token
 *     chunk, so B * H * ceil(T/64) must be at most 804; larger problems
 *     return RDN_ERR_WORKSPACE (with a message giving both sizes) and
 *     nothing is launched.  Use rdn_fwd with a caller workspace for them.
 *   - First call on each device: it looks up the scratch array's device
 *     address (cudaGetSymbolAddress) with that device current, once, and
 *     caches it.  Make that first call before any stream capture.
 *   - All calls share the one array, and each call overwrites every scratch
 *     word it reads before reading it, so nothing needs clearing between
 *     calls.  Calls whose work overlaps on the GPU (different streams, or
 *     different host threads without ordering) race on the array: order
 *     them, e.g. issue them on one stream. */
#define RDN_NOALLOC_SCRATCH_BYTES (64u * 1024u * 1024u)
rdn_status_t rdn_fwd_noalloc(const rdn_fwd_args *args, rdn_stream_t stream);

/* Backward of rdn_fwd (reverse-mode of the same chunkwise computation).
 * Supports RDN_BF16 with Dk = Dv in {64, 128} and RDN_F32 likewise. */
rdn_status_t rdn_bwd(const rdn_bwd_args *args, rdn_stream_t stream);

/* Backward of rla_fwd, Section 3.4 (left formulation): the same arguments,
 * layouts, ownership and errors as rdn_bwd, for the RLA recurrence.
 * fwd.workspace / fwd.S_chunks / fwd.flags refer to an rla_fwd call. */
rdn_status_t rla_bwd(const rdn_bwd_args *args, rdn_stream_t stream);

/* One recurrent step (Section 3.4 recurrence at a single t), states in
 * place; memory-bound: reads and writes S and R once. */
rdn_status_t rdn_decode_step(const rdn_decode_args *args, rdn_stream_t stream);

/* Workspace sizes in bytes for the arguments' shapes (pointers ignored).
 * Return RDN_OK and set *bytes, or an error for invalid shapes. */
rdn_status_t rla_fwd_workspace_size(const rdn_fwd_args *args, size_t *bytes);
/* Device-side failures.  A kernel whose bounded wait for its own copies or
 * tensor-core work gives up (RDN_ERR_TIMEOUT), or that finds its shared
 * memory misaligned (RDN_ERR_CUDA), records the code in a per-device status
 * word, skips the rest of its work and exits, leaving the context usable;
 * the outputs of that call are then invalid.  rdn_device_status waits for
 * `stream`, returns in *status the code recorded since the previous query
 * (RDN_OK if none) and clears it.  The word is shared by all streams of the
 * device.
 * Device state held by the library: the status word and the built-in
 * scratch of rdn_fwd_noalloc are device variables whose addresses the
 * library looks up once per device and keeps for the life of the process.
 * cudaDeviceReset on a device invalidates them: after a reset, do not call
 * the library on that device again in the same process.
 * Test instrumentation: with the environment variable RDN_FAULT_INJECT set
 * to "workspace" or "launch", the forward and backward entry points fail
 * with RDN_ERR_WORKSPACE or RDN_ERR_CUDA after validating their arguments,
 * before enqueueing anything; with "device_wait" the tensor-core forward
 * scan (bf16, Dk = 128), and with "device_wait_bwd" the tensor-core
 * backward chain, makes its first bounded wait give up, records
 * RDN_ERR_TIMEOUT here and drains its work in flight. */
rdn_status_t rdn_device_status(rdn_stream_t stream, int *status);

/* Number of Dk x Dv blocks in each of S_chunks and R_chunks:
 * B * H * ceil(T/64), or with cu_seqlens the bound H * (num_seqs +
 * ceil(T/64)) (slots past the sequences' chunks are left untouched). */
rdn_status_t rdn_chunk_slots(const rdn_fwd_args *args, long long *slots);
rdn_status_t rdn_fwd_workspace_size(const rdn_fwd_args *args, size_t *bytes);
rdn_status_t rla_bwd_workspace_size(const rdn_bwd_args *args, size_t *bytes);
rdn_status_t rdn_bwd_workspace_size(const rdn_bwd_args *args, size_t *bytes);

/* Message describing the last non-OK status returned on this thread
 * ("" if none).  The pointer stays valid until the next call on the
 * thread. */
const char *rdn_last_error(void);

/* Library version string. */
const char *rdn_version(void);

/* Instrumentation (no counterpart in the paper): device time of each launch
 * of the library's own kernels, measured with CUDA events recorded on the
 * stream each kernel is launched on.
 *   rdn_prof_start(capacity)  begins recording the next `capacity` launches
 *                             (any thread, any stream); fails if already
 *                             recording.  Launches beyond capacity are
 *                             counted but not timed.
 *   rdn_prof_stop(out, cap, n) waits for the recorded launches to finish,
 *                             writes up to `cap` records to `out` (may be
 *                             NULL), sets *n to the number of launches seen
 *                             (timed or not) and ends the recording. */
typedef struct {
  char name[40];
  float ms;
} rdn_prof_record;
rdn_status_t rdn_prof_start(int capacity);
rdn_status_t rdn_prof_stop(rdn_prof_record *out, int cap, int *n);

#ifdef __cplusplus
}
#endif

#endif /* RDN_H_ */
