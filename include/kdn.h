/*
 * kdn.h -- C ABI of the GB300 (sm_103a) Kalman Delta Network token-mixer
 * library (libkdn.so).
 *
 * Operations (all from "Kalman Delta Networks"):
 *   kdn_diag_fwd / kdn_iso_fwd
 *       Chunked prefill / training forward of the Diagonal KDN (Prop. 3) and
 *       the Isotropic KDN (Prop. 5; App. E): the Moebius uncertainty scan
 *       (eq. kla-box-mobius, eq. iso-kla-box-mobius), the Kalman gain emitted
 *       from the pre-write predictive variance (eq. kla-box-gain,
 *       eq. iso-kla-box-gain, App. F.1 eq. chunk-gain-emission) and the
 *       asymmetric delta-rule memory scan in compact-WY form (App. F.2,
 *       eq. chunk-memory-wy and eq. chunk-memory-output-state).
 *   kdn_diag_bwd / kdn_iso_bwd
 *       Gradients of the forward.  The paper gives no backward; these are
 *       the exact adjoints of the forward recurrence.
 *   kdn_diag_decode_step / kdn_iso_decode_step
 *       One token of the recurrence (the boxed update of Prop. 3 / Prop. 5)
 *       applied in place to a batch of states.
 *
 * Per token t and head h the layer computes, with alpha_t = exp(g_t):
 *   Diagonal:  phat = alpha^2 p + omega;  kappa = phat k / (r + sum phat k^2)
 *              u = mu k^2 / r;            p' = phat / (1 + u phat)
 *   Isotropic: a = mean_i alpha_i^2 (alpha^2 for scalar decay);
 *              bhat = a b + omega;  beta = bhat / (r + bhat |k|^2); kappa = beta k
 *              u = mu |k|^2 / (d_k r); b' = bhat / (1 + u bhat)
 *   Memory:    S' = (I - kappa k^T) diag(alpha) S + kappa v^T;  o = scale * S'^T q
 *
 * Conventions
 *   Ownership  The caller owns every buffer, device and host.  Entry points
 *              allocate no memory (scratch lives in the caller's workspace),
 *              keep no global state between calls and are reentrant.
 *   Pointers   Device pointers unless stated otherwise, 16-byte aligned.
 *   Streams    `stream` is a cudaStream_t passed as void* (NULL = the legacy
 *              default stream).  Every call is asynchronous on that stream.
 *   Errors     Argument errors are detected before anything is launched and
 *              leave all outputs untouched.  A failed launch returns
 *              KDN_ERR_CUDA.
 *   Inputs     q, k, v, g, omega, r are post-activation values: g = log(alpha)
 *              <= 0 (alpha = sigmoid(.) in the paper), omega > 0, r > 0.  The
 *              library does not normalise q or k and applies no gate
 *              activation.
 *   Layouts    (row-major, last index fastest)
 *              q, k            [B, T, H, dk]        v, o, dO      [B, T, H, dv]
 *              r               [B, T, H]
 *              diag: g, omega  [B, T, H, dk]
 *              iso:  omega     [B, T, H];  g [B, T, H, dk] (decay_per_channel=1)
 *                                           or [B, T, H]     (decay_per_channel=0)
 *              S0, ST, dST, dS0 (float32)   [B, H, dk, dv]
 *              p0, pT, dpT, dp0 (float32)   diag [B, H, dk];  iso [B, H]
 *              Gradients have the layout of the input they belong to.
 *   Dtypes     q, k, v, g, omega, r and dO have desc->dtype (float32 or
 *              bfloat16); o and the input gradients have desc->out_dtype.
 *              State is always float32.  Accumulation is float32; the
 *              bf16 d = 128 forward runs its intra-chunk products on the
 *              tensor cores with tf32 and fp16 operands (Sec. 4.2 products,
 *              float32 accumulators).
 *   Sizes      dk, dv in {32, 64, 128}; T >= 0 (any length; a ragged last
 *              chunk is padded with identity tokens); B, H >= 0.  At most
 *              T = 2^21 tokens, B*H = 65535*1024 sequences and B*T*H =
 *              2^31 - 1 token-heads per call; larger problems return
 *              KDN_ERR_UNSUPPORTED (split them over calls).
 */
#ifndef KDN_H
#define KDN_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KDN_OK = 0,
  KDN_ERR_INVALID_ARG = 1, /* null / misaligned pointer, bad size or field */
  KDN_ERR_UNSUPPORTED = 2, /* valid but not built (e.g. dk = 96) */
  KDN_ERR_WORKSPACE = 3,   /* workspace missing or smaller than required */
  KDN_ERR_CUDA = 4,        /* a CUDA launch or runtime call failed */
  KDN_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
  KDN_ERR_RANGE = 6        /* device status only: a 64-token chunk's cumulative log-decay
                              G_C left a fused kernel's range in some channel (results of
                              that call are invalid).  The single-pass bf16 d = 128
                              diagonal forward (kdn_diag_fwd) takes any decay.  The calls
                              that write or read the backward context (the *_fwd_save /
                              *_bwd_saved pairs, the fused backwards), the isotropic fused
                              forward and the sequence-parallel forward take
                              exp(G_C) >= 1e-36, G_C >= -82.8.  desc->chunk = 32 halves
                              the exposure. */
} kdn_status_t;

typedef enum { KDN_F32 = 0, KDN_BF16 = 1 } kdn_dtype_t;

typedef struct {
  int B, T, H;           /* batch, tokens, heads */
  int dk, dv;            /* key and value head dimensions */
  int chunk;             /* memory-chunk length C_m of App. F.2: 0 (= 64), 32 or 64;
                            a tuning choice, results agree to rounding */
  int dtype;             /* kdn_dtype_t of q, k, v, g, omega, r and dO (the
                            stored dtype of o and the gradients is out_dtype) */
  float mu;              /* information scale of eq. diag-cov-update; <= 0 -> dk */
  float scale;           /* query scale tau of App. F.2; NaN -> 1/sqrt(dk) */
  int decay_per_channel; /* isotropic only: 1 -> g is [B,T,H,dk], 0 -> [B,T,H].
                            Ignored by the diagonal variant (always per channel). */
  int out_dtype;         /* kdn_dtype_t of o and of dq, dk, dv, dg, domega, dr.
                            0 (KDN_F32, the zero-initialised default) keeps the
                            float32 accumulators; KDN_BF16 rounds them once on
                            store. */
  int gates;             /* kdn_gates_t: what g, omega and r hold (below) */
  float r_min;           /* observation-noise floor of KDN_GATES_LOGITS (>= 0) */
} kdn_desc_t;

/* The gate inputs.  KDN_GATES_POST (0, the zero-initialised default): g = log
   alpha <= 0, omega > 0 and r > 0 as the recurrence uses them.  KDN_GATES_LOGITS:
   g, omega and r are the pre-activation values x, y, z of the layer's
   parameterisation (eq. kla-box-parameterization; r_min of Sec. 5):
   alpha = sigmoid(x), omega = softplus(y), r = r_min + softplus(z), applied
   in float32 inside the kernels.  The backward then returns the gradients with
   respect to x, y and z (in dg, domega, dr). */
typedef enum { KDN_GATES_POST = 0, KDN_GATES_LOGITS = 1 } kdn_gates_t;

/* Library version as major*10000 + minor*100 + patch. */
int kdn_version(void);

/* Human-readable name of a status code (static string, never NULL). */
const char *kdn_status_string(kdn_status_t status);

/* Workspace (device scratch) bytes that kdn_*_fwd / kdn_*_bwd need for this
   descriptor; variant 0 = diagonal, 1 = isotropic.  Returns 0 for an invalid
   descriptor.  The workspace must be 256-byte aligned; its contents need no
   initialisation and are clobbered by every call.
   For bf16 inputs with d_k = d_v = 128 and few long sequences (B*H*P <= 152
   for some P >= 4 that divides the T/64 chunks into segments of >= 8 chunks,
   T a multiple of 64) the forward runs sequence-parallel: it cuts each
   sequence into P segments, joined exactly (uncertainty by a scan of per-chunk
   Moebius summaries, memory by the linearity of the chunk recurrence in
   (S_in, v)), and kdn_fwd_workspace_bytes includes its segment buffers
   (160 KB per (batch, head, segment), 2 KB per (batch, head, chunk), and
   2 bytes per element of o, 6 when out_dtype is KDN_BF16).
   A smaller workspace that still holds the single-pass layout (256 bytes)
   runs the single pass. */
size_t kdn_fwd_workspace_bytes(const kdn_desc_t *desc, int variant);
size_t kdn_bwd_workspace_bytes(const kdn_desc_t *desc, int variant);

/* Forward over T tokens (Prop. 3, App. F).
   S0 NULL -> zero initial memory; p0 NULL -> unit initial uncertainty
   (z_0 = [p_0, 1] of eq. chunk-gain-carry with p_0 = 1).
   ST / pT NULL -> final state not written.  o is always written. */
kdn_status_t kdn_diag_fwd(const kdn_desc_t *desc, const void *q, const void *k,
                          const void *v, const void *g, const void *omega,
                          const void *r, const float *S0, const float *p0,
                          void *o, float *ST, float *pT, void *workspace,
                          size_t workspace_bytes, void *stream);

/* Forward of the Isotropic KDN (Prop. 5, App. E); p0 / pT are b_0 / b_T [B,H]. */
kdn_status_t kdn_iso_fwd(const kdn_desc_t *desc, const void *q, const void *k,
                         const void *v, const void *g, const void *omega,
                         const void *r, const float *S0, const float *p0,
                         void *o, float *ST, float *pT, void *workspace,
                         size_t workspace_bytes, void *stream);

/* Backward: gradients of <dO, o> + <dST, ST> + <dpT, pT> with respect to every
   forward input.  It recomputes the forward from the inputs (no saved
   context).  dST / dpT NULL -> zero cotangent.  dS0 / dp0 / dmu NULL -> not
   written; all other gradient pointers are required.  dmu [B,H] float32: the
   gradient with respect to the information scale mu of each sequence (mu
   enters only through u of eq. diag-cov-update / Prop. 5); a mu shared by all
   sequences has the sum.  The gradient of a learned initial uncertainty
   c_{0,h} (p_0 = c_{0,h} in every channel) is the per-head sum of dp0. */
kdn_status_t kdn_diag_bwd(const kdn_desc_t *desc, const void *q, const void *k,
                          const void *v, const void *g, const void *omega,
                          const void *r, const float *S0, const float *p0,
                          const void *dO, const float *dST, const float *dpT,
                          void *dq, void *dk, void *dv, void *dg, void *domega,
                          void *dr, float *dS0, float *dp0, float *dmu, void *workspace,
                          size_t workspace_bytes, void *stream);

kdn_status_t kdn_iso_bwd(const kdn_desc_t *desc, const void *q, const void *k,
                         const void *v, const void *g, const void *omega,
                         const void *r, const float *S0, const float *p0,
                         const void *dO, const float *dST, const float *dpT,
                         void *dq, void *dk, void *dv, void *dg, void *domega,
                         void *dr, float *dS0, float *dp0, float *dmu, void *workspace,
                         size_t workspace_bytes, void *stream);

/* Training pair.  kdn_diag_fwd_save is kdn_diag_fwd that also keeps, in
   `saved`, the context the chunked backward needs (App. F): for every 64-token
   chunk the memory S entering it, its R = U - W S_in, -W, A_qk,
   A = (I + T)^-1 and (Diagonal KDN) Y = V - Kbar S_in as fp16 tiles (96 KB),
   the pre-write variance phat and the cumulative decay gamma of every
   (token, channel) in float32 (64 KB), per-token scalars (2 KB), and the
   float32 uncertainty p entering it.  kdn_diag_bwd_saved is kdn_diag_bwd that starts from that
   context instead of recomputing the forward (same gradients, one kernel).
   kdn_iso_fwd_save / kdn_iso_bwd_saved are the same for the Isotropic KDN.
   Served for bfloat16 activations, dk = dv = 128 and the default chunk; for
   every other descriptor kdn_saved_bytes() returns 0 and the calls return
   KDN_ERR_UNSUPPORTED (use kdn_*_fwd / kdn_*_bwd).
   saved: caller-owned device buffer of kdn_saved_bytes(desc, variant) bytes, 256-byte
   aligned (a smaller or misaligned one -> KDN_ERR_WORKSPACE).  It is written
   by kdn_diag_fwd_save and read by kdn_diag_bwd_saved, which must see the same
   descriptor and the same q, k, v, g, omega, r (and the forward's S0, p0).
   workspace: kdn_fwd_workspace_bytes(desc, variant) bytes for both calls.  The
   other arguments are those of kdn_*_fwd / kdn_*_bwd. */
size_t kdn_saved_bytes(const kdn_desc_t *desc, int variant);

kdn_status_t kdn_diag_fwd_save(const kdn_desc_t *desc, const void *q,
                               const void *k, const void *v, const void *g,
                               const void *omega, const void *r,
                               const float *S0, const float *p0, void *o,
                               float *ST, float *pT, void *saved,
                               size_t saved_bytes, void *workspace,
                               size_t workspace_bytes, void *stream);

kdn_status_t kdn_diag_bwd_saved(const kdn_desc_t *desc, const void *q,
                                const void *k, const void *v, const void *g,
                                const void *omega, const void *r,
                                const void *saved, size_t saved_bytes,
                                const void *dO, const float *dST,
                                const float *dpT, void *dq, void *dk, void *dv,
                                void *dg, void *domega, void *dr, float *dS0,
                                float *dp0, float *dmu, void *workspace,
                                size_t workspace_bytes, void *stream);

kdn_status_t kdn_iso_fwd_save(const kdn_desc_t *desc, const void *q,
                              const void *k, const void *v, const void *g,
                              const void *omega, const void *r,
                              const float *S0, const float *p0, void *o,
                              float *ST, float *pT, void *saved,
                              size_t saved_bytes, void *workspace,
                              size_t workspace_bytes, void *stream);

kdn_status_t kdn_iso_bwd_saved(const kdn_desc_t *desc, const void *q,
                               const void *k, const void *v, const void *g,
                               const void *omega, const void *r,
                               const void *saved, size_t saved_bytes,
                               const void *dO, const float *dST,
                               const float *dpT, void *dq, void *dk, void *dv,
                               void *dg, void *domega, void *dr, float *dS0,
                               float *dp0, float *dmu, void *workspace,
                               size_t workspace_bytes, void *stream);

/* Effective write strength of every token, beta_eff,t = k_t^T kappa_t (the
   coefficient of the residual identity of eq. appendix-effective-write:
   v_t - S_t^T k_t = (1 - beta_eff,t)(v_t - Shat_t^T k_t); 0 <= beta_eff < 1),
   read from the per-token gain scalars a kdn_*_fwd_save call stored in `saved`
   (same descriptor and variant).  Diagonal: 1 - r_t / s_t with
   s_t = r_t + sum_i phat_i k_i^2; Isotropic: beta_t |k_t|^2.
   r: the r input that call was given (logits when desc->gates says so).
   beta_eff: float32 [B,T,H].  One small kernel, asynchronous on `stream`.
   Returns KDN_ERR_UNSUPPORTED for descriptors kdn_*_fwd_save does not serve,
   KDN_ERR_INVALID_ARG for a null or misaligned pointer, KDN_ERR_WORKSPACE when
   saved_bytes < kdn_saved_bytes(desc, variant). */
kdn_status_t kdn_diag_beta_eff(const kdn_desc_t *desc, const void *saved,
                               size_t saved_bytes, const void *r, float *beta_eff,
                               void *stream);
kdn_status_t kdn_iso_beta_eff(const kdn_desc_t *desc, const void *saved,
                              size_t saved_bytes, const void *r, float *beta_eff,
                              void *stream);

/* One decode token for all B*H heads (the update of Prop. 3), in place:
   S [B,H,dk,dv] and p [B,H,dk] are read and overwritten; o [B,H,dv] is
   written.  Per-step inputs drop the T axis: q, k [B,H,dk], v [B,H,dv],
   g, omega [B,H,dk], r [B,H].  desc->T is ignored.  Needs no workspace. */
kdn_status_t kdn_diag_decode_step(const kdn_desc_t *desc, const void *q,
                                  const void *k, const void *v, const void *g,
                                  const void *omega, const void *r, float *S,
                                  float *p, void *o, void *stream);

/* Isotropic decode step (Prop. 5): p is b [B,H]; omega [B,H];
   g [B,H,dk] or [B,H] per desc->decay_per_channel. */
kdn_status_t kdn_iso_decode_step(const kdn_desc_t *desc, const void *q,
                                 const void *k, const void *v, const void *g,
                                 const void *omega, const void *r, float *S,
                                 float *p, void *o, void *stream);

/* Size of the library-owned scratch array used by kdn_diag_fwd_noalloc. */
#define KDN_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

/* Diagonal-KDN forward that allocates nothing and takes no workspace.  The
   paper has no counterpart: this exists for callers that are handed only
   input and output buffers and may not call cudaMalloc (e.g. a latency-
   critical thread where cudaMalloc can stall on a device synchronisation, or
   a framework that forbids allocation outside its own allocator).  Arguments
   and results are those of kdn_diag_fwd without the workspace pair.
   Scratch is a fixed array of KDN_NOALLOC_SCRATCH_BYTES in the library's
   device memory, held by a GPU from the first use of the library on it (CUDA
   loads the module lazily) until the process exits; a problem whose
   single-pass workspace (kdn_fwd_workspace_bytes without the segment buffers
   of the sequence-parallel forward) exceeds it is rejected with
   KDN_ERR_WORKSPACE before anything runs.  The sequence-parallel forward is
   used when its larger workspace fits the array, else the single pass.  The
   first call on a device looks up the array's device address
   (cudaGetSymbolAddress, with that device current) and caches it with the
   device's CUDA context; a later call under another context (after a device
   reset) looks it up again.  Make the first call before any stream capture.
   All calls on a device share the array, so calls that overlap on the GPU
   race and must be serialised by the caller. */
kdn_status_t kdn_diag_fwd_noalloc(const kdn_desc_t *desc, const void *q,
                                  const void *k, const void *v, const void *g,
                                  const void *omega, const void *r,
                                  const float *S0, const float *p0, void *o,
                                  float *ST, float *pT, void *stream);

/* Device status word of the most recent kdn_diag_fwd_noalloc call on the
   current device (kept in the library's scratch array, which the caller cannot
   address): synchronises `stream`, then returns and clears it, as
   kdn_get_device_status does for a workspace (KDN_OK, KDN_ERR_RANGE or
   KDN_ERR_TIMEOUT).  The paper has no counterpart.  Allocates nothing; the
   first call on a device performs the same address look-up as
   kdn_diag_fwd_noalloc. */
kdn_status_t kdn_noalloc_device_status(void *stream);

/* Number of CUDA kernels one call of an entry point launches for this
   descriptor when T > 0 (op 0 = kdn_*_fwd, 1 = kdn_*_bwd, 2 = kdn_*_decode_step,
   3 = kdn_*_fwd_save, 4 = kdn_*_bwd_saved, 5 = kdn_*_beta_eff; variant 0 = diagonal,
   1 = isotropic).  -1 for an invalid descriptor or op, or an op the descriptor
   does not serve.
   Calls with T = 0 launch at most one small fill kernel. */
int kdn_kernel_launches(const kdn_desc_t *desc, int variant, int op);

/* Synchronises `stream`, then returns and clears the device status word kept
   in the first bytes of `workspace`: KDN_OK; KDN_ERR_RANGE when a fused kernel
   met a chunk whose cumulative decay left its range; or KDN_ERR_TIMEOUT when a bounded
   device-side wait of the most recent kdn_*_fwd / kdn_*_bwd call on that
   workspace gave up.  Each of those calls clears the word before it starts. */
kdn_status_t kdn_get_device_status(void *workspace, void *stream);

/* Self-test of the device-side failure reporting: clears the status word of
   `workspace` (any workspace of at least 256 bytes, 256-byte aligned) and
   launches one small kernel. Thread 0 waits, with the bounded wait every
   kernel of this library uses, on an mbarrier phase that nothing completes.
   After 4096 polls, well under a millisecond, the kernel records
   KDN_ERR_TIMEOUT in the word and returns normally, so the CUDA context stays
   usable.
   kdn_get_device_status(workspace, stream) then returns KDN_ERR_TIMEOUT.
   Returns KDN_ERR_INVALID_ARG for a null or misaligned workspace. */
kdn_status_t kdn_selftest_wait_timeout(void *workspace, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* KDN_H */
