// kdn_internal.cuh -- internal types and device helpers shared by the CUDA
// translation units of libkdn.so.  Not part of the public ABI (include/kdn.h).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kdn.h"

namespace kdn {

// ---------------------------------------------------------------------------
// dtype helpers: activations are float32 or bfloat16, arithmetic is float32.

template <typename DT> __device__ __forceinline__ float ld(const void *p, size_t i);
template <> __device__ __forceinline__ float ld<float>(const void *p, size_t i) {
  return static_cast<const float *>(p)[i];
}
template <> __device__ __forceinline__ float ld<__nv_bfloat16>(const void *p, size_t i) {
  return __bfloat162float(static_cast<const __nv_bfloat16 *>(p)[i]);
}
template <typename DT> __device__ __forceinline__ void st(void *p, size_t i, float x);
template <> __device__ __forceinline__ void st<float>(void *p, size_t i, float x) {
  static_cast<float *>(p)[i] = x;
}
template <> __device__ __forceinline__ void st<__nv_bfloat16>(void *p, size_t i, float x) {
  static_cast<__nv_bfloat16 *>(p)[i] = __float2bfloat16_rn(x);
}

// Output store in the caller's output dtype (a uniform runtime choice).
__device__ __forceinline__ void sto(int odt, void *p, size_t i, float x) {
  if (odt == KDN_BF16) static_cast<__nv_bfloat16 *>(p)[i] = __float2bfloat16_rn(x);
  else static_cast<float *>(p)[i] = x;
}

// Gate activations of the layer's parameterisation for KDN_GATES_LOGITS
// inputs: alpha = sigmoid(x), omega = softplus(y), r = r_min + softplus(z).
// softplus(x) = max(x, 0) + log1p(u), u = exp(-|x|) in (0, 1], with log1p(u) taken
// as the fast logarithm of 1 + u: no branch inside the unrolled per-token loops.
// For u below ~1e-4 the rounding of 1 + u costs relative precision in the small
// term log1p(u) ~ u, never more than 6e-8 in absolute terms.
__device__ __forceinline__ float softplus_f(float x) {
  const float u = __expf(-fabsf(x));
  return fmaxf(x, 0.f) + __logf(1.f + u);
}
__device__ __forceinline__ float sigmoid_f(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }
// log alpha from the gate input: g itself, or log sigmoid(x) = -softplus(-x)
__device__ __forceinline__ float gate_logalpha(int gates, float g) {
  return gates ? -softplus_f(-g) : g;
}
__device__ __forceinline__ float gate_omega(int gates, float w) {
  return gates ? softplus_f(w) : w;
}
__device__ __forceinline__ float gate_r(int gates, float rmin, float r) {
  return gates ? rmin + softplus_f(r) : r;
}
// Chain-rule factors from the post-activation gates back to the logits:
// d log(alpha) / dx = 1 - alpha, d omega / dy = sigmoid(y), d r / dz = sigmoid(z).
__device__ __forceinline__ float dgate_logalpha(int gates, float alpha) {
  return gates ? 1.f - alpha : 1.f;
}
__device__ __forceinline__ float dgate_sig(int gates, float y) { return gates ? sigmoid_f(y) : 1.f; }

// A 2x2 Moebius matrix (homogeneous coordinates of the uncertainty) divided by
// its largest entry: the ratio it represents is unchanged, and long products stay
// in range.
__device__ __forceinline__ void renorm4(float &m00, float &m01, float &m10, float &m11) {
  const float s = fmaxf(fmaxf(fabsf(m00), fabsf(m01)), fmaxf(fabsf(m10), fabsf(m11)));
  const float inv = __fdividef(1.f, s);
  m00 *= inv; m01 *= inv; m10 *= inv; m11 *= inv;
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// ---------------------------------------------------------------------------
// Internal argument bundle: everything an entry point received, plus derived
// sizes and the carve-up of the caller's workspace.

struct Args {
  int variant;  // 0 diagonal, 1 isotropic
  int B, T, H, dk, dv;
  int C;        // memory chunk length used by the kernels
  int NC, Tp;   // number of chunks, padded length NC*C
  int P;        // uncertainty entries per head: dk (diag) or 1 (iso)
  int pcd;      // decay has a channel axis (g is [..,dk])
  int dtype;
  int odt;      // dtype of o and of the input gradients
  int chunk;    // chunk length requested in the descriptor (0, 32 or 64)
  int gates;    // kdn_gates_t: post-activation gates or their logits
  float rmin;   // observation-noise floor of the logit parameterisation
  float mu, tau;
  // forward inputs / outputs
  const void *q, *k, *v, *g, *omega, *r;
  const float *S0, *p0;
  void *o;
  float *ST, *pT;
  // backward inputs / outputs
  const void *dO;
  const float *dST, *dpT;
  void *dq, *dk_, *dv_, *dg, *domega, *dr;
  float *dS0, *dp0;
  float *dmu;  // [B,H] gradient with respect to mu (nullable)
  // workspace regions (float32 unless noted)
  unsigned *status;
  float *phat;    // [BH][Tp][P]   predictive variance phat_t (pre-write)
  float *isotok;  // [BH][Tp][2]   isotropic: a_t, |k_t|^2
  float *W, *U;   // [BH][NC][C][dk], [BH][NC][C][dv]
  float *Qb;      // [BH][NC][C][dk]
  float *Aqk;     // [BH][NC][C][C]
  float *Kt;      // [BH][NC][C][dk]
  float *gC;      // [BH][NC][dk]   gamma_C
  float *Sin;     // [BH][NC][dk][dv] chunk-entry memory (backward)
  float *dSout;   // [BH][NC][dk][dv] cotangent of the chunk-exit memory
  float *dR;      // [BH][NC][C][dv]
  float *dkpart;  // [BH][Tp][dk]
  float *dgpart;  // [BH][Tp][dk]
  float *dphloc;  // [BH][Tp][P]
  float *drpart;  // [BH][Tp]
  float *drw;     // [BH][Tp][4]
  float *isoadj;  // [BH][Tp][2]
  unsigned char *fSin;  // fused backward: [BH][NC] context records (S_in, R, -W, A_qk, A)
  float *fpin;          // fused backward: [BH][NC][dk] uncertainty entering each chunk
};

__host__ __device__ inline size_t tok_index(const Args &a, int b, int t, int h) {
  return ((size_t)b * a.T + t) * a.H + h;
}

// Workspace carve-up; returns total bytes.  `bwd` adds the backward regions.
// A forward that runs the fused kernel only needs the status word.
size_t workspace_layout(Args *a, char *base, bool bwd);

// Fused tcgen05 forward (bf16, dk = dv = 128, 64-token chunks).  With
// `save_S` / `save_p` it also stores the context of the fused backward: the
// fp16 image of every chunk's entry memory (32 KB) and the uncertainty entering
// every chunk (128 floats); `write_o` = false skips the outputs o.
// `phi_T` ([B*H][128][128]) selects the transition pass: besides the memory from
// a.S0 with v (to a.ST, its output to a.o, float32), every sequence also carries
// the memory the recurrence reaches from S = I with v = 0, written to phi_T, and
// its output tau Phi_t^T q_t to `o_phi` (fp16, the layout of o); no context then.
bool fused_fwd_supported(const Args &a);
kdn_status_t launch_fused_fwd(const Args &a, cudaStream_t s, unsigned char *save_S = nullptr,
                              float *save_p = nullptr, bool write_o = true, float *phi_T = nullptr,
                              void *o_phi = nullptr);
// Chunked forward of the Diagonal KDN in compact-WY form with tf32 intra-chunk
// products (kdn_wy_fwd.cu): bf16 activations, post-activation gates, dk = dv =
// 128, 64-token chunks; writes o, S_T, p_T where their pointers are non-null,
// and with save_S / save_p the fused backward's context (the layout of
// launch_fused_fwd's saving mode).
bool wy_fwd_supported(const Args &a, bool save);  // save: the context-saving instantiation
kdn_status_t launch_wy_fwd(const Args &a, cudaStream_t s, unsigned char *save_S = nullptr,
                           float *save_p = nullptr);
// beta_eff [B,T,H] (float32) from the per-token gain scalars of a context saved by
// the fused training forward (one launch).
kdn_status_t launch_beta_eff(const Args &a, const void *saved, float *out, cudaStream_t s);
// One bounded wait that runs out (the self-test of kdn_selftest_wait_timeout).
kdn_status_t launch_wait_selftest(unsigned *status, cudaStream_t s);
// Fused tcgen05 backward (Diagonal KDN, bf16, dk = dv = 128, 64-token chunks):
// one reverse sweep per (batch, head) from the saved context in a.fSin / a.fpin.
// launch_fused_bwd first runs the context-saving forward (without o).
bool fused_bwd_supported(const Args &a);
kdn_status_t launch_fused_bwd(const Args &a, cudaStream_t s);
kdn_status_t launch_fused_bwd_sweep(const Args &a, cudaStream_t s);
// Bytes of the saved context for the fused backward (0 if not served): per
// (batch, head) and 64-token chunk one record of fused_ctx_record_bytes(), then
// per chunk the 128 float32 uncertainties entering it.
size_t fused_saved_bytes(const Args &a);
size_t fused_ctx_record_bytes();

// Sequence-parallel forward (kdn_segmented.cu): the number of segments P each
// sequence is cut into (1: not used), the workspace it needs after the common
// layout, and the launcher (gain summaries, scan, one fused run per segment
// carrying memory and transition, the state join, and the output pass).
int seg_count(const Args &a);
// Smallest forward workspace for a descriptor (the single-pass layout; 0 for an
// invalid descriptor); kdn_fwd_workspace_bytes adds the segment buffers.
size_t fwd_min_workspace_bytes(const kdn_desc_t *desc, int variant);
size_t seg_workspace_bytes(const Args &a, int P);
kdn_status_t launch_seg_fwd(const Args &a, int P, char *ws, cudaStream_t s);

// Launchers (each returns KDN_OK or KDN_ERR_CUDA).
kdn_status_t launch_chunked_fwd(const Args &a, cudaStream_t s, bool save_states);
kdn_status_t launch_chunked_bwd(const Args &a, cudaStream_t s);
kdn_status_t launch_decode(const Args &a, float *S, float *p, cudaStream_t s);

// Kernels launched by launch_chunked_fwd / launch_chunked_bwd for these sizes.
int chunked_fwd_launches(const Args &a);
int chunked_bwd_launches(const Args &a);

}  // namespace kdn
