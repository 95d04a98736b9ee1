// kdn_abi.cu -- the extern "C" entry points of libkdn.so (declared in
// include/kdn.h): argument validation, workspace carve-up and dispatch to the
// kernels.  Nothing here allocates memory.
#include <math.h>
#include <stdint.h>

#include "kdn_internal.cuh"

namespace kdn {

int chunked_chunk_len();

namespace {

constexpr size_t kAlign = 256;

size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

bool dim_ok(int d) { return d == 32 || d == 64 || d == 128; }

// Fills the size fields of `a` from the descriptor; returns KDN_OK or an error.
kdn_status_t fill_sizes(const kdn_desc_t *d, int variant, bool decode, Args *a) {
  if (!d) return KDN_ERR_INVALID_ARG;
  if (variant != 0 && variant != 1) return KDN_ERR_INVALID_ARG;
  if (d->B < 0 || d->H < 0 || (!decode && d->T < 0)) return KDN_ERR_INVALID_ARG;
  if (d->dk <= 0 || d->dv <= 0) return KDN_ERR_INVALID_ARG;
  if (!dim_ok(d->dk) || !dim_ok(d->dv)) return KDN_ERR_UNSUPPORTED;
  if (d->chunk != 0 && d->chunk != 32 && d->chunk != 64) return KDN_ERR_INVALID_ARG;
  if (d->dtype != KDN_F32 && d->dtype != KDN_BF16) return KDN_ERR_INVALID_ARG;
  if (d->out_dtype != KDN_F32 && d->out_dtype != KDN_BF16) return KDN_ERR_INVALID_ARG;
  if (variant == 1 && d->decay_per_channel != 0 && d->decay_per_channel != 1)
    return KDN_ERR_INVALID_ARG;
  if (isnan(d->mu) || isinf(d->mu) || isinf(d->scale)) return KDN_ERR_INVALID_ARG;
  if (d->gates != KDN_GATES_POST && d->gates != KDN_GATES_LOGITS) return KDN_ERR_INVALID_ARG;
  if (d->gates == KDN_GATES_LOGITS && !(d->r_min >= 0.f && d->r_min < INFINITY))
    return KDN_ERR_INVALID_ARG;
  const long long BH = (long long)d->B * d->H;
  const int T = decode ? 1 : d->T;
  if (BH > 65535LL * 1024 || T > (1 << 21)) return KDN_ERR_UNSUPPORTED;
  if (BH * (long long)T > (1LL << 31) - 1) return KDN_ERR_UNSUPPORTED;
  *a = Args{};
  a->variant = variant;
  a->B = d->B;
  a->T = T;
  a->H = d->H;
  a->dk = d->dk;
  a->dv = d->dv;
  a->C = chunked_chunk_len();
  a->NC = (T + a->C - 1) / a->C;
  a->Tp = a->NC * a->C;
  a->P = variant == 0 ? d->dk : 1;
  a->pcd = variant == 0 ? 1 : d->decay_per_channel;
  a->dtype = d->dtype;
  a->odt = d->out_dtype;
  a->chunk = d->chunk;
  a->gates = d->gates;
  a->rmin = d->gates == KDN_GATES_LOGITS ? d->r_min : 0.f;
  a->mu = d->mu > 0.f ? d->mu : (float)d->dk;
  a->tau = isnan(d->scale) ? 1.0f / sqrtf((float)d->dk) : d->scale;
  return KDN_OK;
}

// The fused forward serves bf16 activations with dk = dv = 128 and the default
// (or 64-token) chunk; everything else runs the general chunked kernels.
bool use_fused(const Args &a) { return a.chunk != 32 && fused_fwd_supported(a); }
bool use_fused_bwd(const Args &a) { return fused_bwd_supported(a); }

bool ptrs_ok(std::initializer_list<const void *> required,
             std::initializer_list<const void *> optional) {
  for (const void *p : required)
    if (!p || !aligned16(p)) return false;
  for (const void *p : optional)
    if (p && !aligned16(p)) return false;
  return true;
}

__global__ void k_fill(float *p, size_t n, float v) {
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
       e += (size_t)gridDim.x * blockDim.x)
    p[e] = v;
}

// State-only results for T = 0: ST = S0 (or 0), pT = p0 (or 1).
kdn_status_t empty_fwd(const Args &a, cudaStream_t s) {
  const size_t ns = (size_t)a.B * a.H * a.dk * a.dv, np = (size_t)a.B * a.H * a.P;
  if (a.ST) {
    cudaError_t e = a.S0 ? cudaMemcpyAsync(a.ST, a.S0, ns * 4, cudaMemcpyDeviceToDevice, s)
                         : cudaMemsetAsync(a.ST, 0, ns * 4, s);
    if (e != cudaSuccess) return KDN_ERR_CUDA;
  }
  if (a.pT) {
    if (a.p0) {
      if (cudaMemcpyAsync(a.pT, a.p0, np * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return KDN_ERR_CUDA;
    } else if (np) {
      k_fill<<<(unsigned)((np + 255) / 256), 256, 0, s>>>(a.pT, np, 1.f);
    }
  }
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

kdn_status_t empty_bwd(const Args &a, cudaStream_t s) {
  const size_t ns = (size_t)a.B * a.H * a.dk * a.dv, np = (size_t)a.B * a.H * a.P;
  if (a.dmu && cudaMemsetAsync(a.dmu, 0, (size_t)a.B * a.H * sizeof(float), s) != cudaSuccess)
    return KDN_ERR_CUDA;
  if (a.dS0) {
    cudaError_t e = a.dST ? cudaMemcpyAsync(a.dS0, a.dST, ns * 4, cudaMemcpyDeviceToDevice, s)
                          : cudaMemsetAsync(a.dS0, 0, ns * 4, s);
    if (e != cudaSuccess) return KDN_ERR_CUDA;
  }
  if (a.dp0) {
    cudaError_t e = a.dpT ? cudaMemcpyAsync(a.dp0, a.dpT, np * 4, cudaMemcpyDeviceToDevice, s)
                          : cudaMemsetAsync(a.dp0, 0, np * 4, s);
    if (e != cudaSuccess) return KDN_ERR_CUDA;
  }
  return KDN_OK;
}

kdn_status_t fwd_entry(int variant, const kdn_desc_t *d, const void *q, const void *k,
                       const void *v, const void *g, const void *omega, const void *r,
                       const float *S0, const float *p0, void *o, float *ST, float *pT,
                       void *ws, size_t ws_bytes, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, false, &a);
  if (st != KDN_OK) return st;
  const bool work = (size_t)a.B * a.H * a.T > 0;
  if (work && !ptrs_ok({q, k, v, g, omega, r, o}, {S0, p0, ST, pT})) return KDN_ERR_INVALID_ARG;
  if (!work && !ptrs_ok({}, {S0, p0, ST, pT})) return KDN_ERR_INVALID_ARG;
  const size_t base = workspace_layout(&a, nullptr, false);
  int nseg = seg_count(a);
  // a workspace without room for the segment buffers runs the single pass
  if (nseg > 1 && base + seg_workspace_bytes(a, nseg) > ws_bytes) nseg = 1;
  const size_t need = base + (nseg > 1 ? seg_workspace_bytes(a, nseg) : 0);
  if (need > ws_bytes || (need && (!ws || ((uintptr_t)ws % kAlign)))) return KDN_ERR_WORKSPACE;
  workspace_layout(&a, static_cast<char *>(ws), false);
  a.q = q; a.k = k; a.v = v; a.g = g; a.omega = omega; a.r = r;
  a.S0 = S0; a.p0 = p0; a.o = o; a.ST = ST; a.pT = pT;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.status, 0, sizeof(unsigned), s) != cudaSuccess) return KDN_ERR_CUDA;
  if ((size_t)a.B * a.H == 0) return KDN_OK;
  if (a.T == 0) return empty_fwd(a, s);
  if (nseg > 1) return launch_seg_fwd(a, nseg, static_cast<char *>(ws) + base, s);
  if (use_fused(a) && wy_fwd_supported(a, false)) return launch_wy_fwd(a, s);
  if (use_fused(a)) return launch_fused_fwd(a, s);
  return launch_chunked_fwd(a, s, false);
}

kdn_status_t bwd_entry(int variant, const kdn_desc_t *d, const void *q, const void *k,
                       const void *v, const void *g, const void *omega, const void *r,
                       const float *S0, const float *p0, const void *dO, const float *dST,
                       const float *dpT, void *dq, void *dk, void *dv, void *dg, void *domega,
                       void *dr, float *dS0, float *dp0, float *dmu, void *ws,
                       size_t ws_bytes, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, false, &a);
  if (st != KDN_OK) return st;
  const bool work = (size_t)a.B * a.H * a.T > 0;
  if (work && !ptrs_ok({q, k, v, g, omega, r, dO, dq, dk, dv, dg, domega, dr},
                       {S0, p0, dST, dpT, dS0, dp0, dmu}))
    return KDN_ERR_INVALID_ARG;
  if (!work && !ptrs_ok({}, {S0, p0, dST, dpT, dS0, dp0, dmu})) return KDN_ERR_INVALID_ARG;
  const size_t need = workspace_layout(&a, nullptr, true);
  if (need > ws_bytes || (need && (!ws || ((uintptr_t)ws % kAlign)))) return KDN_ERR_WORKSPACE;
  workspace_layout(&a, static_cast<char *>(ws), true);
  a.q = q; a.k = k; a.v = v; a.g = g; a.omega = omega; a.r = r; a.S0 = S0; a.p0 = p0;
  a.dO = dO; a.dST = dST; a.dpT = dpT;
  a.dq = dq; a.dk_ = dk; a.dv_ = dv; a.dg = dg; a.domega = domega; a.dr = dr;
  a.dS0 = dS0; a.dp0 = dp0; a.dmu = dmu;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.status, 0, sizeof(unsigned), s) != cudaSuccess) return KDN_ERR_CUDA;
  if ((size_t)a.B * a.H == 0) return KDN_OK;
  if (a.T == 0) return empty_bwd(a, s);
  if (use_fused_bwd(a)) return launch_fused_bwd(a, s);
  // the general kernels accumulate dmu with atomics
  if (a.dmu && cudaMemsetAsync(a.dmu, 0, (size_t)a.B * a.H * sizeof(float), s) != cudaSuccess)
    return KDN_ERR_CUDA;
  return launch_chunked_bwd(a, s);
}

// Training pair: forward that keeps the fused backward's context in `saved`,
// and the backward sweep that starts from it.
kdn_status_t fwd_save_entry(int variant, const kdn_desc_t *d, const void *q, const void *k, const void *v,
                            const void *g, const void *omega, const void *r, const float *S0,
                            const float *p0, void *o, float *ST, float *pT, void *saved,
                            size_t saved_bytes, void *ws, size_t ws_bytes, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, false, &a);
  if (st != KDN_OK) return st;
  const bool work = (size_t)a.B * a.H * a.T > 0;
  if (work && !use_fused_bwd(a)) return KDN_ERR_UNSUPPORTED;
  // (the diagonal backward reads Y = V - Kbar S_in from the context, which the WY forward writes)
  if (work && variant == 0 && !wy_fwd_supported(a, true)) return KDN_ERR_UNSUPPORTED;
  if (work && !ptrs_ok({q, k, v, g, omega, r, o, saved}, {S0, p0, ST, pT})) return KDN_ERR_INVALID_ARG;
  if (!work && !ptrs_ok({}, {S0, p0, ST, pT})) return KDN_ERR_INVALID_ARG;
  if (work && (saved_bytes < fused_saved_bytes(a) || ((uintptr_t)saved % kAlign)))
    return KDN_ERR_WORKSPACE;
  const size_t need = workspace_layout(&a, nullptr, false);
  if (need > ws_bytes || (need && (!ws || ((uintptr_t)ws % kAlign)))) return KDN_ERR_WORKSPACE;
  workspace_layout(&a, static_cast<char *>(ws), false);
  a.q = q; a.k = k; a.v = v; a.g = g; a.omega = omega; a.r = r;
  a.S0 = S0; a.p0 = p0; a.o = o; a.ST = ST; a.pT = pT;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.status, 0, sizeof(unsigned), s) != cudaSuccess) return KDN_ERR_CUDA;
  if ((size_t)a.B * a.H == 0) return KDN_OK;
  if (a.T == 0) return empty_fwd(a, s);
  const size_t nsv = (size_t)a.B * a.H * ((a.T + 63) / 64) * fused_ctx_record_bytes();
  if (wy_fwd_supported(a, true))
    return launch_wy_fwd(a, s, static_cast<unsigned char *>(saved),
                         reinterpret_cast<float *>(static_cast<char *>(saved) + nsv));
  return launch_fused_fwd(a, s, static_cast<unsigned char *>(saved),
                          reinterpret_cast<float *>(static_cast<char *>(saved) + nsv), true);
}

kdn_status_t bwd_saved_entry(int variant, const kdn_desc_t *d, const void *q, const void *k, const void *v,
                             const void *g, const void *omega, const void *r, const void *saved,
                             size_t saved_bytes, const void *dO, const float *dST,
                             const float *dpT, void *dq, void *dk, void *dv, void *dg,
                             void *domega, void *dr, float *dS0, float *dp0, float *dmu,
                             void *ws, size_t ws_bytes, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, false, &a);
  if (st != KDN_OK) return st;
  const bool work = (size_t)a.B * a.H * a.T > 0;
  if (work && !use_fused_bwd(a)) return KDN_ERR_UNSUPPORTED;
  if (work && !ptrs_ok({q, k, v, g, omega, r, saved, dO, dq, dk, dv, dg, domega, dr},
                       {dST, dpT, dS0, dp0, dmu}))
    return KDN_ERR_INVALID_ARG;
  if (!work && !ptrs_ok({}, {dST, dpT, dS0, dp0, dmu})) return KDN_ERR_INVALID_ARG;
  if (work && (saved_bytes < fused_saved_bytes(a) || ((uintptr_t)saved % kAlign)))
    return KDN_ERR_WORKSPACE;
  const size_t need = workspace_layout(&a, nullptr, false);
  if (need > ws_bytes || (need && (!ws || ((uintptr_t)ws % kAlign)))) return KDN_ERR_WORKSPACE;
  workspace_layout(&a, static_cast<char *>(ws), false);
  a.q = q; a.k = k; a.v = v; a.g = g; a.omega = omega; a.r = r;
  a.dO = dO; a.dST = dST; a.dpT = dpT;
  a.dq = dq; a.dk_ = dk; a.dv_ = dv; a.dg = dg; a.domega = domega; a.dr = dr;
  a.dS0 = dS0; a.dp0 = dp0; a.dmu = dmu;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.status, 0, sizeof(unsigned), s) != cudaSuccess) return KDN_ERR_CUDA;
  if ((size_t)a.B * a.H == 0) return KDN_OK;
  if (a.T == 0) return empty_bwd(a, s);
  const size_t nsv = (size_t)a.B * a.H * ((a.T + 63) / 64) * fused_ctx_record_bytes();
  a.fSin = static_cast<unsigned char *>(const_cast<void *>(saved));
  a.fpin = reinterpret_cast<float *>(static_cast<char *>(const_cast<void *>(saved)) + nsv);
  return launch_fused_bwd_sweep(a, s);
}

kdn_status_t decode_entry(int variant, const kdn_desc_t *d, const void *q, const void *k,
                          const void *v, const void *g, const void *omega, const void *r,
                          float *S, float *p, void *o, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, true, &a);
  if (st != KDN_OK) return st;
  if ((size_t)a.B * a.H == 0) return KDN_OK;
  if (!ptrs_ok({q, k, v, g, omega, r, S, p, o}, {})) return KDN_ERR_INVALID_ARG;
  a.q = q; a.k = k; a.v = v; a.g = g; a.omega = omega; a.r = r; a.o = o;
  return launch_decode(a, S, p, static_cast<cudaStream_t>(stream));
}

kdn_status_t beta_eff_entry(int variant, const kdn_desc_t *d, const void *saved,
                            size_t saved_bytes, const void *r, float *beta_eff, void *stream) {
  Args a;
  kdn_status_t st = fill_sizes(d, variant, false, &a);
  if (st != KDN_OK) return st;
  if ((size_t)a.B * a.H * a.T == 0) return KDN_OK;
  if (!use_fused_bwd(a)) return KDN_ERR_UNSUPPORTED;
  if (!ptrs_ok({saved, r, beta_eff}, {})) return KDN_ERR_INVALID_ARG;
  if (saved_bytes < fused_saved_bytes(a)) return KDN_ERR_WORKSPACE;
  a.r = r;
  return launch_beta_eff(a, saved, beta_eff, static_cast<cudaStream_t>(stream));
}

}  // namespace

size_t fwd_min_workspace_bytes(const kdn_desc_t *desc, int variant) {
  Args a;
  if (fill_sizes(desc, variant, false, &a) != KDN_OK) return 0;
  return workspace_layout(&a, nullptr, false);
}

size_t workspace_layout(Args *a, char *base, bool bwd) {
  const size_t BH = (size_t)a->B * a->H, Tp = a->Tp, NC = a->NC, C = a->C;
  const size_t dk = a->dk, dv = a->dv, P = a->P;
  size_t off = 0;
  auto take = [&](size_t nfloat) -> float * {
    float *p = base ? reinterpret_cast<float *>(base + off) : nullptr;
    off += round_up(nfloat * sizeof(float));
    return p;
  };
  a->status = reinterpret_cast<unsigned *>(take(kAlign / sizeof(float)));
  if (!bwd && use_fused(*a)) return off;
  if (bwd && a->T > 0 && use_fused_bwd(*a)) {
    const size_t NC64 = (a->T + 63) / 64;  // the fused kernels use 64-token chunks
    a->fSin = reinterpret_cast<unsigned char *>(take(BH * NC64 * fused_ctx_record_bytes() / sizeof(float)));
    a->fpin = take(BH * NC64 * dk);
    return off;
  }
  a->phat = take(BH * Tp * P);
  a->isotok = a->variant == 1 ? take(BH * Tp * 2) : nullptr;
  a->W = take(BH * NC * C * dk);
  a->U = take(BH * NC * C * dv);
  a->Qb = take(BH * NC * C * dk);
  a->Aqk = take(BH * NC * C * C);
  a->Kt = take(BH * NC * C * dk);
  a->gC = take(BH * NC * dk);
  if (bwd) {
    a->Sin = take(BH * NC * dk * dv);
    a->dSout = take(BH * NC * dk * dv);
    a->dR = take(BH * NC * C * dv);
    a->dkpart = take(BH * Tp * dk);
    a->dgpart = take(BH * Tp * dk);
    a->dphloc = take(BH * Tp * P);
    a->drpart = take(BH * Tp);
    a->drw = take(BH * Tp * 4);
    a->isoadj = a->variant == 1 ? take(BH * Tp * 2) : nullptr;
  }
  return off;
}

}  // namespace kdn

using namespace kdn;

extern "C" {

int kdn_version(void) { return 100; }

const char *kdn_status_string(kdn_status_t s) {
  switch (s) {
    case KDN_OK: return "KDN_OK";
    case KDN_ERR_INVALID_ARG: return "KDN_ERR_INVALID_ARG";
    case KDN_ERR_UNSUPPORTED: return "KDN_ERR_UNSUPPORTED";
    case KDN_ERR_WORKSPACE: return "KDN_ERR_WORKSPACE";
    case KDN_ERR_CUDA: return "KDN_ERR_CUDA";
    case KDN_ERR_TIMEOUT: return "KDN_ERR_TIMEOUT";
    case KDN_ERR_RANGE: return "KDN_ERR_RANGE";
  }
  return "KDN_ERR_UNKNOWN";
}

size_t kdn_fwd_workspace_bytes(const kdn_desc_t *desc, int variant) {
  Args a;
  if (fill_sizes(desc, variant, false, &a) != KDN_OK) return 0;
  const int nseg = seg_count(a);
  return workspace_layout(&a, nullptr, false) + (nseg > 1 ? seg_workspace_bytes(a, nseg) : 0);
}

size_t kdn_bwd_workspace_bytes(const kdn_desc_t *desc, int variant) {
  Args a;
  if (fill_sizes(desc, variant, false, &a) != KDN_OK) return 0;
  return workspace_layout(&a, nullptr, true);
}

kdn_status_t kdn_diag_fwd(const kdn_desc_t *desc, const void *q, const void *k, const void *v,
                          const void *g, const void *omega, const void *r, const float *S0,
                          const float *p0, void *o, float *ST, float *pT, void *workspace,
                          size_t workspace_bytes, void *stream) {
  return fwd_entry(0, desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, workspace, workspace_bytes,
                   stream);
}

kdn_status_t kdn_iso_fwd(const kdn_desc_t *desc, const void *q, const void *k, const void *v,
                         const void *g, const void *omega, const void *r, const float *S0,
                         const float *p0, void *o, float *ST, float *pT, void *workspace,
                         size_t workspace_bytes, void *stream) {
  return fwd_entry(1, desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, workspace, workspace_bytes,
                   stream);
}

kdn_status_t kdn_diag_bwd(const kdn_desc_t *desc, const void *q, const void *k, const void *v,
                          const void *g, const void *omega, const void *r, const float *S0,
                          const float *p0, const void *dO, const float *dST, const float *dpT,
                          void *dq, void *dk, void *dv, void *dg, void *domega, void *dr,
                          float *dS0, float *dp0, float *dmu, void *workspace,
                          size_t workspace_bytes, void *stream) {
  return bwd_entry(0, desc, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, dq, dk, dv, dg, domega,
                   dr, dS0, dp0, dmu, workspace, workspace_bytes, stream);
}

kdn_status_t kdn_iso_bwd(const kdn_desc_t *desc, const void *q, const void *k, const void *v,
                         const void *g, const void *omega, const void *r, const float *S0,
                         const float *p0, const void *dO, const float *dST, const float *dpT,
                         void *dq, void *dk, void *dv, void *dg, void *domega, void *dr,
                         float *dS0, float *dp0, float *dmu, void *workspace,
                         size_t workspace_bytes, void *stream) {
  return bwd_entry(1, desc, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, dq, dk, dv, dg, domega,
                   dr, dS0, dp0, dmu, workspace, workspace_bytes, stream);
}

size_t kdn_saved_bytes(const kdn_desc_t *desc, int variant) {
  Args a;
  if (fill_sizes(desc, variant, false, &a) != KDN_OK) return 0;
  return fused_saved_bytes(a);
}

kdn_status_t kdn_diag_fwd_save(const kdn_desc_t *desc, const void *q, const void *k,
                               const void *v, const void *g, const void *omega, const void *r,
                               const float *S0, const float *p0, void *o, float *ST, float *pT,
                               void *saved, size_t saved_bytes, void *workspace,
                               size_t workspace_bytes, void *stream) {
  return fwd_save_entry(0, desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, saved, saved_bytes,
                        workspace, workspace_bytes, stream);
}

kdn_status_t kdn_diag_bwd_saved(const kdn_desc_t *desc, const void *q, const void *k,
                                const void *v, const void *g, const void *omega, const void *r,
                                const void *saved, size_t saved_bytes, const void *dO,
                                const float *dST, const float *dpT, void *dq, void *dk, void *dv,
                                void *dg, void *domega, void *dr, float *dS0, float *dp0,
                                float *dmu, void *workspace, size_t workspace_bytes,
                                void *stream) {
  return bwd_saved_entry(0, desc, q, k, v, g, omega, r, saved, saved_bytes, dO, dST, dpT, dq, dk, dv,
                         dg, domega, dr, dS0, dp0, dmu, workspace, workspace_bytes, stream);
}

kdn_status_t kdn_iso_fwd_save(const kdn_desc_t *desc, const void *q, const void *k,
                              const void *v, const void *g, const void *omega, const void *r,
                              const float *S0, const float *p0, void *o, float *ST, float *pT,
                              void *saved, size_t saved_bytes, void *workspace,
                              size_t workspace_bytes, void *stream) {
  return fwd_save_entry(1, desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, saved, saved_bytes,
                        workspace, workspace_bytes, stream);
}

kdn_status_t kdn_iso_bwd_saved(const kdn_desc_t *desc, const void *q, const void *k,
                               const void *v, const void *g, const void *omega, const void *r,
                               const void *saved, size_t saved_bytes, const void *dO,
                               const float *dST, const float *dpT, void *dq, void *dk, void *dv,
                               void *dg, void *domega, void *dr, float *dS0, float *dp0,
                               float *dmu, void *workspace, size_t workspace_bytes,
                               void *stream) {
  return bwd_saved_entry(1, desc, q, k, v, g, omega, r, saved, saved_bytes, dO, dST, dpT, dq, dk, dv,
                         dg, domega, dr, dS0, dp0, dmu, workspace, workspace_bytes, stream);
}

kdn_status_t kdn_diag_decode_step(const kdn_desc_t *desc, const void *q, const void *k,
                                  const void *v, const void *g, const void *omega, const void *r,
                                  float *S, float *p, void *o, void *stream) {
  return decode_entry(0, desc, q, k, v, g, omega, r, S, p, o, stream);
}

kdn_status_t kdn_iso_decode_step(const kdn_desc_t *desc, const void *q, const void *k,
                                 const void *v, const void *g, const void *omega, const void *r,
                                 float *S, float *p, void *o, void *stream) {
  return decode_entry(1, desc, q, k, v, g, omega, r, S, p, o, stream);
}

int kdn_kernel_launches(const kdn_desc_t *desc, int variant, int op) {
  Args a;
  if (fill_sizes(desc, variant, op == 2, &a) != KDN_OK) return -1;
  switch (op) {
    case 0: return seg_count(a) > 1 ? 5 : use_fused(a) ? 1 : chunked_fwd_launches(a);
    case 1: return (a.T > 0 && use_fused_bwd(a)) ? 2 : chunked_bwd_launches(a);
    case 2: return 1;
    case 3:
    case 4:
    case 5: return fused_saved_bytes(a) > 0 ? 1 : -1;
  }
  return -1;
}

kdn_status_t kdn_diag_beta_eff(const kdn_desc_t *desc, const void *saved, size_t saved_bytes,
                               const void *r, float *beta_eff, void *stream) {
  return beta_eff_entry(0, desc, saved, saved_bytes, r, beta_eff, stream);
}

kdn_status_t kdn_iso_beta_eff(const kdn_desc_t *desc, const void *saved, size_t saved_bytes,
                              const void *r, float *beta_eff, void *stream) {
  return beta_eff_entry(1, desc, saved, saved_bytes, r, beta_eff, stream);
}

kdn_status_t kdn_selftest_wait_timeout(void *workspace, void *stream) {
  if (!workspace || ((uintptr_t)workspace % kAlign)) return KDN_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned *status = static_cast<unsigned *>(workspace);
  if (cudaMemsetAsync(status, 0, sizeof(unsigned), s) != cudaSuccess) return KDN_ERR_CUDA;
  return launch_wait_selftest(status, s);
}

kdn_status_t kdn_get_device_status(void *workspace, void *stream) {
  if (!workspace || ((uintptr_t)workspace % kAlign)) return KDN_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned word = 0;
  if (cudaMemcpyAsync(&word, workspace, sizeof word, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return KDN_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return KDN_ERR_CUDA;
  if (word != 0) {
    if (cudaMemsetAsync(workspace, 0, sizeof word, s) != cudaSuccess) return KDN_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return KDN_ERR_CUDA;
    return static_cast<kdn_status_t>(word);
  }
  return KDN_OK;
}

}  // extern "C"
