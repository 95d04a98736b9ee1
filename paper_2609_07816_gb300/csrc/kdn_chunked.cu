// kdn_chunked.cu -- general chunked forward and backward of the Diagonal and
// Isotropic KDN on CUDA cores (float32 arithmetic, any dk, dv in {32,64,128},
// float32 or bfloat16 activations).
//
// The forward is the two-stage scheme of App. F, split into three kernels:
//   k_gain_scan_*  the uncertainty recursion over time (eq. prefix-diag-
//                  uncertainty / eq. iso-kla-box-cov-update), emitting the
//                  pre-write predictive variance phat_t for every token;
//   k_chunk_prep   per chunk, in parallel over chunks: the gain emission
//                  (eq. chunk-gain-emission), the cumulative log-decay G and
//                  gamma = exp(G) (eq. chunk-memory-normalization), the scaled
//                  keys/queries (eq. chunk-memory-scaled-keys), T and A_qk,
//                  A = (I + T)^-1 by forward substitution, W = A Kbar,
//                  U = A V and K_tail (eq. chunk-memory-wy, -tail-output);
//   k_state_fwd    the sequential inter-chunk pass R = U - W S_in,
//                  O = Qbar S_in + A_qk R, S_out = diag(gamma_C) S_in + K_tail^T R
//                  (eq. chunk-memory-output-state), columns of S split across
//                  CTAs (the columns of S are independent given kappa).
// The backward reverses these stages: k_state_bwd carries dS backwards over
// chunks, k_chunk_bwd forms every chunk-local adjoint in parallel, and
// k_gain_bwd_* runs the adjoint of the uncertainty recursion backwards in time.
//
// All chunk-local matrices are float32 in shared memory; intermediates that
// cross kernels live in the caller's workspace.
#include "kdn_internal.cuh"

namespace kdn {
namespace {

constexpr int NT = 256;  // threads per CTA of the chunk kernels
constexpr int CC = 32;   // chunk length of these kernels
constexpr int CW = 32;   // value columns per CTA of the state kernels
constexpr int LC = CC + 1;

#define KDN_TID (int)threadIdx.x

// ---------------------------------------------------------------------------
// Uncertainty recursion over time.

// Tokens are processed in blocks of GU; the inputs of block n+1 are loaded
// into registers before block n is computed, so the loads never sit on the
// loop-carried dependence of the recursion.
constexpr int GU = 16;

template <typename DT>
__global__ void __launch_bounds__(32) k_gain_scan_diag(Args a) {
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int i = blockIdx.y * 32 + threadIdx.x;
  const int dk = a.dk;
  float p = a.p0 ? a.p0[(size_t)bh * dk + i] : 1.f;
  float *out = a.phat + (size_t)bh * a.Tp * dk + i;
  float cg[GU], cw[GU], ck[GU], cr[GU];
  auto load = [&](int t0, float *g_, float *w_, float *k_, float *r_) {
#pragma unroll
    for (int j = 0; j < GU; ++j) {
      const int t = t0 + j;
      g_[j] = 0.f; w_[j] = 0.f; k_[j] = 0.f; r_[j] = 1.f;
      if (t < a.T) {
        const size_t th = tok_index(a, b, t, h);
        g_[j] = gate_logalpha(a.gates, ld<DT>(a.g, th * dk + i));
        w_[j] = gate_omega(a.gates, ld<DT>(a.omega, th * dk + i));
        k_[j] = ld<DT>(a.k, th * dk + i);
        r_[j] = gate_r(a.gates, a.rmin, ld<DT>(a.r, th));
      }
    }
  };
  load(0, cg, cw, ck, cr);
  for (int t0 = 0; t0 < a.T; t0 += GU) {
    float ng[GU], nw[GU], nk[GU], nr[GU];
    load(t0 + GU, ng, nw, nk, nr);
#pragma unroll
    for (int j = 0; j < GU; ++j) {
      if (t0 + j < a.T) {
        const float al2 = expf(2.f * cg[j]);
        const float ph = al2 * p + cw[j];  // eq. diag-covariance-prediction
        out[(size_t)(t0 + j) * dk] = ph;
        const float u = a.mu * ck[j] * ck[j] / cr[j];  // eq. diag-cov-update
        p = ph / (1.f + u * ph);
      }
    }
#pragma unroll
    for (int j = 0; j < GU; ++j) { cg[j] = ng[j]; cw[j] = nw[j]; ck[j] = nk[j]; cr[j] = nr[j]; }
  }
  for (int t = a.T; t < a.Tp; ++t) out[(size_t)t * dk] = 0.f;
  if (a.pT) a.pT[(size_t)bh * dk + i] = p;
}

template <typename DT>
__global__ void __launch_bounds__(32) k_gain_scan_iso(Args a) {
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int lane = threadIdx.x, dk = a.dk;
  __shared__ float s_a[32], s_n2[32], s_w[32], s_r[32];
  float bst = a.p0 ? a.p0[bh] : 1.f;
  for (int t0 = 0; t0 < a.T; t0 += 32) {
    const int t = t0 + lane;
    float aa = 1.f, n2 = 0.f, w = 0.f, rr = 1.f;
    if (t < a.T) {
      const size_t th = tok_index(a, b, t, h);
      float sa = 0.f;
#pragma unroll 8
      for (int i = 0; i < dk; ++i) {
        const float kk = ld<DT>(a.k, th * dk + i);
        n2 += kk * kk;
        if (a.pcd) sa += expf(2.f * gate_logalpha(a.gates, ld<DT>(a.g, th * dk + i)));
      }
      aa = a.pcd ? sa / dk : expf(2.f * gate_logalpha(a.gates, ld<DT>(a.g, th)));
      w = gate_omega(a.gates, ld<DT>(a.omega, th));
      rr = gate_r(a.gates, a.rmin, ld<DT>(a.r, th));
      a.isotok[((size_t)bh * a.Tp + t) * 2 + 0] = aa;
      a.isotok[((size_t)bh * a.Tp + t) * 2 + 1] = n2;
    }
    s_a[lane] = aa;
    s_n2[lane] = n2;
    s_w[lane] = w;
    s_r[lane] = rr;
    __syncwarp();
    if (lane == 0) {
      for (int j = 0; j < 32 && t0 + j < a.T; ++j) {
        const float bhat = s_a[j] * bst + s_w[j];  // eq. iso-kla-box-cov-update
        a.phat[(size_t)bh * a.Tp + t0 + j] = bhat;
        const float u = a.mu * s_n2[j] / (dk * s_r[j]);
        bst = bhat / (1.f + u * bhat);
      }
    }
    __syncwarp();
  }
  for (int t = a.T + lane; t < a.Tp; t += 32) {
    a.phat[(size_t)bh * a.Tp + t] = 0.f;
    a.isotok[((size_t)bh * a.Tp + t) * 2 + 0] = 1.f;
    a.isotok[((size_t)bh * a.Tp + t) * 2 + 1] = 0.f;
  }
  if (lane == 0 && a.pT) a.pT[bh] = bst;
}

// ---------------------------------------------------------------------------
// Chunk-local factors shared by the forward prep and the backward.
// On return (for chunk c of head bh):
//   sK  = Kbar = Gamma (.) K,  sQ = Qbar = tau Gamma (.) Q,  sKk = Kbar^kappa,
//   sT  = strict lower part of Kbar Kbar^kappa^T,  sAqk = lower part of
//   Qbar Kbar^kappa^T,  sA = (I + T)^-1,  s_s = s_t (diag) or beta_t (iso),
//   s_n2 = |k_t|^2 (iso),  s_gC = gamma_C,  sG (optional) = G.
// Tokens past T are identity tokens: k = q = 0, g = 0, r = 1, kappa = 0.

template <int V, typename DT, int DK>
__device__ void prep_core(const Args &a, int c, int bh, float *sK, float *sQ, float *sKk,
                          float *sT, float *sA, float *sAqk, float *s_s, float *s_n2,
                          float *s_gC, float *sG) {
  constexpr int LD = DK + 1;
  const int b = bh / a.H, h = bh % a.H;
  const int tid = KDN_TID, warp = tid / 32, lane = tid % 32;
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int t = idx / DK, i = idx % DK, tt = c * CC + t;
    float kv = 0.f, qv = 0.f;
    if (tt < a.T) {
      const size_t th = tok_index(a, b, tt, h);
      kv = ld<DT>(a.k, th * DK + i);
      qv = ld<DT>(a.q, th * DK + i);
    }
    sK[t * LD + i] = kv;
    sQ[t * LD + i] = qv;
  }
  __syncthreads();
  // gain emission from the pre-write predictive variance (eq. chunk-gain-emission)
  for (int t = warp; t < CC; t += NT / 32) {
    const int tt = c * CC + t;
    const float rr = tt < a.T ? gate_r(a.gates, a.rmin, ld<DT>(a.r, tok_index(a, b, tt, h))) : 1.f;
    if (V == 0) {
      const float *ph = a.phat + ((size_t)bh * a.Tp + tt) * DK;
      float part = 0.f;
      for (int i = lane; i < DK; i += 32) {
        const float kv = sK[t * LD + i];
        part += ph[i] * kv * kv;
      }
      const float s = rr + warp_sum(part);
      if (lane == 0) s_s[t] = s;
      for (int i = lane; i < DK; i += 32) sKk[t * LD + i] = ph[i] * sK[t * LD + i] / s;
    } else {
      float part = 0.f;
      for (int i = lane; i < DK; i += 32) part += sK[t * LD + i] * sK[t * LD + i];
      const float n2 = warp_sum(part);
      const float bhat = a.phat[(size_t)bh * a.Tp + tt];
      const float beta = bhat / (rr + bhat * n2);
      if (lane == 0) { s_s[t] = beta; s_n2[t] = n2; }
      for (int i = lane; i < DK; i += 32) sKk[t * LD + i] = beta * sK[t * LD + i];
    }
  }
  __syncthreads();
  // cumulative decay and the scaled operands (eq. chunk-memory-scaled-keys)
  if (tid < DK) {
    const int i = tid;
    float G = 0.f, gam = 1.f;
    for (int t = 0; t < CC; ++t) {
      const int tt = c * CC + t;
      float gg = 0.f;
      if (tt < a.T) {
        const size_t th = tok_index(a, b, tt, h);
        gg = a.pcd ? gate_logalpha(a.gates, ld<DT>(a.g, th * DK + i)) : gate_logalpha(a.gates, ld<DT>(a.g, th));
      }
      G += gg;
      gam = expf(G);
      if (sG) sG[t * LD + i] = G;
      sK[t * LD + i] *= gam;
      sKk[t * LD + i] /= gam;
      sQ[t * LD + i] *= a.tau * gam;
    }
    s_gC[i] = gam;
  }
  __syncthreads();
  for (int idx = tid; idx < CC * CC; idx += NT) {
    const int r = idx / CC, s = idx % CC;
    float tm = 0.f, aq = 0.f;
    if (s <= r) {
#pragma unroll 8
      for (int i = 0; i < DK; ++i) {
        const float kks = sKk[s * LD + i];
        tm += sK[r * LD + i] * kks;
        aq += sQ[r * LD + i] * kks;
      }
      if (s == r) tm = 0.f;
    }
    sT[r * LC + s] = tm;
    sAqk[r * LC + s] = aq;
  }
  __syncthreads();
  // A = (I + T)^-1, one column per thread by forward substitution
  if (tid < CC) {
    const int j = tid;
    for (int r = 0; r < CC; ++r) {
      float acc = 0.f;
      for (int s = 0; s < r; ++s) acc += sT[r * LC + s] * sA[s * LC + j];
      sA[r * LC + j] = (r == j ? 1.f : 0.f) - acc;
    }
  }
  __syncthreads();
}

template <int DK>
constexpr size_t prep_smem_bytes() {
  return sizeof(float) * (3 * CC * (DK + 1) + CC * 129 + 3 * CC * LC + 2 * CC + DK);
}

template <int V, typename DT, int DK>
__global__ void __launch_bounds__(NT) k_chunk_prep(Args a) {
  constexpr int LD = DK + 1;
  extern __shared__ float sm[];
  float *sK = sm, *sQ = sK + CC * LD, *sKk = sQ + CC * LD, *sV = sKk + CC * LD;
  float *sT = sV + CC * 129, *sA = sT + CC * LC, *sAqk = sA + CC * LC;
  float *s_s = sAqk + CC * LC, *s_n2 = s_s + CC, *s_gC = s_n2 + CC;
  const int bh = blockIdx.x, c = blockIdx.y, tid = KDN_TID;
  const int b = bh / a.H, h = bh % a.H, dv = a.dv;
  prep_core<V, DT, DK>(a, c, bh, sK, sQ, sKk, sT, sA, sAqk, s_s, s_n2, s_gC, nullptr);
  for (int idx = tid; idx < CC * dv; idx += NT) {
    const int t = idx / dv, j = idx % dv, tt = c * CC + t;
    sV[t * 129 + j] = tt < a.T ? ld<DT>(a.v, tok_index(a, b, tt, h) * dv + j) : 0.f;
  }
  __syncthreads();
  const size_t base = (size_t)bh * a.NC + c;
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int r = idx / DK, i = idx % DK;
    float w = 0.f;
    for (int s = 0; s <= r; ++s) w += sA[r * LC + s] * sK[s * LD + i];
    const size_t o = (base * CC + r) * DK + i;
    a.W[o] = w;
    a.Qb[o] = sQ[r * LD + i];
    a.Kt[o] = s_gC[i] * sKk[r * LD + i];
  }
  for (int idx = tid; idx < CC * dv; idx += NT) {
    const int r = idx / dv, j = idx % dv;
    float u = 0.f;
    for (int s = 0; s <= r; ++s) u += sA[r * LC + s] * sV[s * 129 + j];
    a.U[(base * CC + r) * dv + j] = u;
  }
  for (int idx = tid; idx < CC * CC; idx += NT)
    a.Aqk[base * CC * CC + idx] = sAqk[(idx / CC) * LC + idx % CC];
  if (tid < DK) a.gC[base * DK + tid] = s_gC[tid];
}

// ---------------------------------------------------------------------------
// Inter-chunk state passes.  The per-chunk factors (W, Qbar, K_tail, A_qk,
// gamma_C and the chunk's U or dO slice) are double-buffered in shared memory
// with cp.async, so chunk c+1 streams in while chunk c is computed.

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// 16-byte global -> shared copy; zero-filled when `valid` is false
__device__ __forceinline__ void cp16(void *dst, const void *src, bool valid = true) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int DK>
struct StateBuf {
  static constexpr int LD = DK + 4;  // 16-byte aligned rows
  static constexpr int LA = CC + 4;
  static constexpr int LS = CW + 4;
  // floats per buffer: W, Qbar, K_tail, A_qk, gamma_C, and a [C][CW] slice (U or raw dO)
  static constexpr int FLOATS = 3 * CC * LD + CC * LA + DK + CC * LS;
};

// Issues the cp.async copies of chunk c's factors into buffer `buf`.
// `slice` is U (forward, fp32) or dO (backward, bytes of the activation dtype).
template <int DK>
__device__ void issue_chunk_factors(const Args &a, int bh, int c, float *buf, int j0,
                                    bool backward) {
  using SB = StateBuf<DK>;
  float *sW = buf, *sQ = sW + CC * SB::LD, *sKt = sQ + CC * SB::LD, *sAqk = sKt + CC * SB::LD;
  float *sgC = sAqk + CC * SB::LA, *sSl = sgC + DK;
  const size_t base = (size_t)bh * a.NC + c;
  constexpr int RC = DK / 4;  // 16-byte chunks per factor row
  for (int e = KDN_TID; e < CC * RC; e += NT) {
    const int r = e / RC, q = e % RC;
    const size_t o = (base * CC + r) * DK + 4 * q;
    cp16(sW + r * SB::LD + 4 * q, a.W + o);
    cp16(sQ + r * SB::LD + 4 * q, a.Qb + o);
    cp16(sKt + r * SB::LD + 4 * q, a.Kt + o);
  }
  for (int e = KDN_TID; e < CC * (CC / 4); e += NT) {
    const int r = e / (CC / 4), q = e % (CC / 4);
    cp16(sAqk + r * SB::LA + 4 * q, a.Aqk + base * CC * CC + r * CC + 4 * q);
  }
  for (int e = KDN_TID; e < DK / 4; e += NT) cp16(sgC + 4 * e, a.gC + base * DK + 4 * e);
  if (!backward) {
    for (int e = KDN_TID; e < CC * (CW / 4); e += NT) {
      const int r = e / (CW / 4), q = e % (CW / 4);
      cp16(sSl + r * SB::LS + 4 * q, a.U + (base * CC + r) * a.dv + j0 + 4 * q);
    }
  } else {
    // raw dO rows of this slice: CW elements of the activation dtype
    const int es = a.dtype == KDN_BF16 ? 2 : 4;
    const int rc = CW * es / 16;
    const int b = bh / a.H, h = bh % a.H;
    for (int e = KDN_TID; e < CC * rc; e += NT) {
      const int r = e / rc, q = e % rc, tt = c * CC + r;
      const bool valid = tt < a.T;
      const char *src = static_cast<const char *>(a.dO) +
                        ((valid ? tok_index(a, b, tt, h) : 0) * a.dv + j0) * es + 16 * q;
      cp16(reinterpret_cast<char *>(sSl + r * SB::LS) + 16 * q, src, valid);
    }
  }
}

template <int DK>
constexpr size_t state_smem_bytes() {
  using SB = StateBuf<DK>;
  return sizeof(float) * (2 * SB::FLOATS + DK * SB::LS + CC * SB::LS);
}

template <typename DT, int DK>
__global__ void __launch_bounds__(NT) k_state_fwd(Args a, int save_states) {
  using SB = StateBuf<DK>;
  constexpr int LD = SB::LD, LA = SB::LA, LS = SB::LS;
  extern __shared__ __align__(16) float sm[];
  float *bufs = sm, *sS = bufs + 2 * SB::FLOATS, *sR = sS + DK * LS;
  const int bh = blockIdx.x, j0 = blockIdx.y * CW, tid = KDN_TID;
  const int b = bh / a.H, h = bh % a.H, dv = a.dv;
  const size_t sbase = (size_t)bh * DK * dv;
  for (int idx = tid; idx < DK * CW; idx += NT) {
    const int i = idx / CW, j = idx % CW;
    sS[i * LS + j] = a.S0 ? a.S0[sbase + (size_t)i * dv + j0 + j] : 0.f;
  }
  issue_chunk_factors<DK>(a, bh, 0, bufs, j0, false);
  cp_commit();
  for (int c = 0; c < a.NC; ++c) {
    float *buf = bufs + (c & 1) * SB::FLOATS;
    if (c + 1 < a.NC) issue_chunk_factors<DK>(a, bh, c + 1, bufs + ((c + 1) & 1) * SB::FLOATS, j0, false);
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    float *sW = buf, *sQ = sW + CC * LD, *sKt = sQ + CC * LD, *sAqk = sKt + CC * LD;
    float *sgC = sAqk + CC * LA, *sU = sgC + DK;
    const size_t base = (size_t)bh * a.NC + c;
    if (save_states) {
      for (int idx = tid; idx < DK * CW; idx += NT) {
        const int i = idx / CW, j = idx % CW;
        a.Sin[(base * DK + i) * dv + j0 + j] = sS[i * LS + j];
      }
    }
    // R = U - W S_in
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW;
      float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 8
      for (int i = 0; i < DK; i += 2) {
        acc0 += sW[r * LD + i] * sS[i * LS + j];
        acc1 += sW[r * LD + i + 1] * sS[(i + 1) * LS + j];
      }
      sR[r * LS + j] = sU[r * LS + j] - (acc0 + acc1);
    }
    __syncthreads();
    // O = Qbar S_in + A_qk R
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW;
      float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 8
      for (int i = 0; i < DK; i += 2) {
        acc0 += sQ[r * LD + i] * sS[i * LS + j];
        acc1 += sQ[r * LD + i + 1] * sS[(i + 1) * LS + j];
      }
      for (int s2 = 0; s2 <= r; ++s2) acc0 += sAqk[r * LA + s2] * sR[s2 * LS + j];
      const int tt = c * CC + r;
      if (a.o && tt < a.T) sto(a.odt, a.o, tok_index(a, b, tt, h) * dv + j0 + j, acc0 + acc1);
    }
    __syncthreads();
    // S_out = diag(gamma_C) S_in + K_tail^T R
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      float acc0 = sgC[i] * sS[i * LS + j], acc1 = 0.f;
#pragma unroll 8
      for (int s2 = 0; s2 < CC; s2 += 2) {
        acc0 += sKt[s2 * LD + i] * sR[s2 * LS + j];
        acc1 += sKt[(s2 + 1) * LD + i] * sR[(s2 + 1) * LS + j];
      }
      sS[i * LS + j] = acc0 + acc1;
    }
    __syncthreads();
  }
  cp_wait<0>();
  if (a.ST) {
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      a.ST[sbase + (size_t)i * dv + j0 + j] = sS[i * LS + j];
    }
  }
}

// dR = A_qk^T dO + K_tail dS_out,  dS_in = Qbar^T dO + diag(gamma_C) dS_out - W^T dR
template <typename DT, int DK>
__global__ void __launch_bounds__(NT) k_state_bwd(Args a) {
  using SB = StateBuf<DK>;
  constexpr int LD = SB::LD, LA = SB::LA, LS = SB::LS;
  extern __shared__ __align__(16) float sm[];
  float *bufs = sm, *sS = bufs + 2 * SB::FLOATS, *sdR = sS + DK * LS;
  const int bh = blockIdx.x, j0 = blockIdx.y * CW, tid = KDN_TID;
  const int dv = a.dv;
  const size_t sbase = (size_t)bh * DK * dv;
  for (int idx = tid; idx < DK * CW; idx += NT) {
    const int i = idx / CW, j = idx % CW;
    sS[i * LS + j] = a.dST ? a.dST[sbase + (size_t)i * dv + j0 + j] : 0.f;
  }
  if (a.NC > 0) issue_chunk_factors<DK>(a, bh, a.NC - 1, bufs + ((a.NC - 1) & 1) * SB::FLOATS, j0, true);
  cp_commit();
  for (int c = a.NC - 1; c >= 0; --c) {
    float *buf = bufs + (c & 1) * SB::FLOATS;
    if (c > 0) issue_chunk_factors<DK>(a, bh, c - 1, bufs + ((c - 1) & 1) * SB::FLOATS, j0, true);
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    float *sW = buf, *sQ = sW + CC * LD, *sKt = sQ + CC * LD, *sAqk = sKt + CC * LD;
    float *sgC = sAqk + CC * LA;
    const DT *sdO = reinterpret_cast<const DT *>(sgC + DK);
    const size_t base = (size_t)bh * a.NC + c;
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      a.dSout[(base * DK + i) * dv + j0 + j] = sS[i * LS + j];
    }
    // dO row r of the slice starts LS floats apart (raw activation dtype)
    auto dO = [&](int r, int j) -> float {
      const DT *row = reinterpret_cast<const DT *>(reinterpret_cast<const float *>(sdO) + r * LS);
      return ld<DT>(row, j);
    };
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW;
      float acc0 = 0.f, acc1 = 0.f;
      for (int s2 = r; s2 < CC; ++s2) acc0 += sAqk[s2 * LA + r] * dO(s2, j);
#pragma unroll 8
      for (int i = 0; i < DK; i += 2) {
        acc0 += sKt[r * LD + i] * sS[i * LS + j];
        acc1 += sKt[r * LD + i + 1] * sS[(i + 1) * LS + j];
      }
      sdR[r * LS + j] = acc0 + acc1;
      a.dR[(base * CC + r) * dv + j0 + j] = acc0 + acc1;
    }
    __syncthreads();
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      float acc0 = sgC[i] * sS[i * LS + j], acc1 = 0.f;
#pragma unroll 8
      for (int r = 0; r < CC; r += 2) {
        acc0 += sQ[r * LD + i] * dO(r, j) - sW[r * LD + i] * sdR[r * LS + j];
        acc1 += sQ[(r + 1) * LD + i] * dO(r + 1, j) - sW[(r + 1) * LD + i] * sdR[(r + 1) * LS + j];
      }
      sS[i * LS + j] = acc0 + acc1;
    }
    __syncthreads();
  }
  cp_wait<0>();
  if (a.dS0) {
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      a.dS0[sbase + (size_t)i * dv + j0 + j] = sS[i * LS + j];
    }
  }
}

// ---------------------------------------------------------------------------
// Chunk-local adjoints, in parallel over chunks.

template <int DK>
constexpr size_t cbwd_smem_bytes() {
  return sizeof(float) * (8 * CC * (DK + 1) + 5 * CC * LC + 2 * DK * (CW + 1) +
                          4 * CC * (CW + 1) + 2 * CC + 2 * DK);
}

template <int V, typename DT, int DK>
__global__ void __launch_bounds__(NT) k_chunk_bwd(Args a) {
  constexpr int LD = DK + 1, LS = CW + 1;
  extern __shared__ float sm[];
  float *sK = sm, *sQ = sK + CC * LD, *sKk = sQ + CC * LD, *sG = sKk + CC * LD;
  float *sW = sG + CC * LD, *sdQ = sW + CC * LD, *sdKt = sdQ + CC * LD, *sdW = sdKt + CC * LD;
  float *sT = sdW + CC * LD, *sA = sT + CC * LC, *sAqk = sA + CC * LC, *sdAqk = sAqk + CC * LC;
  float *sdA = sdAqk + CC * LC;
  float *sSin = sdA + CC * LC, *sdSo = sSin + DK * LS;
  float *sR = sdSo + DK * LS, *sdR = sR + CC * LS, *sdO = sdR + CC * LS, *sV = sdO + CC * LS;
  float *s_s = sV + CC * LS, *s_n2 = s_s + CC, *s_gC = s_n2 + CC, *s_dgC = s_gC + DK;
  const int bh = blockIdx.x, c = blockIdx.y, tid = KDN_TID;
  const int b = bh / a.H, h = bh % a.H, dv = a.dv;
  const size_t base = (size_t)bh * a.NC + c;

  prep_core<V, DT, DK>(a, c, bh, sK, sQ, sKk, sT, sA, sAqk, s_s, s_n2, s_gC, sG);
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int r = idx / DK, i = idx % DK;
    float w = 0.f;
    for (int s = 0; s <= r; ++s) w += sA[r * LC + s] * sK[s * LD + i];
    sW[r * LD + i] = w;
    sdQ[r * LD + i] = 0.f;
    sdKt[r * LD + i] = 0.f;
    sdW[r * LD + i] = 0.f;
  }
  for (int idx = tid; idx < CC * CC; idx += NT) {
    sdAqk[(idx / CC) * LC + idx % CC] = 0.f;
    sdA[(idx / CC) * LC + idx % CC] = 0.f;
  }
  if (tid < DK) s_dgC[tid] = 0.f;

  for (int j0 = 0; j0 < dv; j0 += CW) {
    __syncthreads();
    for (int idx = tid; idx < DK * CW; idx += NT) {
      const int i = idx / CW, j = idx % CW;
      sSin[i * LS + j] = a.Sin[(base * DK + i) * dv + j0 + j];
      sdSo[i * LS + j] = a.dSout[(base * DK + i) * dv + j0 + j];
    }
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW, tt = c * CC + r;
      sdR[r * LS + j] = a.dR[(base * CC + r) * dv + j0 + j];
      float dov = 0.f, vv = 0.f;
      if (tt < a.T) {
        const size_t th = tok_index(a, b, tt, h);
        dov = ld<DT>(a.dO, th * dv + j0 + j);
        vv = ld<DT>(a.v, th * dv + j0 + j);
      }
      sdO[r * LS + j] = dov;
      sV[r * LS + j] = vv;
    }
    __syncthreads();
    // R = A V - W S_in for this column slice
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW;
      float acc = 0.f;
      for (int s = 0; s <= r; ++s) acc += sA[r * LC + s] * sV[s * LS + j];
#pragma unroll 8
      for (int i = 0; i < DK; ++i) acc -= sW[r * LD + i] * sSin[i * LS + j];
      sR[r * LS + j] = acc;
    }
    __syncthreads();
    // dQbar += dO S_in^T; dK_tail += R dS_out^T; dW -= dR S_in^T
    for (int idx = tid; idx < CC * DK; idx += NT) {
      const int r = idx / DK, i = idx % DK;
      float aq = 0.f, at = 0.f, aw = 0.f;
#pragma unroll 8
      for (int j = 0; j < CW; ++j) {
        const float si = sSin[i * LS + j];
        aq += sdO[r * LS + j] * si;
        at += sR[r * LS + j] * sdSo[i * LS + j];
        aw += sdR[r * LS + j] * si;
      }
      sdQ[r * LD + i] += aq;
      sdKt[r * LD + i] += at;
      sdW[r * LD + i] -= aw;
    }
    if (tid < DK) {
      float acc = 0.f;
      for (int j = 0; j < CW; ++j) acc += sdSo[tid * LS + j] * sSin[tid * LS + j];
      s_dgC[tid] += acc;
    }
    // dA_qk += dO R^T (lower); dA += dR V^T
    for (int idx = tid; idx < CC * CC; idx += NT) {
      const int r = idx / CC, s = idx % CC;
      float aq = 0.f, aa = 0.f;
#pragma unroll 8
      for (int j = 0; j < CW; ++j) {
        aq += sdO[r * LS + j] * sR[s * LS + j];
        aa += sdR[r * LS + j] * sV[s * LS + j];
      }
      if (s <= r) sdAqk[r * LC + s] += aq;
      sdA[r * LC + s] += aa;
    }
    // dV = A^T dR
    for (int idx = tid; idx < CC * CW; idx += NT) {
      const int r = idx / CW, j = idx % CW, tt = c * CC + r;
      float acc = 0.f;
      for (int s = r; s < CC; ++s) acc += sA[s * LC + r] * sdR[s * LS + j];
      if (tt < a.T) sto(a.odt, a.dv_, tok_index(a, b, tt, h) * dv + j0 + j, acc);
    }
  }
  __syncthreads();
  // dA += dW Kbar^T;  dgamma_C += colsum(dK_tail (.) Kbar^kappa)
  for (int idx = tid; idx < CC * CC; idx += NT) {
    const int r = idx / CC, s = idx % CC;
    float acc = 0.f;
#pragma unroll 8
    for (int i = 0; i < DK; ++i) acc += sdW[r * LD + i] * sK[s * LD + i];
    sdA[r * LC + s] += acc;
  }
  if (tid < DK) {
    float acc = 0.f;
    for (int r = 0; r < CC; ++r) acc += sdKt[r * LD + tid] * sKk[r * LD + tid];
    s_dgC[tid] += acc;
  }
  __syncthreads();
  // dQbar += dA_qk Kbar^kappa; dKbar^kappa = dA_qk^T Qbar + gamma_C dK_tail (into sdKt);
  // dKbar = A^T dW (into sW); X = A^T dA (into sT)
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int r = idx / DK, i = idx % DK;
    float aq = 0.f, ak = 0.f, akb = 0.f;
    for (int s = 0; s <= r; ++s) aq += sdAqk[r * LC + s] * sKk[s * LD + i];
    for (int m = r; m < CC; ++m) {
      ak += sdAqk[m * LC + r] * sQ[m * LD + i];
      akb += sA[m * LC + r] * sdW[m * LD + i];
    }
    sdQ[r * LD + i] += aq;
    sdKt[r * LD + i] = ak + s_gC[i] * sdKt[r * LD + i];
    sW[r * LD + i] = akb;
  }
  for (int idx = tid; idx < CC * CC; idx += NT) {
    const int r = idx / CC, s = idx % CC;
    float acc = 0.f;
    for (int m = r; m < CC; ++m) acc += sA[m * LC + r] * sdA[m * LC + s];
    sT[r * LC + s] = acc;
  }
  __syncthreads();
  // dT = strict lower part of -X A^T (into sdA)
  for (int idx = tid; idx < CC * CC; idx += NT) {
    const int r = idx / CC, s = idx % CC;
    float acc = 0.f;
    if (s < r)
      for (int m = 0; m <= s; ++m) acc -= sT[r * LC + m] * sA[s * LC + m];
    sdA[r * LC + s] = acc;
  }
  __syncthreads();
  // dKbar += dT Kbar^kappa; dKbar^kappa += dT^T Kbar
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int r = idx / DK, i = idx % DK;
    float a1 = 0.f, a2 = 0.f;
    for (int s = 0; s < r; ++s) a1 += sdA[r * LC + s] * sKk[s * LD + i];
    for (int m = r + 1; m < CC; ++m) a2 += sdA[m * LC + r] * sK[m * LD + i];
    sW[r * LD + i] += a1;
    sdKt[r * LD + i] += a2;
  }
  __syncthreads();
  // Back through the scaling by gamma = exp(G): dq, the key/gain cotangents,
  // and dG (stored into sdQ).
  for (int idx = tid; idx < CC * DK; idx += NT) {
    const int t = idx / DK, i = idx % DK, tt = c * CC + t;
    const float gam = expf(sG[t * LD + i]);
    const float dKb = sW[t * LD + i], dKkb = sdKt[t * LD + i], dQb = sdQ[t * LD + i];
    float dG = dKb * sK[t * LD + i] - dKkb * sKk[t * LD + i] + dQb * sQ[t * LD + i];
    if (t == CC - 1) dG += s_dgC[i] * s_gC[i];
    if (tt < a.T) sto(a.odt, a.dq, tok_index(a, b, tt, h) * DK + i, a.tau * dQb * gam);
    sW[t * LD + i] = dKb * gam;       // dK from the memory path
    sdKt[t * LD + i] = dKkb / gam;    // d kappa
    sdQ[t * LD + i] = dG;
    sKk[t * LD + i] *= gam;           // kappa
  }
  __syncthreads();
  // reverse cumulative sum over the chunk: dg_j = sum_{r >= j} dG_r
  if (tid < DK) {
    float acc = 0.f;
    for (int t = CC - 1; t >= 0; --t) {
      acc += sdQ[t * LD + tid];
      sdQ[t * LD + tid] = acc;
    }
  }
  __syncthreads();
  // local part of the gain adjoint, one warp per token
  const int warp = tid / 32, lane = tid % 32;
  for (int t = warp; t < CC; t += NT / 32) {
    const int tt = c * CC + t;
    const size_t row = (size_t)bh * a.Tp + tt;
    float rr = 1.f;
    if (tt < a.T) rr = gate_r(a.gates, a.rmin, ld<DT>(a.r, tok_index(a, b, tt, h)));
    float kv[DK / 32];
#pragma unroll
    for (int m = 0; m < DK / 32; ++m) {
      const int i = lane + 32 * m;
      kv[m] = tt < a.T ? ld<DT>(a.k, tok_index(a, b, tt, h) * DK + i) : 0.f;
    }
    if (V == 0) {
      const float s = s_s[t];
      float cpart = 0.f;
#pragma unroll
      for (int m = 0; m < DK / 32; ++m) {
        const int i = lane + 32 * m;
        cpart += sdKt[t * LD + i] * sKk[t * LD + i];
      }
      const float ds = -warp_sum(cpart) / s;
#pragma unroll
      for (int m = 0; m < DK / 32; ++m) {
        const int i = lane + 32 * m;
        const float dkap = sdKt[t * LD + i];
        const float ph = a.phat[row * DK + i];
        a.dphloc[row * DK + i] = dkap * kv[m] / s + ds * kv[m] * kv[m];
        a.dkpart[row * DK + i] = sW[t * LD + i] + dkap * ph / s + 2.f * ds * ph * kv[m];
        a.dgpart[row * DK + i] = sdQ[t * LD + i];
      }
      if (lane == 0) a.drpart[row] = ds;
    } else {
      const float beta = s_s[t], n2 = s_n2[t];
      float bpart = 0.f;
#pragma unroll
      for (int m = 0; m < DK / 32; ++m) bpart += sdKt[t * LD + lane + 32 * m] * kv[m];
      const float dbeta = warp_sum(bpart);
      const float bhat = a.phat[row];
      const float den = rr + bhat * n2;
      const float dn2 = -dbeta * beta * beta;
#pragma unroll
      for (int m = 0; m < DK / 32; ++m) {
        const int i = lane + 32 * m;
        a.dkpart[row * DK + i] = sW[t * LD + i] + beta * sdKt[t * LD + i] + 2.f * kv[m] * dn2;
        a.dgpart[row * DK + i] = sdQ[t * LD + i];
      }
      if (lane == 0) {
        a.dphloc[row] = dbeta * rr / (den * den);
        a.drpart[row] = -dbeta * beta / den;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Adjoint of the uncertainty recursion, backwards in time.

template <typename DT>
__global__ void __launch_bounds__(32) k_gain_bwd_diag(Args a) {
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int lane = threadIdx.x, i = blockIdx.y * 32 + lane, dk = a.dk;
  float dp = a.dpT ? a.dpT[(size_t)bh * dk + i] : 0.f;
  float dmu_acc = 0.f;  // this channel's part of dL/dmu
  const size_t hrow = (size_t)bh * a.Tp;
  const float p_init = a.p0 ? a.p0[(size_t)bh * dk + i] : 1.f;
  // per token: phat, k, r, g, local dphat, dk and dg partials; blocks of GU
  // tokens walk backwards with the next (earlier) block prefetched
  float cph[GU], ck[GU], cr[GU], cg[GU], cdl[GU], cdk[GU], cdg[GU];
  auto load = [&](int t0, float *ph_, float *k_, float *r_, float *g_, float *dl_, float *dk_,
                  float *dg_) {
#pragma unroll
    for (int j = 0; j < GU; ++j) {
      const int t = t0 + j;
      ph_[j] = 0.f; k_[j] = 0.f; r_[j] = 1.f; g_[j] = 0.f; dl_[j] = 0.f; dk_[j] = 0.f; dg_[j] = 0.f;
      if (t >= 0 && t < a.T) {
        const size_t th = tok_index(a, b, t, h), row = hrow + t;
        ph_[j] = a.phat[row * dk + i];
        k_[j] = ld<DT>(a.k, th * dk + i);
        r_[j] = gate_r(a.gates, a.rmin, ld<DT>(a.r, th));
        g_[j] = gate_logalpha(a.gates, ld<DT>(a.g, th * dk + i));
        dl_[j] = a.dphloc[row * dk + i];
        dk_[j] = a.dkpart[row * dk + i];
        dg_[j] = a.dgpart[row * dk + i];
      }
    }
  };
  const int nblk = (a.T + GU - 1) / GU;
  int t0 = (nblk - 1) * GU;
  load(t0, cph, ck, cr, cg, cdl, cdk, cdg);
  for (; t0 >= 0; t0 -= GU) {
    float nph[GU], nk[GU], nr[GU], ng[GU], ndl[GU], ndk[GU], ndg[GU];
    load(t0 - GU, nph, nk, nr, ng, ndl, ndk, ndg);
    // posterior variance before the block: p_{t0-1}
    float pprev_block = p_init;
    if (t0 > 0) {
      const float u1 = a.mu * nk[GU - 1] * nk[GU - 1] / nr[GU - 1];
      pprev_block = nph[GU - 1] / (1.f + u1 * nph[GU - 1]);
    }
    // p_t for every token of the block (from phat_t and u_t)
    float pt[GU];
#pragma unroll
    for (int j = 0; j < GU; ++j) {
      const float u = a.mu * ck[j] * ck[j] / cr[j];
      pt[j] = cph[j] / (1.f + u * cph[j]);
    }
#pragma unroll
    for (int j = GU - 1; j >= 0; --j) {
      const int t = t0 + j;
      if (t < a.T) {
        const size_t th = tok_index(a, b, t, h), row = hrow + t;
        const float u = a.mu * ck[j] * ck[j] / cr[j];
        const float den = 1.f + u * cph[j];
        const float dph = dp / (den * den) + cdl[j];
        const float du = -dp * pt[j] * pt[j];
        dmu_acc += du * ck[j] * ck[j] / cr[j];  // u = mu k^2 / r
        const float dkk = cdk[j] + du * 2.f * a.mu * ck[j] / cr[j];
        const float drp = warp_sum(-du * u / cr[j]);
        if (lane == 0) a.drw[row * 4 + blockIdx.y] = drp;
        const float pprev = j > 0 ? pt[j - 1] : pprev_block;
        const float al2 = expf(2.f * cg[j]);
        // logit gates: d omega / dy = sigmoid(y), d log alpha / dx = 1 - alpha
        const float fw = a.gates ? sigmoid_f(ld<DT>(a.omega, th * dk + i)) : 1.f;
        const float fg = a.gates ? -expm1f(cg[j]) : 1.f;
        sto(a.odt, a.domega, th * dk + i, dph * fw);
        sto(a.odt, a.dg, th * dk + i, (cdg[j] + 2.f * al2 * pprev * dph) * fg);
        sto(a.odt, a.dk_, th * dk + i, dkk);
        dp = al2 * dph;
      }
    }
#pragma unroll
    for (int j = 0; j < GU; ++j) {
      cph[j] = nph[j]; ck[j] = nk[j]; cr[j] = nr[j]; cg[j] = ng[j];
      cdl[j] = ndl[j]; cdk[j] = ndk[j]; cdg[j] = ndg[j];
    }
  }
  if (a.dp0) a.dp0[(size_t)bh * dk + i] = dp;
  if (a.dmu) {
    dmu_acc = warp_sum(dmu_acc);
    if (lane == 0) atomicAdd(a.dmu + bh, dmu_acc);
  }
}

template <typename DT>
__global__ void k_finalize_dr_diag(Args a) {
  const size_t n = (size_t)a.B * a.H * a.T;
  const int nw = a.dk / 32;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
       e += (size_t)gridDim.x * blockDim.x) {
    const int bh = (int)(e / a.T), t = (int)(e % a.T);
    const size_t row = (size_t)bh * a.Tp + t;
    float acc = a.drpart[row];
    for (int w = 0; w < nw; ++w) acc += a.drw[row * 4 + w];
    const size_t th = tok_index(a, bh / a.H, t, bh % a.H);
    if (a.gates) acc *= sigmoid_f(ld<DT>(a.r, th));  // d r / dz
    sto(a.odt, a.dr, th, acc);
  }
}

template <typename DT>
__global__ void __launch_bounds__(32) k_gain_bwd_iso(Args a) {
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int lane = threadIdx.x;
  __shared__ float s_ph[33], s_a[33], s_n2[33], s_r[33], s_dl[32], s_dr[32], s_o1[32], s_o2[32], s_dw[32];
  float db = a.dpT ? a.dpT[bh] : 0.f;
  float dmu_acc = 0.f;  // dL/dmu of this sequence (lane 0)
  const size_t hrow = (size_t)bh * a.Tp;
  const int nblk = (a.T + 31) / 32;
  for (int blk = nblk - 1; blk >= 0; --blk) {
    const int t0 = blk * 32;
    // lane j stages token t0 + j; slot 32 holds token t0 - 1
    for (int j = lane; j < 33; j += 32) {
      const int t = j < 32 ? t0 + j : t0 - 1;
      float ph = 0.f, aa = 1.f, n2 = 0.f, rr = 1.f;
      if (t >= 0 && t < a.T) {
        const size_t row = hrow + t;
        ph = a.phat[row];
        aa = a.isotok[row * 2 + 0];
        n2 = a.isotok[row * 2 + 1];
        rr = gate_r(a.gates, a.rmin, ld<DT>(a.r, tok_index(a, b, t, h)));
        if (j < 32) {
          s_dl[j] = a.dphloc[row];
          s_dr[j] = a.drpart[row];
        }
      }
      s_ph[j] = ph; s_a[j] = aa; s_n2[j] = n2; s_r[j] = rr;
    }
    __syncwarp();
    if (lane == 0) {
      for (int j = 31; j >= 0; --j) {
        const int t = t0 + j;
        if (t >= a.T) continue;
        const float bhat = s_ph[j], rr = s_r[j];
        const float u = a.mu * s_n2[j] / (a.dk * rr);
        const float den = 1.f + u * bhat;
        const float bt = bhat / den;
        const float dbh = db / (den * den) + s_dl[j];
        const float du = -db * bt * bt;
        dmu_acc += du * s_n2[j] / (a.dk * rr);  // u = mu |k|^2 / (dk r)
        s_dr[j] += -du * u / rr;
        float bprev;
        if (j > 0 || t > 0) {
          const int jj = j > 0 ? j - 1 : 32;
          const float u1 = a.mu * s_n2[jj] / (a.dk * s_r[jj]);
          bprev = s_ph[jj] / (1.f + u1 * s_ph[jj]);
        } else {
          bprev = a.p0 ? a.p0[bh] : 1.f;
        }
        s_o1[j] = du * a.mu / (a.dk * rr);  // d|k|^2 through u
        s_o2[j] = bprev * dbh;              // d a_t
        s_dw[j] = dbh;
        db = s_a[j] * dbh;
      }
    }
    __syncwarp();
    {
      const int t = t0 + lane;
      if (t < a.T) {
        const size_t row = hrow + t;
        a.drpart[row] = s_dr[lane];
        a.isoadj[row * 2 + 0] = s_o1[lane];
        a.isoadj[row * 2 + 1] = s_o2[lane];
        const size_t th = tok_index(a, b, t, h);
        const float fw = a.gates ? sigmoid_f(ld<DT>(a.omega, th)) : 1.f;  // d omega / dy
        sto(a.odt, a.domega, th, s_dw[lane] * fw);
      }
    }
    __syncwarp();
  }
  if (lane == 0 && a.dp0) a.dp0[bh] = db;
  if (lane == 0 && a.dmu) atomicAdd(a.dmu + bh, dmu_acc);
}

// per token: dk += 2 k d|k|^2, dg += d a_t * d a_t / d g, dr -> output dtype
template <typename DT, int DK>
__global__ void __launch_bounds__(DK) k_finalize_iso(Args a) {
  const int e = blockIdx.x;  // token-head index over B*H*T
  const int bh = e / a.T, t = e % a.T, b = bh / a.H, h = bh % a.H;
  const int i = threadIdx.x;
  const size_t th = tok_index(a, b, t, h), row = (size_t)bh * a.Tp + t;
  const float dn2 = a.isoadj[row * 2 + 0], da = a.isoadj[row * 2 + 1];
  const float kk = ld<DT>(a.k, th * DK + i);
  sto(a.odt, a.dk_, th * DK + i, a.dkpart[row * DK + i] + 2.f * kk * dn2);
  if (a.pcd) {
    const float lal = gate_logalpha(a.gates, ld<DT>(a.g, th * DK + i));
    const float al2 = expf(2.f * lal);
    const float fg = a.gates ? -expm1f(lal) : 1.f;  // d log alpha / dx
    sto(a.odt, a.dg, th * DK + i, (a.dgpart[row * DK + i] + 2.f * al2 * da / DK) * fg);
  } else {
    __shared__ float red[DK / 32];
    float part = warp_sum(a.dgpart[row * DK + i]);
    if (i % 32 == 0) red[i / 32] = part;
    __syncthreads();
    if (i == 0) {
      float tot = 0.f;
      for (int w = 0; w < DK / 32; ++w) tot += red[w];
      const float lal = gate_logalpha(a.gates, ld<DT>(a.g, th));
      const float al2 = expf(2.f * lal);
      const float fg = a.gates ? -expm1f(lal) : 1.f;  // d log alpha / dx
      sto(a.odt, a.dg, th, (tot + 2.f * al2 * da) * fg);
    }
  }
  if (i == 0) {
    const float fr = a.gates ? sigmoid_f(ld<DT>(a.r, th)) : 1.f;  // d r / dz
    sto(a.odt, a.dr, th, a.drpart[row] * fr);
  }
}

// ---------------------------------------------------------------------------
// Launch helpers

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

template <int V, typename DT, int DK>
kdn_status_t fwd_impl(const Args &a, cudaStream_t s, bool save) {
  const int BH = a.B * a.H;
  if (V == 0) k_gain_scan_diag<DT><<<dim3(BH, DK / 32), 32, 0, s>>>(a);
  else k_gain_scan_iso<DT><<<BH, 32, 0, s>>>(a);
  const size_t ps = prep_smem_bytes<DK>();
  if (set_smem(k_chunk_prep<V, DT, DK>, ps) != cudaSuccess) return KDN_ERR_CUDA;
  k_chunk_prep<V, DT, DK><<<dim3(BH, a.NC), NT, ps, s>>>(a);
  const size_t ss = state_smem_bytes<DK>();
  if (set_smem(k_state_fwd<DT, DK>, ss) != cudaSuccess) return KDN_ERR_CUDA;
  k_state_fwd<DT, DK><<<dim3(BH, a.dv / CW), NT, ss, s>>>(a, save ? 1 : 0);
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

template <int V, typename DT, int DK>
kdn_status_t bwd_impl(const Args &a0, cudaStream_t s) {
  Args a = a0;
  a.o = nullptr;
  a.ST = nullptr;
  a.pT = nullptr;
  kdn_status_t st0 = fwd_impl<V, DT, DK>(a, s, true);
  if (st0 != KDN_OK) return st0;
  const int BH = a.B * a.H;
  const size_t ss = state_smem_bytes<DK>();
  if (set_smem(k_state_bwd<DT, DK>, ss) != cudaSuccess) return KDN_ERR_CUDA;
  k_state_bwd<DT, DK><<<dim3(BH, a.dv / CW), NT, ss, s>>>(a);
  const size_t cs = cbwd_smem_bytes<DK>();
  if (set_smem(k_chunk_bwd<V, DT, DK>, cs) != cudaSuccess) return KDN_ERR_CUDA;
  k_chunk_bwd<V, DT, DK><<<dim3(BH, a.NC), NT, cs, s>>>(a);
  if (V == 0) {
    k_gain_bwd_diag<DT><<<dim3(BH, DK / 32), 32, 0, s>>>(a);
    k_finalize_dr_diag<DT><<<1024, 256, 0, s>>>(a);
  } else {
    k_gain_bwd_iso<DT><<<BH, 32, 0, s>>>(a);
    k_finalize_iso<DT, DK><<<BH * a.T, DK, 0, s>>>(a);
  }
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

template <int V, typename DT>
kdn_status_t fwd_dk(const Args &a, cudaStream_t s, bool save) {
  switch (a.dk) {
    case 32: return fwd_impl<V, DT, 32>(a, s, save);
    case 64: return fwd_impl<V, DT, 64>(a, s, save);
    case 128: return fwd_impl<V, DT, 128>(a, s, save);
  }
  return KDN_ERR_UNSUPPORTED;
}

template <int V, typename DT>
kdn_status_t bwd_dk(const Args &a, cudaStream_t s) {
  switch (a.dk) {
    case 32: return bwd_impl<V, DT, 32>(a, s);
    case 64: return bwd_impl<V, DT, 64>(a, s);
    case 128: return bwd_impl<V, DT, 128>(a, s);
  }
  return KDN_ERR_UNSUPPORTED;
}

}  // namespace

int chunked_chunk_len() { return CC; }

int chunked_fwd_launches(const Args &) { return 3; }
int chunked_bwd_launches(const Args &a) { return chunked_fwd_launches(a) + 4; }

kdn_status_t launch_chunked_fwd(const Args &a, cudaStream_t s, bool save_states) {
  if (a.variant == 0)
    return a.dtype == KDN_BF16 ? fwd_dk<0, __nv_bfloat16>(a, s, save_states)
                               : fwd_dk<0, float>(a, s, save_states);
  return a.dtype == KDN_BF16 ? fwd_dk<1, __nv_bfloat16>(a, s, save_states)
                             : fwd_dk<1, float>(a, s, save_states);
}

kdn_status_t launch_chunked_bwd(const Args &a, cudaStream_t s) {
  if (a.variant == 0)
    return a.dtype == KDN_BF16 ? bwd_dk<0, __nv_bfloat16>(a, s) : bwd_dk<0, float>(a, s);
  return a.dtype == KDN_BF16 ? bwd_dk<1, __nv_bfloat16>(a, s) : bwd_dk<1, float>(a, s);
}

}  // namespace kdn
