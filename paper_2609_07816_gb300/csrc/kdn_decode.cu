// kdn_decode.cu -- one decode token of the Diagonal / Isotropic KDN for every
// (batch, head): the boxed update of Prop. 3 / Prop. 5 applied in place.
//
// The step is bound by HBM traffic on the float32 memory S (2 * dk * dv * 4
// bytes per head).  One CTA owns one head; its 8 warps split the dk rows and
// every lane holds a dv/32-wide strip of each of its rows in registers, so S
// is read once and written once.  Using
//   delta = v - (D S)^T k,   o = tau (D S)^T q + tau delta (kappa^T q),
//   S'    = D S + kappa delta^T,
// both reductions over rows come from the same read of S.
#include "kdn_internal.cuh"

namespace kdn {
namespace {

constexpr int DNT = 256;

template <int CPL> struct Vec;
template <> struct Vec<1> { using T = float; };
template <> struct Vec<2> { using T = float2; };
template <> struct Vec<4> { using T = float4; };

template <int CPL>
__device__ __forceinline__ void vload(const float *p, float *x) {
  typename Vec<CPL>::T v = *reinterpret_cast<const typename Vec<CPL>::T *>(p);
  const float *f = reinterpret_cast<const float *>(&v);
#pragma unroll
  for (int n = 0; n < CPL; ++n) x[n] = f[n];
}
template <int CPL>
__device__ __forceinline__ void vstore(float *p, const float *x) {
  typename Vec<CPL>::T v;
  float *f = reinterpret_cast<float *>(&v);
#pragma unroll
  for (int n = 0; n < CPL; ++n) f[n] = x[n];
  *reinterpret_cast<typename Vec<CPL>::T *>(p) = v;
}

// G: the gate inputs are logits (compile-time, so that post-activation inputs
// carry none of the activation code)
template <int V, typename DT, int DK, int DV, int G>
__global__ void __launch_bounds__(DNT) k_decode(Args a, float *S, float *P) {
  constexpr int RPW = DK / 8;   // rows per warp
  constexpr int CPL = DV / 32;  // columns per lane
  constexpr int NWK = DK / 32;  // warps that carry one key channel per lane
  __shared__ float s_ak[DK], s_aq[DK], s_al[DK], s_kap[DK];
  __shared__ float s_red[8][DV], s_red2[8][DV], s_delta[DV];
  __shared__ float s_part[4][4], s_sc[2];
  const int bh = blockIdx.x, tid = threadIdx.x, warp = tid / 32, lane = tid % 32;
  const size_t sb = (size_t)bh * DK * DV;
  float s[RPW][CPL];
#pragma unroll
  for (int m = 0; m < RPW; ++m) vload<CPL>(S + sb + (size_t)(warp * RPW + m) * DV + lane * CPL, s[m]);

  // gain (eq. kla-box-gain / eq. iso-kla-box-gain) and uncertainty update
  const size_t th = (size_t)bh;  // per-step inputs are [B,H,..]
  float kk = 0.f, qq = 0.f, al = 1.f, x0 = 0.f, x1 = 0.f, x2 = 0.f, ph = 0.f;
  if (tid < DK) {
    const int i = tid;
    kk = ld<DT>(a.k, th * DK + i);
    qq = ld<DT>(a.q, th * DK + i);
    const float gg = (V == 0 || a.pcd) ? ld<DT>(a.g, th * DK + i) : ld<DT>(a.g, th);
    al = G ? sigmoid_f(gg) : expf(gg);
    if (V == 0) {
      ph = al * al * P[(size_t)bh * DK + i] + gate_omega(G, ld<DT>(a.omega, th * DK + i));
      x0 = ph * kk * kk;  // -> sum phat k^2
      x1 = ph * kk * qq;  // -> sum phat k q
    } else {
      x0 = al * al;       // -> a_t * dk
      x1 = kk * kk;       // -> |k|^2
      x2 = kk * qq;       // -> k^T q
    }
    x0 = warp_sum(x0);
    x1 = warp_sum(x1);
    x2 = warp_sum(x2);
    if (lane == 0) { s_part[warp][0] = x0; s_part[warp][1] = x1; s_part[warp][2] = x2; }
  }
  __syncthreads();
  if (tid < DK) {
    float t0 = 0.f, t1 = 0.f, t2 = 0.f;
#pragma unroll
    for (int w = 0; w < NWK; ++w) { t0 += s_part[w][0]; t1 += s_part[w][1]; t2 += s_part[w][2]; }
    const int i = tid;
    const float rr = gate_r(G, a.rmin, ld<DT>(a.r, th));
    float kap, kq;
    if (V == 0) {
      const float sden = rr + t0;
      kap = ph * kk / sden;
      kq = t1 / sden;
      const float u = a.mu * kk * kk / rr;
      P[(size_t)bh * DK + i] = ph / (1.f + u * ph);
    } else {
      const float aa = a.pcd ? t0 / DK : al * al;
      const float bhat = aa * P[bh] + gate_omega(G, ld<DT>(a.omega, th));
      const float beta = bhat / (rr + bhat * t1);
      kap = beta * kk;
      kq = beta * t2;
      __syncwarp();
      if (i == 0) {
        const float u = a.mu * t1 / (DK * rr);
        s_sc[1] = bhat / (1.f + u * bhat);
      }
    }
    s_ak[i] = al * kk;
    s_aq[i] = al * qq;
    s_al[i] = al;
    s_kap[i] = kap;
    if (i == 0) s_sc[0] = kq;
  }
  __syncthreads();
  if (V == 1 && tid == 0) P[bh] = s_sc[1];

  // column sums of (D S)^T k and (D S)^T q over this warp's rows
  float pa[CPL], pb[CPL];
#pragma unroll
  for (int n = 0; n < CPL; ++n) { pa[n] = 0.f; pb[n] = 0.f; }
#pragma unroll
  for (int m = 0; m < RPW; ++m) {
    const int i = warp * RPW + m;
    const float ak = s_ak[i], aq = s_aq[i];
#pragma unroll
    for (int n = 0; n < CPL; ++n) { pa[n] += ak * s[m][n]; pb[n] += aq * s[m][n]; }
  }
#pragma unroll
  for (int n = 0; n < CPL; ++n) { s_red[warp][lane * CPL + n] = pa[n]; s_red2[warp][lane * CPL + n] = pb[n]; }
  __syncthreads();
  if (tid < DV) {
    const int j = tid;
    float sa = 0.f, sq = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) { sa += s_red[w][j]; sq += s_red2[w][j]; }
    const float delta = ld<DT>(a.v, th * DV + j) - sa;
    s_delta[j] = delta;
    sto(a.odt, a.o, th * DV + j, a.tau * (sq + delta * s_sc[0]));
  }
  __syncthreads();
  float dl[CPL];
#pragma unroll
  for (int n = 0; n < CPL; ++n) dl[n] = s_delta[lane * CPL + n];
#pragma unroll
  for (int m = 0; m < RPW; ++m) {
    const int i = warp * RPW + m;
    const float ali = s_al[i], kai = s_kap[i];
#pragma unroll
    for (int n = 0; n < CPL; ++n) s[m][n] = ali * s[m][n] + kai * dl[n];
    vstore<CPL>(S + sb + (size_t)i * DV + lane * CPL, s[m]);
  }
}

template <int V, typename DT, int DK, int G>
kdn_status_t dec_dv(const Args &a, float *S, float *P, cudaStream_t s) {
  const int BH = a.B * a.H;
  switch (a.dv) {
    case 32: k_decode<V, DT, DK, 32, G><<<BH, DNT, 0, s>>>(a, S, P); break;
    case 64: k_decode<V, DT, DK, 64, G><<<BH, DNT, 0, s>>>(a, S, P); break;
    case 128: k_decode<V, DT, DK, 128, G><<<BH, DNT, 0, s>>>(a, S, P); break;
    default: return KDN_ERR_UNSUPPORTED;
  }
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

template <int V, typename DT, int G>
kdn_status_t dec_dk(const Args &a, float *S, float *P, cudaStream_t s) {
  switch (a.dk) {
    case 32: return dec_dv<V, DT, 32, G>(a, S, P, s);
    case 64: return dec_dv<V, DT, 64, G>(a, S, P, s);
    case 128: return dec_dv<V, DT, 128, G>(a, S, P, s);
  }
  return KDN_ERR_UNSUPPORTED;
}

template <int V, typename DT>
kdn_status_t dec_gates(const Args &a, float *S, float *P, cudaStream_t s) {
  return a.gates ? dec_dk<V, DT, 1>(a, S, P, s) : dec_dk<V, DT, 0>(a, S, P, s);
}

}  // namespace

kdn_status_t launch_decode(const Args &a, float *S, float *P, cudaStream_t s) {
  if (a.variant == 0)
    return a.dtype == KDN_BF16 ? dec_gates<0, __nv_bfloat16>(a, S, P, s)
                               : dec_gates<0, float>(a, S, P, s);
  return a.dtype == KDN_BF16 ? dec_gates<1, __nv_bfloat16>(a, S, P, s)
                             : dec_gates<1, float>(a, S, P, s);
}

}  // namespace kdn
