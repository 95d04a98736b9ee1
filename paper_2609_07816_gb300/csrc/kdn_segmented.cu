// kdn_segmented.cu -- sequence-parallel forward for a few long sequences.
//
// The fused forward walks the chunks of one (batch, head) in one CTA, so with
// B*H far below the SM count most of the GPU idles (one long sequence per head).
// Here every sequence is cut into P segments of whole 64-token chunks that run
// as B*P "virtual" sequences of the fused kernel, and the pieces are joined
// exactly:
//
//  * Uncertainty.  One token's update of p (Prop. 3; Prop. 5 for the scalar b)
//    is a Moebius map, a 2x2 matrix on homogeneous coordinates (n, d) with
//    p = n / d:  M_t = [[a_t, omega_t], [u_t a_t, 1 + u_t omega_t]], a_t = alpha_t^2
//    (iso: the mean of alpha_t^2 over channels), u_t = mu k_t^2 / r_t (iso:
//    mu |k_t|^2 / (d_k r_t)).  The ordered product of a chunk's 64 matrices
//    summarises the chunk (the associative form of the uncertainty scan); a scan
//    over chunk summaries gives the uncertainty entering every segment.
//  * Memory.  With the gains fixed, the chunked recurrence (App. F) is linear in
//    (S_in, v) jointly, so a segment's exit memory is Phi S_in + S_out|(S_in = 0),
//    where the transition Phi (d_k x d_k) is the exit memory of a run from S = I
//    with v = 0.  One fused pass carries both memories (they share every gain
//    and WY factor; only the state products are doubled).  A short sequential
//    pass over segments then gives every segment's exact entry memory, and a last
//    run of all segments writes o.
//
// Cost: two fused runs over T / P tokens instead of one over T (the first with
// a second state pass), plus two light passes over the gates; used when P >= 4
// segments of >= 8 chunks fit.
#include "kdn_internal.cuh"

namespace kdn {
namespace {

constexpr int D = 128;       // d_k = d_v served by the fused kernels
constexpr int CM = 64;       // their chunk length
constexpr int kSegCtas = 152;  // one CTA per SM of a GB300 (152 SMs)
constexpr int kMinSegChunks = 8;

using bf16 = __nv_bfloat16;

// Diagonal KDN: per (chunk, batch*head) and channel, the ordered product of the
// chunk's 64 token matrices (later tokens on the left), renormalised by its
// largest entry every 4 tokens (all entries are non-negative).  One warp per
// chunk, four adjacent channels per lane (8-byte loads of a 256-byte row).
constexpr int kCompWarps = 4;
template <int G>  // G: logit gates (compile-time)
__global__ void __launch_bounds__(32 * kCompWarps) k_seg_comp_diag(const Args a, float4 *comp) {
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * kCompWarps + (threadIdx.x >> 5), bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H, i0 = 4 * lane;
  const int NC = a.T / CM;
  if (c >= NC) return;
  float m[4][4];
#pragma unroll
  for (int q = 0; q < 4; ++q) { m[q][0] = 1.f; m[q][1] = 0.f; m[q][2] = 0.f; m[q][3] = 1.f; }
  const bf16 *kb = static_cast<const bf16 *>(a.k), *gb = static_cast<const bf16 *>(a.g);
  const bf16 *wb = static_cast<const bf16 *>(a.omega);
  for (int t0 = 0; t0 < CM; t0 += 4) {
    uint2 kr[4], gr[4], wr[4];
    float rr[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const size_t th = tok_index(a, b, c * CM + t0 + u, h);
      kr[u] = *reinterpret_cast<const uint2 *>(kb + th * D + i0);
      gr[u] = *reinterpret_cast<const uint2 *>(gb + th * D + i0);
      wr[u] = *reinterpret_cast<const uint2 *>(wb + th * D + i0);
      rr[u] = a.mu / gate_r(G, a.rmin, ld<bf16>(a.r, th));
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&kr[u].x));
      const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&kr[u].y));
      const float2 g01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&gr[u].x));
      const float2 g23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&gr[u].y));
      const float2 w01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&wr[u].x));
      const float2 w23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&wr[u].y));
      const float kv[4] = {k01.x, k01.y, k23.x, k23.y}, gv[4] = {g01.x, g01.y, g23.x, g23.y};
      const float wv[4] = {w01.x, w01.y, w23.x, w23.y};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float al2, w;
        if (G) {
          const float al = sigmoid_f(gv[q]);
          al2 = al * al;
          w = softplus_f(wv[q]);
        } else {
          al2 = __expf(2.f * gv[q]);
          w = wv[q];
        }
        const float uu = rr[u] * kv[q] * kv[q];
        // rows of M_t: [al2, w] and u * [al2, w] + [0, 1]
        const float n00 = al2 * m[q][0] + w * m[q][2];
        const float n01 = al2 * m[q][1] + w * m[q][3];
        m[q][2] = fmaf(uu, n00, m[q][2]);
        m[q][3] = fmaf(uu, n01, m[q][3]);
        m[q][0] = n00;
        m[q][1] = n01;
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) renorm4(m[q][0], m[q][1], m[q][2], m[q][3]);
  }
  float4 *dst = comp + ((size_t)bh * NC + c) * D + i0;
#pragma unroll
  for (int q = 0; q < 4; ++q) dst[q] = make_float4(m[q][0], m[q][1], m[q][2], m[q][3]);
}

// Isotropic KDN: one thread per token forms M_t; the 64 matrices are multiplied
// in order by a shuffle tree within each warp, then the two warp products.
template <int G>  // G: logit gates (compile-time)
__global__ void __launch_bounds__(CM) k_seg_comp_iso(const Args a, float4 *comp) {
  const int c = blockIdx.x, bh = blockIdx.y, b = bh / a.H, h = bh % a.H;
  const int tid = threadIdx.x, lane = tid & 31;
  const int NC = a.T / CM;
  const size_t th = tok_index(a, b, c * CM + tid, h);
  float n2 = 0.f, al2 = 0.f;
  const uint4 *kr = reinterpret_cast<const uint4 *>(static_cast<const bf16 *>(a.k) + th * D);
#pragma unroll 4
  for (int e = 0; e < D / 8; ++e) {
    const uint4 x = kr[e];
    const uint32_t wv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&wv[q]));
      n2 = fmaf(f.x, f.x, n2);
      n2 = fmaf(f.y, f.y, n2);
    }
  }
  if (a.pcd) {
    const uint4 *gr = reinterpret_cast<const uint4 *>(static_cast<const bf16 *>(a.g) + th * D);
#pragma unroll 4
    for (int e = 0; e < D / 8; ++e) {
      const uint4 x = gr[e];
      const uint32_t wv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&wv[q]));
        if (G) {
          const float ax = sigmoid_f(f.x), ay = sigmoid_f(f.y);
          al2 += ax * ax + ay * ay;
        } else {
          al2 += __expf(2.f * f.x) + __expf(2.f * f.y);
        }
      }
    }
    al2 *= 1.f / D;
  } else {
    const float x = ld<bf16>(a.g, th);
    if (G) {
      const float al = sigmoid_f(x);
      al2 = al * al;
    } else {
      al2 = __expf(2.f * x);
    }
  }
  const float w = gate_omega(G, ld<bf16>(a.omega, th));
  const float r = gate_r(G, a.rmin, ld<bf16>(a.r, th));
  const float uu = a.mu * n2 / ((float)a.dk * r);
  float m00 = al2, m01 = w, m10 = uu * al2, m11 = fmaf(uu, w, 1.f);
  renorm4(m00, m01, m10, m11);
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    // lane l (l % 2off == 0) holds tokens [l, l + off); the partner the next off
    const float p00 = __shfl_down_sync(0xffffffffu, m00, off);
    const float p01 = __shfl_down_sync(0xffffffffu, m01, off);
    const float p10 = __shfl_down_sync(0xffffffffu, m10, off);
    const float p11 = __shfl_down_sync(0xffffffffu, m11, off);
    if ((lane & (2 * off - 1)) == 0) {
      float n00 = p00 * m00 + p01 * m10, n01 = p00 * m01 + p01 * m11;
      float n10 = p10 * m00 + p11 * m10, n11 = p10 * m01 + p11 * m11;
      renorm4(n00, n01, n10, n11);
      m00 = n00; m01 = n01; m10 = n10; m11 = n11;
    }
  }
  __shared__ float4 s_w[2];
  if (lane == 0) s_w[tid >> 5] = make_float4(m00, m01, m10, m11);
  __syncthreads();
  if (tid == 0) {
    const float4 lo = s_w[0], hi = s_w[1];
    float n00 = hi.x * lo.x + hi.y * lo.z, n01 = hi.x * lo.y + hi.y * lo.w;
    float n10 = hi.z * lo.x + hi.w * lo.z, n11 = hi.z * lo.y + hi.w * lo.w;
    renorm4(n00, n01, n10, n11);
    comp[(size_t)bh * NC + c] = make_float4(n00, n01, n10, n11);
  }
}

// Uncertainty entering every segment, stored as the initial uncertainty of its
// virtual sequence (b * P + j, h).  Two levels: threads (entry, group) multiply
// the chunk summaries of segments group, group + 8, ... in order (the loads of 8
// chunks issued ahead of their dependent products) and store each segment's
// product over the summary of its first chunk, which only they read; then one
// thread per entry (channel for diag, head for iso) runs the segment products
// from p_0 (or 1).
constexpr int kScanGroups = 8;
__global__ void __launch_bounds__(D * kScanGroups) k_seg_scan(const Args a, float4 *comp,
                                                              int nseg, float *pseg) {
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int i = threadIdx.x % D, grp = threadIdx.x / D;
  const int Pn = a.variant == 0 ? D : 1;
  const int NC = a.T / CM, P = NC / nseg;
  float4 *cm = comp + (size_t)bh * NC * Pn + i;
  if (i < Pn) {
    for (int j = grp; j < P; j += kScanGroups) {
      float m00 = 1.f, m01 = 0.f, m10 = 0.f, m11 = 1.f;
      const int end = (j + 1) * nseg;
      for (int c0 = j * nseg; c0 < end; c0 += 8) {
        float4 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          x[u] = c0 + u < end ? cm[(size_t)(c0 + u) * Pn] : make_float4(1.f, 0.f, 0.f, 1.f);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float n00 = fmaf(x[u].x, m00, x[u].y * m10), n01 = fmaf(x[u].x, m01, x[u].y * m11);
          const float n10 = fmaf(x[u].z, m00, x[u].w * m10), n11 = fmaf(x[u].z, m01, x[u].w * m11);
          m00 = n00; m01 = n01; m10 = n10; m11 = n11;
        }
        renorm4(m00, m01, m10, m11);
      }
      cm[(size_t)j * nseg * Pn] = make_float4(m00, m01, m10, m11);
    }
  }
  __syncthreads();
  if (grp != 0 || i >= Pn) return;
  float z0 = a.p0 ? a.p0[(size_t)bh * Pn + i] : 1.f, z1 = 1.f;
  for (int j = 0; j < P; ++j) {
    pseg[((size_t)(b * P + j) * a.H + h) * Pn + i] = z0 / z1;
    const float4 x = cm[(size_t)j * nseg * Pn];
    const float n = fmaf(x.x, z0, x.y * z1), d = fmaf(x.z, z0, x.w * z1);
    const float inv = 1.f / fmaxf(fabsf(n), fabsf(d));
    z0 = n * inv;
    z1 = d * inv;
  }
}

// Entry memory of every segment j >= 1:  S_in(1) = Sv(0),
// S_in(j + 1) = Phi(j) S_in(j) + Sv(j), with Sv(j) the exit memory of the run
// from S_in = 0 (the true S_0 for j = 0) and Phi(j) the exit memory of the run
// from S = I with v = 0.  Columns of the memory are independent: a CTA owns 16
// of them for one (batch, head); thread (row, half) holds 8 entries.
__global__ void __launch_bounds__(256) k_seg_combine(const Args a, int P, const float *Sv,
                                                     const float *Sphi, float *S0seg) {
  __shared__ __align__(16) float sS[D][16];
  const int bh = blockIdx.y, b = bh / a.H, h = bh % a.H;
  const int tid = threadIdx.x, row = tid >> 1, half = tid & 1;
  const int col = blockIdx.x * 16 + half * 8;
  auto ent = [&](int j) { return ((size_t)(b * P + j) * a.H + h) * D * D; };
  float acc[8];
  {
    const float4 *src = reinterpret_cast<const float4 *>(Sv + ent(0) + (size_t)row * D + col);
    const float4 x0 = src[0], x1 = src[1];
    acc[0] = x0.x; acc[1] = x0.y; acc[2] = x0.z; acc[3] = x0.w;
    acc[4] = x1.x; acc[5] = x1.y; acc[6] = x1.z; acc[7] = x1.w;
  }
  for (int j = 1; j < P; ++j) {
    float4 *dst = reinterpret_cast<float4 *>(S0seg + ent(j) + (size_t)row * D + col);
    dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    if (j == P - 1) break;
#pragma unroll
    for (int u = 0; u < 8; ++u) sS[row][half * 8 + u] = acc[u];
    __syncthreads();
    const float4 *sv = reinterpret_cast<const float4 *>(Sv + ent(j) + (size_t)row * D + col);
    const float4 y0 = sv[0], y1 = sv[1];
    acc[0] = y0.x; acc[1] = y0.y; acc[2] = y0.z; acc[3] = y0.w;
    acc[4] = y1.x; acc[5] = y1.y; acc[6] = y1.z; acc[7] = y1.w;
    const float4 *phi = reinterpret_cast<const float4 *>(Sphi + ent(j) + (size_t)row * D);
#pragma unroll 4
    for (int k4 = 0; k4 < D / 4; ++k4) {
      const float4 f = phi[k4];
      const float fv[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float4 s0 = *reinterpret_cast<const float4 *>(&sS[4 * k4 + q][half * 8]);
        const float4 s1 = *reinterpret_cast<const float4 *>(&sS[4 * k4 + q][half * 8 + 4]);
        acc[0] = fmaf(fv[q], s0.x, acc[0]); acc[1] = fmaf(fv[q], s0.y, acc[1]);
        acc[2] = fmaf(fv[q], s0.z, acc[2]); acc[3] = fmaf(fv[q], s0.w, acc[3]);
        acc[4] = fmaf(fv[q], s1.x, acc[4]); acc[5] = fmaf(fv[q], s1.y, acc[5]);
        acc[6] = fmaf(fv[q], s1.z, acc[6]); acc[7] = fmaf(fv[q], s1.w, acc[7]);
      }
    }
    __syncthreads();
  }
}

}  // namespace

int seg_count(const Args &a) {
  if (!fused_fwd_supported(a) || a.chunk == 32 || a.T % CM) return 1;
  const int nc = a.T / CM;
  const long long bh = (long long)a.B * a.H;
  int best = 1;
  for (int p = 4; p * kMinSegChunks <= nc; ++p)
    if (nc % p == 0 && bh * p <= kSegCtas) best = p;
  return best;
}

size_t seg_workspace_bytes(const Args &a, int P) {
  const size_t BH = (size_t)a.B * a.H, Pn = a.variant == 0 ? D : 1, NC = a.T / CM;
  auto r = [](size_t x) { return (x + 255) / 256 * 256; };
  return r(BH * NC * Pn * 16) + r(BH * P * Pn * 4) * 2 + r(BH * P * D * D * 4) * 3;
}

kdn_status_t launch_seg_fwd(const Args &a, int P, char *ws, cudaStream_t s) {
  const size_t BH = (size_t)a.B * a.H, Pn = a.variant == 0 ? D : 1, NC = a.T / CM;
  const size_t nS = (size_t)D * D, seqS = (size_t)a.H * nS;
  auto r = [](size_t x) { return (x + 255) / 256 * 256; };
  char *p = ws;
  float4 *comp = reinterpret_cast<float4 *>(p); p += r(BH * NC * Pn * 16);
  float *pseg = reinterpret_cast<float *>(p); p += r(BH * P * Pn * 4);
  float *pbuf = reinterpret_cast<float *>(p); p += r(BH * P * Pn * 4);
  float *S0seg = reinterpret_cast<float *>(p); p += r(BH * P * nS * 4);
  float *Sv = reinterpret_cast<float *>(p); p += r(BH * P * nS * 4);
  float *Sphi = reinterpret_cast<float *>(p);

  if (cudaMemsetAsync(S0seg, 0, BH * P * nS * 4, s) != cudaSuccess) return KDN_ERR_CUDA;
  if (a.S0 && cudaMemcpy2DAsync(S0seg, (size_t)P * seqS * 4, a.S0, seqS * 4, seqS * 4, a.B,
                                cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KDN_ERR_CUDA;

  // uncertainty entering every segment
  const dim3 gc((unsigned)NC, (unsigned)BH);
  if (a.variant == 0)
    (a.gates ? k_seg_comp_diag<1> : k_seg_comp_diag<0>)
        <<<dim3((unsigned)((NC + kCompWarps - 1) / kCompWarps), (unsigned)BH), 32 * kCompWarps,
           0, s>>>(a, comp);
  else
    (a.gates ? k_seg_comp_iso<1> : k_seg_comp_iso<0>)<<<gc, CM, 0, s>>>(a, comp);
  k_seg_scan<<<(unsigned)BH, D * kScanGroups, 0, s>>>(a, comp, (int)(NC / P), pseg);
  if (cudaGetLastError() != cudaSuccess) return KDN_ERR_CUDA;

  // the segments as B * P sequences of T / P tokens
  Args sa = a;
  sa.B = a.B * P;
  sa.T = a.T / P;
  sa.NC = (sa.T + a.C - 1) / a.C;
  sa.Tp = sa.NC * a.C;
  sa.p0 = pseg;
  sa.o = nullptr;
  sa.pT = nullptr;
  // (1) one pass carries two memories through every segment: from S_in = 0 (S_0
  // for the first segment) with v, and from S = I with v = 0 (the transition Phi)
  sa.S0 = S0seg;
  sa.ST = Sv;
  kdn_status_t st = launch_fused_fwd(sa, s, nullptr, nullptr, false, Sphi);
  if (st != KDN_OK) return st;
  // exact entry memories
  k_seg_combine<<<dim3(D / 16, (unsigned)BH), 256, 0, s>>>(a, P, Sv, Sphi, S0seg);
  if (cudaGetLastError() != cudaSuccess) return KDN_ERR_CUDA;
  // (2) every segment from its exact entry state: o, and the final state
  sa.S0 = S0seg;
  sa.o = a.o;
  sa.ST = a.ST ? Sphi : nullptr;
  sa.pT = a.pT ? pbuf : nullptr;
  st = launch_fused_fwd(sa, s);
  if (st != KDN_OK) return st;
  if (a.ST && cudaMemcpy2DAsync(a.ST, seqS * 4, Sphi + (size_t)(P - 1) * seqS, (size_t)P * seqS * 4,
                                seqS * 4, a.B, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KDN_ERR_CUDA;
  const size_t seqP = (size_t)a.H * Pn;
  if (a.pT && cudaMemcpy2DAsync(a.pT, seqP * 4, pbuf + (size_t)(P - 1) * seqP, (size_t)P * seqP * 4,
                                seqP * 4, a.B, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KDN_ERR_CUDA;
  return KDN_OK;
}

}  // namespace kdn
