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
//    and WY factor; only the state products are doubled) and writes both
//    outputs per token.  A short sequential pass over segments then gives every
//    segment's exact entry memory S_in(j).
//  * Output.  By the same linearity o_t = o_v,t + S_in(j)^T o_Phi,t: one dense
//    128 x 128 product per token on the tensor cores (k_seg_out).
//
// Cost: one fused run over T / P tokens (with a second state pass) instead of
// one over T, plus light passes over the gates and the outputs; used when
// P >= 4 segments of >= 8 chunks fit.
#include "kdn_internal.cuh"
#include "kdn_sm103.cuh"
#include "kdn_fused_common.cuh"

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

// Entry memory of every segment:  S_in(0) = S_0 (0 when absent), then
// S_in(j + 1) = Phi(j) S_in(j) + Sv(j), with Sv(j) the exit memory of segment j
// run from S_in = 0 with v and Phi(j) its exit memory from S = I with v = 0;
// S_in(P) is the final memory S_T (written when ST is given).  Columns of the
// memory are independent: a CTA owns 16 of them for one (batch, head); thread
// (row, half) holds 8 entries.
// Every S_in(j) also goes to `img` as the fp16 B operand of the output pass
// (32 KB per segment: two slabs of 64 value columns, rows = key channels,
// 128-byte swizzle), so that pass fetches it with one bulk copy.
__global__ void __launch_bounds__(256) k_seg_combine(const Args a, int P, const float *Sv,
                                                     const float *Sphi, float *ST,
                                                     unsigned char *img) {
  __shared__ __align__(16) float sS[D][16];
  const int bh = blockIdx.y, b = bh / a.H, h = bh % a.H;
  const int tid = threadIdx.x, row = tid >> 1, half = tid & 1;
  const int col = blockIdx.x * 16 + half * 8;
  auto ent = [&](int j) { return ((size_t)(b * P + j) * a.H + h) * D * D; };
  auto put_img = [&](int j, const float *x) {
    unsigned char *dst = img + ((size_t)(b * P + j) * a.H + h) * 32768;
    fused::sm16(dst, (col >> 6) * 16384 + fused::chunk_off(row, (col & 63) >> 3)) = fused::pack_h8(x);
  };
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (a.S0) {  // S_in(0) = S_0
    const float4 *src = reinterpret_cast<const float4 *>(a.S0 + ((size_t)bh * D + row) * D + col);
    const float4 x0 = src[0], x1 = src[1];
    acc[0] = x0.x; acc[1] = x0.y; acc[2] = x0.z; acc[3] = x0.w;
    acc[4] = x1.x; acc[5] = x1.y; acc[6] = x1.z; acc[7] = x1.w;
  }
  put_img(0, acc);
  for (int j = 0; j < P; ++j) {  // acc = S_in(j)
    if (j == P - 1 && !ST) break;
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
    if (j + 1 < P) {
      put_img(j + 1, acc);
    } else {
      float4 *dst = reinterpret_cast<float4 *>(ST + (size_t)bh * D * D + (size_t)row * D + col);
      dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
      dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    }
  }
}

// Exact output of every token:  o_t = o_v,t + S_in(j)^T o_Phi,t, with o_v the
// output of the run from S_in = 0 with v, o_Phi,t = tau Phi_t^T q_t that of the
// transition run, and S_in(j) the entry memory of the token's segment j (the
// recurrence is linear in S_in).  One CTA per (128-token tile, head, batch):
// TMA brings the o_Phi tile (fp16, K-major A) and a bulk copy the fp16 image of
// S_in(j) (MN-major B, written by k_seg_combine); eight tcgen05 MMAs
// (M = N = 128, K = 16 each) form o_Phi S_in in TMEM.  With float32 o (which
// then already holds o_v) the epilogue stages the product and a TMA reduce-add
// adds it to o; with bf16 o it loads o_v from the workspace, adds, rounds and
// stores.  Segments are whole 64-token chunks, so a tile whose second half
// starts a new segment also forms o_Phi S_in(j + 1) for that half.  96 KB of
// shared memory and 256 TMEM columns: two CTAs per SM.
constexpr int kOutT = 128, kOutThreads = 128;
constexpr int kOutSmem = 32768 + 65536 + 64 + 1024;
constexpr uint32_t kOutWait = 1u << 25;

__global__ void __launch_bounds__(kOutThreads, 2)
    k_seg_out(const __grid_constant__ CUtensorMap m_ophi, const __grid_constant__ CUtensorMap m_ov,
              const __grid_constant__ CUtensorMap m_o, const Args a, int P,
              const unsigned char *img) {
  using namespace sm103;
  using namespace fused;
  extern __shared__ unsigned char smraw[];
  unsigned char *sm =
      reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  unsigned char *sA = sm, *sB = sm + 32768;  // after the MMAs: [0, 64K) float32 staging,
                                             // [64K, 96K) bf16 staging
  uint64_t *bars = reinterpret_cast<uint64_t *>(sm + 98304);
  uint64_t *bar_a = bars, *bar_o = bars + 1, *bar_m = bars + 2;
  uint32_t *s_tbase = reinterpret_cast<uint32_t *>(bars + 4);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int t0 = blockIdx.x * kOutT, h = blockIdx.y, b = blockIdx.z;
  const bool obf = a.odt == KDN_BF16;
  // segments of the two 64-token halves (a last tile may hold only the first;
  // the TMA fills and clips the tokens past T)
  const int seg = t0 / (a.T / P), seg2 = t0 + 64 < a.T ? (t0 + 64) / (a.T / P) : seg;
  const bool two = seg2 != seg;
  if (tid == 0) {
    mbar_init(bar_a, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_m, 1);
    fence_mbar_init();
    mbar_expect_tx(bar_a, 32768u * (two ? 3 : 2));
    for (int sl = 0; sl < 2; ++sl)
      for (int th = 0; th < 2; ++th)  // slab sl: rows 0..63 (th 0), 64..127 (th 1)
        tma_load_4d(sA + sl * 16384 + th * 8192, &m_ophi, bar_a, 64 * sl, h, t0 + 64 * th, b);
    for (int u = 0; u < (two ? 2 : 1); ++u)
      bulk_g2s(sB + u * 32768, img + ((size_t)(b * P + seg + u) * a.H + h) * 32768, 32768, bar_a);
  }
  if (warp == 0) {
    tmem_alloc(s_tbase, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tb = *s_tbase;
  bool ok = true, o_issued = false;
  if (tid == 0) {
    ok = mbar_wait(bar_a, 0, kOutWait);
    if (ok) {
      const uint32_t id = idesc_f16(128, 128, 0, 1), A = smem_u32(sA), B = smem_u32(sB);
      for (int u = 0; u < (two ? 2 : 1); ++u)
        for (int kk = 0; kk < 8; ++kk)
          umma_bf16(tb + 128 * u, sw128_desc(A + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                    sw128_desc(B + u * 32768 + kk * 2048, 16384, 1024), id, kk > 0);
      umma_commit(bar_m);
      ok = mbar_wait(bar_m, 0, kOutWait);
      if (ok && obf) {  // o_v (float32, workspace) over the operands the MMAs have read
        mbar_expect_tx(bar_o, 65536);
        o_issued = true;
        for (int bx = 0; bx < 4; ++bx)
          for (int th = 0; th < 2; ++th)
            tma_load_4d(sm + (bx * 2 + th) * 8192, &m_ov, bar_o, 32 * bx, h, t0 + 64 * th, b);
        ok = mbar_wait(bar_o, 0, kOutWait);
      }
    }
  }
  ok = __syncthreads_and(ok);
  if (ok) {
    tc_fence_after();
    // token t = tid: TMEM lane t; float32 row t % 64 of box (column group, t / 64)
    const int t = tid, r = t & 63, th = t >> 6;
    const uint32_t acc = tb + ((two && th) ? 128u : 0u);  // the second half's segment
    for (int j0 = 0; j0 < D; j0 += 16) {
      float v[16];
      tmem_ld16(acc + ((uint32_t)(32 * warp) << 16) + j0, v);
      const int bx = j0 >> 5, cc = (j0 & 31) >> 2;
      unsigned char *box = sm + (bx * 2 + th) * 8192;
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        uint4 &u = sm16(box, chunk_off(r, cc + m));
        if (obf) {
          v[4 * m] += __uint_as_float(u.x);
          v[4 * m + 1] += __uint_as_float(u.y);
          v[4 * m + 2] += __uint_as_float(u.z);
          v[4 * m + 3] += __uint_as_float(u.w);
        } else {
          u = make_uint4(__float_as_uint(v[4 * m]), __float_as_uint(v[4 * m + 1]),
                         __float_as_uint(v[4 * m + 2]), __float_as_uint(v[4 * m + 3]));
        }
      }
      if (obf) {  // boxes of 64 bf16 columns
        const int bb = j0 >> 6, c2 = (j0 & 63) >> 3;
        unsigned char *ob = sm + 65536 + (bb * 2 + th) * 8192;
        sm16(ob, chunk_off(r, c2)) = pack_bf8(v);
        sm16(ob, chunk_off(r, c2 + 1)) = pack_bf8(v + 8);
      }
    }
    fence_proxy_async();
  }
  __syncthreads();
  if (tid == 0) {
    if (ok) {
      if (obf) {
        for (int bb = 0; bb < 2; ++bb)
          for (int th = 0; th < 2; ++th)
            tma_store_4d(&m_o, sm + 65536 + (bb * 2 + th) * 8192, 64 * bb, h, t0 + 64 * th, b);
      } else {  // o += o_Phi S_in
        for (int bx = 0; bx < 4; ++bx)
          for (int th = 0; th < 2; ++th)
            tma_add_4d(&m_o, sm + (bx * 2 + th) * 8192, 32 * bx, h, t0 + 64 * th, b);
      }
      bulk_commit();
      bulk_wait_all();
    } else {
      atomicExch(a.status, (unsigned)KDN_ERR_TIMEOUT);
      mbar_wait(bar_a, 0, kOutWait);  // copies in flight land before the CTA leaves
      if (o_issued) mbar_wait(bar_o, 0, kOutWait);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tb, 256);
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
  const size_t ntok = (size_t)a.B * a.T * a.H * D;  // o_Phi (fp16); o_v (fp32) unless o is
  return r(BH * NC * Pn * 16) + r(BH * P * Pn * 4) * 2 + r(BH * P * D * D * 4) * 2 +
         r(BH * P * 32768) + r(ntok * 2) + (a.odt == KDN_BF16 ? r(ntok * 4) : 0);
}

kdn_status_t launch_seg_fwd(const Args &a, int P, char *ws, cudaStream_t s) {
  const size_t BH = (size_t)a.B * a.H, Pn = a.variant == 0 ? D : 1, NC = a.T / CM;
  const size_t nS = (size_t)D * D;
  auto r = [](size_t x) { return (x + 255) / 256 * 256; };
  char *p = ws;
  float4 *comp = reinterpret_cast<float4 *>(p); p += r(BH * NC * Pn * 16);
  float *pseg = reinterpret_cast<float *>(p); p += r(BH * P * Pn * 4);
  float *pbuf = reinterpret_cast<float *>(p); p += r(BH * P * Pn * 4);
  float *Sv = reinterpret_cast<float *>(p); p += r(BH * P * nS * 4);
  float *Sphi = reinterpret_cast<float *>(p); p += r(BH * P * nS * 4);
  unsigned char *img = reinterpret_cast<unsigned char *>(p); p += r(BH * P * 32768);
  const size_t ntok = (size_t)a.B * a.T * a.H * D;
  void *ophi = p; p += r(ntok * 2);
  // output of the run from S_in = 0: float32, in o itself unless o is bf16
  float *ov = a.odt == KDN_BF16 ? reinterpret_cast<float *>(p) : static_cast<float *>(a.o);


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

  // (1) the segments as B * P sequences of T / P tokens, in one pass that carries
  // two memories: from S_in = 0 with v, and from S = I with v = 0 (the
  // transition Phi), with both outputs per token
  Args sa = a;
  sa.B = a.B * P;
  sa.T = a.T / P;
  sa.NC = (sa.T + a.C - 1) / a.C;
  sa.Tp = sa.NC * a.C;
  sa.p0 = pseg;
  sa.S0 = nullptr;  // every segment from S_in = 0; S_0 enters through the join
  sa.ST = Sv;
  sa.o = ov;
  sa.odt = KDN_F32;
  sa.pT = a.pT ? pbuf : nullptr;
  kdn_status_t st = launch_fused_fwd(sa, s, nullptr, nullptr, true, Sphi, ophi);
  if (st != KDN_OK) return st;
  // (2) exact entry memories (as fp16 operand images) from S_in(0) = S_0, and the final one
  k_seg_combine<<<dim3(D / 16, (unsigned)BH), 256, 0, s>>>(a, P, Sv, Sphi, a.ST, img);
  if (cudaGetLastError() != cudaSuccess) return KDN_ERR_CUDA;
  // (3) exact outputs o = o_v + S_in^T o_Phi
  CUtensorMap m_ophi, m_ov, m_o;
  if (!fused::make_map(&m_ophi, ophi, a, false, true) || !fused::make_map(&m_ov, ov, a, true) ||
      !fused::make_map(&m_o, a.o, a, a.odt != KDN_BF16))
    return KDN_ERR_CUDA;
  if (cudaFuncSetAttribute(k_seg_out, cudaFuncAttributeMaxDynamicSharedMemorySize, kOutSmem) !=
      cudaSuccess)
    return KDN_ERR_CUDA;
  k_seg_out<<<dim3((unsigned)((a.T + kOutT - 1) / kOutT), (unsigned)a.H, (unsigned)a.B), kOutThreads, kOutSmem,
              s>>>(m_ophi, m_ov, m_o, a, P, img);
  if (cudaGetLastError() != cudaSuccess) return KDN_ERR_CUDA;
  const size_t seqP = (size_t)a.H * Pn;
  if (a.pT && cudaMemcpy2DAsync(a.pT, seqP * 4, pbuf + (size_t)(P - 1) * seqP, (size_t)P * seqP * 4,
                                seqP * 4, a.B, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KDN_ERR_CUDA;
  return KDN_OK;
}

}  // namespace kdn
