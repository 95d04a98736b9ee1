// kdn_fused_fwd.cu -- fused chunked forward of the Diagonal / Isotropic KDN
// for bfloat16 activations with d_k = d_v = 128 and memory chunks of C = 64
// tokens (App. F), on the tcgen05 tensor cores of sm_103a.
//
// One CTA owns one (batch, head) and walks its chunks in order.  The memory S
// (128 x 128 float32) stays in tensor memory (TMEM) for the whole sequence;
// every activation tile is read from HBM once by TMA and o is written once.
// Per chunk (notation of App. F.2, Kbar = Gamma.K, Kk = Kbar^kappa, Qbar = tau Gamma.Q):
//   gain     uncertainty recursion per channel (Diagonal) or per head
//            (Isotropic) and the gain kappa_t emitted from the pre-write
//            variance (eq. chunk-gain-emission); cumulative decay gamma
//   MMA-T    [Kbar; Qbar] Kk^T          -> T (strict lower) and A_qk (lower)
//   solve    A = (I + T)^-1 on CUDA cores (16x16 blocked substitution, fp32)
//   MMA-W/U  [A; 0] Kbar, [A; 0] V      -> W, [U; 0]
//   MMA-S1   [U; 0] += [-W; Qbar] S_in  -> [R; Qbar S_in]
//   MMA-O    (.) += [0; A_qk] R         -> rows 64..127 hold O
//   MMA-S2   S = diag(gamma_C) S_in + K_tail^T R   (eq. chunk-memory-output-state)
// All MMAs are cta_group::1, M = 128, 16-bit operands in 128-byte-swizzled
// shared memory, fp32 accumulators in TMEM.  Operands are reused across
// layouts: a [tokens][channels] tile is K-major for one product and MN-major
// for another.
// Precision: the operands of MMA-T carry the decay factors exp(+-G) and need
// bf16's exponent range, so each is split into two bf16 terms (hi + lo) and
// the product takes three MMAs (hi.hi + lo.hi + hi.lo).  The state products
// MMA-S1, MMA-O and MMA-S2 have range-bounded operands and run in fp16, whose
// 10-bit mantissa is 8x finer than bf16's.  With single bf16 operands the
// intra-chunk intermediates (R, A_qk) are ~10x larger than the output and the
// error reaches ~3% of RMS(o); with this split it stays below ~0.5%.
//
// Limits of this kernel: bf16 inputs, dk = dv = 128, per-chunk cumulative
// log-decay above about -80 in every channel (exp(-G) must stay finite in
// fp32; with alpha = sigmoid(x) that needs an average alpha > 0.29 over a
// 64-token chunk).  Every wait on an mbarrier is bounded; on timeout the
// kernel records KDN_ERR_TIMEOUT in the workspace status word and returns.
#include <cudaTypedefs.h>

#include <mutex>

#include "kdn_internal.cuh"
#include "kdn_sm103.cuh"

namespace kdn {
namespace {

using namespace sm103;

constexpr int FT = 256;   // threads
constexpr int CM = 64;    // chunk length
constexpr int D = 128;    // head dim (dk = dv)
constexpr uint32_t kWaitIters = 1u << 25;

// shared-memory map (bytes from the 1024-aligned base)
// The raw TMA tiles of k and q are interleaved per 64-channel slab so that,
// once overwritten in place, they form the 128-row operand [Kbar; Qbar]:
//   slab s (16 KB) = [k or Kbar, channels 64s..64s+63 (rows 0..63);
//                     q or Qbar, same channels        (rows 64..127)].
constexpr int OFF_KQ = 0;                 // raw k|q -> hi part of [Kbar; Qbar]   32 KB
constexpr int OFF_W = OFF_KQ + 32768;     // raw omega -> hi part of Kk           16 KB
constexpr int OFF_G = OFF_W + 16384;      // raw g (per-channel decay)            16 KB
constexpr int OFF_A1L = OFF_G + 16384;    // lo part of [Kbar; Qbar] -> [-W; Qbar] fp16
constexpr int OFF_B1L = OFF_A1L + 32768;  // lo part of Kk -> K_tail fp16         16 KB
constexpr int OFF_VR = OFF_B1L + 16384;   // V tile (TMA), later R in fp16        16 KB
constexpr int OFF_A2 = OFF_VR + 16384;    // [A; 0] bf16 -> [0; A_qk] fp16        16 KB
constexpr int OFF_B3 = OFF_A2 + 16384;    // S_in fp16 (MN-major)                 32 KB
constexpr int OFF_F = OFF_B3 + 32768;     // fp32 scratch: Y [64][128] / T, A [64][65] + X
constexpr int F_BYTES = 2 * 64 * 65 * 4 + 3 * 256 * 4;  // 36352 >= 32768
constexpr int OFF_SM = OFF_F + F_BYTES;                  // small arrays
constexpr int SMALL_FLOATS = 64 * 6 + 128 * 2;
constexpr int OFF_BAR = OFF_SM + SMALL_FLOATS * 4;
constexpr int SMEM_BYTES = OFF_BAR + 64 + 1024;  // + alignment slack

struct FusedParams {
  Args a;
  int has_g_map;  // per-channel decay tile through TMA
  int has_w_map;  // per-channel omega tile through TMA (diag)
};

__device__ __forceinline__ float bf(const unsigned char *base, int slab_bytes, int row, int col) {
  const int s = col >> 6;
  return __bfloat162float(
      *reinterpret_cast<const __nv_bfloat16 *>(base + s * slab_bytes + sw128_off(row, col & 63)));
}
__device__ __forceinline__ void bfw(unsigned char *base, int slab_bytes, int row, int col, float x) {
  const int s = col >> 6;
  *reinterpret_cast<__nv_bfloat16 *>(base + s * slab_bytes + sw128_off(row, col & 63)) =
      __float2bfloat16_rn(x);
}

__device__ __forceinline__ void hw(unsigned char *base, int slab_bytes, int row, int col, float x) {
  const int s = col >> 6;
  *reinterpret_cast<__half *>(base + s * slab_bytes + sw128_off(row, col & 63)) = __float2half_rn(x);
}
// x ~ hi + lo with both parts in bf16 (about 16 significant bits together)
__device__ __forceinline__ void bfw2(unsigned char *hi, unsigned char *lo, int slab_bytes, int row,
                                     int col, float x) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  const int s = col >> 6;
  const uint32_t off = s * slab_bytes + sw128_off(row, col & 63);
  *reinterpret_cast<__nv_bfloat16 *>(hi + off) = h;
  *reinterpret_cast<__nv_bfloat16 *>(lo + off) = __float2bfloat16_rn(x - __bfloat162float(h));
}
__device__ __forceinline__ float bf2(const unsigned char *hi, const unsigned char *lo,
                                     int slab_bytes, int row, int col) {
  return bf(hi, slab_bytes, row, col) + bf(lo, slab_bytes, row, col);
}

template <int V>
__global__ void __launch_bounds__(FT, 1)
    k_fused_fwd(const __grid_constant__ CUtensorMap mq, const __grid_constant__ CUtensorMap mk,
                const __grid_constant__ CUtensorMap mv, const __grid_constant__ CUtensorMap mg,
                const __grid_constant__ CUtensorMap mw, const FusedParams P) {
  const Args &a = P.a;
  extern __shared__ unsigned char smraw[];
  unsigned char *sm =
      reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  unsigned char *kq = sm + OFF_KQ;    // k rows 0..63, q rows 64..127 of each 16 KB slab
  unsigned char *rw = sm + OFF_W, *rg = sm + OFF_G;
  unsigned char *a1l = sm + OFF_A1L, *b1l = sm + OFF_B1L;
  unsigned char *vr = sm + OFF_VR, *a2 = sm + OFF_A2, *b3 = sm + OFF_B3;
  float *fs = reinterpret_cast<float *>(sm + OFF_F);
  float *s_r = reinterpret_cast<float *>(sm + OFF_SM);  // [64] r_t
  float *s_x = s_r + 64;     // [64] s_t (diag) / beta_t (iso)
  float *s_n2 = s_x + 64;    // [64] |k|^2 (iso)
  float *s_a = s_n2 + 64;    // [64] a_t (iso)
  float *s_om = s_a + 64;    // [64] omega_t (iso)
  float *s_gs = s_om + 64;   // [64] scalar g_t (iso, scalar decay)
  float *s_gC = s_gs + 64;   // [128] gamma_C
  float *s_b = s_gC + 128;   // [1] isotropic carry b
  uint64_t *bars = reinterpret_cast<uint64_t *>(sm + OFF_BAR);
  uint64_t *bar_raw = bars, *bar_v = bars + 1, *bar_mma = bars + 2;
  uint32_t *s_tbase = reinterpret_cast<uint32_t *>(bars + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wq = warp & 3, wh = warp >> 2;
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int NC = (a.T + CM - 1) / CM;
  const bool pcd = (V == 0) || a.pcd;
  const uint32_t raw_bytes = 8192u * (4 + (P.has_g_map ? 2 : 0) + (P.has_w_map ? 2 : 0));

  if (tid == 0) {
    mbar_init(bar_raw, 1);
    mbar_init(bar_v, 1);
    mbar_init(bar_mma, 1);
    fence_mbar_init();
    prefetch_tmap(&mq);
    prefetch_tmap(&mk);
    prefetch_tmap(&mv);
    if (P.has_g_map) prefetch_tmap(&mg);
    if (P.has_w_map) prefetch_tmap(&mw);
    s_b[0] = (V == 1) ? (a.p0 ? a.p0[bh] : 1.f) : 0.f;
  }
  if (warp == 0) {
    tmem_alloc(s_tbase, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tb = *s_tbase;
  const uint32_t TS = tb, TD1 = tb + 128, TW = tb + 256, TU = tb + 384;
  const uint32_t lane_base = (uint32_t)(32 * wq) << 16;

  // Raw tiles of chunk c arrive on bar_raw in two groups: the decay tile as
  // soon as its buffer is free, then k, q, omega once [Kbar; Qbar] and Kk have
  // been consumed.  The single expect_tx covers both groups.
  auto issue_raw_g = [&](int c) {
    mbar_expect_tx(bar_raw, raw_bytes);
    if (P.has_g_map)
      for (int s = 0; s < 2; ++s) tma_load_4d(rg + s * 8192, &mg, bar_raw, 64 * s, h, c * CM, b);
  };
  auto issue_raw_kqw = [&](int c) {
    for (int s = 0; s < 2; ++s) {
      tma_load_4d(kq + s * 16384, &mk, bar_raw, 64 * s, h, c * CM, b);
      tma_load_4d(kq + s * 16384 + 8192, &mq, bar_raw, 64 * s, h, c * CM, b);
      if (P.has_w_map) tma_load_4d(rw + s * 8192, &mw, bar_raw, 64 * s, h, c * CM, b);
    }
  };
  auto issue_v = [&](int c) {
    mbar_expect_tx(bar_v, 16384);
    for (int s = 0; s < 2; ++s) tma_load_4d(vr + s * 8192, &mv, bar_v, 64 * s, h, c * CM, b);
  };
  if (tid == 0 && NC > 0) {
    issue_raw_g(0);
    issue_raw_kqw(0);
    issue_v(0);
  }

  // initial memory S_0 -> TMEM (row = key channel i, column = value j)
  {
    const int i = 32 * wq + lane;
    for (int c0 = 0; c0 < 64; c0 += 16) {
      float v[16];
      const int j0 = 64 * wh + c0;
      if (a.S0) {
        const float4 *src = reinterpret_cast<const float4 *>(a.S0 + ((size_t)bh * D + i) * D + j0);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          float4 x = src[u];
          v[4 * u] = x.x; v[4 * u + 1] = x.y; v[4 * u + 2] = x.z; v[4 * u + 3] = x.w;
        }
      } else {
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = 0.f;
      }
      tmem_st16(TS + lane_base + j0, v);
    }
    tmem_st_wait();
  }
  // uncertainty carry (diag: one channel per thread of warps 0-3)
  float pcarry = 1.f;
  if (V == 0 && tid < D && a.p0) pcarry = a.p0[(size_t)bh * D + tid];
  // per-token scalars of the next chunk, prefetched into registers
  float nr = 1.f, nom = 0.f, ng = 0.f;
  auto load_scalars = [&](int c) {
    if (tid < CM) {
      const int t = c * CM + tid;
      nr = 1.f; nom = 0.f; ng = 0.f;
      if (c < NC && t < a.T) {
        const size_t th = tok_index(a, b, t, h);
        nr = ld<__nv_bfloat16>(a.r, th);
        if (V == 1) {
          nom = ld<__nv_bfloat16>(a.omega, th);
          if (!a.pcd) ng = ld<__nv_bfloat16>(a.g, th);
        }
      }
    }
  };
  load_scalars(0);

  uint32_t mma_phase = 0;
  bool ok = true;
  const uint32_t id_T = idesc_bf16(128, 64, 0, 0);
  const uint32_t id_WU = idesc_bf16(128, 128, 0, 1);
  const uint32_t ih_S1 = idesc_f16(128, 128, 0, 1);
  const uint32_t ih_S2 = idesc_f16(128, 128, 1, 1);
  auto mma_wait = [&]() -> bool {
    bool r = mbar_wait(bar_mma, mma_phase & 1, kWaitIters);
    ++mma_phase;
    return __syncthreads_and(r);
  };

  for (int c = 0; c < NC && ok; ++c) {
    // ---- [1] raw tiles and per-token scalars of this chunk
    if (tid < CM) {
      s_r[tid] = nr;
      s_om[tid] = nom;
      s_gs[tid] = ng;
    }
    ok = __syncthreads_and(mbar_wait(bar_raw, c & 1, kWaitIters));
    if (!ok) break;
    load_scalars(c + 1);

    // ---- [2] gain, decay and the scaled operand tiles (hi/lo bf16 pairs)
    if (V == 0) {
      if (tid < D) {
        // warps 0-3: uncertainty recursion of channel i (eq. prefix-diag-uncertainty);
        // Kbar overwrites raw k, the unscaled gain X = phat k / gamma overwrites raw omega
        const int i = tid;
        float p = pcarry, e = 1.f;
        for (int t = 0; t < CM; ++t) {
          const float gg = bf(rg, 8192, t, i), w = bf(rw, 8192, t, i), kk = bf(kq, 16384, t, i);
          const float al = __expf(gg);
          e *= al;
          const float ph = al * al * p + w;  // eq. diag-covariance-prediction
          fs[t * D + i] = ph * kk * kk;      // summand of s_t
          bfw2(rw, b1l, 8192, t, i, __fdividef(ph * kk, e));
          bfw2(kq, a1l, 16384, t, i, e * kk);
          const float u = a.mu * kk * kk / s_r[t];
          p = __fdividef(ph, 1.f + u * ph);
        }
        pcarry = p;
      } else {
        // warps 4-7: cumulative decay and Qbar of channel i (overwrites raw q)
        const int i = tid - D;
        float e = 1.f;
        for (int t = 0; t < CM; ++t) {
          e *= __expf(bf(rg, 8192, t, i));
          bfw2(kq, a1l, 16384, 64 + t, i, a.tau * e * bf(kq, 16384, 64 + t, i));
        }
        s_gC[i] = e;
      }
    } else {
      // isotropic: per-token reductions a_t and |k_t|^2
      for (int t = warp * 8; t < warp * 8 + 8; ++t) {
        float n2 = 0.f, sa = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int i = lane + 32 * j;
          const float kk = bf(kq, 16384, t, i);
          n2 += kk * kk;
          if (pcd) {
            const float al = __expf(bf(rg, 8192, t, i));
            sa += al * al;
          }
        }
        n2 = warp_sum(n2);
        sa = warp_sum(sa);
        if (lane == 0) {
          s_n2[t] = n2;
          const float al = __expf(s_gs[t]);
          s_a[t] = pcd ? sa / D : al * al;
        }
      }
      __syncthreads();
      if (tid < D) {
        const int i = tid;
        float e = 1.f;
        for (int t = 0; t < CM; ++t) {
          const float gg = pcd ? bf(rg, 8192, t, i) : s_gs[t];
          e *= __expf(gg);
          const float kk = bf(kq, 16384, t, i);
          bfw2(rw, b1l, 8192, t, i, __fdividef(kk, e));
          bfw2(kq, a1l, 16384, t, i, e * kk);
          bfw2(kq, a1l, 16384, 64 + t, i, a.tau * e * bf(kq, 16384, 64 + t, i));
        }
        s_gC[i] = e;
      } else if (tid == D) {
        // scalar recursion of Prop. 5 (eq. iso-kla-box-cov-update, -gain)
        float bb = s_b[0];
        for (int t = 0; t < CM; ++t) {
          const float bhat = s_a[t] * bb + s_om[t];
          const float rr = s_r[t];
          s_x[t] = __fdividef(bhat, rr + bhat * s_n2[t]);
          const float u = a.mu * s_n2[t] / (D * rr);
          bb = __fdividef(bhat, 1.f + u * bhat);
        }
        s_b[0] = bb;
      }
    }
    __syncthreads();
    if (tid == 0 && c + 1 < NC) issue_raw_g(c + 1);  // the decay tile is no longer read
    // ---- [3] Kk = X / s_t (diag) or beta_t X (iso), kept as a hi/lo pair
    for (int t = warp * 8; t < warp * 8 + 8; ++t) {
      float sc;
      if (V == 0) {
        float part = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) part += fs[t * D + lane + 32 * j];
        sc = 1.f / (s_r[t] + warp_sum(part));
      } else {
        sc = s_x[t];
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = lane + 32 * j;
        bfw2(rw, b1l, 8192, t, i, sc * bf2(rw, b1l, 8192, t, i));
      }
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    // ---- [4] MMA-T: D1 = [Kbar; Qbar] Kk^T, hi.hi + lo.hi + hi.lo
    if (tid == 0) {
      tc_fence_after();
      const uint32_t AH = smem_u32(kq), AL = smem_u32(a1l), BH = smem_u32(rw), BL = smem_u32(b1l);
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t ao = (kk >> 2) * 16384 + (kk & 3) * 32, bo = (kk >> 2) * 8192 + (kk & 3) * 32;
        const uint64_t ah = sw128_desc(AH + ao, 16, 1024), bh_ = sw128_desc(BH + bo, 16, 1024);
        umma_bf16(TD1, ah, bh_, id_T, kk > 0);
        umma_bf16(TD1, sw128_desc(AL + ao, 16, 1024), bh_, id_T, 1);
        umma_bf16(TD1, ah, sw128_desc(BL + bo, 16, 1024), id_T, 1);
      }
      umma_commit(bar_mma);
    }
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    // ---- [5] T -> fp32 smem, A = (I + T)^-1
    float *sT = fs, *sA = fs + 64 * 65, *sX = fs + 2 * 64 * 65;
    if (wq < 2) {
      const int r = 32 * wq + lane;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int s0 = 32 * wh + c0;
        tmem_ld16(TD1 + lane_base + s0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u) sT[r * 65 + s0 + u] = (s0 + u < r) ? v[u] : 0.f;
      }
    }
    __syncthreads();
    if (tid < 64) {
      const int bI = tid >> 4, j = tid & 15, o0 = bI * 16;
      for (int r = 0; r < 16; ++r) {
        float acc = (r == j) ? 1.f : 0.f;
        for (int s = j; s < r; ++s) acc -= sT[(o0 + r) * 65 + o0 + s] * sA[(o0 + s) * 65 + o0 + j];
        sA[(o0 + r) * 65 + o0 + j] = (r >= j) ? acc : 0.f;
      }
    }
    __syncthreads();
    for (int L = 1; L < 4; ++L) {
      const int nb = 4 - L;
      for (int e = tid; e < nb * 256; e += FT) {
        const int J = e >> 8, rr = (e >> 4) & 15, cc = e & 15, I = J + L;
        float acc = 0.f;
        for (int K = J; K < I; ++K)
#pragma unroll
          for (int m = 0; m < 16; ++m)
            acc += sT[(16 * I + rr) * 65 + 16 * K + m] * sA[(16 * K + m) * 65 + 16 * J + cc];
        sX[J * 256 + rr * 16 + cc] = acc;
      }
      __syncthreads();
      for (int e = tid; e < nb * 256; e += FT) {
        const int J = e >> 8, rr = (e >> 4) & 15, cc = e & 15, I = J + L;
        float acc = 0.f;
        for (int m = 0; m <= rr; ++m) acc += sA[(16 * I + rr) * 65 + 16 * I + m] * sX[J * 256 + m * 16 + cc];
        sA[(16 * I + rr) * 65 + 16 * J + cc] = -acc;
      }
      __syncthreads();
    }
    // [A; 0] -> a2 (bf16, K-major, K = 64 source tokens)
    for (int e = tid; e < 128 * 64; e += FT) {
      const int r = e >> 6, s = e & 63;
      const float val = (r < 64 && s <= r) ? sA[r * 65 + s] : 0.f;
      *reinterpret_cast<__nv_bfloat16 *>(a2 + sw128_off(r, s)) = __float2bfloat16_rn(val);
    }
    fence_proxy_async();
    ok = __syncthreads_and(mbar_wait(bar_v, c & 1, kWaitIters));
    if (!ok) break;
    tc_fence_before();
    __syncthreads();
    // ---- [6] MMA-W, MMA-U (bf16; Kbar enters as its hi part)
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A2 = smem_u32(a2), KQ = smem_u32(kq), VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t ad = sw128_desc(A2 + kk * 32, 16, 1024);
        umma_bf16(TW, ad, sw128_desc(KQ + kk * 2048, 16384, 1024), id_WU, kk > 0);
        umma_bf16(TU, ad, sw128_desc(VR + kk * 2048, 8192, 1024), id_WU, kk > 0);
      }
      umma_commit(bar_mma);
    }
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    // ---- [7] fp16 operands of the state products:
    //   a1l rows 0..63 <- -W, rows 64..127 <- Qbar;  a2 <- [0; A_qk];
    //   b3 <- S_in (and diag(gamma_C) S_in back to TMEM);  b1l <- K_tail
    if (wq < 2) {
      const int r = 32 * wq + lane;
      for (int c0 = 0; c0 < 64; c0 += 16) {
        float v[16];
        const int j0 = 64 * wh + c0;
        tmem_ld16(TW + lane_base + j0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u) hw(a1l, 16384, r, j0 + u, -v[u]);
      }
      for (int s = 32 * wh; s < 32 * wh + 32; ++s)
        *reinterpret_cast<__half *>(a2 + sw128_off(r, s)) = __float2half_rn(0.f);
    } else {
      const int r = 32 * wq + lane - 64;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int s0 = 32 * wh + c0;
        tmem_ld16(TD1 + lane_base + s0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u)
          *reinterpret_cast<__half *>(a2 + sw128_off(64 + r, s0 + u)) =
              __float2half_rn(s0 + u <= r ? v[u] : 0.f);
      }
    }
    {
      const int i = 32 * wq + lane;
      const float gC = s_gC[i];
      for (int c0 = 0; c0 < 64; c0 += 16) {
        float v[16];
        const int j0 = 64 * wh + c0;
        tmem_ld16(TS + lane_base + j0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          hw(b3, 16384, i, j0 + u, v[u]);
          v[u] *= gC;
        }
        tmem_st16(TS + lane_base + j0, v);
      }
    }
    for (int e = tid; e < CM * D; e += FT) {
      const int t = e >> 7, i = e & 127;
      hw(a1l, 16384, 64 + t, i, bf2(kq, a1l, 16384, 64 + t, i));
      hw(b1l, 8192, t, i, s_gC[i] * bf2(rw, b1l, 8192, t, i));
    }
    tmem_st_wait();
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && c + 1 < NC) issue_raw_kqw(c + 1);  // raw k, q, omega buffers are free
    // ---- [8] MMA-S1 (fp16): [U; 0] += [-W; Qbar] S_in
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A1 = smem_u32(a1l), B3 = smem_u32(b3);
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(TU, sw128_desc(A1 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                  sw128_desc(B3 + kk * 2048, 16384, 1024), ih_S1, 1);
      umma_commit(bar_mma);
    }
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    // ---- [9] R -> fp16 vr (MN-major [64 tok][128 dv])
    if (wq < 2) {
      const int t = 32 * wq + lane;
      for (int c0 = 0; c0 < 64; c0 += 16) {
        float v[16];
        const int j0 = 64 * wh + c0;
        tmem_ld16(TU + lane_base + j0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u) hw(vr, 8192, t, j0 + u, v[u]);
      }
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    // ---- [10] MMA-O and MMA-S2 (fp16)
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A2 = smem_u32(a2), B1 = smem_u32(b1l), VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t bd = sw128_desc(VR + kk * 2048, 8192, 1024);
        umma_bf16(TU, sw128_desc(A2 + kk * 32, 16, 1024), bd, ih_S1, 1);
        umma_bf16(TS, sw128_desc(B1 + kk * 2048, 8192, 1024), bd, ih_S2, 1);
      }
      umma_commit(bar_mma);
    }
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    if (tid == 0 && c + 1 < NC) issue_v(c + 1);  // R in vr has been consumed
    // ---- [11] O (rows 64..127 of TU) -> global
    if (wq >= 2) {
      const int t = 32 * wq + lane - 64, tt = c * CM + t;
      for (int c0 = 0; c0 < 64; c0 += 16) {
        float v[16];
        const int j0 = 64 * wh + c0;
        tmem_ld16(TU + lane_base + j0, v);
        if (tt < a.T) {
          const size_t o = tok_index(a, b, tt, h) * D + j0;
          if (a.odt == KDN_BF16) {
            __nv_bfloat162 *dst = reinterpret_cast<__nv_bfloat162 *>(static_cast<__nv_bfloat16 *>(a.o) + o);
#pragma unroll
            for (int u = 0; u < 8; ++u) dst[u] = __floats2bfloat162_rn(v[2 * u], v[2 * u + 1]);
          } else {
            float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(a.o) + o);
#pragma unroll
            for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }

  if (ok) {
    // final state
    if (a.ST) {
      const int i = 32 * wq + lane;
      for (int c0 = 0; c0 < 64; c0 += 16) {
        float v[16];
        const int j0 = 64 * wh + c0;
        tmem_ld16(TS + lane_base + j0, v);
        float4 *dst = reinterpret_cast<float4 *>(a.ST + ((size_t)bh * D + i) * D + j0);
#pragma unroll
        for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    }
    if (a.pT) {
      if (V == 0 && tid < D) a.pT[(size_t)bh * D + tid] = pcarry;
      if (V == 1 && tid == 0) a.pT[bh] = s_b[0];
    }
  } else {
    if (tid == 0) atomicExch(a.status, (unsigned)KDN_ERR_TIMEOUT);
    // let copies already in flight land before the CTA's shared memory goes away
    if (tid == 0) {
      mbar_wait(bar_raw, 0, kWaitIters);
      mbar_wait(bar_raw, 1, kWaitIters);
      mbar_wait(bar_v, 0, kWaitIters);
      mbar_wait(bar_v, 1, kWaitIters);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tb, 512);
}

// ---------------------------------------------------------------------------
// host side

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void *p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// [B, T, H, 128] bf16 tensor, box = 64 channels x 1 head x 64 tokens x 1 batch
bool make_map(CUtensorMap *m, const void *ptr, const Args &a) {
  auto enc = encoder();
  if (!enc) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)a.H, (cuuint64_t)a.T, (cuuint64_t)a.B};
  cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)a.H * D * 2,
                           (cuuint64_t)a.T * a.H * D * 2};
  cuuint32_t box[4] = {64, 1, 64, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims, strides, box,
             es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool fused_fwd_supported(const Args &a) {
  return a.dtype == KDN_BF16 && a.dk == D && a.dv == D && a.T > 0;
}

int fused_fwd_smem_bytes() { return SMEM_BYTES; }

kdn_status_t launch_fused_fwd(const Args &a, cudaStream_t s) {
  FusedParams P;
  P.a = a;
  P.has_g_map = (a.variant == 0 || a.pcd) ? 1 : 0;
  P.has_w_map = a.variant == 0 ? 1 : 0;
  CUtensorMap mq, mk, mv, mg, mw;
  if (!make_map(&mq, a.q, a) || !make_map(&mk, a.k, a) || !make_map(&mv, a.v, a))
    return KDN_ERR_CUDA;
  mg = mq;
  mw = mq;
  if (P.has_g_map && !make_map(&mg, a.g, a)) return KDN_ERR_CUDA;
  if (P.has_w_map && !make_map(&mw, a.omega, a)) return KDN_ERR_CUDA;
  const int BH = a.B * a.H;
  if (a.variant == 0) {
    if (cudaFuncSetAttribute(k_fused_fwd<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES) != cudaSuccess)
      return KDN_ERR_CUDA;
    k_fused_fwd<0><<<BH, FT, SMEM_BYTES, s>>>(mq, mk, mv, mg, mw, P);
  } else {
    if (cudaFuncSetAttribute(k_fused_fwd<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES) != cudaSuccess)
      return KDN_ERR_CUDA;
    k_fused_fwd<1><<<BH, FT, SMEM_BYTES, s>>>(mq, mk, mv, mg, mw, P);
  }
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

}  // namespace kdn
