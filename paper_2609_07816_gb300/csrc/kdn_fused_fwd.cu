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
// decay exp(G_C) >= 1e-36 (G_C >= -82.8) in every channel, so that 1/gamma
// stays a normal fp32 number; that is an average alpha above 0.27 over a
// 64-token chunk.  A chunk below it is recorded as KDN_ERR_RANGE in the
// workspace status word.  Every wait on an mbarrier is bounded; on timeout the
// kernel records KDN_ERR_TIMEOUT in the workspace status word and returns.
//
// Instantiations (template <V, G, SD, PH>, described at the kernel): the
// variant, logit gates, the isotropic KDN with one decay per head (exact
// single-MMA intra-chunk products on the raw tiles), and the transition pass of
// the sequence-parallel forward (a second memory from S = I with v = 0).  This
// file also holds k_beta_eff, which reads the gain scalars a training forward
// saved.
#include "kdn_internal.cuh"
#include "kdn_sm103.cuh"
#include "kdn_fused_common.cuh"

namespace kdn {
namespace {

using namespace sm103;
using namespace fused;

constexpr int FT = 512;   // threads (16 warps)
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
constexpr int OFF_F = OFF_B3 + 32768;     // fp32 scratch: gamma [64][128] / T, A [64][LT] + X
constexpr int F_BYTES = 2 * 64 * LT * 4 + 3 * 256 * 4;  // 37888 >= 32768
constexpr int OFF_SM = OFF_F + F_BYTES;                  // small arrays
constexpr int SMALL_FLOATS = 64 * 11 + 128 * 3;
constexpr int OFF_BAR = OFF_SM + SMALL_FLOATS * 4;
constexpr int SMEM_BYTES = OFF_BAR + 64 + 1024;  // + alignment slack

// n consecutive floats of 16-byte-aligned shared memory, by float4
__device__ __forceinline__ void ld_f8(const float *p, float *x) {
  const float4 a0 = reinterpret_cast<const float4 *>(p)[0], a1 = reinterpret_cast<const float4 *>(p)[1];
  x[0] = a0.x; x[1] = a0.y; x[2] = a0.z; x[3] = a0.w; x[4] = a1.x; x[5] = a1.y; x[6] = a1.z; x[7] = a1.w;
}
__device__ __forceinline__ void ld_f16(const float *p, float *x) {
  ld_f8(p, x);
  ld_f8(p + 8, x + 8);
}

struct FusedParams {
  Args a;
  int has_g_map;  // per-channel decay tile through TMA
  int has_w_map;  // per-channel omega tile through TMA (diag)
  int write_o;    // 0: the outputs o are not written (state-saving pass of the backward)
  float *phi_T;   // PH: [BH][128][128] transition of the whole sequence (from S = I, v = 0)
  unsigned char *save_S;  // optional [BH][NC] context records of the backward (kCtxBytes each)
  float *save_p;          // optional [BH][NC][128] uncertainty carry entering each chunk
};

// G: the gate inputs are logits (KDN_GATES_LOGITS), a compile-time choice so
// that the post-activation path carries none of the activation code.
// SD: isotropic KDN with one decay per head (decay_per_channel = 0).  Gamma is
// then a per-token scalar and factors out of every intra-chunk product:
//   T_ts = beta_s (k_t . k_s) gamma_t / gamma_s,
//   A_qk,ts = tau beta_s (q_t . k_s) gamma_t / gamma_s,
//   W = (A diag(gamma)) K,
// so MMA-T runs once per K step on the raw bf16 k and q tiles (exact products,
// no hi/lo split) and the decay ratios and beta_s are applied in fp32 when T and
// A_qk leave TMEM; no Gamma-scaled operand tile is formed.
// PH: besides the memory S (from S_0, with v), carry the transition Phi of the
// sequence, the memory the same recurrence reaches from S = I with v = 0
// (dk = dv).  Both share every gain, T, A and W; Phi's state pass is
// R_Phi = -W Phi_in, Phi_out = diag(gamma_C) Phi_in + K_tail^T R_Phi.  Per token
// it writes o from the memory (float32, map mo) and o_Phi = tau Phi_t^T q_t, the
// output the transition state would give (fp16, map mo2); the sequence-parallel
// forward joins the segments with the two end states and then forms the exact
// output o + S_in^T o_Phi.  No context is saved.
template <int V, int G, int SD, int PH>
__global__ void __launch_bounds__(FT, 1)
    k_fused_fwd(const __grid_constant__ CUtensorMap mq, const __grid_constant__ CUtensorMap mk,
                const __grid_constant__ CUtensorMap mv, const __grid_constant__ CUtensorMap mg,
                const __grid_constant__ CUtensorMap mw, const __grid_constant__ CUtensorMap mo,
                const __grid_constant__ CUtensorMap mo2, const FusedParams P) {
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
  float *s_bh = s_a + 64;    // [64] bhat_t (iso)
  float *s_bp = s_bh + 64;   // [64] b_{t-1} (iso)
  float *s_om = s_bp + 64;   // [64] omega_t (iso)
  float *s_gs = s_om + 64;   // [64] scalar g_t (iso, scalar decay)
  float *s_ri = s_gs + 64;   // [64] 1 / r_t
  float *s_gC = s_ri + 64;   // [128] gamma_C
  float *s_b = s_gC + 128;   // [1] isotropic carry b
  float *s_p = s_b + 128;    // [128] diagonal carry p (per channel)
  float *s_gm = s_p + 128;   // [64] gamma_t (SD: one value per token)
  float *s_kf = s_gm + 64;   // [64] beta_t / gamma_t (SD)
  uint64_t *bars = reinterpret_cast<uint64_t *>(sm + OFF_BAR);
  uint64_t *bar_raw = bars, *bar_v = bars + 1, *bar_mma = bars + 2;
  uint32_t *s_tbase = reinterpret_cast<uint32_t *>(bars + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wq = warp & 3, wg = warp >> 2;  // TMEM lane quarter, column group
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int NC = (a.T + CM - 1) / CM;
  const bool pcd = (V == 0) || a.pcd;
  // the copies (TMA loads, context and output stores) are issued by lane 0 of warp 15,
  // not by the MMA issuer: each TMA operation holds the issuing warp for tens of cycles
  const bool io = tid == 480;
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
  // PH: Phi takes the columns of MMA-T's output, which then shares TW's (T has been
  // read before MMA-W writes W, and A_qk is not needed without o)
  const uint32_t TS = tb, TPH = tb + 128, TD1 = PH ? tb + 256 : tb + 128, TW = tb + 256, TU = tb + 384;
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
  if (io && NC > 0) {
    issue_raw_g(0);
    issue_raw_kqw(0);
    issue_v(0);
  }

  // initial memory S_0 -> TMEM (row = key channel i, column = value j)
  {
    const int i = 32 * wq + lane;
    for (int c0 = 0; c0 < 32; c0 += 16) {
      float v[16];
      const int j0 = 32 * wg + c0;
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
      if (PH) {  // Phi_0 = I
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = (i == j0 + u) ? 1.f : 0.f;
        tmem_st16(TPH + lane_base + j0, v);
      }
    }
    tmem_st_wait();
  }
  // uncertainty carry (diag: one value per channel)
  if (V == 0 && tid < D) s_p[tid] = a.p0 ? a.p0[(size_t)bh * D + tid] : 1.f;
  // per-token scalars of the next chunk, prefetched into registers
  float nr = 1.f, nom = 0.f, ng = 0.f;
  auto load_scalars = [&](int c) {
    if (tid < CM) {
      const int t = c * CM + tid;
      nr = 1.f; nom = 0.f; ng = 0.f;
      if (c < NC && t < a.T) {
        const size_t th = tok_index(a, b, t, h);
        nr = gate_r(G, a.rmin, ld<__nv_bfloat16>(a.r, th));
        if (V == 1) {
          nom = gate_omega(G, ld<__nv_bfloat16>(a.omega, th));
          if (!a.pcd) ng = gate_logalpha(G, ld<__nv_bfloat16>(a.g, th));
        }
      }
    }
  };
  load_scalars(0);

  uint32_t mma_phase = 0;
  bool ok = true;
  const uint32_t id_T = idesc_bf16(128, 64, 0, 0);
  const uint32_t id_WU = idesc_bf16(128, 128, 0, 1), id_U = idesc_f16(128, 128, 0, 1);
  const uint32_t ih_S1 = idesc_f16(128, 128, 0, 1);
  const uint32_t ih_S2 = idesc_f16(128, 128, 1, 1);
  // One thread polls the MMA-completion barrier; the CTA barrier then orders every
  // thread's TMEM reads after it (each caller issues tcgen05.fence::after_thread_sync).
  auto mma_wait = [&]() -> bool {
    bool r = true;
    if (tid == 0) r = mbar_wait(bar_mma, mma_phase & 1, kWaitIters);
    ++mma_phase;
    return __syncthreads_and(r);
  };

  for (int c = 0; c < NC && ok; ++c) {
    // ---- [1] raw tiles and per-token scalars of this chunk
    if (tid < CM) {
      s_r[tid] = nr;
      s_ri[tid] = 1.f / nr;
      s_om[tid] = nom;
      s_gs[tid] = ng;
    }
    if (io) bulk_wait_read();  // O staging and the saved S image have been read
    if (P.save_p && tid < D)
      P.save_p[((size_t)bh * NC + c) * D + tid] = (V == 0) ? s_p[tid] : s_b[0];
    unsigned char *ctx = P.save_S ? P.save_S + ((size_t)bh * NC + c) * kCtxBytes : nullptr;
    ok = __syncthreads_and(mbar_wait(bar_raw, c & 1, kWaitIters));
    if (!ok) break;
    load_scalars(c + 1);

    // ---- [2] the sequential recursions of this chunk, split into four quarters
    //          of 16 tokens: each quarter first forms the Moebius product of its
    //          tokens (independent of the carry; eq. chunk-gain-summary), the
    //          products are combined into the state entering each quarter
    //          (eq. chunk-gain-carry), then every quarter runs its own 16 steps
    //          (eq. chunk-gain-local-prefix, -emission).  Results go to fp32
    //          scratch: phat to b3, gamma to fs (both free here).
    // alpha and omega from the per-channel gate tiles (log alpha or logits); with
    // logit gates the zero-filled tokens past T are kept identity updates
    const int t_valid = a.T - c * CM;
    auto tile_alpha = [&](float x, int t) {
      return G ? (t < t_valid ? sigmoid_f(x) : 1.f) : __expf(x);
    };
    auto tile_omega = [&](float y, int t) {
      return G ? (t < t_valid ? softplus_f(y) : 0.f) : y;
    };
    float *Pb = reinterpret_cast<float *>(b3);  // [64][128] phat_t
    float *Eb = fs;                             // [64][128] gamma_t
    float *sQ = reinterpret_cast<float *>(a2);  // [4][128][5] per-quarter summaries (a2 is free)
    float carry_out = 0.f, gc_out = 0.f;        // written after the closing barrier
    {
      const int i = tid & (D - 1), qq = tid >> 7, t0 = 16 * qq;
      if (V == 0) {
        float al[16], w[16], uk[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float kk = bf(kq, 16384, t0 + j, i);
          al[j] = tile_alpha(bf(rg, 8192, t0 + j, i), t0 + j);
          w[j] = tile_omega(bf(rw, 8192, t0 + j, i), t0 + j);
          uk[j] = a.mu * kk * kk * s_ri[t0 + j];
        }
        // a quarter's summary is read by the later quarters only: the last one skips it
        if (qq < 3) {
          float m00 = 1.f, m01 = 0.f, m10 = 0.f, m11 = 1.f, eq = 1.f;
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float a2_ = al[j] * al[j], ua2 = uk[j] * a2_, d1 = 1.f + uk[j] * w[j];
            const float n00 = a2_ * m00 + w[j] * m10, n01 = a2_ * m01 + w[j] * m11;
            const float n10 = ua2 * m00 + d1 * m10, n11 = ua2 * m01 + d1 * m11;
            m00 = n00; m01 = n01; m10 = n10; m11 = n11;
            eq *= al[j];
            if ((j & 7) == 7) {  // renormalise by the largest magnitude (n/d is scale free)
              const float sc = __frcp_rn(fmaxf(fmaxf(fabsf(m00), fabsf(m01)), fmaxf(fabsf(m10), fabsf(m11))));
              m00 *= sc; m01 *= sc; m10 *= sc; m11 *= sc;
            }
          }
          float *mine = sQ + (qq * D + i) * 5;
          mine[0] = m00; mine[1] = m01; mine[2] = m10; mine[3] = m11; mine[4] = eq;
        }
        __syncthreads();
        float n = s_p[i], d = 1.f, e = 1.f;
        for (int q2 = 0; q2 < qq; ++q2) {
          const float *o = sQ + (q2 * D + i) * 5;
          const float nn = o[0] * n + o[1] * d, dd = o[2] * n + o[3] * d;
          const float sc = __frcp_rn(fmaxf(fabsf(nn), fabsf(dd)));
          n = nn * sc;
          d = dd * sc;
          e *= o[4];
        }
        float p = __fdividef(n, d);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          e *= al[j];
          const float ph = al[j] * al[j] * p + w[j];  // eq. diag-covariance-prediction
          Pb[(t0 + j) * D + i] = ph;
          Eb[(t0 + j) * D + i] = e;
          p = __fdividef(ph, 1.f + uk[j] * ph);     // eq. prefix-diag-uncertainty
        }
        carry_out = p;
        gc_out = e;
      } else {
        // per-token reductions a_t and |k_t|^2, one half-warp per token
        for (int m = 0; m < 2; ++m) {
          const int t = 32 * m + 2 * warp + (lane >> 4), c8 = lane & 15, sl = c8 >> 3, cc = c8 & 7;
          float kv[8];
          unpack_bf8(sm16(kq, sl * 16384 + chunk_off(t, cc)), kv);
          float n2 = 0.f, sa = 0.f;
#pragma unroll
          for (int j = 0; j < 8; ++j) n2 += kv[j] * kv[j];
          if (pcd) {
            float gv[8];
            unpack_bf8(sm16(rg, sl * 8192 + chunk_off(t, cc)), gv);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float al = tile_alpha(gv[j], t);
              sa += al * al;
            }
          }
#pragma unroll
          for (int o = 8; o > 0; o >>= 1) {
            n2 += __shfl_xor_sync(0xffffffffu, n2, o);
            sa += __shfl_xor_sync(0xffffffffu, sa, o);
          }
          if (c8 == 0) {
            s_n2[t] = n2;
            const float al = __expf(s_gs[t]);
            s_a[t] = pcd ? sa / D : al * al;
          }
        }
        __syncthreads();
        // cumulative decay of channel i within this quarter (SD: per token, below)
        float el[16], eq = 1.f;
        if (!SD) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            eq *= pcd ? tile_alpha(bf(rg, 8192, t0 + j, i), t0 + j) : __expf(s_gs[t0 + j]);
            el[j] = eq;
          }
          sQ[(qq * D + i) * 5 + 4] = eq;
        }
        // scalar uncertainty of the chunk (Prop. 5, eq. iso-kla-box-mobius) by an
        // ordered scan of the token matrices M_t = [[a, w], [u a, 1 + u w]] in one
        // warp: lane l holds tokens 2l, 2l + 1; after the scan it holds the product
        // of tokens 0 .. 2l + 1 (later tokens on the left, renormalised by the
        // largest entry), and the exclusive product gives b_{t-1} for its tokens
        // from the carry b entering the chunk
        if (warp == 0) {
          const int ta = 2 * lane, tb = ta + 1;
          auto tok_m = [&](int t, float &m00, float &m01, float &m10, float &m11) {
            const float at = s_a[t], wt = s_om[t], ut = a.mu * s_n2[t] * s_ri[t] * (1.f / D);
            m00 = at; m01 = wt; m10 = ut * at; m11 = fmaf(ut, wt, 1.f);
          };
          float a00, a01, a10, a11, b00, b01, b10, b11;
          tok_m(ta, a00, a01, a10, a11);
          tok_m(tb, b00, b01, b10, b11);
          // pair product M_tb M_ta
          float m00 = b00 * a00 + b01 * a10, m01 = b00 * a01 + b01 * a11;
          float m10 = b10 * a00 + b11 * a10, m11 = b10 * a01 + b11 * a11;
          renorm4(m00, m01, m10, m11);
#pragma unroll
          for (int off = 1; off < 32; off <<= 1) {
            const float p00 = __shfl_up_sync(0xffffffffu, m00, off);
            const float p01 = __shfl_up_sync(0xffffffffu, m01, off);
            const float p10 = __shfl_up_sync(0xffffffffu, m10, off);
            const float p11 = __shfl_up_sync(0xffffffffu, m11, off);
            if (lane >= off) {
              float n00 = m00 * p00 + m01 * p10, n01 = m00 * p01 + m01 * p11;
              float n10 = m10 * p00 + m11 * p10, n11 = m10 * p01 + m11 * p11;
              renorm4(n00, n01, n10, n11);
              m00 = n00; m01 = n01; m10 = n10; m11 = n11;
            }
          }
          // exclusive product (tokens 0 .. ta - 1) applied to the carry [b, 1]
          float e00 = __shfl_up_sync(0xffffffffu, m00, 1), e01 = __shfl_up_sync(0xffffffffu, m01, 1);
          float e10 = __shfl_up_sync(0xffffffffu, m10, 1), e11 = __shfl_up_sync(0xffffffffu, m11, 1);
          if (lane == 0) { e00 = 1.f; e01 = 0.f; e10 = 0.f; e11 = 1.f; }
          const float bin = s_b[0];
          float n = fmaf(e00, bin, e01), d = fmaf(e10, bin, e11);
          const float bpa = __fdividef(n, d);                       // b_{ta - 1}
          const float nn = fmaf(a00, n, a01 * d), dd = fmaf(a10, n, a11 * d);
          const float bpb = __fdividef(nn, dd);                     // b_{ta}
          const float bha = fmaf(s_a[ta], bpa, s_om[ta]);           // eq. iso-kla-box-cov-update
          const float bhb = fmaf(s_a[tb], bpb, s_om[tb]);
          s_bp[ta] = bpa; s_bh[ta] = bha;
          s_bp[tb] = bpb; s_bh[tb] = bhb;
          const float xa = __fdividef(bha, s_r[ta] + bha * s_n2[ta]);  // beta_t, eq. iso-kla-box-gain
          const float xb = __fdividef(bhb, s_r[tb] + bhb * s_n2[tb]);
          s_x[ta] = xa;
          s_x[tb] = xb;
          if (lane == 31)  // b_63 leaves the chunk
            carry_out = __fdividef(bhb, 1.f + a.mu * s_n2[tb] * s_ri[tb] * (1.f / D) * bhb);
          if (SD) {
            // gamma_t = prod_{s <= t} alpha_s by a product scan over the lanes' pairs
            const float aa = __expf(s_gs[ta]), ab = __expf(s_gs[tb]);
            float pr = aa * ab;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
              const float pv = __shfl_up_sync(0xffffffffu, pr, off);
              if (lane >= off) pr *= pv;
            }
            float ex = __shfl_up_sync(0xffffffffu, pr, 1);
            if (lane == 0) ex = 1.f;
            const float ga = ex * aa, gb = ga * ab;
            s_gm[ta] = ga;
            s_gm[tb] = gb;
            s_kf[ta] = xa * __frcp_rn(ga);
            s_kf[tb] = xb * __frcp_rn(gb);
          }
        }
        __syncthreads();
        if (SD) {  // gamma is the same in every channel: the context keeps the 64 values
          gc_out = s_gm[CM - 1];
        } else {
          float pre = 1.f;
          for (int q2 = 0; q2 < qq; ++q2) pre *= sQ[(q2 * D + i) * 5 + 4];
#pragma unroll
          for (int j = 0; j < 16; ++j) Eb[(t0 + j) * D + i] = pre * el[j];
          gc_out = pre * eq;
        }
      }
      __syncthreads();
      if (qq == 3) {
        s_gC[i] = gc_out;
        check_gamma_range(gc_out, a.status);
        if (V == 0) s_p[i] = carry_out;
      }
      if (V == 1 && tid == 31) s_b[0] = carry_out;  // lane 31 of warp 0 formed b_63
    }
    fence_proxy_async();  // phat / gamma are read by the bulk copies below
    __syncthreads();
    if (io && c + 1 < NC) issue_raw_g(c + 1);  // the decay tile is no longer read
    if (io && P.save_S) {  // phat and gamma into the backward context
      if (V == 0) bulk_s2g(ctx + kCtxPh, Pb, 32768);
      if (SD) bulk_s2g(ctx + kCtxGa, s_gm, CM * 4);  // one gamma per token
      else bulk_s2g(ctx + kCtxGa, Eb, 32768);
      bulk_commit();
    }
    // ---- [3] operand tiles, 16-byte chunks (t, 8 channels), one half-warp per token:
    //   Kk = phat k / (s_t gamma) (diag, s_t = r_t + sum phat k^2) or beta_t k / gamma (iso)
    //   Kbar = gamma k, Qbar = tau gamma q; each as a hi/lo bf16 pair, written over
    //   the raw tiles (hi) and into the lo buffers.  SD: none (MMA-T reads the raw tiles)
    for (int m = 0; m < (SD ? 0 : 2); ++m) {
      const int t = 32 * m + 2 * warp + (lane >> 4), c8 = lane & 15, sl = c8 >> 3, cc = c8 & 7;
      const uint32_t ok16 = sl * 16384 + chunk_off(t, cc), oq16 = ok16 + 8192;
      const uint32_t o8 = sl * 8192 + chunk_off(t, cc);
      float kv[8], qv[8], ev[8], xv[8];
      unpack_bf8(sm16(kq, ok16), kv);
      unpack_bf8(sm16(kq, oq16), qv);
      {
        const float4 *ep = reinterpret_cast<const float4 *>(Eb + t * D + 8 * c8);
        const float4 e0 = ep[0], e1 = ep[1];
        ev[0] = e0.x; ev[1] = e0.y; ev[2] = e0.z; ev[3] = e0.w;
        ev[4] = e1.x; ev[5] = e1.y; ev[6] = e1.z; ev[7] = e1.w;
      }
      if (V == 0) {
        const float4 *pp = reinterpret_cast<const float4 *>(Pb + t * D + 8 * c8);
        const float4 p0 = pp[0], p1 = pp[1];
        const float ph[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
        float y = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) y += ph[j] * kv[j] * kv[j];
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) y += __shfl_xor_sync(0xffffffffu, y, o);
        const float st = s_r[t] + y, sc = 1.f / st;  // eq. kla-box-gain
        if (c8 == 0) s_x[t] = st;
#pragma unroll
        for (int j = 0; j < 8; ++j) xv[j] = __fdividef(ph[j] * kv[j] * sc, ev[j]);
      } else {
        const float beta = s_x[t];
#pragma unroll
        for (int j = 0; j < 8; ++j) xv[j] = __fdividef(beta * kv[j], ev[j]);
      }
      uint4 lo;
      sm16(rw, o8) = split_bf8(xv, &lo);
      sm16(b1l, o8) = lo;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        xv[j] = ev[j] * kv[j];
        qv[j] = a.tau * ev[j] * qv[j];
      }
      sm16(kq, ok16) = split_bf8(xv, &lo);
      sm16(a1l, ok16) = lo;
      sm16(kq, oq16) = split_bf8(qv, &lo);
      sm16(a1l, oq16) = lo;
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    if (io && P.save_S) {  // per-token scalars of the gain into the backward context
      bulk_s2g(ctx + kCtxTok, s_x, 5 * 64 * 4);
      bulk_commit();
    }
    // ---- [4] MMA-T: D1 = [Kbar; Qbar] Kk^T, hi.hi + lo.hi + hi.lo
    if (tid == 0) {
      tc_fence_after();
      const uint32_t AH = smem_u32(kq), AL = smem_u32(a1l), BH = smem_u32(rw), BL = smem_u32(b1l);
      for (int kk = 0; SD && kk < 8; ++kk) {  // [K; Q] K^T on the raw tiles (B: rows 0..63)
        const uint64_t ad = sw128_desc(AH + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
        umma_bf16(TD1, ad, ad, id_T, kk > 0);
      }
      for (int kk = 0; !SD && kk < 8; ++kk) {
        const uint32_t ao = (kk >> 2) * 16384 + (kk & 3) * 32, bo = (kk >> 2) * 8192 + (kk & 3) * 32;
        const uint64_t ah = sw128_desc(AH + ao, 16, 1024), bh_ = sw128_desc(BH + bo, 16, 1024);
        umma_bf16(TD1, ah, bh_, id_T, kk > 0);
        umma_bf16(TD1, sw128_desc(AL + ao, 16, 1024), bh_, id_T, 1);
        umma_bf16(TD1, ah, sw128_desc(BL + bo, 16, 1024), id_T, 1);
      }
      umma_commit(bar_mma);
    }
    // V -> fp16 in place while MMA-T runs (the tile arrived during the previous chunk);
    // on a timeout the MMA is still waited for before leaving
    const bool v_ok = __syncthreads_and(mbar_wait(bar_v, c & 1, kWaitIters));
    if (v_ok) {
      for (int e = tid; e < 64 * 16; e += FT) {
        const uint32_t off = (e >> 9) * 8192 + chunk_off((e >> 3) & 63, e & 7);  // slab, row, chunk
        float v[8];
        unpack_bf8(sm16(vr, off), v);
        sm16(vr, off) = pack_h8(v);
      }
    }
    if (io && P.save_S) bulk_wait_read();  // phat / gamma have left b3 / fs
    ok = mma_wait() && v_ok;
    if (!ok) break;
    tc_fence_after();
    // ---- [5] T -> fp32 smem, A = (I + T)^-1 by 16x16 blocks:
    //   diagonal blocks D_I = (I + T_II)^-1 by column substitution (rows across a half-warp),
    //   then A_IJ = -D_I sum_{K=J}^{I-1} T_IK A_KJ level by level (I - J = 1, 2, 3)
    float *sT = fs, *sA = fs + 64 * LT, *sX = fs + 2 * 64 * LT;
    unsigned char *af = reinterpret_cast<unsigned char *>(fs);  // [A; 0] fp16, 16 KB over T
    if (wq < 2) {
      const int r = 32 * wq + lane, s0 = 16 * wg;
      float v[16];
      tmem_ld16(TD1 + lane_base + s0, v);
      float kf[16];
      if (SD) ld_f16(s_kf + s0, kf);
      const float gr = SD ? s_gm[r] : 1.f;
#pragma unroll
      for (int u = 0; u < 16; ++u)  // SD: T_ts = beta_s gamma_t / gamma_s (k_t . k_s)
        v[u] = (s0 + u >= r) ? 0.f : (SD ? v[u] * (gr * kf[u]) : v[u]);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<float4 *>(sT + r * LT + s0 + 4 * u) = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
    } else if (PH) {
      // A_qk leaves TMEM now: MMA-W overwrites it (TD1 = TW).  fp16 into rows
      // 64..127 of a2, which MMA-W reads only into accumulator rows nobody reads
      const int r = 32 * wq + lane - 64, s0 = 16 * wg;
      float v[16];
      tmem_ld16(TD1 + lane_base + s0, v);
      float kf[16];
      if (SD) ld_f16(s_kf + s0, kf);
      const float fq = SD ? a.tau * s_gm[r] : 1.f;
#pragma unroll
      for (int u = 0; u < 16; ++u)
        v[u] = (s0 + u > r) ? 0.f : (SD ? v[u] * (fq * kf[u]) : v[u]);
      sm16(a2, chunk_off(64 + r, s0 >> 3)) = pack_h8(v);
      sm16(a2, chunk_off(64 + r, (s0 >> 3) + 1)) = pack_h8(v + 8);
    }
    __syncthreads();
    tri_inverse64(sT, sA, sX);
    // [A; 0] -> a2 (bf16, K-major, K = 64 source tokens), 16-byte chunks
    for (int e = tid; e < 128 * 8; e += FT) {
      const int r = e >> 3, cc = e & 7;
      float v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int sidx = 8 * cc + j;
        v[j] = (r < 64 && sidx <= r) ? sA[r * LT + sidx] : 0.f;
      }
      if (PH && r >= 64) {
        // rows 64..127 of a2 hold A_qk (PH)
      } else if (SD) {  // W = (A diag(gamma)) K
        float w[8], gm[8];
        ld_f8(s_gm + 8 * cc, gm);
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = v[j] * gm[j];
        sm16(a2, chunk_off(r, cc)) = pack_bf8(w);
      } else {
        sm16(a2, chunk_off(r, cc)) = pack_bf8(v);
      }
      sm16(af, chunk_off(r, cc)) = pack_h8(v);  // [A; 0] fp16 for MMA-U (over the dead T tile)
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    // ---- [6] MMA-W (bf16; Kbar enters as its hi part), MMA-U (fp16)
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A2 = smem_u32(a2), AF = smem_u32(af), KQ = smem_u32(kq), VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk) {
        umma_bf16(TW, sw128_desc(A2 + kk * 32, 16, 1024), sw128_desc(KQ + kk * 2048, 16384, 1024), id_WU,
                  kk > 0);
        umma_bf16(TU, sw128_desc(AF + kk * 32, 16, 1024), sw128_desc(VR + kk * 2048, 8192, 1024), id_U,
                  kk > 0);
      }
      umma_commit(bar_mma);
    }
    tc_fence_after();
    // While MMA-W/U run, the state operands that depend on neither W nor U
    // (MMA-T has finished reading their buffers; MMA-W/U read a2, kq rows 0..63,
    // af and vr):  b3 <- S_in fp16 and diag(gamma_C) S_in back to TMEM;
    // a1l rows 64..127 <- Qbar fp16;  b1l <- K_tail fp16
    {
      const int i = 32 * wq + lane;
      const float gC = s_gC[i];
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TS + lane_base + j0, v);
        sm16(b3, sl * 16384 + chunk_off(i, cc0)) = pack_h8(v);
        sm16(b3, sl * 16384 + chunk_off(i, cc0 + 1)) = pack_h8(v + 8);
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] *= gC;
        tmem_st16(TS + lane_base + j0, v);
      }
    }
    for (int m = 0; m < 2; ++m) {
      const int t = 32 * m + 2 * warp + (lane >> 4), c8 = lane & 15, sl = c8 >> 3, cc = c8 & 7;
      const uint32_t oq16 = sl * 16384 + 8192 + chunk_off(t, cc), o8 = sl * 8192 + chunk_off(t, cc);
      float hv[8], lv[8];
      if (SD) {  // Qbar = tau gamma_t q_t, K_tail = gamma_C beta_t k_t / gamma_t from the raw tiles
        unpack_bf8(sm16(kq, oq16), hv);
        const float fq = a.tau * s_gm[t], fk = s_kf[t];
#pragma unroll
        for (int j = 0; j < 8; ++j) hv[j] *= fq;
        sm16(a1l, oq16) = pack_h8(hv);
        unpack_bf8(sm16(kq, oq16 - 8192), hv);
#pragma unroll
        for (int j = 0; j < 8; ++j) hv[j] *= s_gC[8 * c8 + j] * fk;
        sm16(b1l, o8) = pack_h8(hv);
        continue;
      }
      unpack_bf8(sm16(kq, oq16), hv);
      unpack_bf8(sm16(a1l, oq16), lv);
#pragma unroll
      for (int j = 0; j < 8; ++j) hv[j] += lv[j];
      sm16(a1l, oq16) = pack_h8(hv);
      unpack_bf8(sm16(rw, o8), hv);
      unpack_bf8(sm16(b1l, o8), lv);
#pragma unroll
      for (int j = 0; j < 8; ++j) hv[j] = s_gC[8 * c8 + j] * (hv[j] + lv[j]);
      sm16(b1l, o8) = pack_h8(hv);
    }
    tmem_st_wait();
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    // kq and rw are free: MMA-T and MMA-W have read them, the Qbar and K_tail
    // conversions above have finished (the wait's barrier)
    if (io && c + 1 < NC) issue_raw_kqw(c + 1);
    if (io && P.save_S) {  // A fp16 [t][s] into the backward context
      bulk_s2g(ctx + kCtxA, af, 8192);
      bulk_commit();
    }
    // ---- [7] the remaining fp16 operands of the state products:
    //   a1l rows 0..63 <- -W;  a2 <- [0; A_qk]  (a2 held [A; 0] for MMA-W)
    if (wq < 2) {
      const int r = 32 * wq + lane;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TW + lane_base + j0, v);
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = -v[u];
        sm16(a1l, sl * 16384 + chunk_off(r, cc0)) = pack_h8(v);
        sm16(a1l, sl * 16384 + chunk_off(r, cc0 + 1)) = pack_h8(v + 8);
      }
      for (int cc = 2 * wg; cc < 2 * wg + 2; ++cc) sm16(a2, chunk_off(r, cc)) = make_uint4(0, 0, 0, 0);
    } else if (!PH) {
      const int r = 32 * wq + lane - 64, s0 = 16 * wg;
      float v[16];
      tmem_ld16(TD1 + lane_base + s0, v);
      float kf[16];
      if (SD) ld_f16(s_kf + s0, kf);
      const float fq = SD ? a.tau * s_gm[r] : 1.f;
#pragma unroll
      for (int u = 0; u < 16; ++u)  // SD: A_qk,ts = tau beta_s gamma_t / gamma_s (q_t . k_s)
        v[u] = (s0 + u > r) ? 0.f : (SD ? v[u] * (fq * kf[u]) : v[u]);
      sm16(a2, chunk_off(64 + r, s0 >> 3)) = pack_h8(v);
      sm16(a2, chunk_off(64 + r, (s0 >> 3) + 1)) = pack_h8(v + 8);
    }
    if (PH) {  // Phi_in -> fp16 in fs (laid out like S_in in b3); diag(gamma_C) Phi_in back to TMEM
      unsigned char *b4 = reinterpret_cast<unsigned char *>(fs);
      const int i = 32 * wq + lane;
      const float gC = s_gC[i];
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TPH + lane_base + j0, v);
        sm16(b4, sl * 16384 + chunk_off(i, cc0)) = pack_h8(v);
        sm16(b4, sl * 16384 + chunk_off(i, cc0 + 1)) = pack_h8(v + 8);
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] *= gC;
        tmem_st16(TPH + lane_base + j0, v);
      }
      tmem_st_wait();
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    if (io && P.save_S) {  // S_in, -W and A_qk into the backward context
      bulk_s2g(ctx + kCtxS, b3, 32768);
      bulk_s2g(ctx + kCtxW, a1l, 8192);
      bulk_s2g(ctx + kCtxW + 8192, a1l + 16384, 8192);
      bulk_s2g(ctx + kCtxAqk, a2 + 8192, 8192);
      bulk_commit();
    }
    // ---- [8] MMA-S1 (fp16): [U; 0] += [-W; Qbar] S_in
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A1 = smem_u32(a1l), B3 = smem_u32(b3);
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(TU, sw128_desc(A1 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                  sw128_desc(B3 + kk * 2048, 16384, 1024), ih_S1, 1);
      if (PH) {  // [R_Phi; .] = [-W; Qbar] Phi_in  (U = 0: v = 0 for Phi)
        const uint32_t B4 = smem_u32(fs);
        for (int kk = 0; kk < 8; ++kk)
          umma_bf16(TW, sw128_desc(A1 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                    sw128_desc(B4 + kk * 2048, 16384, 1024), ih_S1, kk > 0);
      }
      umma_commit(bar_mma);
    }
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    // ---- [9] R -> fp16 vr (MN-major [64 tok][128 dv])
    if (wq < 2) {
      const int t = 32 * wq + lane;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TU + lane_base + j0, v);
        sm16(vr, sl * 8192 + chunk_off(t, cc0)) = pack_h8(v);
        sm16(vr, sl * 8192 + chunk_off(t, cc0 + 1)) = pack_h8(v + 8);
        if (PH) {  // R_Phi -> fs (Phi_in has been read), the same layout
          unsigned char *rp = reinterpret_cast<unsigned char *>(fs);
          tmem_ld16(TW + lane_base + j0, v);
          sm16(rp, sl * 8192 + chunk_off(t, cc0)) = pack_h8(v);
          sm16(rp, sl * 8192 + chunk_off(t, cc0 + 1)) = pack_h8(v + 8);
        }
      }
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    if (io && P.save_S) {  // R into the backward context
      bulk_s2g(ctx + kCtxR, vr, 16384);
      bulk_commit();
    }
    // ---- [10] MMA-O and MMA-S2 (fp16)
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A2 = smem_u32(a2), B1 = smem_u32(b1l), VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t bd = sw128_desc(VR + kk * 2048, 8192, 1024);
        umma_bf16(TU, sw128_desc(A2 + kk * 32, 16, 1024), bd, ih_S1, 1);
        umma_bf16(TS, sw128_desc(B1 + kk * 2048, 8192, 1024), bd, ih_S2, 1);
        if (PH) {  // O_Phi += A_qk R_Phi;  Phi += K_tail^T R_Phi
          const uint64_t bp = sw128_desc(smem_u32(fs) + kk * 2048, 8192, 1024);
          umma_bf16(TW, sw128_desc(A2 + kk * 32, 16, 1024), bp, ih_S1, 1);
          umma_bf16(TPH, sw128_desc(B1 + kk * 2048, 8192, 1024), bp, ih_S2, 1);
        }
      }
      umma_commit(bar_mma);
    }
    if (io && P.save_S) bulk_wait_read();  // the saved R and A have left vr and fs
    if (!(ok = mma_wait())) break;
    tc_fence_after();
    if (io && c + 1 < NC) issue_v(c + 1);  // R in vr has been consumed
    // ---- [11] O (rows 64..127 of TU) -> 128-byte-swizzled staging tiles in fs
    //           -> TMA bulk tensor stores (rows past T are not written)
    if (wq >= 2 && P.write_o) {
      const int t = 32 * wq + lane - 64;
      unsigned char *stg = reinterpret_cast<unsigned char *>(fs);
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0;
        tmem_ld16(TU + lane_base + j0, v);
        if (a.odt == KDN_BF16) {
          // box = 64 bf16 columns: box j0 / 64, chunks (j0 % 64) / 8 + {0, 1}
          const int bx = j0 >> 6, cc = (j0 & 63) >> 3;
          sm16(stg, bx * 8192 + chunk_off(t, cc)) = pack_bf8(v);
          sm16(stg, bx * 8192 + chunk_off(t, cc + 1)) = pack_bf8(v + 8);
        } else {
          // box = 32 fp32 columns: box j0 / 32, chunks (j0 % 32) / 4 + {0..3}
          const int bx = j0 >> 5, cc = (j0 & 31) >> 2;
#pragma unroll
          for (int m = 0; m < 4; ++m)
            sm16(stg, bx * 8192 + chunk_off(t, cc + m)) =
                make_uint4(__float_as_uint(v[4 * m]), __float_as_uint(v[4 * m + 1]),
                           __float_as_uint(v[4 * m + 2]), __float_as_uint(v[4 * m + 3]));
        }
        if (PH) {  // O_Phi (rows 64..127 of TW) -> fp16 staging in a2, boxes of 64 columns
          tmem_ld16(TW + lane_base + j0, v);
          const int bx = j0 >> 6, cc = (j0 & 63) >> 3;
          sm16(a2, bx * 8192 + chunk_off(t, cc)) = pack_h8(v);
          sm16(a2, bx * 8192 + chunk_off(t, cc + 1)) = pack_h8(v + 8);
        }
      }
    }
    fence_proxy_async();
    __syncthreads();
    if (io && P.write_o) {
      const unsigned char *stg = reinterpret_cast<const unsigned char *>(fs);
      const int nbox = a.odt == KDN_BF16 ? 2 : 4, bw = a.odt == KDN_BF16 ? 64 : 32;
      for (int bx = 0; bx < nbox; ++bx) tma_store_4d(&mo, stg + bx * 8192, bx * bw, h, c * CM, b);
      if (PH)
        for (int bx = 0; bx < 2; ++bx) tma_store_4d(&mo2, a2 + bx * 8192, bx * 64, h, c * CM, b);
      bulk_commit();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }

  if (ok) {
    // final state
    if (a.ST) {
      const int i = 32 * wq + lane;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0;
        tmem_ld16(TS + lane_base + j0, v);
        float4 *dst = reinterpret_cast<float4 *>(a.ST + ((size_t)bh * D + i) * D + j0);
#pragma unroll
        for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    }
    if (PH && P.phi_T) {
      const int i = 32 * wq + lane;
      for (int c0 = 0; c0 < 32; c0 += 16) {
        float v[16];
        const int j0 = 32 * wg + c0;
        tmem_ld16(TPH + lane_base + j0, v);
        float4 *dst = reinterpret_cast<float4 *>(P.phi_T + ((size_t)bh * D + i) * D + j0);
#pragma unroll
        for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    }
    if (a.pT) {
      if (V == 0 && tid < D) a.pT[(size_t)bh * D + tid] = s_p[tid];
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
  if (io) bulk_wait_all();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tb, 512);
}

// Effective write strength beta_eff,t = k_t^T kappa_t of every token (eq.
// appendix-effective-write: v - S_t^T k = (1 - beta_eff)(v - Shat_t^T k)), from
// the per-token gain scalars a training forward saved: Diagonal KDN
// kappa = phat k / s_t, so k^T kappa = (s_t - r_t) / s_t = 1 - r_t / s_t;
// Isotropic KDN kappa = beta_t k, so k^T kappa = beta_t |k_t|^2.  One thread per
// token, one CTA per (chunk, batch * head).
__global__ void __launch_bounds__(CM) k_beta_eff(const Args a, const unsigned char *saved, float *out) {
  const int c = blockIdx.x, bh = blockIdx.y, t = threadIdx.x;
  const int b = bh / a.H, h = bh % a.H, NC = (a.T + CM - 1) / CM, tt = c * CM + t;
  if (tt >= a.T) return;
  const float *tok = reinterpret_cast<const float *>(saved + ((size_t)bh * NC + c) * kCtxBytes + kCtxTok);
  const size_t th = tok_index(a, b, tt, h);
  if (a.variant == 0) {
    const float rr = gate_r(a.gates, a.rmin, ld<__nv_bfloat16>(a.r, th));
    out[th] = 1.f - rr / tok[t];
  } else {
    out[th] = tok[t] * tok[CM + t];
  }
}

// Self-test of the bounded waits: thread 0 waits on phase 0 of an mbarrier that
// nothing ever arrives on, with the same helper and a short poll limit (4096
// polls, well under a millisecond), and the CTA reports the timeout in the status
// word exactly as the fused kernels do.  No fault, trap or unbounded loop.
__global__ void __launch_bounds__(32) k_wait_selftest(unsigned *status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  const bool ok = threadIdx.x != 0 || mbar_wait(&bar, 0, 1u << 12);
  if (!__syncthreads_and(ok) && threadIdx.x == 0) atomicExch(status, (unsigned)KDN_ERR_TIMEOUT);
}

// ---------------------------------------------------------------------------
// host side

}  // namespace

kdn_status_t launch_wait_selftest(unsigned *status, cudaStream_t s) {
  k_wait_selftest<<<1, 32, 0, s>>>(status);
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

kdn_status_t launch_beta_eff(const Args &a, const void *saved, float *out, cudaStream_t s) {
  const int NC = (a.T + CM - 1) / CM;
  k_beta_eff<<<dim3((unsigned)NC, (unsigned)(a.B * a.H)), CM, 0, s>>>(
      a, static_cast<const unsigned char *>(saved), out);
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

bool fused_fwd_supported(const Args &a) {
  return a.dtype == KDN_BF16 && a.dk == D && a.dv == D && a.T > 0;
}

int fused_fwd_smem_bytes() { return SMEM_BYTES; }

kdn_status_t launch_fused_fwd(const Args &a, cudaStream_t s, unsigned char *save_S,
                              float *save_p, bool write_o, float *phi_T, void *o_phi) {
  // the transition pass writes o (float32) and o_Phi, and no context
  if (phi_T && (save_S || save_p || !write_o || !o_phi || a.odt != KDN_F32))
    return KDN_ERR_INVALID_ARG;
  FusedParams P;
  P.a = a;
  P.has_g_map = (a.variant == 0 || a.pcd) ? 1 : 0;
  P.has_w_map = a.variant == 0 ? 1 : 0;
  P.write_o = write_o ? 1 : 0;
  P.phi_T = phi_T;
  P.save_S = save_S;
  P.save_p = save_p;
  CUtensorMap mq, mk, mv, mg, mw, mo, mo2;
  if (!make_map(&mq, a.q, a) || !make_map(&mk, a.k, a) || !make_map(&mv, a.v, a))
    return KDN_ERR_CUDA;
  if (P.write_o ? !make_map(&mo, a.o, a, a.odt != KDN_BF16) : !make_map(&mo, a.q, a))
    return KDN_ERR_CUDA;
  if (phi_T ? !make_map(&mo2, o_phi, a, false, true) : !make_map(&mo2, a.q, a)) return KDN_ERR_CUDA;
  mg = mq;
  mw = mq;
  if (P.has_g_map && !make_map(&mg, a.g, a)) return KDN_ERR_CUDA;
  if (P.has_w_map && !make_map(&mw, a.omega, a)) return KDN_ERR_CUDA;
  const int BH = a.B * a.H;
  const int sd = a.variant == 1 && !a.pcd;
  using K = decltype(&k_fused_fwd<0, 0, 0, 0>);
  // [variant][gates][scalar decay][transition]
  static const K kerns[2][2][2][2] = {
      {{{k_fused_fwd<0, 0, 0, 0>, k_fused_fwd<0, 0, 0, 1>}, {nullptr, nullptr}},
       {{k_fused_fwd<0, 1, 0, 0>, k_fused_fwd<0, 1, 0, 1>}, {nullptr, nullptr}}},
      {{{k_fused_fwd<1, 0, 0, 0>, k_fused_fwd<1, 0, 0, 1>}, {k_fused_fwd<1, 0, 1, 0>, k_fused_fwd<1, 0, 1, 1>}},
       {{k_fused_fwd<1, 1, 0, 0>, k_fused_fwd<1, 1, 0, 1>}, {k_fused_fwd<1, 1, 1, 0>, k_fused_fwd<1, 1, 1, 1>}}}};
  const K kern = kerns[a.variant][a.gates ? 1 : 0][sd][phi_T ? 1 : 0];
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES) !=
      cudaSuccess)
    return KDN_ERR_CUDA;
  kern<<<BH, FT, SMEM_BYTES, s>>>(mq, mk, mv, mg, mw, mo, mo2, P);
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

}  // namespace kdn
