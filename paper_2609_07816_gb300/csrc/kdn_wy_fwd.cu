// kdn_wy_fwd.cu -- chunked forward of the Diagonal KDN in compact-WY form
// (App. F.2, eq. chunk-memory-wy / chunk-memory-output-state) for bfloat16
// activations, d_k = d_v = 128 and chunks of C = 64 tokens, on the tcgen05
// tensor cores of sm_103a.
//
// One CTA (16 warps) owns one (batch, head) and walks its chunks in order; the
// 128 x 128 float32 memory S stays in tensor memory for the whole sequence,
// every activation tile is read once by TMA and o is written once.  Per chunk,
// with G_t = sum_{u<=t} g_u the cumulative log-decay inside the chunk (per
// channel) and gamma_t = exp(G_t):
//
//   gain     warps 0-3, one thread per key channel, run the uncertainty
//            recursion of Prop. 3 over the 64 tokens (eq. diag-cov-update,
//            eq. prefix-diag-uncertainty).  Each thread writes
//              Kk'_t = phat_t k_t exp(c - G_t)          (tf32, MMA-T operand)
//              K'_t  = phat_t k_t exp(G_C - G_t)        (fp16, tensor memory)
//            where c = G_C / 2 is a per-channel reference in the middle of
//            the chunk's decay range.
//   prepare  warps 4-11, one thread per (4 channels, 8 tokens), form
//              Kbar_t = k_t exp(G_t - c), Qbar_t = tau q_t exp(G_t - c)  (tf32)
//              -Kbar_t = -gamma_t k_t, Qbar_t = tau gamma_t q_t        (fp16)
//   MMA-T    [Kbar; Qbar] Kk'^T (tf32) = [T'; A'_qk].  The ratios
//            exp(G_t - G_s) of App. F.2 are exact products of the two
//            referenced factors, each within exp(+-|G_C| / 2).
//            s_t = r_t + sum_i phat_t,i k_t,i^2 (the denominator of the gain,
//            eq. kla-box-gain) is r_t plus the diagonal of T'.
//   MMA-KS   [-Kbar; Qbar] S_in = [-Kbar S_in; Qbar S_in]  (fp16), on the tensor
//            cores while the CUDA cores solve
//   solve    with L = diag(s) + strict_lower(T'), A = (I + T)^-1 = diag(s) L^-1
//            (T = strict_lower(T') diag(1/s)) on CUDA cores in fp32.
//   MMA-R    R = U - W S_in = A (V - Kbar S_in)  (fp16; W = A Kbar, U = A V of
//            eq. chunk-memory-wy are only formed for the backward's context)
//   MMA-O    O = Qbar S_in + A'_qk R'          with R' = diag(1/s) R
//   MMA-S2   S_out = diag(gamma_C) S_in + K'^T R'   (K' in tensor memory)
// so that A'_qk R' = A_qk R and K'^T R' = K_tail^T R of eq.
// chunk-memory-output-state, with A_qk = lower(A'_qk) diag(1/s).  Every MMA
// accumulates in float32 in tensor memory.
//
// The chunk is a chain of dependent stages inside one CTA, and the gain (run one
// chunk ahead on its own warps) is as long as the rest: the kernel is bound by
// that latency, not by HBM or shared-memory throughput.  Every per-element pass
// still reads and writes 8 or 16 bytes per shared-memory instruction wherever the
// layout allows (the gain's per-channel recursion is the exception), and the
// next chunk's TMA operations are issued from a thread outside the MMA issuer's
// warp while every main warp waits for MMA-T.
//
// Range: the referenced factors stay finite while the chunk's cumulative
// log-decay G_C >= -160 in every channel (average alpha >= 0.082 over 64
// tokens).  A chunk below that (flagged by the gain warps, for every channel
// at once) runs in range mode: the main warps form T' and A'_qk on the CUDA
// cores from exp(G_t - G_s), s <= t, which never exceeds 1, in place of MMA-T;
// gamma_t and K' are then formed from G_t directly.  The context-saving
// instantiation keeps the referenced form (the fused backward it feeds divides
// by gamma and reports exp(G_C) < 1e-36 as KDN_ERR_RANGE).
//
// Logit gates (LG): g, omega, r hold the logits x, y, z of the layer's
// parameterisation (Sec. 5): log alpha = -softplus(-x), omega = softplus(y),
// r = r_min + softplus(z), formed in float32.  The gain forms log alpha once per
// element and keeps it in its column of the Kk' tile until the recursion
// overwrites it; the prepare pass forms its own.  The tokens past T are identity
// updates: their rows of the g and omega tiles are set to logits whose
// activations are exactly alpha = 1 and omega = 0, so no pass masks elements.
//
// Every wait on an mbarrier is bounded; on timeout the kernel records
// KDN_ERR_TIMEOUT in the status word, waits (bounded) for its copies in flight,
// frees its tensor memory and returns.
#include <type_traits>

#include "kdn_internal.cuh"
#include "kdn_sm103.cuh"
#include "kdn_fused_common.cuh"

namespace kdn {
namespace {

using namespace sm103;
using namespace fused;

constexpr int WT = 512;  // threads
constexpr int CM = 64;   // chunk length
constexpr int D = 128;   // d_k = d_v
constexpr uint32_t kWait = 1u << 25;
constexpr uint32_t kDrain = 1u << 14;  // bounded waits of the failure path
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kMinHalfG = -80.f;  // c = G_C / 2 below this: out of range
constexpr int kPrepThreads = 256;   // warps 4-11: the preparing pass
constexpr int kMain = 384;          // warps 4-15: everything but the gain
constexpr int kBarMain = 2, kBarGain = 3;  // named barriers (0 = __syncthreads)
constexpr int kTmaThread = 224;  // warp 7, lane 0: issues each chunk's next-chunk TMA operations

// shared-memory map (bytes from the 1024-aligned base)
constexpr int LT = 68;          // row stride (floats) of the fp32 T and A tiles
constexpr int O_RK = 0;        // raw k  [64 t][128 i] bf16, two 64-channel slabs   16 KB
constexpr int O_RG = 16384;    // raw g                                          16 KB
constexpr int O_RW = 32768;    // raw omega                                      16 KB
constexpr int O_V = 49152;     // V (TMA bf16), then Y fp16, then R' fp16 [64 s][128 j]  16 KB
constexpr int O_TA = 65536;    // tf32 [Kbar; Qbar] [128][128], four 32-channel slabs 64 KB
constexpr int O_TB = 133120;   // tf32 Kk' [64][128], four slabs                   32 KB
constexpr int O_Q = 165888;    // q (TMA, one chunk ahead; the preparing pass)    16 KB
constexpr int O_AS1 = 182272;  // fp16 [-Kbar; Qbar] [128][128], two slabs (MMA-KS A) 32 KB
constexpr int O_SMALL = 215040;
// after MMA-T has read the tf32 tiles (T and A run 2 KB past the tf32 tile)
constexpr int O_S16 = O_TA;                      // fp16 S_in [128 i][128 j], two slabs (MMA-KS B)
constexpr int O_SWT = O_TA + 32768;              // fp32 T' [64][LT]
constexpr int O_SWA = O_SWT + 64 * LT * 4;       // fp32 L^-1 [64][LT]
static_assert(O_SWA + 64 * LT * 4 <= O_TB, "T and A tiles overlap the Kk' tile");
constexpr int O_AWU = O_SWT;           // fp16 [A; 0] [128][64] (MMA-R A), over T' after the solve
// small arrays (floats); r and mu / r per token for two chunks (the gain works one chunk ahead)
constexpr int SM_R = 0, SM_MUR = 128, SM_S = 256, SM_IS = 320, SM_C = 384, SM_GC = 512,
              SM_PART = 640, SM_OOR = 640 + 8 * 128, SM_FLOATS = SM_OOR + 16;
constexpr int O_BAR = O_SMALL + SM_FLOATS * 4;
constexpr int O_SX = O_BAR + 64;       // scratch of the solve: 2 x 256 floats
constexpr int O_SY = O_SX + 2048;      //                       32 x 32 floats
constexpr int SMEM_BYTES = O_SY + 4096 + 1024;
static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");

// tensor-memory columns (512 allocated)
constexpr uint32_t TC_S = 0, TC_D1 = 128, TC_KT = 192, TC_W = 256, TC_U = 384;

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcpf(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float lg2f(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// softplus(x) = max(x, 0) + log(1 + exp(-|x|)), from the two approximate base-2
// operations with subnormals flushed (exactly 0 below x = -88)
__device__ __forceinline__ float softplus_w(float x) {
  return fmaxf(x, 0.f) + kLn2 * lg2f(1.f + ex2f(-fabsf(x) * kLog2e));
}
// round to tf32 (nearest, ties away): the tensor core reads the top 19 bits
__device__ __forceinline__ float tf32r(float x) {
  uint32_t u;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(u) : "f"(x));
  return __uint_as_float(u);
}
// byte offset of fp32 element (row, col) of a 128-byte-swizzled tile with 32
// elements per row
__device__ __forceinline__ uint32_t sw32_off(uint32_t row, uint32_t col) {
  return row * 128u + ((((col >> 2) ^ (row & 7u)) << 4) | ((col & 3u) << 2));
}
__device__ __forceinline__ void bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// named barrier that also returns the OR of a predicate over its n threads
__device__ __forceinline__ bool bar_or(int id, int n, bool p) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred pi, po;\n setp.ne.u32 pi, %1, 0;\n barrier.cta.red.or.pred po, %2, %3, pi;\n"
      " selp.u32 %0, 1, 0, po;\n}"
      : "=r"(r)
      : "r"((uint32_t)p), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void umma_tf32(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                          uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// A operand in tensor memory: lane = row, 32-bit column c holds the 16-bit
// elements 2c (low half) and 2c + 1 of that row
__device__ __forceinline__ void umma_f16_tA(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                            uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d),
      "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void tmem_st4u(uint32_t taddr, const uint32_t *v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr),
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3])
               : "memory");
}
// four bf16 (8 bytes) -> floats
__device__ __forceinline__ void unpack_bf4(uint2 u, float *v) {
  v[0] = __uint_as_float(u.x << 16);
  v[1] = __uint_as_float(u.x & 0xffff0000u);
  v[2] = __uint_as_float(u.y << 16);
  v[3] = __uint_as_float(u.y & 0xffff0000u);
}
__device__ __forceinline__ uint2 pack_h4(float a0, float a1, float a2, float a3) {
  uint2 u;
  __half2 h0 = __floats2half2_rn(a0, a1), h1 = __floats2half2_rn(a2, a3);
  u.x = *reinterpret_cast<uint32_t *>(&h0);
  u.y = *reinterpret_cast<uint32_t *>(&h1);
  return u;
}
// byte offset of the 4 bf16 / fp16 channels i0..i0+3 (i0 % 4 == 0) of row t
// in a 128-byte-swizzled [t][64] slab
__device__ __forceinline__ uint32_t sw128_off4(uint32_t t, uint32_t i0) {
  return t * 128u + (((((i0 & 63u) >> 3) ^ (t & 7u)) << 4) | ((i0 & 7u) << 1));
}

// X = L^-1 for the lower triangular 64 x 64 fp32 L = diag(s) + strict_lower(T')
// held in sT (row stride LT; only the lower triangle is read), with
// s_t = r_t + T'_tt, into sA (its strict upper triangle zero), by 16 x 16
// blocks: the diagonal blocks D_I = L_II^-1 by forward substitution (one thread
// per column), then the 32 x 32 halves
//   X_10 = -D_1 L_10 D_0,  X_32 = -D_3 L_32 D_2,
// and the lower-left quarter X_21 = -X22 L21 X11 (X11, X22 the 32 x 32
// diagonal halves), each output thread forming four adjacent columns from
// 16-byte loads.  s_t and 1 / s_t go to s_s, s_is.  Called by the kMain
// threads tid = 0 .. kMain - 1 of warps 4-15 (named-barrier synchronisation).
template <class Side>
__device__ __forceinline__ void wy_inverse(int tid, const float *sT, float *sA, float *sX, float *sY,
                                           const float *s_r, float *s_s, float *s_is,
                                           unsigned char *awu, Side side) {
  const int w = tid >> 5;  // main warp 0 .. 11 (lane quarter w & 3)
  if (tid < 64) {
    // column c of D_I: x_r = (delta_rc - sum_{m<r} L_rm x_m) / L_rr, rows read 16 bytes at a time
    const int o = 16 * (tid >> 4), c = tid & 15;
    const float *tb = sT + o * (LT + 1);
    float x[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      float lr[16];
#pragma unroll
      for (int j = 0; 4 * j <= r; ++j) {
        const float4 t4 = *reinterpret_cast<const float4 *>(tb + r * LT + 4 * j);
        lr[4 * j] = t4.x; lr[4 * j + 1] = t4.y; lr[4 * j + 2] = t4.z; lr[4 * j + 3] = t4.w;
      }
      const float lrr = s_r[o + r] + lr[r];  // s_t = r_t + sum_i phat k^2 (eq. kla-box-gain)
      const float inv = rcpf(lrr);
      if (r == c) {
        s_s[o + r] = lrr;
        s_is[o + r] = inv;
      }
      float acc0 = (r == c) ? 1.f : 0.f, acc1 = 0.f;
#pragma unroll
      for (int m = 0; m < r; ++m) {
        if (m & 1) acc1 = fmaf(-lr[m], x[m], acc1);
        else acc0 = fmaf(-lr[m], x[m], acc0);
      }
      x[r] = (acc0 + acc1) * inv;  // x[r] = 0 for r < c
    }
    float *ab = sA + o * (LT + 1) + c;
#pragma unroll
    for (int r = 0; r < 16; ++r) ab[r * LT] = x[r];
  } else if ((w & 3) < 2) {
    side();  // warps 4, 5, 8, 9 of the main group (lane quarters 0, 1)
  } else {
    // zero the strictly upper 16 x 16 blocks (I < J): 6 blocks x 16 rows x 4 float4
    const int z = 64 * (w >> 2) + 32 * ((w & 3) - 2) + (tid & 31);  // 0 .. 191
    for (int e = z; e < 384; e += 192) {
      const int blk = e >> 6, rr = (e >> 2) & 15, q4 = e & 3;
      const int I = blk < 3 ? 0 : (blk < 5 ? 1 : 2);
      const int J = blk < 3 ? blk + 1 : (blk < 5 ? blk - 1 : 3);
      *reinterpret_cast<float4 *>(sA + (16 * I + rr) * LT + 16 * J + 4 * q4) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  bar_sync(kBarMain, kMain);
  // X_10, X_32: one thread per (block, row, 4 columns)
  const int blk = tid >> 6, r2 = (tid >> 2) & 15, cq2 = 4 * (tid & 3);
  const int C0 = 32 * blk, R0 = C0 + 16;
  if (tid < 128) {
    const float *tp = sT + (R0 + r2) * LT + C0;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 t4 = *reinterpret_cast<const float4 *>(tp + 4 * j);
      const float tv[4] = {t4.x, t4.y, t4.z, t4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 a4 = *reinterpret_cast<const float4 *>(sA + (C0 + 4 * j + u) * LT + C0 + cq2);
        acc.x = fmaf(tv[u], a4.x, acc.x);
        acc.y = fmaf(tv[u], a4.y, acc.y);
        acc.z = fmaf(tv[u], a4.z, acc.z);
        acc.w = fmaf(tv[u], a4.w, acc.w);
      }
    }
    *reinterpret_cast<float4 *>(sX + blk * 256 + r2 * 16 + cq2) = acc;
  }
  bar_sync(kBarMain, kMain);
  if (tid < 128) {
    const float *dp = sA + (R0 + r2) * LT + R0;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 d4 = *reinterpret_cast<const float4 *>(dp + 4 * j);
      const float dv[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 x4 = *reinterpret_cast<const float4 *>(sX + blk * 256 + (4 * j + u) * 16 + cq2);
        acc.x = fmaf(dv[u], x4.x, acc.x);
        acc.y = fmaf(dv[u], x4.y, acc.y);
        acc.z = fmaf(dv[u], x4.z, acc.z);
        acc.w = fmaf(dv[u], x4.w, acc.w);
      }
    }
    *reinterpret_cast<float4 *>(sA + (R0 + r2) * LT + C0 + cq2) = make_float4(-acc.x, -acc.y, -acc.z, -acc.w);
  }
  bar_sync(kBarMain, kMain);
  // Y = L21 X11 (32 x 32 x 32): one thread per (row, 4 columns)
  const int r3 = tid >> 3, cq3 = 4 * (tid & 7);
  if (tid < 256) {
    const float *tp = sT + (32 + r3) * LT;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 t4 = *reinterpret_cast<const float4 *>(tp + 4 * j);
      const float tv[4] = {t4.x, t4.y, t4.z, t4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 a4 = *reinterpret_cast<const float4 *>(sA + (4 * j + u) * LT + cq3);
        acc.x = fmaf(tv[u], a4.x, acc.x);
        acc.y = fmaf(tv[u], a4.y, acc.y);
        acc.z = fmaf(tv[u], a4.z, acc.z);
        acc.w = fmaf(tv[u], a4.w, acc.w);
      }
    }
    *reinterpret_cast<float4 *>(sY + r3 * 32 + cq3) = acc;
  }
  bar_sync(kBarMain, kMain);
  // T' is dead from here on: [A; 0] fp16 [128 t][64 s] (A = diag(s) L^-1) is written over it.
  // X_21 = -X22 Y by threads 0..255, straight to fp16; threads 256..383 convert the rest.
  if (tid < 256) {
    const float *dp = sA + (32 + r3) * LT + 32;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 d4 = *reinterpret_cast<const float4 *>(dp + 4 * j);
      const float dv[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 y4 = *reinterpret_cast<const float4 *>(sY + (4 * j + u) * 32 + cq3);
        acc.x = fmaf(dv[u], y4.x, acc.x);
        acc.y = fmaf(dv[u], y4.y, acc.y);
        acc.z = fmaf(dv[u], y4.z, acc.z);
        acc.w = fmaf(dv[u], y4.w, acc.w);
      }
    }
    const int r = 32 + r3;
    const float sr = -s_s[r];
    *reinterpret_cast<uint2 *>(awu + chunk_off(r, cq3 >> 3) + 2 * (cq3 & 4)) =
        pack_h4(sr * acc.x, sr * acc.y, sr * acc.z, sr * acc.w);
  } else {
    // rows 0..31 (8 column chunks), rows 32..63 columns 32..63 (4 chunks), rows 64..127 zero
    for (int e = tid - 256; e < 896; e += 128) {
      int r, cc;
      if (e < 256) {
        r = e >> 3;
        cc = e & 7;
      } else if (e < 384) {
        r = 32 + ((e - 256) >> 2);
        cc = 4 + (e & 3);
      } else {
        r = 64 + ((e - 384) >> 3);
        cc = e & 7;
      }
      float v[8];
      if (r < 64) {
        const float sr = s_s[r];
        const float4 a0 = *reinterpret_cast<const float4 *>(sA + r * LT + 8 * cc);
        const float4 a1 = *reinterpret_cast<const float4 *>(sA + r * LT + 8 * cc + 4);
        const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = (8 * cc + j <= r) ? sr * av[j] : 0.f;
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = 0.f;
      }
      sm16(awu, chunk_off(r, cc)) = pack_h8(v);
    }
  }
}

// fp32 G_t of the range mode: [64 t][128 i], 512-byte rows, 16-byte groups of four
// channels XOR-swizzled by the row
__device__ __forceinline__ uint32_t g_off(int t, int i4) {
  return (uint32_t)t * 512u + ((uint32_t)(i4 ^ (t & 31)) << 4);
}

// Range mode: a chunk whose cumulative log-decay leaves the range of the
// referenced factors (G_C < -160 in some channel) forms
//   T'_ts   = sum_i k_t,i phat_s,i k_s,i exp(G_t,i - G_s,i)
//   A'qk_ts = tau sum_i q_t,i phat_s,i k_s,i exp(G_t,i - G_s,i)      (s <= t)
// from the cumulative log-decay differences themselves (App. F.2): every ratio
// exp(G_t - G_s), s <= t, lies in (0, 1].  Inputs: raw k, q (bf16 tiles), G (fp32,
// g_off layout) and phat k (fp32 in the layout of the Kk' tile).  Outputs: T' into
// sT and A'_qk into sA (fp32 [64][LT]), zero above the diagonal.  One thread per
// (row t, group of four columns); rows t and 63 - t together have 17 groups.
__device__ __noinline__ void direct_products(int tid, const unsigned char *rk, const unsigned char *rq,
                                                const unsigned char *gbuf, const unsigned char *tb,
                                                float tau, float *sT, float *sA) {
  for (int e = tid; e < 32 * 17; e += kMain) {
    const int pr = e / 17, j = e - 17 * pr, n0 = (pr >> 2) + 1;
    const int t = j < n0 ? pr : 63 - pr;
    const int s0 = 4 * (j < n0 ? j : j - n0);
    float aT[4] = {0.f, 0.f, 0.f, 0.f}, aQ[4] = {0.f, 0.f, 0.f, 0.f};
    for (int i4 = 0; i4 < 32; ++i4) {
      const int i0 = 4 * i4;
      const uint32_t sl8 = (uint32_t)(i0 >> 6) * 8192u;
      float kv[4], qv[4];
      unpack_bf4(*reinterpret_cast<const uint2 *>(rk + sl8 + sw128_off4(t, i0)), kv);
      unpack_bf4(*reinterpret_cast<const uint2 *>(rq + sl8 + sw128_off4(t, i0)), qv);
      const float4 gt = *reinterpret_cast<const float4 *>(gbuf + g_off(t, i4));
      const unsigned char *pkb = tb + (i0 >> 5) * 8192;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int sidx = s0 + u;
        const float4 gs = *reinterpret_cast<const float4 *>(gbuf + g_off(sidx, i4));
        const float4 pk = *reinterpret_cast<const float4 *>(pkb + sw32_off(sidx, i0 & 31));
        // columns above the diagonal are clamped to finite values and masked below
        const float e0 = ex2f(fminf(gt.x - gs.x, 0.f) * kLog2e) * pk.x;
        const float e1 = ex2f(fminf(gt.y - gs.y, 0.f) * kLog2e) * pk.y;
        const float e2 = ex2f(fminf(gt.z - gs.z, 0.f) * kLog2e) * pk.z;
        const float e3 = ex2f(fminf(gt.w - gs.w, 0.f) * kLog2e) * pk.w;
        aT[u] = fmaf(kv[0], e0, fmaf(kv[1], e1, fmaf(kv[2], e2, fmaf(kv[3], e3, aT[u]))));
        aQ[u] = fmaf(qv[0], e0, fmaf(qv[1], e1, fmaf(qv[2], e2, fmaf(qv[3], e3, aQ[u]))));
      }
    }
    *reinterpret_cast<float4 *>(sT + t * LT + s0) =
        make_float4(s0 <= t ? aT[0] : 0.f, s0 + 1 <= t ? aT[1] : 0.f, s0 + 2 <= t ? aT[2] : 0.f,
                    s0 + 3 <= t ? aT[3] : 0.f);
    *reinterpret_cast<float4 *>(sA + t * LT + s0) =
        make_float4(s0 <= t ? tau * aQ[0] : 0.f, s0 + 1 <= t ? tau * aQ[1] : 0.f,
                    s0 + 2 <= t ? tau * aQ[2] : 0.f, s0 + 3 <= t ? tau * aQ[3] : 0.f);
  }
  for (int e = tid; e < 64 * 16; e += kMain) {
    const int t = e >> 4, s0 = 4 * (e & 15);
    if (s0 > t) {
      *reinterpret_cast<float4 *>(sT + t * LT + s0) = make_float4(0.f, 0.f, 0.f, 0.f);
      *reinterpret_cast<float4 *>(sA + t * LT + s0) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

struct WyParams {
  Args a;
  unsigned char *save_S;  // SV: [BH][NC] context records of the backward (kCtxBytes each)
  float *save_p;          // SV: [BH][NC][128] uncertainty carry entering each chunk
};

// SV: besides o, S_T and p_T (each written when its pointer is non-null), keep
// the chunked backward's context: per chunk the fp16 tiles S_in, R, -W, A_qk,
// A = (I + T)^-1 and Y = V - Kbar S_in in the 128-byte-swizzled layout of the
// fused backward (all but A_qk staged in shared memory and bulk-copied),
// phat and gamma in float32 [64 t][128 i], s_t per token, and the uncertainty
// entering the chunk.  The arithmetic is the same with and without it.

template <int SV, int LG>  // LG: g, omega, r hold the logits x, y, z of the gates
__global__ void __launch_bounds__(WT, 1)
    k_wy_fwd(const __grid_constant__ CUtensorMap mk, const __grid_constant__ CUtensorMap mg,
             const __grid_constant__ CUtensorMap mw, const __grid_constant__ CUtensorMap mv,
             const __grid_constant__ CUtensorMap mq, const WyParams P) {
  const Args &a = P.a;
  extern __shared__ unsigned char smraw[];
  unsigned char *sm =
      reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  unsigned char *rk = sm + O_RK, *rg = sm + O_RG, *rw = sm + O_RW, *vr = sm + O_V, *rq = sm + O_Q;
  unsigned char *ta = sm + O_TA, *tb = sm + O_TB, *as1 = sm + O_AS1;
  unsigned char *s16 = sm + O_S16, *awu = sm + O_AWU;
  float *sT = reinterpret_cast<float *>(sm + O_SWT), *sA = reinterpret_cast<float *>(sm + O_SWA);
  unsigned char *wst = sm + O_SWA;  // context: -W fp16 staged over L^-1 after the solve
  float *sX = reinterpret_cast<float *>(sm + O_SX), *sY = reinterpret_cast<float *>(sm + O_SY);
  float *sf = reinterpret_cast<float *>(sm + O_SMALL);
  float *s_r = sf + SM_R, *s_mur = sf + SM_MUR, *s_s = sf + SM_S, *s_is = sf + SM_IS;
  float *s_c = sf + SM_C, *s_gC = sf + SM_GC, *s_part = sf + SM_PART;
  // per chunk (slot c & 1): some channel's decay left the range of the referenced factors
  int *s_oor = reinterpret_cast<int *>(sf + SM_OOR);
  uint64_t *bars = reinterpret_cast<uint64_t *>(sm + O_BAR);
  uint64_t *bar_raw = bars, *bar_v = bars + 1, *bar_mma = bars + 2, *bar_q = bars + 3;
  uint64_t *bar_t = bars + 4;  // MMA-T completions (one a chunk)
  uint64_t *bar_w = bars + 5;  // MMA-W completions (context mode only, one a chunk)
  uint32_t *s_tbase = reinterpret_cast<uint32_t *>(bars + 6);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wq = warp & 3, wg = warp >> 2;  // TMEM lane quarter, column group
  const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
  const int NC = (a.T + CM - 1) / CM;
  const bool issuer = tid == 128;
  const uint32_t lane_base = (uint32_t)(32 * wq) << 16;

  if (issuer) {
    mbar_init(bar_raw, 1);
    mbar_init(bar_v, 1);
    mbar_init(bar_mma, 1);
    mbar_init(bar_q, 1);
    mbar_init(bar_t, 1);
    mbar_init(bar_w, 1);
    fence_mbar_init();
    prefetch_tmap(&mk);
    prefetch_tmap(&mg);
    prefetch_tmap(&mw);
    prefetch_tmap(&mv);
    prefetch_tmap(&mq);
  }
  if (warp == 0) {
    tmem_alloc(s_tbase, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *s_tbase;
  const uint32_t TS = tbase + TC_S, TD1 = tbase + TC_D1, TKT = tbase + TC_KT, TW = tbase + TC_W,
                 TU = tbase + TC_U;

  // k, g, omega of chunk c (the gain and the preparing pass), q of chunk c (the
  // preparing pass), V of chunk c (once MMA-O / MMA-S2 of chunk c - 1 has read R')
  auto issue_raw = [&](int c) {
    mbar_expect_tx(bar_raw, 49152);
    for (int s = 0; s < 2; ++s) {
      tma_load_4d(rk + s * 8192, &mk, bar_raw, 64 * s, h, c * CM, b);
      tma_load_4d(rg + s * 8192, &mg, bar_raw, 64 * s, h, c * CM, b);
      tma_load_4d(rw + s * 8192, &mw, bar_raw, 64 * s, h, c * CM, b);
    }
  };
  auto issue_q = [&](int c) {
    mbar_expect_tx(bar_q, 16384);
    for (int s = 0; s < 2; ++s) tma_load_4d(rq + s * 8192, &mq, bar_q, 64 * s, h, c * CM, b);
  };
  auto issue_v = [&](int c) {
    mbar_expect_tx(bar_v, 16384);
    for (int s = 0; s < 2; ++s) tma_load_4d(vr + s * 8192, &mv, bar_v, 64 * s, h, c * CM, b);
  };
  if (issuer && NC > 0) {
    issue_raw(0);
    issue_q(0);
    issue_v(0);
    if (NC > 1) {
      for (int s = 0; s < 2; ++s) {
        tma_prefetch_4d(&mk, 64 * s, h, CM, b);
        tma_prefetch_4d(&mg, 64 * s, h, CM, b);
        tma_prefetch_4d(&mw, 64 * s, h, CM, b);
        tma_prefetch_4d(&mq, 64 * s, h, CM, b);
      }
    }
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
          const float4 x = src[u];
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

  // roles: warps 0-3 run the gain one chunk ahead; warps 4-15 (the main warps)
  // prepare the operands (warps 4-11), store o (warps 14, 15), and run every
  // tensor-core and solve stage, synchronised among themselves by named barriers
  const bool gain = tid < 128;
  const bool prep = tid >= 128 && tid < 128 + kPrepThreads;
  const int mt = tid - 128;           // main thread 0 .. kMain - 1
  const int wgm = (warp >> 2) - 1;    // main warps: 0, 1, 2 within a lane quarter
  float p = 1.f;                      // gain threads: uncertainty carry of channel tid
  if (gain && a.p0) p = a.p0[(size_t)bh * D + tid];
  float rnext = 1.f;                  // gain threads tid < 64: r of the next chunk's token tid
  auto load_r = [&](int c) {
    if (tid < CM) {
      rnext = 1.f;
      if (c < NC && c * CM + tid < a.T) {
        const float z = ld<__nv_bfloat16>(a.r, tok_index(a, b, c * CM + tid, h));
        rnext = LG ? a.rmin + softplus_w(z) : z;  // r = r_min + softplus(z) (Sec. 5)
      }
    }
  };
  load_r(0);

  uint32_t mph = 0;  // main threads: completions of bar_mma observed (three per chunk:
                     // MMA-KS, MMA-R, MMA-O / MMA-S2)
  auto mma_wait_main = [&]() -> bool {
    const bool r = mbar_wait(bar_mma, mph & 1, kWait);
    ++mph;
    return r;
  };
  const uint32_t id_T = idesc_tf32(128, 64);
  const uint32_t id_16 = idesc_f16(128, 128, 0, 1);  // A K-major, B MN-major

  // ---- the gain of chunk c (warps 0-3): r and mu / r of its tokens into buffer
  //      c & 1, the recursion over its 64 tokens.  Its Kk' tile may be written
  //      once MMA-T of chunk c - 1 has read the previous one.
  auto gain_chunk = [&](int c) -> bool {
    const int i = tid, sb = c & 1;
    float *sr = s_r + 64 * sb, *smur = s_mur + 64 * sb;
    if (tid < CM) {
      sr[tid] = rnext;
      smur[tid] = a.mu / rnext;
    }
    load_r(c + 1);
    bar_sync(kBarGain, 128);
    bool g_ok = mbar_wait(bar_raw, c & 1, kWait);
    const unsigned char *pg = rg + (i >> 6) * 8192, *pw = rw + (i >> 6) * 8192, *pk = rk + (i >> 6) * 8192;
    const int cl = i & 63;
    // element (t, i) of a raw slab: row t, 128-byte swizzle
    auto raw = [&](const unsigned char *base, int t) {
      return __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(base + sw128_off(t, cl)));
    };
    // log alpha and omega from the tile's values
    auto lga = [&](float x) { return LG ? -softplus_w(-x) : x; };
    auto omg = [&](float y) { return LG ? softplus_w(y) : y; };
    // logit gates: the tokens past T must be identity updates (alpha = 1, omega = 0).
    // Their rows of the g and omega tiles, zero-filled by TMA, get the logits +-1e30,
    // whose activations are exactly those (softplus(-1e30) = 0), so that no pass
    // masks its elements; the preparing pass reads the same rows
    if (LG && a.T - c * CM < CM) {
      const __nv_bfloat16 big = __float2bfloat16_rn(1e30f), nbig = __float2bfloat16_rn(-1e30f);
      for (int t = a.T - c * CM; t < CM; ++t) {
        *reinterpret_cast<__nv_bfloat16 *>(rg + (i >> 6) * 8192 + sw128_off(t, cl)) = big;
        *reinterpret_cast<__nv_bfloat16 *>(rw + (i >> 6) * 8192 + sw128_off(t, cl)) = nbig;
      }
    }
    unsigned char *pb = tb + (i >> 5) * 8192;
    const int cb = i & 31;
    // logit gates: log alpha is formed once per element here and kept (fp32) in this
    // channel's column of the Kk' tile, which the loop below overwrites token by token
    // after reading it; the tile is free once MMA-T of chunk c - 1 has read it
    if (LG && c > 0) g_ok = mbar_wait(bar_t, (c - 1) & 1, kWait) && g_ok;
    auto lga_t = [&](int t) {  // log alpha of token t in the loop
      return LG ? *reinterpret_cast<const float *>(pb + sw32_off(t, cb)) : lga(raw(pg, t));
    };
    // G_C, and the sums of the chunk's eight 8-token segments for the preparing pass
    // (which reads them at the next chunk boundary; it is done with the previous chunk's)
    // (logit gates: 16 tokens at a time, their loads ahead of the stores of log alpha,
    // which the compiler must otherwise keep in order with the next loads)
    float GC = 0.f;
    if constexpr (!LG) {
#pragma unroll
      for (int sg = 0; sg < 8; ++sg) {
        const int t = 8 * sg;
        const float ss = ((raw(pg, t) + raw(pg, t + 1)) + (raw(pg, t + 2) + raw(pg, t + 3))) +
                         ((raw(pg, t + 4) + raw(pg, t + 5)) + (raw(pg, t + 6) + raw(pg, t + 7)));
        s_part[sg * D + i] = ss;
        GC += ss;
      }
    } else {
#pragma unroll
    for (int s2 = 0; s2 < 4; ++s2) {
      float x[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) x[j] = lga(raw(pg, 16 * s2 + j));
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const float *y = x + 8 * h2;
        const float ss = ((y[0] + y[1]) + (y[2] + y[3])) + ((y[4] + y[5]) + (y[6] + y[7]));
        s_part[(2 * s2 + h2) * D + i] = ss;
        GC += ss;
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) *reinterpret_cast<float *>(pb + sw32_off(16 * s2 + j, cb)) = x[j];
    }
    }
    const float cref = 0.5f * GC;
    s_c[i] = cref;
    // out of the referenced factors' range in some channel: this chunk forms T' and A'_qk
    // from exp(G_t - G_s) directly
    // (the training forward keeps the referenced form: its context feeds a backward
    // that needs exp(G_C) >= 1e-36, and such chunks are reported instead)
    const bool oor = !SV && bar_or(kBarGain, 128, cref < kMinHalfG);
    if (tid == 0) s_oor[sb] = oor ? 1 : 0;
    float Gt = 0.f;  // G_t of this channel (range mode)
    unsigned char *gctx = SV ? P.save_S + ((size_t)bh * NC + c) * kCtxBytes : nullptr;
    if (SV) P.save_p[((size_t)bh * NC + c) * D + i] = p;
    float *cph = SV ? reinterpret_cast<float *>(gctx + kCtxPh) + i : nullptr;
    float f = ex2f(cref * kLog2e);                // exp(c - G_t), G_{-1} = 0
    const float E2 = ex2f((GC - cref) * kLog2e);  // exp(G_C - c)
    const uint32_t tkt = TKT + (uint32_t)((c & 1) * 32);
    float gb[8], wb[8], kb8[8], mb[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      gb[j] = lga_t(j);
      wb[j] = omg(raw(pw, j));
      kb8[j] = raw(pk, j);
    }
    {
      const float4 m0 = *reinterpret_cast<const float4 *>(smur), m1 = *reinterpret_cast<const float4 *>(smur + 4);
      mb[0] = m0.x; mb[1] = m0.y; mb[2] = m0.z; mb[3] = m0.w; mb[4] = m1.x; mb[5] = m1.y; mb[6] = m1.z; mb[7] = m1.w;
    }
    if (!LG && c > 0) g_ok = mbar_wait(bar_t, (c - 1) & 1, kWait) && g_ok;  // Kk' of chunk c - 1 has been read
    // the chunk in blocks of 8 tokens; the next block's inputs are loaded
    // before the current block's outputs are stored
    if (oor) {
      // range mode (rare): Kk' is replaced by phat k itself, and K' is formed from G_t
      // directly; a compact loop without the prefetching of the referenced mode
#pragma unroll 1
      for (int blk = 0; blk < 8; ++blk) {
        uint32_t kt[4];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int t = 8 * blk + j;
          const float lg = lga_t(t), kk = raw(pk, t);
          const float al = ex2f(lg * kLog2e);
          const float ph = fmaf(al * al, p, omg(raw(pw, t)));
          const float den = fmaf(kk * kk * smur[t], ph, 1.f);
          p = ph * rcpf(den);
          Gt += lg;
          const float pkv = ph * kk;
          if (SV) cph[t * D] = ph;
          *reinterpret_cast<float *>(pb + sw32_off(t, cb)) = pkv;
          const uint32_t hb =
              (uint32_t)__half_as_ushort(__float2half_rn(pkv * ex2f((GC - Gt) * kLog2e)));
          if ((j & 1) == 0) kt[j >> 1] = hb;
          else kt[j >> 1] |= hb << 16;
        }
        tmem_st4u(tkt + lane_base + (uint32_t)(4 * blk), kt);
      }
    } else {
#pragma unroll
      for (int blk = 0; blk < 8; ++blk) {
        float gn[8], wn[8], kn[8], mn[8];
        if (blk < 7) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int t = 8 * (blk + 1) + j;
            gn[j] = lga_t(t);
            wn[j] = omg(raw(pw, t));
            kn[j] = raw(pk, t);
          }
          const float4 m0 = *reinterpret_cast<const float4 *>(smur + 8 * (blk + 1));
          const float4 m1 = *reinterpret_cast<const float4 *>(smur + 8 * (blk + 1) + 4);
          mn[0] = m0.x; mn[1] = m0.y; mn[2] = m0.z; mn[3] = m0.w; mn[4] = m1.x; mn[5] = m1.y; mn[6] = m1.z; mn[7] = m1.w;
        }
        uint32_t kt[4];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int t = 8 * blk + j;
          const float al = ex2f(gb[j] * kLog2e), a2 = al * al;
          const float ph = fmaf(a2, p, wb[j]);               // eq. diag-covariance-prediction
          const float u = kb8[j] * kb8[j] * mb[j];
          const float den = fmaf(u, ph, 1.f);
          const float x = rcpf(al * den);
          p = ph * (x * al);                                  // eq. prefix-diag-uncertainty
          f *= x * den;                                       // / alpha_t
          const float pkv = ph * kb8[j];
          if (SV) cph[t * D] = ph;
          *reinterpret_cast<float *>(pb + sw32_off(t, cb)) = tf32r(pkv * f);
          const uint32_t hb = (uint32_t)__half_as_ushort(__float2half_rn(pkv * (f * E2)));
          if ((j & 1) == 0) kt[j >> 1] = hb;
          else kt[j >> 1] |= hb << 16;
        }
        tmem_st4u(tkt + lane_base + (uint32_t)(4 * blk), kt);
        if (blk < 7) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            gb[j] = gn[j];
            wb[j] = wn[j];
            kb8[j] = kn[j];
            mb[j] = mn[j];
          }
        }
      }
    }
    tmem_st_wait();
    fence_proxy_async();
    return g_ok;
  };

  bool mine = true;    // this thread's waits so far; combined at the CTA-wide barriers
  bool failed = false;
  if (gain && NC > 0) mine = gain_chunk(0);

  for (int c = 0; c < NC; ++c) {
    const uint32_t tkt = TKT + (uint32_t)((c & 1) * 32);
    unsigned char *ctx = SV ? P.save_S + ((size_t)bh * NC + c) * kCtxBytes : nullptr;
    if (SV && issuer) bulk_wait_read();  // the previous chunk's context tiles have left shared memory
    // ---- [0] the previous chunk's MMA-O / MMA-S2 must be done before V is brought
    //          into its R' buffer; the gain of this chunk is done (its warps arrive here)
    if (!gain) mine = mbar_wait(bar_raw, c & 1, kWait) && mine;
    if (issuer && c > 0) {
      mine = mma_wait_main() && mine;  // MMA-O / MMA-S2 of chunk c - 1
      if (mine) issue_v(c);
    } else if (!gain && c > 0) {
      ++mph;
    }
    tc_fence_before();
    if (!__syncthreads_and(mine)) {
      failed = true;
      break;
    }
    tc_fence_after();

    // ---- [1] operand preparation (warps 4-11) and the previous chunk's output
    //          (warps 14, 15); the gain of this chunk is already done
    if (prep) {
      const int pi = mt;
      const int i0 = 4 * (pi & 31), seg = pi >> 5, t0 = 8 * seg;
      const uint32_t sl8 = (uint32_t)(i0 >> 6) * 8192u;  // 64-channel slab of a [t][64] 16-bit tile
      // the chunk's g for this thread's 8 tokens and 4 channels (8 bytes a token)
      uint2 gq[8];
      const bool oor = !SV && s_oor[c & 1] != 0;
      // (logit gates: the rows past T hold logits whose log alpha is exactly 0)
      auto unpack_lga = [&](uint2 u, float *gv) {
        unpack_bf4(u, gv);
        if (LG) {
#pragma unroll
          for (int w = 0; w < 4; ++w) gv[w] = -softplus_w(-gv[w]);
        }
      };
#pragma unroll
      for (int j = 0; j < 8; ++j) gq[j] = *reinterpret_cast<const uint2 *>(rg + sl8 + sw128_off4(t0 + j, i0));
      // G at the start of this thread's segment from the segment sums the gain formed
      float cr[4], G[4] = {0.f, 0.f, 0.f, 0.f}, Ec[4], gm[4];
      {
        const float4 c4 = *reinterpret_cast<const float4 *>(s_c + i0);
        cr[0] = c4.x; cr[1] = c4.y; cr[2] = c4.z; cr[3] = c4.w;
      }
      for (int s2 = 0; s2 < seg; ++s2) {
        const float4 p4 = *reinterpret_cast<const float4 *>(s_part + s2 * D + i0);
        G[0] += p4.x; G[1] += p4.y; G[2] += p4.z; G[3] += p4.w;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) Ec[u] = ex2f(cr[u] * kLog2e);
      mine = mbar_wait(bar_q, c & 1, kWait) && mine;
      unsigned char *pa = ta + (i0 >> 5) * 16384, *pqh = as1 + (i0 >> 6) * 16384;
      const int cc = i0 & 31;
      auto prep_loop = [&](auto range_mode) {
        constexpr bool RM = decltype(range_mode)::value;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int t = t0 + j;
          float gv[4], kv[4], qv[4], e[4];
          unpack_lga(gq[j], gv);
          unpack_bf4(*reinterpret_cast<const uint2 *>(rk + sl8 + sw128_off4(t, i0)), kv);
          unpack_bf4(*reinterpret_cast<const uint2 *>(rq + sl8 + sw128_off4(t, i0)), qv);
          if constexpr (RM) {  // G_t itself for the direct products; gamma_t = exp(G_t) (may underflow)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              G[u] += gv[u];
              gm[u] = ex2f(G[u] * kLog2e);
              qv[u] *= a.tau;
            }
            *reinterpret_cast<float4 *>(ta + g_off(t, i0 >> 2)) = make_float4(G[0], G[1], G[2], G[3]);
          } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              G[u] += gv[u];
              e[u] = ex2f((G[u] - cr[u]) * kLog2e);
              gm[u] = e[u] * Ec[u];
              qv[u] *= a.tau;
            }
            *reinterpret_cast<float4 *>(pa + sw32_off(t, cc)) =
                make_float4(tf32r(e[0] * kv[0]), tf32r(e[1] * kv[1]), tf32r(e[2] * kv[2]), tf32r(e[3] * kv[3]));
            *reinterpret_cast<float4 *>(pa + sw32_off(64 + t, cc)) =
                make_float4(tf32r(e[0] * qv[0]), tf32r(e[1] * qv[1]), tf32r(e[2] * qv[2]), tf32r(e[3] * qv[3]));
          }
          *reinterpret_cast<uint2 *>(pqh + sw128_off4(t, i0)) =
              pack_h4(-gm[0] * kv[0], -gm[1] * kv[1], -gm[2] * kv[2], -gm[3] * kv[3]);
          *reinterpret_cast<uint2 *>(pqh + sw128_off4(64 + t, i0)) =
              pack_h4(gm[0] * qv[0], gm[1] * qv[1], gm[2] * qv[2], gm[3] * qv[3]);
          if (SV)
            *reinterpret_cast<float4 *>(reinterpret_cast<float *>(ctx + kCtxGa) + t * D + i0) =
                make_float4(gm[0], gm[1], gm[2], gm[3]);
        }
      };
      if (oor) prep_loop(std::true_type{});
      else prep_loop(std::false_type{});
      if (seg == 7) {
        *reinterpret_cast<float4 *>(s_gC + i0) = make_float4(gm[0], gm[1], gm[2], gm[3]);
        // the fused backward divides by the saved gamma: it needs gamma_C >= 1e-36
        if (SV)
          for (int u = 0; u < 4; ++u) check_gamma_range(gm[u], a.status);
      }
    } else if (!gain && wq >= 2 && wgm == 2 && c > 0 && a.o) {  // warps 14, 15: O of chunk c - 1
      const int t = 32 * (wq - 2) + lane, tt = (c - 1) * CM + t;
      for (int j0 = 0; j0 < D; j0 += 16) {
        float v[16];
        tmem_ld16(TU + lane_base + j0, v);
        if (tt < a.T) {
          const size_t base = tok_index(a, b, tt, h) * D + j0;
          if (a.odt == KDN_BF16) {
            uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.o) + base);
            dst[0] = pack_bf8(v);
            dst[1] = pack_bf8(v + 8);
          } else {
            float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(a.o) + base);
#pragma unroll
            for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
          }
        }
      }
    }
    fence_proxy_async();
    tc_fence_before();
    if (!__syncthreads_and(mine)) {
      failed = true;
      break;
    }

    // ---- [2] MMA-T; the next chunk's k, g, omega and q.  In range mode the main
    //          warps form T' and A'_qk on the CUDA cores instead, and the issuer
    //          completes the MMA-T barrier's phase by hand once they are done.
    const bool oor = !SV && s_oor[c & 1] != 0;
    auto issue_next = [&]() {
      if (c + 1 < NC) {
        issue_raw(c + 1);
        issue_q(c + 1);
        for (int s = 0; s < 2; ++s) tma_prefetch_4d(&mv, 64 * s, h, (c + 1) * CM, b);
      }
      if (c + 2 < NC) {  // chunk c + 2 into L2: its tiles are loaded during chunk c + 1
        for (int s = 0; s < 2; ++s) {
          tma_prefetch_4d(&mk, 64 * s, h, (c + 2) * CM, b);
          tma_prefetch_4d(&mg, 64 * s, h, (c + 2) * CM, b);
          tma_prefetch_4d(&mw, 64 * s, h, (c + 2) * CM, b);
          tma_prefetch_4d(&mq, 64 * s, h, (c + 2) * CM, b);
        }
      }
    };
    if (issuer && !oor) {
      tc_fence_after();
      const uint32_t A0 = smem_u32(ta), B0 = smem_u32(tb);
      for (int kk = 0; kk < 16; ++kk)
        umma_tf32(TD1, sw128_desc(A0 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                  sw128_desc(B0 + (kk >> 2) * 8192 + (kk & 3) * 32, 16, 1024), id_T, kk > 0);
      umma_commit(bar_t);
    }
    // the next chunk's tiles (the raw tiles are free: the preparing pass is done), from a
    // main thread outside the MMA issuer's warp: its ~20 TMA operations then overlap
    // MMA-T, for which every main warp waits anyway
    if (tid == kTmaThread && !oor) issue_next();
    if (gain) {
      // the next chunk's gain, overlapping this chunk's remaining stages
      if (c + 1 < NC) mine = gain_chunk(c + 1) && mine;
      continue;
    }
    if (oor) {
      direct_products(mt, rk, rq, ta, tb, a.tau, sT, sA);
      bar_sync(kBarMain, kMain);
      if (issuer) {  // the raw tiles and phat k have been read
        mbar_arrive(bar_t);
        issue_next();
      }
    }
    mine = mbar_wait(bar_t, c & 1, kWait) && mine;
    tc_fence_after();

    // ---- [3] T' (with its diagonal) out of TMEM; A'_qk -> fp16 pairs in place (the
    //          A operand of MMA-O); S_in -> fp16; V -> fp16
    if (wq < 2 && !oor) {  // T' rows 0..63, lower triangle with the diagonal -> fp32 tile
      const int t = 32 * wq + lane;
      for (int g = wgm; g < 4; g += 3) {
        const int s0 = 16 * g;
        float v[16];
        tmem_ld16(TD1 + lane_base + s0, v);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          float4 o;
          o.x = (s0 + 4 * u + 0 <= t) ? v[4 * u + 0] : 0.f;
          o.y = (s0 + 4 * u + 1 <= t) ? v[4 * u + 1] : 0.f;
          o.z = (s0 + 4 * u + 2 <= t) ? v[4 * u + 2] : 0.f;
          o.w = (s0 + 4 * u + 3 <= t) ? v[4 * u + 3] : 0.f;
          *reinterpret_cast<float4 *>(sT + t * LT + s0 + 4 * u) = o;
        }
      }
    } else if (wgm == 0) {
      // A'_qk rows 64..127, lower triangle: columns 16g .. 16g + 15 -> fp16 pairs in
      // columns 8g .. 8g + 7 (each column is read before it is overwritten)
      const int t = 32 * (wq - 2) + lane;
      for (int g = 0; g < 4; ++g) {
        float v[16], hv[8];
        if (oor) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float4 x4 = *reinterpret_cast<const float4 *>(sA + t * LT + 16 * g + 4 * u);
            v[4 * u] = x4.x; v[4 * u + 1] = x4.y; v[4 * u + 2] = x4.z; v[4 * u + 3] = x4.w;
          }
        } else {
          tmem_ld16(TD1 + lane_base + 16 * g, v);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const __half2 h2 = __floats2half2_rn((16 * g + 2 * j <= t) ? v[2 * j] : 0.f,
                                               (16 * g + 2 * j + 1 <= t) ? v[2 * j + 1] : 0.f);
          hv[j] = __uint_as_float(*reinterpret_cast<const uint32_t *>(&h2));
        }
        tmem_st8(TD1 + lane_base + 8 * g, hv);
      }
    }
    {  // S_in -> fp16 (MN-major B of MMA-KS); diag(gamma_C) S_in back to TMEM
      const int i = 32 * wq + lane;
      const float gC = s_gC[i];
      for (int g = wgm; g < 8; g += 3) {
        float v[16];
        const int j0 = 16 * g, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TS + lane_base + j0, v);
        sm16(s16, sl * 16384 + chunk_off(i, cc0)) = pack_h8(v);
        sm16(s16, sl * 16384 + chunk_off(i, cc0 + 1)) = pack_h8(v + 8);
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] *= gC;
        tmem_st16(TS + lane_base + j0, v);
      }
    }
    tmem_st_wait();
    fence_proxy_async();
    tc_fence_before();
    bar_sync(kBarMain, kMain);
    tc_fence_after();
    // MMA-KS: TU = [-Kbar; Qbar] S_in (fp16), while the CUDA cores solve
    if (issuer) {
      const uint32_t A1 = smem_u32(as1), B1 = smem_u32(s16);
      for (int kk = 0; kk < 8; ++kk)
        umma_bf16(TU, sw128_desc(A1 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                  sw128_desc(B1 + kk * 2048, 16384, 1024), id_16, kk > 0);
      umma_commit(bar_mma);
      if (SV) {
        bulk_s2g(ctx + kCtxS, s16, 32768);
        bulk_commit();
      }
    }

    // ---- [4] A = (I + T)^-1 = diag(s) L^-1 with L = diag(s) + strict_lower(T')
    //          (T = strict_lower(T') diag(1/s)), then [A; 0] fp16 over T';
    //          Y = V - Kbar S_in (rows 0..63 of TU plus V) -> fp16 in place over V, by warps
    //          8, 9, 12, 13 while warps 4, 5 solve the diagonal blocks
    {
      auto y_side = [&]() {
        const bool ks_ok = mma_wait_main();  // MMA-KS
        const bool v_ok = mbar_wait(bar_v, c & 1, kWait);
        mine = ks_ok && v_ok && mine;
        tc_fence_after();
        const int t = 32 * wq + lane;
        for (int g = wgm - 1; g < 8; g += 2) {
          float v[16], vv[16];
          const int j0 = 16 * g, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
          tmem_ld16(TU + lane_base + j0, v);
          const uint32_t o0 = sl * 8192 + chunk_off(t, cc0), o1 = sl * 8192 + chunk_off(t, cc0 + 1);
          unpack_bf8(sm16(vr, o0), vv);
          unpack_bf8(sm16(vr, o1), vv + 8);
#pragma unroll
          for (int u = 0; u < 16; ++u) v[u] += vv[u];
          sm16(vr, o0) = pack_h8(v);
          sm16(vr, o1) = pack_h8(v + 8);
        }
      };
      wy_inverse(mt, sT, sA, sX, sY, s_r + 64 * (c & 1), s_s, s_is, awu, y_side);
      if (!(wq < 2 && wgm >= 1)) ++mph;  // MMA-KS, observed by the Y warps
    }
    if (SV) {
      if (wq >= 2 && wgm == 0) {  // A_qk = lower(A'_qk) diag(1/s) into the context
        const int t = 32 * (wq - 2) + lane;
        for (int h2 = 0; h2 < 2; ++h2) {
          float pv[16];
          tmem_ld16(TD1 + lane_base + 16 * h2, pv);  // 32 fp16 of columns 32 h2 ..
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            const int cc = 4 * h2 + q4;
            float v8[8];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t bits = __float_as_uint(pv[4 * q4 + j]);
              const float2 f2 = __half22float2(*reinterpret_cast<const __half2 *>(&bits));
              v8[2 * j] = f2.x * s_is[8 * cc + 2 * j];
              v8[2 * j + 1] = f2.y * s_is[8 * cc + 2 * j + 1];
            }
            *reinterpret_cast<uint4 *>(ctx + kCtxAqk + chunk_off(t, cc)) = pack_h8(v8);
          }
        }
      }
      if (mt < CM) reinterpret_cast<float *>(ctx + kCtxTok)[mt] = s_s[mt];
    }
    fence_proxy_async();
    tc_fence_before();
    bar_sync(kBarMain, kMain);

    // ---- [5] (context only) -W = A (-Kbar) into TW, then to the context
    if (SV) {
      if (issuer) {
        bulk_s2g(ctx + kCtxA, awu, 8192);
        bulk_s2g(ctx + kCtxY, vr, 16384);  // Y, before R' is written over it
        bulk_commit();
        tc_fence_after();
        const uint32_t AW = smem_u32(awu), KN = smem_u32(as1);
        for (int kk = 0; kk < 4; ++kk)  // B = rows 0..63 of [-Kbar; Qbar], MN-major
          umma_bf16(TW, sw128_desc(AW + kk * 32, 16, 1024), sw128_desc(KN + kk * 2048, 16384, 1024),
                    id_16, kk > 0);
        umma_commit(bar_w);  // its own barrier: MMA-KS may not have been observed yet
      }
    }
    // ---- [6] (context only) -W out of TMEM
    if (SV) {  // -W of the context (rows 0..63 of TW), once MMA-W has completed
      mine = mbar_wait(bar_w, c & 1, kWait) && mine;
      tc_fence_after();
      if (wq < 2) {  // into the fp32 L^-1 tile, dead since the solve, for one bulk copy
        const int t = 32 * wq + lane;
        for (int g = wgm; g < 8; g += 3) {
          float v[16];
          const int j0 = 16 * g, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
          tmem_ld16(TW + lane_base + j0, v);
          sm16(wst, sl * 8192 + chunk_off(t, cc0)) = pack_h8(v);
          sm16(wst, sl * 8192 + chunk_off(t, cc0 + 1)) = pack_h8(v + 8);
        }
      }
      fence_proxy_async();
      tc_fence_before();
      bar_sync(kBarMain, kMain);  // TW is free for MMA-R
      if (issuer) {
        bulk_s2g(ctx + kCtxW, wst, 16384);
        bulk_commit();
      }
    }

    // ---- [7] MMA-R: TW = [A; 0] Y = [R; 0]  (fp16)
    if (issuer) {
      // (context: the copy of Y has left shared memory before MMA-R completes, after
      // which R' is written over Y; the copy of -W, committed after it, may still run)
      if (SV) bulk_wait_read_but1();
      tc_fence_after();
      const uint32_t AW = smem_u32(awu), VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk)
        umma_bf16(TW, sw128_desc(AW + kk * 32, 16, 1024), sw128_desc(VR + kk * 2048, 8192, 1024), id_16,
                  kk > 0);
      umma_commit(bar_mma);
    }
    mine = mma_wait_main() && mine;
    tc_fence_after();

    // ---- [8] R' = diag(1/s) R -> fp16 [t][j] (MN-major B), over Y
    if (wq < 2) {
      const int t = 32 * wq + lane;
      const float ist = s_is[t];
      for (int g = wgm; g < 8; g += 3) {
        float v[16];
        const int j0 = 16 * g, sl = j0 >> 6, cc0 = (j0 & 63) >> 3;
        tmem_ld16(TW + lane_base + j0, v);
        if (SV) {  // R for the context, staged over [A; 0] (MMA-R has read it) for one bulk copy
          sm16(awu, sl * 8192 + chunk_off(t, cc0)) = pack_h8(v);
          sm16(awu, sl * 8192 + chunk_off(t, cc0 + 1)) = pack_h8(v + 8);
        }
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] *= ist;
        sm16(vr, sl * 8192 + chunk_off(t, cc0)) = pack_h8(v);
        sm16(vr, sl * 8192 + chunk_off(t, cc0 + 1)) = pack_h8(v + 8);
      }
    }
    fence_proxy_async();
    tc_fence_before();
    bar_sync(kBarMain, kMain);

    // ---- [9] MMA-O (rows 64..127 of TU += A'_qk R', A'_qk in TMEM) and
    //          MMA-S2 (S += K'^T R', K' in TMEM)
    if (issuer) {
      if (SV) {
        bulk_s2g(ctx + kCtxR, awu, 16384);
        bulk_commit();
      }
      tc_fence_after();
      const uint32_t VR = smem_u32(vr);
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t bd = sw128_desc(VR + kk * 2048, 8192, 1024);
        umma_f16_tA(TU, TD1 + (uint32_t)(kk * 8), bd, id_16, 1);
        umma_f16_tA(TS, tkt + (uint32_t)(kk * 8), bd, id_16, 1);
      }
      umma_commit(bar_mma);
    }
  }

  if (!failed && NC > 0) {
    if (!gain) mine = mma_wait_main() && mine;  // MMA-O / MMA-S2 of the last chunk
    tc_fence_before();
    failed = !__syncthreads_and(mine);
    tc_fence_after();
  }
  if (!failed) {
    if (!gain && wq >= 2 && NC > 0 && a.o) {  // O of the last chunk
      const int t = 32 * (wq - 2) + lane, tt = (NC - 1) * CM + t;
      for (int g = wgm; g < 8; g += 3) {
        float v[16];
        const int j0 = 16 * g;
        tmem_ld16(TU + lane_base + j0, v);
        if (tt < a.T) {
          const size_t base = tok_index(a, b, tt, h) * D + j0;
          if (a.odt == KDN_BF16) {
            uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.o) + base);
            dst[0] = pack_bf8(v);
            dst[1] = pack_bf8(v + 8);
          } else {
            float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(a.o) + base);
#pragma unroll
            for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
          }
        }
      }
    }
    if (!gain && a.ST) {
      const int i = 32 * wq + lane;
      for (int g = wgm; g < 8; g += 3) {
        float v[16];
        const int j0 = 16 * g;
        tmem_ld16(TS + lane_base + j0, v);
        float4 *dst = reinterpret_cast<float4 *>(a.ST + ((size_t)bh * D + i) * D + j0);
#pragma unroll
        for (int u = 0; u < 4; ++u) dst[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    }
    if (a.pT && gain) a.pT[(size_t)bh * D + tid] = p;
  } else {
    if (tid == 0) atomicExch(a.status, (unsigned)KDN_ERR_TIMEOUT);
    // copies and MMAs in flight land before the CTA's memory goes away
    // (short bounds: a copy or MMA that was issued lands within microseconds,
    // and a phase that was never armed must not hold the call for long)
    if (issuer) {
      for (int k = 0; k < 6; ++k) {
        mbar_wait(bars + k, 0, kDrain);
        mbar_wait(bars + k, 1, kDrain);
      }
    }
  }
  if (SV && issuer) bulk_wait_all();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tbase, 512);
}

}  // namespace

bool wy_fwd_supported(const Args &a, bool save) {
  (void)save;
  return a.variant == 0 && (a.gates == KDN_GATES_POST || a.gates == KDN_GATES_LOGITS) &&
         a.dtype == KDN_BF16 && a.dk == D && a.dv == D && a.T > 0 && a.chunk != 32;
}

kdn_status_t launch_wy_fwd(const Args &a, cudaStream_t s, unsigned char *save_S, float *save_p) {
  if (!wy_fwd_supported(a, save_S != nullptr) || (!save_S) != (!save_p)) return KDN_ERR_UNSUPPORTED;
  WyParams P;
  P.a = a;
  P.save_S = save_S;
  P.save_p = save_p;
  CUtensorMap mk, mg, mw, mv, mq;
  if (!make_map(&mk, a.k, a) || !make_map(&mg, a.g, a) || !make_map(&mw, a.omega, a) ||
      !make_map(&mv, a.v, a) || !make_map(&mq, a.q, a))
    return KDN_ERR_CUDA;
  const bool lg = a.gates == KDN_GATES_LOGITS;
  const auto kern = save_S ? (lg ? k_wy_fwd<1, 1> : k_wy_fwd<1, 0>) : (lg ? k_wy_fwd<0, 1> : k_wy_fwd<0, 0>);
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES) !=
      cudaSuccess)
    return KDN_ERR_CUDA;
  kern<<<a.B * a.H, WT, SMEM_BYTES, s>>>(mk, mg, mw, mv, mq, P);
  return cudaGetLastError() == cudaSuccess ? KDN_OK : KDN_ERR_CUDA;
}

}  // namespace kdn
