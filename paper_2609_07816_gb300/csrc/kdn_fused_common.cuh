// kdn_fused_common.cuh -- helpers shared by the fused tcgen05 forward and
// backward kernels: 16-byte chunk access to 128-byte-swizzled 16-bit tiles,
// bf16/fp16 packing, the hi/lo bf16 split, and the host-side TMA descriptors
// for [B, T, H, 128] activation tensors.
#pragma once

#include <cudaTypedefs.h>

#include <mutex>

#include "kdn_internal.cuh"
#include "kdn_sm103.cuh"

namespace kdn {
namespace fused {

using namespace sm103;

__device__ __forceinline__ float bf(const unsigned char *base, int slab_bytes, int row, int col) {
  const int s = col >> 6;
  return __bfloat162float(
      *reinterpret_cast<const __nv_bfloat16 *>(base + s * slab_bytes + sw128_off(row, col & 63)));
}
// 16-byte chunk `cc` (8 consecutive 2-byte elements) of row `row` in a
// 128-byte-swizzled slab.
__device__ __forceinline__ uint32_t chunk_off(int row, int cc) {
  return (uint32_t)row * 128u + ((uint32_t)(cc ^ (row & 7)) << 4);
}
__device__ __forceinline__ void unpack_bf8(uint4 u, float *v) {
  const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __bfloat1622float2(h[j]);
    v[2 * j] = f.x;
    v[2 * j + 1] = f.y;
  }
}
__device__ __forceinline__ uint4 pack_bf8(const float *v) {
  uint4 u;
  __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
  return u;
}
__device__ __forceinline__ uint4 pack_h8(const float *v) {
  uint4 u;
  __half2 *h = reinterpret_cast<__half2 *>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) h[j] = __floats2half2_rn(v[2 * j], v[2 * j + 1]);
  return u;
}
// x ~ hi + lo, both bf16: returns hi, writes the lo chunk
__device__ __forceinline__ uint4 split_bf8(const float *x, uint4 *lo) {
  float h[8], l[8];
  const uint4 hi = pack_bf8(x);
  unpack_bf8(hi, h);
#pragma unroll
  for (int j = 0; j < 8; ++j) l[j] = x[j] - h[j];
  *lo = pack_bf8(l);
  return hi;
}
__device__ __forceinline__ uint4 &sm16(unsigned char *base, uint32_t off) {
  return *reinterpret_cast<uint4 *>(base + off);
}
__device__ __forceinline__ void unpack_h8(uint4 u, float *v) {
  const __half2 *h = reinterpret_cast<const __half2 *>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __half22float2(h[j]);
    v[2 * j] = f.x;
    v[2 * j + 1] = f.y;
  }
}

// Per-chunk record of the backward context written by the fused forward in
// its saving mode (byte offsets; every tile is the 128-byte-swizzled 16-bit
// image the kernels use in shared memory):
//   S_in  fp16 [128 i][128 j] as two 64-column slabs          32 KB
//   R     fp16 [64 s][128 j] as two slabs                      16 KB
//   -W    fp16 [64 t][128 i] as two slabs                      16 KB
//   A_qk  fp16 [64 t][64 s] (lower triangle)                    8 KB
//   A     fp16 [64 t][64 s] (lower triangle)                    8 KB
//   phat  fp32 [64 t][128 i] (diag; pre-write variance)        32 KB
//   gamma fp32 [64 t][128 i] (cumulative decay in the chunk)   32 KB
//   per-token fp32 [5][64]: s_t (diag) or beta_t, then |k_t|^2, a_t, bhat_t,
//         b_{t-1} (iso)                                          2 KB
//   Y = V - Kbar S_in  fp16 [64 t][128 j] as two slabs (diag; the
//         tile R = A Y was formed from)                          16 KB
constexpr int kCtxS = 0, kCtxR = 32768, kCtxW = 49152, kCtxAqk = 65536, kCtxA = 73728;
constexpr int kCtxPh = 81920, kCtxGa = 114688, kCtxTok = 147456, kCtxY = 149504;
constexpr int kCtxBytes = 165888;

// Smallest cumulative decay gamma_C = exp(G_C) of a chunk the fused kernels
// accept: they divide by gamma (Kk = kappa / gamma), which must stay a normal
// fp32 number.  Below it a kernel records KDN_ERR_RANGE in the status word.
constexpr float kMinGammaC = 1e-36f;
__device__ __forceinline__ void check_gamma_range(float gC, unsigned *status) {
  if (!(gC >= kMinGammaC)) atomicCAS(status, 0u, (unsigned)KDN_ERR_RANGE);
}

// Row stride (floats) of the fp32 T and A tiles: 16-byte rows, conflict-free.
constexpr int LT = 68;

// Level L (= I - J) of the blocked inverse below: one thread per (block J, row,
// 4 columns), float4 operands; X_IJ = sum_{K=J}^{I-1} T_IK A_KJ, then A_IJ = -D_I X_IJ.
template <int L>
__device__ __forceinline__ void tri_inverse_level(const float *sT, float *sA, float *sX) {
  constexpr int nb = 4 - L;
  const int tid = threadIdx.x;
  const int J = tid >> 6, rr = (tid >> 2) & 15, cg = tid & 3, I = J + L;
  if (J < nb) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < L; ++k) {
      const int K = J + k;
      const float *tr = sT + (16 * I + rr) * LT + 16 * K;
      const float *ac = sA + (16 * K) * LT + 16 * J + 4 * cg;
#pragma unroll
      for (int m4 = 0; m4 < 4; ++m4) {
        const float4 t4 = *reinterpret_cast<const float4 *>(tr + 4 * m4);
        const float tv[4] = {t4.x, t4.y, t4.z, t4.w};
#pragma unroll
        for (int mm = 0; mm < 4; ++mm) {
          const float4 a4 = *reinterpret_cast<const float4 *>(ac + (4 * m4 + mm) * LT);
          acc.x += tv[mm] * a4.x;
          acc.y += tv[mm] * a4.y;
          acc.z += tv[mm] * a4.z;
          acc.w += tv[mm] * a4.w;
        }
      }
    }
    *reinterpret_cast<float4 *>(sX + J * 256 + rr * 16 + 4 * cg) = acc;
  }
  __syncthreads();
  if (J < nb) {
    const float *dr = sA + (16 * I + rr) * LT + 16 * I;
    const float *xc = sX + J * 256 + 4 * cg;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int m4 = 0; m4 < 4; ++m4) {
      const float4 d4 = *reinterpret_cast<const float4 *>(dr + 4 * m4);
      const float dv[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
      for (int mm = 0; mm < 4; ++mm) {
        const float4 x4 = *reinterpret_cast<const float4 *>(xc + (4 * m4 + mm) * 16);
        acc.x += dv[mm] * x4.x;
        acc.y += dv[mm] * x4.y;
        acc.z += dv[mm] * x4.z;
        acc.w += dv[mm] * x4.w;
      }
    }
    *reinterpret_cast<float4 *>(sA + (16 * I + rr) * LT + 16 * J + 4 * cg) =
        make_float4(-acc.x, -acc.y, -acc.z, -acc.w);
  }
  __syncthreads();
}

// A = (I + T)^-1 for a strictly lower triangular 64 x 64 fp32 T (row stride
// LT, zero on and above the diagonal), by 16 x 16 blocks, with 512 threads:
// diagonal blocks D_I = (I + T_II)^-1 by column substitution (rows across a
// half-warp), then A_IJ = -D_I sum_{K=J}^{I-1} T_IK A_KJ level by level
// (I - J = 1, 2, 3).  sX holds 3 x 256 floats of scratch.  Entries of A above
// the diagonal are left unwritten except inside the diagonal blocks (zero).
// Contains block-wide barriers; every thread of the CTA must call it.
__device__ __forceinline__ void tri_inverse64(const float *sT, float *sA, float *sX) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  {
    // diagonal block I = warp / 4, columns c, c + 1 (c = 4 (warp % 4) + 2 (lane / 16));
    // lane % 16 is the row.  Column substitution: once x_s is final it is broadcast
    // along the half-warp and every lower row subtracts T_rs x_s.
    const int o0 = 16 * (warp >> 2), rr = lane & 15, cl = 4 * (warp & 3) + 2 * (lane >> 4);
    float trow[16];
#pragma unroll
    for (int u = 0; u < 4; ++u) {  // 0 for columns >= rr
      const float4 t4 = *reinterpret_cast<const float4 *>(sT + (o0 + rr) * LT + o0 + 4 * u);
      trow[4 * u] = t4.x; trow[4 * u + 1] = t4.y; trow[4 * u + 2] = t4.z; trow[4 * u + 3] = t4.w;
    }
    float x0 = (rr == cl) ? 1.f : 0.f, x1 = (rr == cl + 1) ? 1.f : 0.f;
#pragma unroll
    for (int s2 = 0; s2 < 15; ++s2) {
      const float y0 = __shfl_sync(0xffffffffu, x0, s2, 16);
      const float y1 = __shfl_sync(0xffffffffu, x1, s2, 16);
      x0 -= trow[s2] * y0;
      x1 -= trow[s2] * y1;
    }
    sA[(o0 + rr) * LT + o0 + cl] = x0;  // zero above the diagonal
    sA[(o0 + rr) * LT + o0 + cl + 1] = x1;
  }
  __syncthreads();
  // off-diagonal levels, each with its K sum fully unrolled
  tri_inverse_level<1>(sT, sA, sX);
  tri_inverse_level<2>(sT, sA, sX);
  tri_inverse_level<3>(sT, sA, sX);
}

inline PFN_cuTensorMapEncodeTiled_v12000 encoder() {
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

// [B, T, H, 128] tensor of 2- or 4-byte elements; box = 128 bytes of channels
// x 1 head x 64 tokens x 1 batch, 128-byte swizzle.
// f16: fp16 elements (else bf16) when not fp32.
inline bool make_map(CUtensorMap *m, const void *ptr, const Args &a, bool fp32 = false,
                     bool f16 = false) {
  auto enc = encoder();
  if (!enc) return false;
  const cuuint64_t es_bytes = fp32 ? 4 : 2;
  constexpr int D = 128;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)a.H, (cuuint64_t)a.T, (cuuint64_t)a.B};
  cuuint64_t strides[3] = {(cuuint64_t)D * es_bytes, (cuuint64_t)a.H * D * es_bytes,
                           (cuuint64_t)a.T * a.H * D * es_bytes};
  cuuint32_t box[4] = {fp32 ? 32u : 64u, 1, 64, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  const CUtensorMapDataType dt = fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                 : f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                       : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  return enc(m, dt, 4,
             const_cast<void *>(ptr), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}


}  // namespace fused
}  // namespace kdn
