// k_gemm.cu -- fp32 SIMT GEMM for the contractions of the fp32 path:
// the input projection of layers > 1 (a5), the output-layer backward (a10)
// and the weight-gradient / input-gradient contractions (a12).  fp32 FMA keeps
// the fp32 path within its parity bound (tf32 tensor cores would not).
//
// 64 x 64 output tile per CTA, 16-deep k slabs staged in shared memory,
// 256 threads with a 4 x 4 register tile each.  Ragged edges are zero-filled.
// Split-K over gridDim.z writes partial tiles that a separate pass reduces in
// a fixed order, so results do not depend on scheduling.
#include "bkt_internal.h"

namespace bkt {

namespace {
constexpr int BM = 64, BN = 64, BK = 16;
}

template <bool AT, bool BT>
__global__ void __launch_bounds__(256) gemm_f32_kernel(GemmArgs g) {
  __shared__ __align__(16) float As[BK][BM + 4];
  __shared__ __align__(16) float Bs[BK][BN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN, z = blockIdx.z;
  const int splits = g.P ? g.splits : 1;
  int chunk = (g.K + splits - 1) / splits;
  chunk = (chunk + BK - 1) / BK * BK;
  const int kb = z * chunk, ke = min(g.K, kb + chunk);
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = kb; k0 < ke; k0 += BK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = tid + i * 256;
      int mm, kk;
      if (!AT) {
        mm = e >> 4;
        kk = e & 15;
      } else {
        kk = e >> 6;
        mm = e & 63;
      }
      const int m = m0 + mm, k = k0 + kk;
      float v = 0.f;
      if (m < g.M && k < ke) v = AT ? g.A[(int64_t)k * g.lda + m] : g.A[(int64_t)m * g.lda + k];
      As[kk][mm] = v;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = tid + i * 256;
      int nn, kk;
      if (!BT) {
        kk = e >> 6;
        nn = e & 63;
      } else {
        nn = e >> 4;
        kk = e & 15;
      }
      const int n = n0 + nn, k = k0 + kk;
      float v = 0.f;
      if (n < g.N && k < ke) {
        if (BT) {
          v = g.B[(int64_t)n * g.ldb + k];
        } else {
          const int row = g.gather ? g.gather[k] : k;
          if (row >= 0) v = g.B[(int64_t)row * g.ldb + n];
        }
      }
      Bs[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      const float4 a = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
      const float4 b = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= g.N) continue;
      if (g.P) {
        g.P[(int64_t)z * g.M * g.N + (int64_t)m * g.N + n] = acc[i][j];
      } else {
        float v = acc[i][j];
        if (g.bias) v += g.bias[n];
        float *c = g.C + (int64_t)m * g.ldc + n;
        if (g.accumulate) v += *c;
        *c = v;
      }
    }
  }
}

cudaError_t launch_gemm_f32(bool a_t, bool b_t, const GemmArgs &g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  const int splits = g.P ? g.splits : 1;
  if (g.P && splits < 1) return cudaErrorInvalidValue;
  if (g.K <= 0 && !g.P) return cudaErrorInvalidValue;
  dim3 grid((g.M + BM - 1) / BM, (g.N + BN - 1) / BN, splits);
  if (grid.y > 65535u || grid.z > 65535u) return cudaErrorInvalidConfiguration;
  if (!a_t && !b_t) gemm_f32_kernel<false, false><<<grid, 256, 0, s>>>(g);
  else if (!a_t && b_t) gemm_f32_kernel<false, true><<<grid, 256, 0, s>>>(g);
  else if (a_t && !b_t) gemm_f32_kernel<true, false><<<grid, 256, 0, s>>>(g);
  else gemm_f32_kernel<true, true><<<grid, 256, 0, s>>>(g);
  return cudaGetLastError();
}

}  // namespace bkt
