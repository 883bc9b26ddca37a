// k_wgrad.cu -- reductions over the token axis for the weight gradients
// (a10, a12): the narrow first-layer contraction [dW_ih | db] = dz^T [X | 1]
// (X has in_dim <= 16 columns, so it is a bandwidth-bound pass over dz), and
// the fixed-order sum of split-K partial tiles, scattered straight into the
// flat gradient layout.
#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

// Sums the split partials in order and scatters column n of row m to
// out1[m*D1 + n], out2[m*D2 + n - D1] or out3[m] (the ones column).
__global__ void wgrad_reduce_kernel(const float *__restrict__ P, int splits, int M, int N, int D1, int D2,
                                    float *__restrict__ out1, float *__restrict__ out2, float *__restrict__ out3) {
  const int64_t total = (int64_t)M * N;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int z = 0; z < splits; ++z) s += P[(int64_t)z * total + i];
    const int m = (int)(i / N), n = (int)(i % N);
    if (n < D1) out1[(int64_t)m * D1 + n] = s;
    else if (n < D1 + D2) out2[(int64_t)m * D2 + (n - D1)] = s;
    else out3[m] = s;
  }
}

// Narrow case G[m][n] = sum_k A[k][m] [X[k] | 1][n] with X of D <= 16
// columns: one thread per m keeps D+1 sums over its token range (A read
// coalesced along m, X rows broadcast), partials P[z][m][n] as above.
template <int D>
__global__ void narrow_wgrad_kernel(const float *__restrict__ A, int64_t lda, int M, const float *__restrict__ X,
                                    int K, float *__restrict__ P, int splits) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  const int z = blockIdx.y;
  if (m >= M) return;
  const int chunk = (K + splits - 1) / splits;
  const int k0 = z * chunk, k1 = min(K, k0 + chunk);
  float acc[D + 1];
#pragma unroll
  for (int j = 0; j <= D; ++j) acc[j] = 0.f;
  // eight independent loads of A in flight per thread
  int k = k0;
  for (; k + 8 <= k1; k += 8) {
    float a[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) a[u] = A[(int64_t)(k + u) * lda + m];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
#pragma unroll
      for (int j = 0; j < D; ++j) acc[j] = fmaf(a[u], __ldg(X + (int64_t)(k + u) * D + j), acc[j]);
      acc[D] += a[u];
    }
  }
  for (; k < k1; ++k) {
    const float a = A[(int64_t)k * lda + m];
#pragma unroll
    for (int j = 0; j < D; ++j) acc[j] = fmaf(a, __ldg(X + (int64_t)k * D + j), acc[j]);
    acc[D] += a;
  }
  float *out = P + ((int64_t)z * M + m) * (D + 1);
#pragma unroll
  for (int j = 0; j <= D; ++j) out[j] = acc[j];
}

cudaError_t launch_narrow_wgrad(const float *A, int64_t lda, int M, const float *X, int D, int K, float *P,
                                size_t part_floats, int sm_count, float *out_w, float *out_b, cudaStream_t s) {
  if (M <= 0 || K <= 0) return cudaSuccess;
  const int mb = (M + 255) / 256;
  int splits = std::max(1, std::min(2 * sm_count / mb, K / 32));
  splits = std::min(splits, 1024);
  while (splits > 1 && (size_t)splits * M * (D + 1) > part_floats) --splits;
  dim3 grid(mb, splits);
  switch (D) {
#define BKT_NW(DD) \
  case DD: narrow_wgrad_kernel<DD><<<grid, 256, 0, s>>>(A, lda, M, X, K, P, splits); break;
    BKT_NW(1) BKT_NW(2) BKT_NW(3) BKT_NW(4) BKT_NW(5) BKT_NW(6) BKT_NW(7) BKT_NW(8)
    BKT_NW(9) BKT_NW(10) BKT_NW(11) BKT_NW(12) BKT_NW(13) BKT_NW(14) BKT_NW(15) BKT_NW(16)
#undef BKT_NW
    default: return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t total = (int64_t)M * (D + 1);
  int blocks = (int)std::min<int64_t>(4096, (total + 255) / 256);
  wgrad_reduce_kernel<<<blocks, 256, 0, s>>>(P, splits, M, D + 1, D, 0, out_w, nullptr, out_b);
  return cudaGetLastError();
}

cudaError_t launch_splitk_sum(const float *P, int splits, int M, int N, float *out, cudaStream_t s) {
  const int64_t total = (int64_t)M * N;
  if (total <= 0) return cudaSuccess;
  int blocks = (int)std::min<int64_t>(4096, (total + 255) / 256);
  wgrad_reduce_kernel<<<blocks, 256, 0, s>>>(P, splits, M, N, N, 0, out, nullptr, nullptr);
  return cudaGetLastError();
}

}  // namespace bkt
