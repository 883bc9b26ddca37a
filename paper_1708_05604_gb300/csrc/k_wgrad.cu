// k_wgrad.cu -- reductions over the token axis for the weight gradients
// (a10, a12): the narrow first-layer contraction [dW_ih | db] = dz^T [X | 1]
// (X has in_dim <= 16 columns, so it is a bandwidth-bound pass over dz), and
// the fixed-order sum of split-K partial tiles, scattered straight into the
// flat gradient layout.
#include <algorithm>
#include <cstdint>

#include "bkt_internal.h"

namespace bkt {

// Sums the split partials P[z][i], i < M*N, in a fixed order and scatters
// column n of row m to out1[m*D1 + n], out2[m*D2 + n - D1] or out3[m] (the
// ones column).  A block holds 32 consecutive outputs (coalesced along i);
// its 8 warps take interleaved groups of splits z = g, g+8, ... with four
// independent running sums each (so loads overlap instead of waiting on one
// another), and warp 0 adds the 8 group sums in order: the result depends
// only on `splits`, never on scheduling.
__global__ void __launch_bounds__(256) wgrad_reduce_kernel(const float *__restrict__ P, int splits, int M, int N,
                                                           int D1, int D2, float *__restrict__ out1,
                                                           float *__restrict__ out2, float *__restrict__ out3) {
  __shared__ float part[8][33];
  const int64_t total = (int64_t)M * N;
  const int tx = threadIdx.x & 31, g = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * 32 + tx;
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  if (i < total) {
    int z = g;
    for (; z + 24 < splits; z += 32) {
      a0 += P[(int64_t)z * total + i];
      a1 += P[(int64_t)(z + 8) * total + i];
      a2 += P[(int64_t)(z + 16) * total + i];
      a3 += P[(int64_t)(z + 24) * total + i];
    }
    if (z < splits) a0 += P[(int64_t)z * total + i];
    if (z + 8 < splits) a1 += P[(int64_t)(z + 8) * total + i];
    if (z + 16 < splits) a2 += P[(int64_t)(z + 16) * total + i];
  }
  part[g][tx] = (a0 + a1) + (a2 + a3);
  __syncthreads();
  if (g == 0 && i < total) {
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) s += part[k][tx];
    const int m = (int)(i / N), n = (int)(i % N);
    if (n < D1) out1[(int64_t)m * D1 + n] = s;
    else if (n < D1 + D2) out2[(int64_t)m * D2 + (n - D1)] = s;
    else out3[m] = s;
  }
}

static cudaError_t launch_reduce(const float *P, int splits, int M, int N, int D1, int D2, float *o1, float *o2,
                                 float *o3, cudaStream_t s) {
  const int64_t total = (int64_t)M * N;
  if (total <= 0) return cudaSuccess;
  const int64_t blocks = (total + 31) / 32;
  if (blocks > 0x7fffffff) return cudaErrorInvalidConfiguration;
  wgrad_reduce_kernel<<<(unsigned)blocks, 256, 0, s>>>(P, splits, M, N, D1, D2, o1, o2, o3);
  return cudaGetLastError();
}

// Narrow case G[m][n] = sum_k A[k][m] [X[k] | 1][n] with X of D <= 16
// columns, partials P[z][m][n] over token chunk z.  A bandwidth-bound pass
// over A: with M and lda multiples of 4 a thread keeps 4 (D+1) sums for four
// consecutive columns (otherwise one column).  The block first stages its
// chunk's rows [X | 1] in shared memory, zero past the chunk's end; tokens
// then go in groups of 16 whose A rows are loaded from clamped (always
// valid) rows one group ahead, and a group is summed with plain FMAs against
// the staged rows: no branch and no select stands between a load and the
// loads behind it (a warp issues in order), the ones column forms the bias
// sum and the zero rows cancel the clamped tail.
template <int D, int VEC>
__global__ void __launch_bounds__(128) narrow_wgrad_kernel(const float *__restrict__ A, int64_t lda, int M,
                                                           const float *__restrict__ X, int K,
                                                           float *__restrict__ P, int chunk) {
  constexpr int U = 16, DX = D + 1;
  extern __shared__ float xs[];  // [chunk][D + 1]
  const int z = blockIdx.y;
  const int k0 = z * chunk, k1 = min(K, k0 + chunk);
  for (int i = threadIdx.x; i < chunk * DX; i += blockDim.x) {
    const int k = k0 + i / DX, j = i % DX;
    xs[i] = k < k1 ? (j < D ? X[(int64_t)k * D + j] : 1.f) : 0.f;
  }
  __syncthreads();
  const int m0 = (blockIdx.x * blockDim.x + threadIdx.x) * VEC;
  if (m0 >= M) return;
  float acc[VEC][DX];
#pragma unroll
  for (int c = 0; c < VEC; ++c)
#pragma unroll
    for (int j = 0; j < DX; ++j) acc[c][j] = 0.f;
  const float *acol = A + m0;
  auto load_group = [&](int k, float (&v)[U][VEC]) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const float *row = acol + (int64_t)min(k + u, k1 - 1) * lda;
      if constexpr (VEC == 4) {
        const float4 a = __ldg(reinterpret_cast<const float4 *>(row));
        v[u][0] = a.x;
        v[u][1] = a.y;
        v[u][2] = a.z;
        v[u][3] = a.w;
      } else {
        v[u][0] = __ldg(row);
      }
    }
  };
  auto add_group = [&](int k, const float (&v)[U][VEC]) {
    const float *xr = xs + (k - k0) * DX;
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int j = 0; j < DX; ++j) {
        const float x = xr[u * DX + j];
#pragma unroll
        for (int c = 0; c < VEC; ++c) acc[c][j] = fmaf(v[u][c], x, acc[c][j]);
      }
  };
  float va[U][VEC], vb[U][VEC];
  int k = k0;
  load_group(k, va);
  while (k < k1) {
    if (k + U < k1) load_group(k + U, vb);
    add_group(k, va);
    k += U;
    if (k >= k1) break;
    if (k + U < k1) load_group(k + U, va);
    add_group(k, vb);
    k += U;
  }
#pragma unroll
  for (int c = 0; c < VEC; ++c) {
    float *out = P + ((int64_t)z * M + m0 + c) * DX;
#pragma unroll
    for (int j = 0; j < DX; ++j) out[j] = acc[c][j];
  }
}

cudaError_t launch_narrow_wgrad(const float *A, int64_t lda, int M, const float *X, int D, int K, float *P,
                                size_t part_floats, int sm_count, float *out_w, float *out_b, cudaStream_t s) {
  if (M <= 0 || K <= 0) return cudaSuccess;
  if (D < 1 || D > 16) return cudaErrorInvalidValue;
  const bool vec = (M % 4 == 0) && (lda % 4 == 0) && (reinterpret_cast<uintptr_t>(A) % 16 == 0);
  const int per_thread = vec ? 4 : 1;
  const int mb = (M / per_thread + 127) / 128;
  // at least four blocks of 128 threads per SM when the batch allows (a
  // thread streams 64 tokens or more; chunks are whole 16-token groups), and
  // a chunk's [X | 1] rows within 48 KB of shared memory
  const int max_chunk = std::max(16, (int)((48 * 1024 / (4 * (D + 1))) & ~15));
  int splits = std::max(1, std::max(std::min(4 * sm_count / mb, K / 64), K / 2048));
  splits = std::max(splits, (K + max_chunk - 1) / max_chunk);
  splits = std::min(splits, 1024);
  while (splits > 1 && (size_t)splits * M * (D + 1) > part_floats) --splits;
  const int chunk = (((K + splits - 1) / splits) + 15) & ~15;
  splits = (K + chunk - 1) / chunk;
  const size_t smem = (size_t)chunk * (D + 1) * sizeof(float);
  dim3 grid(mb, splits);
  switch (D) {
#define BKT_NW(DD)                                                                                           \
  case DD: {                                                                                                 \
    const void *kv = vec ? (const void *)narrow_wgrad_kernel<DD, 4> : (const void *)narrow_wgrad_kernel<DD, 1>; \
    if (smem > 48 * 1024) {                                                                                  \
      cudaError_t e = ensure_smem(kv, smem);                                                                 \
      if (e != cudaSuccess) return e;                                                                        \
    }                                                                                                        \
    if (vec) narrow_wgrad_kernel<DD, 4><<<grid, 128, smem, s>>>(A, lda, M, X, K, P, chunk);                 \
    else narrow_wgrad_kernel<DD, 1><<<grid, 128, smem, s>>>(A, lda, M, X, K, P, chunk);                     \
    break;                                                                                                   \
  }
    BKT_NW(1) BKT_NW(2) BKT_NW(3) BKT_NW(4) BKT_NW(5) BKT_NW(6) BKT_NW(7) BKT_NW(8)
    BKT_NW(9) BKT_NW(10) BKT_NW(11) BKT_NW(12) BKT_NW(13) BKT_NW(14) BKT_NW(15) BKT_NW(16)
#undef BKT_NW
    default: return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_reduce(P, splits, M, D + 1, D, 0, out_w, nullptr, out_b, s);
}

cudaError_t launch_splitk_sum(const float *P, int splits, int M, int N, float *out, cudaStream_t s) {
  return launch_reduce(P, splits, M, N, N, 0, out, nullptr, nullptr, s);
}

}  // namespace bkt
