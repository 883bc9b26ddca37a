// k_wgrad.cu -- fused weight-gradient contraction over the token axis (a10,
// a12), fp32 FMA:
//   G[m][n] = sum_k A[k][m] * Bv[k][n]
// where A is dZ (or dlogit) [tokens x M] and Bv is a virtual [tokens x N]
// matrix [ B1[k] | B2[gather(k)] | 1 ]: the layer input X (for dW_ih), the
// previous-step hidden state h_{t-1} of the same row and direction (for
// dW_hh; rows with no previous step read zeros), and a column of ones (for
// the bias).  One pass reads dZ once for all three gradients.
//
// Tiles of 128 (M) x 64 (N) per CTA, 8-token k slabs double-buffered through
// registers, 256 threads with an 8 x 4 register tile each.  The token range is
// split across gridDim.z; partial tiles are summed in a fixed order by the
// scatter-reduce, which writes straight into the flat gradient layout.
#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

namespace {
constexpr int WM = 128, WN = 64, WK = 8;
}

template <bool VA>
__global__ void __launch_bounds__(256) wgrad_kernel(WgradArgs g) {
  __shared__ __align__(16) float As[2][WK][WM];
  __shared__ __align__(16) float Bs[2][WK][WN];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.x * WM, n0 = blockIdx.y * WN, z = blockIdx.z;
  int chunk = (g.K + g.splits - 1) / g.splits;
  chunk = (chunk + WK - 1) / WK * WK;
  const int kb = z * chunk, ke = min(g.K, kb + chunk);
  const int D12 = g.D1 + g.D2;

  // per-thread load coordinates
  const int ak = tid >> 5, am = (tid & 31) * 4;  // A: one float4 (or 4 scalars) per thread
  float4 ra;
  float rb[2];
  auto load_a = [&](int k0) {
    const int k = k0 + ak, m = m0 + am;
    if (k < ke) {
      const float *src = g.A + (int64_t)k * g.lda + m;
      if (VA && m + 3 < g.M) {
        ra = *reinterpret_cast<const float4 *>(src);
      } else {
        ra.x = (m < g.M) ? src[0] : 0.f;
        ra.y = (m + 1 < g.M) ? src[1] : 0.f;
        ra.z = (m + 2 < g.M) ? src[2] : 0.f;
        ra.w = (m + 3 < g.M) ? src[3] : 0.f;
      }
    } else {
      ra = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  auto load_b = [&](int k0) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int e = tid + i * 256;
      const int kk = e >> 6, nn = e & 63;
      const int k = k0 + kk, n = n0 + nn;
      float v = 0.f;
      if (k < ke && n < g.N) {
        if (n < g.D1) {
          v = g.B1[(int64_t)k * g.ldb1 + n];
        } else if (n < D12) {
          const int row = g.gather2 ? g.gather2[k] : k;
          if (row >= 0) v = g.B2[(int64_t)row * g.ldb2 + (n - g.D1)];
        } else {
          v = 1.f;
        }
      }
      rb[i] = v;
    }
  };
  auto store = [&](int buf) {
    *reinterpret_cast<float4 *>(&As[buf][ak][am]) = ra;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int e = tid + i * 256;
      Bs[buf][e >> 6][e & 63] = rb[i];
    }
  };

  float acc[8][4];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  if (kb < ke) {
    load_a(kb);
    load_b(kb);
    store(0);
  }
  __syncthreads();
  int buf = 0;
  for (int k0 = kb; k0 < ke; k0 += WK) {
    const bool more = k0 + WK < ke;
    if (more) {
      load_a(k0 + WK);
      load_b(k0 + WK);
    }
#pragma unroll
    for (int kk = 0; kk < WK; ++kk) {
      const float4 a0 = *reinterpret_cast<const float4 *>(&As[buf][kk][ty * 8]);
      const float4 a1 = *reinterpret_cast<const float4 *>(&As[buf][kk][ty * 8 + 4]);
      const float4 b = *reinterpret_cast<const float4 *>(&Bs[buf][kk][tx * 4]);
      const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    if (more) store(buf ^ 1);
    __syncthreads();
    buf ^= 1;
  }
  float *P = g.P + (int64_t)z * g.M * g.N;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = m0 + ty * 8 + i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n < g.N) P[(int64_t)m * g.N + n] = acc[i][j];
    }
  }
}

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

int wgrad_splits(int M, int N, int K, int sm_count, size_t part_floats) {
  const int tiles = ((M + WM - 1) / WM) * ((N + WN - 1) / WN);
  int s = (2 * sm_count + tiles - 1) / tiles;
  s = std::min(s, std::max(1, K / 64));
  s = std::max(1, std::min(s, 64));
  while (s > 1 && (size_t)s * M * N > part_floats) --s;
  return s;
}

cudaError_t launch_wgrad(const WgradArgs &g, float *out1, float *out2, float *out3, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.splits < 1 || g.N != g.D1 + g.D2 + g.ones) return cudaErrorInvalidValue;
  dim3 grid((g.M + WM - 1) / WM, (g.N + WN - 1) / WN, g.splits);
  const bool va = (g.lda % 4 == 0) && ((reinterpret_cast<uintptr_t>(g.A) & 15) == 0);
  if (va) wgrad_kernel<true><<<grid, 256, 0, s>>>(g);
  else wgrad_kernel<false><<<grid, 256, 0, s>>>(g);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t total = (int64_t)g.M * g.N;
  int blocks = (int)std::min<int64_t>(4096, (total + 255) / 256);
  wgrad_reduce_kernel<<<blocks, 256, 0, s>>>(g.P, g.splits, g.M, g.N, g.D1, g.D2, out1, out2, out3);
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
