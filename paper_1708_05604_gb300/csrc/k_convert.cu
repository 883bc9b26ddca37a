// k_convert.cu -- operand preparation for the bf16 tensor-core contractions
// (all HBM-bound):
//   cast_bf16:      fp32 [R x C] -> bf16 [R x C] (row-major, own strides;
//                   optionally reading row src_row[r] instead of r, a
//                   negative index giving zeros)
//   colsum:         P[z][m] = sum over the rows of chunk z of A[r][m]
// The bf16 GEMM reads token-major operands directly (MN-major tiles), so the
// contractions over tokens need only bf16 copies of dz, h_{t-1} and the layer
// input, which the tensor-core recurrent kernels write themselves; the casts
// here serve the other recurrent kernels.
#include <cuda_bf16.h>

#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

__global__ void cast_bf16_kernel(const float *__restrict__ src, int64_t lds, const int32_t *__restrict__ src_row,
                                 int R, int C, __nv_bfloat16 *__restrict__ dst, int64_t ldd) {
  const int c2 = C / 2;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < (int64_t)R * c2;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(i / c2), c = (int)(i % c2) * 2;
    const int sr = src_row ? src_row[r] : r;
    const float2 v = sr >= 0 ? *reinterpret_cast<const float2 *>(src + (int64_t)sr * lds + c) : make_float2(0.f, 0.f);
    *reinterpret_cast<__nv_bfloat162 *>(dst + (int64_t)r * ldd + c) = __floats2bfloat162_rn(v.x, v.y);
  }
  if (C & 1)
    for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
      const int sr = src_row ? src_row[r] : (int)r;
      dst[r * ldd + C - 1] = __float2bfloat16_rn(sr >= 0 ? src[(int64_t)sr * lds + C - 1] : 0.f);
    }
}

cudaError_t launch_gather_cast_bf16(const float *src, int64_t lds, const int32_t *src_row, int R, int C, void *dst,
                                    int64_t ldd, cudaStream_t s) {
  if (R <= 0 || C <= 0) return cudaSuccess;
  if ((lds & 1) || (ldd & 1) || (reinterpret_cast<uintptr_t>(src) & 7) || (reinterpret_cast<uintptr_t>(dst) & 3))
    return cudaErrorInvalidValue;
  const int64_t work = (int64_t)R * (C / 2 + 1);
  const int blocks = (int)std::min<int64_t>(8192, (work + 255) / 256);
  cast_bf16_kernel<<<blocks, 256, 0, s>>>(src, lds, src_row, R, C, reinterpret_cast<__nv_bfloat16 *>(dst), ldd);
  return cudaGetLastError();
}

cudaError_t launch_cast_bf16(const float *src, int64_t lds, int R, int C, void *dst, int64_t ldd, cudaStream_t s) {
  return launch_gather_cast_bf16(src, lds, nullptr, R, C, dst, ldd, s);
}

// fp32 [R x C] -> two fp32 [C x R] arrays hi, lo, each a tf32 value (11
// significant bits) with |x - hi - lo| <= 2^-22 |x|, for the split-precision
// tensor-core GEMM; optional row gather as above.
__global__ void transpose_split_kernel(const float *__restrict__ src, int64_t lds, const int32_t *__restrict__ src_row,
                                       int R, int C, float *__restrict__ hi, float *__restrict__ lo, int64_t ldd) {
  __shared__ float tile[32][33];
  const int r0 = blockIdx.x * 32, c0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
#pragma unroll
  for (int i = 0; i < 32; i += 8) {
    const int r = r0 + ty + i, c = c0 + tx;
    float v = 0.f;
    if (r < R && c < C) {
      const int sr = src_row ? src_row[r] : r;
      if (sr >= 0) v = src[(int64_t)sr * lds + c];
    }
    tile[ty + i][tx] = v;
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < 32; i += 8) {
    const int c = c0 + ty + i, r = r0 + tx;
    if (c < C && r < R) {
      // both parts rounded to the nearest tf32 value (11 significant bits),
      // so the tensor core uses them exactly: |x - hi - lo| <= 2^-22 |x|
      const float x = tile[tx][ty + i];
      const float h = __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
      const float l = __uint_as_float((__float_as_uint(x - h) + 0x1000u) & 0xFFFFE000u);
      hi[(int64_t)c * ldd + r] = h;
      lo[(int64_t)c * ldd + r] = l;
    }
  }
}

cudaError_t launch_transpose_split(const float *src, int64_t lds, const int32_t *src_row, int R, int C, float *hi,
                                   float *lo, int64_t ldd, cudaStream_t s) {
  if (R <= 0 || C <= 0) return cudaSuccess;
  dim3 grid((R + 31) / 32, (C + 31) / 32);
  if (grid.y > 65535u) return cudaErrorInvalidConfiguration;
  transpose_split_kernel<<<grid, dim3(32, 8), 0, s>>>(src, lds, src_row, R, C, hi, lo, ldd);
  return cudaGetLastError();
}

// fp32 [R x C] (stride lds) -> hi, lo [R x C] (stride ldd >= C) as in the
// transposing split; padding columns C..ldd-1 are left untouched.
__global__ void split_rows_kernel(const float *__restrict__ src, int64_t lds, int R, int C, float *__restrict__ hi,
                                  float *__restrict__ lo, int64_t ldd) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < (int64_t)R * C;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(i / C), c = (int)(i % C);
    const float x = src[(int64_t)r * lds + c];
    const float h = __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
    const float l = __uint_as_float((__float_as_uint(x - h) + 0x1000u) & 0xFFFFE000u);
    hi[(int64_t)r * ldd + c] = h;
    lo[(int64_t)r * ldd + c] = l;
  }
}

cudaError_t launch_split_rows(const float *src, int64_t lds, int R, int C, float *hi, float *lo, int64_t ldd,
                              cudaStream_t s) {
  if (R <= 0 || C <= 0) return cudaSuccess;
  const int blocks = (int)std::min<int64_t>(8192, ((int64_t)R * C + 255) / 256);
  split_rows_kernel<<<blocks, 256, 0, s>>>(src, lds, R, C, hi, lo, ldd);
  return cudaGetLastError();
}

// P[z][m] = sum of A[r][m] over the rows of chunk z (ceil(R / splits) rows).
// A block holds 32 columns (coalesced along m); its 8 warps take rows
// r0 + g, r0 + g + 8, ... with four running sums each, and warp 0 adds the 8
// group sums in a fixed order.
__global__ void __launch_bounds__(256) colsum_kernel(const float *__restrict__ A, int64_t lda, int R, int M,
                                                     float *__restrict__ P, int chunk) {
  __shared__ float part[8][33];
  const int tx = threadIdx.x & 31, g = threadIdx.x >> 5;
  const int m = blockIdx.x * 32 + tx, z = blockIdx.y;
  const int r0 = z * chunk, r1 = min(R, r0 + chunk);
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  if (m < M) {
    int r = r0 + g;
    for (; r + 24 < r1; r += 32) {
      a0 += A[(int64_t)r * lda + m];
      a1 += A[(int64_t)(r + 8) * lda + m];
      a2 += A[(int64_t)(r + 16) * lda + m];
      a3 += A[(int64_t)(r + 24) * lda + m];
    }
    if (r < r1) a0 += A[(int64_t)r * lda + m];
    if (r + 8 < r1) a1 += A[(int64_t)(r + 8) * lda + m];
    if (r + 16 < r1) a2 += A[(int64_t)(r + 16) * lda + m];
  }
  part[g][tx] = (a0 + a1) + (a2 + a3);
  __syncthreads();
  if (g == 0 && m < M) {
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) s += part[k][tx];
    P[(int64_t)z * M + m] = s;
  }
}

int colsum_splits(int R, int M, size_t part_floats) {
  const size_t cap = M > 0 ? part_floats / (size_t)M : 1;
  return (int)std::max<size_t>(1, std::min<size_t>(std::min<size_t>((R + 255) / 256, cap), 65535));
}

cudaError_t launch_colsum(const float *A, int64_t lda, int R, int M, float *P, int splits, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (splits < 1 || splits > 65535) return cudaErrorInvalidValue;
  const int chunk = (R + splits - 1) / splits;
  dim3 grid((M + 31) / 32, splits);
  colsum_kernel<<<grid, 256, 0, s>>>(A, lda, R, M, P, chunk);
  return cudaGetLastError();
}

}  // namespace bkt
