// k_misc.cu -- the bandwidth-bound kernels of the step: the packed-layout
// gather (a4), the narrow input projection (a5 for in_dim <= 16) and the SGD
// update (a13).
#include "bkt_internal.h"

namespace bkt {

// ---------------------------------------------------------------------------
// a4.  One CTA per time step t; thread r < batch_size(t) owns token
// (t, r) = tok_off[t] + r.  The caller's rows are read where they lie
// (x + (row_xoff[r] + t) * in_dim), so the batch can be any subset of a
// resident dataset.
__global__ void layout_kernel(DevIdx ix, const float *__restrict__ x, int in_dim,
                              float *__restrict__ X, int32_t *__restrict__ tok_t,
                              int32_t *__restrict__ tok_r, int32_t *__restrict__ prev_f,
                              int32_t *__restrict__ prev_b) {
  const int t = blockIdx.x;
  const int base = ix.tok_off[t];
  const int nb = ix.tok_off[t + 1] - base;
  for (int r = threadIdx.x; r < nb; r += blockDim.x) {
    const int tok = base + r;
    tok_t[tok] = t;
    tok_r[tok] = r;
    prev_f[tok] = t > 0 ? ix.tok_off[t - 1] + r : -1;
    prev_b[tok] = (t + 1 < ix.row_len[r]) ? ix.tok_off[t + 1] + r : -1;
    const float *src = x + (ix.row_xoff[r] + t) * (int64_t)in_dim;
    float *dst = X + (int64_t)tok * in_dim;
    if (in_dim == 4 && ((reinterpret_cast<uintptr_t>(src) & 15) == 0)) {
      *reinterpret_cast<float4 *>(dst) = __ldg(reinterpret_cast<const float4 *>(src));
    } else {
      for (int k = 0; k < in_dim; ++k) dst[k] = __ldg(src + k);
    }
  }
}

cudaError_t launch_layout(const DevIdx &ix, const float *x, int in_dim, float *X, int32_t *tok_t,
                          int32_t *tok_r, int32_t *const *prev_tok, cudaStream_t s) {
  int threads = ((ix.b + 31) / 32) * 32;
  if (threads > 1024) threads = 1024;
  layout_kernel<<<ix.T, threads, 0, s>>>(ix, x, in_dim, X, tok_t, tok_r, prev_tok[0], prev_tok[1]);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a5 with a narrow input.  A CTA stages its chunk of token rows of X in
// shared memory; thread i owns output columns 4i .. 4i+3 of one direction
// (their W rows and biases in registers) and writes each token's four values
// as one 16-byte store, coalesced along n; no FMA waits on a global load.
constexpr int kProjTok = 64;

template <int D>
__global__ void __launch_bounds__(128) proj_narrow_kernel(const float *__restrict__ X, int n_tok,
                                                         const float *__restrict__ params, int64_t w_off,
                                                         int64_t w_stride, int H, float *Z0, float *Z1) {
  __shared__ float xs[kProjTok * D];
  const int d = blockIdx.z;
  const int G = 4 * H;
  const int t0 = blockIdx.y * kProjTok;
  const int t1 = min(n_tok, t0 + kProjTok);
  for (int i = threadIdx.x; i < (t1 - t0) * D; i += blockDim.x) xs[i] = X[(int64_t)t0 * D + i];
  __syncthreads();
  const int n0 = 4 * (blockIdx.x * 128 + threadIdx.x);  // this thread's outputs n0 .. n0+3 (4H % 4 == 0)
  if (n0 >= G) return;
  const float *W = params + w_off + d * w_stride;
  const float *bias = W + (int64_t)G * D + (int64_t)G * H;
  float w[4][D], bn[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
#pragma unroll
    for (int k = 0; k < D; ++k) w[c][k] = W[(int64_t)(n0 + c) * D + k];
    bn[c] = bias[n0 + c];
  }
  float *Z = d == 0 ? Z0 : Z1;
  for (int tok = t0; tok < t1; ++tok) {
    const float *x = xs + (tok - t0) * D;
    float4 z = make_float4(bn[0], bn[1], bn[2], bn[3]);
#pragma unroll
    for (int k = 0; k < D; ++k) {
      const float xk = x[k];
      z.x = fmaf(w[0][k], xk, z.x);
      z.y = fmaf(w[1][k], xk, z.y);
      z.z = fmaf(w[2][k], xk, z.z);
      z.w = fmaf(w[3][k], xk, z.w);
    }
    *reinterpret_cast<float4 *>(Z + (int64_t)tok * G + n0) = z;
  }
}

cudaError_t launch_proj_narrow(const float *X, int n_tok, int in_dim, const float *params, int64_t w_off,
                               int64_t w_stride, int H, int dirs, float *const *Z, cudaStream_t s) {
  dim3 grid((H + 127) / 128, (n_tok + kProjTok - 1) / kProjTok, dirs);  // 4H outputs, 4 per thread
  float *Z1 = dirs > 1 ? Z[1] : Z[0];
  if (((reinterpret_cast<uintptr_t>(Z[0]) | reinterpret_cast<uintptr_t>(Z1)) & 15) != 0) return cudaErrorInvalidValue;
  switch (in_dim) {
#define BKT_CASE(D) \
  case D:           \
    proj_narrow_kernel<D><<<grid, 128, 0, s>>>(X, n_tok, params, w_off, w_stride, H, Z[0], Z1); \
    break;
    BKT_CASE(1) BKT_CASE(2) BKT_CASE(3) BKT_CASE(4) BKT_CASE(5) BKT_CASE(6) BKT_CASE(7) BKT_CASE(8)
    BKT_CASE(9) BKT_CASE(10) BKT_CASE(11) BKT_CASE(12) BKT_CASE(13) BKT_CASE(14) BKT_CASE(15) BKT_CASE(16)
#undef BKT_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a13: theta <- theta - lr * g, 16-byte vectors over the aligned body.
__global__ void sgd_kernel(float *__restrict__ p, const float *__restrict__ g, int64_t n, float lr, int vec) {
  const int64_t n4 = vec ? n / 4 : 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  float4 *p4 = reinterpret_cast<float4 *>(p);
  const float4 *g4 = reinterpret_cast<const float4 *>(g);
  for (int64_t i = i0; i < n4; i += stride) {
    float4 a = p4[i];
    const float4 b = g4[i];
    a.x = fmaf(-lr, b.x, a.x);
    a.y = fmaf(-lr, b.y, a.y);
    a.z = fmaf(-lr, b.z, a.z);
    a.w = fmaf(-lr, b.w, a.w);
    p4[i] = a;
  }
  for (int64_t i = n4 * 4 + i0; i < n; i += stride) p[i] = fmaf(-lr, g[i], p[i]);
}

cudaError_t launch_sgd(float *p, const float *g, int64_t n, float lr, cudaStream_t s) {
  const int vec = ((reinterpret_cast<uintptr_t>(p) | reinterpret_cast<uintptr_t>(g)) & 15) == 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (n / 4 + 255) / 256;
  if (blocks > 4LL * sms) blocks = 4LL * sms;
  if (blocks < 1) blocks = 1;
  sgd_kernel<<<(int)blocks, 256, 0, s>>>(p, g, n, lr, vec);
  return cudaGetLastError();
}

// a13 with ADADELTA (Zeiler 2012, Algorithm 1): three running arrays per
// parameter, 28 bytes of HBM traffic per parameter.
__device__ __forceinline__ void adadelta_one(float &p, float g, float &eg2, float &edx2, float rho, float eps,
                                             float lr) {
  eg2 = fmaf(rho, eg2, (1.f - rho) * (g * g));
  const float dx = sqrtf(edx2 + eps) / sqrtf(eg2 + eps) * g;
  edx2 = fmaf(rho, edx2, (1.f - rho) * (dx * dx));
  p = fmaf(-lr, dx, p);
}

__global__ void adadelta_kernel(float *__restrict__ p, const float *__restrict__ g, float *__restrict__ eg2,
                                float *__restrict__ edx2, int64_t n, float rho, float eps, float lr, int vec) {
  const int64_t n4 = vec ? n / 4 : 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  for (int64_t i = i0; i < n4; i += stride) {
    float4 a = reinterpret_cast<float4 *>(p)[i];
    const float4 b = reinterpret_cast<const float4 *>(g)[i];
    float4 e = reinterpret_cast<float4 *>(eg2)[i];
    float4 x = reinterpret_cast<float4 *>(edx2)[i];
    adadelta_one(a.x, b.x, e.x, x.x, rho, eps, lr);
    adadelta_one(a.y, b.y, e.y, x.y, rho, eps, lr);
    adadelta_one(a.z, b.z, e.z, x.z, rho, eps, lr);
    adadelta_one(a.w, b.w, e.w, x.w, rho, eps, lr);
    reinterpret_cast<float4 *>(p)[i] = a;
    reinterpret_cast<float4 *>(eg2)[i] = e;
    reinterpret_cast<float4 *>(edx2)[i] = x;
  }
  for (int64_t i = n4 * 4 + i0; i < n; i += stride) adadelta_one(p[i], g[i], eg2[i], edx2[i], rho, eps, lr);
}

cudaError_t launch_adadelta(float *p, const float *g, float *eg2, float *edx2, int64_t n, float rho, float eps,
                            float lr, cudaStream_t s) {
  const uintptr_t any = reinterpret_cast<uintptr_t>(p) | reinterpret_cast<uintptr_t>(g) |
                        reinterpret_cast<uintptr_t>(eg2) | reinterpret_cast<uintptr_t>(edx2);
  const int vec = (any & 15) == 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (n / 4 + 255) / 256;
  if (blocks > 4LL * sms) blocks = 4LL * sms;
  if (blocks < 1) blocks = 1;
  adadelta_kernel<<<(int)blocks, 256, 0, s>>>(p, g, eg2, edx2, n, rho, eps, lr, vec);
  return cudaGetLastError();
}

// Section III.B step 5, eq. 3 (alpha = 1): v[i] <- v[i] / K - beta prev[i],
// with v the element-wise sum of the K replicas' parameters (what an
// all-reduce with the sum operation leaves on every replica): an IEEE
// division, then one fused multiply-add; 12 bytes of HBM traffic per
// parameter.
__global__ void average_models_kernel(float *__restrict__ v, const float *__restrict__ prev, int64_t n, float K,
                                      float beta, int vec) {
  const int64_t n4 = vec ? n / 4 : 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  for (int64_t i = i0; i < n4; i += stride) {
    float4 a = reinterpret_cast<float4 *>(v)[i];
    const float4 b = reinterpret_cast<const float4 *>(prev)[i];
    a.x = fmaf(-beta, b.x, __fdiv_rn(a.x, K));
    a.y = fmaf(-beta, b.y, __fdiv_rn(a.y, K));
    a.z = fmaf(-beta, b.z, __fdiv_rn(a.z, K));
    a.w = fmaf(-beta, b.w, __fdiv_rn(a.w, K));
    reinterpret_cast<float4 *>(v)[i] = a;
  }
  for (int64_t i = n4 * 4 + i0; i < n; i += stride) v[i] = fmaf(-beta, prev[i], __fdiv_rn(v[i], K));
}

cudaError_t launch_average_models(float *v, const float *prev, int64_t n, int K, float beta, cudaStream_t s) {
  const int vec = ((reinterpret_cast<uintptr_t>(v) | reinterpret_cast<uintptr_t>(prev)) & 15) == 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (n / 4 + 255) / 256;
  if (blocks > 4LL * sms) blocks = 4LL * sms;
  if (blocks < 1) blocks = 1;
  average_models_kernel<<<(int)blocks, 256, 0, s>>>(v, prev, n, (float)K, beta, vec);
  return cudaGetLastError();
}

}  // namespace bkt
