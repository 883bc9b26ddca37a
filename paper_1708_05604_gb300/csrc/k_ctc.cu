// k_ctc.cu -- the CTC forward/backward tables (a8) and the softmax
// gradient (a9).
//
// CTC follows Graves et al. 2006 (the paper's ref. [15]) in log space.  Over
// thousands of steps fp32 log-probabilities reach magnitudes of 1e3-1e4,
// where an fp32 ulp is ~1e-3 and the posterior exp(alpha + beta - ln p)
// would lose three digits.  So each table row is kept relative to a running
// offset: every few steps the row is shifted by its maximum, the shifts are
// summed in double for ln p, and the stored rows hold alpha_t minus the
// offset, values of magnitude tens at most.  The posterior normalises per
// time step,
//   gamma_t(s) = exp(a_t(s) + b_t(s) - lse_s'(a_t(s') + b_t(s'))),
// which is exactly alpha beta / p because sum_s alpha_t(s) beta_t(s) = p at
// every t, and is independent of the offsets.
#include <math_constants.h>

#include "bkt_internal.h"

namespace bkt {

constexpr int kMaxClasses = 128;

// ---------------------------------------------------------------------------
// a8.  One CTA per (row, direction).  Thread i owns extended-label positions
// s = i + j * blockDim (j < SPT).  blockIdx.y = 0 computes
//   alpha_t(s) = lp_t(l'_s) + lse(alpha_{t-1}(s), alpha_{t-1}(s-1),
//                                  [l'_s != blank, l'_s != l'_{s-2}] alpha_{t-1}(s-2)),
// blockIdx.y = 1 the mirror image over time and s,
//   bh_t(s) = lp_t(l'_s) + lse(bh_{t+1}(s), bh_{t+1}(s+1),
//                               [l'_{s+2} != blank, l'_{s+2} != l'_s] bh_{t+1}(s+2)),
// where bh_t(s) = beta_t(s) + lp_t(l'_s) (beta with the emission at t).
// Both start from the two admissible end positions.  Each step keeps one
// CTA barrier: step t reads row t-1 from one shared buffer and writes row t
// into the other.  Every 8 steps the row maximum is reduced (one max per
// warp) and folded in on the next step.  Emissions are prefetched 8 steps
// ahead into registers.
namespace {

// The recursion's serial chain runs T steps; the hardware exp2/log2
// approximations keep each step short.  Their error (a few ulp on arguments
// in (-inf, 0] and on sums in [1, 3]) is re-anchored every step by the
// running-maximum shift, so it does not grow with T.
__device__ __forceinline__ float lse3(float a, float b, float c) {
  const float m = fmaxf(a, fmaxf(b, c));
  if (m == -CUDART_INF_F) return -CUDART_INF_F;
  return m + __logf(__expf(a - m) + __expf(b - m) + __expf(c - m));
}

__device__ __forceinline__ float lse2(float a, float b) {
  const float m = fmaxf(a, b);
  if (m == -CUDART_INF_F) return -CUDART_INF_F;
  return m + __logf(__expf(a - m) + __expf(b - m));
}

constexpr int kPre = 8;  // emission prefetch depth (steps)

// Read-only global load issued where it is written: a volatile asm statement
// keeps the compiler from sinking a prefetch next to its use kPre steps later.
__device__ __forceinline__ float ld_prefetch(const float *p) {
  float v;
  asm volatile("ld.global.nc.f32 %0, [%1];" : "=f"(v) : "l"(p));
  return v;
}

}  // namespace

template <int SPT>
__global__ void __launch_bounds__(512) ctc_tables_kernel(DevIdx ix, const float *__restrict__ logp, int C, int blank,
                                                         const int32_t *__restrict__ labels,
                                                         float *__restrict__ alpha, float *__restrict__ beta,
                                                         float *__restrict__ loss, int32_t *__restrict__ row_ok,
                                                         int32_t *__restrict__ status) {
  extern __shared__ float sm[];
  const int r = blockIdx.x;
  const bool fwd = blockIdx.y == 0;
  const int L = ix.row_len[r];
  const int U = ix.row_lab_len[r];
  const int S = 2 * U + 1;
  const int SP = ix.S_max + 4;
  float *buf0 = sm, *buf1 = sm + SP;
  float *wmax = sm + 2 * SP;  // [2][32]
  int *toff = reinterpret_cast<int *>(wmax + 64);  // [L] packed offsets of this row's time steps
  const int nw = blockDim.x >> 5;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int32_t *lab = labels + ix.row_lab_off[r];
  float *tab = (fwd ? alpha : beta) + ix.row_ctc_off[r];

  // label checks; a bad row is reported and skipped
  int bad = 0;
  for (int u = tid; u < U; u += blockDim.x) {
    const int v = lab[u];
    bad |= (v < 0 || v >= C || v == blank);
  }
  bad = __syncthreads_or(bad);
  if (bad) {
    if (tid == 0 && fwd) {
      atomicOr(status, 1);
      row_ok[r] = 0;
      loss[ix.row_orig[r]] = CUDART_NAN_F;
    }
    return;
  }

  int ext[SPT];
  bool allow2[SPT], valid[SPT];
#pragma unroll
  for (int j = 0; j < SPT; ++j) {
    const int s = tid + j * blockDim.x;
    valid[j] = s < S;
    ext[j] = (s & 1) ? lab[(s - 1) >> 1] : blank;
    allow2[j] = false;
    if (valid[j] && (s & 1)) {
      if (fwd) allow2[j] = s >= 3 && lab[(s - 1) >> 1] != lab[(s - 3) >> 1];
      else allow2[j] = s + 2 < S && lab[(s + 1) >> 1] != lab[(s - 1) >> 1];
    }
    if (!valid[j]) ext[j] = blank;
  }
  // sentinels: both buffers, both ends
  for (int i = tid; i < SP; i += blockDim.x) {
    buf0[i] = -CUDART_INF_F;
    buf1[i] = -CUDART_INF_F;
  }
  // the time offsets live in shared memory: an emission prefetch is then one
  // global load, not two dependent ones
  for (int i = tid; i < L; i += blockDim.x) toff[i] = ix.tok_off[i];
  __syncthreads();

  const float *lprow = logp + (int64_t)r * C;  // token (t, r) = tok_off[t] + r
  auto emis = [&](int step, int j) -> float {
    const int t = fwd ? step : L - 1 - step;
    return ld_prefetch(lprow + (int64_t)toff[t] * C + ext[j]);
  };
  const int d1 = fwd ? -1 : 1, d2 = fwd ? -2 : 2;

  // step 0: the two admissible start positions
  float lmx = -CUDART_INF_F;
#pragma unroll
  for (int j = 0; j < SPT; ++j) {
    const int s = tid + j * blockDim.x;
    if (!valid[j]) continue;
    const bool start = fwd ? (s <= 1) : (s >= S - 2);
    const float v = start ? emis(0, j) : -CUDART_INF_F;
    buf0[s + 2] = v;
    lmx = fmaxf(lmx, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lmx = fmaxf(lmx, __shfl_xor_sync(0xffffffffu, lmx, o));
  if (lane == 0) wmax[wid] = lmx;

  float em[SPT][kPre];
#pragma unroll
  for (int u = 0; u < kPre; ++u)
#pragma unroll
    for (int j = 0; j < SPT; ++j) em[j][u] = (1 + u < L) ? emis(1 + u, j) : 0.f;
  __syncthreads();

  double M = 0.0;  // sum of the row maxima folded in so far
  int p = 0;
  for (int base = 1; base < L; base += kPre) {
#pragma unroll
    for (int u = 0; u < kPre; ++u) {
      const int step = base + u;
      if (step >= L) break;
      const float *cur = p ? buf1 : buf0;
      float *nxt = p ? buf0 : buf1;
      // the row is re-anchored to its maximum every kPre steps; in between a
      // row can rise by at most ln 3 per step, so values stay small
      float mprev = 0.f;
      if (u == 0) {
        const float *wm = wmax + p * 32;
        mprev = wm[0];
        for (int i = 1; i < nw; ++i) mprev = fmaxf(mprev, wm[i]);
      }
      const int tprev = fwd ? step - 1 : L - step;
      float lm = -CUDART_INF_F;
#pragma unroll
      for (int j = 0; j < SPT; ++j) {
        const int s = tid + j * blockDim.x;
        if (!valid[j]) continue;
        const float a0 = cur[s + 2];
        const float a1 = cur[s + 2 + d1];
        const float a2 = allow2[j] ? cur[s + 2 + d2] : -CUDART_INF_F;
        const float l3 = lse3(a0, a1, a2);
        const float v = (l3 == -CUDART_INF_F) ? -CUDART_INF_F : (l3 - mprev) + em[j][u];
        tab[(int64_t)tprev * S + s] = a0 - mprev;
        nxt[s + 2] = v;
        lm = fmaxf(lm, v);
        em[j][u] = (step + kPre < L) ? emis(step + kPre, j) : 0.f;
      }
      if (u == 0 && tid == 0) M += (double)mprev;  // fp64 is slow here: once per re-anchoring, one thread
      if (u == kPre - 1 || step == L - 1) {  // uniform over the CTA
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) lm = fmaxf(lm, __shfl_xor_sync(0xffffffffu, lm, o));
        if (lane == 0) wmax[(p ^ 1) * 32 + wid] = lm;
      }
      p ^= 1;
      __syncthreads();
    }
  }
  // last row: normalise, store, and (forward) finish ln p
  const float *cur = p ? buf1 : buf0;
  const float *wm = wmax + p * 32;
  float mlast = wm[0];
  for (int i = 1; i < nw; ++i) mlast = fmaxf(mlast, wm[i]);
  const int tlast = fwd ? L - 1 : 0;
#pragma unroll
  for (int j = 0; j < SPT; ++j) {
    const int s = tid + j * blockDim.x;
    if (valid[j]) tab[(int64_t)tlast * S + s] = cur[s + 2] - mlast;
  }
  if (fwd && tid == 0) {
    const float e1 = cur[S - 1 + 2];
    const float e2 = S >= 2 ? cur[S - 2 + 2] : -CUDART_INF_F;
    const float l2 = lse2(e1, e2);
    const bool ok = l2 != -CUDART_INF_F;
    row_ok[r] = ok ? 1 : 0;
    loss[ix.row_orig[r]] = ok ? (float)(-(M + (double)l2)) : CUDART_INF_F;
  }
}

cudaError_t launch_ctc_tables(const DevIdx &ix, const float *logp, int C, int blank, const int32_t *labels,
                              float *alpha, float *beta, float *loss, int32_t *row_ok, int32_t *status,
                              cudaStream_t s) {
  const int S = ix.S_max;
  int spt = 1;
  while (spt < 4 && (S + spt - 1) / spt > 512) spt *= 2;
  if ((S + spt - 1) / spt > 512) return cudaErrorInvalidValue;
  int threads = ((S + spt - 1) / spt + 31) / 32 * 32;
  const size_t smem = (size_t)(2 * (S + 4) + 64 + ix.T) * sizeof(float);
  if (smem > 48 * 1024) {
    const void *k = spt == 1 ? (const void *)ctc_tables_kernel<1>
                             : spt == 2 ? (const void *)ctc_tables_kernel<2> : (const void *)ctc_tables_kernel<4>;
    cudaError_t e = ensure_smem(k, smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid(ix.b, 2);
  switch (spt) {
    case 1: ctc_tables_kernel<1><<<grid, threads, smem, s>>>(ix, logp, C, blank, labels, alpha, beta, loss, row_ok, status); break;
    case 2: ctc_tables_kernel<2><<<grid, threads, smem, s>>>(ix, logp, C, blank, labels, alpha, beta, loss, row_ok, status); break;
    default: ctc_tables_kernel<4><<<grid, threads, smem, s>>>(ix, logp, C, blank, labels, alpha, beta, loss, row_ok, status); break;
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a9.  One warp per token (t, r):
//   v(s) = a_t(s) + bh_t(s) - lp_t(l'_s)  (log of alpha_t(s) beta_t(s), offset)
//   gamma(s) = exp(v(s) - lse_s v)
//   dlogit[k] = exp(lp_t(k)) - sum_{s: l'_s = k} gamma(s)
// written over the log-probabilities in place.  Blank mass is a warp sum;
// label mass goes through a per-warp shared row.  Rows without an alignment
// (or with a bad label) get zeros.
__global__ void __launch_bounds__(256) ctc_grad_kernel(DevIdx ix, float *__restrict__ lp_dl, int C, int blank,
                                                       const int32_t *__restrict__ labels,
                                                       const float *__restrict__ alpha,
                                                       const float *__restrict__ beta,
                                                       const int32_t *__restrict__ row_ok) {
  __shared__ float acc[8][kMaxClasses];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int tok = blockIdx.x * 8 + w;
  if (tok >= ix.n_tok) return;
  const int t = ix.tok_t[tok], r = ix.tok_r[tok];
  float *row = lp_dl + (int64_t)tok * C;
  float lpk[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) lpk[j] = (lane + 32 * j < C) ? row[lane + 32 * j] : 0.f;
#pragma unroll
  for (int j = 0; j < 4; ++j) acc[w][lane + 32 * j] = 0.f;
  float out[4] = {0.f, 0.f, 0.f, 0.f};
  if (row_ok[r]) {
    const int U = ix.row_lab_len[r], S = 2 * U + 1;
    const int32_t *lab = labels + ix.row_lab_off[r];
    const float *a = alpha + ix.row_ctc_off[r] + (int64_t)t * S;
    const float *b = beta + ix.row_ctc_off[r] + (int64_t)t * S;
    const float lpb = row[blank];
    float mx = -CUDART_INF_F;
    for (int s = lane; s < S; s += 32) {
      const float e = (s & 1) ? row[lab[(s - 1) >> 1]] : lpb;
      mx = fmaxf(mx, a[s] + b[s] - e);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float se = 0.f;
    for (int s = lane; s < S; s += 32) {
      const float e = (s & 1) ? row[lab[(s - 1) >> 1]] : lpb;
      se += expf(a[s] + b[s] - e - mx);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
    const float lz = mx + logf(se);
    float blank_mass = 0.f;
    __syncwarp();
    for (int s = lane; s < S; s += 32) {
      const int k = (s & 1) ? lab[(s - 1) >> 1] : blank;
      const float e = (s & 1) ? row[k] : lpb;
      const float g = expf(a[s] + b[s] - e - lz);
      if (s & 1) atomicAdd(&acc[w][k], g);
      else blank_mass += g;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) blank_mass += __shfl_xor_sync(0xffffffffu, blank_mass, o);
    __syncwarp();
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int k = lane + 32 * j;
      out[j] = expf(lpk[j]) - acc[w][k] - (k == blank ? blank_mass : 0.f);
    }
  }
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (lane + 32 * j < C) row[lane + 32 * j] = out[j];
}

cudaError_t launch_ctc_grad(const DevIdx &ix, float *lp_dl, int C, int blank, const int32_t *labels,
                            const float *alpha, const float *beta, const int32_t *row_ok, cudaStream_t s) {
  if (C > kMaxClasses) return cudaErrorInvalidValue;
  const int blocks = (ix.n_tok + 7) / 8;
  ctc_grad_kernel<<<blocks, 256, 0, s>>>(ix, lp_dl, C, blank, labels, alpha, beta, row_ok);
  return cudaGetLastError();
}

}  // namespace bkt
