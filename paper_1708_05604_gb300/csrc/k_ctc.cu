// k_ctc.cu -- the CTC forward/backward tables (a8) and the softmax
// gradient (a9).
//
// CTC follows Graves et al. 2006 (the paper's ref. [15]) in log space, kept
// here in base-2 logarithms so that the recursion's exponentials and
// logarithms are the hardware exp2/log2 without a scale.  Over thousands of
// steps fp32 log-probabilities reach magnitudes of 1e3-1e4, where an fp32 ulp
// is ~1e-3 and the posterior exp(alpha + beta - ln p) would lose three digits.
// So each table row is kept relative to a running offset: every 8 steps the
// row is shifted by a recent row maximum, the shifts are summed in double for
// ln p, and the stored rows hold log2 alpha_t minus the offset, values of
// magnitude tens at most.  The posterior normalises per time step,
//   gamma_t(s) = 2^(a_t(s) + b_t(s) - lse2_s'(a_t(s') + b_t(s'))),
// which is exactly alpha beta / p because sum_s alpha_t(s) beta_t(s) = p at
// every t, and is independent of the offsets.
//
// An entry no path reaches holds the finite value kNeg = -1e30 instead of
// -inf: the log-sum-exp then needs no special case (2^(kNeg - m) is 0 and
// kNeg plus a term of ordinary size is kNeg), and a sequence has no
// alignment when its end value is below kDead = -1e20 (a log2-probability no
// finite fp32 input of ordinary range reaches).
#include <math_constants.h>

#include <cstdlib>

#include "bkt_internal.h"

namespace bkt {

constexpr int kMaxClasses = 128;

namespace {
constexpr float kLog2e = 1.4426950408889634f;
constexpr double kLn2 = 0.6931471805599453;
constexpr float kNeg = -1e30f;
constexpr float kDead = -1e20f;
}  // namespace

// ---------------------------------------------------------------------------
// a8.  One CTA of W warps per (row, direction); blockIdx.y = 0 computes the
// forward table
//   alpha_t(s) = lp_t(l'_s) + lse(alpha_{t-1}(s), alpha_{t-1}(s-1),
//                                  [l'_s != blank, l'_s != l'_{s-2}] alpha_{t-1}(s-2)),
// blockIdx.y = 1 the table bh_t(s) = beta_t(s) + lp_t(l'_s) (beta with the
// emission at t), whose recursion runs backwards in time and over s+1, s+2.
// Both directions run the same code: the backward one works on the reversed
// position p = S-1-s with the reversed label string, where its recursion
// reads p-1, p-2 like the forward one and its skip rule becomes the forward
// rule, and on reversed time.  Both start from positions p in {0, 1}.
//
// Lane l of warp w owns the K consecutive positions p = (32w + l) K + j and
// keeps its part of the previous row in registers: the two values below its
// first position come from the lane below by a shuffle, and across warps from
// a two-value exchange slot per warp that the step's CTA barrier publishes
// (W = 1 needs no barrier).  With K even, position parity is fixed per j, so
// the blank positions (two-term lse) and the label positions (three-term lse,
// the skip term masked by adding kNeg where the rule forbids it) never
// diverge within a warp.  Positions past S are never stored and never feed a
// position below S.
//
// A lane loads its own K emissions of each step with plain read-only loads
// kBlock steps ahead into registers: the loop body is unrolled over two blocks
// of kBlock steps, consuming one register buffer while filling the other, so
// no loaded value is moved before use.  The body has no branch (loads past
// the end read the last row again) and the warp count is a template
// parameter, so the compiler can schedule loads, stores and the exchange into
// the gaps of the serial chain; a warp issues in order, and a branch would
// put each piece's latency on the chain.  At the start of every block the row
// is shifted by the row maximum taken two steps earlier (its reduction
// overlaps a step), rounded down to a whole number.
namespace {

constexpr int kBlock = 8;  // steps between re-anchorings; emissions are loaded this many steps ahead

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// log2(2^a + 2^b) and log2(2^a + 2^b + 2^c): the largest term is 2^0 = 1 and
// is not evaluated.  The approximations' error (a few ulp on arguments in
// (-inf, 0] and on sums in [1, 3]) does not grow with T: every step adds it
// once to values of ordinary size.
__device__ __forceinline__ float lse2b(float a, float b) {
  const float m = fmaxf(a, b);
  return m + lg2(1.f + ex2(fminf(a, b) - m));
}
__device__ __forceinline__ float lse3b(float a, float b, float c) {
  const float hi = fmaxf(a, b), lo = fminf(a, b);
  const float m = fmaxf(hi, c), mid = fminf(hi, c);
  return m + lg2(1.f + ex2(mid - m) + ex2(lo - m));
}

// A read-only load issued where it is written: the volatile statement keeps
// the compiler from sinking the prefetch next to its use kBlock steps later.
__device__ __forceinline__ float ld_prefetch(const float *p) {
  float v;
  asm volatile("ld.global.nc.f32 %0, [%1];" : "=f"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

}  // namespace

size_t ctc_tables_smem(int W, int T) { return (6 * (size_t)W + 4) * sizeof(float) + (size_t)T * sizeof(int32_t); }

template <int K, bool MW>
__global__ void __launch_bounds__(K >= 16 ? 1024 : 512)
    ctc_tables_kernel(DevIdx ix, const float *__restrict__ logp, int C, int blank, const int32_t *__restrict__ labels,
                      float *__restrict__ alpha, float *__restrict__ beta, float *__restrict__ loss,
                      int32_t *__restrict__ row_ok, int32_t *__restrict__ status) {
  extern __shared__ float sm[];
  const int r = blockIdx.x;
  const bool fwd = blockIdx.y == 0;
  const int L = ix.row_len[r];
  const int U = ix.row_lab_len[r];
  const int S = 2 * U + 1;
  const int W = MW ? (int)(blockDim.x >> 5) : 1;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  float *xch = sm;                      // [2][W][2] last two values of each warp's part
  float *wmx = xch + 4 * W;             // [W] per-warp row maxima (2W reserved)
  float *fin = wmx + 2 * W;             // [4] the two end positions (forward)
  int *toff = reinterpret_cast<int *>(fin + 4);  // [L] packed offsets of this row's time steps
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
      atomicOr(status, kErrLabel);
      row_ok[r] = 0;
      loss[ix.row_orig[r]] = CUDART_NAN_F;
    }
    return;
  }

  // this lane's positions p0 .. p0+K-1: emission column, skip mask, table column
  const int p0 = (wid * 32 + lane) * K;
  int ecol[K], tcol[K];
  float mk[K];
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const int p = p0 + j;
    ecol[j] = blank;
    mk[j] = kNeg;
    if (p < S && (p & 1)) {
      const int u = (p - 1) >> 1;
      const int lu = lab[fwd ? u : U - 1 - u];
      ecol[j] = lu;
      if (p >= 3 && lu != lab[fwd ? u - 1 : U - u]) mk[j] = 0.f;
    }
    tcol[j] = fwd ? p : S - 1 - p;
  }
  for (int i = tid; i < L; i += blockDim.x) toff[i] = ix.tok_off[i];
  __syncthreads();

  // this lane's emissions of `step`; past the end, those of the last step
  auto load_step = [&](int step, float *dst) {
    const int sc = min(step, L - 1);
    const int t = fwd ? sc : L - 1 - sc;
    const float *lrow = logp + ((int64_t)toff[t] + r) * C;
#pragma unroll
    for (int j = 0; j < K; ++j) dst[j] = ld_prefetch(lrow + ecol[j]);
  };
  float e[2 * kBlock][K];  // two register buffers of kBlock steps

  // step 0: the two admissible start positions
  float v[K];
  {
    const int t0 = fwd ? 0 : L - 1;
    const float *lp0 = logp + ((int64_t)toff[t0] + r) * C;
    float *rowp = tab + (int64_t)t0 * S;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      v[j] = (p0 + j <= 1 && p0 + j < S) ? lp0[ecol[j]] * kLog2e : kNeg;
      if (p0 + j < S) rowp[tcol[j]] = v[j];
    }
  }
  if (MW) {
    if (lane == 31) xch[wid * 2 + 1] = v[K - 1];
    if (lane == (K >= 2 ? 31 : 30)) xch[wid * 2] = v[K >= 2 ? K - 2 : 0];
  }
#pragma unroll
  for (int d = 0; d < kBlock; ++d) load_step(1 + d, e[d]);
  __syncthreads();

  // Shifts are whole numbers in log2 units (powers of two), at most 2^24 in
  // magnitude, summed exactly in int64 by every thread without a branch.
  long long M = 0;
  float anchor = 0.f;
  for (int base = 1; base < L; base += 2 * kBlock) {
#pragma unroll
    for (int u = 0; u < 2 * kBlock; ++u) {  // step base+u uses buffer slot u
      const int step = base + u;
      if (step >= L) break;
      const float *xprev = xch + ((step - 1) & 1) * 2 * W;
      // the two positions below this lane's first one, from the previous row
      float n1 = __shfl_up_sync(0xffffffffu, v[K - 1], 1);
      float n2 = K >= 2 ? __shfl_up_sync(0xffffffffu, v[K >= 2 ? K - 2 : 0], 1)
                        : __shfl_up_sync(0xffffffffu, v[0], 2);
      if (MW) {
        if (lane == 0) {
          n1 = wid ? xprev[(wid - 1) * 2 + 1] : kNeg;
          n2 = wid ? xprev[(wid - 1) * 2] : kNeg;
        }
        if (K == 1 && lane == 1) n2 = wid ? xprev[(wid - 1) * 2 + 1] : kNeg;
      } else {
        if (lane == 0) n1 = n2 = kNeg;
        if (K == 1 && lane == 1) n2 = kNeg;
      }
      float shift = 0.f;
      if (u % kBlock == 0) {
        shift = anchor;
        M += (long long)anchor;
      }
      const int t = fwd ? step : L - 1 - step;
      float *rowp = tab + (int64_t)t * S;
      // in place from the top: v[j-1], v[j-2] still hold the previous row
#pragma unroll
      for (int j = K - 1; j >= 0; --j) {
        const float a0 = v[j];
        const float a1 = j >= 1 ? v[j >= 1 ? j - 1 : 0] : n1;
        const float a2 = j >= 2 ? v[j >= 2 ? j - 2 : 0] : (j == 1 ? n1 : n2);
        float l;
        if (K % 2 == 0 && (j & 1) == 0) l = lse2b(a0, a1);  // p even: a blank
        else l = lse3b(a0, a1, a2 + mk[j]);
        v[j] = fmaf(e[u][j], kLog2e, l - shift);
        if (p0 + j < S) rowp[tcol[j]] = v[j];
      }
      if (u % kBlock == kBlock - 2) {  // the next shift: this row's maximum (a dead row is not shifted)
        float m = v[0];
#pragma unroll
        for (int j = 1; j < K; ++j) m = fmaxf(m, v[j]);
        m = warp_max(m);
        if (!MW) anchor = m > kDead ? fminf(fmaxf(floorf(m), -16777216.f), 16777216.f) : 0.f;
        else if (lane == 0) wmx[wid] = m;
      }
      if (MW) {
        float *xcur = xch + (step & 1) * 2 * W;
        if (lane == 31) xcur[wid * 2 + 1] = v[K - 1];
        if (lane == (K >= 2 ? 31 : 30)) xcur[wid * 2] = v[K >= 2 ? K - 2 : 0];
        if (u % kBlock == kBlock - 1) {  // published by the barrier of step kBlock-2
          float m = wmx[0];
          for (int i = 1; i < W; ++i) m = fmaxf(m, wmx[i]);
          anchor = m > kDead ? fminf(fmaxf(floorf(m), -16777216.f), 16777216.f) : 0.f;
        }
      }
      load_step(step + kBlock, e[(u + kBlock) % (2 * kBlock)]);
      if (MW) __syncthreads();
    }
  }
  // forward: ln p from the two end positions of the last row
  if (fwd) {
#pragma unroll
    for (int j = 0; j < K; ++j) {
      if (p0 + j == S - 1) fin[1] = v[j];
      if (p0 + j == S - 2) fin[0] = v[j];
    }
    if (S < 2 && tid == 0) fin[0] = kNeg;
    __syncthreads();
    if (tid == 0) {
      const float l2 = lse2b(fin[0], fin[1]);
      const bool ok = l2 > kDead;
      row_ok[r] = ok ? 1 : 0;
      if (!ok) atomicAdd(status + 1, 1);  // counted in the ctx (no alignment is not an error)
      loss[ix.row_orig[r]] = ok ? (float)(-((double)M + (double)l2) * kLn2) : CUDART_INF_F;
    }
  }
}

namespace {
// Positions per lane (measured on GB300: one position per lane while one warp
// covers the label, then two, over up to 16 warps); BKT_CTC_K overrides.
int ctc_lanes_k(int S) {
  static const int forced = [] {
    const char *e = getenv("BKT_CTC_K");
    const int k = e ? atoi(e) : 0;
    return (k == 1 || k == 2 || k == 4 || k == 8 || k == 16) ? k : 0;
  }();
  if (forced) return forced;
  if (S <= 32) return 1;
  if (S <= 16 * 64) return 2;
  if (S <= 16 * 128) return 4;
  if (S <= 16 * 256) return 8;
  return 16;
}
}  // namespace

cudaError_t launch_ctc_tables(const DevIdx &ix, const float *logp, int C, int blank, const int32_t *labels,
                              float *alpha, float *beta, float *loss, int32_t *row_ok, int32_t *status,
                              cudaStream_t s) {
  if (C > kMaxClasses) return cudaErrorInvalidValue;
  const int S = ix.S_max;
  const int K = ctc_lanes_k(S);
  const int W = (S + 32 * K - 1) / (32 * K);
  if (W > (K >= 16 ? 32 : 16)) return cudaErrorInvalidValue;
  const size_t smem = ctc_tables_smem(W, ix.T);
  const bool mw = W > 1;
#define BKT_CTC_FN(k) (mw ? (const void *)ctc_tables_kernel<k, true> : (const void *)ctc_tables_kernel<k, false>)
  const void *kfn = K == 1 ? BKT_CTC_FN(1) : K == 2 ? BKT_CTC_FN(2) : K == 4 ? BKT_CTC_FN(4) : K == 8 ? BKT_CTC_FN(8) : BKT_CTC_FN(16);
#undef BKT_CTC_FN
  if (smem > 48 * 1024) {
    cudaError_t e = ensure_smem(kfn, smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid(ix.b, 2);
  const int threads = 32 * W;
#define BKT_CTC_GO(k)                                                                                          \
  (mw ? ctc_tables_kernel<k, true><<<grid, threads, smem, s>>>(ix, logp, C, blank, labels, alpha, beta, loss,   \
                                                               row_ok, status)                                 \
      : ctc_tables_kernel<k, false><<<grid, threads, smem, s>>>(ix, logp, C, blank, labels, alpha, beta, loss,  \
                                                                row_ok, status))
  switch (K) {
    case 1: BKT_CTC_GO(1); break;
    case 2: BKT_CTC_GO(2); break;
    case 4: BKT_CTC_GO(4); break;
    case 8: BKT_CTC_GO(8); break;
    default: BKT_CTC_GO(16); break;
  }
#undef BKT_CTC_GO
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a9.  One warp per token (t, r):
//   v(s) = a_t(s) + bh_t(s) - log2(e) lp_t(l'_s)  (log2 of alpha_t(s) beta_t(s), offset)
//   gamma(s) = 2^(v(s) - lse2_s v)
//   dlogit[k] = exp(lp_t(k)) - sum_{s: l'_s = k} gamma(s)
// For labels of up to 256 extended positions each lane keeps the v(s) of its
// positions in registers, so the tables, labels and emissions are read once.
// written over the log-probabilities in place, and (when dl_hi is set) as
// the tf32 hi + lo split the dY GEMM reads, rows padded to ld_split (both
// parts rounded to nearest: |x - hi - lo| <= 2^-22 |x|).  Blank mass is a
// warp sum; label mass goes through a per-warp shared row.  Rows without an
// alignment (or with a bad label) get zeros.
template <int JC>  // JC > 0: v(s) of positions s = lane + 32 j (j < JC) kept in registers (S <= 32 JC)
__global__ void __launch_bounds__(256) ctc_grad_kernel(DevIdx ix, float *__restrict__ lp_dl, int C, int blank,
                                                       const int32_t *__restrict__ labels,
                                                       const float *__restrict__ alpha,
                                                       const float *__restrict__ beta,
                                                       const int32_t *__restrict__ row_ok,
                                                       float *__restrict__ dl_hi, float *__restrict__ dl_lo,
                                                       int64_t ld_split) {
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
    float blank_mass = 0.f;
    __syncwarp();
    if (JC > 0) {
      // one pass of loads: label, emission and both tables of each position
      float v[JC > 0 ? JC : 1];
      int k[JC > 0 ? JC : 1];
      float mx = -CUDART_INF_F;
#pragma unroll
      for (int j = 0; j < JC; ++j) {
        const int s = lane + 32 * j;
        k[j] = blank;
        v[j] = -CUDART_INF_F;
        if (s < S) {  // positions past S read nothing
          if (s & 1) k[j] = lab[(s - 1) >> 1];
          const float e = (s & 1) ? row[k[j]] : lpb;
          v[j] = a[s] + b[s] - kLog2e * e;
        }
        mx = fmaxf(mx, v[j]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float se = 0.f;
#pragma unroll
      for (int j = 0; j < JC; ++j) se += exp2f(v[j] - mx);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
      const float lz = mx + log2f(se);
#pragma unroll
      for (int j = 0; j < JC; ++j) {
        const int s = lane + 32 * j;
        if (s < S) {
          const float gm = exp2f(v[j] - lz);
          if (s & 1) atomicAdd(&acc[w][k[j]], gm);
          else blank_mass += gm;
        }
      }
    } else {
      float mx = -CUDART_INF_F;
      for (int s = lane; s < S; s += 32) {
        const float e = (s & 1) ? row[lab[(s - 1) >> 1]] : lpb;
        mx = fmaxf(mx, a[s] + b[s] - kLog2e * e);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float se = 0.f;
      for (int s = lane; s < S; s += 32) {
        const float e = (s & 1) ? row[lab[(s - 1) >> 1]] : lpb;
        se += exp2f(a[s] + b[s] - kLog2e * e - mx);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
      const float lz = mx + log2f(se);
      for (int s = lane; s < S; s += 32) {
        const int kk = (s & 1) ? lab[(s - 1) >> 1] : blank;
        const float e = (s & 1) ? row[kk] : lpb;
        const float gm = exp2f(a[s] + b[s] - kLog2e * e - lz);
        if (s & 1) atomicAdd(&acc[w][kk], gm);
        else blank_mass += gm;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) blank_mass += __shfl_xor_sync(0xffffffffu, blank_mass, o);
    __syncwarp();
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int kk = lane + 32 * j;
      out[j] = expf(lpk[j]) - acc[w][kk] - (kk == blank ? blank_mass : 0.f);
    }
  }
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (lane + 32 * j < C) row[lane + 32 * j] = out[j];
  if (dl_hi) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int kk = lane + 32 * j;
      if (kk < (int)ld_split) {  // the padding columns get zeros
        const float x = kk < C ? out[j] : 0.f;
        const float hv = __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
        const float lv = __uint_as_float((__float_as_uint(x - hv) + 0x1000u) & 0xFFFFE000u);
        dl_hi[(int64_t)tok * ld_split + kk] = hv;
        dl_lo[(int64_t)tok * ld_split + kk] = lv;
      }
    }
  }
}

cudaError_t launch_ctc_grad(const DevIdx &ix, float *lp_dl, int C, int blank, const int32_t *labels,
                            const float *alpha, const float *beta, const int32_t *row_ok, float *dl_hi, float *dl_lo,
                            int64_t ld_split, cudaStream_t s) {
  if (C > kMaxClasses || (dl_hi && (ld_split < C || ld_split > kMaxClasses || !dl_lo))) return cudaErrorInvalidValue;
  const int blocks = (ix.n_tok + 7) / 8;
  // labels up to 256 extended positions keep each position's value in registers
  if (ix.S_max <= 32 * 8)
    ctc_grad_kernel<8><<<blocks, 256, 0, s>>>(ix, lp_dl, C, blank, labels, alpha, beta, row_ok, dl_hi, dl_lo, ld_split);
  else
    ctc_grad_kernel<0><<<blocks, 256, 0, s>>>(ix, lp_dl, C, blank, labels, alpha, beta, row_ok, dl_hi, dl_lo, ld_split);
  return cudaGetLastError();
}

}  // namespace bkt
