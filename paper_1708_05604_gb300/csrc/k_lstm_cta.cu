// k_lstm_cta.cu -- single-CTA persistent recurrent kernels for H <= 128
// (a6 forward, a11 BPTT).
//
// Same recurrence as the cluster kernels (gates i, f, g, o; the reverse
// direction over each sequence's own length), but one CTA holds the whole
// 4H x H fp32 W_hh of its direction, so a time step needs no inter-SM
// exchange at all: two CTA barriers per step are the only synchronisation.
// For H = 128 the matrix is 256 KB, more than shared memory: each thread keeps
// RK of its H weights in registers and the remaining H - RK in shared memory
// (laid out so a warp reads 512 consecutive bytes).
//
// Forward, 4H threads, thread t owns gate row t:
//   phase A (all threads): z_t = Zx[t] + W_hh[t,:] . h_{s-1}   (h broadcast
//            from shared memory), activation of row t (tanh for the g block,
//            sigmoid otherwise), written to shared memory and, in place over
//            Zx, to global memory;
//   phase B (threads t < H = unit t): c = f c + i g, h = o tanh(c).
// BPTT, 4H threads, thread t = (q, k) owns the column segment
// W_hh[q*H .. q*H+H-1, k]:
//   phase B (threads t < H = unit t): dh = dY + sum_q part[q][t]; dc, dz of
//            the four gates (written in place over the gates);
//   phase A (all threads): part[q][k] = sum_i W_hh[q*H+i, k] dz[q*H+i].
// A CTA owns BC consecutive rows of the length-sorted batch (BC = 1 when the
// batch fits the GPU) and stops after its longest row.  Per-step global loads
// are issued one step ahead.
#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

namespace {

constexpr int kTokCap = 8192;  // time offsets staged in shared memory up to this T

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + expf(-x)); }

}  // namespace

template <int H, int RK, int BC>
__global__ void __launch_bounds__(4 * H, 1) lstm_fwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, SK = H - RK, H4 = H / 4;
  extern __shared__ __align__(16) float sm[];
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SK/4][G]
  float *hs = sm + SK * G;                       // [2][BC][H]
  float *zs = hs + 2 * BC * H;                   // [BC][G]
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(zs + BC * G);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x;
  const int q = t / H;
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;

  const float *Wrow = a.Whh[d] + (size_t)t * H;
  float wr[RK > 0 ? RK : 1];
#pragma unroll
  for (int i = 0; i < RK; ++i) wr[i] = __ldg(Wrow + i);
  for (int i4 = 0; i4 < SK / 4; ++i4) {
    const float *w = Wrow + RK + 4 * i4;
    Ws4[i4 * G + t] = make_float4(__ldg(w), __ldg(w + 1), __ldg(w + 2), __ldg(w + 3));
  }
  for (int i = t; i < 2 * BC * H; i += G) hs[i] = 0.f;
  if (toff_sm)
    for (int i = t; i <= T; i += G) toff_s[i] = a.ix.tok_off[i];
  int len[BC];
#pragma unroll
  for (int b = 0; b < BC; ++b) len[b] = (r0 + b < a.ix.b) ? a.ix.row_len[r0 + b] : 0;
  const int Tg = len[0];
  __syncthreads();

  float *__restrict__ Z = a.Z[d];
  float *__restrict__ Cs = a.Cst[d];
  float *__restrict__ Y = a.Y;
  auto tok_at = [&](int b, int s) {
    const int tt = d == 0 ? s : len[b] - 1 - s;
    return toff[tt] + r0 + b;
  };
  float zn[BC], cst[BC];
  int tokn[BC];
#pragma unroll
  for (int b = 0; b < BC; ++b) {
    cst[b] = 0.f;
    tokn[b] = 0;
    zn[b] = 0.f;
    if (len[b] > 0) {
      tokn[b] = tok_at(b, 0);
      zn[b] = Z[(size_t)tokn[b] * G + t];
    }
  }
  for (int s = 0; s < Tg; ++s) {
    const int p = s & 1;
    float zc[BC];
    int tc[BC];
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      zc[b] = zn[b];
      tc[b] = tokn[b];
      if (s + 1 < len[b]) {
        tokn[b] = tok_at(b, s + 1);
        zn[b] = Z[(size_t)tokn[b] * G + t];
      }
    }
    // phase A
    float acc[BC];
#pragma unroll
    for (int b = 0; b < BC; ++b) acc[b] = 0.f;
    const float4 *h4 = reinterpret_cast<const float4 *>(hs + p * BC * H);
#pragma unroll
    for (int i4 = 0; i4 < RK / 4; ++i4) {
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        const float4 hv = h4[b * H4 + i4];
        float x = fmaf(wr[4 * i4], hv.x, acc[b]);
        x = fmaf(wr[4 * i4 + 1], hv.y, x);
        x = fmaf(wr[4 * i4 + 2], hv.z, x);
        acc[b] = fmaf(wr[4 * i4 + 3], hv.w, x);
      }
    }
#pragma unroll 8
    for (int i4 = 0; i4 < SK / 4; ++i4) {
      const float4 w = Ws4[i4 * G + t];
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        const float4 hv = h4[b * H4 + RK / 4 + i4];
        float x = fmaf(w.x, hv.x, acc[b]);
        x = fmaf(w.y, hv.y, x);
        x = fmaf(w.z, hv.z, x);
        acc[b] = fmaf(w.w, hv.w, x);
      }
    }
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s < len[b]) {
        const float z = acc[b] + zc[b];
        const float v = (q == 2) ? tanhf(z) : sigm(z);
        zs[b * G + t] = v;
        Z[(size_t)tc[b] * G + t] = v;
      }
    }
    __syncthreads();
    // phase B
    if (t < H) {
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        if (s < len[b]) {
          const float ig = zs[b * G + t], fg = zs[b * G + H + t], gg = zs[b * G + 2 * H + t],
                      og = zs[b * G + 3 * H + t];
          cst[b] = fmaf(fg, cst[b], ig * gg);
          const float h = og * tanhf(cst[b]);
          hs[(p ^ 1) * BC * H + b * H + t] = h;
          Cs[(size_t)tc[b] * H + t] = cst[b];
          Y[(size_t)tc[b] * DH + d * H + t] = h;
        }
      }
    }
    __syncthreads();
  }
}

template <int H, int RK, int BC>
__global__ void __launch_bounds__(4 * H, 1) lstm_bwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, SK = H - RK;
  extern __shared__ __align__(16) float sm[];
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SK/4][G], W[q*H+RK+4*i4 .. +3][k]
  float *dzs = sm + SK * G;                      // [BC][G]
  float *red = dzs + BC * G;                     // [BC][G] partials, index q*H + k
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(red + BC * G);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x;
  const int q = t / H, k = t % H;
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;

  const float *Wcol = a.Whh[d] + (size_t)q * H * H + k;  // W[q*H + i][k] = Wcol[i*H]
  float wc[RK > 0 ? RK : 1];
#pragma unroll
  for (int i = 0; i < RK; ++i) wc[i] = __ldg(Wcol + (size_t)i * H);
  for (int i4 = 0; i4 < SK / 4; ++i4) {
    const float *w = Wcol + (size_t)(RK + 4 * i4) * H;
    Ws4[i4 * G + t] = make_float4(__ldg(w), __ldg(w + H), __ldg(w + 2 * H), __ldg(w + 3 * H));
  }
  if (toff_sm)
    for (int i = t; i <= T; i += G) toff_s[i] = a.ix.tok_off[i];
  int len[BC];
#pragma unroll
  for (int b = 0; b < BC; ++b) len[b] = (r0 + b < a.ix.b) ? a.ix.row_len[r0 + b] : 0;
  const int Tg = len[0];
  __syncthreads();

  float *__restrict__ Z = a.Z[d];
  const float *__restrict__ Cs = a.Cst[d];
  const float *__restrict__ dY = a.dY;
  auto tok_at = [&](int b, int s) {
    const int tt = d == 0 ? s : len[b] - 1 - s;
    return toff[tt] + r0 + b;
  };
  // unit t's prefetched inputs (threads t < H)
  float gn[BC][4], cn[BC], cpn[BC], dyn[BC], dc[BC];
  int tokn[BC];
  auto prefetch = [&](int b, int s) {
    const int tk = tok_at(b, s);
    tokn[b] = tk;
#pragma unroll
    for (int g = 0; g < 4; ++g) gn[b][g] = Z[(size_t)tk * G + g * H + t];
    cn[b] = Cs[(size_t)tk * H + t];
    cpn[b] = s > 0 ? Cs[(size_t)tok_at(b, s - 1) * H + t] : 0.f;
    dyn[b] = dY[(size_t)tk * DH + d * H + t];
  };
#pragma unroll
  for (int b = 0; b < BC; ++b) {
    dc[b] = 0.f;
    tokn[b] = 0;
    cn[b] = cpn[b] = dyn[b] = 0.f;
#pragma unroll
    for (int g = 0; g < 4; ++g) gn[b][g] = 0.f;
    if (t < H && Tg - 1 < len[b]) prefetch(b, Tg - 1);
  }
  for (int s = Tg - 1; s >= 0; --s) {
    // phase B
    if (t < H) {
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        if (s < len[b]) {
          float dh_rec = 0.f;
          if (s + 1 < len[b])
            dh_rec = red[b * G + t] + red[b * G + H + t] + red[b * G + 2 * H + t] + red[b * G + 3 * H + t];
          const float ig = gn[b][0], fg = gn[b][1], gg = gn[b][2], og = gn[b][3];
          const float ct = cn[b], cp = cpn[b];
          const float dh = dyn[b] + dh_rec;
          const int tk = tokn[b];
          if (s - 1 >= 0 && s - 1 < len[b]) prefetch(b, s - 1);
          const float tch = tanhf(ct);
          float dcv = fmaf(dh * og, 1.f - tch * tch, dc[b]);
          const float dzi = dcv * gg * ig * (1.f - ig);
          const float dzf = dcv * cp * fg * (1.f - fg);
          const float dzg = dcv * ig * (1.f - gg * gg);
          const float dzo = dh * tch * og * (1.f - og);
          dc[b] = dcv * fg;
          dzs[b * G + t] = dzi;
          dzs[b * G + H + t] = dzf;
          dzs[b * G + 2 * H + t] = dzg;
          dzs[b * G + 3 * H + t] = dzo;
          float *zr = Z + (size_t)tk * G + t;
          zr[0] = dzi;
          zr[H] = dzf;
          zr[2 * H] = dzg;
          zr[3 * H] = dzo;
        }
      }
    }
    __syncthreads();
    // phase A
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s < len[b]) {
        const float4 *dz4 = reinterpret_cast<const float4 *>(dzs + b * G + q * H);
        float acc = 0.f;
#pragma unroll
        for (int i4 = 0; i4 < RK / 4; ++i4) {
          const float4 v = dz4[i4];
          float x = fmaf(wc[4 * i4], v.x, acc);
          x = fmaf(wc[4 * i4 + 1], v.y, x);
          x = fmaf(wc[4 * i4 + 2], v.z, x);
          acc = fmaf(wc[4 * i4 + 3], v.w, x);
        }
#pragma unroll 8
        for (int i4 = 0; i4 < SK / 4; ++i4) {
          const float4 w = Ws4[i4 * G + t];
          const float4 v = dz4[RK / 4 + i4];
          float x = fmaf(w.x, v.x, acc);
          x = fmaf(w.y, v.y, x);
          x = fmaf(w.z, v.z, x);
          acc = fmaf(w.w, v.w, x);
        }
        red[b * G + q * H + k] = acc;
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
namespace {

size_t cta_smem_bytes(bool bwd, int H, int RK, int BC, int T) {
  const size_t f = bwd ? (size_t)(H - RK) * 4 * H + 2 * (size_t)BC * 4 * H
                       : (size_t)(H - RK) * 4 * H + 2 * (size_t)BC * H + (size_t)BC * 4 * H;
  const size_t i = (T + 1 <= kTokCap) ? (size_t)(T + 1) : 0;
  return (f + i) * 4 + 16;
}

template <int H, int RK, int BC>
cudaError_t launch_cta(const RecArgs &a, bool bwd, cudaStream_t s) {
  const size_t smem = cta_smem_bytes(bwd, H, RK, BC, a.ix.T);
  const int ng = (a.ix.b + BC - 1) / BC;
  if (bwd) {
    cudaError_t e = cudaFuncSetAttribute(lstm_bwd_cta_kernel<H, RK, BC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    lstm_bwd_cta_kernel<H, RK, BC><<<ng * a.dirs, 4 * H, smem, s>>>(a);
  } else {
    cudaError_t e = cudaFuncSetAttribute(lstm_fwd_cta_kernel<H, RK, BC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    lstm_fwd_cta_kernel<H, RK, BC><<<ng * a.dirs, 4 * H, smem, s>>>(a);
  }
  return cudaGetLastError();
}

template <int H, int RK>
cudaError_t launch_cta_bc(const RecArgs &a, int bc, bool bwd, cudaStream_t s) {
  switch (bc) {
    case 1: return launch_cta<H, RK, 1>(a, bwd, s);
    case 2: return launch_cta<H, RK, 2>(a, bwd, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool cta_supported(int H) { return H == 32 || H == 64 || H == 128; }

int cta_rows_per_block(int H, int b, int dirs, int sm_count) {
  (void)H;
  return (b * dirs > sm_count) ? 2 : 1;
}

cudaError_t launch_lstm_cta(const RecArgs &a, int bc, bool bwd, cudaStream_t s) {
  switch (a.H) {
    case 32: return launch_cta_bc<32, 32>(a, bc, bwd, s);
    case 64: return launch_cta_bc<64, 64>(a, bc, bwd, s);
    case 128: return launch_cta_bc<128, 64>(a, bc, bwd, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bkt
