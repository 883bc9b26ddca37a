// k_lstm_cta.cu -- single-CTA persistent recurrent kernels for H <= 128
// (a6 forward, a11 BPTT).
//
// Same recurrence as the cluster kernels (gates i, f, g, o; the reverse
// direction over each sequence's own length), but one CTA holds the whole
// 4H x H fp32 W_hh of its direction, so a time step needs no inter-SM
// exchange at all: two CTA barriers per step are the only synchronisation.
// For H = 128 the matrix is 256 KB, more than shared memory.  2H threads each
// own two rows (or, in BPTT, two column segments), keep RK weights of each in
// registers (192 registers for H = 128) and the rest in shared memory (laid
// out so a warp reads 512 consecutive bytes).  Each h value read from shared
// memory feeds both rows, so a step moves half the shared-memory bytes of a
// one-row-per-thread layout, which was bound by shared-memory bandwidth.
//
// Forward, 2H threads, thread t owns gate rows t (i or f) and t + 2H (g or o):
//   phase A (all threads): z_r = Zx[r] + W_hh[r,:] . h_{s-1}   (h broadcast
//            from shared memory), activation of row r (tanh for the g block,
//            sigmoid otherwise), written to shared memory and, in place over
//            Zx, to global memory;
//   phase B (threads t < H = unit t): c = f c + i g, h = o tanh(c).
// BPTT, 2H threads, thread t = (q, kc) owns the column segments
// W_hh[q*H .. q*H+H-1, k] for k = kc and kc + H/2 of gate block q:
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
__global__ void __launch_bounds__(2 * H, 1) lstm_fwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, NTH = 2 * H, SK = H - RK, H4 = H / 4;
  extern __shared__ __align__(16) float sm[];
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SK/4][2][NTH]
  float *hs = sm + 2 * SK * NTH;                 // [2][BC][H]
  float *zs = hs + 2 * BC * H;                   // [BC][G]
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(zs + BC * G);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x;
  const bool lo_half = t < H;  // rows t (i or f) and t + 2H (g or o)
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;

  const float *W0 = a.Whh[d] + (size_t)t * H;
  const float *W1 = a.Whh[d] + (size_t)(t + NTH) * H;
  float w0[RK], w1[RK];
#pragma unroll
  for (int i = 0; i < RK; ++i) {
    w0[i] = __ldg(W0 + i);
    w1[i] = __ldg(W1 + i);
  }
  for (int i4 = 0; i4 < SK / 4; ++i4) {
    const float *u = W0 + RK + 4 * i4, *v = W1 + RK + 4 * i4;
    Ws4[(2 * i4) * NTH + t] = make_float4(__ldg(u), __ldg(u + 1), __ldg(u + 2), __ldg(u + 3));
    Ws4[(2 * i4 + 1) * NTH + t] = make_float4(__ldg(v), __ldg(v + 1), __ldg(v + 2), __ldg(v + 3));
  }
  for (int i = t; i < 2 * BC * H; i += NTH) hs[i] = 0.f;
  if (toff_sm)
    for (int i = t; i <= T; i += NTH) toff_s[i] = a.ix.tok_off[i];
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
  float zn0[BC], zn1[BC], cst[BC];
  int tokn[BC];
#pragma unroll
  for (int b = 0; b < BC; ++b) {
    cst[b] = 0.f;
    tokn[b] = 0;
    zn0[b] = zn1[b] = 0.f;
    if (len[b] > 0) {
      tokn[b] = tok_at(b, 0);
      zn0[b] = Z[(size_t)tokn[b] * G + t];
      zn1[b] = Z[(size_t)tokn[b] * G + NTH + t];
    }
  }
  for (int s = 0; s < Tg; ++s) {
    const int p = s & 1;
    float zc0[BC], zc1[BC];
    int tc[BC];
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      zc0[b] = zn0[b];
      zc1[b] = zn1[b];
      tc[b] = tokn[b];
      if (s + 1 < len[b]) {
        tokn[b] = tok_at(b, s + 1);
        zn0[b] = Z[(size_t)tokn[b] * G + t];
        zn1[b] = Z[(size_t)tokn[b] * G + NTH + t];
      }
    }
    // phase A: two rows per thread, two accumulators per row
    float a0[BC], a1[BC], e0[BC], e1[BC];
#pragma unroll
    for (int b = 0; b < BC; ++b) a0[b] = a1[b] = e0[b] = e1[b] = 0.f;
    const float4 *h4 = reinterpret_cast<const float4 *>(hs + p * BC * H);
#pragma unroll
    for (int i4 = 0; i4 < RK / 4; ++i4) {
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        const float4 hv = h4[b * H4 + i4];
        a0[b] = fmaf(w0[4 * i4], hv.x, a0[b]);
        a1[b] = fmaf(w1[4 * i4], hv.x, a1[b]);
        e0[b] = fmaf(w0[4 * i4 + 1], hv.y, e0[b]);
        e1[b] = fmaf(w1[4 * i4 + 1], hv.y, e1[b]);
        a0[b] = fmaf(w0[4 * i4 + 2], hv.z, a0[b]);
        a1[b] = fmaf(w1[4 * i4 + 2], hv.z, a1[b]);
        e0[b] = fmaf(w0[4 * i4 + 3], hv.w, e0[b]);
        e1[b] = fmaf(w1[4 * i4 + 3], hv.w, e1[b]);
      }
    }
#pragma unroll
    for (int i4 = 0; i4 < SK / 4; ++i4) {
      const float4 u = Ws4[(2 * i4) * NTH + t];
      const float4 v = Ws4[(2 * i4 + 1) * NTH + t];
#pragma unroll
      for (int b = 0; b < BC; ++b) {
        const float4 hv = h4[b * H4 + RK / 4 + i4];
        a0[b] = fmaf(u.x, hv.x, a0[b]);
        a1[b] = fmaf(v.x, hv.x, a1[b]);
        e0[b] = fmaf(u.y, hv.y, e0[b]);
        e1[b] = fmaf(v.y, hv.y, e1[b]);
        a0[b] = fmaf(u.z, hv.z, a0[b]);
        a1[b] = fmaf(v.z, hv.z, a1[b]);
        e0[b] = fmaf(u.w, hv.w, e0[b]);
        e1[b] = fmaf(v.w, hv.w, e1[b]);
      }
    }
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s < len[b]) {
        const float v0 = sigm(a0[b] + e0[b] + zc0[b]);                       // i or f
        const float z1 = a1[b] + e1[b] + zc1[b];
        const float v1 = lo_half ? tanhf(z1) : sigm(z1);                      // g or o
        zs[b * G + t] = v0;
        zs[b * G + NTH + t] = v1;
        Z[(size_t)tc[b] * G + t] = v0;
        Z[(size_t)tc[b] * G + NTH + t] = v1;
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
__global__ void __launch_bounds__(2 * H, 1) lstm_bwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, NTH = 2 * H, SK = H - RK;
  extern __shared__ __align__(16) float sm[];
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SK/4][2][NTH]: W[q*H+RK+4*i4 .. +3][k], k = kc, kc+H/2
  float *dzs = sm + 2 * SK * NTH;                // [BC][G]
  float *red = dzs + BC * G;                     // [BC][G] partials, index q*H + k
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(red + BC * G);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x;
  constexpr int H2 = H / 2;
  const int q = t / H2, kc = t % H2;  // columns kc and kc + H/2 of gate block q
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;

  const float *C0 = a.Whh[d] + (size_t)q * H * H + kc;       // W[q*H + i][kc] = C0[i*H]
  const float *C1 = a.Whh[d] + (size_t)q * H * H + kc + H2;  // W[q*H + i][kc + H/2]
  float w0[RK], w1[RK];
#pragma unroll
  for (int i = 0; i < RK; ++i) {
    w0[i] = __ldg(C0 + (size_t)i * H);
    w1[i] = __ldg(C1 + (size_t)i * H);
  }
  for (int i4 = 0; i4 < SK / 4; ++i4) {
    const float *u = C0 + (size_t)(RK + 4 * i4) * H, *v = C1 + (size_t)(RK + 4 * i4) * H;
    Ws4[(2 * i4) * NTH + t] = make_float4(__ldg(u), __ldg(u + H), __ldg(u + 2 * H), __ldg(u + 3 * H));
    Ws4[(2 * i4 + 1) * NTH + t] = make_float4(__ldg(v), __ldg(v + H), __ldg(v + 2 * H), __ldg(v + 3 * H));
  }
  if (toff_sm)
    for (int i = t; i <= T; i += NTH) toff_s[i] = a.ix.tok_off[i];
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
            dh_rec = (red[b * G + t] + red[b * G + H + t]) + (red[b * G + 2 * H + t] + red[b * G + 3 * H + t]);
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
    // phase A: two columns of one gate block per thread (one dz read feeds
    // both), two accumulators each
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s < len[b]) {
        const float4 *d0 = reinterpret_cast<const float4 *>(dzs + b * G + q * H);
        float a0 = 0.f, a1 = 0.f, e0 = 0.f, e1 = 0.f;
#pragma unroll
        for (int i4 = 0; i4 < RK / 4; ++i4) {
          const float4 x = d0[i4];
          a0 = fmaf(w0[4 * i4], x.x, a0);
          a1 = fmaf(w1[4 * i4], x.x, a1);
          e0 = fmaf(w0[4 * i4 + 1], x.y, e0);
          e1 = fmaf(w1[4 * i4 + 1], x.y, e1);
          a0 = fmaf(w0[4 * i4 + 2], x.z, a0);
          a1 = fmaf(w1[4 * i4 + 2], x.z, a1);
          e0 = fmaf(w0[4 * i4 + 3], x.w, e0);
          e1 = fmaf(w1[4 * i4 + 3], x.w, e1);
        }
#pragma unroll
        for (int i4 = 0; i4 < SK / 4; ++i4) {
          const float4 u = Ws4[(2 * i4) * NTH + t], v = Ws4[(2 * i4 + 1) * NTH + t];
          const float4 x = d0[RK / 4 + i4];
          a0 = fmaf(u.x, x.x, a0);
          a1 = fmaf(v.x, x.x, a1);
          e0 = fmaf(u.y, x.y, e0);
          e1 = fmaf(v.y, x.y, e1);
          a0 = fmaf(u.z, x.z, a0);
          a1 = fmaf(v.z, x.z, a1);
          e0 = fmaf(u.w, x.w, e0);
          e1 = fmaf(v.w, x.w, e1);
        }
        red[b * G + q * H + kc] = a0 + e0;
        red[b * G + q * H + kc + H2] = a1 + e1;
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
namespace {

size_t cta_smem_bytes(bool bwd, int H, int RK, int BC, int T) {
  const size_t f = bwd ? (size_t)(H - RK) * 4 * H + 2 * (size_t)BC * 4 * H
                       : (size_t)(H - RK) * 4 * H + 2 * (size_t)BC * H + (size_t)BC * 4 * H;  // W: 2 rows x (H-RK) x 2H threads
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
    lstm_bwd_cta_kernel<H, RK, BC><<<ng * a.dirs, 2 * H, smem, s>>>(a);
  } else {
    cudaError_t e = cudaFuncSetAttribute(lstm_fwd_cta_kernel<H, RK, BC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    lstm_fwd_cta_kernel<H, RK, BC><<<ng * a.dirs, 2 * H, smem, s>>>(a);
  }
  return cudaGetLastError();
}

template <int H, int RK1, int RK2>
cudaError_t launch_cta_bc(const RecArgs &a, int bc, bool bwd, cudaStream_t s) {
  switch (bc) {
    case 1: return launch_cta<H, RK1, 1>(a, bwd, s);
    case 2: return launch_cta<H, RK2, 2>(a, bwd, s);
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
    case 32: return launch_cta_bc<32, 32, 32>(a, bc, bwd, s);
    case 64: return launch_cta_bc<64, 64, 48>(a, bc, bwd, s);
    case 128: return launch_cta_bc<128, 96, 64>(a, bc, bwd, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bkt
