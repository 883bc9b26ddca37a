// k_lstm.cu -- persistent recurrent kernels of the stacked LSTM (a6, a11).
//
// LSTM (the paper's ref. [1]), gates i, f, g, o, no peepholes:
//   z_t = Zx_t + W_hh h_{t-1}          (Zx_t = W_ih x_t + b, precomputed)
//   i, f, o = sigmoid(z), g = tanh(z); c_t = f c_{t-1} + i g; h_t = o tanh(c_t)
// The reverse direction runs each sequence over its own length (t = L-1..0).
//
// Geometry.  One thread-block cluster of `cs` CTAs owns one direction and a
// group of `bc` consecutive rows of the length-sorted batch; clusters are
// independent, so rows of different groups never wait on each other and a
// group stops after its own longest row (Section III.A's point: padded steps
// are never executed).  CTA c of the cluster owns hidden units
// [c*Hc, (c+1)*Hc), Hc = H/cs: it keeps the 4*Hc rows of W_hh that feed
// those units in shared memory for the whole sequence (fp32, padded rows to
// spread banks) and updates their cell state in registers.  Each step:
//   forward:  every CTA reads the full h_{t-1} of its rows from its own
//             shared memory, computes its gate slice, and writes its h_t
//             slice into the shared memory of all cs CTAs (DSMEM stores);
//   backward: every CTA turns dh into dz for its units, forms the partial
//             W_hh^T dz over its 4*Hc rows for all H columns, and scatters
//             each column block to the CTA that owns it (a reduce-scatter
//             over DSMEM, summed in a fixed order);
// then one cluster barrier (arrive.release / wait.acquire).  Buffers are
// double-buffered by step parity, so one barrier per step suffices.  The
// per-step global traffic (Zx / gates / cell / dY) is prefetched one step
// ahead.  Only hardware cluster barriers are waited on: every CTA of a
// cluster runs the same number of steps, so no barrier can be left waiting.
#include <cooperative_groups.h>

#include <algorithm>

#include "bkt_internal.h"

namespace cg = cooperative_groups;

namespace bkt {

namespace {

constexpr int kTokSmemCap = 8192;  // time offsets staged in shared memory up to this T

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + expf(-x)); }

__device__ __forceinline__ int h_pad(int H) { return ((H + 3) & ~3) + 4; }

}  // namespace

// Shared-memory carve-up (floats): [W slice][h double buffer | dz + reduce
// slots][time offsets][row lengths].
__host__ __device__ inline size_t rec_smem_bytes(bool bwd, bool ws, int H, int cs, int bc, int T) {
  const int Hc = H / cs, HP = ((H + 3) & ~3) + 4;
  size_t f = ws ? (size_t)4 * Hc * HP : 0;
  if (!bwd) f += (size_t)2 * bc * HP;
  else f += (size_t)bc * (4 * Hc + 4) + (size_t)2 * cs * bc * Hc;
  size_t i = (size_t)(T + 1 <= kTokSmemCap ? T + 1 : 0) + bc;
  return (f + i) * 4 + 16;
}

template <bool WS>
__global__ void __launch_bounds__(512, 1) lstm_fwd_kernel(RecArgs a, int cs, int bc, int ks) {
  cg::cluster_group cluster = cg::this_cluster();
  extern __shared__ __align__(16) float sm[];
  const int tid = threadIdx.x;
  const int H = a.H, Hc = H / cs, HP = h_pad(H), HV = (H + 3) & ~3, G = 4 * H, DH = a.dirs * H;
  const int c = (int)cluster.block_rank();
  const int cid = blockIdx.x / cs;
  const int n_groups = (a.ix.b + bc - 1) / bc;
  const int d = cid / n_groups, grp = cid % n_groups;
  const int r0 = grp * bc;
  const int T = a.ix.T;
  float *Ws = sm;
  float *hb = sm + (WS ? 4 * Hc * HP : 0);
  int *toff_s = reinterpret_cast<int *>(hb + 2 * bc * HP);
  const bool toff_in_smem = T + 1 <= kTokSmemCap;
  int *rl = toff_s + (toff_in_smem ? T + 1 : 0);
  const int *toff = toff_in_smem ? toff_s : a.ix.tok_off;
  const float *__restrict__ Whh = a.Whh[d];

  if (WS) {
    for (int i = tid; i < 4 * Hc * HV; i += blockDim.x) {
      const int row = i / HV, k = i % HV;
      const int q = row / Hc, j = row % Hc;
      Ws[row * HP + k] = k < H ? __ldg(Whh + (size_t)(q * H + c * Hc + j) * H + k) : 0.f;
    }
  }
  for (int i = tid; i < 2 * bc * HP; i += blockDim.x) hb[i] = 0.f;
  if (toff_in_smem)
    for (int i = tid; i <= T; i += blockDim.x) toff_s[i] = a.ix.tok_off[i];
  for (int i = tid; i < bc; i += blockDim.x) rl[i] = (r0 + i < a.ix.b) ? a.ix.row_len[r0 + i] : 0;
  const int Tg = (r0 < a.ix.b) ? a.ix.row_len[r0] : 0;
  cluster.sync();  // every CTA initialised before any DSMEM store

  const int pairs = bc * Hc;
  const int pi = tid / ks, kp = tid % ks;
  const bool has = pi < pairs;
  const int bb = has ? pi / Hc : 0, j = has ? pi % Hc : 0;
  const int my_len = has ? rl[bb] : 0;
  const int r = r0 + bb;
  const int col = c * Hc + j;
  const unsigned lane = tid & 31;
  const unsigned gmask = ks >= 32 ? 0xffffffffu : (((1u << ks) - 1u) << (lane & ~(unsigned)(ks - 1)));
  float *__restrict__ Z = a.Z[d];
  float *__restrict__ Cs = a.Cst[d];
  float *__restrict__ Y = a.Y;
  auto tok_at = [&](int s) {
    const int t = d == 0 ? s : my_len - 1 - s;
    return toff[t] + r;
  };
  float cst = 0.f;
  float zn[4] = {0.f, 0.f, 0.f, 0.f};
  int tokn = 0;
  if (my_len > 0) {
    tokn = tok_at(0);
#pragma unroll
    for (int q = 0; q < 4; ++q) zn[q] = Z[(size_t)tokn * G + q * H + col];
  }
  for (int s = 0; s < Tg; ++s) {
    const int p = s & 1;
    const bool act = s < my_len;
    float zx[4] = {zn[0], zn[1], zn[2], zn[3]};
    const int tok = tokn;
    if (s + 1 < my_len) {
      tokn = tok_at(s + 1);
#pragma unroll
      for (int q = 0; q < 4; ++q) zn[q] = Z[(size_t)tokn * G + q * H + col];
    }
    if (act) {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
      const float *hrow = hb + (p * bc + bb) * HP;
      for (int k = 4 * kp; k < HV; k += 4 * ks) {
        const float4 h4 = *reinterpret_cast<const float4 *>(hrow + k);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float4 w4;
          if (WS) w4 = *reinterpret_cast<const float4 *>(Ws + (q * Hc + j) * HP + k);
          else w4 = __ldg(reinterpret_cast<const float4 *>(Whh + (size_t)(q * H + col) * H + k));
          float t0 = fmaf(w4.x, h4.x, acc[q]);
          t0 = fmaf(w4.y, h4.y, t0);
          t0 = fmaf(w4.z, h4.z, t0);
          acc[q] = fmaf(w4.w, h4.w, t0);
        }
      }
      for (int o = ks >> 1; o > 0; o >>= 1)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[q] += __shfl_xor_sync(gmask, acc[q], o);
      const float ig = sigm(acc[0] + zx[0]);
      const float fg = sigm(acc[1] + zx[1]);
      const float gg = tanhf(acc[2] + zx[2]);
      const float og = sigm(acc[3] + zx[3]);
      cst = fmaf(fg, cst, ig * gg);
      const float h = og * tanhf(cst);
      if (kp == 0) {
        float *zr = Z + (size_t)tok * G + col;
        zr[0] = ig;
        zr[H] = fg;
        zr[2 * H] = gg;
        zr[3 * H] = og;
        Cs[(size_t)tok * H + col] = cst;
        Y[(size_t)tok * DH + d * H + col] = h;
      }
      float *dst = hb + ((p ^ 1) * bc + bb) * HP + col;
      for (int q = kp; q < cs; q += ks) *cluster.map_shared_rank(dst, q) = h;
    }
    cluster.sync();
  }
}

template <bool WS>
__global__ void __launch_bounds__(512, 1) lstm_bwd_kernel(RecArgs a, int cs, int bc, int ks) {
  cg::cluster_group cluster = cg::this_cluster();
  extern __shared__ __align__(16) float sm[];
  const int tid = threadIdx.x;
  const int H = a.H, Hc = H / cs, HP = h_pad(H), HV = (H + 3) & ~3, G = 4 * H, DH = a.dirs * H;
  const int RZ = 4 * Hc + 4;  // padded dz row
  const int c = (int)cluster.block_rank();
  const int cid = blockIdx.x / cs;
  const int n_groups = (a.ix.b + bc - 1) / bc;
  const int d = cid / n_groups, grp = cid % n_groups;
  const int r0 = grp * bc;
  const int T = a.ix.T;
  float *Ws = sm;
  float *dzs = sm + (WS ? 4 * Hc * HP : 0);
  float *red = dzs + bc * RZ;  // [2][cs][bc][Hc]
  int *toff_s = reinterpret_cast<int *>(red + 2 * cs * bc * Hc);
  const bool toff_in_smem = T + 1 <= kTokSmemCap;
  int *rl = toff_s + (toff_in_smem ? T + 1 : 0);
  const int *toff = toff_in_smem ? toff_s : a.ix.tok_off;
  const float *__restrict__ Whh = a.Whh[d];

  if (WS) {
    for (int i = tid; i < 4 * Hc * HV; i += blockDim.x) {
      const int row = i / HV, k = i % HV;
      const int q = row / Hc, j = row % Hc;
      Ws[row * HP + k] = k < H ? __ldg(Whh + (size_t)(q * H + c * Hc + j) * H + k) : 0.f;
    }
  }
  if (toff_in_smem)
    for (int i = tid; i <= T; i += blockDim.x) toff_s[i] = a.ix.tok_off[i];
  for (int i = tid; i < bc; i += blockDim.x) rl[i] = (r0 + i < a.ix.b) ? a.ix.row_len[r0 + i] : 0;
  const int Tg = (r0 < a.ix.b) ? a.ix.row_len[r0] : 0;
  cluster.sync();

  const int pairs = bc * Hc;
  const int pi = tid / ks, kp = tid % ks;
  const bool has = pi < pairs;
  const int bb = has ? pi / Hc : 0, j = has ? pi % Hc : 0;
  const int my_len = has ? rl[bb] : 0;
  const int r = r0 + bb;
  const int col = c * Hc + j;
  float *__restrict__ Z = a.Z[d];
  const float *__restrict__ Cs = a.Cst[d];
  const float *__restrict__ dY = a.dY;
  auto tok_at = [&](int s) {
    const int t = d == 0 ? s : my_len - 1 - s;
    return toff[t] + r;
  };
  // prefetched inputs of the next step to process
  float gn[4] = {0.f, 0.f, 0.f, 0.f}, cn = 0.f, cpn = 0.f, dyn = 0.f;
  int tokn = 0;
  auto prefetch = [&](int s) {
    tokn = tok_at(s);
#pragma unroll
    for (int q = 0; q < 4; ++q) gn[q] = Z[(size_t)tokn * G + q * H + col];
    cn = Cs[(size_t)tokn * H + col];
    cpn = s > 0 ? Cs[(size_t)tok_at(s - 1) * H + col] : 0.f;
    dyn = dY[(size_t)tokn * DH + d * H + col];
  };
  if (Tg - 1 < my_len && Tg > 0) prefetch(Tg - 1);
  float dc = 0.f;
  int nact = 0;
  for (int s = Tg - 1; s >= 0; --s) {
    const int p = s & 1;
    const bool act = s < my_len;
    float dh_rec = 0.f;
    if (act && s + 1 < my_len) {
      const float *rp = red + (size_t)(p ^ 1) * cs * bc * Hc + bb * Hc + j;
      for (int q = 0; q < cs; ++q) dh_rec += rp[(size_t)q * bc * Hc];
    }
    const float ig = gn[0], fg = gn[1], gg = gn[2], og = gn[3];
    const float ct = cn, cp = cpn, dy = dyn;
    const int tok = tokn;
    if (s - 1 >= 0 && s - 1 < my_len) prefetch(s - 1);
    if (act) {
      const float dh = dy + dh_rec;
      const float tc = tanhf(ct);
      dc = fmaf(dh * og, 1.f - tc * tc, dc);
      const float dzi = dc * gg * ig * (1.f - ig);
      const float dzf = dc * cp * fg * (1.f - fg);
      const float dzg = dc * ig * (1.f - gg * gg);
      const float dzo = dh * tc * og * (1.f - og);
      dc *= fg;
      if (kp == 0) {
        float *zr = Z + (size_t)tok * G + col;
        zr[0] = dzi;
        zr[H] = dzf;
        zr[2 * H] = dzg;
        zr[3 * H] = dzo;
        float *dr = dzs + bb * RZ + j;
        dr[0] = dzi;
        dr[Hc] = dzf;
        dr[2 * Hc] = dzg;
        dr[3 * Hc] = dzo;
      }
    }
    __syncthreads();
    while (nact < bc && rl[nact] > s) ++nact;
    // partial dh_{prev}[b][k] = sum over this CTA's 4*Hc rows of W_hh[row][k] dz[b][row]
    const int items = nact * H;
    for (int it = tid; it < items; it += blockDim.x) {
      const int b2 = it / H, k = it % H;
      const float *dz = dzs + b2 * RZ;
      float sum = 0.f;
      if (WS) {
        const float *wc = Ws + k;
        for (int row = 0; row < 4 * Hc; ++row) sum = fmaf(wc[row * HP], dz[row], sum);
      } else {
        for (int q = 0; q < 4; ++q) {
          const float *wc = Whh + (size_t)(q * H + c * Hc) * H + k;
          for (int jr = 0; jr < Hc; ++jr) sum = fmaf(__ldg(wc + (size_t)jr * H), dz[q * Hc + jr], sum);
        }
      }
      const int owner = k / Hc, jj = k % Hc;
      float *dst = red + ((size_t)(p * cs + c) * bc + b2) * Hc + jj;
      *cluster.map_shared_rank(dst, owner) = sum;
    }
    cluster.sync();
  }
}

// ---------------------------------------------------------------------------
namespace {

int pick_ks(int pairs, int H) {
  int ks = 1;
  while (ks < 8 && pairs * ks * 2 <= 256 && 4 * ks * 2 <= ((H + 3) & ~3)) ks *= 2;
  return ks;
}

template <typename K>
bool cluster_fits(K kernel, int cs, int threads, size_t smem) {
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (cs > 8 && cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cs, 1, 1);
  cfg.blockDim = dim3(threads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cs;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return n > 0;
}

}  // namespace

RecGeom plan_recurrent(int H, int b, int dirs, int sm_count, bool bf16) {
  const int Tcap = kTokSmemCap - 1;
  const size_t lim = 220 * 1024;
  RecGeom g{};
  if (bf16 && tc_rec_supported(H)) {
    const int resident = tc_clusters_resident();
    if (resident > 0) {
      g.mode = 3;
      g.cs = 8;
      g.bc = resident;
      g.ks = 1;
      g.threads = 512;
      g.w_smem = 0;
      return g;
    }
  }
  if (cta_supported(H)) {
    g.mode = 1;
    g.cs = 1;
    g.bc = cta_rows_per_block(H, b, dirs, sm_count);
    g.ks = 1;
    g.threads = 4 * H;
    g.w_smem = 1;
    return g;
  }
  if (cl_cluster_size(H) > 0) {
    const int bc = plan_cl_rows(H, b, dirs);
    if (bc > 0) {
      g.mode = 2;
      g.cs = cl_cluster_size(H);
      g.bc = bc;
      g.ks = 1;
      g.threads = 256;
      g.w_smem = 1;
      return g;
    }
  }
  int cs = 16;
  while (cs > 1 && (H % cs != 0 || H / cs < 8)) cs >>= 1;
  for (;; cs >>= 1) {
    const int Hc = H / cs;
    const int ng = std::max(1, sm_count / (dirs * cs));
    int bc = (b + ng - 1) / ng;
    while (bc > 1 && bc * Hc > 512) bc = (bc + 1) / 2;
    const int pairs = bc * Hc;
    const int ks = pick_ks(pairs, H);
    const int threads = std::min(512, std::max(64, ((pairs * ks + 31) / 32) * 32));
    size_t sf = rec_smem_bytes(false, true, H, cs, bc, Tcap), sb = rec_smem_bytes(true, true, H, cs, bc, Tcap);
    bool ws = true;
    if ((sf > lim || sb > lim) && H % 4 == 0) {
      ws = false;  // W_hh slice read from L2 every step
      sf = rec_smem_bytes(false, false, H, cs, bc, Tcap);
      sb = rec_smem_bytes(true, false, H, cs, bc, Tcap);
    }
    g.cs = cs;
    g.bc = bc;
    g.ks = ks;
    g.threads = threads;
    g.w_smem = ws ? 1 : 0;
    g.smem_fwd = sf;
    g.smem_bwd = sb;
    if (cs == 1) break;
    const bool ok = ws ? (cluster_fits(lstm_fwd_kernel<true>, cs, threads, sf) &&
                          cluster_fits(lstm_bwd_kernel<true>, cs, threads, sb))
                       : (cluster_fits(lstm_fwd_kernel<false>, cs, threads, sf) &&
                          cluster_fits(lstm_bwd_kernel<false>, cs, threads, sb));
    if (ok) break;
  }
  return g;
}

namespace {

template <typename K>
cudaError_t launch_rec(K kernel, const RecArgs &a, const RecGeom &g, bool bwd, cudaStream_t s) {
  const int ng = (a.ix.b + g.bc - 1) / g.bc;
  const size_t smem = rec_smem_bytes(bwd, g.w_smem != 0, a.H, g.cs, g.bc, a.ix.T);
  cudaError_t e = ensure_smem((const void *)kernel, smem, g.cs > 8);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ng * a.dirs * g.cs, 1, 1);
  cfg.blockDim = dim3(g.threads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = g.cs;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, a, g.cs, g.bc, g.ks);
}

}  // namespace

cudaError_t launch_lstm_fwd(const RecArgs &a, const RecGeom &g, cudaStream_t s) {
  if (g.mode == 3) return launch_lstm_tc(a, g.bc, false, s);
  if (g.mode == 1) return launch_lstm_cta(a, g.bc, false, s);
  if (g.mode == 2) return launch_lstm_cl(a, g.bc, false, s);
  if (a.H % g.cs != 0) return cudaErrorInvalidValue;
  if (!g.w_smem && (a.H % 4) != 0) return cudaErrorInvalidValue;
  return g.w_smem ? launch_rec(lstm_fwd_kernel<true>, a, g, false, s) : launch_rec(lstm_fwd_kernel<false>, a, g, false, s);
}

cudaError_t launch_lstm_bwd(const RecArgs &a, const RecGeom &g, cudaStream_t s) {
  if (g.mode == 3) return launch_lstm_tc(a, g.bc, true, s);
  if (g.mode == 1) return launch_lstm_cta(a, g.bc, true, s);
  if (g.mode == 2) return launch_lstm_cl(a, g.bc, true, s);
  if (a.H % g.cs != 0) return cudaErrorInvalidValue;
  if (!g.w_smem && (a.H % 4) != 0) return cudaErrorInvalidValue;
  return g.w_smem ? launch_rec(lstm_bwd_kernel<true>, a, g, true, s) : launch_rec(lstm_bwd_kernel<false>, a, g, true, s);
}

}  // namespace bkt
