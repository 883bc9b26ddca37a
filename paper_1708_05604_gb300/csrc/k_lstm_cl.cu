// k_lstm_cl.cu -- register-tiled cluster kernels of the recurrence for
// H = 256 and H = 512 (a6 forward, a11 BPTT).
//
// The fp32 W_hh of one direction (1 MB at H = 256, 4 MB at H = 512) does not
// fit one SM, so a thread-block cluster of CS CTAs shares it: CTA c owns the
// Hc = H / CS hidden units [c Hc, (c+1) Hc), i.e. 4 Hc gate rows, 256 KB of
// weights per CTA (CS = 4 at H = 256, CS = 16 at H = 512), kept for the whole
// sequence half in registers and half in shared memory.  A cluster owns BC
// consecutive rows of the length-sorted batch and runs as many steps as its
// longest row; clusters never wait on each other.
//
// Forward step (z_t = Zx_t + W_hh h_{t-1}; gates i, f, g, o):
//   thread (u, kl) holds rows {q H + c Hc + u : q = i, f, g, o} of W_hh over
//   the 64 columns kl*64 .. kl*64 + 63 and forms 4 x BC partial dot products
//   against h_{t-1}; a shuffle reduce-scatter over the KS = H / 64 threads of
//   a unit leaves each lane whole gate sets (or a gate pair, swapped with its
//   neighbour), so the cell state stays in registers.  The CTA's slice of h_t
//   is then sent to every CTA of the cluster.
// BPTT step: (B) dh = dY + W_hh^T dz_{t+1} (the sum of the CS partials this
//   CTA received for its units), dz of the four gates; (A) thread (cg, rs)
//   holds the 64 local gate rows rs*64 .. rs*64 + 63 over the 4 columns
//   4 cg .. 4 cg + 3 and forms the partial W_hh^T dz over its rows for all BC
//   rows; a reduce-scatter over the row slices finishes the CTA's partial,
//   and each column block is sent to the CTA that owns those units.
//
// Exchange.  Remote writes are st.async stores into a double-buffered
// receive array of the destination, each completing bytes on the
// destination's mbarrier for that buffer; a CTA waits only for its own
// mbarrier (every source sends the same byte count each step, zeros for rows
// that have ended).  A step's send happens after the CTA barrier that closes
// every read of the buffer it will reuse two steps later, so the data
// dependence itself orders reuse and no cluster-wide barrier is needed per
// step.  Every wait is bounded: on expiry the kernel sets bit 4 of the status
// word, leaves its loop at the next CTA barrier, sleeps 20 us so that stores
// its peers issued before they gave up can land, and all CTAs meet at a final
// cluster barrier.  (A peer gives up only after its own bounded wait, at
// least 256 polls after its last store.)
#include <cstdint>

#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

namespace {

constexpr int kClThreads = 256;
#ifndef BKT_CL_FWD_REG_COLS
#define BKT_CL_FWD_REG_COLS 32
#endif
constexpr int kClFwdRegCols = BKT_CL_FWD_REG_COLS;  // multiple of 4, at most 64
constexpr int kClTokCap = 8192;  // time offsets staged in shared memory up to this T
constexpr int kClPolls = 1 << 22;
constexpr int32_t kErrExchange = kErrExchWait;

// Gate nonlinearities from the exponential intrinsic: sigma(x) = 1 / (1 + e^-x)
// and tanh(x) = 1 - 2 / (1 + e^2x) (absolute error a few 1e-8; both saturate
// correctly when the exponential overflows to +inf or underflows to 0).
__device__ __forceinline__ float sigm_cl(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }
__device__ __forceinline__ float tanh_cl(float x) { return 1.f - __fdividef(2.f, 1.f + __expf(2.f * x)); }

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t peer_addr(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ uint32_t cta_rank_in_cluster() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_barrier_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void mbar_init1(uint32_t mb) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mb) : "memory");
}
// One local arrival plus `bytes` of transactions complete the phase.
__device__ __forceinline__ void mbar_arm(uint32_t mb, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t mb, uint32_t parity, int cap) {
  for (int i = 0; i < cap; ++i) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(mb), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}
// 16-byte remote store that completes 16 bytes on the remote mbarrier.
__device__ __forceinline__ void st_async4(uint32_t raddr, float4 v, uint32_t rmbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(raddr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rmbar)
               : "memory");
}

// Per-thread asynchronous 4-byte copy global -> shared (the next step's
// inputs are requested a whole step before they are read).
__device__ __forceinline__ void cp_async4_cl(float *dst, const float *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit_cl() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_all_cl() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Reduce-scatter of N values over the KS lanes that differ in lane bits
// 0 .. log2(KS)-1: on return v[0 .. N/KS - 1] of lane l holds the sums of
// positions (l % KS) * N/KS .. (l % KS + 1) * N/KS - 1.
template <int N, int KS>
__device__ __forceinline__ void reduce_scatter_lanes(float (&v)[N], int lane) {
  constexpr int kStages = KS == 1 ? 0 : KS == 2 ? 1 : KS == 4 ? 2 : KS == 8 ? 3 : 4;
  static_assert((1 << kStages) == KS && KS <= 16, "KS is a power of two <= 16");
#pragma unroll
  for (int st = 0; st < kStages; ++st) {
    const int m = KS >> (st + 1);
    const int half = (N >> st) / 2;
    const bool hi = (lane & m) != 0;
#pragma unroll
    for (int i = 0; i < N / 2; ++i) {
      if (i < half) {
        const float send = hi ? v[i] : v[i + half];
        const float keep = hi ? v[i + half] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, m);
      }
    }
  }
}

template <int H, int CS, int BC, int NH>
struct ClGeom {
  static constexpr int Hc = H / CS;          // hidden units per CTA
  static constexpr int KS = H / 64;          // 64-column slices (forward)
  static constexpr int R = 4 * Hc;           // gate rows per CTA
  static constexpr int RSL = R / 64;         // 64-row slices (BPTT)
  static constexpr int BH = BC / NH;         // rows per half
  static constexpr int HPAD = H + 4 * KS;    // h row: 4 floats of padding after each slice
  static constexpr int DZS = R * BH + 4 * RSL;  // dz buffer of a half: [R][BH], 4 floats after each 64 rows
  static constexpr uint32_t kXBytes = BH * H * 4;  // bytes a CTA receives per half and step
  static_assert(Hc * KS == kClThreads && (H / 4) * RSL == kClThreads, "256 threads per CTA");
  static_assert(Hc % 4 == 0 && BH % 4 == 0 && BC == BH * NH, "float4 exchange");
  static constexpr int PPT = (Hc * BH + kClThreads - 1) / kClThreads;  // BPTT pairs per thread and half
  static constexpr int RKF = kClFwdRegCols;   // forward: W columns of a 64-column slice kept in registers
  static size_t fwd_floats() { return (size_t)(64 - RKF) * 4 * kClThreads + 2 * NH * BH * (HPAD + Hc); }
  static size_t bwd_floats() {
    return (size_t)32 * kClThreads * 4 + 2 * NH * (DZS + (size_t)CS * BH * Hc) + (size_t)2 * NH * kClThreads * PPT * 8;
  }
};

size_t cl_tail_bytes(int NH, int T) { return 16 * NH + (T + 1 <= kClTokCap ? (size_t)(T + 1) * 4 : 0); }

}  // namespace

// Rows of a cluster are processed as NH halves of BH rows, one after the
// other within a step, each with its own receive buffers and mbarriers, so
// the exchange of one half overlaps the arithmetic of the other.
// The body of one cluster: direction d, rows r0 .. r0 + BC - 1.
template <int H, int CS, int BC, int NH>
__device__ __forceinline__ void fwd_cl_body(const RecArgs &a, float *sm, const int d, const int r0) {
  using Gm = ClGeom<H, CS, BC, NH>;
  constexpr int Hc = Gm::Hc, KS = Gm::KS, HPAD = Gm::HPAD, BH = Gm::BH, G = 4 * H, NTH = kClThreads;
  constexpr int NV = 4 * BH, NPL = NV / KS;  // partial sums per thread, per lane after the reduction
  static_assert(NPL == 2 || NPL % 4 == 0, "a lane finishes whole units or one gate pair");
  constexpr int RPL = NPL >= 4 ? NPL / 4 : 1;  // rows of a half finished per lane
  constexpr int SEND4 = BH * Hc / 4;           // float4 sent to each CTA per half and step
  constexpr int RK = Gm::RKF, SK4 = (64 - RK) / 4;  // register columns, shared float4 columns
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SK4][4][NTH] columns RK..63 of each slice
  float *hb = sm + SK4 * 4 * NTH * 4;            // [NH][2][BH][HPAD] received h
  float *stg = hb + 2 * NH * BH * HPAD;          // [NH][2][BH][Hc] this CTA's h slice
  uint64_t *mb = reinterpret_cast<uint64_t *>(stg + 2 * NH * BH * Hc);  // [NH][2]
  int *toff_s = reinterpret_cast<int *>(mb + 2 * NH);
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kClTokCap;
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;

  const int t = threadIdx.x, lane = t & 31;
  const int kl = t % KS, u = t / KS;
  const uint32_t c = cta_rank_in_cluster();
  const int gu = (int)c * Hc + u, kb = kl * 64;
  const int DH = a.dirs * H;
  const float *__restrict__ Whh = a.Whh[d];

  float w[4][RK];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float *row = Whh + (size_t)(q * H + gu) * H + kb;
#pragma unroll
    for (int k = 0; k < RK; ++k) w[q][k] = __ldg(row + k);
#pragma unroll
    for (int j = 0; j < SK4; ++j) {
      const float *p = row + RK + 4 * j;
      Ws4[(j * 4 + q) * NTH + t] = make_float4(__ldg(p), __ldg(p + 1), __ldg(p + 2), __ldg(p + 3));
    }
  }
  if (toff_sm)
    for (int i = t; i <= T; i += NTH) toff_s[i] = a.ix.tok_off[i];
  const int Tg = (r0 < a.ix.b) ? a.ix.row_len[r0] : 0;
  if (t == 0) {
    for (int i = 0; i < 2 * NH; ++i) mbar_init1(smem_addr(&mb[i]));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_barrier_all();  // barriers initialised everywhere before any remote store
  if (t == 0)
    for (int h = 0; h < NH; ++h) {
      if (Tg >= 2) mbar_arm(smem_addr(&mb[2 * h]), Gm::kXBytes);
      if (Tg >= 3) mbar_arm(smem_addr(&mb[2 * h + 1]), Gm::kXBytes);
    }

  float *__restrict__ Z = a.Z[d];
  float *__restrict__ Cs = a.Cst[d];
  float *__restrict__ Y = a.Y;
  // lane ownership after the reduction (rows counted within a half): rows
  // kl*RPL + rr with all four gates, or (NPL == 2) row kl/2 with gates
  // 2*(kl&1), 2*(kl&1)+1
  auto own_row = [&](int rr) { return NPL >= 4 ? kl * RPL + rr : kl >> 1; };
  auto own_gate = [&](int j) { return NPL >= 4 ? (j & 3) : 2 * (kl & 1) + j; };
  int olen[NH][RPL];  // lengths of the owned rows (read directly: a runtime index into an array would live in local memory)
#pragma unroll
  for (int h = 0; h < NH; ++h)
#pragma unroll
    for (int rr = 0; rr < RPL; ++rr) {
      const int r = r0 + h * BH + own_row(rr);
      olen[h][rr] = r < a.ix.b ? a.ix.row_len[r] : 0;
    }
  auto tok_at = [&](int h, int rr, int s) {
    const int tt = d == 0 ? s : olen[h][rr] - 1 - s;
    return toff[tt] + r0 + h * BH + own_row(rr);
  };
  auto zx_at = [&](int h, int j, int s) {  // owned pre-activation j of step s (0 once the row has ended)
    const int rr = NPL >= 4 ? j / 4 : 0;
    return (s < olen[h][rr]) ? Z[(size_t)tok_at(h, rr, s) * G + own_gate(j) * H + gu] : 0.f;
  };
  // the next step's pre-activations are loaded into registers one step ahead
  // (a shared-memory ring with asynchronous copies measured slower here)
  float zn[NH][NPL], cst[NH][RPL];
#pragma unroll
  for (int h = 0; h < NH; ++h) {
#pragma unroll
    for (int j = 0; j < NPL; ++j) zn[h][j] = zx_at(h, j, 0);
#pragma unroll
    for (int rr = 0; rr < RPL; ++rr) cst[h][rr] = 0.f;
  }
  bool ok = true, stop = false;
  const int cap = a.wf.poll_cap > 0 ? a.wf.poll_cap : kClPolls;
  // failure-detection hook: CTA 0 of the cluster withholds its exchange data
  const bool withhold = (a.wf.withhold & kWithholdExchange) && c == 0;

  for (int s = 0; s < Tg && !stop; ++s) {
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      float zc[NPL];
#pragma unroll
      for (int j = 0; j < NPL; ++j) zc[j] = zn[h][j];
      if (s + 1 < Tg) {
#pragma unroll
        for (int j = 0; j < NPL; ++j) zn[h][j] = zx_at(h, j, s + 1);
      }
      float acc[NV];
#pragma unroll
      for (int i = 0; i < NV; ++i) acc[i] = 0.f;
      if (s > 0) {  // h_{-1} = 0
        const int e = s - 1;
        ok = mbar_wait_bounded(smem_addr(&mb[2 * h + (e & 1)]), (e >> 1) & 1, cap) && ok;
        // re-arm only a phase that completed: arriving again on a phase whose
        // wait ran out would over-arrive on it (its one arrival is spent)
        if (t == 0 && ok && e + 2 <= Tg - 2) mbar_arm(smem_addr(&mb[2 * h + (e & 1)]), Gm::kXBytes);
        const float *hv = hb + (2 * h + (e & 1)) * BH * HPAD + kb + 4 * kl;
#pragma unroll
        for (int k4 = 0; k4 < RK / 4; ++k4) {
#pragma unroll
          for (int b = 0; b < BH; ++b) {
            const float4 h4 = *reinterpret_cast<const float4 *>(hv + b * HPAD + 4 * k4);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float x = fmaf(w[q][4 * k4], h4.x, acc[b * 4 + q]);
              x = fmaf(w[q][4 * k4 + 1], h4.y, x);
              x = fmaf(w[q][4 * k4 + 2], h4.z, x);
              acc[b * 4 + q] = fmaf(w[q][4 * k4 + 3], h4.w, x);
            }
          }
        }
#pragma unroll
        for (int j = 0; j < SK4; ++j) {
          float4 wv[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) wv[q] = Ws4[(j * 4 + q) * NTH + t];
#pragma unroll
          for (int b = 0; b < BH; ++b) {
            const float4 h4 = *reinterpret_cast<const float4 *>(hv + b * HPAD + RK + 4 * j);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float x = fmaf(wv[q].x, h4.x, acc[b * 4 + q]);
              x = fmaf(wv[q].y, h4.y, x);
              x = fmaf(wv[q].z, h4.z, x);
              acc[b * 4 + q] = fmaf(wv[q].w, h4.w, x);
            }
          }
        }
      }
      reduce_scatter_lanes<NV, KS>(acc, lane);
      float *sg = stg + (2 * h + (s & 1)) * BH * Hc;
      if constexpr (NPL >= 4) {
#pragma unroll
        for (int rr = 0; rr < RPL; ++rr) {
          float hval = 0.f;
          if (s < olen[h][rr]) {
            const float ig = sigm_cl(acc[rr * 4] + zc[rr * 4]);
            const float fg = sigm_cl(acc[rr * 4 + 1] + zc[rr * 4 + 1]);
            const float gg = tanh_cl(acc[rr * 4 + 2] + zc[rr * 4 + 2]);
            const float og = sigm_cl(acc[rr * 4 + 3] + zc[rr * 4 + 3]);
            cst[h][rr] = fmaf(fg, cst[h][rr], ig * gg);
            hval = og * tanh_cl(cst[h][rr]);
            const size_t tk = (size_t)tok_at(h, rr, s);
            float *zr = Z + tk * G + gu;
            zr[0] = ig;
            zr[H] = fg;
            zr[2 * H] = gg;
            zr[3 * H] = og;
            Cs[tk * H + gu] = cst[h][rr];
            Y[tk * DH + d * H + gu] = hval;
          }
          sg[own_row(rr) * Hc + u] = hval;
        }
      } else {
        const int pr = kl & 1;  // pr 0: (i, f), pr 1: (g, o)
        const float a0 = pr ? tanh_cl(acc[0] + zc[0]) : sigm_cl(acc[0] + zc[0]);
        const float a1 = sigm_cl(acc[1] + zc[1]);
        const float x0 = __shfl_xor_sync(0xffffffffu, a0, 1), x1 = __shfl_xor_sync(0xffffffffu, a1, 1);
        const float ig = pr ? x0 : a0, fg = pr ? x1 : a1, gg = pr ? a0 : x0, og = pr ? a1 : x1;
        float hval = 0.f;
        if (s < olen[h][0]) {
          cst[h][0] = fmaf(fg, cst[h][0], ig * gg);
          hval = og * tanh_cl(cst[h][0]);
          const size_t tk = (size_t)tok_at(h, 0, s);
          Z[tk * G + (2 * pr) * H + gu] = a0;
          Z[tk * G + (2 * pr + 1) * H + gu] = a1;
          if (pr) {
            Cs[tk * H + gu] = cst[h][0];
            Y[tk * DH + d * H + gu] = hval;
          }
        }
        if (!pr) sg[own_row(0) * Hc + u] = hval;
      }
      if (__syncthreads_or(!ok)) {
        if (t == 0) atomicOr(a.status, kErrExchange);
        stop = true;
        break;
      }
      if (s + 1 < Tg && !withhold) {  // exchange s of half h: this CTA's slice to every CTA of the cluster
        const uint32_t dst0 = smem_addr(hb + (2 * h + (s & 1)) * BH * HPAD), mbl = smem_addr(&mb[2 * h + (s & 1)]);
        for (int n = t; n < CS * SEND4; n += NTH) {
          const int peer = n / SEND4, rem = n % SEND4, b = rem / (Hc / 4), u4 = rem % (Hc / 4);
          const float4 v = *reinterpret_cast<const float4 *>(sg + b * Hc + 4 * u4);
          const int k = (int)c * Hc + 4 * u4;
          const uint32_t dst = dst0 + 4u * (uint32_t)(b * HPAD + k + (k >> 6) * 4);
          st_async4(peer_addr(dst, peer), v, peer_addr(mbl, peer));
        }
      }
    }
  }
  // after an abort, stores a peer issued before it gave up may still be in
  // flight toward this CTA: give them time to land before the cluster exits
  if (stop) __nanosleep(20000);
  cluster_barrier_all();  // no CTA leaves while a peer may still address its shared memory
}

// The body of one cluster: direction d, rows r0 .. r0 + BC - 1.
template <int H, int CS, int BC, int NH>
__device__ __forceinline__ void bwd_cl_body(const RecArgs &a, float *sm, const int d, const int r0) {
  using Gm = ClGeom<H, CS, BC, NH>;
  constexpr int Hc = Gm::Hc, RSL = Gm::RSL, BH = Gm::BH, G = 4 * H, NTH = kClThreads, DZS = Gm::DZS;
  constexpr int NV = 4 * BH, NPL = NV / RSL;  // partials per thread, per lane after the reduction
  static_assert(NPL % 4 == 0, "a lane finishes whole float4 column groups");
  constexpr int PAIRS = Hc * BH, PPT = Gm::PPT;  // (unit, row) pairs of a half
  float4 *Wb4 = reinterpret_cast<float4 *>(sm);  // [32][NTH] rows 32..63 of each row slice
  float *dzs = sm + 32 * NTH * 4;                // [NH][2][DZS] dz of this CTA's gate rows
  float *red = dzs + 2 * NH * DZS;               // [NH][2][CS][BH][Hc] received partials of W_hh^T dz
  float *ring = red + 2 * NH * CS * BH * Hc;     // [NH][2][PPT][8][NTH] phase B inputs of this and the next step
  uint64_t *mb = reinterpret_cast<uint64_t *>(ring + 2 * NH * NTH * PPT * 8);  // [NH][2]
  int *toff_s = reinterpret_cast<int *>(mb + 2 * NH);
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kClTokCap;
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;

  const int t = threadIdx.x, lane = t & 31;
  const int rs = t % RSL, cgp = t / RSL, k0 = 4 * cgp;
  const uint32_t c = cta_rank_in_cluster();
  const int DH = a.dirs * H;
  const float *__restrict__ Whh = a.Whh[d];
  auto dz_at = [&](int r, int b) { return r * BH + (r >> 6) * 4 + b; };

  // local gate row r = q * Hc + uu is global row q * H + c * Hc + uu
  float wr[32][4];
#pragma unroll
  for (int j = 0; j < 64; ++j) {
    const int r = rs * 64 + j;
    const float *p = Whh + (size_t)((r / Hc) * H + (int)c * Hc + r % Hc) * H + k0;
    const float4 v = make_float4(__ldg(p), __ldg(p + 1), __ldg(p + 2), __ldg(p + 3));
    if (j < 32) {
      wr[j][0] = v.x;
      wr[j][1] = v.y;
      wr[j][2] = v.z;
      wr[j][3] = v.w;
    } else {
      Wb4[(j - 32) * NTH + t] = v;
    }
  }
  if (toff_sm)
    for (int i = t; i <= T; i += NTH) toff_s[i] = a.ix.tok_off[i];
  const int Tg = (r0 < a.ix.b) ? a.ix.row_len[r0] : 0;
  if (t == 0) {
    for (int i = 0; i < 2 * NH; ++i) mbar_init1(smem_addr(&mb[i]));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_barrier_all();
  if (t == 0)
    for (int h = 0; h < NH; ++h) {
      if (Tg >= 2) mbar_arm(smem_addr(&mb[2 * h]), Gm::kXBytes);
      if (Tg >= 3) mbar_arm(smem_addr(&mb[2 * h + 1]), Gm::kXBytes);
    }

  float *__restrict__ Z = a.Z[d];
  const float *__restrict__ Cs = a.Cst[d];
  const float *__restrict__ dY = a.dY;
  // phase B pairs of half h: pair index i -> unit i % Hc, row h*BH + i / Hc
  int plen[NH][PPT];  // row lengths of the pairs (0 for pairs past the end)
#pragma unroll
  for (int h = 0; h < NH; ++h)
#pragma unroll
    for (int p = 0; p < PPT; ++p) {
      const int i = t + p * NTH, r = r0 + h * BH + i / Hc;
      plen[h][p] = (i < PAIRS && r < a.ix.b) ? a.ix.row_len[r] : 0;
    }
  auto tok_at = [&](int h, int p, int s) {
    const int tt = d == 0 ? s : plen[h][p] - 1 - s;
    return toff[tt] + r0 + h * BH + (t + p * NTH) / Hc;
  };
  // phase B inputs of step s (gates, c_t, c_{t-1}, dY) into ring slot s & 1;
  // value v of a thread sits at slot + v * NTH, so a warp's copies and reads
  // touch consecutive words (no bank conflicts)
  auto slot_of = [&](int h, int p, int s) { return ring + ((size_t)(2 * h + (s & 1)) * PPT + p) * 8 * NTH + t; };
  auto issue = [&](int h, int p, int s) {
    const int i = t + p * NTH;
    const int gu = (int)c * Hc + i % Hc;
    if (i < PAIRS && s >= 0 && s < plen[h][p]) {
      float *sl = slot_of(h, p, s);
      const size_t tk = (size_t)tok_at(h, p, s);
#pragma unroll
      for (int q = 0; q < 4; ++q) cp_async4_cl(sl + q * NTH, Z + tk * G + q * H + gu);
      cp_async4_cl(sl + 4 * NTH, Cs + tk * H + gu);
      if (s > 0) cp_async4_cl(sl + 5 * NTH, Cs + (size_t)tok_at(h, p, s - 1) * H + gu);
      else sl[5 * NTH] = 0.f;
      cp_async4_cl(sl + 6 * NTH, dY + tk * DH + d * H + gu);
    }
  };
  float dc[NH][PPT];
#pragma unroll
  for (int h = 0; h < NH; ++h)
#pragma unroll
    for (int p = 0; p < PPT; ++p) {
      dc[h][p] = 0.f;
      issue(h, p, Tg - 1);
    }
  cp_commit_cl();
  bool ok = true, stop = false;
  const int cap = a.wf.poll_cap > 0 ? a.wf.poll_cap : kClPolls;
  // failure-detection hook: CTA 0 of the cluster withholds its exchange data
  const bool withhold = (a.wf.withhold & kWithholdExchange) && c == 0;

  for (int it = 0; it < Tg && !stop; ++it) {
    const int s = Tg - 1 - it;
    cp_wait_all_cl();  // this step's inputs, requested one step ago
#pragma unroll
    for (int h = 0; h < NH; ++h)
#pragma unroll
      for (int p = 0; p < PPT; ++p) issue(h, p, s - 1);  // a row that starts later gets its first step too
    cp_commit_cl();
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      if (it > 0) {
        const int e = it - 1;
        ok = mbar_wait_bounded(smem_addr(&mb[2 * h + (e & 1)]), (e >> 1) & 1, cap) && ok;
        // re-arm only a phase that completed: arriving again on a phase whose
        // wait ran out would over-arrive on it (its one arrival is spent)
        if (t == 0 && ok && e + 2 <= Tg - 2) mbar_arm(smem_addr(&mb[2 * h + (e & 1)]), Gm::kXBytes);
      }
      float *dzb = dzs + (2 * h + (it & 1)) * DZS;
      // phase B
#pragma unroll
      for (int p = 0; p < PPT; ++p) {
        const int i = t + p * NTH;
        if (i >= PAIRS) continue;
        const int uu = i % Hc, b = i / Hc, gu = (int)c * Hc + uu;
        if (s < plen[h][p]) {
          const float *sl = slot_of(h, p, s);
          const float ig = sl[0], fg = sl[NTH], gg = sl[2 * NTH], og = sl[3 * NTH];
          const float ct = sl[4 * NTH], cp = sl[5 * NTH], dy = sl[6 * NTH];
          float dh_rec = 0.f;
          if (s + 1 < plen[h][p]) {
            const float *rp = red + (size_t)(2 * h + ((it - 1) & 1)) * CS * BH * Hc + b * Hc + uu;
#pragma unroll
            for (int cc = 0; cc < CS; ++cc) dh_rec += rp[cc * BH * Hc];
          }
          const float dh = dy + dh_rec;
          const float tch = tanh_cl(ct);
          const float dcv = fmaf(dh * og, 1.f - tch * tch, dc[h][p]);
          const float dzi = dcv * gg * ig * (1.f - ig);
          const float dzf = dcv * cp * fg * (1.f - fg);
          const float dzg = dcv * ig * (1.f - gg * gg);
          const float dzo = dh * tch * og * (1.f - og);
          dc[h][p] = dcv * fg;
          const size_t tk = (size_t)tok_at(h, p, s);
          float *zr = Z + tk * G + gu;
          zr[0] = dzi;
          zr[H] = dzf;
          zr[2 * H] = dzg;
          zr[3 * H] = dzo;
          dzb[dz_at(uu, b)] = dzi;
          dzb[dz_at(Hc + uu, b)] = dzf;
          dzb[dz_at(2 * Hc + uu, b)] = dzg;
          dzb[dz_at(3 * Hc + uu, b)] = dzo;
        } else {
#pragma unroll
          for (int q = 0; q < 4; ++q) dzb[dz_at(q * Hc + uu, b)] = 0.f;
        }
      }
      if (__syncthreads_or(!ok)) {
        if (t == 0) atomicOr(a.status, kErrExchange);
        stop = true;
        break;
      }
      if (it + 1 >= Tg || withhold) continue;  // dh_{-1} is not needed
      // phase A: partial W_hh^T dz over this thread's 64 rows, columns k0..k0+3
      // (a [batch row][gate row] dz layout made phase B cheaper but this loop
      // slower, a net loss)
      float acc[NV];
#pragma unroll
      for (int i = 0; i < NV; ++i) acc[i] = 0.f;
#pragma unroll
      for (int j = 0; j < 64; ++j) {
        const int r = rs * 64 + j;
        float wv[4];
        if (j < 32) {
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) wv[cc] = wr[j][cc];
        } else {
          const float4 v = Wb4[(j - 32) * NTH + t];
          wv[0] = v.x;
          wv[1] = v.y;
          wv[2] = v.z;
          wv[3] = v.w;
        }
#pragma unroll
        for (int m = 0; m < BH / 4; ++m) {
          const float4 z4 = *reinterpret_cast<const float4 *>(dzb + dz_at(r, 4 * m));
          const float zz[4] = {z4.x, z4.y, z4.z, z4.w};
#pragma unroll
          for (int bb = 0; bb < 4; ++bb)
#pragma unroll
            for (int cc = 0; cc < 4; ++cc)
              acc[(4 * m + bb) * 4 + cc] = fmaf(wv[cc], zz[bb], acc[(4 * m + bb) * 4 + cc]);
        }
      }
      reduce_scatter_lanes<NV, RSL>(acc, lane);
      // lane holds rows rs*(NPL/4) .. + NPL/4 - 1 of the half, columns k0..k0+3 -> the owner of those units
      const uint32_t owner = (uint32_t)(k0 / Hc);
      const int uo = k0 % Hc;
      const uint32_t dst0 =
          smem_addr(red + (size_t)(2 * h + (it & 1)) * CS * BH * Hc + (size_t)c * BH * Hc + uo);
      const uint32_t rmb = peer_addr(smem_addr(&mb[2 * h + (it & 1)]), owner);
#pragma unroll
      for (int rr = 0; rr < NPL / 4; ++rr) {
        const int b = rs * (NPL / 4) + rr;
        st_async4(peer_addr(dst0 + 4u * (uint32_t)(b * Hc), owner),
                  make_float4(acc[rr * 4], acc[rr * 4 + 1], acc[rr * 4 + 2], acc[rr * 4 + 3]), rmb);
      }
    }
  }
  cp_wait_all_cl();
  if (stop) __nanosleep(20000);  // in-flight peer stores after an abort (see the forward kernel)
  cluster_barrier_all();
}

// ---------------------------------------------------------------------------
// Cluster layout of a launch.  Clusters of 4 rows step faster than
// clusters of 8 (at H = 512, 16-CTA clusters, half the FMAs per CTA and
// step), but at most 7 such 16-CTA clusters fit on the GPU at once.  As in
// the tensor-core kernels, the longest rows of the length-sorted batch go to
// n4 four-row clusters per direction and the shortest to n8 eight-row
// clusters, with dirs (n4 + n8) no more than the resident clusters.
namespace {

struct ClSplit {
  int n4, n8;  // clusters per direction of 4 and of 8 rows
};

}  // namespace

template <int H, int CS>
__global__ void __launch_bounds__(kClThreads, 1) lstm_fwd_cl_kernel(RecArgs a, ClSplit sp) {
  extern __shared__ __align__(16) float sm[];
  const int cid = blockIdx.x / CS, per = sp.n4 + sp.n8;
  const int d = cid / per, g = cid % per;
  if (g < sp.n4)
    fwd_cl_body<H, CS, 4, 1>(a, sm, d, 4 * g);
  else
    fwd_cl_body<H, CS, 8, 1>(a, sm, d, 4 * sp.n4 + 8 * (g - sp.n4));
}

template <int H, int CS>
__global__ void __launch_bounds__(kClThreads, 1) lstm_bwd_cl_kernel(RecArgs a, ClSplit sp) {
  extern __shared__ __align__(16) float sm[];
  const int cid = blockIdx.x / CS, per = sp.n4 + sp.n8;
  const int d = cid / per, g = cid % per;
  if (g < sp.n4)
    bwd_cl_body<H, CS, 4, 1>(a, sm, d, 4 * g);
  else
    bwd_cl_body<H, CS, 8, 1>(a, sm, d, 4 * sp.n4 + 8 * (g - sp.n4));
}

namespace {

template <int H, int CS, int BC>
size_t cl_smem_one(bool bwd, int T) {
  using Gm = ClGeom<H, CS, BC, 1>;
  return (bwd ? Gm::bwd_floats() : Gm::fwd_floats()) * 4 + cl_tail_bytes(1, T);
}
// dynamic shared memory of a launch: the larger of the two bodies' layouts
template <int H, int CS>
size_t cl_smem(bool bwd, int T) {
  return std::max(cl_smem_one<H, CS, 4>(bwd, T), cl_smem_one<H, CS, 8>(bwd, T));
}

cudaLaunchConfig_t cl_config(int cs, int clusters, size_t smem, cudaStream_t s, cudaLaunchAttribute *attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(clusters * cs, 1, 1);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr->id = cudaLaunchAttributeClusterDimension;
  attr->val.clusterDim.x = cs;
  attr->val.clusterDim.y = 1;
  attr->val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

ClSplit cl_split(int b, int dirs, int max_clusters) {
  const int groups = (b + 3) / 4;                    // 4-row groups per direction
  const int per = std::max(1, max_clusters / dirs);  // clusters per direction resident at once
  ClSplit sp;
  if (groups <= per) {
    sp.n4 = groups;
    sp.n8 = 0;
  } else if (groups - per >= (groups + 1) / 2) {
    sp.n4 = 0;  // eight rows everywhere (clusters beyond the resident ones wait)
    sp.n8 = (groups + 1) / 2;
  } else {
    sp.n8 = groups - per;  // each eight-row cluster saves one cluster
    sp.n4 = groups - 2 * sp.n8;
  }
  return sp;
}

template <int H, int CS>
cudaError_t launch_cl(const RecArgs &a, int max_clusters, bool bwd, cudaStream_t s) {
  if (a.ix.b <= 0 || a.ix.T <= 0) return cudaSuccess;
  if (max_clusters <= 0 || a.dirs < 1 || a.dirs > 2) return cudaErrorInvalidValue;
  const ClSplit sp = cl_split(a.ix.b, a.dirs, max_clusters);
  const size_t smem = cl_smem<H, CS>(bwd, a.ix.T);
  const int clusters = (sp.n4 + sp.n8) * a.dirs;
  cudaLaunchAttribute attr;
  cudaLaunchConfig_t cfg = cl_config(CS, clusters, smem, s, &attr);
  if (bwd) {
    auto k = lstm_bwd_cl_kernel<H, CS>;
    cudaError_t e = ensure_smem((const void *)k, smem, CS > 8);
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&cfg, k, a, sp);
  }
  auto k = lstm_fwd_cl_kernel<H, CS>;
  cudaError_t e = ensure_smem((const void *)k, smem, CS > 8);
  if (e != cudaSuccess) return e;
  return cudaLaunchKernelEx(&cfg, k, a, sp);
}

// Clusters of the forward and the BPTT kernel that can be resident at once
// (0: the configuration cannot launch on this device).
template <int H, int CS>
int cl_resident(int T) {
  int lo = 1 << 30;
  for (int bwd = 0; bwd < 2; ++bwd) {
    const size_t smem = cl_smem<H, CS>(bwd != 0, T);
    cudaLaunchAttribute attr;
    int n = 0;
    cudaError_t e;
    cudaLaunchConfig_t cfg = cl_config(CS, 1, smem, 0, &attr);
    if (bwd) {
      auto k = lstm_bwd_cl_kernel<H, CS>;
      e = ensure_smem((const void *)k, smem, CS > 8);
      if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, k, &cfg);
    } else {
      auto k = lstm_fwd_cl_kernel<H, CS>;
      e = ensure_smem((const void *)k, smem, CS > 8);
      if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, k, &cfg);
    }
    if (e != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    lo = std::min(lo, n);
  }
  return lo;
}

}  // namespace

int cl_cluster_size(int H) { return H == 256 ? 4 : H == 512 ? 16 : 0; }

int plan_cl_rows(int H, int b, int dirs) {
  (void)b;
  (void)dirs;
  const int T = kClTokCap - 1;
  if (H == 256) return cl_resident<256, 4>(T);
  if (H == 512) return cl_resident<512, 16>(T);
  return 0;
}

cudaError_t launch_lstm_cl(const RecArgs &a, int max_clusters, bool bwd, cudaStream_t s) {
  if (a.H == 256) return launch_cl<256, 4>(a, max_clusters, bwd, s);
  if (a.H == 512) return launch_cl<512, 16>(a, max_clusters, bwd, s);
  return cudaErrorInvalidValue;
}

}  // namespace bkt
