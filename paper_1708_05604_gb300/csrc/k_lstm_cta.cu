// k_lstm_cta.cu -- single-CTA persistent recurrent kernels for H in {32, 64,
// 128} (a6 forward, a11 BPTT).
//
// Same recurrence as the cluster kernels (gates i, f, g, o; the reverse
// direction over each sequence's own length), but one CTA holds the whole
// 4H x H fp32 W_hh of its direction, so a time step needs no inter-SM
// exchange at all.
//
// Register tiling.  2H threads; lane l of warp w belongs to row group
// rg = 4w + l/8 and k slice ks = l % 8.  Row group rg is the 16 gate rows of
// units u0..u0+3 (u0 = 4 rg), ordered [i, f, g, o] per unit; k slice ks is the
// KPT = H/8 columns ks*KPT .. ks*KPT+KPT-1.  Each thread keeps its 16 x KPT
// tile of W_hh for the whole sequence: RKK columns in registers (192 weights
// at H = 128); the other SKK = KPT - RKK columns sit in tensor memory (TMEM)
// in the forward kernel, one 16-weight column per tcgen05.ld, and in shared
// memory in BPTT.  The forward matvec interleaves its two parts: the load of
// TMEM column j + 1 is in flight while the thread runs the register FMAs of
// block j + 1, so the TMEM reads (64 KB per step at H = 128) overlap the FMA
// pipe instead of following it, as shared-memory operands did (0.94 -> 0.72
// us per step).  BPTT's column sums over the 16 rows of a tile run as short
// chains per column; with TMEM columns between register blocks they lost
// their overlap and the step got slower (0.89 -> 1.0 us), so BPTT streams
// its SKK columns from shared memory.  A
// thread reads only the KPT values of h (forward) or the 16 values of dz
// (backward) that its tile needs, so the shared-memory bytes per step stay
// small; a shared-memory broadcast of all of h to every thread would cost
// 1 KB of load bandwidth per thread per step.
//
// Forward step: 16 partial dot products per thread over its k slice; an
// 8-lane shuffle reduce-scatter leaves lane ks with rows 2ks, 2ks+1 of the
// group, i.e. (i, f) or (g, o) of unit u0 + ks/2; activations; the two lanes
// of a unit swap their pair and both update c = f c + i g, h = o tanh(c);
// h goes to the other half of a double buffer; one CTA barrier.
// BPTT step: (B) lanes 2j, 2j+1 form dh = dY + sum of the per-warp partials
// of W_hh^T dz for unit j, and dz of its four gates (written in place over the
// gates); barrier; (A) each thread multiplies its tile by the 16 dz values of
// its rows, a shuffle reduce-scatter over the warp's four row groups sums the
// tile products per column, and each warp stores its column partials;
// barrier.
// A CTA owns BC consecutive rows of the length-sorted batch (BC = 1 when the
// batch fits the GPU) and stops after its longest row.  Each thread keeps the
// global inputs of the next kPF steps in flight with asynchronous copies into
// a small shared-memory ring (global-memory latency under load is about one
// time step).
#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

namespace {

constexpr int kTokCap = 8192;  // time offsets staged in shared memory up to this T
constexpr int kPF = 4;         // steps of per-step global inputs kept in flight
constexpr int kRing = kPF + 1; // ring slots: a copy never lands in the slot read this step

// Gate nonlinearities from the exponential intrinsic: sigma(x) = 1 / (1 + e^-x)
// and tanh(x) = 1 - 2 / (1 + e^2x) (absolute error a few 1e-8; both saturate
// correctly when the exponential overflows to +inf or underflows to 0).
__device__ __forceinline__ float sigm(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }
__device__ __forceinline__ float tanh_g(float x) { return 1.f - __fdividef(2.f, 1.f + __expf(2.f * x)); }

// The step inputs are whole rows (Zx or gates, cell states, dY), copied to a
// shared-memory ring in 16-byte asynchronous pieces by all threads together:
// one commit group per step.  A thread reads pieces other threads copied, so
// a step's group is completed one step early (wait_group kPF-2 at the top of
// the previous step) and published by that step's closing barrier.
__device__ __forceinline__ void cp_async16(float *dst, const float *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait_pending() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// TMEM part of the W_hh tile.  Thread t of warp w owns TMEM lane
// 32 (w % 4) + t % 32 (the lanes a warp may access) and, within it, the SKK
// x 16 columns from (w / 4) SKK 16: column 16 kk + ri holds weight
// (ri, RKK + kk) of its tile.  Columns per lane: SKK 16 for each warp that
// shares the lane quadrant.
template <int NTH, int SKK>
__host__ __device__ constexpr int tm_cols() {
  return SKK == 0 ? 0 : (NTH > 128 ? 2 : 1) * SKK * 16;
}
__device__ __forceinline__ void tm_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// Allocated by warp 0; every thread returns the base address (a CTA-wide
// barrier inside).  The allocation waits while another CTA on the SM holds
// the columns; none of the recurrent kernels waits on another CTA.
template <int NCOL>
__device__ __forceinline__ uint32_t tm_alloc(uint32_t *slot, int warp) {
  static_assert(NCOL >= 32 && NCOL <= 512 && (NCOL & (NCOL - 1)) == 0, "TMEM allocations are powers of 2 in 32..512");
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(slot))),
                 "r"(NCOL)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  return *slot;
}
template <int NCOL>
__device__ __forceinline__ void tm_free(uint32_t base, int warp) {
  tm_fence_before();
  __syncthreads();
  tm_fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(base), "r"(NCOL) : "memory");
}
__device__ __forceinline__ void tm_st16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}
__device__ __forceinline__ void tm_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, "
      "[%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
// Completes this thread's tcgen05.ld; the loaded registers pass through the
// wait, so no use of them is scheduled ahead of it.
__device__ __forceinline__ void tm_wait16(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
// The tile of the thread: RKK columns into w, the other SKK into TMEM at tw.
template <int H, int RKK, int SKK>
__device__ __forceinline__ void load_tile(const float *__restrict__ Whh, int u0, int kb, uint32_t tw,
                                          float (&w)[16][RKK > 0 ? RKK : 1]) {
#pragma unroll
  for (int ri = 0; ri < 16; ++ri) {
    const float *row = Whh + (size_t)((ri & 3) * H + u0 + (ri >> 2)) * H + kb;
#pragma unroll
    for (int kk = 0; kk < RKK; ++kk) w[ri][kk] = __ldg(row + kk);
  }
  if constexpr (SKK > 0) {
#pragma unroll 1
    for (int kk = 0; kk < SKK; ++kk) {
      uint32_t v[16];
#pragma unroll
      for (int ri = 0; ri < 16; ++ri)
        v[ri] = __float_as_uint(__ldg(Whh + (size_t)((ri & 3) * H + u0 + (ri >> 2)) * H + kb + RKK + kk));
      tm_st16(tw + 16 * kk, v);
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  }
}

// Reduce-scatter over the 8 lanes of a k-slice group (lane bits 0..2): on
// return, lane l holds the group sums of positions 2(l%8) and 2(l%8)+1.
__device__ __forceinline__ void reduce_scatter8(const float (&v)[16], int lane, float &o0, float &o1) {
  const bool b2 = (lane >> 2) & 1, b1 = (lane >> 1) & 1, b0 = lane & 1;
  float r8[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float send = b2 ? v[i] : v[i + 8], keep = b2 ? v[i + 8] : v[i];
    r8[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
  }
  float r4[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float send = b1 ? r8[i] : r8[i + 4], keep = b1 ? r8[i + 4] : r8[i];
    r4[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
  }
  const float s0 = b0 ? r4[0] : r4[2], k0 = b0 ? r4[2] : r4[0];
  const float s1 = b0 ? r4[1] : r4[3], k1 = b0 ? r4[3] : r4[1];
  o0 = k0 + __shfl_xor_sync(0xffffffffu, s0, 1);
  o1 = k1 + __shfl_xor_sync(0xffffffffu, s1, 1);
}

// Reduce-scatter of KPT column sums over the warp's four row groups (lane
// bits 3, 4): on return, lane holds the sums of columns
// rgl*(KPT/4) .. rgl*(KPT/4) + KPT/4 - 1 of its slice (rgl = lane / 8).
template <int KPT>
__device__ __forceinline__ void reduce_groups(const float (&v)[KPT], int lane, float (&out)[KPT / 4]) {
  const bool b4 = (lane >> 4) & 1, b3 = (lane >> 3) & 1;
  float r[KPT / 2];
#pragma unroll
  for (int i = 0; i < KPT / 2; ++i) {
    const float send = b4 ? v[i] : v[i + KPT / 2], keep = b4 ? v[i + KPT / 2] : v[i];
    r[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
  }
#pragma unroll
  for (int i = 0; i < KPT / 4; ++i) {
    const float send = b3 ? r[i] : r[i + KPT / 4], keep = b3 ? r[i + KPT / 4] : r[i];
    out[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
  }
}

}  // namespace

template <int H, int RKK, int BC>
__global__ void __launch_bounds__(2 * H, 1) lstm_fwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, NTH = 2 * H, KPT = H / 8, SKK = KPT - RKK, HS = KPT + 4;
  constexpr int NCOL = tm_cols<NTH, SKK>();
  static_assert(SKK % 4 == 0 && RKK % 4 == 0, "k split in float4 steps");
  extern __shared__ __align__(16) float sm[];
  __shared__ uint32_t tslot;
  float *hs = sm;                                // [2][BC][8 slices][HS]
  float *zr = hs + 2 * BC * 8 * HS;              // [BC][kRing][4H] Zx rows of upcoming steps
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(zr + BC * kRing * G);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x, lane = t & 31;
  const int ks = lane & 7, rg = (t >> 5) * 4 + (lane >> 3);
  const int u0 = 4 * rg, kb = ks * KPT;
  const int unit = u0 + (ks >> 1), pair = ks & 1;  // after the reduce-scatter
  const int q0 = 2 * pair;                         // this lane's gates q0, q0 + 1
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;
  const float *__restrict__ Whh = a.Whh[d];

  uint32_t tbase = 0, tw = 0;
  if constexpr (NCOL > 0) {
    tbase = tm_alloc<NCOL>(&tslot, t >> 5);
    tw = tbase + ((32u * ((t >> 5) & 3)) << 16) + (uint32_t)((t >> 7) * SKK * 16);
  }
  float w[16][RKK > 0 ? RKK : 1];
  load_tile<H, RKK, SKK>(Whh, u0, kb, tw, w);
  for (int i = t; i < 2 * BC * 8 * HS; i += NTH) hs[i] = 0.f;
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
  const int zo0 = q0 * H + unit, zo1 = zo0 + H;  // offsets of this lane's gates in a Z row
  const int hslot = (unit / KPT) * HS + unit % KPT;
  auto tok_at = [&](int b, int s) {
    const int tt = d == 0 ? s : len[b] - 1 - s;
    return toff[tt] + r0 + b;
  };
  float cst[BC];
  // token of step s of row b at a clamped (always valid) time; meaningful
  // only while s < len[b].  The prefetch reads it one step before its copy
  // needs it, so the copy's address waits on no load (a warp issues in order)
  auto tok_clamped = [&](int b, int s) {
    const int last = max(len[b] - 1, 0);
    const int tt = d == 0 ? min(s, last) : max(last - s, 0);
    return toff[tt] + r0 + b;
  };
  auto issue_at = [&](int b, int s, int tk) {  // the Zx row of step s of row b (token tk) into its ring slot
    if (s < len[b]) {
      const float *src = Z + (size_t)tk * G;
      float *slot = zr + ((size_t)b * kRing + s % kRing) * G;
      for (int i = t; i < G / 4; i += NTH) cp_async16(slot + 4 * i, src + 4 * i);
    }
  };
#pragma unroll
  for (int b = 0; b < BC; ++b) cst[b] = 0.f;
  for (int j = 0; j < kPF; ++j) {
#pragma unroll
    for (int b = 0; b < BC; ++b) issue_at(b, j, tok_clamped(b, j));
    cp_commit();
  }
  int tk_pf[BC];  // token of step s + kPF
#pragma unroll
  for (int b = 0; b < BC; ++b) tk_pf[b] = tok_clamped(b, kPF);
  cp_wait_pending<kPF - 1>();  // step 0's rows
  __syncthreads();
  for (int s = 0; s < Tg; ++s) {
    const int p = s & 1;
    cp_wait_pending<kPF - 2>();  // step s + 1's rows, published by this step's barrier
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s >= len[b]) continue;  // uniform over the CTA
      const float *slot = zr + ((size_t)b * kRing + s % kRing) * G;
      const float zc0 = slot[zo0], zc1 = slot[zo1];
      const int tc = tok_at(b, s);
      issue_at(b, s + kPF, tk_pf[b]);
      tk_pf[b] = tok_clamped(b, s + kPF + 1);
      const float *hv = hs + (p * BC + b) * 8 * HS + ks * HS;
      float acc[16];
#pragma unroll
      for (int ri = 0; ri < 16; ++ri) acc[ri] = 0.f;
      // register block j (columns 4j .. 4j + 3), then TMEM column RKK + j,
      // whose load was issued before block j
      constexpr int NR = RKK / 4, NJ = NR > SKK ? NR : SKK;
      uint32_t wt[16];
      if constexpr (SKK > 0) tm_ld16(tw, wt);
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        if (j < NR) {
          const float4 h4 = *reinterpret_cast<const float4 *>(hv + 4 * j);
#pragma unroll
          for (int ri = 0; ri < 16; ++ri) {
            float x = fmaf(w[ri][4 * j], h4.x, acc[ri]);
            x = fmaf(w[ri][4 * j + 1], h4.y, x);
            x = fmaf(w[ri][4 * j + 2], h4.z, x);
            acc[ri] = fmaf(w[ri][4 * j + 3], h4.w, x);
          }
        }
        if (j < SKK) {
          tm_wait16(wt);
          const float hk = hv[RKK + j];
#pragma unroll
          for (int ri = 0; ri < 16; ++ri) acc[ri] = fmaf(__uint_as_float(wt[ri]), hk, acc[ri]);
          if (j + 1 < SKK) tm_ld16(tw + 16 * (j + 1), wt);
        }
      }
      float v0, v1;
      reduce_scatter8(acc, lane, v0, v1);
      // lane pair 0 holds (i, f), pair 1 holds (g, o) of `unit`
      const float a0 = pair ? tanh_g(v0 + zc0) : sigm(v0 + zc0);
      const float a1 = sigm(v1 + zc1);
      Z[(size_t)tc * G + zo0] = a0;
      Z[(size_t)tc * G + zo1] = a1;
      const float x0 = __shfl_xor_sync(0xffffffffu, a0, 1), x1 = __shfl_xor_sync(0xffffffffu, a1, 1);
      const float ig = pair ? x0 : a0, fg = pair ? x1 : a1, gg = pair ? a0 : x0, og = pair ? a1 : x1;
      cst[b] = fmaf(fg, cst[b], ig * gg);
      const float h = og * tanh_g(cst[b]);
      if (pair == 0) {
        hs[((p ^ 1) * BC + b) * 8 * HS + hslot] = h;
      } else {
        Cs[(size_t)tc * H + unit] = cst[b];
        Y[(size_t)tc * DH + d * H + unit] = h;
      }
    }
    cp_commit();
    __syncthreads();
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  if constexpr (NCOL > 0) tm_free<NCOL>(tbase, t >> 5);
}

template <int H, int RKK, int BC>
__global__ void __launch_bounds__(2 * H, 1) lstm_bwd_cta_kernel(RecArgs a) {
  constexpr int G = 4 * H, NTH = 2 * H, KPT = H / 8, SKK = KPT - RKK, NW = NTH / 32;
  static_assert(SKK % 4 == 0 && RKK % 4 == 0 && KPT % 4 == 0, "k split in float4 steps");
  extern __shared__ __align__(16) float sm[];
  float4 *Ws4 = reinterpret_cast<float4 *>(sm);  // [SKK/4][16][NTH]
  float *dzs = sm + SKK * 16 * NTH;              // [BC][H][4] unit-major dz
  float *red = dzs + BC * G;                     // [BC][NW][H] per-warp column partials
  float *ring = red + BC * NW * H;               // [BC][kRing][7H] input rows of upcoming steps
  const int T = a.ix.T;
  const bool toff_sm = T + 1 <= kTokCap;
  int *toff_s = reinterpret_cast<int *>(ring + BC * kRing * 7 * H);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int ks = lane & 7, rgl = lane >> 3, rg = warp * 4 + rgl;
  const int u0 = 4 * rg, kb = ks * KPT;
  const int unit = t >> 1, pair = t & 1;  // phase B: lanes 2j, 2j+1 serve unit j
  const int n_groups = (a.ix.b + BC - 1) / BC;
  const int d = blockIdx.x / n_groups, grp = blockIdx.x % n_groups;
  const int r0 = grp * BC;
  const int DH = a.dirs * H;
  const float *__restrict__ Whh = a.Whh[d];

  float w[16][RKK > 0 ? RKK : 1];
#pragma unroll
  for (int ri = 0; ri < 16; ++ri) {
    const float *row = Whh + (size_t)((ri & 3) * H + u0 + (ri >> 2)) * H + kb;
#pragma unroll
    for (int kk = 0; kk < RKK; ++kk) w[ri][kk] = __ldg(row + kk);
#pragma unroll
    for (int k4 = 0; k4 < SKK / 4; ++k4) {
      const float *p = row + RKK + 4 * k4;
      Ws4[(k4 * 16 + ri) * NTH + t] = make_float4(__ldg(p), __ldg(p + 1), __ldg(p + 2), __ldg(p + 3));
    }
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
  // phase B inputs of step s, kPF steps ahead: the gate row [4H], c_t [H],
  // c_{t-1} [H] (zeros at the start) and dY [H] of the row, in 16-byte pieces
  float dc[BC];
  // token of step s of row b at a clamped (always valid) time; meaningful
  // only while 0 <= s < len[b].  The prefetch reads the tokens of its step
  // one step before its copies need them, so no copy address waits on a load
  auto tok_clamped = [&](int b, int s) {
    const int last = max(len[b] - 1, 0);
    const int tt = d == 0 ? min(max(s, 0), last) : max(last - max(s, 0), 0);
    return toff[tt] + r0 + b;
  };
  auto issue = [&](int b, int s, int tk, int tp) {  // tp: token of step s - 1 (used when s > 0)
    if (s >= 0 && s < len[b]) {
      if (s == 0) tp = -1;
      float *slot = ring + ((size_t)b * kRing + s % kRing) * 7 * H;
      for (int i = t; i < 7 * H / 4; i += NTH) {
        const int q = 4 * i;  // float offset in the slot
        if (q < 4 * H) cp_async16(slot + q, Z + (size_t)tk * G + q);
        else if (q < 5 * H) cp_async16(slot + q, Cs + (size_t)tk * H + (q - 4 * H));
        else if (q < 6 * H) {
          if (tp >= 0) cp_async16(slot + q, Cs + (size_t)tp * H + (q - 5 * H));
          else *reinterpret_cast<float4 *>(slot + q) = make_float4(0.f, 0.f, 0.f, 0.f);
        } else cp_async16(slot + q, dY + (size_t)tk * DH + d * H + (q - 6 * H));
      }
    }
  };
#pragma unroll
  for (int b = 0; b < BC; ++b) dc[b] = 0.f;
  for (int j = 0; j < kPF; ++j) {
#pragma unroll
    for (int b = 0; b < BC; ++b) issue(b, Tg - 1 - j, tok_clamped(b, Tg - 1 - j), tok_clamped(b, Tg - 2 - j));
    cp_commit();
  }
  int tk_pf[BC], tp_pf[BC];  // tokens of steps s - kPF and s - kPF - 1
#pragma unroll
  for (int b = 0; b < BC; ++b) {
    tk_pf[b] = tok_clamped(b, Tg - 1 - kPF);
    tp_pf[b] = tok_clamped(b, Tg - 2 - kPF);
  }
  cp_wait_pending<kPF - 1>();  // the first step's rows
  __syncthreads();
  for (int s = Tg - 1; s >= 0; --s) {
    cp_wait_pending<kPF - 2>();  // step s - 1's rows, published by this step's barriers
    // phase B: dz of unit j from dh = dY + recurrent part
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s >= len[b]) continue;  // uniform over the CTA
      float dh_rec = 0.f;
      if (s + 1 < len[b]) {
        const float *rp = red + (size_t)b * NW * H + unit;
#pragma unroll
        for (int wi = 0; wi < NW; ++wi) dh_rec += rp[wi * H];
      }
      const float *slot = ring + ((size_t)b * kRing + s % kRing) * 7 * H;
      const float ig = slot[unit], fg = slot[H + unit], gg = slot[2 * H + unit], og = slot[3 * H + unit];
      const float ct = slot[4 * H + unit], cp = slot[5 * H + unit];
      const float dh = slot[6 * H + unit] + dh_rec;
      const int tk = tok_at(b, s);
      const float tch = tanh_g(ct);
      const float dcv = fmaf(dh * og, 1.f - tch * tch, dc[b]);
      const float dzi = dcv * gg * ig * (1.f - ig);
      const float dzf = dcv * cp * fg * (1.f - fg);
      const float dzg = dcv * ig * (1.f - gg * gg);
      const float dzo = dh * tch * og * (1.f - og);
      dc[b] = dcv * fg;
      const float z0 = pair ? dzg : dzi, z1 = pair ? dzo : dzf;
      *reinterpret_cast<float2 *>(dzs + ((size_t)b * H + unit) * 4 + 2 * pair) = make_float2(z0, z1);
      Z[(size_t)tk * G + (2 * pair) * H + unit] = z0;
      Z[(size_t)tk * G + (2 * pair + 1) * H + unit] = z1;
    }
    // the prefetch of step s - kPF, for every row active or not: steps run
    // backwards, so a shorter row becomes active only later and needs its
    // first kPF steps in flight by then
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      issue(b, s - kPF, tk_pf[b], tp_pf[b]);
      tk_pf[b] = tp_pf[b];  // the next step's token is this one's predecessor
      tp_pf[b] = tok_clamped(b, s - kPF - 2);
    }
    cp_commit();
    __syncthreads();
    // phase A: column partials of W_hh^T dz over this warp's 16 x 4 rows
#pragma unroll
    for (int b = 0; b < BC; ++b) {
      if (s >= len[b]) continue;
      const float4 *dz4 = reinterpret_cast<const float4 *>(dzs + ((size_t)b * H + u0) * 4);
      float dz[16];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 v = dz4[u];
        dz[4 * u] = v.x;
        dz[4 * u + 1] = v.y;
        dz[4 * u + 2] = v.z;
        dz[4 * u + 3] = v.w;
      }
      float part[KPT];
#pragma unroll
      for (int kk = 0; kk < RKK; ++kk) {
        float x = 0.f;
#pragma unroll
        for (int ri = 0; ri < 16; ++ri) x = fmaf(w[ri][kk], dz[ri], x);
        part[kk] = x;
      }
#pragma unroll
      for (int k4 = 0; k4 < SKK / 4; ++k4) {
        float x0 = 0.f, x1 = 0.f, x2 = 0.f, x3 = 0.f;
#pragma unroll
        for (int ri = 0; ri < 16; ++ri) {
          const float4 wv = Ws4[(k4 * 16 + ri) * NTH + t];
          x0 = fmaf(wv.x, dz[ri], x0);
          x1 = fmaf(wv.y, dz[ri], x1);
          x2 = fmaf(wv.z, dz[ri], x2);
          x3 = fmaf(wv.w, dz[ri], x3);
        }
        part[RKK + 4 * k4] = x0;
        part[RKK + 4 * k4 + 1] = x1;
        part[RKK + 4 * k4 + 2] = x2;
        part[RKK + 4 * k4 + 3] = x3;
      }
      float out[KPT / 4];
      reduce_groups<KPT>(part, lane, out);
      // lane (rgl, ks) now holds columns kb + rgl*(KPT/4) .. + KPT/4 - 1
      float *dst = red + ((size_t)b * NW + warp) * H + kb + rgl * (KPT / 4);
#pragma unroll
      for (int i = 0; i < KPT / 4; ++i) dst[i] = out[i];
    }
    __syncthreads();
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// ---------------------------------------------------------------------------
namespace {

size_t cta_smem_bytes(bool bwd, int H, int RKK, int BC, int T) {
  const int KPT = H / 8, SKK = KPT - RKK, NTH = 2 * H;
  const size_t wf = (size_t)SKK * 16 * NTH;  // BPTT's shared-memory weights (the forward's are in TMEM)
  const size_t f = bwd ? wf + (size_t)BC * 4 * H + (size_t)BC * (NTH / 32) * H + (size_t)BC * kRing * 7 * H
                       : (size_t)2 * BC * 8 * (KPT + 4) + (size_t)BC * kRing * 4 * H;
  const size_t i = (T + 1 <= kTokCap) ? (size_t)(T + 1) : 0;
  return (f + i) * 4 + 16;
}

template <int H, int RKK, int BC>
cudaError_t launch_cta(const RecArgs &a, bool bwd, cudaStream_t s) {
  const size_t smem = cta_smem_bytes(bwd, H, RKK, BC, a.ix.T);
  const int ng = (a.ix.b + BC - 1) / BC;
  if (bwd) {
    cudaError_t e = ensure_smem((const void *)lstm_bwd_cta_kernel<H, RKK, BC>, smem);
    if (e != cudaSuccess) return e;
    lstm_bwd_cta_kernel<H, RKK, BC><<<ng * a.dirs, 2 * H, smem, s>>>(a);
  } else {
    cudaError_t e = ensure_smem((const void *)lstm_fwd_cta_kernel<H, RKK, BC>, smem);
    if (e != cudaSuccess) return e;
    lstm_fwd_cta_kernel<H, RKK, BC><<<ng * a.dirs, 2 * H, smem, s>>>(a);
  }
  return cudaGetLastError();
}

// Columns of the k slice held in registers (RKK of KPT = H/8) for one and two
// batch rows per CTA.
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
    case 32: return launch_cta_bc<32, 4, 4>(a, bc, bwd, s);
    case 64: return launch_cta_bc<64, 8, 4>(a, bc, bwd, s);
    case 128: return launch_cta_bc<128, 12, 8>(a, bc, bwd, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bkt
