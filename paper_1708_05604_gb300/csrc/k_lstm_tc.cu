// k_lstm_tc.cu -- the recurrence of the bf16 configuration at H = 256 on the
// 5th-generation tensor cores (a6 forward, a11 BPTT).
//
// One step of the recurrence is a small dense contraction per batch row:
// forward z_t = Zx_t + W_hh h_{t-1} ([4H x H] by [H]), BPTT
// dh_{t-1} = W_hh^T dz_t.  A thread-block cluster of 8 CTAs owns one
// direction and N = 16 or 32 consecutive rows of the length-sorted batch;
// CTA c owns the hidden units [32c, 32c + 32), i.e. the 128 gate rows
// {q H + 32c + u : q = i, f, g, o; u < 32}, and keeps its slice of W_hh for
// the whole sequence in tensor memory as the A operand of tcgen05.mma, split
// into two parts, with fp32 accumulation in TMEM; the cell state, h, the
// gates and every elementwise step stay fp32.  Forward: w = w_hi + 2^-11 w_lo
// in fp16 (about 22 significant bits) times h_{t-1} rounded to fp16
// (relative error 2^-12 in each h, within the bf16 input projection's 2^-9),
// two products per step.  BPTT: w = w_hi + w_lo in bf16 (16 bits) and dz_t
// split the same way (bf16 keeps the range that small gradients need), the
// three products hi*hi + hi*lo + lo*hi (relative error near 2^-16).  W never
// leaves the SM: per step only N rows of h (or dz) are read from shared
// memory.
//
// A team is 16 rows of the batch with its own MMAs, TMEM accumulators,
// exchange buffers, mbarriers and named barrier.  A one-team cluster runs its
// team on all 16 warps; a two-team cluster runs two teams of 8 warps that
// share only W in TMEM (one team's MMAs and exchange wait overlap the other's
// elementwise work).  A launch gives the longest rows to one-team clusters,
// which step faster, and the rest to two-team clusters, within the clusters
// that fit on the GPU at once (see the launch code at the end).
//
// Forward: TMEM lane 32 q + u holds gate row q H + 32c + u (A = the W slice,
// K = the 256 units; hi part in columns 0 .. 127, scaled lo part in
// 128 .. 255).
// BPTT: A = the W slice transposed in two 128-unit halves (lane m = unit
// 128 hf + m), K = the CTA's 128 gate rows in the order 4u + q.  Operands in
// shared memory use the K-major layout without swizzle: 8 x 16-byte core
// matrices, element (n, k) at (k / 8) * 16 N + n * 16 + (k % 8) * 2 bytes, so
// the 32 units of one CTA are one contiguous 64 N-byte block.
//
// Forward step: once h_{t-1} has arrived, four issuing threads (product x
// half of K) issue 8 MMAs each into their own accumulators and commit them
// to an mbarrier; each warp then reads one TMEM lane quarter (one gate for
// the 32 units) for C rows, adds Zx and the four accumulators (the lo ones
// scaled by 2^-11), applies sigma or tanh and leaves the gates in shared
// memory, where thread (w, lane) finds the four gates of unit `lane` for
// its rows, updates c in registers, stages c and h, and stages h_t in fp16
// for st.async stores to every CTA of the cluster (16-byte remote stores
// completing bytes on the receiver's mbarrier; double-buffered by step
// parity, so the data dependence orders buffer reuse).  The warps that
// issue no MMAs write the staged outputs to global memory and bring in Zx
// during the next step's exchange wait and MMAs.
// BPTT step: dh = dY + the sum of the 8 partials of W_hh^T dz_{t+1} received
// for this CTA's units, then dc and dz of the four gates (bf16, and fp32 in
// place of the gates for layer 1, and split to the B operand); four issuing
// threads (six with one team) form this CTA's partial W_hh^T dz over its 128
// gate rows for all 256 units (two 128-lane halves), and each warp sends
// its 16-byte pieces of the 32-unit blocks straight to the CTAs that own
// them.  Above layer 1 the bias gradient is summed in the kernel.
//
// Every wait is bounded (status bit 4 on expiry, as in the other cluster
// kernels); on an abort the kernel still waits for its last MMA batch before
// it frees TMEM, sleeps 20 us so peers' in-flight stores land, and meets its
// peers at a final cluster barrier.  A CTA takes all 512 TMEM columns; its
// shared-memory request (>= 140 KB) keeps any other TMEM user off its SM.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>

#include <algorithm>

#include "bkt_internal.h"

namespace bkt {

namespace {

constexpr int kTH = 256;           // hidden units
constexpr int kTCS = 8;            // CTAs per cluster
constexpr int kTHc = kTH / kTCS;   // units per CTA
constexpr int kTTokCap = 8192;     // time offsets staged in shared memory up to this T
constexpr int kTPolls = 1 << 22;
// One CTA per SM, and no bf16 GEMM CTA (97 KB at its smallest) beside it:
// each CTA holds all of TMEM for the whole sequence.
constexpr size_t kTSmemFloor = 140 * 1024;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCol = 256;  // first accumulator column (A operands take 0 .. 255)

// kind::f16 instruction descriptor: D fp32, A and B bf16 (format 1 at bits
// 7 and 10) or fp16 (format 0), both K-major, N >> 3 at bit 17, M = 128
// (>> 4 at bit 24).
template <int N, bool F16 = false>
__host__ __device__ constexpr uint32_t tc_idesc() {
  return (1u << 4) | (F16 ? 0u : (1u << 7) | (1u << 10)) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

__device__ __forceinline__ uint32_t sa(const void *p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }
__device__ __forceinline__ uint32_t peer(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void mb_init(uint32_t mb, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(mb), "r"(count) : "memory");
}
__device__ __forceinline__ void mb_arm(uint32_t mb, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mb_arrive(uint32_t mb) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(mb) : "memory");
}
__device__ __forceinline__ bool mb_wait(uint32_t mb, uint32_t parity, int cap) {
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
__device__ __forceinline__ void st_async16(uint32_t raddr, uint4 v, uint32_t rmbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(raddr),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(rmbar)
               : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
// Shared-memory descriptor of a K-major operand without swizzle: core
// matrices of 8 rows x 16 bytes, `lbo` bytes apart along K, `sbo` along N.
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version
  return d;                // swizzle mode 0: none
}
// The same for a K-major operand in the 128-byte swizzle: rows of 128 B
// (64 bf16 of K) whose 16-byte chunks are permuted by chunk ^ (row % 8),
// 8-row groups 1024 B apart (the tile 1024-byte aligned).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
  uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;            // leading byte offset (unused in this mode)
  d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset
  d |= (uint64_t)1 << 46;            // descriptor version
  d |= (uint64_t)2 << 61;            // 128-byte swizzle
  return d;
}
// D (TMEM) (+)= A (TMEM) * B (shared memory)
__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d),
      "r"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar) : "memory");
}
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&v)[8]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr), "r"(v[0]),
               "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
               : "memory");
}
// C = N / 4 consecutive columns of this thread's lane, added into x (C = 4 or 8).
template <int C>
__device__ __forceinline__ void tmem_ld_add(uint32_t taddr, float (&x)[C]) {
  uint32_t r[C];
  if constexpr (C == 4) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(taddr)
                 : "memory");
  } else {
    static_assert(C == 8, "4 or 8 columns per thread");
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr)
                 : "memory");
  }
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < C; ++j) x[j] += __uint_as_float(r[j]);
}

// x = hi + lo, both bf16 (hi rounded to nearest, lo the rounded rest).
__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16 &hi, __nv_bfloat16 &lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}
__device__ __forceinline__ uint32_t pack2(__nv_bfloat16 a, __nv_bfloat16 b) {
  return (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16);
}
__device__ __forceinline__ uint32_t bf2u(__nv_bfloat162 v) { return pack2(v.x, v.y); }
// x = hi + 2^-11 lo, both fp16: hi rounded to nearest, lo the rounded rest
// scaled by 2^11 so that it keeps fp16's full precision (the rest alone is
// often subnormal); hi + 2^-11 lo carries about 22 significant bits
constexpr float kF16LoScale = 2048.f;
__device__ __forceinline__ void split_f16(float x, __half &hi, __half &lo) {
  hi = __float2half_rn(x);
  lo = __float2half_rn((x - __half2float(hi)) * kF16LoScale);
}
__device__ __forceinline__ uint32_t pack2h(__half a, __half b) {
  return (uint32_t)__half_as_ushort(a) | ((uint32_t)__half_as_ushort(b) << 16);
}
__device__ __forceinline__ uint32_t pack2bf(float a, float b) {
  return pack2(__float2bfloat16_rn(a), __float2bfloat16_rn(b));
}
// 16-byte asynchronous copy global -> shared; `bytes` = 0 fills zeros.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int K>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(K) : "memory");
}
// C consecutive columns of this thread's lane, not yet waited for
template <int C>
__device__ __forceinline__ void tmem_ld_raw(uint32_t taddr, uint32_t (&r)[C]) {
  if constexpr (C == 4) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(taddr)
                 : "memory");
  } else {
    static_assert(C == 8, "4 or 8 columns per thread");
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr)
                 : "memory");
  }
}
// Gate nonlinearities from the exponential intrinsic (as in the other
// recurrent kernels): sigma(x) = 1 / (1 + e^-x), tanh(x) = 1 - 2 / (1 + e^2x).
__device__ __forceinline__ float tanh_tc(float x) { return 1.f - __fdividef(2.f, 1.f + __expf(2.f * x)); }
// Four values of one nonlinearity with one reciprocal: with d_k = 1 + e^{a_k}
// (a_k = -x for sigma, 2x for tanh, clamped at 20 so that the product of the
// four stays finite), 1 / d_k = (prod_{j != k} d_j) / (prod_j d_j).  The
// clamp changes sigma(x) only for x < -20 and tanh(x) only for x > 10, by
// less than 5e-9.
template <bool TANH>
__device__ __forceinline__ void act4(float (&x)[4]) {
  float dd[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) dd[k] = 1.f + __expf(fminf(TANH ? 2.f * x[k] : -x[k], 20.f));
  const float d01 = dd[0] * dd[1], d23 = dd[2] * dd[3];
  const float r = __fdividef(1.f, d01 * d23);
  const float r23 = r * d23, r01 = r * d01;
  const float inv[4] = {dd[1] * r23, dd[0] * r23, dd[3] * r01, dd[2] * r01};
#pragma unroll
  for (int k = 0; k < 4; ++k) x[k] = TANH ? 1.f - 2.f * inv[k] : inv[k];
}

// Named barrier of one team (id >= 1; id 0 is __syncthreads) of n threads,
// and the same barrier returning the OR of a predicate over them.
__device__ __forceinline__ void team_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ bool team_sync_or(int id, int n, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred a, b;\n\tsetp.ne.u32 a, %1, 0;\n\tbar.red.or.pred b, %2, %3, a;\n\tselp.u32 %0, 1, 0, b;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)p), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// Shared-memory layout (bytes): one region of kTeam bytes per team, then the
// TMEM address slot, the lengths of the cluster's rows and the time offsets.
template <int N>
struct TcBwdLayout {
  static constexpr uint32_t kB = N * 128 * 2;      // one B operand (dz hi or lo): N rows x 128 gate rows, 128-byte swizzle
  static constexpr int kRS = kTHc + 8;             // floats per (source, row) of received partials (32 units + pad)
  static constexpr uint32_t kRed = kTCS * N * kRS * 4;     // received partials per parity
  static constexpr uint32_t kStepBytes = kTCS * kTHc * N * 4;
  static constexpr uint32_t oB = 0;                // [2 hi/lo][kB]
  static constexpr uint32_t oRed = oB + 2 * kB;    // [2 parity][8 src][N rows][kRS] fp32
  static constexpr uint32_t oStg = oRed + 2 * kRed;  // [8 owners][N rows][32 units] fp32 partials to send
  static constexpr uint32_t oBar = oStg + kTCS * N * kTHc * 4;  // rbar[2], mmabar
  static constexpr uint32_t kTeam = (oBar + 32 + 1023) & ~1023u;  // keeps each team's B operand 1024-byte aligned
};

template <int N>
struct TcFwdLayout {
  static constexpr uint32_t kB = N * kTH * 2;          // h_{t-1} in fp16: N rows x 256 units
  static constexpr uint32_t kSlice = 64 * N;           // one CTA's 32 units of it
  static constexpr uint32_t kStepBytes = kTCS * kSlice;
  static constexpr uint32_t oB = 0;                    // [2 parity][kB]
  // staging of h_t: [2 parity][4 unit octets][N rows][16 B], the octets
  // 16 N + 16 bytes apart so that a warp's stores of one row (four octets)
  // fall in distinct banks
  static constexpr uint32_t kOct = 16 * N + 16;
  static constexpr uint32_t kStgS = 4 * kOct;
  static constexpr uint32_t oStg = oB + 2 * kB;
  static constexpr uint32_t kRowF = 4 * kTHc;                    // floats of one row: [4 gates][32 units]
  static constexpr uint32_t oGate = oStg + 2 * kStgS;            // [2 parity][N][4][32] fp32 activated gates
  static constexpr uint32_t oCell = oGate + 2 * N * kRowF * 4;   // [2 parity][c, h][N][32] fp32
  static constexpr uint32_t oZx = oCell + 2 * 2 * N * kTHc * 4;  // [3 stages][N][4][32] fp32 Zx
  static constexpr uint32_t oBar = oZx + 3 * N * kRowF * 4;      // xbar[2], mmabar
  static constexpr uint32_t kTeam = oBar + 32;
  static_assert(oGate % 16 == 0 && oCell % 16 == 0 && oZx % 16 == 0, "16-byte staging rows");
};

template <typename L, int N, int TM>
struct TcSmem {
  static constexpr uint32_t oSlot = TM * L::kTeam;
  static constexpr uint32_t oLen = oSlot + 16;
  static constexpr uint32_t oToff = oLen + 4 * N * TM;
  static_assert(L::kTeam % 16 == 0, "team regions keep 16-byte operand alignment");
};

// Dynamic shared memory of a launch: the larger of the one- and two-team
// layouts (BPTT: + 1 KB to align its base to 1024 bytes), then the time
// offsets when they fit under the per-block limit (else they are read from
// global memory; only the warps that move data read them).
constexpr uint32_t kSmemMax = 232448;
__host__ __device__ constexpr uint32_t umax(uint32_t x, uint32_t y) { return x > y ? x : y; }
template <int N>
__host__ __device__ constexpr uint32_t tc_base(bool bwd) {
  return bwd ? umax(TcSmem<TcBwdLayout<N>, N, 1>::oToff, TcSmem<TcBwdLayout<N>, N, 2>::oToff) + 1024
             : umax(TcSmem<TcFwdLayout<N>, N, 1>::oToff, TcSmem<TcFwdLayout<N>, N, 2>::oToff);
}
template <int N>
__host__ __device__ constexpr int tc_tok_cap(bool bwd) {
  return (int)((kSmemMax - tc_base<N>(bwd)) / 4) < kTTokCap ? (int)((kSmemMax - tc_base<N>(bwd)) / 4) : kTTokCap;
}

template <int N>
size_t tc_smem_bytes(bool bwd, int T) {
  const size_t need = tc_base<N>(bwd) + (T + 1 <= tc_tok_cap<N>(bwd) ? (size_t)(T + 1) * 4 : 0);
  return std::max(need, kTSmemFloor);
}

}  // namespace

// Teams.  A CTA's 16 warps form TM teams of TW = 16 / TM warps; team k owns
// N consecutive rows of the cluster's R = TM N and runs its own recurrence
// over them: its own MMAs and accumulators, exchange buffers, mbarriers and
// a named barrier, so that with two teams one team's MMAs and exchange wait
// overlap the other team's elementwise work (they share W in TMEM only).
// Thread roles inside a team: warp w of TW reads TMEM lane quarter w % 4
// and columns C (w / 4) .. + C - 1 (C = 4 N / TW) of each accumulator, lane
// l of it TMEM lane 32 (w % 4) + l; the elementwise phases give thread (w, l)
// unit l of the CTA's 32 and rows P w .. P w + P - 1 (P = N / TW).
// Forward kernel.  TMEM lane m = 32 q + u holds gate q of unit u, so warp
// quarter q holds one gate for 32 consecutive units (coalesced Zx loads and
// gate stores, a warp-uniform nonlinearity); the four gates of a (unit, row)
// meet through shared memory, then thread (w, lane) updates the cell of unit
// `lane` for its P rows.  (A lane order 4u + q, with the gates swapped by
// shuffles inside groups of four lanes, measured 10 % slower per step.)
// The body of one cluster: direction d, rows rc .. rc + TM N - 1.
//
// A step's chain (exchange, MMAs, gates, cell update, exchange) touches
// only shared memory and TMEM.  The step's outputs go to a staging area
// (gates and c, h in fp32, double-buffered by step parity), and during the
// next step's exchange wait and MMAs the team's warps that issue no MMAs
// (warps 4 .. TW - 1) write them to global memory as 16-byte pieces and
// bring Zx of two steps ahead into a three-stage ring with asynchronous
// copies.  (A step's stores, ~14 KB per CTA, take ~450 cycles at the SM's
// ~32 bytes per clock to L2, measured; inside the gate and cell phases, or
// issued by every warp after the send, they lengthened the step.)
template <int N, int TM>
__device__ __forceinline__ void fwd_tc_body(const RecArgs &a, uint8_t *smem, const int d, const int rc) {
  using Lay = TcFwdLayout<N>;
  using Sm = TcSmem<Lay, N, TM>;
  constexpr int H = kTH, G = 4 * H, kTThreads = 512, TW = 16 / TM, TT = 32 * TW, QW = TW / 4, C = N / QW,
                P = N / TW, R = N * TM, RF = Lay::kRowF, NWK = TT - 128;
  static_assert(C == 4 || C == 8, "4 or 8 accumulator columns per thread");
  static_assert(P * TW == N, "whole rows per warp");
  static_assert(NWK > 0, "warps 4 .. TW - 1 of a team move the step's data");
  constexpr uint32_t idesc = tc_idesc<N, true>();
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int tm = warp / TW, wt = warp % TW, tt = t % TT;  // team; warp and thread within it
  uint8_t *team = smem + tm * Lay::kTeam;
  uint8_t *Bb = team + Lay::oB;
  uint8_t *stg = team + Lay::oStg;
  float *gate = reinterpret_cast<float *>(team + Lay::oGate);
  float *cell = reinterpret_cast<float *>(team + Lay::oCell);
  float *zx = reinterpret_cast<float *>(team + Lay::oZx);
  uint64_t *bar = reinterpret_cast<uint64_t *>(team + Lay::oBar);
  uint32_t *tslot = reinterpret_cast<uint32_t *>(smem + Sm::oSlot);
  int *rlen_c = reinterpret_cast<int *>(smem + Sm::oLen);
  const int *rlen = rlen_c + tm * N;
  int *toff_s = reinterpret_cast<int *>(smem + Sm::oToff);

  const int q = wt & 3, cs = wt >> 2;  // TMEM lane quarter = gate; column slice
  const int col0 = C * cs;
  const uint32_t c = cluster_rank();
  const int gu = (int)c * kTHc + lane;      // the unit of this lane (both phases)
  const int r0 = rc + tm * N;
  const int DH = a.dirs * H, T = a.ix.T;
  const bool toff_sm = T + 1 <= tc_tok_cap<N>(false);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int cap = a.wf.poll_cap > 0 ? a.wf.poll_cap : kTPolls;
  const bool withhold = (a.wf.withhold & kWithholdExchange) && c == 0;
  const int bid = 1 + tm;
  float *__restrict__ Z = a.Z[d];
  float *__restrict__ Cs = a.Cst[d];
  float *__restrict__ Y = a.Y;
  __nv_bfloat16 *__restrict__ Yb = reinterpret_cast<__nv_bfloat16 *>(a.Yb);
  __nv_bfloat16 *__restrict__ Hs = reinterpret_cast<__nv_bfloat16 *>(a.Hs[d]);
  // token of row n (of the team) at step s of its direction
  auto tok_of = [&](int n, int L, int s) { return (size_t)(toff[d == 0 ? s : L - 1 - s] + r0 + n); };
  // Zx of step sl into ring stage sl % 3 (zeros for rows that have ended),
  // pieces w0, w0 + nw, ... of the team's 32 N 16-byte pieces
  auto load_zx = [&](int sl, int w0, int nw) {
    const uint32_t zs = sa(zx + (sl % 3) * N * RF);
    for (int i = w0; i < N * 32; i += nw) {
      const int n = i >> 5, qq = (i >> 3) & 3, ch = i & 7, L = rlen[n];
      const bool act = sl < L;
      const float *src = Z + (act ? tok_of(n, L, sl) * G : 0) + qq * H + c * kTHc + 4 * ch;
      cp_async16(zs + (uint32_t)((n * 4 + qq) * kTHc + 4 * ch) * 4u, src, act ? 16u : 0u);
    }
  };
  // the staged outputs of step sp: gates in place of Zx; c, h; the bf16 h
  // as Y's copy and as h_{t-1} of the row's next token
  auto store_step = [&](int sp, int w0, int nw) {
    const float *gs = gate + (sp & 1) * N * RF;
    const float *cl = cell + (sp & 1) * 2 * N * kTHc;
    for (int i = w0; i < N * 32; i += nw) {
      const int n = i >> 5, qq = (i >> 3) & 3, ch = i & 7, L = rlen[n];
      if (sp < L)
        *reinterpret_cast<float4 *>(Z + tok_of(n, L, sp) * G + qq * H + c * kTHc + 4 * ch) =
            *reinterpret_cast<const float4 *>(gs + (n * 4 + qq) * kTHc + 4 * ch);
    }
    for (int i = w0; i < N * 8; i += nw) {
      const int n = i >> 3, ch = i & 7, L = rlen[n];
      if (sp < L) {
        const size_t tk = tok_of(n, L, sp);
        *reinterpret_cast<float4 *>(Cs + tk * H + c * kTHc + 4 * ch) =
            *reinterpret_cast<const float4 *>(cl + n * kTHc + 4 * ch);
        if (Y)
          *reinterpret_cast<float4 *>(Y + tk * DH + d * H + c * kTHc + 4 * ch) =
              *reinterpret_cast<const float4 *>(cl + (N + n) * kTHc + 4 * ch);
      }
    }
    if (Yb || Hs) {
      for (int i = w0; i < N * 4; i += nw) {
        const int n = i >> 2, ch = i & 3, L = rlen[n];
        if (sp < L) {
          const float4 h0 = *reinterpret_cast<const float4 *>(cl + (N + n) * kTHc + 8 * ch);
          const float4 h1 = *reinterpret_cast<const float4 *>(cl + (N + n) * kTHc + 8 * ch + 4);
          const uint4 v = make_uint4(pack2bf(h0.x, h0.y), pack2bf(h0.z, h0.w), pack2bf(h1.x, h1.y), pack2bf(h1.z, h1.w));
          if (Yb) *reinterpret_cast<uint4 *>(Yb + tok_of(n, L, sp) * DH + d * H + c * kTHc + 8 * ch) = v;
          if (Hs && sp + 1 < L) *reinterpret_cast<uint4 *>(Hs + tok_of(n, L, sp + 1) * H + c * kTHc + 8 * ch) = v;
        }
      }
    }
  };

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(tslot)), "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
#pragma unroll
  for (int k = 0; k < TM; ++k)
    for (uint32_t i = t; i < 2 * Lay::kB / 16; i += kTThreads)
      reinterpret_cast<uint4 *>(smem + k * Lay::kTeam + Lay::oB)[i] = make_uint4(0, 0, 0, 0);
  if (toff_sm)
    for (int i = t; i <= T; i += kTThreads) toff_s[i] = a.ix.tok_off[i];
  if (t < R) rlen_c[t] = rc + t < a.ix.b ? a.ix.row_len[rc + t] : 0;
  if (t == 0) {
#pragma unroll
    for (int k = 0; k < TM; ++k) {
      uint64_t *b = reinterpret_cast<uint64_t *>(smem + k * Lay::kTeam + Lay::oBar);
      mb_init(sa(&b[0]), 1);
      mb_init(sa(&b[1]), 1);
      mb_init(sa(&b[2]), 4);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  fence_proxy();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t tl = tmem + ((uint32_t)(32 * q) << 16);
  // Zx of the first two steps; the rows' first h_{t-1} (zero)
  load_zx(0, tt, TT);
  load_zx(1, tt, TT);
  cp_commit();
  if (Hs)
    for (int i = tt; i < N * 4; i += TT) {
      const int n = i >> 2, ch = i & 3, L = rlen[n];
      if (L > 0) *reinterpret_cast<uint4 *>(Hs + tok_of(n, L, 0) * H + c * kTHc + 8 * ch) = make_uint4(0, 0, 0, 0);
    }
  // W_hh slice into TMEM (warps 0 .. 3, warp q = lane quarter q): lane
  // 32 q + u holds row q H + 32c + u
  if (warp < 4) {
    const float *wrow = a.Whh[d] + (size_t)(q * H + gu) * H;
#pragma unroll 1
    for (int c0 = 0; c0 < 128; c0 += 8) {
      uint32_t hi[8], lo[8];
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(wrow + 2 * (c0 + j)));
        __half h0, l0, h1, l1, h2, l2, h3, l3;
        split_f16(v.x, h0, l0);
        split_f16(v.y, h1, l1);
        split_f16(v.z, h2, l2);
        split_f16(v.w, h3, l3);
        hi[j] = pack2h(h0, h1);
        lo[j] = pack2h(l0, l1);
        hi[j + 1] = pack2h(h2, h3);
        lo[j + 1] = pack2h(l2, l3);
      }
      tmem_st8(tl + c0, hi);
      tmem_st8(tl + 128 + c0, lo);
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  }
  cp_wait<0>();
  fence_before();
  __syncthreads();
  const int Tg = rlen[0];
  cluster_sync_all();
  if (tt == 0) {
    if (Tg >= 2) mb_arm(sa(&bar[0]), Lay::kStepBytes);
    if (Tg >= 3) mb_arm(sa(&bar[1]), Lay::kStepBytes);
  }

  int lenp[P];  // lengths of this thread's cell rows
#pragma unroll
  for (int j = 0; j < P; ++j) lenp[j] = rlen[P * wt + j];
  float cst[P];
#pragma unroll
  for (int j = 0; j < P; ++j) cst[j] = 0.f;
  // MMA issuers: lane 0 of the team's warps 0 .. 3; issuer i forms W_hi h
  // (i < 2) or W_lo h (i >= 2) over k-steps 8 (i % 2) .. + 7 into its own
  // accumulator
  const int prod = (lane == 0 && wt < 4) ? wt : -1;
  const uint32_t acc0 = kAccCol + 32u * (uint32_t)(4 * tm);  // the team's four accumulators
  bool ok = true, stop = false;
  int mma_issued = 0, mma_seen = 0;

  for (int s = 0; s < Tg && !stop; ++s) {
    const int e = s - 1;
    if (s > 0 && prod >= 0) {
      ok = mb_wait(sa(&bar[e & 1]), (e >> 1) & 1, cap) && ok;
      if (tt == 0 && ok && e + 2 <= Tg - 2) mb_arm(sa(&bar[e & 1]), Lay::kStepBytes);
      if (ok) {
        fence_proxy();
        fence_after();
        const uint32_t bsel = sa(Bb + (e & 1) * Lay::kB);
        const uint32_t asel = tmem + (prod >= 2 ? 128u : 0u);
        const uint32_t dcol = tmem + acc0 + 32u * (uint32_t)prod;
        const int j0 = 8 * (prod & 1);
#pragma unroll
        for (int j = j0; j < j0 + 8; ++j)
          mma_ts(dcol, asel + 8 * j, desc_kmajor(bsel + (uint32_t)(2 * j) * (16u * N), 16 * N, 128), idesc, j > j0);
        mma_commit(sa(&bar[2]));
      } else {
        mb_arrive(sa(&bar[2]));
      }
    }
    // the movers: step s - 1's outputs out, Zx of step s + 2 in (one
    // asynchronous-copy group per step)
    if (wt >= 4) {
      if (s > 0) store_step(s - 1, tt - 128, NWK);
      if (s + 2 < Tg) load_zx(s + 2, tt - 128, NWK);
      cp_commit();
    }
    const float *zs = zx + (s % 3) * N * RF;
    float acc[C];
#pragma unroll
    for (int k = 0; k < C; ++k) acc[k] = zs[((col0 + k) * 4 + q) * kTHc + lane];
    if (s > 0) {
      ++mma_issued;
      const bool got = mb_wait(sa(&bar[2]), (uint32_t)(e & 1), cap);
      if (got) ++mma_seen;
      ok = got && ok;
      fence_after();
      uint32_t r[4][C];
#pragma unroll
      for (int p = 0; p < 4; ++p) tmem_ld_raw<C>(tl + acc0 + 32 * p + col0, r[p]);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
      for (int k = 0; k < C; ++k)
        acc[k] += (__uint_as_float(r[0][k]) + __uint_as_float(r[1][k])) +
                  (__uint_as_float(r[2][k]) + __uint_as_float(r[3][k])) * (1.f / kF16LoScale);
    }
    // gate q of unit `lane` for this thread's columns (uniform per warp)
    const uint32_t par = (uint32_t)(s & 1);
    float *gs = gate + par * N * RF;
#pragma unroll
    for (int k0 = 0; k0 < C; k0 += 4) {
      float v[4] = {acc[k0], acc[k0 + 1], acc[k0 + 2], acc[k0 + 3]};
      if (q == 2)
        act4<true>(v);
      else
        act4<false>(v);
#pragma unroll
      for (int k = 0; k < 4; ++k) gs[((col0 + k0 + k) * 4 + q) * kTHc + lane] = v[k];
    }
    fence_before();
    // an issuer that gave up on the exchange stops the whole team
    if (team_sync_or(bid, TT, !ok)) {
      if (tt == 0) atomicOr(a.status, kErrExchWait);
      stop = true;
      break;
    }
    // cell update of unit `lane`, rows P wt + j
    uint8_t *sg = stg + par * Lay::kStgS;
    float *cl = cell + par * 2 * N * kTHc;
#pragma unroll
    for (int j = 0; j < P; ++j) {
      const int n = P * wt + j;
      const float ig = gs[(n * 4 + 0) * kTHc + lane], fg = gs[(n * 4 + 1) * kTHc + lane];
      const float gg = gs[(n * 4 + 2) * kTHc + lane], og = gs[(n * 4 + 3) * kTHc + lane];
      const float cn = fmaf(fg, cst[j], ig * gg);
      float h = og * tanh_tc(cn);
      if (s < lenp[j])
        cst[j] = cn;
      else
        h = 0.f;
      cl[n * kTHc + lane] = cn;
      cl[(N + n) * kTHc + lane] = h;
      const uint32_t off = (uint32_t)(lane >> 3) * Lay::kOct + (uint32_t)n * 16u + (uint32_t)(lane & 7) * 2u;
      *reinterpret_cast<__half *>(sg + off) = __float2half_rn(h);
    }
    if (wt >= 4) cp_wait<1>();  // Zx of step s + 1 has landed (seen by all after the barrier)
    team_sync(bid, TT);
    if (s + 1 < Tg && !withhold) {
      constexpr int kPieces = Lay::kSlice / 16;
      const uint32_t dst0 = sa(Bb + par * Lay::kB) + c * (uint32_t)Lay::kSlice;
      const uint32_t mbl = sa(&bar[par]);
#pragma unroll
      for (int i = tt; i < kTCS * kPieces; i += TT) {
        // piece pc = (octet, row): 16 pc bytes into the K-major slice
        const int pr = i / kPieces, pc = i % kPieces;
        const uint32_t o = (uint32_t)pc * 16u, so = (uint32_t)(pc / N) * Lay::kOct + (uint32_t)(pc % N) * 16u;
        const uint4 v = *reinterpret_cast<const uint4 *>(sg + so);
        st_async16(peer(dst0 + o, (uint32_t)pr), v, peer(mbl, (uint32_t)pr));
      }
    }
  }
  if (!stop && Tg > 0) store_step(Tg - 1, tt, TT);  // the last step's outputs
  cp_wait<0>();
  if (mma_seen < mma_issued) mb_wait(sa(&bar[2]), (uint32_t)((mma_issued - 1) & 1), kTPolls);
  if (stop) __nanosleep(20000);
  fence_before();
  cluster_sync_all();
  fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// The body of one cluster: direction d, rows rc .. rc + TM N - 1 (smem
// 1024-byte aligned).
template <int N, int TM>
__device__ __forceinline__ void bwd_tc_body(const RecArgs &a, uint8_t *smem, const int d, const int rc, const int gcl,
                                            const int ncl) {
  using Lay = TcBwdLayout<N>;
  using Sm = TcSmem<Lay, N, TM>;
  constexpr int H = kTH, G = 4 * H, kTThreads = 512, TW = 16 / TM, TT = 32 * TW, QW = TW / 4, C = N / QW,
                P = N / TW, R = N * TM, RS = Lay::kRS;
  // Accumulators per 128-unit half: with one team, one per product (three
  // issuers per half); with two, one per half of the k-steps (two issuers
  // per half, each forming all three products), so that both teams'
  // accumulators fit the 256 free TMEM columns at 32-column spacing.
  constexpr int AH = TM == 1 ? 3 : 2;
  static_assert(C == 4 || C == 8, "4 or 8 accumulator columns per thread");
  static_assert(P * TW == N && 2 * AH <= TW, "whole rows per warp; an issuer per warp");
  constexpr uint32_t idesc = tc_idesc<N>();
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int tm = warp / TW, wt = warp % TW, tt = t % TT;
  uint8_t *team = smem + tm * Lay::kTeam;
  uint8_t *Bz = team + Lay::oB;
  float *red = reinterpret_cast<float *>(team + Lay::oRed);
  float *pst = reinterpret_cast<float *>(team + Lay::oStg);
  uint64_t *bar = reinterpret_cast<uint64_t *>(team + Lay::oBar);
  uint32_t *tslot = reinterpret_cast<uint32_t *>(smem + Sm::oSlot);
  int *rlen_c = reinterpret_cast<int *>(smem + Sm::oLen);
  const int *rlen = rlen_c + tm * N;
  int *toff_s = reinterpret_cast<int *>(smem + Sm::oToff);

  const int qt = wt & 3, cs = wt >> 2;
  const int col0 = C * cs;
  const int u = lane;  // phase B: unit `lane`, rows P wt + j
  const uint32_t c = cluster_rank();
  const int gu = (int)c * kTHc + u;
  const int r0 = rc + tm * N;
  const int DH = a.dirs * H, T = a.ix.T;
  const bool toff_sm = T + 1 <= tc_tok_cap<N>(true);
  const int *toff = toff_sm ? toff_s : a.ix.tok_off;
  const int cap = a.wf.poll_cap > 0 ? a.wf.poll_cap : kTPolls;
  const bool withhold = (a.wf.withhold & kWithholdExchange) && c == 0;
  const int bid = 1 + tm;

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(tslot)), "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
#pragma unroll
  for (int k = 0; k < TM; ++k)
    for (uint32_t i = t; i < 2 * Lay::kB / 16; i += kTThreads)
      reinterpret_cast<uint4 *>(smem + k * Lay::kTeam + Lay::oB)[i] = make_uint4(0, 0, 0, 0);
  if (toff_sm)
    for (int i = t; i <= T; i += kTThreads) toff_s[i] = a.ix.tok_off[i];
  if (t < R) rlen_c[t] = rc + t < a.ix.b ? a.ix.row_len[rc + t] : 0;
  if (t == 0) {
#pragma unroll
    for (int k = 0; k < TM; ++k) {
      uint64_t *b = reinterpret_cast<uint64_t *>(smem + k * Lay::kTeam + Lay::oBar);
      mb_init(sa(&b[0]), 1);
      mb_init(sa(&b[1]), 1);
      mb_init(sa(&b[2]), 2 * AH);  // one commit from each of the team's MMA issuers
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t tl = tmem + ((uint32_t)(32 * qt) << 16);
  // W_hh^T into TMEM (warps 0 .. 7): half hf = warp / 4 holds units
  // 128 hf + m in lane m; K = the CTA's gate rows k = 4 uu + qq (global row
  // qq H + 32c + uu); hi part in columns 128 hf .. + 63, lo part 64 after
  if (warp < 8) {
    const int hf = warp >> 2;
    const float *W = a.Whh[d];
    const int col = 128 * hf + 32 * qt + lane;
#pragma unroll 1
    for (int k0 = 0; k0 < 128; k0 += 16) {
      uint32_t hi[8], lo[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int k = k0 + 2 * j;
        const float w0 = __ldg(W + (size_t)((k & 3) * H + (int)c * kTHc + (k >> 2)) * H + col);
        const float w1 = __ldg(W + (size_t)(((k + 1) & 3) * H + (int)c * kTHc + ((k + 1) >> 2)) * H + col);
        __nv_bfloat16 h0, l0, h1, l1;
        split_bf16(w0, h0, l0);
        split_bf16(w1, h1, l1);
        hi[j] = pack2(h0, h1);
        lo[j] = pack2(l0, l1);
      }
      tmem_st8(tl + 128 * hf + k0 / 2, hi);
      tmem_st8(tl + 128 * hf + 64 + k0 / 2, lo);
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  const int Tg = rlen[0];
  cluster_sync_all();
  if (tt == 0) {
    if (Tg >= 2) mb_arm(sa(&bar[0]), Lay::kStepBytes);
    if (Tg >= 3) mb_arm(sa(&bar[1]), Lay::kStepBytes);
  }

  float *__restrict__ Z = a.Z[d];
  const float *__restrict__ Cs = a.Cst[d];
  const float *__restrict__ dY = a.dY;
  __nv_bfloat16 *__restrict__ dZb = reinterpret_cast<__nv_bfloat16 *>(a.dZb[d]);
  int len[P];  // lengths of this thread's rows P wt + j
#pragma unroll
  for (int j = 0; j < P; ++j) len[j] = rlen[P * wt + j];
  auto tok_at = [&](int j, int s) { return toff[d == 0 ? s : len[j] - 1 - s] + r0 + P * wt + j; };
  // phase B inputs of a step, loaded two steps ahead: gates i, f, g, o,
  // c_t, dY (c_{t-1} is the next step's c_t, zero before the first step)
  float in[P][6], nx[P][6], nx2[P][6];
  auto load_in = [&](int s, float (&v)[P][6]) {
#pragma unroll
    for (int j = 0; j < P; ++j) {
      if (s >= 0 && s < len[j]) {
        const size_t tk = (size_t)tok_at(j, s);
#pragma unroll
        for (int g = 0; g < 4; ++g) v[j][g] = Z[tk * G + g * H + gu];
        v[j][4] = Cs[tk * H + gu];
        v[j][5] = dY[tk * DH + d * H + gu];
      } else {
#pragma unroll
        for (int g = 0; g < 6; ++g) v[j][g] = 0.f;
      }
    }
  };
  load_in(Tg - 1, nx);
  load_in(Tg - 2, nx2);
  float dc[P];
#pragma unroll
  for (int j = 0; j < P; ++j) dc[j] = 0.f;
  // db of unit u, per gate, over this thread's rows and steps (fp32)
  float dbs[4] = {0.f, 0.f, 0.f, 0.f};
  const bool dz32 = !a.no_dz32;
  // MMA issuers: lane 0 of the team's warps 0 .. 2 AH - 1; issuer i works on
  // half i / AH into accumulator i of the team (AH = 3: product i % 3 of
  // W_hi dz_hi, W_hi dz_lo, W_lo dz_hi over all eight k-steps; AH = 2: all
  // three products over k-steps 4 (i % 2) .. + 3)
  const int iss = (lane == 0 && wt < 2 * AH) ? wt : -1;
  const uint32_t acc0 = kAccCol + 32u * (uint32_t)(2 * AH * tm);  // the team's 2 AH accumulators
  bool ok = true, stop = false;
  int mma_issued = 0, mma_seen = 0;
  const uint32_t bh = sa(Bz);

  for (int it = 0; it < Tg && !stop; ++it) {
    const int s = Tg - 1 - it;
#pragma unroll
    for (int j = 0; j < P; ++j)
#pragma unroll
      for (int g = 0; g < 6; ++g) {
        in[j][g] = nx[j][g];
        nx[j][g] = nx2[j][g];
      }
    load_in(s - 2, nx2);
    const float *rp = nullptr;
    if (it > 0) {
      const int e = it - 1;
      ok = mb_wait(sa(&bar[e & 1]), (e >> 1) & 1, cap) && ok;
      if (tt == 0 && ok && e + 2 <= Tg - 2) mb_arm(sa(&bar[e & 1]), Lay::kStepBytes);
      rp = red + (size_t)(e & 1) * (kTCS * N * RS) + u;
    }
    // phase B: dh, dc and dz of unit u for rows P wt + j
#pragma unroll
    for (int j = 0; j < P; ++j) {
      const int n = P * wt + j;
      float dz4[4] = {0.f, 0.f, 0.f, 0.f};
      if (s < len[j]) {
        float dh = in[j][5];
        if (rp) {
#pragma unroll
          for (int src = 0; src < kTCS; ++src) dh += rp[((size_t)src * N + n) * RS];
        }
        // c_{t-1}: the c_t of step s - 1 (zero when s is the row's first step)
        const float ig = in[j][0], fg = in[j][1], gg = in[j][2], og = in[j][3], ct = in[j][4], cp = nx[j][4];
        const float tch = tanh_tc(ct);
        const float dcv = fmaf(dh * og, 1.f - tch * tch, dc[j]);
        dz4[0] = dcv * gg * ig * (1.f - ig);
        dz4[1] = dcv * cp * fg * (1.f - fg);
        dz4[2] = dcv * ig * (1.f - gg * gg);
        dz4[3] = dh * tch * og * (1.f - og);
        dc[j] = dcv * fg;
        if (dz32) {
          float *zr = Z + (size_t)tok_at(j, s) * G + gu;
          zr[0] = dz4[0];
          zr[H] = dz4[1];
          zr[2 * H] = dz4[2];
          zr[3 * H] = dz4[3];
        }
#pragma unroll
        for (int g = 0; g < 4; ++g) dbs[g] += dz4[g];
      } else {
        dc[j] = 0.f;
      }
      // B operand: k = 4u .. 4u + 3 of row n (8 bytes of each part), in
      // 64-k atom u / 16 at 16-byte chunk (u % 16) / 2 swizzled by n % 8, so
      // that a warp's 32 stores fill two whole 128-byte rows
      // (hi rounded to nearest, lo the rounded rest, two values per conversion)
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(dz4[0], dz4[1]), h23 = __floats2bfloat162_rn(dz4[2], dz4[3]);
      const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
      const __nv_bfloat162 l01 = __floats2bfloat162_rn(dz4[0] - f01.x, dz4[1] - f01.y);
      const __nv_bfloat162 l23 = __floats2bfloat162_rn(dz4[2] - f23.x, dz4[3] - f23.y);
      if (dZb && s < len[j]) {  // bf16 dz for the bf16 contractions
        __nv_bfloat16 *zb = dZb + (size_t)tok_at(j, s) * G + gu;
        zb[0] = h01.x;
        zb[H] = h01.y;
        zb[2 * H] = h23.x;
        zb[3 * H] = h23.y;
      }
      const uint32_t off = (uint32_t)(u >> 4) * (128u * N) + (uint32_t)n * 128u +
                           (uint32_t)((((u & 15) >> 1) ^ (n & 7)) * 16) + (uint32_t)(u & 1) * 8u;
      *reinterpret_cast<uint2 *>(Bz + off) = make_uint2(bf2u(h01), bf2u(h23));
      *reinterpret_cast<uint2 *>(Bz + Lay::kB + off) = make_uint2(bf2u(l01), bf2u(l23));
    }
    fence_proxy();
    fence_before();
    if (team_sync_or(bid, TT, !ok)) {
      if (tt == 0) atomicOr(a.status, kErrExchWait);
      stop = true;
      break;
    }
    fence_after();
    if (it + 1 >= Tg) continue;  // dh_{-1} is not needed
    // this CTA's partial W_hh^T dz for all 256 units (two halves of 128 lanes)
    if (iss >= 0) {
      const int hf = iss / AH, ia = iss % AH;
      const uint32_t dcol = tmem + acc0 + 32u * (uint32_t)iss;
      const uint32_t abase = tmem + 128u * (uint32_t)hf;
      auto one = [&](int j, int p, bool accum) {
        const uint32_t asel = abase + (p == 2 ? 64u : 0u);
        const uint32_t bsel = bh + (p == 1 ? Lay::kB : 0u);
        mma_ts(dcol, asel + 8 * j, desc_sw128(bsel + (uint32_t)(j >> 2) * (128u * N) + (uint32_t)(j & 3) * 32u), idesc, accum);
      };
      if constexpr (AH == 3) {
#pragma unroll
        for (int j = 0; j < 128 / 16; ++j) one(j, ia, j > 0);
      } else {
#pragma unroll
        for (int jj = 0; jj < 4; ++jj)
#pragma unroll
          for (int p = 0; p < 3; ++p) one(4 * ia + jj, p, jj > 0 || p > 0);
      }
      mma_commit(sa(&bar[2]));
    }
    ++mma_issued;
    const bool got = mb_wait(sa(&bar[2]), (uint32_t)((mma_issued - 1) & 1), cap);
    if (got) ++mma_seen;
    ok = got && ok;
    fence_after();
    float p0[C], p1[C];
#pragma unroll
    for (int k = 0; k < C; ++k) p0[k] = p1[k] = 0.f;
#pragma unroll
    for (int i = 0; i < AH; ++i) {
      tmem_ld_add<C>(tl + acc0 + 32 * i + col0, p0);
      tmem_ld_add<C>(tl + acc0 + 32 * (AH + i) + col0, p1);
    }
    // stage the partials by owner (unit 32 qt + lane of half hf belongs to
    // CTA qt + 4 hf), rows contiguous, so that each remote store is a whole
    // 16-byte piece of consecutive memory on both sides; the warp's pieces
    // (its C rows for owners qt and qt + 4) are its own, so it sends them
    // as soon as it has staged them
#pragma unroll
    for (int k = 0; k < C; ++k) {
      pst[((qt)*N + col0 + k) * kTHc + lane] = p0[k];
      pst[((qt + 4) * N + col0 + k) * kTHc + lane] = p1[k];
    }
    __syncwarp();
    if (!withhold && got) {
      const uint32_t par = (uint32_t)(it & 1);
      const uint32_t mbl = sa(&bar[par]);
      constexpr int kWP = C * (kTHc / 4);  // pieces per owner
#pragma unroll
      for (int i = lane; i < 2 * kWP; i += 32) {
        const int owner = qt + 4 * (i / kWP), rem = i % kWP, n = col0 + rem / (kTHc / 4), ch = rem % (kTHc / 4);
        const uint4 v = *reinterpret_cast<const uint4 *>(pst + (owner * N + n) * kTHc + 4 * ch);
        const uint32_t dst = sa(red) + (((par * kTCS + c) * N + n) * RS + 4 * ch) * 4u;
        st_async16(peer(dst, (uint32_t)owner), v, peer(mbl, (uint32_t)owner));
      }
    }
    fence_before();  // the accumulators are read before the next step's MMAs overwrite them
  }
  if (mma_seen < mma_issued) mb_wait(sa(&bar[2]), (uint32_t)((mma_issued - 1) & 1), kTPolls);
  if (a.dbp) {
    // db: the 16 warps' sums (both teams) meet in the first team's send
    // staging, then one thread per (gate, unit) adds them in warp order
    // and writes the cluster's partial (deterministic)
    float *red4 = reinterpret_cast<float *>(smem + Lay::oStg);  // [16 warps][4][32]
    __syncthreads();
#pragma unroll
    for (int g = 0; g < 4; ++g) red4[(warp * 4 + g) * kTHc + lane] = dbs[g];
    __syncthreads();
    if (t < 4 * kTHc) {
      const int g = t >> 5;
      float v = 0.f;
      for (int w = 0; w < kTThreads / 32; ++w) v += red4[(w * 4 + g) * kTHc + lane];
      a.dbp[((size_t)d * ncl + gcl) * G + g * H + (int)c * kTHc + lane] = v;
    }
  }
  if (stop) __nanosleep(20000);
  fence_before();
  cluster_sync_all();
  fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// ---------------------------------------------------------------------------
// Cluster layout of a launch.  A cluster of one team (16 rows on all 16
// warps) takes a step in about 1.7 us, a cluster of two teams (32 rows, 8
// warps each) about 2.9 us: the step is latency-bound, and two teams only
// partly hide each other's waits.  So one-team clusters are used wherever
// they fit: the longest rows of the length-sorted batch go to n1 one-team
// clusters per direction, the shortest to n2 two-team clusters, with
// dirs (n1 + n2) no more than the 8-CTA clusters that can be resident at
// once (15 on a 152-SM GB300; a cluster beyond them would start only when
// another ends, after the rows it was meant to run beside).
namespace {

constexpr int kTN = 16;  // rows per team: the N of the MMAs

struct TcSplit {
  int n1, n2;  // clusters per direction of one team (16 rows) and of two teams (32 rows)
};

}  // namespace

template <int N>
__global__ void __launch_bounds__(512, 1) lstm_fwd_tc_kernel(RecArgs a, TcSplit sp) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int cid = blockIdx.x / kTCS, per = sp.n1 + sp.n2;
  const int d = cid / per, g = cid % per;
  if (g < sp.n1)
    fwd_tc_body<N, 1>(a, smem, d, N * g);
  else
    fwd_tc_body<N, 2>(a, smem, d, N * sp.n1 + 2 * N * (g - sp.n1));
}

template <int N>
__global__ void __launch_bounds__(512, 1) lstm_bwd_tc_kernel(RecArgs a, TcSplit sp) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int cid = blockIdx.x / kTCS, per = sp.n1 + sp.n2;
  const int d = cid / per, g = cid % per;
  if (g < sp.n1)
    bwd_tc_body<N, 1>(a, smem, d, N * g, g, per);
  else
    bwd_tc_body<N, 2>(a, smem, d, N * sp.n1 + 2 * N * (g - sp.n1), g, per);
}

namespace {

size_t tc_smem(bool bwd, int T) { return tc_smem_bytes<kTN>(bwd, T); }
static_assert(tc_base<kTN>(false) <= kSmemMax && tc_base<kTN>(true) <= kSmemMax, "team layouts fit a CTA");

cudaLaunchConfig_t tc_config(int clusters, size_t smem, cudaStream_t s, cudaLaunchAttribute *attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(clusters * kTCS, 1, 1);
  cfg.blockDim = dim3(512, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr->id = cudaLaunchAttributeClusterDimension;
  attr->val.clusterDim.x = kTCS;
  attr->val.clusterDim.y = 1;
  attr->val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// 8-CTA clusters of one kernel that can be resident at once (0: cannot launch).
template <typename K>
int tc_resident_one(K k, size_t smem) {
  cudaLaunchAttribute attr;
  int n = 0;
  cudaError_t e = ensure_smem((const void *)k, smem);
  cudaLaunchConfig_t cfg = tc_config(1, smem, 0, &attr);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, k, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

TcSplit tc_split(int b, int dirs, int max_clusters) {
  const int groups = (b + kTN - 1) / kTN;                // 16-row groups per direction
  const int per = std::max(1, max_clusters / dirs);      // clusters per direction resident at once
  TcSplit sp;
  if (groups <= per) {
    sp.n1 = groups;
    sp.n2 = 0;
  } else if (groups - per >= (groups + 1) / 2) {
    sp.n1 = 0;  // two teams everywhere (clusters beyond the resident ones wait)
    sp.n2 = (groups + 1) / 2;
  } else {
    sp.n2 = groups - per;  // each two-team cluster saves one cluster
    sp.n1 = groups - 2 * sp.n2;
  }
  return sp;
}

}  // namespace

bool tc_rec_supported(int H) {
  static const bool off = [] {
    const char *e = getenv("BKT_REC_TC");
    return e && e[0] == '0';
  }();
  return H == kTH && !off;
}

int tc_clusters_per_dir(int b, int dirs, int max_clusters) {
  const TcSplit sp = tc_split(b, dirs, max_clusters);
  return sp.n1 + sp.n2;
}

int tc_clusters_resident() {
  const int f = tc_resident_one(lstm_fwd_tc_kernel<kTN>, tc_smem(false, kTTokCap - 1));
  const int b = tc_resident_one(lstm_bwd_tc_kernel<kTN>, tc_smem(true, kTTokCap - 1));
  return std::min(f, b);
}

cudaError_t launch_lstm_tc(const RecArgs &a, int max_clusters, bool bwd, cudaStream_t s) {
  if (a.ix.b <= 0 || a.ix.T <= 0) return cudaSuccess;
  if (a.H != kTH || max_clusters <= 0 || a.dirs < 1 || a.dirs > 2) return cudaErrorInvalidValue;
  const TcSplit sp = tc_split(a.ix.b, a.dirs, max_clusters);
  const size_t smem = tc_smem(bwd, a.ix.T);
  const int clusters = (sp.n1 + sp.n2) * a.dirs;
  cudaLaunchAttribute attr;
  cudaLaunchConfig_t cfg = tc_config(clusters, smem, s, &attr);
  if (bwd) {
    auto k = lstm_bwd_tc_kernel<kTN>;
    cudaError_t e = ensure_smem((const void *)k, smem);
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&cfg, k, a, sp);
  }
  auto k = lstm_fwd_tc_kernel<kTN>;
  cudaError_t e = ensure_smem((const void *)k, smem);
  if (e != cudaSuccess) return e;
  return cudaLaunchKernelEx(&cfg, k, a, sp);
}

}  // namespace bkt
