// k_gemm_tc.cu -- GEMMs on the 5th-generation tensor cores (tcgen05, TMEM
// accumulators):
//   gemm_bf16_tc_kernel    bf16 operands fed by TMA, one tile per CTA: the
//                          bf16 path's split-K weight gradients;
//   gemm_bf16_tc_persistent_kernel
//                          the same contraction, persistent with two TMEM
//                          accumulators: the bf16 path's input projections
//                          and input gradients (no split);
//   gemm_tf32x3_tc_kernel  fp32 split into tf32 hi + lo (3 MMAs per product),
//                          operands fed by TMA: the fp32 path's logits (with
//                          a log-softmax epilogue), dY, projections and dX,
//                          and weight gradients with unaligned operand rows;
//   gemm_tf32x3_tn_kernel  the same split, read token-major and split while
//                          loading: the fp32 path's weight gradients.
// The bf16 kernel:
//   D[m][n] (+)= sum_k A[m][k] * B[n][k]  (+ bias[n]),   fp32 accumulation
// A [M x K] and B [N x K] are bf16 with K contiguous (row-major); D is fp32.
//
// One CTA computes a 128 x 256 tile.  Warp 0 (one lane) streams 64-wide k
// slabs of A and B into shared memory with TMA (128-byte swizzle) through a
// 4-stage mbarrier ring; warp 1 (one lane) issues tcgen05.mma (M=128, N=256,
// K=16 per instruction) into a 256-column TMEM accumulator and releases each
// stage with tcgen05.commit; after the last slab all four warps read the
// accumulator back with tcgen05.ld (warp w owns TMEM lanes 32w..32w+31, i.e.
// tile rows) and write fp32 to global memory.  The token range can be split
// over gridDim.z, each split writing its own partial tile.  Every mbarrier
// wait is bounded: on expiry the CTA records an error flag, still waits for
// its issued MMAs through the final commit, waits (bounded) for the TMA loads
// it armed, frees TMEM and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "bkt_internal.h"

namespace bkt {

namespace {

constexpr int TBM = 128, TBN = 256, TBK = 64;
constexpr uint32_t kAStage = TBM * TBK * 2;  // 16 KB
constexpr uint32_t kBStage = TBN * TBK * 2;  // 32 KB
constexpr uint32_t kTxBytes = kAStage + kBStage;
// shared memory of the one-tile-per-CTA kernel with `stages` ring stages (4:
// the split-K weight gradients, one CTA per SM)
constexpr size_t tc_smem_for(int stages) { return 1024 + (size_t)stages * (kAStage + kBStage) + 256; }
constexpr uint32_t kWaitPolls = 1u << 22;
// kind::f16 instruction descriptor: D fp32 (bit 4), A and B bf16 (bits 7, 10),
// K-major unless bit 15 (A) / bit 16 (B) marks an MN-major operand, N >> 3 at
// bit 17, M >> 4 at bit 24.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(TBN >> 3) << 17) |
                            ((uint32_t)(TBM >> 4) << 24);
constexpr uint32_t kIdescAmn = 1u << 15, kIdescBmn = 1u << 16;
constexpr uint32_t kMnChunk = 64 * TBK * 2;  // one 64-element MN chunk of a 64-k slab (8 KB)

__device__ __forceinline__ uint32_t su32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(n) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t a) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(a), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity; false on expiry.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, uint32_t cap = kWaitPolls) {
  for (uint32_t i = 0; i < cap; ++i)
    if (mbar_try(a, parity)) return true;
  return false;
}
// The poll cap of a launch: the failure-detection hook's, else the built-in one.
__device__ __forceinline__ uint32_t wait_cap(const WaitFaults &wf) {
  return wf.poll_cap > 0 ? (uint32_t)wf.poll_cap : kWaitPolls;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(mbar)
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint32_t mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar) : "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// Shared-memory matrix descriptor of a K-major tile written by TMA with the
// 128-byte swizzle: rows of 128 B, 8-row groups 1024 B apart.  (An MN-major
// tile is 64-element MN chunks of `lbo` bytes, see sw128_desc_mn.)
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;            // leading byte offset (not used by swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset
  d |= (uint64_t)1 << 46;            // descriptor version
  d |= (uint64_t)2 << 61;            // 128-byte swizzle
  return d;
}
// The same for an MN-major tile (a token-major operand read without a
// transpose): each 128-byte row holds 64 consecutive M (or N) elements of one
// k; rows of consecutive k, 8-row groups 1024 B apart; the 64-element chunks
// along M (N) are `lbo` bytes apart.
__device__ __forceinline__ uint64_t sw128_desc_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;  // leading byte offset: next 64-element MN chunk
  d |= (uint64_t)(1024 >> 4) << 32;              // stride byte offset: next 8 k
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 3xTF32 variant: fp32 operands split as a = hi + lo (hi = a with the low 13
// mantissa bits cleared, exactly representable in tf32); the tile product is
// A_hi B_hi + A_hi B_lo + A_lo B_hi with fp32 accumulation, which leaves a
// relative error near 2^-20 per product.  128 x 128 tiles, 32-wide k slabs
// (128 bytes of fp32 per row), 3 stages of {A_hi, A_lo, B_hi, B_lo}.
constexpr int FBM = 128, FBN = 128, FBK = 32, FSTAGES = 3;
constexpr uint32_t kFTile = FBM * FBK * 4;  // 16 KB
constexpr uint32_t kFStage = 4 * kFTile;
constexpr size_t kFSmem = 1024 + (size_t)FSTAGES * kFStage + 256;
// kind::tf32 descriptor: D fp32 (bit 4), A and B tf32 (format 2 at bits 7, 10)
constexpr uint32_t kIdescTf32 = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(FBN >> 3) << 17) |
                                ((uint32_t)(FBM >> 4) << 24);

__device__ __forceinline__ void tc_mma_tf32(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

}  // namespace

template <int TSTAGES>
__global__ void __launch_bounds__(128, TSTAGES <= 2 ? 2 : 1)
    gemm_bf16_tc_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, TcGemmArgs g) {
  extern __shared__ uint8_t tc_smem_raw[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *sA = base;
  uint8_t *sB = base + TSTAGES * kAStage;
  uint64_t *bars = reinterpret_cast<uint64_t *>(sB + TSTAGES * kBStage);  // full[S], empty[S], done
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2 * TSTAGES + 1);
  int *abort_s = reinterpret_cast<int *>(tslot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * TBM, n0 = blockIdx.y * TBN;
  const int splits = g.P ? g.splits : 1;
  const int nkb = (g.K + TBK - 1) / TBK;
  const int chunk = (nkb + splits - 1) / splits;
  const int kb0 = blockIdx.z * chunk;
  const int nk = max(0, min(nkb, kb0 + chunk) - kb0);
  const uint32_t full0 = su32(bars), empty0 = su32(bars + TSTAGES), done = su32(bars + 2 * TSTAGES);

  if (threadIdx.x == 0) {
    for (int s = 0; s < TSTAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    *abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tslot)), "r"(TBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  const uint32_t cap = wait_cap(g.wf);
  if (warp == 0) {
    if (lane == 0) {  // TMA producer
      int last_phase[TSTAGES];  // phase of each stage's last armed load (-1: none)
#pragma unroll
      for (int s = 0; s < TSTAGES; ++s) last_phase[s] = -1;
      for (int i = 0; i < nk; ++i) {
        const int s = i % TSTAGES;
        if (i >= TSTAGES && !mbar_wait(empty0 + 8 * s, ((i / TSTAGES) - 1) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        if (i == 0 && (g.wf.withhold & kWithholdTma)) continue;  // failure-detection hook
        mbar_expect_tx(full0 + 8 * s, kTxBytes);
        const int kx = (kb0 + i) * TBK;
        // K-major: one 128-row box; MN-major: 64-element chunks of 64 k rows
        if (!g.a_mn) {
          tma_load_2d(su32(sA + s * kAStage), &ta, kx, m0, full0 + 8 * s);
        } else {
#pragma unroll
          for (int ch = 0; ch < TBM / 64; ++ch)
            tma_load_2d(su32(sA + s * kAStage + ch * kMnChunk), &ta, m0 + 64 * ch, kx, full0 + 8 * s);
        }
        if (!g.b_mn) {
          tma_load_2d(su32(sB + s * kBStage), &tb, kx, n0, full0 + 8 * s);
        } else {
#pragma unroll
          for (int ch = 0; ch < TBN / 64; ++ch)
            tma_load_2d(su32(sB + s * kBStage + ch * kMnChunk), &tb, n0 + 64 * ch, kx, full0 + 8 * s);
        }
        last_phase[s] = i / TSTAGES;
      }
      // after an abort, loads issued to stages the MMA warp never consumed
      // may still be in flight: wait (bounded) until every armed stage has
      // landed before the CTA can exit and its shared memory be reused
#pragma unroll
      for (int s = 0; s < TSTAGES; ++s)
        if (last_phase[s] >= 0 && !mbar_wait(full0 + 8 * s, last_phase[s] & 1, cap)) *abort_s = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      int issued = 0;
      for (int i = 0; i < nk; ++i) {
        const int s = i % TSTAGES;
        if (!mbar_wait(full0 + 8 * s, (i / TSTAGES) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = su32(sA + s * kAStage), b0 = su32(sB + s * kBStage);
        const uint32_t idesc = kIdesc | (g.a_mn ? kIdescAmn : 0u) | (g.b_mn ? kIdescBmn : 0u);
#pragma unroll
        for (int kk = 0; kk < TBK / 16; ++kk) {
          // k step kk: 32 bytes into each K-major row, or 16 rows (2 KB) of an MN-major tile
          const uint64_t ad = g.a_mn ? sw128_desc_mn(a0 + kk * 2048, kMnChunk) : sw128_desc(a0 + kk * 32);
          const uint64_t bd = g.b_mn ? sw128_desc_mn(b0 + kk * 2048, kMnChunk) : sw128_desc(b0 + kk * 32);
          tc_mma(tmem, ad, bd, idesc, (i > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(empty0 + 8 * s);
        ++issued;
      }
      // the final commit tracks every MMA issued above
      if (issued > 0) tc_commit(done);
      else mbar_arrive(done);
    }
    __syncwarp();
  }

  // epilogue: TMEM -> registers -> shared memory -> global.  TMEM lane = tile
  // row, so a thread holds one row; each 32-column chunk goes through a
  // per-warp staging block (the idle A stages: every MMA has completed) and
  // leaves as float4 stores that cover four whole 128-byte row pieces per
  // instruction (one row per thread would touch 32 rows per instruction)
  const bool ready_t = mbar_wait(done, 0, cap);
  if (!ready_t) *abort_s = 1;
  const bool ready = __all_sync(0xffffffffu, ready_t);  // uniform per warp: the chunk loop below syncs the warp
  tc_fence_after();
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  float *out_base;
  int64_t ld;
  if (g.P) {
    out_base = g.P + (int64_t)blockIdx.z * g.M * g.N;
    ld = g.N;
  } else {
    out_base = g.D;
    ld = g.ldd;
  }
  const bool vec = ((ld & 3) == 0) && ((reinterpret_cast<uintptr_t>(out_base) & 15) == 0);
  constexpr int kSt = 36;  // staging row stride (floats): 16-byte pieces of 8 consecutive rows hit distinct banks
  float *stg = reinterpret_cast<float *>(sA) + warp * 32 * kSt;
  const int cq = lane & 7, rq = lane >> 3;  // write phase: columns 4 cq .. 4 cq + 3 of rows rq + 4 i
#pragma unroll 1
  for (int c0 = 0; c0 < TBN; c0 += 32) {
    uint32_t v[32];
    __syncwarp();
    tmem_ld32(trow + c0, v);
    const int nb = n0 + c0;
    if (!ready || nb >= g.N) continue;  // uniform across the warp
#pragma unroll
    for (int j = 0; j < 32; j += 4)
      *reinterpret_cast<float4 *>(stg + lane * kSt + j) =
          nk > 0 ? make_float4(__uint_as_float(v[j]), __uint_as_float(v[j + 1]), __uint_as_float(v[j + 2]),
                               __uint_as_float(v[j + 3]))
                 : make_float4(0.f, 0.f, 0.f, 0.f);
    __syncwarp();
    const int n = nb + 4 * cq;
    float4 bias4 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (!g.P && g.bias) {
      bias4.x = n < g.N ? g.bias[n] : 0.f;
      bias4.y = n + 1 < g.N ? g.bias[n + 1] : 0.f;
      bias4.z = n + 2 < g.N ? g.bias[n + 2] : 0.f;
      bias4.w = n + 3 < g.N ? g.bias[n + 3] : 0.f;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = rq + 4 * i, m = m0 + warp * 32 + r;
      if (m >= g.M) continue;
      float4 x = *reinterpret_cast<const float4 *>(stg + r * kSt + 4 * cq);
      x.x += bias4.x;
      x.y += bias4.y;
      x.z += bias4.z;
      x.w += bias4.w;
      float *o = out_base + (int64_t)m * ld + n;
      if (vec && n + 4 <= g.N) {
        if (!g.P && g.accumulate) {
          const float4 y = *reinterpret_cast<const float4 *>(o);
          x.x += y.x;
          x.y += y.y;
          x.z += y.z;
          x.w += y.w;
        }
        *reinterpret_cast<float4 *>(o) = x;
      } else {
        const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (n + j < g.N) o[j] = xs[j] + ((!g.P && g.accumulate) ? o[j] : 0.f);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TBN) : "memory");
  if (threadIdx.x == 0 && *abort_s && g.err) atomicOr(g.err, kErrTcWait);
}

// Persistent variant for contractions without a split (the projections and
// dX): one CTA per SM walks the tiles n-fastest (m0 = (t / tiles_n) * 128),
// t = blockIdx.x, blockIdx.x + gridDim.x, ...  Warp 0 (one lane) streams
// the k slabs of every tile through a 4-stage TMA ring; warp 1 (one lane)
// issues each tile's MMAs into one of two 256-column TMEM accumulators in
// turn and commits it to that accumulator's `full` barrier; warps 2 .. 5
// (TMEM lane quarters 2, 3, 0, 1) drain the other accumulator to global
// memory through their own staging blocks and release it on its `empty`
// barrier, so a tile's epilogue overlaps the next tile's loads and MMAs.
constexpr int kPStages = 4, kPThreads = 192, kPSt = 36;
constexpr size_t kPStgBytes = 4 * 32 * kPSt * 4;
constexpr size_t kPSmem = 1024 + (size_t)kPStages * (kAStage + kBStage) + kPStgBytes + 256;

__global__ void __launch_bounds__(kPThreads, 1)
    gemm_bf16_tc_persistent_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                                   const __grid_constant__ CUtensorMap ta2, const __grid_constant__ CUtensorMap tb2,
                                   TcGemmArgs g) {
  extern __shared__ uint8_t tc_smem_raw[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *sA = base;
  uint8_t *sB = base + kPStages * kAStage;
  float *stg_all = reinterpret_cast<float *>(sB + kPStages * kBStage);
  uint64_t *bars = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(stg_all) + kPStgBytes);
  // full[S], empty[S], acc_full[2], acc_empty[2], done
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2 * kPStages + 5);
  int *abort_s = reinterpret_cast<int *>(tslot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles_m = (g.M + TBM - 1) / TBM, tiles_n = (g.N + TBN - 1) / TBN, total = tiles_m * tiles_n;
  // k slabs of the first pair, then of the second (if any)
  const int nkb1 = (g.K + TBK - 1) / TBK, nkb = nkb1 + (g.A2 ? (g.K2 + TBK - 1) / TBK : 0);
  const uint32_t full0 = su32(bars), empty0 = su32(bars + kPStages), afull0 = su32(bars + 2 * kPStages),
                 aempty0 = su32(bars + 2 * kPStages + 2), done = su32(bars + 2 * kPStages + 4);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(afull0 + 8 * b, 1);
      mbar_init(aempty0 + 8 * b, 4);  // one arrival per epilogue warp
    }
    mbar_init(done, 1);
    *abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tslot)), "r"(2 * TBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t cap = wait_cap(g.wf);

  if (warp == 0) {
    if (lane == 0) {  // TMA producer
      int last_phase[kPStages];  // phase of each stage's last armed load (-1: none)
#pragma unroll
      for (int s = 0; s < kPStages; ++s) last_phase[s] = -1;
      int it = 0;
      bool stop = false;
      for (int t = blockIdx.x; t < total && !stop; t += gridDim.x) {
        const int m0 = (t / tiles_n) * TBM, n0 = (t % tiles_n) * TBN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kPStages;
          if (it >= kPStages && !mbar_wait(empty0 + 8 * s, ((it / kPStages) - 1) & 1, cap)) {
            *abort_s = 1;
            stop = true;
            break;
          }
          if (it == 0 && (g.wf.withhold & kWithholdTma)) continue;  // failure-detection hook
          mbar_expect_tx(full0 + 8 * s, kTxBytes);
          const bool second = kb >= nkb1;
          const int kx = (second ? kb - nkb1 : kb) * TBK;
          const CUtensorMap *ma = second ? &ta2 : &ta, *mb = second ? &tb2 : &tb;
          if (!g.a_mn) {
            tma_load_2d(su32(sA + s * kAStage), ma, kx, m0, full0 + 8 * s);
          } else {
#pragma unroll
            for (int ch = 0; ch < TBM / 64; ++ch)
              tma_load_2d(su32(sA + s * kAStage + ch * kMnChunk), ma, m0 + 64 * ch, kx, full0 + 8 * s);
          }
          if (!g.b_mn) {
            tma_load_2d(su32(sB + s * kBStage), mb, kx, n0, full0 + 8 * s);
          } else {
#pragma unroll
            for (int ch = 0; ch < TBN / 64; ++ch)
              tma_load_2d(su32(sB + s * kBStage + ch * kMnChunk), mb, n0 + 64 * ch, kx, full0 + 8 * s);
          }
          last_phase[s] = it / kPStages;
        }
      }
      // loads issued to stages that no MMA consumed may still be in flight
      // after an abort: wait (bounded) until every armed stage has landed
#pragma unroll
      for (int s = 0; s < kPStages; ++s)
        if (last_phase[s] >= 0 && !mbar_wait(full0 + 8 * s, last_phase[s] & 1, cap)) *abort_s = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      int it = 0, lt = 0, issued = 0;
      bool stop = false;
      const uint32_t idesc = kIdesc | (g.a_mn ? kIdescAmn : 0u) | (g.b_mn ? kIdescBmn : 0u);
      for (int t = blockIdx.x; t < total && !stop; t += gridDim.x, ++lt) {
        const int ab = lt & 1;
        if (lt >= 2 && !mbar_wait(aempty0 + 8 * ab, ((lt >> 1) - 1) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(ab * TBN);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kPStages;
          if (!mbar_wait(full0 + 8 * s, (it / kPStages) & 1, cap)) {
            *abort_s = 1;
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = su32(sA + s * kAStage), b0 = su32(sB + s * kBStage);
#pragma unroll
          for (int kk = 0; kk < TBK / 16; ++kk) {
            const uint64_t ad = g.a_mn ? sw128_desc_mn(a0 + kk * 2048, kMnChunk) : sw128_desc(a0 + kk * 32);
            const uint64_t bd = g.b_mn ? sw128_desc_mn(b0 + kk * 2048, kMnChunk) : sw128_desc(b0 + kk * 32);
            tc_mma(d, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(empty0 + 8 * s);
          ++issued;
        }
        if (!stop) tc_commit(afull0 + 8 * ab);
      }
      // the final commit tracks every MMA issued above
      if (issued > 0) tc_commit(done);
      else mbar_arrive(done);
    }
    __syncwarp();
  } else {
    // epilogue: warp w owns TMEM lane quarter w % 4 (tile rows 32 (w % 4) ..);
    // each 32-column chunk goes through the warp's staging block and leaves
    // as float4 stores covering four whole 128-byte row pieces
    const int q = warp & 3;
    float *stg = stg_all + (warp - 2) * 32 * kPSt;
    const int cq = lane & 7, rq = lane >> 3;  // write phase: columns 4 cq .. + 3 of rows rq + 4 i
    int lt = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++lt) {
      const int ab = lt & 1;
      const bool ready_t = mbar_wait(afull0 + 8 * ab, (lt >> 1) & 1, cap);
      if (!ready_t) *abort_s = 1;
      if (!__all_sync(0xffffffffu, ready_t)) break;  // uniform per warp
      tc_fence_after();
      const int m0 = (t / tiles_n) * TBM, n0 = (t % tiles_n) * TBN;
      const uint32_t trow = tmem + (uint32_t)(ab * TBN) + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int c0 = 0; c0 < TBN; c0 += 32) {
        uint32_t v[32];
        __syncwarp();
        tmem_ld32(trow + c0, v);
        const int nb = n0 + c0;
        if (nb >= g.N) continue;  // uniform across the warp
#pragma unroll
        for (int j = 0; j < 32; j += 4)
          *reinterpret_cast<float4 *>(stg + lane * kPSt + j) = make_float4(
              __uint_as_float(v[j]), __uint_as_float(v[j + 1]), __uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]));
        __syncwarp();
        const int n = nb + 4 * cq;
        float4 bias4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (g.bias) {
          bias4.x = n < g.N ? g.bias[n] : 0.f;
          bias4.y = n + 1 < g.N ? g.bias[n + 1] : 0.f;
          bias4.z = n + 2 < g.N ? g.bias[n + 2] : 0.f;
          bias4.w = n + 3 < g.N ? g.bias[n + 3] : 0.f;
        }
        const bool vec = ((g.ldd & 3) == 0) && ((reinterpret_cast<uintptr_t>(g.D) & 15) == 0);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int r = rq + 4 * i, m = m0 + q * 32 + r;
          if (m >= g.M) continue;
          float4 x = *reinterpret_cast<const float4 *>(stg + r * kPSt + 4 * cq);
          x.x += bias4.x;
          x.y += bias4.y;
          x.z += bias4.z;
          x.w += bias4.w;
          float *o = g.D + (int64_t)m * g.ldd + n;
          if (vec && n + 4 <= g.N) {
            if (g.accumulate) {
              const float4 y = *reinterpret_cast<const float4 *>(o);
              x.x += y.x;
              x.y += y.y;
              x.z += y.z;
              x.w += y.w;
            }
            *reinterpret_cast<float4 *>(o) = x;
          } else {
            const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (n + j < g.N) o[j] = xs[j] + (g.accumulate ? o[j] : 0.f);
          }
        }
      }
      // every tcgen05.ld of this accumulator has completed (each waited):
      // hand it back to the issuer
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(aempty0 + 8 * ab);
    }
  }
  // no MMA may be in flight when TMEM is freed
  if (!mbar_wait(done, 0, cap)) *abort_s = 1;
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * TBN) : "memory");
  if (threadIdx.x == 0 && *abort_s && g.err) atomicOr(g.err, kErrTcWait);
}


__global__ void __launch_bounds__(128, 1)
    gemm_tf32x3_tc_kernel(const __grid_constant__ CUtensorMap tah, const __grid_constant__ CUtensorMap tal,
                          const __grid_constant__ CUtensorMap tbh, const __grid_constant__ CUtensorMap tbl,
                          TcGemmArgs g) {
  extern __shared__ uint8_t tc_smem_raw[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(base + FSTAGES * kFStage);  // full[S], empty[S], done
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2 * FSTAGES + 1);
  int *abort_s = reinterpret_cast<int *>(tslot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * FBM, n0 = blockIdx.y * FBN;
  const int splits = g.P ? g.splits : 1;
  const int nkb = (g.K + FBK - 1) / FBK;
  const int chunk = (nkb + splits - 1) / splits;
  const int kb0 = blockIdx.z * chunk;
  const int nk = max(0, min(nkb, kb0 + chunk) - kb0);
  const uint32_t full0 = su32(bars), empty0 = su32(bars + FSTAGES), done = su32(bars + 2 * FSTAGES);

  if (threadIdx.x == 0) {
    for (int s = 0; s < FSTAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    *abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tslot)), "r"(FBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  const uint32_t cap = wait_cap(g.wf);
  if (warp == 0) {
    if (lane == 0) {  // TMA producer
      int last_phase[FSTAGES];  // phase of each stage's last armed load (-1: none)
#pragma unroll
      for (int s = 0; s < FSTAGES; ++s) last_phase[s] = -1;
      for (int i = 0; i < nk; ++i) {
        const int s = i % FSTAGES;
        if (i >= FSTAGES && !mbar_wait(empty0 + 8 * s, ((i / FSTAGES) - 1) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        if (i == 0 && (g.wf.withhold & kWithholdTma)) continue;  // failure-detection hook
        uint8_t *st = base + s * kFStage;
        mbar_expect_tx(full0 + 8 * s, kFStage);
        const int kx = (kb0 + i) * FBK;
        tma_load_2d(su32(st), &tah, kx, m0, full0 + 8 * s);
        tma_load_2d(su32(st + kFTile), &tal, kx, m0, full0 + 8 * s);
        tma_load_2d(su32(st + 2 * kFTile), &tbh, kx, n0, full0 + 8 * s);
        tma_load_2d(su32(st + 3 * kFTile), &tbl, kx, n0, full0 + 8 * s);
        last_phase[s] = i / FSTAGES;
      }
      // drain the armed stages before the CTA can exit (see the bf16 kernel)
#pragma unroll
      for (int s = 0; s < FSTAGES; ++s)
        if (last_phase[s] >= 0 && !mbar_wait(full0 + 8 * s, last_phase[s] & 1, cap)) *abort_s = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      int issued = 0;
      for (int i = 0; i < nk; ++i) {
        const int s = i % FSTAGES;
        if (!mbar_wait(full0 + 8 * s, (i / FSTAGES) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        tc_fence_after();
        const uint32_t ah = su32(base + s * kFStage), al = ah + kFTile, bh = ah + 2 * kFTile, bl = ah + 3 * kFTile;
#pragma unroll
        for (int kk = 0; kk < FBK / 8; ++kk) {
          const uint32_t o = kk * 32;
          tc_mma_tf32(tmem, sw128_desc(ah + o), sw128_desc(bh + o), kIdescTf32, (i > 0 || kk > 0) ? 1u : 0u);
          tc_mma_tf32(tmem, sw128_desc(ah + o), sw128_desc(bl + o), kIdescTf32, 1u);
          tc_mma_tf32(tmem, sw128_desc(al + o), sw128_desc(bh + o), kIdescTf32, 1u);
        }
        tc_commit(empty0 + 8 * s);
        ++issued;
      }
      if (issued > 0) tc_commit(done);
      else mbar_arrive(done);
    }
    __syncwarp();
  }

  const bool ready = mbar_wait(done, 0, cap);
  if (!ready) *abort_s = 1;
  tc_fence_after();
  const int m = m0 + warp * 32 + lane;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  const bool write = ready && m < g.M;
  float *out;
  int64_t ld;
  if (g.P) {
    out = g.P + (int64_t)blockIdx.z * g.M * g.N + (int64_t)m * g.N;
    ld = g.N;
  } else {
    out = g.D + (int64_t)m * g.ldd;
    ld = g.ldd;
  }
  const bool vec = ((ld & 3) == 0) && ((reinterpret_cast<uintptr_t>(g.P ? g.P : g.D) & 15) == 0);
  if (g.logsoftmax) {
    // the whole row (N <= FBN columns, one tile) is in this thread's TMEM
    // lane: bias, then x - max - ln sum exp(x - max) over the N columns
    float x[FBN];
#pragma unroll
    for (int c0 = 0; c0 < FBN; c0 += 32) {
      uint32_t v[32];
      __syncwarp();
      tmem_ld32(trow + c0, v);
#pragma unroll
      for (int j = 0; j < 32; ++j) x[c0 + j] = __uint_as_float(v[j]);
    }
    if (write) {
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < FBN; ++j)
        if (j < g.N) {
          x[j] = (nk > 0 ? x[j] : 0.f) + (g.bias ? g.bias[j] : 0.f);
          mx = fmaxf(mx, x[j]);
        }
      float se = 0.f;
#pragma unroll
      for (int j = 0; j < FBN; ++j)
        if (j < g.N) se += expf(x[j] - mx);
      const float lz = mx + logf(se);
#pragma unroll
      for (int j = 0; j < FBN; ++j)
        if (j < g.N) out[j] = x[j] - lz;
    }
  } else
#pragma unroll 1
  for (int c0 = 0; c0 < FBN; c0 += 32) {
    uint32_t v[32];
    __syncwarp();
    tmem_ld32(trow + c0, v);
    if (!write) continue;
    const int nb = n0 + c0;
    if (nb >= g.N) continue;
    float x[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) x[j] = nk > 0 ? __uint_as_float(v[j]) : 0.f;
    if (!g.P) {
      if (g.bias)
#pragma unroll
        for (int j = 0; j < 32; ++j) x[j] += (nb + j < g.N) ? g.bias[nb + j] : 0.f;
      if (g.accumulate)
#pragma unroll
        for (int j = 0; j < 32; ++j) x[j] += (nb + j < g.N) ? out[nb + j] : 0.f;
    }
    if (vec && nb + 32 <= g.N) {
#pragma unroll
      for (int j = 0; j < 32; j += 4)
        *reinterpret_cast<float4 *>(out + nb + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (nb + j < g.N) out[nb + j] = x[j];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(FBN) : "memory");
  if (threadIdx.x == 0 && *abort_s && g.err) atomicOr(g.err, kErrTcWait);
}

// ---------------------------------------------------------------------------
// 3xTF32 contraction over the token axis with token-major operands:
//   D[m][n] = sum_k A[k][m] * B[g(k)][n]
// (A [K x M], B [rows x N], both fp32 row-major with M or N contiguous and
// 16-byte aligned rows, M and N multiples of 4; g an optional row gather, -1
// giving a zero row), as the weight gradients need (k = token), without
// transposed and split copies of the operands.
//
// Eight converter warps and one MMA warp.  Per 32-token slab a converter
// thread loads a 4 x 4 block of each tile (tokens 4 kc .. 4 kc + 3 of the
// slab, rows r0 .. r0 + 3) as four 16-byte vectors, two slabs ahead, into
// registers; out-of-range rows read a zero vector in global memory instead,
// so no instruction consumes a loaded value before its slab is converted (a
// warp issues in order).  Converting a slab transposes the block in
// registers, splits each value into tf32 hi + lo (truncating: hi = x with the
// low 13 mantissa bits cleared, lo = (x - hi) likewise, |x - hi - lo| <=
// 2^-20 |x|) and stores four 16-byte K-major chunks per tile in the 128-byte
// swizzled layout TMA would produce (chunk c of row r at chunk position
// c ^ (r & 7)), into one of kTnStages MMA stages; the warp then makes its
// stores visible to the tensor core (fence.proxy.async) and arrives on the
// stage's full barrier.  The MMA warp waits on it, issues the twelve MMAs and
// commits them to the stage's empty barrier, which the converter warps wait
// on before refilling the stage.  Converter warps never wait for each other.
// A thread's gather indices are loaded two slabs before the vectors they
// address; the loop is unrolled over two slabs to keep the prefetch
// registers statically named.  Every wait is bounded; on expiry the CTA
// records an error flag.  The epilogue splits the 128 accumulator columns
// between the two converter warps of each TMEM lane quarter.
namespace {

constexpr int kTnConv = 256;                      // converter threads (warps 0-7)
constexpr int kTnThreads = kTnConv + 32;          // + the MMA warp
constexpr int kTnStages = 3;                      // converted (MMA) stages
constexpr size_t kTnSmem = 1024 + (size_t)kTnStages * kFStage + 256;

__device__ __align__(16) float g_tn_zero[4];      // the zero vector out-of-range rows read

__device__ __forceinline__ void split_tf32_trunc(float x, float &h, float &l) {
  h = __uint_as_float(__float_as_uint(x) & 0xFFFFE000u);
  l = __uint_as_float(__float_as_uint(x - h) & 0xFFFFE000u);
}
// A read-only 16-byte load issued where it is written (volatile: not moved
// toward its use two slabs later).
__device__ __forceinline__ float4 ldg4_pinned(const float *p) {
  float4 v;
  asm volatile("ld.global.nc.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p));
  return v;
}

}  // namespace

__global__ void __launch_bounds__(kTnThreads, 1) gemm_tf32x3_tn_kernel(TnGemmArgs g) {
  extern __shared__ uint8_t tc_smem_raw[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(base + kTnStages * kFStage);  // full[S], empty[S], done
  uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2 * kTnStages + 1);
  int *abort_s = reinterpret_cast<int *>(tslot + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * FBM, n0 = blockIdx.y * FBN;
  const int nkb = (g.K + FBK - 1) / FBK;
  const int chunk = (nkb + g.splits - 1) / g.splits;
  const int kb0 = blockIdx.z * chunk;
  const int nk = max(0, min(nkb, kb0 + chunk) - kb0);
  const int kbase = kb0 * FBK;
  const int ntok = max(0, min(nk * FBK, g.K - kbase));
  const uint32_t full0 = su32(bars), empty0 = su32(bars + kTnStages), done = su32(bars + 2 * kTnStages);

  if (tid == 0) {
    for (int s = 0; s < kTnStages; ++s) {
      mbar_init(full0 + 8 * s, kTnConv / 32);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    *abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tslot)), "r"(FBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  const uint32_t cap = wait_cap(g.wf);
  if (warp == kTnConv / 32) {  // the MMA warp
    if (lane == 0) {
      int issued = 0;
      for (int i = 0; i < nk; ++i) {
        const int s = i % kTnStages;
        if (!mbar_wait(full0 + 8 * s, (i / kTnStages) & 1, cap)) {
          *abort_s = 1;
          break;
        }
        tc_fence_after();
        const uint32_t ah = su32(base + s * kFStage), al = ah + kFTile, bh = ah + 2 * kFTile, bl = ah + 3 * kFTile;
#pragma unroll
        for (int kk = 0; kk < FBK / 8; ++kk) {
          const uint32_t o = kk * 32;
          tc_mma_tf32(tmem, sw128_desc(ah + o), sw128_desc(bh + o), kIdescTf32, (i > 0 || kk > 0) ? 1u : 0u);
          tc_mma_tf32(tmem, sw128_desc(ah + o), sw128_desc(bl + o), kIdescTf32, 1u);
          tc_mma_tf32(tmem, sw128_desc(al + o), sw128_desc(bh + o), kIdescTf32, 1u);
        }
        tc_commit(empty0 + 8 * s);
        ++issued;
      }
      // the final commit tracks every MMA issued above
      if (issued > 0) tc_commit(done);
      else mbar_arrive(done);
    }
    __syncwarp();
  } else {  // converters
    // geometry: warp w covers rows 32 (w & 3) .. +31 and k chunks 4 (w >> 2)
    // .. +3; lane l takes rows r0 .. r0+3 with r0 = 32 (w & 3) + 4 rb, rb =
    // l & 7, and chunk kc = 4 (w >> 2) + ((rb >> 1) + (l >> 3)) mod 4, so
    // that the eight lanes of each quarter warp (one 128-bit shared store
    // phase) write eight distinct swizzled chunk positions
    const int rb = lane & 7;
    const int r0 = 32 * (warp & 3) + 4 * rb, kc = 4 * (warp >> 2) + (((rb >> 1) + (lane >> 3)) & 3);
    const bool a_in = m0 + r0 < g.M, b_in = n0 + r0 < g.N;  // M, N multiples of 4: a block is in or out
    const float *acol = g.A + (m0 + r0), *bcol = g.B + (n0 + r0);
    // B rows of this thread's tokens of slab i (gather read at clamped
    // positions; validity is checked where the rows are used); a uniform
    // branch, so that no select waits for the loaded indices
    const bool gathered = g.gather && ntok > 0;
    auto rows_of = [&](int i, int (&br)[4]) {
      if (gathered) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) br[kk] = __ldg(g.gather + kbase + min(i * FBK + 4 * kc + kk, ntok - 1));
      } else {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) br[kk] = kbase + i * FBK + 4 * kc + kk;
      }
    };
    auto load = [&](int i, const int (&br)[4], float4 (&va)[4], float4 (&vb)[4]) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int kl = i * FBK + 4 * kc + kk;
        const bool kin = kl < ntok;
        va[kk] = ldg4_pinned(kin && a_in ? acol + (int64_t)(kbase + kl) * g.lda : g_tn_zero);
        vb[kk] = ldg4_pinned(kin && b_in && br[kk] >= 0 ? bcol + (int64_t)br[kk] * g.ldb : g_tn_zero);
      }
    };
    bool fail = false;
    auto slab = [&](int i, float4 (&va)[4], float4 (&vb)[4], int (&br)[4]) -> bool {
      const int s = i % kTnStages;
      if (i >= kTnStages && !mbar_wait(empty0 + 8 * s, ((i / kTnStages) - 1) & 1, cap)) {
        fail = true;
        return false;
      }
      uint8_t *st = base + s * kFStage;
#pragma unroll
      for (int mm = 0; mm < 4; ++mm) {
        const int r = r0 + mm;
        const uint32_t off = (uint32_t)r * 128u + ((uint32_t)(kc ^ (r & 7)) << 4);
        auto el = [](const float4 &v, int q) { return q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w; };
        float4 ah, al, bh, bl;
        split_tf32_trunc(el(va[0], mm), ah.x, al.x);
        split_tf32_trunc(el(va[1], mm), ah.y, al.y);
        split_tf32_trunc(el(va[2], mm), ah.z, al.z);
        split_tf32_trunc(el(va[3], mm), ah.w, al.w);
        split_tf32_trunc(el(vb[0], mm), bh.x, bl.x);
        split_tf32_trunc(el(vb[1], mm), bh.y, bl.y);
        split_tf32_trunc(el(vb[2], mm), bh.z, bl.z);
        split_tf32_trunc(el(vb[3], mm), bh.w, bl.w);
        *reinterpret_cast<float4 *>(st + off) = ah;
        *reinterpret_cast<float4 *>(st + kFTile + off) = al;
        *reinterpret_cast<float4 *>(st + 2 * kFTile + off) = bh;
        *reinterpret_cast<float4 *>(st + 3 * kFTile + off) = bl;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      // (failure-detection hook: the first slab is never published)
      if (lane == 0 && !(i == 0 && (g.wf.withhold & kWithholdTma))) mbar_arrive(full0 + 8 * s);
      // the vectors of slab i + 2 (rows loaded two slabs ago), then the rows of slab i + 4
      load(i + 2, br, va, vb);
      rows_of(i + 4, br);
      return true;
    };

    float4 a0[4], b0[4], a1[4], b1[4];  // slabs of even and odd index
    int r_even[4], r_odd[4];
    rows_of(0, r_even);
    load(0, r_even, a0, b0);
    rows_of(1, r_odd);
    load(1, r_odd, a1, b1);
    rows_of(2, r_even);
    rows_of(3, r_odd);
    for (int i = 0; i < nk; i += 2) {
      if (!slab(i, a0, b0, r_even)) break;
      if (i + 1 < nk && !slab(i + 1, a1, b1, r_odd)) break;
    }
    if (fail) *abort_s = 1;
  }

  const bool ready = mbar_wait(done, 0, cap);
  tc_fence_after();
  __syncthreads();
  const bool aborted = *abort_s != 0;
  if (warp < kTnConv / 32) {
    const int quarter = warp & 3, half = warp >> 2;
    const int m = m0 + quarter * 32 + lane;
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    const bool write = ready && !aborted && m < g.M;
    float *out = g.P ? g.P + (int64_t)blockIdx.z * g.M * g.N + (int64_t)m * g.N : g.D + (int64_t)m * g.ldd;
#pragma unroll 1
    for (int cc = half * (FBN / 2); cc < (half + 1) * (FBN / 2); cc += 32) {
      uint32_t v[32];
      __syncwarp();
      tmem_ld32(trow + cc, v);
      if (!write) continue;
      const int nb = n0 + cc;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (nb + j < g.N) out[nb + j] = nk > 0 ? __uint_as_float(v[j]) : 0.f;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(FBN) : "memory");
  if (tid == 0 && (aborted || !ready) && g.err) atomicOr(g.err, kErrTcWait);
}

// ---------------------------------------------------------------------------
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D map over a row-major [rows x inner] matrix with row stride `ld`
// elements; boxes of 128 bytes (inner) x box_rows with the 128-byte swizzle.
bool make_map(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows, int64_t ld, uint32_t box_rows,
              bool fp32 = false) {
  auto fn = encode_fn();
  if (!fn) return false;
  const int esz = fp32 ? 4 : 2;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * esz};
  cuuint32_t box[2] = {(cuuint32_t)(128 / esz), box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(map, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            const_cast<void *>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int tc_splits(int M, int N, int K, int sm_count, size_t part_floats) {
  const int tiles = ((M + TBM - 1) / TBM) * ((N + TBN - 1) / TBN);
  const int nkb = (K + TBK - 1) / TBK;
  int s = std::max(1, sm_count / std::max(1, tiles));
  s = std::min(s, std::max(1, nkb / 4));  // at least 4 k slabs per split
  s = std::min(s, 64);
  while (s > 1 && (size_t)s * M * N > part_floats) --s;
  return s;
}

cudaError_t launch_gemm_bf16_tc(const TcGemmArgs &g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.K <= 0 || (g.lda & 7) || (g.ldb & 7) || (reinterpret_cast<uintptr_t>(g.A) & 15) ||
      (reinterpret_cast<uintptr_t>(g.B) & 15) || (g.P && g.splits < 1) || (!g.P && !g.D))
    return cudaErrorInvalidValue;
  if (g.A2 && (g.P || !g.B2 || g.K2 <= 0 || ((reinterpret_cast<uintptr_t>(g.A2) | reinterpret_cast<uintptr_t>(g.B2)) & 15)))
    return cudaErrorInvalidValue;
  CUtensorMap ta, tb, ta2, tb2;
  // K-major operands are [rows x K]; MN-major ones [K x rows] (rows contiguous)
  const bool okA = g.a_mn ? make_map(&ta, g.A, (uint64_t)g.M, (uint64_t)g.K, g.lda, TBK)
                          : make_map(&ta, g.A, (uint64_t)g.K, (uint64_t)g.M, g.lda, TBM);
  const bool okB = g.b_mn ? make_map(&tb, g.B, (uint64_t)g.N, (uint64_t)g.K, g.ldb, TBK)
                          : make_map(&tb, g.B, (uint64_t)g.K, (uint64_t)g.N, g.ldb, TBN);
  if (!okA || !okB) return cudaErrorInvalidValue;
  if (g.A2) {
    const bool okA2 = g.a_mn ? make_map(&ta2, g.A2, (uint64_t)g.M, (uint64_t)g.K2, g.lda, TBK)
                             : make_map(&ta2, g.A2, (uint64_t)g.K2, (uint64_t)g.M, g.lda, TBM);
    const bool okB2 = g.b_mn ? make_map(&tb2, g.B2, (uint64_t)g.N, (uint64_t)g.K2, g.ldb, TBK)
                             : make_map(&tb2, g.B2, (uint64_t)g.K2, (uint64_t)g.N, g.ldb, TBN);
    if (!okA2 || !okB2) return cudaErrorInvalidValue;
  } else {
    ta2 = ta;
    tb2 = tb;
  }
  dim3 grid((g.M + TBM - 1) / TBM, (g.N + TBN - 1) / TBN, g.P ? g.splits : 1);
  if (grid.y > 65535u || grid.z > 65535u) return cudaErrorInvalidConfiguration;
  if (!g.P) {
    // persistent: one CTA per SM over the tiles
    static int sms[64] = {0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (sms[dev] == 0) {
      int n = 0;
      e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return e;
      sms[dev] = n;
    }
    e = ensure_smem((const void *)gemm_bf16_tc_persistent_kernel, kPSmem);
    if (e != cudaSuccess) return e;
    const int64_t tiles = (int64_t)grid.x * grid.y;
    const unsigned blocks = (unsigned)std::min<int64_t>(tiles, sms[dev]);
    gemm_bf16_tc_persistent_kernel<<<blocks, kPThreads, kPSmem, s>>>(ta, tb, ta2, tb2, g);
  } else {
    cudaError_t e = ensure_smem((const void *)gemm_bf16_tc_kernel<4>, tc_smem_for(4));
    if (e != cudaSuccess) return e;
    gemm_bf16_tc_kernel<4><<<grid, 128, tc_smem_for(4), s>>>(ta, tb, g);
  }
  return cudaGetLastError();
}

int tf32x3_splits(int M, int N, int K, int sm_count, size_t part_floats) {
  const int tiles = ((M + FBM - 1) / FBM) * ((N + FBN - 1) / FBN);
  const int nkb = (K + FBK - 1) / FBK;
  int s = std::max(1, sm_count / std::max(1, tiles));
  s = std::min(s, std::max(1, nkb / 4));
  // at most 4096 tokens per accumulator: keeps fp32 accumulation chains short
  s = std::max(s, (K + 4095) / 4096);
  s = std::min(s, 64);
  while (s > 1 && (size_t)s * M * N > part_floats) --s;
  return s;
}

cudaError_t launch_gemm_tf32x3_tc(const TcGemmArgs &g, const void *A_lo, const void *B_lo, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.K <= 0 || (g.lda & 3) || (g.ldb & 3) || ((reinterpret_cast<uintptr_t>(g.A) | reinterpret_cast<uintptr_t>(g.B) |
                                                   reinterpret_cast<uintptr_t>(A_lo) | reinterpret_cast<uintptr_t>(B_lo)) &
                                                  15) ||
      (g.P && g.splits < 1) || (!g.P && !g.D))
    return cudaErrorInvalidValue;
  if (g.logsoftmax && (g.P || g.N > FBN || g.accumulate)) return cudaErrorInvalidValue;
  CUtensorMap tah, tal, tbh, tbl;
  if (!make_map(&tah, g.A, (uint64_t)g.K, (uint64_t)g.M, g.lda, FBM, true) ||
      !make_map(&tal, A_lo, (uint64_t)g.K, (uint64_t)g.M, g.lda, FBM, true) ||
      !make_map(&tbh, g.B, (uint64_t)g.K, (uint64_t)g.N, g.ldb, FBN, true) ||
      !make_map(&tbl, B_lo, (uint64_t)g.K, (uint64_t)g.N, g.ldb, FBN, true))
    return cudaErrorInvalidValue;
  cudaError_t e = ensure_smem((const void *)gemm_tf32x3_tc_kernel, kFSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((g.M + FBM - 1) / FBM, (g.N + FBN - 1) / FBN, g.P ? g.splits : 1);
  if (grid.y > 65535u || grid.z > 65535u) return cudaErrorInvalidConfiguration;
  gemm_tf32x3_tc_kernel<<<grid, 128, kFSmem, s>>>(tah, tal, tbh, tbl, g);
  return cudaGetLastError();
}

int tf32x3_tn_splits(int M, int N, int K, int sm_count, size_t part_floats) {
  return tf32x3_splits(M, N, K, sm_count, part_floats);
}

cudaError_t launch_gemm_tf32x3_tn(const TnGemmArgs &g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.K <= 0 || g.splits < 1 || (!g.P && (!g.D || g.splits != 1)) || !g.A || !g.B) return cudaErrorInvalidValue;
  // 16-byte pieces: every row of both tiles starts 16-byte aligned and no
  // piece straddles the end of a row
  if (((g.lda | g.ldb | g.M | g.N) & 3) != 0 ||
      ((reinterpret_cast<uintptr_t>(g.A) | reinterpret_cast<uintptr_t>(g.B)) & 15) != 0)
    return cudaErrorInvalidValue;
  cudaError_t e = ensure_smem((const void *)gemm_tf32x3_tn_kernel, kTnSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((g.M + FBM - 1) / FBM, (g.N + FBN - 1) / FBN, g.splits);
  if (grid.y > 65535u || grid.z > 65535u) return cudaErrorInvalidConfiguration;
  gemm_tf32x3_tn_kernel<<<grid, kTnThreads, kTnSmem, s>>>(g);
  return cudaGetLastError();
}

}  // namespace bkt
