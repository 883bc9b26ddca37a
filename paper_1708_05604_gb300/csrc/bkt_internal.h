// bkt_internal.h -- declarations shared by the host step engine and the CUDA
// kernels of libbkt.  Not part of the public ABI (see include/bkt.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "bkt.h"

#include <map>
#include <mutex>
#include <utility>

namespace bkt {

// Raises `func`'s dynamic shared-memory limit to at least `bytes` on the
// current device, calling the runtime only when the limit must grow (a
// cudaFuncSetAttribute per launch costs microseconds of host time per
// kernel, many times per step).  `cluster16` also allows 16-CTA clusters.
inline cudaError_t ensure_smem(const void *func, size_t bytes, bool cluster16 = false) {
  static std::mutex mu;
  static std::map<std::pair<int, const void *>, size_t> granted;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  auto it = granted.find({dev, func});
  if (it != granted.end() && it->second >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess && cluster16) e = cudaFuncSetAttribute(func, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) granted[{dev, func}] = bytes;
  return e;
}

// Device-side view of one packed mini-batch.  Rows are the batch's sequences
// sorted by length, longest first (stable), so the sequences still running at
// time t are rows 0 .. batch_size(t)-1 and token (t, r) sits at
// tok_off[t] + r of the time-major packed arrays.
struct DevIdx {
  int32_t b;       // sequences in the batch
  int32_t T;       // longest length
  int32_t n_tok;   // sum of lengths
  int32_t S_max;   // largest 2U+1 in the batch
  const int32_t *row_len;      // [b]
  const int32_t *row_lab_len;  // [b]
  const int32_t *row_orig;     // [b] position of the row in the caller's batch
  const int64_t *row_xoff;     // [b] first feature row in the caller's x
  const int64_t *row_lab_off;  // [b] first label in the caller's labels
  const int64_t *row_ctc_off;  // [b] offset of the row's [L x S] CTC tables
  const int32_t *tok_off;      // [T+1]
  const int32_t *tok_t;        // [n_tok] time index of each packed token
  const int32_t *tok_r;        // [n_tok] row of each packed token
  int64_t n_cells;             // host bookkeeping: sum_i L_i (2 U_i + 1), the CTC table cells
};

// Failure-detection hooks of a ctx (bkt_ctx_set_wait_faults): the poll cap
// of every bounded wait (0: the kernel's built-in cap) and the withhold bits.
struct WaitFaults {
  int32_t poll_cap;
  int32_t withhold;
};
constexpr int32_t kWithholdExchange = 1;  // BKT_WITHHOLD_EXCHANGE
constexpr int32_t kWithholdTma = 2;       // BKT_WITHHOLD_TMA

// Device error flags (word 0 of the status block; word 1 counts sequences
// without a CTC alignment).
constexpr int32_t kErrLabel = 1;     // a label outside 1..C-1
constexpr int32_t kErrTcWait = 2;    // a tensor-core pipeline wait ran out
constexpr int32_t kErrExchWait = 4;  // a recurrent cluster exchange wait ran out
constexpr int kStatusWords = 4;

// Records per-kernel CUDA events when timing is on (owned by the ctx).
// Each launch carries its algorithmic work (see bkt_kernel_time in bkt.h).
struct Work {
  double flops = 0, bytes = 0;
  int64_t steps = 0;
};
struct KernelTimer {
  virtual ~KernelTimer() {}
  virtual void begin(const char *name, const Work &w, cudaStream_t s) = 0;
  virtual void end(cudaStream_t s) = 0;
};

// Every launcher below enqueues on `s` and returns the launch status.

// a4: fills tok_t / tok_r, the previous-step token of every token for each
// direction (prev_tok[0]: (t-1, r); prev_tok[1]: (t+1, r); -1 where the
// direction starts), and gathers the caller's feature rows into the packed
// time-major X [n_tok x in_dim].
cudaError_t launch_layout(const DevIdx &ix, const float *x, int in_dim, float *X,
                          int32_t *tok_t, int32_t *tok_r, int32_t *const *prev_tok,
                          cudaStream_t s);

// a5 for a narrow input (in_dim <= 16): Z_d[tok][n] = b_d[n] + W_d[n] . X[tok]
// for both directions; W_d = params + w_off + d * w_stride, b_d follows W_hh.
cudaError_t launch_proj_narrow(const float *X, int n_tok, int in_dim, const float *params,
                               int64_t w_off, int64_t w_stride, int H, int dirs,
                               float *const *Z, cudaStream_t s);

// [out_w | out_b][m] = sum over the K token rows of A[k][m] [X[k] | 1] for an
// input X of D <= 16 columns (out_w row-major [M x D]); fixed summation order.
cudaError_t launch_narrow_wgrad(const float *A, int64_t lda, int M, const float *X, int D, int K, float *P,
                                size_t part_floats, int sm_count, float *out_w, float *out_b, cudaStream_t s);
// out[m*N + n] = sum_z P[z][m][n] (fixed order).
cudaError_t launch_splitk_sum(const float *P, int splits, int M, int N, float *out, cudaStream_t s);

// Operand preparation for the bf16 GEMMs (k_convert.cu).
cudaError_t launch_cast_bf16(const float *src, int64_t lds, int R, int C, void *dst, int64_t ldd, cudaStream_t s);
// dst[r][c] = bf16(src[src_row[r]][c]), zeros where src_row[r] < 0.
cudaError_t launch_gather_cast_bf16(const float *src, int64_t lds, const int32_t *src_row, int R, int C, void *dst,
                                    int64_t ldd, cudaStream_t s);
// P[z][m] = sum of A[r][m] over row chunk z of ceil(R / splits) rows (P
// holds splits * M floats), then launch_splitk_sum finishes the sums;
// colsum_splits picks about 256 rows per chunk within part_floats.
int colsum_splits(int R, int M, size_t part_floats);
cudaError_t launch_colsum(const float *A, int64_t lda, int R, int M, float *P, int splits, cudaStream_t s);
// hi[c][r] + lo[c][r] = src[src_row ? src_row[r] : r][c] to 2^-22 relative,
// hi and lo both tf32 values (zeros where src_row[r] < 0).
cudaError_t launch_transpose_split(const float *src, int64_t lds, const int32_t *src_row, int R, int C, float *hi,
                                   float *lo, int64_t ldd, cudaStream_t s);
// The same split without transposing (row-major, destination stride ldd).
cudaError_t launch_split_rows(const float *src, int64_t lds, int R, int C, float *hi, float *lo, int64_t ldd,
                              cudaStream_t s);

// bf16 tensor-core GEMM (k_gemm_tc.cu):
//   D[m][n] (+)= sum_k A[m][k] B[n][k] (+ bias[n]); A, B bf16, K-major (A
//   stored [M x K], B [N x K], K contiguous) or, with a_mn / b_mn, MN-major
//   (A stored [K x M], B [K x N]: token-major operands read without a
//   transpose); lda, ldb multiples of 8 elements, 16-byte aligned bases; D
//   fp32 row-major.
//   P != null: split the k range over `splits` and write partial tiles
//   P[z][m][n] instead (D, bias, accumulate unused).  err: device flag word
//   (bit 1 set if a pipeline wait timed out).
struct TcGemmArgs {
  int M, N, K;
  const void *A; int64_t lda;
  const void *B; int64_t ldb;
  float *D; int64_t ldd;
  const float *bias;
  int accumulate;
  float *P; int splits;
  int32_t *err;
  int logsoftmax;  // 3xTF32 GEMM only: replace each output row by its log-softmax (N <= 128, no split)
  WaitFaults wf;   // poll cap / withheld first slab (failure-detection tests)
  int a_mn, b_mn;  // bf16 GEMM only: operand stored MN-major (see above)
  // bf16 GEMM without a split only: a second pair summed into the same
  // tile, D = A B^T + A2 B2^T (A2 [M x K2], B2 like B; same strides and
  // layouts), e.g. both directions' dX in one contraction (null: none)
  const void *A2, *B2; int K2;
};
int tc_splits(int M, int N, int K, int sm_count, size_t part_floats);
cudaError_t launch_gemm_bf16_tc(const TcGemmArgs &g, cudaStream_t s);
// fp32 GEMM on the tensor cores with split precision (3xTF32): A = A (hi) +
// A_lo, B = B (hi) + B_lo, all fp32 row-major with K contiguous (lda, ldb
// multiples of 4, 16-byte aligned); D (or partials) as for the bf16 GEMM.
int tf32x3_splits(int M, int N, int K, int sm_count, size_t part_floats);
cudaError_t launch_gemm_tf32x3_tc(const TcGemmArgs &g, const void *A_lo, const void *B_lo, cudaStream_t s);
// The same 3xTF32 contraction over the token axis with token-major operands,
// split and swizzled while loading: D[m][n] = sum_k A[k*lda + m] B[g(k)*ldb + n]
// (g = gather, or the identity when null; a negative entry gives a zero row).
// Writes partials P[split][M][N] (D with ldd when splits == 1 and P is null).
// lda, ldb, M and N must be multiples of 4 and A, B 16-byte aligned.
struct TnGemmArgs {
  int M, N, K;
  const float *A; int64_t lda;
  const float *B; int64_t ldb;
  const int32_t *gather;
  float *D; int64_t ldd;
  float *P; int splits;
  int32_t *err;
  WaitFaults wf;
};
int tf32x3_tn_splits(int M, int N, int K, int sm_count, size_t part_floats);
cudaError_t launch_gemm_tf32x3_tn(const TnGemmArgs &g, cudaStream_t s);

// a8: log-space CTC forward (alpha) and backward (beta-hat) tables, one CTA
// per (row, direction); writes the per-sequence loss and the row's flag, and
// counts rows without an alignment in status[1].
cudaError_t launch_ctc_tables(const DevIdx &ix, const float *logp, int C, int blank,
                              const int32_t *labels, float *alpha, float *beta,
                              float *loss, int32_t *row_ok, int32_t *status,
                              cudaStream_t s);

// a9: dlogit = softmax - posterior, written over logp in place, and also as
// tf32 hi + lo parts [n_tok x ld_split] for the dY GEMM (when dl_hi is set).
cudaError_t launch_ctc_grad(const DevIdx &ix, float *logp_dlogit, int C, int blank, const int32_t *labels,
                            const float *alpha, const float *beta, const int32_t *row_ok, float *dl_hi, float *dl_lo,
                            int64_t ld_split, cudaStream_t s);

// Geometry of the recurrent kernels for one layer.
//   mode 1: one CTA per bc rows holds all of W_hh (H in {32, 64, 128});
//   mode 2: register-tiled clusters of cs CTAs, 4 or 8 rows each (H in
//           {256, 512}); bc = the clusters that can be resident at once;
//   mode 3: tensor-core clusters of 8 CTAs, 16 or 32 rows each, W_hh in
//           TMEM (H = 256 with bf16 contractions); bc = the clusters that
//           can be resident at once;
//   mode 0: a cluster of cs CTAs per bc rows splits the hidden units (any H).
struct RecGeom {
  int mode;
  int cs;        // CTAs per cluster (hidden units split cs ways)
  int bc;        // batch rows per cluster
  int ks;        // threads sharing one (row, unit) pair along k (power of 2 <= 8)
  int threads;   // threads per CTA
  int w_smem;    // 1: the CTA's W_hh slice lives in shared memory
  size_t smem_fwd, smem_bwd;
};
RecGeom plan_recurrent(int H, int b, int dirs, int sm_count, bool bf16);

// a6: persistent recurrent forward for both directions of one layer.
//   Z[d]  [n_tok x 4H] pre-activations in, activated gates (i,f,g,o) out
//   Cst[d] [n_tok x H] cell states; Y [n_tok x dirs*H] hidden outputs
//   Whh[d] = recurrent weights [4H x H] of direction d
struct RecArgs {
  DevIdx ix;
  int H, dirs;
  float *Z[2];
  float *Cst[2];
  const float *Whh[2];
  float *Y;            // forward: fp32 h [n_tok x dirs*H] (the tensor-core kernels take null: no fp32 copy)
  const float *dY;     // backward: d loss / d Y of this layer [n_tok x dirs*H]
  int32_t *status;     // device error flags (bit 4: a cluster exchange wait timed out)
  WaitFaults wf;       // poll cap / withheld exchange (failure-detection tests)
  // bf16 copies for the bf16 contractions, written by the kernels that
  // rec_writes_bf16() names (null: not wanted):
  void *Yb;            // forward: bf16 Y [n_tok x dirs*H]
  void *Hs[2];         // forward: bf16 h_{t-1} of every token of direction d [n_tok x H] (zeros at the start)
  void *dZb[2];        // backward: bf16 dz [n_tok x 4H]
  // backward, tensor-core kernels only:
  float *dbp;          // db as one partial sum per cluster, [dirs][clusters per direction][4H] (null: not formed)
  int no_dz32;         // 1: dz only as the bf16 copy, not over the gates in fp32
};
cudaError_t launch_lstm_fwd(const RecArgs &a, const RecGeom &g, cudaStream_t s);
// Whether the kernels of geometry g write RecArgs' bf16 copies.
inline bool rec_writes_bf16(const RecGeom &g) { return g.mode == 3; }
// a11: BPTT for both directions; Z[d] holds the gates on entry and dz on exit.
cudaError_t launch_lstm_bwd(const RecArgs &a, const RecGeom &g, cudaStream_t s);

// Register-tiled cluster kernels for H = 256 and 512 (k_lstm_cl.cu):
// CTAs per cluster for H (0: not handled there), how many of their clusters
// can be resident at once (0: they cannot launch), and the launch, which
// lays the batch's rows out over 4- and 8-row clusters, at most
// max_clusters of them.
int cl_cluster_size(int H);
int plan_cl_rows(int H, int b, int dirs);
cudaError_t launch_lstm_cl(const RecArgs &a, int max_clusters, bool bwd, cudaStream_t s);

// Tensor-core cluster kernels for H = 256 on the bf16 path (k_lstm_tc.cu):
// whether H is handled there (BKT_REC_TC=0 in the environment turns them
// off), how many of their 8-CTA clusters can be resident at once (0: they
// cannot launch), and the launch, which lays the batch's rows out over at
// most max_clusters clusters.
bool tc_rec_supported(int H);
int tc_clusters_resident();
cudaError_t launch_lstm_tc(const RecArgs &a, int max_clusters, bool bwd, cudaStream_t s);
// clusters per direction that a launch of b rows uses (their db partials)
int tc_clusters_per_dir(int b, int dirs, int max_clusters);

// Single-CTA recurrent kernels (k_lstm_cta.cu).
bool cta_supported(int H);
int cta_rows_per_block(int H, int b, int dirs, int sm_count);
cudaError_t launch_lstm_cta(const RecArgs &a, int bc, bool bwd, cudaStream_t s);

// a13
cudaError_t launch_sgd(float *p, const float *g, int64_t n, float lr, cudaStream_t s);
// Section III.B step 5, eq. 3: see bkt_average_models in bkt.h
cudaError_t launch_average_models(float *v, const float *prev, int64_t n, int K, float beta, cudaStream_t s);
// a13, ADADELTA: see bkt_adadelta_update in bkt.h
cudaError_t launch_adadelta(float *p, const float *g, float *eg2, float *edx2, int64_t n, float rho, float eps,
                            float lr, cudaStream_t s);

// ---------------------------------------------------------------------------
// Device buffers of one step (see the step engine in bkt_api.cpp).
constexpr int kMaxLayers = 64;
struct StepBufs {
  float *X;                                   // packed input [NT x in_dim]
  float *Y[kMaxLayers];                       // layer outputs [NT x dirs*H]
  float *Z[2 * kMaxLayers];                   // per layer*dirs+dir: Zx / gates / dz [NT x 4H]
  float *Cst[2 * kMaxLayers];                 // cell states [NT x H]
  float *logit;                               // log-probabilities / dlogit [NT x C]
  float *DXh, *DXl;                           // split dz for dX while the side stream holds AT (or null)
  float *part2;                               // partials of layer 1's narrow weight gradient on the main stream (or null)
  size_t part2_floats;
  float *alpha, *beta;                        // CTC tables, sum_i L_i (2 U_i + 1) each
  float *dY;                                  // dloss/dY of the current layer [NT x dirs*H]
  float *part;                                // split-K partial sums
  size_t part_floats;
  int32_t *tok_t, *tok_r, *prev_tok[2];       // [NT] each
  int32_t *row_ok;                            // [b]
  int32_t *status;                            // device error flags [kStatusWords]
  void *idx_dev;                              // per-step index block
  // split-precision (3xTF32) operands of the fp32 contractions over tokens
  float *AT, *ATl;                            // [max(4H, C) x NTq] transposed dz / dlogit, hi and lo
  float *BTf, *BTl;                           // [dirs*H x NTq] transposed X, h_{t-1} or Y, hi and lo
  float *Lh, *Ll;                             // [NT x Cp] dlogit split, rows padded to Cp = C rounded to 4
  float *Wh, *Wl;                             // [Cp x dirs*H] W_out split (or its transpose)
  float *Woh, *Wol;                           // [C x DHp] W_out split for the logits (made at the step's start)
  float *WoTh, *WoTl;                         // [dirs*H x Cp] W_out transposed and split for dY
  // bf16 GEMM path only (null otherwise); token-major, read by the GEMMs as
  // K-major (projection, dX) or MN-major (weight gradients) operands
  void *Yb[kMaxLayers];                       // [NT x dirs*H] bf16 Y of layers 0 .. L-2
  void *Hs[2 * kMaxLayers];                   // per layer*dirs+dir: [NT x H] bf16 h_{t-1}
  void *dZb[2 * kMaxLayers];                  // per layer*dirs+dir: [NT x 4H] bf16 dz
  float *dbp[kMaxLayers];                     // layers > 0: db partials of the tensor-core BPTT [dirs x ceil(b/16) x 4H]
  void *Wb[2 * kMaxLayers];                   // per layer*dirs+dir (layers > 0): [4H x dirs*H] bf16 W_ih
};

// Records an error message for bkt_last_error() and returns `code`.
int report_error(int code, const char *fmt, ...);

// Runs one training step with every buffer carved out of `scratch`
// (`scratch_bytes` long, 256-byte aligned device memory), allocating
// nothing.  Host-side checks return BKT_EINVAL, including a batch whose
// workspace does not fit.
int step_on_scratch(const bkt_model_cfg *cfg, const bkt_batch *batch, const float *params,
                    float *grads, float *loss, cudaStream_t s, void *scratch, size_t scratch_bytes,
                    int sm_count);

}  // namespace bkt
