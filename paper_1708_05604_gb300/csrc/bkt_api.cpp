// bkt_api.cpp -- host side of libbkt: the bucketing planner (Section III.A of
// arXiv 1708.05604), the step context and the step engine that enqueues the
// CUDA kernels of one training step (Section IV).  Entry points are declared,
// with their contracts, in include/bkt.h.
#include "../../include/bkt.h"

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "bkt_internal.h"
#include "nvtx_range.h"

namespace {

thread_local std::string g_err;

int set_err(int code, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

int vset_err(int code, const char *fmt, va_list ap) {
  char buf[512];
  vsnprintf(buf, sizeof buf, fmt, ap);
  g_err = buf;
  return code;
}

int cuda_err(const char *what, cudaError_t e) {
  return set_err(BKT_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// Planner.
constexpr int64_t kDpInf = int64_t(1) << 62;

uint64_t splitmix64_next(uint64_t &state) {
  state += 0x9E3779B97F4A7C15ULL;
  uint64_t z = state;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

}  // namespace

struct bkt_plan {
  std::vector<int32_t> bounds, order, batch_off, batch_bucket;
  int64_t dp_cost = 0, padded = 0, unpadded = 0;
};

extern "C" int bkt_plan_buckets_ordered(const int32_t *lengths, int64_t n, int32_t Q, int32_t batch,
                                        uint64_t seed, uint64_t epoch, int32_t batch_order, bkt_plan **out) {
  bkt::NvtxRange range("bkt_plan_buckets");
  if (!out) return set_err(BKT_EINVAL, "bkt_plan_buckets: out is NULL");
  if (batch_order < BKT_ORDER_ASCENDING || batch_order > BKT_ORDER_SHUFFLE_BATCHES)
    return set_err(BKT_EINVAL, "bkt_plan_buckets: unknown batch order %d", batch_order);
  *out = nullptr;
  if (!lengths || n < 1) return set_err(BKT_EINVAL, "bkt_plan_buckets: no lengths");
  if (Q < 1 || batch < 1) return set_err(BKT_EINVAL, "bkt_plan_buckets: n_buckets and batch must be >= 1");
  if (n > INT32_MAX - 1) return set_err(BKT_EINVAL, "bkt_plan_buckets: too many sequences");
  int32_t lmax = 0;
  int64_t total = 0;
  for (int64_t i = 0; i < n; ++i) {
    if (lengths[i] < 1) return set_err(BKT_EINVAL, "bkt_plan_buckets: lengths[%lld] = %d < 1", (long long)i, lengths[i]);
    lmax = std::max(lmax, lengths[i]);
    total += lengths[i];
  }
  if (Q > lmax) return set_err(BKT_EINVAL, "bkt_plan_buckets: %d buckets but the longest sequence has length %d", Q, lmax);

  bkt_plan *p = new (std::nothrow) bkt_plan;
  if (!p) return set_err(BKT_ENOMEM, "bkt_plan_buckets: out of host memory");
  try {
    // Histogram f[l] and its prefix sums F[i] = f[0] + ... + f[i]; the
    // charge of a group (j, i] with upper bound i is i * (F[i] - F[j]).
    const int32_t nf = lmax + 1;
    std::vector<int64_t> F(nf, 0);
    for (int64_t i = 0; i < n; ++i) F[lengths[i]] += 1;
    for (int32_t l = 1; l < nf; ++l) F[l] += F[l - 1];
    // dp rows q-1 and q, back-pointers for every q.  The charge
    // w(j, i) = i (F[i] - F[j]) satisfies the quadrangle inequality
    // (w(a,c) + w(b,d) - w(a,d) - w(b,c) = (c - d)(F[b] - F[a]) <= 0 for
    // a <= b <= c <= d), so the largest minimising j of row i is
    // non-decreasing in i and a divide-and-conquer over i finds, for every i,
    // the same minimum and the same largest argmin as the full scan (j
    // descending, strict "<"), in O(Q n log n) instead of O(Q n^2).
    std::vector<int64_t> prev_row(nf, kDpInf), row(nf, kDpInf);
    std::vector<int32_t> back((size_t)(Q + 1) * nf, -1);
    prev_row[0] = 0;
    struct Range {
      int32_t lo, hi, jlo, jhi;
    };
    std::vector<Range> todo;
    for (int32_t q = 1; q <= Q; ++q) {
      std::fill(row.begin(), row.end(), kDpInf);
      int32_t *bq = back.data() + (size_t)q * nf;
      // dp[q-1][j] is finite only for j >= q-1.
      todo.clear();
      if (q < nf) todo.push_back({q, nf - 1, q - 1, nf - 2});
      while (!todo.empty()) {
        const Range r = todo.back();
        todo.pop_back();
        if (r.lo > r.hi) continue;
        const int32_t i = r.lo + (r.hi - r.lo) / 2;
        const int64_t Fi = F[i];
        int64_t best = kDpInf;
        int32_t arg = -1;
        for (int32_t j = std::min(i - 1, r.jhi); j >= std::max(q - 1, r.jlo); --j) {
          const int64_t v = (int64_t)i * (Fi - F[j]) + prev_row[j];
          if (v < best) {  // strict: ties keep the larger j
            best = v;
            arg = j;
          }
        }
        row[i] = best;
        bq[i] = arg;
        const int32_t split = arg >= 0 ? arg : r.jlo;
        todo.push_back({r.lo, i - 1, r.jlo, split});
        todo.push_back({i + 1, r.hi, split, r.jhi});
      }
      std::swap(prev_row, row);
    }
    if (prev_row[lmax] >= kDpInf) {
      delete p;
      return set_err(BKT_EINVAL, "bkt_plan_buckets: infeasible bucket count");
    }
    p->dp_cost = prev_row[lmax];
    p->bounds.assign(Q, 0);
    for (int32_t q = Q, cur = lmax; q >= 1; --q) {
      p->bounds[q - 1] = cur;
      cur = back[(size_t)q * nf + cur];
    }
    // Bucket of every length value, then counting sort by bucket.
    std::vector<int32_t> bucket_of_len(nf, 0);
    for (int32_t q = 0, l = 1; l < nf; ++l) {
      while (l > p->bounds[q]) ++q;
      bucket_of_len[l] = q;
    }
    std::vector<int64_t> start(Q + 1, 0);
    for (int64_t i = 0; i < n; ++i) start[bucket_of_len[lengths[i]] + 1] += 1;
    for (int32_t q = 0; q < Q; ++q) start[q + 1] += start[q];
    p->order.resize(n);
    {
      std::vector<int64_t> fill(start.begin(), start.end() - 1);
      for (int64_t i = 0; i < n; ++i) p->order[fill[bucket_of_len[lengths[i]]]++] = (int32_t)i;
    }
    uint64_t state = seed + (epoch + 1ULL) * 0x9E3779B97F4A7C15ULL;
    for (int32_t q = 0; q < Q; ++q) {
      int32_t *lst = p->order.data() + start[q];
      const int64_t m = start[q + 1] - start[q];
      for (int64_t k = m - 1; k >= 1; --k) {
        const int64_t j = (int64_t)(splitmix64_next(state) % (uint64_t)(k + 1));
        std::swap(lst[k], lst[j]);
      }
    }
    // mini-batches: consecutive chunks of each bucket, buckets ascending
    std::vector<int64_t> cut_s, cut_e;
    std::vector<int32_t> cut_q;
    for (int32_t q = 0; q < Q; ++q) {
      for (int64_t s = start[q]; s < start[q + 1]; s += batch) {
        const int64_t e = std::min<int64_t>(s + batch, start[q + 1]);
        int32_t mx = 0;
        for (int64_t r = s; r < e; ++r) mx = std::max(mx, lengths[p->order[r]]);
        cut_s.push_back(s);
        cut_e.push_back(e);
        cut_q.push_back(q);
        p->padded += (e - s) * (int64_t)mx;
      }
    }
    // emission order of the batches (the bucket-ordering strategies that
    // Section V leaves to future work); the shuffles continue the stream
    const int64_t nb = (int64_t)cut_q.size();
    std::vector<int64_t> seq(nb);
    for (int64_t b = 0; b < nb; ++b) seq[b] = b;
    if (batch_order == BKT_ORDER_DESCENDING || batch_order == BKT_ORDER_SHUFFLE_BUCKETS) {
      std::vector<int32_t> qs(Q);
      for (int32_t q = 0; q < Q; ++q) qs[q] = batch_order == BKT_ORDER_DESCENDING ? Q - 1 - q : q;
      if (batch_order == BKT_ORDER_SHUFFLE_BUCKETS)
        for (int64_t k = Q - 1; k >= 1; --k) {
          const int64_t j = (int64_t)(splitmix64_next(state) % (uint64_t)(k + 1));
          std::swap(qs[k], qs[j]);
        }
      int64_t w = 0;
      for (int32_t qi = 0; qi < Q; ++qi)
        for (int64_t b = 0; b < nb; ++b)
          if (cut_q[b] == qs[qi]) seq[w++] = b;
    } else if (batch_order == BKT_ORDER_SHUFFLE_BATCHES) {
      for (int64_t k = nb - 1; k >= 1; --k) {
        const int64_t j = (int64_t)(splitmix64_next(state) % (uint64_t)(k + 1));
        std::swap(seq[k], seq[j]);
      }
    }
    std::vector<int32_t> emitted(n);
    int64_t pos = 0;
    for (int64_t i = 0; i < nb; ++i) {
      const int64_t b = seq[i];
      p->batch_off.push_back((int32_t)pos);
      p->batch_bucket.push_back(cut_q[b]);
      for (int64_t r = cut_s[b]; r < cut_e[b]; ++r) emitted[pos++] = p->order[r];
    }
    p->order.swap(emitted);
    p->batch_off.push_back((int32_t)n);
    p->unpadded = total;
  } catch (const std::bad_alloc &) {
    delete p;
    return set_err(BKT_ENOMEM, "bkt_plan_buckets: out of host memory");
  }
  *out = p;
  return BKT_OK;
}

extern "C" int bkt_plan_buckets(const int32_t *lengths, int64_t n, int32_t Q, int32_t batch,
                                uint64_t seed, uint64_t epoch, bkt_plan **out) {
  return bkt_plan_buckets_ordered(lengths, n, Q, batch, seed, epoch, BKT_ORDER_ASCENDING, out);
}

extern "C" int bkt_plan_get(const bkt_plan *p, bkt_plan_view *v) {
  if (!p || !v) return set_err(BKT_EINVAL, "bkt_plan_get: NULL argument");
  v->n_buckets = (int32_t)p->bounds.size();
  v->bounds = p->bounds.data();
  v->dp_cost = p->dp_cost;
  v->n_seqs = (int64_t)p->order.size();
  v->order = p->order.data();
  v->n_batches = (int32_t)p->batch_bucket.size();
  v->batch_off = p->batch_off.data();
  v->batch_bucket = p->batch_bucket.data();
  v->padded_timesteps = p->padded;
  v->unpadded_timesteps = p->unpadded;
  return BKT_OK;
}

extern "C" void bkt_plan_free(bkt_plan *p) { delete p; }

extern "C" const char *bkt_last_error(void) { return g_err.c_str(); }

// ---------------------------------------------------------------------------
// Parameters.
namespace {

bool cfg_ok(const bkt_model_cfg *c) {
  return c && c->n_layers >= 1 && c->n_layers <= bkt::kMaxLayers &&
         (c->bidirectional == 0 || c->bidirectional == 1) && c->in_dim >= 1 && c->in_dim <= 16 &&
         c->hidden >= 1 && c->hidden <= 2048 && c->n_classes >= 2 && c->n_classes <= 128 && c->blank >= 0 &&
         c->blank < c->n_classes && (c->gemm_precision == BKT_GEMM_FP32 || c->gemm_precision == BKT_GEMM_BF16);
}

struct Layout {
  int dirs, H, C, L, D0;
  int64_t w_ih[2 * bkt::kMaxLayers];  // offset of W_ih of (layer, dir) at [l*dirs + d]
  int64_t w_out, b_out, total;
  int D(int l) const { return l == 0 ? D0 : dirs * H; }
  int64_t w_hh(int l, int d) const { return w_ih[l * dirs + d] + (int64_t)4 * H * D(l); }
  int64_t bias(int l, int d) const { return w_hh(l, d) + (int64_t)4 * H * H; }
  int64_t stride(int l) const { return (int64_t)4 * H * (D(l) + H + 1); }
};

Layout make_layout(const bkt_model_cfg *c) {
  Layout lo;
  lo.dirs = c->bidirectional ? 2 : 1;
  lo.H = c->hidden;
  lo.C = c->n_classes;
  lo.L = c->n_layers;
  lo.D0 = c->in_dim;
  int64_t off = 0;
  for (int l = 0; l < lo.L; ++l)
    for (int d = 0; d < lo.dirs; ++d) {
      lo.w_ih[l * lo.dirs + d] = off;
      off += lo.stride(l);
    }
  lo.w_out = off;
  off += (int64_t)lo.C * lo.dirs * lo.H;
  lo.b_out = off;
  off += lo.C;
  lo.total = off;
  return lo;
}

// Layout of the per-step index block (same in staging and on the device).
struct IdxLayout {
  size_t row_len, row_lab_len, row_orig, row_xoff, row_lab_off, row_ctc_off, tok_off, bytes;
};
IdxLayout idx_layout(int32_t b, int64_t T) {
  IdxLayout L;
  size_t o = 0;
  auto take = [&](size_t n) {
    size_t r = o;
    o += (n + 15) & ~size_t(15);
    return r;
  };
  L.row_len = take(4 * (size_t)b);
  L.row_lab_len = take(4 * (size_t)b);
  L.row_orig = take(4 * (size_t)b);
  L.row_xoff = take(8 * (size_t)b);
  L.row_lab_off = take(8 * (size_t)b);
  L.row_ctc_off = take(8 * (size_t)b);
  L.tok_off = take(4 * (size_t)(T + 1));
  L.bytes = o;
  return L;
}

// Host checks of one batch against capacities.  On success: tokens, the
// largest 2U+1 and the CTC table cells sum_i L_i (2 U_i + 1).
int check_batch(const bkt_batch *bt, int64_t max_tokens, int32_t max_batch, int32_t max_label_len,
                int64_t *n_tok, int32_t *S_max, int64_t *ctc_cells) {
  const int32_t b = bt->n_seq;
  if (b < 1 || b > max_batch) return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: n_seq %d outside 1..%d", b, max_batch);
  if (!bt->lengths || !bt->x_offsets || !bt->label_lengths || !bt->label_offsets || !bt->x || !bt->labels)
    return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: NULL batch array");
  int64_t nt = 0, cells = 0;
  int32_t sm = 1;
  for (int32_t i = 0; i < b; ++i) {
    if (bt->lengths[i] < 1) return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: lengths[%d] = %d < 1", i, bt->lengths[i]);
    if (bt->label_lengths[i] < 0 || bt->label_lengths[i] > max_label_len)
      return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: label_lengths[%d] = %d outside 0..%d", i, bt->label_lengths[i],
                     max_label_len);
    if (bt->x_offsets[i] < 0 || bt->label_offsets[i] < 0)
      return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: negative offset for sequence %d", i);
    nt += bt->lengths[i];
    sm = std::max(sm, 2 * bt->label_lengths[i] + 1);
    cells += (int64_t)bt->lengths[i] * (2 * bt->label_lengths[i] + 1);
  }
  if (nt > max_tokens)
    return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: %lld tokens exceed the capacity %lld", (long long)nt,
                   (long long)max_tokens);
  *n_tok = nt;
  *S_max = sm;
  *ctc_cells = cells;
  return BKT_OK;
}

// a4, host part: with `perm` the batch's stable longest-first order, fills
// the index block at `st` and returns its device view at `dev`.
bkt::DevIdx fill_index_block(const bkt_batch *bt, const int32_t *perm, int32_t T, int64_t n_tok, int32_t S_max,
                             const IdxLayout &il, char *st, char *dev, int32_t *tok_t, int32_t *tok_r) {
  const int32_t b = bt->n_seq;
  int32_t *row_len = (int32_t *)(st + il.row_len), *row_lab_len = (int32_t *)(st + il.row_lab_len),
          *row_orig = (int32_t *)(st + il.row_orig), *tok_off = (int32_t *)(st + il.tok_off);
  int64_t *row_xoff = (int64_t *)(st + il.row_xoff), *row_lab_off = (int64_t *)(st + il.row_lab_off),
          *row_ctc_off = (int64_t *)(st + il.row_ctc_off);
  int64_t ctc_off = 0;
  for (int32_t r = 0; r < b; ++r) {
    const int32_t i = perm[r];
    row_len[r] = bt->lengths[i];
    row_lab_len[r] = bt->label_lengths[i];
    row_orig[r] = i;
    row_xoff[r] = bt->x_offsets[i];
    row_lab_off[r] = bt->label_offsets[i];
    row_ctc_off[r] = ctc_off;
    ctc_off += (int64_t)bt->lengths[i] * (2 * bt->label_lengths[i] + 1);
  }
  int32_t active = b, acc = 0;
  for (int32_t t = 0; t < T; ++t) {
    while (active > 0 && row_len[active - 1] <= t) --active;
    tok_off[t] = acc;
    acc += active;
  }
  tok_off[T] = acc;
  bkt::DevIdx ix;
  ix.b = b;
  ix.T = T;
  ix.n_tok = (int32_t)n_tok;
  ix.S_max = S_max;
  ix.row_len = (const int32_t *)(dev + il.row_len);
  ix.row_lab_len = (const int32_t *)(dev + il.row_lab_len);
  ix.row_orig = (const int32_t *)(dev + il.row_orig);
  ix.row_xoff = (const int64_t *)(dev + il.row_xoff);
  ix.row_lab_off = (const int64_t *)(dev + il.row_lab_off);
  ix.row_ctc_off = (const int64_t *)(dev + il.row_ctc_off);
  ix.tok_off = (const int32_t *)(dev + il.tok_off);
  ix.tok_t = tok_t;
  ix.tok_r = tok_r;
  return ix;
}

struct Launch {
  bkt::KernelTimer *timer;
  cudaStream_t s;
  const char *failed = nullptr;
  cudaError_t err = cudaSuccess;
  template <typename F>
  bool run(const char *name, const bkt::Work &wk, F &&f) {
    if (failed) return false;
    bkt::NvtxRange range(name);
    if (timer) timer->begin(name, wk, s);
    cudaError_t e = f();
    if (timer) timer->end(s);
    if (e != cudaSuccess) {
      failed = name;
      err = e;
      return false;
    }
    return true;
  }
};

// Algorithmic work of a launch (bkt_kernel_time): contraction flops,
// minimum DRAM bytes, serial time steps.
bkt::Work flops_w(double f, int64_t steps = 0) {
  bkt::Work w;
  w.flops = f;
  w.steps = steps;
  return w;
}
bkt::Work bytes_w(double b, int64_t steps = 0) {
  bkt::Work w;
  w.bytes = b;
  w.steps = steps;
  return w;
}
// a GEMM of 2 M N K flops; an element-wise pass over R x C values reading
// `rb` and writing `wb` bytes per value
bkt::Work gemm_w(double M, double N, double K) { return flops_w(2.0 * M * N * K); }
bkt::Work pass_w(double R, double C, double rb, double wb) { return bytes_w(R * C * (rb + wb)); }

// Largest M x N block a token reduction writes: [W_out | b_out] or
// [W_ih | W_hh | b] of one layer and direction.
size_t max_reduce_block(const Layout &lo) {
  const size_t DH = (size_t)lo.dirs * lo.H, H = lo.H;
  const size_t Dm = std::max<size_t>(DH, (size_t)lo.D0);
  return std::max<size_t>((size_t)lo.C * (DH + 1), 4 * H * (Dm + H + 1));
}

// Enqueues every kernel of one step (a4 gather .. a12) on `s`.
// `side` (with its two events) is an optional second stream: the output
// layer's weight gradient runs there, overlapping dY and the top layer's BPTT.
int enqueue_kernels(const bkt_model_cfg &cfg, const Layout &lo, const bkt::StepBufs &w, const bkt::RecGeom *geom,
                    const bkt::DevIdx &ix, const bkt_batch *bt, const float *params, float *grads, float *loss,
                    cudaStream_t s, bkt::KernelTimer *timer, int sm_count, cudaStream_t side = nullptr,
                    cudaEvent_t fork_ev = nullptr, cudaEvent_t join_ev = nullptr, bkt::WaitFaults wf = {}) {
  const int H = lo.H, dirs = lo.dirs, DH = dirs * H, C = lo.C, NT = ix.n_tok;
  const bool bf16 = cfg.gemm_precision == BKT_GEMM_BF16;
  Launch L{timer, s};
  Launch Ls{timer, side ? side : s};

  // ---- W_out in the two split forms the output layer needs (rows for the
  // logits, transposed for dY); they depend on the parameters only, so with
  // a side stream they run beside the forward pass
  const int DHp = (DH + 3) & ~3;  // split rows padded to 16 bytes for TMA
  const int Cp = (C + 3) & ~3;
  if (side) {
    cudaError_t e = cudaEventRecord(fork_ev, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(side, fork_ev, 0);
    if (e != cudaSuccess) return cuda_err("fork to the side stream", e);
  }
  Ls.run("split_rows", pass_w(C, DH, 4, 8),
         [&] { return bkt::launch_split_rows(params + lo.w_out, DH, C, DH, w.Woh, w.Wol, DHp, Ls.s); });
  Ls.run("transpose_split", pass_w(C, DH, 4, 8), [&] {
    return bkt::launch_transpose_split(params + lo.w_out, DH, nullptr, C, DH, w.WoTh, w.WoTl, Cp, Ls.s);
  });
  if (side) {
    cudaError_t e = cudaEventRecord(join_ev, side);
    if (e != cudaSuccess) return cuda_err("record on the side stream", e);
  }

  // ---- a4: packed time-major input
  L.run("layout_gather", bytes_w((double)NT * (8.0 * lo.D0 + 16.0)), [&] { return bkt::launch_layout(ix, bt->x, lo.D0, w.X, w.tok_t, w.tok_r, w.prev_tok, s); });

  // ---- forward, layer by layer
  for (int l = 0; l < lo.L; ++l) {
    bkt::NvtxRange layer_range("forward layer");
    float *Zl[2] = {w.Z[l * dirs], dirs > 1 ? w.Z[l * dirs + 1] : nullptr};
    if (l == 0) {
      // a5, narrow input: both directions in one launch
      L.run("proj_narrow", bytes_w(4.0 * NT * (lo.D0 + 4.0 * H * dirs)), [&] {
        return bkt::launch_proj_narrow(w.X, NT, lo.D0, params, lo.w_ih[0], lo.stride(0), H, dirs, Zl, s);
      });
    } else if (bf16) {
      // a5 on the tensor cores: Zx = bf16(Y_{l-1}) bf16(W_ih)^T + b, fp32
      // accumulation; bf16(Y_{l-1}) was written by layer l-1's recurrent
      // kernel (or cast after it); bf16(W_ih) is kept for dX
      for (int d = 0; d < dirs; ++d) {
        void *Wb = w.Wb[l * dirs + d];
        L.run("cast_bf16", pass_w(4.0 * H, DH, 4, 2), [&] {
          return bkt::launch_cast_bf16(params + lo.w_ih[l * dirs + d], DH, 4 * H, DH, Wb, DH, s);
        });
        bkt::TcGemmArgs g{};
        g.M = NT;
        g.N = 4 * H;
        g.K = DH;
        g.A = w.Yb[l - 1];
        g.lda = DH;
        g.B = Wb;
        g.ldb = DH;
        g.D = Zl[d];
        g.ldd = 4 * H;
        g.bias = params + lo.bias(l, d);
        g.err = w.status;
        g.wf = wf;
        L.run("gemm_tc", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_bf16_tc(g, s); });
      }
    } else {
      // a5 in fp32 on the tensor cores (3xTF32): Zx = Y_{l-1} W_ih^T + b; both
      // operands are K-contiguous, split into hi + lo rows padded to 16 bytes
      const int DHq = (DH + 3) & ~3;
      L.run("split_rows", pass_w(NT, DH, 4, 8),
            [&] { return bkt::launch_split_rows(w.Y[l - 1], DH, NT, DH, w.AT, w.ATl, DHq, s); });
      for (int d = 0; d < dirs; ++d) {
        L.run("split_rows", pass_w(4.0 * H, DH, 4, 8), [&] {
          return bkt::launch_split_rows(params + lo.w_ih[l * dirs + d], DH, 4 * H, DH, w.Wh, w.Wl, DHq, s);
        });
        bkt::TcGemmArgs g{};
        g.M = NT;
        g.N = 4 * H;
        g.K = DH;
        g.A = w.AT;
        g.lda = DHq;
        g.B = w.Wh;
        g.ldb = DHq;
        g.D = Zl[d];
        g.ldd = 4 * H;
        g.bias = params + lo.bias(l, d);
        g.err = w.status;
        g.wf = wf;
        L.run("gemm_tf32x3", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_tf32x3_tc(g, w.ATl, w.Wl, s); });
      }
    }
    bkt::RecArgs ra{};
    ra.ix = ix;
    ra.H = H;
    ra.dirs = dirs;
    for (int d = 0; d < dirs; ++d) {
      ra.Z[d] = Zl[d];
      ra.Cst[d] = w.Cst[l * dirs + d];
      ra.Whh[d] = params + lo.w_hh(l, d);
    }
    ra.Y = w.Y[l];
    ra.status = w.status;
    ra.wf = wf;
    if (bf16) {  // the bf16 copies the contractions read (written by the kernel when it can)
      ra.Yb = l + 1 < lo.L ? w.Yb[l] : nullptr;
      for (int d = 0; d < dirs; ++d) ra.Hs[d] = w.Hs[l * dirs + d];
      // below the top layer only the bf16 copies are read when the kernel
      // writes them (projection, dW_ih and dW_hh): no fp32 h
      if (l + 1 < lo.L && bkt::rec_writes_bf16(geom[l])) ra.Y = nullptr;
    }
    L.run("lstm_fwd", flops_w(8.0 * H * H * (double)NT * dirs, ix.T), [&] { return bkt::launch_lstm_fwd(ra, geom[l], s); });
    if (bf16 && l + 1 < lo.L && !bkt::rec_writes_bf16(geom[l]))
      L.run("cast_bf16", pass_w(NT, DH, 4, 2), [&] { return bkt::launch_cast_bf16(w.Y[l], DH, NT, DH, w.Yb[l], DH, s); });
  }

  // ---- a7: output layer and log-softmax
  bkt::NvtxRange output_range("output layer and CTC");
  // logits = Y W_out^T + b_out on the tensor cores (3xTF32; both operands are
  // already K-contiguous, so they are split without transposing); the
  // GEMM's epilogue holds whole rows (C <= 128 columns in one tile) and
  // writes their log-softmax
  float *Ytop = w.Y[lo.L - 1];
  L.run("split_rows", pass_w(NT, DH, 4, 8), [&] { return bkt::launch_split_rows(Ytop, DH, NT, DH, w.BTf, w.BTl, DHp, s); });
  if (side) {
    cudaError_t e = cudaStreamWaitEvent(s, join_ev, 0);  // the W_out splits
    if (e != cudaSuccess) return cuda_err("wait for the side stream", e);
  }
  {
    bkt::TcGemmArgs g{};
    g.M = NT;
    g.N = C;
    g.K = DH;
    g.A = w.BTf;
    g.lda = DHp;
    g.B = w.Woh;
    g.ldb = DHp;
    g.D = w.logit;
    g.ldd = C;
    g.bias = params + lo.b_out;
    g.logsoftmax = 1;
    g.err = w.status;
    g.wf = wf;
    L.run("gemm_tf32x3", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_tf32x3_tc(g, w.BTl, w.Wol, s); });
  }
  // ---- a8, a9: CTC
  L.run("ctc_tables", bytes_w(16.0 * (double)ix.n_cells, ix.T), [&] {
    return bkt::launch_ctc_tables(ix, w.logit, C, cfg.blank, bt->labels, w.alpha, w.beta, loss, w.row_ok, w.status, s);
  });
  L.run("ctc_grad", bytes_w(8.0 * (double)ix.n_cells + 8.0 * NT * C + 8.0 * NT * Cp), [&] {  // dlogit in place, and its split for dY
    return bkt::launch_ctc_grad(ix, w.logit, C, cfg.blank, bt->labels, w.alpha, w.beta, w.row_ok, w.Lh, w.Ll, Cp, s);
  });

  // ---- a10: output layer backward
  // fp32 contractions over tokens on the tensor cores (3xTF32).  Operands
  // with 16-byte aligned rows are read token-major by the fused kernel
  // (split and swizzled while loading); others (dlogit: C = 81 columns) are
  // transposed and split first for the TMA-fed GEMM.  Measured on GB300:
  // dW_hh at H = 128, 32 us fused against 66 us; at H = 512, 1.22 ms
  // against 1.31 ms.
  const int NTq = (NT + 7) & ~7;
  // the transposed split of A left in AT by the last fallback call: dW_ih of
  // a layer above the first reuses the one its dW_hh made (nothing else
  // writes AT between them)
  const float *at_src = nullptr;
  auto tn_reduce_on = [&](Launch &X, const float *A, int64_t lda, int M, const float *B, int64_t ldb,
                          const int32_t *gather, int N, float *out) {
    const bool fused = ((lda | ldb | M | N) & 3) == 0 &&
                       ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B)) & 15) == 0;
    if (fused) {
      bkt::TnGemmArgs g{};
      g.M = M;
      g.N = N;
      g.K = NT;
      g.A = A;
      g.lda = lda;
      g.B = B;
      g.ldb = ldb;
      g.gather = gather;
      g.P = w.part;
      g.splits = bkt::tf32x3_tn_splits(M, N, NT, sm_count, w.part_floats);
      g.err = w.status;
      g.wf = wf;
      X.run("gemm_tf32x3_tn", gemm_w(M, N, NT), [&] { return bkt::launch_gemm_tf32x3_tn(g, X.s); });
      X.run("splitk_sum", pass_w(M, N, 4.0 * g.splits, 4),
            [&] { return bkt::launch_splitk_sum(w.part, g.splits, M, N, out, X.s); });
      return;
    }
    if (at_src != A) {
      X.run("transpose_split", pass_w(NT, M, 4, 8),
            [&] { return bkt::launch_transpose_split(A, lda, nullptr, NT, M, w.AT, w.ATl, NTq, X.s); });
      at_src = A;
    }
    X.run("transpose_split", pass_w(NT, N, 4, 8),
          [&] { return bkt::launch_transpose_split(B, ldb, gather, NT, N, w.BTf, w.BTl, NTq, X.s); });
    bkt::TcGemmArgs g{};
    g.M = M;
    g.N = N;
    g.K = NT;
    g.A = w.AT;
    g.lda = NTq;
    g.B = w.BTf;
    g.ldb = NTq;
    g.P = w.part;
    g.splits = bkt::tf32x3_splits(M, N, NT, sm_count, w.part_floats);
    g.err = w.status;
    g.wf = wf;
    X.run("gemm_tf32x3", gemm_w(M, N, NT), [&] { return bkt::launch_gemm_tf32x3_tc(g, w.ATl, w.BTl, X.s); });
    X.run("splitk_sum", pass_w(M, N, 4.0 * g.splits, 4),
          [&] { return bkt::launch_splitk_sum(w.part, g.splits, M, N, out, X.s); });
  };
  auto bias_sum_on = [&](Launch &X, const float *A, int64_t lda, int M, float *out) {
    const int splits = bkt::colsum_splits(NT, M, w.part_floats);
    X.run("colsum", bytes_w(4.0 * NT * M + 4.0 * splits * M),
          [&] { return bkt::launch_colsum(A, lda, NT, M, w.part, splits, X.s); });
    X.run("splitk_sum", pass_w(1, M, 4.0 * splits, 4),
          [&] { return bkt::launch_splitk_sum(w.part, splits, 1, M, out, X.s); });
  };
  // [dW_out | db_out] = dlogit^T [Y | 1]; with a side stream it overlaps dY
  // and the top layer's BPTT (the side stream runs all weight gradients in
  // order and is joined at the end of the step)
  if (side) {
    cudaError_t e = cudaEventRecord(fork_ev, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(side, fork_ev, 0);
    if (e != cudaSuccess) return cuda_err("fork to the side stream", e);
  }
  tn_reduce_on(Ls, w.logit, C, C, Ytop, DH, nullptr, DH, grads + lo.w_out);
  bias_sum_on(Ls, w.logit, C, C, grads + lo.b_out);
  {
    // dY = dlogit W_out on the tensor cores: dlogit split by the CTC gradient
    // (rows padded to a multiple of 4 floats, TMA strides), W_out split
    // transposed at the step's start
    bkt::TcGemmArgs g{};
    g.M = NT;
    g.N = DH;
    g.K = C;
    g.A = w.Lh;
    g.lda = Cp;
    g.B = w.WoTh;
    g.ldb = Cp;
    g.D = w.dY;
    g.ldd = DH;
    g.err = w.status;
    g.wf = wf;
    L.run("gemm_tf32x3", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_tf32x3_tc(g, w.Ll, w.WoTl, s); });
  }

  output_range.end();
  // ---- a11, a12: BPTT and weight gradients, top layer first.  With a side
  // stream, a layer's weight gradients run there (after its BPTT) while the
  // main stream goes on with dX and the BPTT of the layer below; the side
  // stream's scratch (AT, BT, part) is its own, dX uses separate buffers.
  auto fork_to_side = [&]() -> int {
    if (!side) return BKT_OK;
    cudaError_t e = cudaEventRecord(fork_ev, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(side, fork_ev, 0);
    return e == cudaSuccess ? BKT_OK : cuda_err("fork to the side stream", e);
  };
  for (int l = lo.L - 1; l >= 0; --l) {
    bkt::NvtxRange layer_range("BPTT layer");
    bkt::RecArgs ra{};
    ra.ix = ix;
    ra.H = H;
    ra.dirs = dirs;
    for (int d = 0; d < dirs; ++d) {
      ra.Z[d] = w.Z[l * dirs + d];
      ra.Cst[d] = w.Cst[l * dirs + d];
      ra.Whh[d] = params + lo.w_hh(l, d);
    }
    ra.Y = w.Y[l];
    ra.status = w.status;
    ra.dY = w.dY;
    ra.wf = wf;
    const bool fused_bf16 = bkt::rec_writes_bf16(geom[l]);
    if (bf16)
      for (int d = 0; d < dirs; ++d) ra.dZb[d] = w.dZb[l * dirs + d];
    // tensor-core BPTT above layer 1: db as per-cluster partials, and dz only
    // in bf16 (nothing else reads the fp32 dz there)
    const bool tc_db = bf16 && l > 0 && geom[l].mode == 3 && w.dbp[l];
    if (tc_db) {
      ra.dbp = w.dbp[l];
      ra.no_dz32 = 1;
    }
    L.run("lstm_bwd", flops_w(8.0 * H * H * (double)NT * dirs, ix.T), [&] { return bkt::launch_lstm_bwd(ra, geom[l], s); });
    if (bf16 && !fused_bf16)
      for (int d = 0; d < dirs; ++d)
        L.run("cast_bf16", pass_w(NT, 4.0 * H, 4, 2), [&] {
          return bkt::launch_cast_bf16(w.Z[l * dirs + d], 4 * H, NT, 4 * H, w.dZb[l * dirs + d], 4 * H, s);
        });
    if (int rc = fork_to_side()) return rc;
    Launch &X = Ls;  // the weight gradients of layer l
    const int D = lo.D(l);
    const float *Xl = (l == 0) ? w.X : w.Y[l - 1];
    // layer 1's narrow [dW_ih | db] goes to the main stream (own partials)
    // when it has nothing else left, beside the side stream's dW_hh work
    const bool narrow_main = side && l == 0 && w.part2;
    auto narrow_on = [&](const float *dZ, float *ow, float *ob) {
      Launch &Y = narrow_main ? L : X;
      float *P = narrow_main ? w.part2 : w.part;
      const size_t PF = narrow_main ? w.part2_floats : w.part_floats;
      Y.run("narrow_wgrad", bytes_w(4.0 * NT * (4.0 * H + D)), [&] {
        return bkt::launch_narrow_wgrad(dZ, 4 * H, 4 * H, Xl, D, NT, P, PF, sm_count, ow, ob, Y.s);
      });
    };
    if (bf16) {
      // token-axis contractions on the tensor cores, reading the token-major
      // bf16 copies as MN-major tiles (no transposes): A = dz [NT x 4H]
      auto tc_reduce = [&](const void *A, const void *B, int N, float *out) {
        bkt::TcGemmArgs g{};
        g.M = 4 * H;
        g.N = N;
        g.K = NT;
        g.A = A;
        g.lda = 4 * H;
        g.a_mn = 1;
        g.B = B;
        g.ldb = N;
        g.b_mn = 1;
        g.P = w.part;
        g.splits = bkt::tc_splits(g.M, g.N, NT, sm_count, w.part_floats);
        g.err = w.status;
        g.wf = wf;
        X.run("gemm_tc", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_bf16_tc(g, X.s); });
        X.run("splitk_sum", pass_w(g.M, g.N, 4.0 * g.splits, 4),
              [&] { return bkt::launch_splitk_sum(w.part, g.splits, g.M, g.N, out, X.s); });
      };
      for (int d = 0; d < dirs; ++d) {
        const float *dZ = w.Z[l * dirs + d];
        void *dZb = w.dZb[l * dirs + d], *Hs = w.Hs[l * dirs + d];
        // dW_hh = dz^T h_{t-1} (bf16 h_{t-1}: from the recurrent kernel, or
        // gathered here through the previous-token index)
        if (!fused_bf16)
          X.run("cast_bf16", pass_w(NT, H, 4, 2), [&] {
            return bkt::launch_gather_cast_bf16(w.Y[l] + d * H, DH, w.prev_tok[d], NT, H, Hs, H, X.s);
          });
        tc_reduce(dZb, Hs, H, grads + lo.w_hh(l, d));
        if (l == 0) {
          // narrow input: [dW_ih | db] = dz^T [X | 1] in fp32
          narrow_on(dZ, grads + lo.w_ih[l * dirs + d], grads + lo.bias(l, d));
        } else {
          tc_reduce(dZb, w.Yb[l - 1], D, grads + lo.w_ih[l * dirs + d]);
          if (tc_db) {
            const int ncl = bkt::tc_clusters_per_dir(ix.b, dirs, geom[l].bc);
            X.run("splitk_sum", pass_w(1, 4 * H, 4.0 * ncl, 4), [&] {
              return bkt::launch_splitk_sum(w.dbp[l] + (size_t)d * ncl * 4 * H, ncl, 1, 4 * H, grads + lo.bias(l, d), X.s);
            });
          } else {
            bias_sum_on(X, dZ, 4 * H, 4 * H, grads + lo.bias(l, d));
          }
        }
      }
    } else {
      for (int d = 0; d < dirs; ++d) {
        // dW_hh = dz^T h_{t-1}; h_{t-1} of token (t, r) is the row's previous
        // token in its direction (zeros at the start)
        const float *dZ = w.Z[l * dirs + d];
        tn_reduce_on(X, dZ, 4 * H, 4 * H, w.Y[l] + d * H, DH, w.prev_tok[d], H, grads + lo.w_hh(l, d));
        if (l == 0) {
          // narrow input: [dW_ih | db] = dz^T [X | 1] streamed over dz
          narrow_on(dZ, grads + lo.w_ih[l * dirs + d], grads + lo.bias(l, d));
        } else {
          tn_reduce_on(X, dZ, 4 * H, 4 * H, Xl, D, nullptr, D, grads + lo.w_ih[l * dirs + d]);
          bias_sum_on(X, dZ, 4 * H, 4 * H, grads + lo.bias(l, d));
        }
      }
    }
    if (l > 0 && bf16) {
      // dX = sum_d dz_d W_ih,d on the tensor cores as one contraction over
      // both directions' 4H (bf16 W_ih as cast for the projection, read
      // MN-major): no second pass over dY
      bkt::TcGemmArgs g{};
      g.M = NT;
      g.N = DH;
      g.K = 4 * H;
      g.A = w.dZb[l * dirs];
      g.lda = 4 * H;
      g.B = w.Wb[l * dirs];
      g.ldb = DH;
      g.b_mn = 1;
      if (dirs == 2) {
        g.A2 = w.dZb[l * dirs + 1];
        g.B2 = w.Wb[l * dirs + 1];
        g.K2 = 4 * H;
      }
      g.D = w.dY;
      g.ldd = DH;
      g.err = w.status;
      g.wf = wf;
      L.run("gemm_tc", gemm_w(g.M, g.N, (double)g.K + g.K2), [&] { return bkt::launch_gemm_bf16_tc(g, s); });
    } else if (l > 0) {
      // dX = dz W_ih in fp32 on the tensor cores (3xTF32): dz rows are
      // K-contiguous already, W_ih is transposed while it is split
      float *dxa = w.DXh ? w.DXh : w.AT, *dxl = w.DXl ? w.DXl : w.ATl;
      if (side && !w.DXh) return set_err(BKT_EINVAL, "internal: dX buffers missing for the side stream");
      if (dxa == w.AT) at_src = nullptr;  // AT is overwritten here
      for (int d = 0; d < dirs; ++d) {
        L.run("split_rows", pass_w(NT, 4.0 * H, 4, 8), [&] {
          return bkt::launch_split_rows(w.Z[l * dirs + d], 4 * H, NT, 4 * H, dxa, dxl, 4 * H, s);
        });
        L.run("transpose_split", pass_w(4.0 * H, DH, 4, 8), [&] {
          return bkt::launch_transpose_split(params + lo.w_ih[l * dirs + d], DH, nullptr, 4 * H, DH, w.Wh, w.Wl,
                                             4 * H, s);
        });
        bkt::TcGemmArgs g{};
        g.M = NT;
        g.N = DH;
        g.K = 4 * H;
        g.A = dxa;
        g.lda = 4 * H;
        g.B = w.Wh;
        g.ldb = 4 * H;
        g.D = w.dY;
        g.ldd = DH;
        g.accumulate = d > 0;
        g.err = w.status;
        g.wf = wf;
        L.run("gemm_tf32x3", gemm_w(g.M, g.N, g.K), [&] { return bkt::launch_gemm_tf32x3_tc(g, dxl, w.Wl, s); });
      }
    }
  }
  if (side) {  // every gradient is written before the step's work on `s` ends
    cudaError_t e = cudaEventRecord(join_ev, side);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, join_ev, 0);
    if (e != cudaSuccess) return cuda_err("join the side stream", e);
  }
  if (L.failed) return cuda_err(L.failed, L.err);
  if (Ls.failed) return cuda_err(Ls.failed, Ls.err);
  return BKT_OK;
}

}  // namespace

extern "C" int64_t bkt_param_count(const bkt_model_cfg *cfg) {
  if (!cfg_ok(cfg)) return 0;
  return make_layout(cfg).total;
}

// ---------------------------------------------------------------------------
// Context.
namespace {

struct EventTimer : bkt::KernelTimer {
  struct Rec {
    const char *name;
    bkt::Work work;
    cudaEvent_t a, b;
  };
  struct Total {
    const char *name;
    int64_t launches;
    double ms;
    double flops, bytes;
    int64_t steps;
  };
  std::vector<Rec> pending;
  std::vector<cudaEvent_t> pool;
  std::vector<Total> totals;  // first-seen order; names are static strings
  bool on = false;
  cudaEvent_t get() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  void begin(const char *name, const bkt::Work &wk, cudaStream_t s) override {
    if (!on) return;
    if (pending.size() >= 32768) fold();
    Rec r{name, wk, get(), get()};
    cudaEventRecord(r.a, s);
    pending.push_back(r);
  }
  void end(cudaStream_t s) override {
    if (!on || pending.empty()) return;
    cudaEventRecord(pending.back().b, s);
  }
  void fold() {
    for (auto &r : pending) {
      float ms = 0.f;
      cudaEventSynchronize(r.b);
      cudaEventElapsedTime(&ms, r.a, r.b);
      Total *t = nullptr;
      for (auto &x : totals)
        if (std::strcmp(x.name, r.name) == 0) t = &x;
      if (!t) {
        totals.push_back(Total{r.name, 0, 0.0, 0.0, 0.0, 0});
        t = &totals.back();
      }
      t->launches += 1;
      t->ms += ms;
      t->flops += r.work.flops;
      t->bytes += r.work.bytes;
      t->steps += r.work.steps;
      pool.push_back(r.a);
      pool.push_back(r.b);
    }
    pending.clear();
  }
  ~EventTimer() override {
    for (auto &r : pending) {
      cudaEventDestroy(r.a);
      cudaEventDestroy(r.b);
    }
    for (auto e : pool) cudaEventDestroy(e);
  }
};

constexpr int kStageSlots = 4;

}  // namespace

struct bkt_ctx {
  bkt_model_cfg cfg;
  Layout lo;
  int64_t max_tokens;
  int32_t max_batch, max_label_len, S_cap;
  int device = 0, sm_count = 0;
  std::vector<void *> allocs;
  bkt::StepBufs w{};
  size_t idx_bytes = 0;
  // pinned staging ring for the per-step index block
  void *stage = nullptr;
  cudaEvent_t stage_ev[kStageSlots] = {};
  bool stage_used[kStageSlots] = {};
  int stage_next = 0;
  cudaStream_t last_stream = nullptr;
  cudaStream_t side = nullptr;  // output-layer weight gradient overlaps BPTT here
  cudaEvent_t fork_ev = nullptr, join_ev = nullptr;
  EventTimer timer;
  bkt::WaitFaults wf{};  // failure-detection hooks (off)
  bkt::RecGeom geom[bkt::kMaxLayers] = {};

  ~bkt_ctx() {
    if (fork_ev) cudaEventDestroy(fork_ev);
    if (join_ev) cudaEventDestroy(join_ev);
    if (side) cudaStreamDestroy(side);
    for (int i = 0; i < kStageSlots; ++i)
      if (stage_ev[i]) cudaEventDestroy(stage_ev[i]);
    if (stage) cudaFreeHost(stage);
    for (void *p : allocs) cudaFree(p);
  }
  template <typename T>
  cudaError_t alloc(T **p, size_t count) {
    void *q = nullptr;
    cudaError_t e = cudaMalloc(&q, std::max<size_t>(count, 1) * sizeof(T));
    if (e == cudaSuccess) {
      allocs.push_back(q);
      *p = (T *)q;
    }
    return e;
  }
};

extern "C" int bkt_ctx_create(const bkt_model_cfg *cfg, int64_t max_tokens, int32_t max_batch,
                              int32_t max_label_len, bkt_ctx **out) {
  if (!out) return set_err(BKT_EINVAL, "bkt_ctx_create: out is NULL");
  *out = nullptr;
  if (!cfg_ok(cfg)) return set_err(BKT_EINVAL, "bkt_ctx_create: invalid model cfg");
  if (max_tokens < 1 || max_tokens > (int64_t)INT32_MAX / 4 || max_batch < 1 || max_batch > 4096 ||
      max_label_len < 0 || max_label_len > 4096)
    return set_err(BKT_EINVAL, "bkt_ctx_create: capacity out of range");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_err("cudaGetDevice", e);
  bkt_ctx *c = new (std::nothrow) bkt_ctx;
  if (!c) return set_err(BKT_ENOMEM, "bkt_ctx_create: out of host memory");
  c->cfg = *cfg;
  c->lo = make_layout(cfg);
  c->max_tokens = max_tokens;
  c->max_batch = max_batch;
  c->max_label_len = max_label_len;
  c->S_cap = 2 * max_label_len + 1;
  c->device = dev;
  e = cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) {
    delete c;
    return cuda_err("cudaDeviceGetAttribute", e);
  }
  const Layout &lo = c->lo;
  bkt::StepBufs &w = c->w;
  const size_t NT = (size_t)max_tokens, DH = (size_t)lo.dirs * lo.H, H = lo.H;
#define BKT_ALLOC(ptr, n)                                                                       \
  do {                                                                                          \
    const size_t bytes_ = (size_t)(n) * sizeof(*(ptr));                                         \
    e = c->alloc(&(ptr), (n));                                                                  \
    if (e != cudaSuccess) {                                                                     \
      delete c;                                                                                 \
      return set_err(BKT_ENOMEM, "bkt_ctx_create: cudaMalloc of %zu bytes failed: %s", bytes_, \
                     cudaGetErrorName(e));                                                      \
    }                                                                                           \
  } while (0)
  BKT_ALLOC(w.X, NT * cfg->in_dim);
  for (int l = 0; l < lo.L; ++l) {
    BKT_ALLOC(w.Y[l], NT * DH);
    for (int d = 0; d < lo.dirs; ++d) {
      BKT_ALLOC(w.Z[l * lo.dirs + d], NT * 4 * H);
      BKT_ALLOC(w.Cst[l * lo.dirs + d], NT * H);
    }
  }
  BKT_ALLOC(w.logit, NT * lo.C);
  BKT_ALLOC(w.alpha, NT * (size_t)c->S_cap);
  BKT_ALLOC(w.beta, NT * (size_t)c->S_cap);
  BKT_ALLOC(w.dY, NT * DH);
  // split-K partials: at most 64 splits of the largest weight block
  w.part_floats = 64 * max_reduce_block(lo);
  BKT_ALLOC(w.part, w.part_floats);
  BKT_ALLOC(w.tok_t, NT);
  BKT_ALLOC(w.tok_r, NT);
  BKT_ALLOC(w.prev_tok[0], NT);
  BKT_ALLOC(w.prev_tok[1], NT);
  BKT_ALLOC(w.row_ok, (size_t)max_batch);
  BKT_ALLOC(w.status, bkt::kStatusWords);
  {
    const size_t NTq = (NT + 7) & ~size_t(7), MA = std::max<size_t>(4 * H, (size_t)lo.C);
    BKT_ALLOC(w.AT, MA * NTq);
    BKT_ALLOC(w.ATl, MA * NTq);
    const size_t DHp = (DH + 3) & ~size_t(3), Cp = ((size_t)lo.C + 3) & ~size_t(3);
    BKT_ALLOC(w.BTf, DHp * NTq);
    BKT_ALLOC(w.BTl, DHp * NTq);
    BKT_ALLOC(w.Lh, NT * Cp);
    BKT_ALLOC(w.Ll, NT * Cp);
    // W_out split; for fp32 stacks also W_ih (and its transpose) of a layer > 0
    const size_t WW = std::max(Cp * DHp, (lo.L > 1 && cfg->gemm_precision != BKT_GEMM_BF16) ? 4 * (size_t)H * DHp : 0);
    BKT_ALLOC(w.Wh, WW);
    BKT_ALLOC(w.Wl, WW);
    BKT_ALLOC(w.Woh, (size_t)lo.C * DHp);
    BKT_ALLOC(w.Wol, (size_t)lo.C * DHp);
    BKT_ALLOC(w.WoTh, (size_t)DH * Cp);
    BKT_ALLOC(w.WoTl, (size_t)DH * Cp);
    if (lo.L > 1 && cfg->gemm_precision != BKT_GEMM_BF16) {  // dX operands beside the side stream's AT
      BKT_ALLOC(w.DXh, NT * 4 * (size_t)H);
      BKT_ALLOC(w.DXl, NT * 4 * (size_t)H);
    }
    // layer 1's narrow weight gradient: up to 1024 token chunks of 4H x (in_dim+1) partials
    w.part2_floats = (size_t)1024 * 4 * H * (cfg->in_dim + 1);
    BKT_ALLOC(w.part2, w.part2_floats);
  }
  if (cfg->gemm_precision == BKT_GEMM_BF16) {
    uint16_t *p = nullptr;
    for (int l = 0; l < lo.L; ++l) {
      if (l + 1 < lo.L) {
        BKT_ALLOC(p, NT * DH);
        w.Yb[l] = p;
      }
      for (int d = 0; d < lo.dirs; ++d) {
        BKT_ALLOC(p, NT * H);
        w.Hs[l * lo.dirs + d] = p;
        BKT_ALLOC(p, NT * 4 * H);
        w.dZb[l * lo.dirs + d] = p;
        if (l > 0) {
          BKT_ALLOC(p, 4 * H * DH);
          w.Wb[l * lo.dirs + d] = p;
        }
      }
      if (l > 0) BKT_ALLOC(w.dbp[l], (size_t)lo.dirs * ((max_batch + 15) / 16) * 4 * H);
    }
  }
  IdxLayout il = idx_layout(max_batch, max_tokens);
  c->idx_bytes = il.bytes;
  {
    char *p = nullptr;
    BKT_ALLOC(p, il.bytes);
    w.idx_dev = p;
  }
#undef BKT_ALLOC
  e = cudaMemset(w.status, 0, bkt::kStatusWords * sizeof(int32_t));
  if (e != cudaSuccess) {
    delete c;
    return cuda_err("cudaMemset", e);
  }
  e = cudaMallocHost(&c->stage, il.bytes * kStageSlots);
  if (e != cudaSuccess) {
    delete c;
    return set_err(BKT_ENOMEM, "bkt_ctx_create: cudaMallocHost failed: %s", cudaGetErrorName(e));
  }
  for (int i = 0; i < kStageSlots; ++i) {
    e = cudaEventCreateWithFlags(&c->stage_ev[i], cudaEventDisableTiming);
    if (e != cudaSuccess) {
      delete c;
      return cuda_err("cudaEventCreate", e);
    }
  }
  {
    cudaError_t e2 = cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking);
    if (e2 == cudaSuccess) e2 = cudaEventCreateWithFlags(&c->fork_ev, cudaEventDisableTiming);
    if (e2 == cudaSuccess) e2 = cudaEventCreateWithFlags(&c->join_ev, cudaEventDisableTiming);
    if (e2 != cudaSuccess) {
      delete c;
      return cuda_err("side stream", e2);
    }
  }
  for (int l = 0; l < lo.L; ++l)
    c->geom[l] = bkt::plan_recurrent(lo.H, max_batch, lo.dirs, c->sm_count, cfg->gemm_precision == BKT_GEMM_BF16);
  *out = c;
  return BKT_OK;
}

extern "C" void bkt_ctx_destroy(bkt_ctx *c) {
  if (!c) return;
  cudaSetDevice(c->device);
  cudaDeviceSynchronize();
  delete c;
}

extern "C" int bkt_ctx_set_timing(bkt_ctx *c, int32_t enable) {
  if (!c) return set_err(BKT_EINVAL, "bkt_ctx_set_timing: NULL ctx");
  c->timer.fold();
  c->timer.totals.clear();
  c->timer.on = enable != 0;
  return BKT_OK;
}

extern "C" int bkt_ctx_kernel_times(bkt_ctx *c, bkt_kernel_time *out, int32_t cap, int32_t *n_out) {
  if (!c || !n_out) return set_err(BKT_EINVAL, "bkt_ctx_kernel_times: NULL argument");
  c->timer.fold();
  int32_t n = 0;
  for (const auto &t : c->timer.totals) {
    if (out && n < cap) {
      out[n].name = t.name;
      out[n].launches = t.launches;
      out[n].total_ms = t.ms;
      out[n].flops = t.flops;
      out[n].bytes = t.bytes;
      out[n].serial_steps = t.steps;
    }
    ++n;
  }
  *n_out = n;
  return BKT_OK;
}

namespace {
// Waits for the ctx's work and reads status word `i`; with `clear`, zeroes it.
int read_status_word(bkt_ctx *c, int i, int32_t *v, bool clear) {
  cudaError_t e = cudaSetDevice(c->device);
  if (e != cudaSuccess) return cuda_err("cudaSetDevice", e);
  e = cudaStreamSynchronize(c->last_stream);
  if (e == cudaSuccess && c->side) e = cudaStreamSynchronize(c->side);
  if (e != cudaSuccess) return cuda_err("cudaStreamSynchronize", e);
  e = cudaMemcpy(v, c->w.status + i, sizeof *v, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_err("cudaMemcpy(status)", e);
  if (clear && *v != 0) {
    e = cudaMemset(c->w.status + i, 0, sizeof *v);
    if (e != cudaSuccess) return cuda_err("cudaMemset(status)", e);
  }
  return BKT_OK;
}
}  // namespace

extern "C" int bkt_ctx_sync_status(bkt_ctx *c) {
  if (!c) return set_err(BKT_EINVAL, "bkt_ctx_sync_status: NULL ctx");
  int32_t st = 0;
  if (int rc = read_status_word(c, 0, &st, true)) return rc;
  if (st != 0) {
    const bool timeout = (st & (bkt::kErrTcWait | bkt::kErrExchWait)) != 0;
    return set_err(timeout ? BKT_ETIMEOUT : BKT_EDEVICE, "device check failed (flags 0x%x):%s%s%s", st,
                   (st & bkt::kErrLabel) ? " a label is out of range or equals the blank;" : "",
                   (st & bkt::kErrTcWait) ? " a tensor-core pipeline wait timed out;" : "",
                   (st & bkt::kErrExchWait) ? " a recurrent cluster exchange wait timed out;" : "");
  }
  return BKT_OK;
}

extern "C" int bkt_ctx_infeasible_count(bkt_ctx *c, int64_t *count) {
  if (!c || !count) return set_err(BKT_EINVAL, "bkt_ctx_infeasible_count: NULL argument");
  int32_t v = 0;
  if (int rc = read_status_word(c, 1, &v, true)) return rc;
  *count = v;
  return BKT_OK;
}

extern "C" int bkt_ctx_set_wait_faults(bkt_ctx *c, int32_t poll_cap, int32_t withhold) {
  if (!c) return set_err(BKT_EINVAL, "bkt_ctx_set_wait_faults: NULL ctx");
  if (poll_cap < 0 || (withhold & ~(BKT_WITHHOLD_EXCHANGE | BKT_WITHHOLD_TMA)) != 0)
    return set_err(BKT_EINVAL, "bkt_ctx_set_wait_faults: poll_cap %d or withhold bits 0x%x out of range", poll_cap,
                   withhold);
  c->wf.poll_cap = poll_cap == 0 ? 0 : std::max(poll_cap, 256);
  c->wf.withhold = withhold;
  return BKT_OK;
}

extern "C" int bkt_adadelta_update(float *params, const float *grads, float *eg2, float *edx2, int64_t n,
                                   float rho, float eps, float lr, void *stream) {
  if (n < 0 || (n > 0 && (!params || !grads || !eg2 || !edx2)))
    return set_err(BKT_EINVAL, "bkt_adadelta_update: bad arguments");
  if (!(rho >= 0.f && rho < 1.f) || !(eps > 0.f) || !(lr >= 0.f))
    return set_err(BKT_EINVAL, "bkt_adadelta_update: need 0 <= rho < 1, eps > 0, lr >= 0");
  if (n == 0) return BKT_OK;
  cudaError_t e = bkt::launch_adadelta(params, grads, eg2, edx2, n, rho, eps, lr, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_err("adadelta kernel launch", e);
  return BKT_OK;
}

extern "C" int bkt_average_models(float *v, const float *prev, int64_t n, int32_t n_models, float beta,
                                  void *stream) {
  if (n < 0 || n_models < 1 || (n > 0 && (!v || !prev)) || !(beta >= 0.f))
    return set_err(BKT_EINVAL, "bkt_average_models: bad arguments");
  if (n == 0) return BKT_OK;
  cudaError_t e = bkt::launch_average_models(v, prev, n, n_models, beta, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_err("average kernel launch", e);
  return BKT_OK;
}

extern "C" int bkt_sgd_update(float *params, const float *grads, int64_t n, float lr, void *stream) {
  if (n < 0 || (n > 0 && (!params || !grads))) return set_err(BKT_EINVAL, "bkt_sgd_update: bad arguments");
  if (n == 0) return BKT_OK;
  cudaError_t e = bkt::launch_sgd(params, grads, n, lr, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_err("sgd kernel launch", e);
  return BKT_OK;
}

// ---------------------------------------------------------------------------
// The step through a ctx.
extern "C" int bkt_lstm_ctc_step(bkt_ctx *c, const bkt_batch *bt, const float *params, float *grads, float *loss,
                                 void *stream) {
  bkt::NvtxRange range("bkt_lstm_ctc_step");
  if (!c || !bt || !params || !grads || !loss) return set_err(BKT_EINVAL, "bkt_lstm_ctc_step: NULL argument");
  int64_t n_tok = 0, cells = 0;
  int32_t S_max = 1;
  int rc = check_batch(bt, c->max_tokens, c->max_batch, c->max_label_len, &n_tok, &S_max, &cells);
  if (rc != BKT_OK) return rc;
  const int32_t b = bt->n_seq;
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaSetDevice(c->device);
  if (e != cudaSuccess) return cuda_err("cudaSetDevice", e);

  // ---- a4 (host part): stable sort by length, longest first; time offsets.
  std::vector<int32_t> perm(b);
  for (int32_t i = 0; i < b; ++i) perm[i] = i;
  std::stable_sort(perm.begin(), perm.end(),
                   [&](int32_t x, int32_t y) { return bt->lengths[x] > bt->lengths[y]; });
  const int32_t T = bt->lengths[perm[0]];
  IdxLayout il = idx_layout(b, T);
  const int slot = c->stage_next;
  c->stage_next = (slot + 1) % kStageSlots;
  if (c->stage_used[slot]) {
    e = cudaEventSynchronize(c->stage_ev[slot]);
    if (e != cudaSuccess) return cuda_err("cudaEventSynchronize(stage)", e);
  }
  char *st = (char *)c->stage + (size_t)slot * c->idx_bytes;
  bkt::DevIdx ix = fill_index_block(bt, perm.data(), T, n_tok, S_max, il, st, (char *)c->w.idx_dev, c->w.tok_t,
                                    c->w.tok_r);
  e = cudaMemcpyAsync(c->w.idx_dev, st, il.bytes, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_err("cudaMemcpyAsync(index block)", e);
  e = cudaEventRecord(c->stage_ev[slot], s);
  if (e != cudaSuccess) return cuda_err("cudaEventRecord(stage)", e);
  c->stage_used[slot] = true;
  c->last_stream = s;
  ix.n_cells = cells;
  return enqueue_kernels(c->cfg, c->lo, c->w, c->geom, ix, bt, params, grads, loss, s,
                         c->timer.on ? &c->timer : nullptr, c->sm_count, c->side, c->fork_ev, c->join_ev, c->wf);
}

// ---------------------------------------------------------------------------
// The step on caller-provided scratch (no allocation anywhere on this path:
// fixed-size host arrays, a pageable staging buffer, buffers carved out of
// the scratch range).
int bkt::report_error(int code, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  const int r = vset_err(code, fmt, ap);
  va_end(ap);
  return r;
}

namespace {

constexpr int32_t kScratchMaxBatch = 512;
constexpr int32_t kScratchMaxLabel = 1023;
constexpr size_t kScratchStageBytes = 256 * 1024;
alignas(64) char g_scratch_stage[kScratchStageBytes];
std::mutex g_scratch_stage_mu;

// Bump allocator over a caller-provided range (256-byte aligned pieces).
struct Carve {
  char *base;
  size_t cap, used = 0;
  template <typename T>
  T *take(size_t count) {
    const size_t off = (used + 255) & ~size_t(255);
    used = off + std::max<size_t>(count, 1) * sizeof(T);
    return reinterpret_cast<T *>(base + off);
  }
};

}  // namespace

int bkt::step_on_scratch(const bkt_model_cfg *cfg, const bkt_batch *bt, const float *params, float *grads,
                         float *loss, cudaStream_t s, void *scratch, size_t scratch_bytes, int sm_count) {
  bkt::NvtxRange range("bkt_lstm_ctc_step_static");
  if (!cfg_ok(cfg)) return set_err(BKT_EINVAL, "bkt_lstm_ctc_step_static: invalid model cfg");
  if (!bt || !params || !grads || !loss) return set_err(BKT_EINVAL, "bkt_lstm_ctc_step_static: NULL argument");
  int64_t n_tok = 0, cells = 0;
  int32_t S_max = 1;
  int rc = check_batch(bt, (int64_t)INT32_MAX / 4, kScratchMaxBatch, kScratchMaxLabel, &n_tok, &S_max, &cells);
  if (rc != BKT_OK) return rc;
  const Layout lo = make_layout(cfg);
  const int32_t b = bt->n_seq;
  // stable insertion sort, longest first
  int32_t perm[kScratchMaxBatch];
  for (int32_t i = 0; i < b; ++i) {
    int32_t j = i;
    while (j > 0 && bt->lengths[perm[j - 1]] < bt->lengths[i]) {
      perm[j] = perm[j - 1];
      --j;
    }
    perm[j] = i;
  }
  const int32_t T = bt->lengths[perm[0]];
  const IdxLayout il = idx_layout(b, T);
  if (il.bytes > kScratchStageBytes)
    return set_err(BKT_EINVAL, "bkt_lstm_ctc_step_static: the longest sequence (%d steps) is too long for this entry point", T);

  // carve the workspace
  const size_t NT = (size_t)n_tok, DH = (size_t)lo.dirs * lo.H, H = lo.H;
  Carve cv{(char *)scratch, scratch_bytes};
  StepBufs w{};
  w.X = cv.take<float>(NT * cfg->in_dim);
  for (int l = 0; l < lo.L; ++l) {
    w.Y[l] = cv.take<float>(NT * DH);
    for (int d = 0; d < lo.dirs; ++d) {
      w.Z[l * lo.dirs + d] = cv.take<float>(NT * 4 * H);
      w.Cst[l * lo.dirs + d] = cv.take<float>(NT * H);
    }
  }
  w.logit = cv.take<float>(NT * lo.C);
  w.alpha = cv.take<float>((size_t)cells);
  w.beta = cv.take<float>((size_t)cells);
  w.dY = cv.take<float>(NT * DH);
  w.tok_t = cv.take<int32_t>(NT);
  w.tok_r = cv.take<int32_t>(NT);
  w.prev_tok[0] = cv.take<int32_t>(NT);
  w.prev_tok[1] = cv.take<int32_t>(NT);
  w.row_ok = cv.take<int32_t>((size_t)b);
  w.status = cv.take<int32_t>(kStatusWords);
  w.idx_dev = cv.take<char>(il.bytes);
  {
    const size_t NTq = (NT + 7) & ~size_t(7), MA = std::max<size_t>(4 * H, (size_t)lo.C);
    w.AT = cv.take<float>(MA * NTq);
    w.ATl = cv.take<float>(MA * NTq);
    const size_t DHp = (DH + 3) & ~size_t(3), Cp = ((size_t)lo.C + 3) & ~size_t(3);
    w.BTf = cv.take<float>(DHp * NTq);
    w.BTl = cv.take<float>(DHp * NTq);
    w.Lh = cv.take<float>(NT * Cp);
    w.Ll = cv.take<float>(NT * Cp);
    const size_t WW = std::max(Cp * DHp, (lo.L > 1 && cfg->gemm_precision != BKT_GEMM_BF16) ? 4 * (size_t)H * DHp : 0);
    w.Wh = cv.take<float>(WW);
    w.Wl = cv.take<float>(WW);
    w.Woh = cv.take<float>((size_t)lo.C * DHp);
    w.Wol = cv.take<float>((size_t)lo.C * DHp);
    w.WoTh = cv.take<float>((size_t)DH * Cp);
    w.WoTl = cv.take<float>((size_t)DH * Cp);
  }
  if (cfg->gemm_precision == BKT_GEMM_BF16) {
    for (int l = 0; l < lo.L; ++l) {
      if (l + 1 < lo.L) w.Yb[l] = cv.take<uint16_t>(NT * DH);
      for (int d = 0; d < lo.dirs; ++d) {
        w.Hs[l * lo.dirs + d] = cv.take<uint16_t>(NT * H);
        w.dZb[l * lo.dirs + d] = cv.take<uint16_t>(NT * 4 * H);
        if (l > 0 && d == 0) w.dbp[l] = cv.take<float>((size_t)lo.dirs * ((b + 15) / 16) * 4 * H);
        if (l > 0) w.Wb[l * lo.dirs + d] = cv.take<uint16_t>(4 * H * DH);
      }
    }
  }
  // split-K partials get the rest: at least one split of the largest block
  const size_t min_part = max_reduce_block(lo);
  w.part = cv.take<float>(min_part);
  const size_t need = cv.used;
  if (need > scratch_bytes)
    return set_err(BKT_EINVAL,
                   "bkt_lstm_ctc_step_static: this batch needs %zu bytes of scratch but the static array holds %zu "
                   "(use a bkt_ctx for larger batches)",
                   need, scratch_bytes);
  w.part_floats = min_part + (scratch_bytes - need) / sizeof(float);
  w.part_floats = std::min(w.part_floats, 64 * min_part);

  RecGeom geom[kMaxLayers];
  const RecGeom g0 = plan_recurrent(lo.H, b, lo.dirs, sm_count, cfg->gemm_precision == BKT_GEMM_BF16);
  for (int l = 0; l < lo.L; ++l) geom[l] = g0;

  cudaError_t e = cudaMemsetAsync(w.status, 0, kStatusWords * sizeof(int32_t), s);
  if (e != cudaSuccess) return cuda_err("cudaMemsetAsync(status)", e);
  DevIdx ix;
  {
    // pageable source: the call returns once the bytes are staged, so the
    // buffer is free again when the lock is released
    std::lock_guard<std::mutex> lk(g_scratch_stage_mu);
    ix = fill_index_block(bt, perm, T, n_tok, S_max, il, g_scratch_stage, (char *)w.idx_dev, w.tok_t, w.tok_r);
    e = cudaMemcpyAsync(w.idx_dev, g_scratch_stage, il.bytes, cudaMemcpyHostToDevice, s);
  }
  if (e != cudaSuccess) return cuda_err("cudaMemcpyAsync(index block)", e);
  ix.n_cells = cells;
  return enqueue_kernels(*cfg, lo, w, geom, ix, bt, params, grads, loss, s, nullptr, sm_count);
}
