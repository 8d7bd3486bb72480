// api.cu -- the extern "C" entry points declared in include/tt.h: argument
// validation (before anything touches the GPU), workspace carving and the
// launch sequences of align / transfer / verify / step.
#include <atomic>
#include <cmath>
#include <algorithm>
#include <cstdint>
#include <cstring>

#include "tt_device.cuh"
#include "tt_launch.h"
#include "tt_shard.h"

namespace {

using namespace tt;

std::atomic<int> g_last_cuda_error{0};
std::atomic<int32_t> g_epoch{0x2b6f1000};  // tags each call's row-pass error word

int32_t next_epoch() { return ++g_epoch; }

tt_status cuda_fail(cudaError_t e) {
  g_last_cuda_error.store(int(e));
  return TT_ERR_CUDA;
}

// Loads all kernels on the current device once, before the first launch there
// (two threads that both find a device not yet done load it twice, which is
// harmless: loading and setting attributes are idempotent).
cudaError_t ensure_loaded() {
  static std::atomic<bool> done[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && done[dev].load(std::memory_order_acquire)) return cudaSuccess;
  if ((e = preload_align()) != cudaSuccess) return e;
  if ((e = preload_rowpass()) != cudaSuccess) return e;
  if ((e = preload_decide()) != cudaSuccess) return e;
  if ((e = preload_filter()) != cudaSuccess) return e;
  if ((e = preload_nucleus()) != cudaSuccess) return e;
  if ((e = preload_pen()) != cudaSuccess) return e;
  if ((e = preload_shard()) != cudaSuccess) return e;
  if (dev >= 0 && dev < 64) done[dev].store(true, std::memory_order_release);
  return cudaSuccess;
}

int sm_count_current() {
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < 64) {
    const int c = cached[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  if (dev < 64) cached[dev].store(n, std::memory_order_relaxed);
  return n;
}

bool batch_ok(const tt_batch* b) {
  if (!b || b->B < 0 || b->n_draft < 0 || b->n_target < 0) return false;
  if (b->B == 0) return true;
  if (!b->draft_off || !b->target_off) return false;
  if (b->max_k < 1 || b->max_k > TT_MAX_K || b->max_m < 1 || b->max_m > TT_MAX_M) return false;
  if (int64_t(b->n_target) + b->B > INT32_MAX) return false;
  return true;
}

bool dtype_ok(int32_t dt) { return dt == TT_F32 || dt == TT_BF16; }

// Logits rows usable by the vectorised row pass.
bool logits_ok(const tt_logits* L, int64_t rows_needed) {
  if (!L || !L->data || !dtype_ok(L->dtype)) return false;
  if (L->n_cols < 1 || int64_t(L->n_cols) > int64_t(kMaxChunksPerRow) * kChunk) return false;
  if (L->row_stride < L->n_cols || L->n_rows < rows_needed) return false;
  const int64_t esz = L->dtype == TT_F32 ? 4 : 2;
  if ((reinterpret_cast<uintptr_t>(L->data) & 15) != 0) return false;
  if ((L->row_stride * esz) % 16 != 0) return false;
  return true;
}

bool params_ok(const tt_params* p) {
  if (!p) return false;
  if (!(p->temp_draft > 0.f) || !std::isfinite(p->temp_draft)) return false;
  if (!(p->temp_target > 0.f) || !std::isfinite(p->temp_target)) return false;
  if (p->full_q != 0 && p->full_q != 1) return false;
  if (p->top_k_draft < 0 || p->top_k_draft > TT_MAX_TOP_K) return false;
  if (p->top_k_target < 0 || p->top_k_target > TT_MAX_TOP_K) return false;
  if (!(p->top_p_draft > 0.f) || std::isnan(p->top_p_draft)) return false;
  if (!(p->top_p_target > 0.f) || std::isnan(p->top_p_target)) return false;
  if (!(p->rep_penalty_draft > 0.f) || !std::isfinite(p->rep_penalty_draft)) return false;
  if (!(p->rep_penalty_target > 0.f) || !std::isfinite(p->rep_penalty_target)) return false;
  return true;
}

// Repetition penalties on: per family, and the batch's histories usable.
bool pen_draft(const tt_params* p) { return p->rep_penalty_draft != 1.f; }
bool pen_target(const tt_params* p) { return p->rep_penalty_target != 1.f; }
bool history_ok(const int32_t* off, const int32_t* cols, int32_t n) {
  return n >= 0 && (off == nullptr ? n == 0 : (n == 0 || cols != nullptr));
}

PenSizes pen_sizes(const tt_batch* b, bool on_d, bool on_t) {
  PenSizes p;
  p.on_d = on_d;
  p.on_t = on_t;
  p.n_hist_d = on_d && b->hist_off_d ? b->n_hist_d : 0;
  p.n_hist_t = on_t && b->hist_off_t ? b->n_hist_t : 0;
  return p;
}

// The per-request sets of the penalized families (one small kernel).
cudaError_t launch_pen_sets(const tt_batch* batch, const RowSet& d, const RowSet& t, bool on_d,
                            bool on_t, const int32_t* dcols, const int32_t* tcols,
                            const Workspace& ws, cudaStream_t s) {
  PenArgs a;
  std::memset(&a, 0, sizeof a);
  a.B = batch->B;
  a.on_d = on_d;
  a.on_t = on_t;
  a.V_d = d.V;
  a.V_t = t.V;
  a.nch_d = d.nch;
  a.nch_t = t.nch;
  a.unit_d = d.unit_cols;
  a.unit_t = t.unit_cols;
  a.nlist_d = d.nlist;
  a.nlist_t = t.nlist;
  a.n_draft = batch->n_draft;
  a.n_target = batch->n_target;
  a.n_hist_d = batch->hist_off_d ? batch->n_hist_d : 0;
  a.n_hist_t = batch->hist_off_t ? batch->n_hist_t : 0;
  a.hist_off_d = batch->hist_off_d;
  a.hist_cols_d = batch->hist_cols_d;
  a.hist_off_t = batch->hist_off_t;
  a.hist_cols_t = batch->hist_cols_t;
  a.draft_off = batch->draft_off;
  a.draft_cols = dcols;
  a.target_off = batch->target_off;
  a.target_cols = tcols;
  a.pen_d = ws.pen_d;
  a.pbase_d = ws.pbase_d;
  a.pcnt_d = ws.pcnt_d;
  a.pstart_d = ws.pstart_d;
  a.pen_t = ws.pen_t;
  a.pbase_t = ws.pbase_t;
  a.pcnt_t = ws.pcnt_t;
  a.pstart_t = ws.pstart_t;
  a.pstatus = ws.pstatus;
  return launch_pen_prep(a, s);
}

// A nucleus family's row set: the row pass writes the compensated partials of
// all its columns, and the nucleus kernel finds each row's kept set from them
// and the row's logits.
void attach_nucleus(RowSet& r, bool on) { r.nucleus = on ? 1 : 0; }

// A family's row set sees its penalty arrays.
void attach_pen(RowSet& r, bool on, float theta, PenEntry* pen, const int32_t* pbase,
                const int32_t* pcnt, const int32_t* pstart) {
  if (!on) return;
  r.pen = pen;
  r.pbase = pbase;
  r.pcnt = pcnt;
  r.pstart = pstart;
  r.penalty = theta;
}

int k_draft(const tt_params* p) { return p->top_k_draft; }
int k_target(const tt_params* p) { return p->top_k_target; }
// Nucleus families: top-p without top-k (a kept set over the whole row).
bool nuc_draft(const tt_params* p) { return p->top_k_draft == 0 && p->top_p_draft < 1.f; }
bool nuc_target(const tt_params* p) { return p->top_k_target == 0 && p->top_p_target < 1.f; }

// Shards usable by tt_verify_sharded: 1..TT_MAX_SHARDS logits arrays of
// rows_needed rows that tile the row in order from column 0; V = the row width.
bool shards_ok(const tt_shards* sh, int64_t rows_needed, int32_t* V) {
  if (!sh || sh->S < 1 || sh->S > TT_MAX_SHARDS || !sh->shards || !sh->col0) return false;
  int64_t c = 0;
  for (int s = 0; s < sh->S; ++s) {
    if (!logits_ok(&sh->shards[s], rows_needed)) return false;
    if (sh->col0[s] != c) return false;
    c += sh->shards[s].n_cols;
  }
  if (c > INT32_MAX) return false;
  *V = int32_t(c);
  return true;
}

ShardWorkspace shard_workspace(void* base, const tt_batch* batch, const tt_shards* sh) {
  int32_t nch[TT_MAX_SHARDS] = {0};
  for (int s = 0; s < sh->S; ++s) nch[s] = n_chunks(sh->shards[s].n_cols);
  return shard_layout(base, int64_t(batch->n_target) + batch->B, sh->S, nch);
}

bool vocab_ok(const tt_vocab* v) {
  return v && v->bytes && v->offsets && v->n_tokens >= 1 && v->n_bytes >= 0;
}

float log2e_over(float T) { return float(1.4426950408889634 / double(T)); }

RowSet rowset(const tt_logits* L, Partial* part, const uint8_t* need, float T) {
  RowSet r;
  r.data = static_cast<const char*>(L->data);
  r.stride_bytes = L->row_stride * (L->dtype == TT_F32 ? 4 : 2);
  r.V = L->n_cols;
  r.nch = n_chunks(L->n_cols);
  r.scale = log2e_over(T);
  r.n_rows = L->n_rows;
  r.part = part;
  r.need = need;
  r.top_k = 0;
  r.cand = nullptr;
  r.nlist = L->dtype == TT_F32 ? r.nch : (r.nch + 1) / 2;
  r.nucleus = 0;
  r.pen = nullptr;
  r.pbase = r.pcnt = r.pstart = nullptr;
  r.penalty = 1.f;
  r.unit_cols = L->dtype == TT_F32 ? kChunk : 2 * kChunk;
  return r;
}

RowSet no_rows() {
  RowSet r;
  std::memset(&r, 0, sizeof r);
  r.nch = 1;
  r.nlist = 1;
  return r;
}

// Kept sets of the filtered families among d (rows_d rows) and t (rows_t);
// penalized families find each row's request and position from the batch.
cudaError_t launch_kept_sets(const RowSet& d, int64_t rows_d, const RowSet& t, int64_t rows_t,
                             const tt_params* prm, const Workspace& ws, cudaStream_t s,
                             bool pdl, const tt_batch* batch = nullptr, int dt_d = TT_F32,
                             int dt_t = TT_F32) {
  KeptArgs k;
  std::memset(&k, 0, sizeof k);
  if (batch) {
    k.B = batch->B;
    k.n_target = batch->n_target;
    k.n_draft = batch->n_draft;
    k.target_off = batch->target_off;
    k.draft_off = batch->draft_off;
  }
  k.dt_d = dt_d;
  k.dt_t = dt_t;
  k.d = d;
  k.t = t;
  k.rows_d = d.top_k > 0 ? rows_d : 0;
  k.rows_t = t.top_k > 0 ? rows_t : 0;
  k.top_p_d = prm->top_p_draft;
  k.top_p_t = prm->top_p_target;
  k.kept_d = ws.kept_d;
  k.kept_t = ws.kept_t;
  k.head_d = ws.head_d;
  k.head_t = ws.head_t;
  return launch_kept(k, s, sm_count_current(), pdl);
}

// Kept sets of the nucleus families among d and t (top-p without top-k).
cudaError_t launch_nucleus_sets(const RowSet& d, int64_t rows_d, const RowSet& t, int64_t rows_t,
                                const tt_params* prm, const Workspace& ws, int dt_d, int dt_t,
                                const tt_batch* batch, const int32_t* tcols, cudaStream_t s,
                                bool pdl) {
  KeptArgs k;
  std::memset(&k, 0, sizeof k);
  k.d = d;
  k.t = t;
  k.rows_d = d.nucleus ? rows_d : 0;
  k.rows_t = t.nucleus ? rows_t : 0;
  k.top_p_d = prm->top_p_draft;
  k.top_p_t = prm->top_p_target;
  k.head_d = ws.head_d;
  k.head_t = ws.head_t;
  k.um_d = ws.um_d;
  k.um_t = ws.um_t;
  k.dt_d = dt_d;
  k.dt_t = dt_t;
  k.B = batch->B;
  k.n_target = batch->n_target;
  k.target_off = batch->target_off;
  k.target_cols = tcols;
  k.draft_off = batch->draft_off;
  k.n_draft = batch->n_draft;
  return launch_nucleus(k, s, sm_count_current(), pdl);
}

void attach_kept(DecideArgs& d, const Workspace& ws) {
  d.kept_d = ws.kept_d;
  d.kept_t = ws.kept_t;
  d.head_d = ws.head_d;
  d.head_t = ws.head_t;
  d.um_d = ws.um_d;
  d.um_t = ws.um_t;
}

// Share of the target rows the step's row pass streams before it waits for
// the alignment (in eighths): half, or seven eighths when the batch holds so
// many draft tokens (B x max_k of 32768 and more, each a row of the DTW tile)
// that the alignment outlasts half of the target rows; the rest is drawn
// dynamically after the wait.
int pre_wait_eighths(const tt_batch* b) {
  return int64_t(b->B) * b->max_k >= 32768 ? 7 : 4;
}

void record(const tt_params* p, int i, cudaStream_t s) {
  if (p->events && p->events[i]) cudaEventRecord(static_cast<cudaEvent_t>(p->events[i]), s);
}

tt_status fill_align_args(const tt_batch* bt, const tt_vocab* vd, const tt_vocab* vt,
                          const tt_params* prm, AlignArgs& a) {
  std::memset(&a, 0, sizeof a);
  a.B = bt->B;
  a.n_draft = bt->n_draft;
  a.n_target = bt->n_target;
  a.max_k = bt->max_k;
  a.max_m = bt->max_m;
  a.window = prm->window;
  a.draft_off = bt->draft_off;
  a.draft_ids = bt->draft_ids;
  a.target_off = bt->target_off;
  a.target_ids = bt->target_ids;
  a.vd = *vd;
  a.vt = *vt;
  a.tile_w = align_tile_width(bt->max_k, bt->max_m, prm->window);
  a.smem_per_warp = align_smem_per_warp(bt->max_k, bt->max_m, a.tile_w);
  if (a.smem_per_warp > size_t(kAlignSmemMax)) return TT_ERR_UNSUPPORTED;
  // pairs spread over the SMs (one warp each while the batch is small), at
  // most kAlignWarpsMax warps and 96 KB per CTA; before the row pass,
  // launch_align caps the grid at one CTA per SM, whose warps then loop over
  // the pairs
  int wpb = int(size_t(96 * 1024) / a.smem_per_warp);
  const int spread = (bt->B + sm_count_current() - 1) / sm_count_current();
  wpb = std::min(wpb, std::min(kAlignWarpsMax, spread));
  a.warps_per_block = wpb < 1 ? 1 : wpb;
  return TT_OK;
}

}  // namespace

namespace tt {
tt_status record_cuda_error(cudaError_t e) { return cuda_fail(e); }

tt_status step_check(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                     const tt_logits* draft, const float* draft_probs, const tt_logits* target,
                     const tt_params* prm, const tt_step_out* out, size_t* need) {
  *need = 0;
  if (!batch_ok(batch) || !params_ok(prm)) return TT_ERR_INVALID_ARG;
  if (!out || !out->accepted || !out->next_token || !out->status) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!vocab_ok(vd) || !vocab_ok(vt)) return TT_ERR_INVALID_ARG;
  if ((batch->n_draft > 0 && !batch->draft_ids) || (batch->n_target > 0 && !batch->target_ids))
    return TT_ERR_INVALID_ARG;
  const bool full_q = prm->full_q != 0;
  const bool from_logits = draft_probs == nullptr || full_q;
  if (!logits_ok(target, int64_t(batch->n_target) + batch->B)) return TT_ERR_INVALID_ARG;
  if (from_logits && !logits_ok(draft, batch->n_draft)) return TT_ERR_INVALID_ARG;
  if (full_q && draft->n_cols != target->n_cols) return TT_ERR_INVALID_ARG;
  // given draft probabilities are taken as they are (no draft filter)
  const int kd = from_logits ? k_draft(prm) : 0, kt = k_target(prm);
  const bool nd = from_logits && nuc_draft(prm), nt = nuc_target(prm);
  // full-q: both families filtered or neither, and no nucleus family
  if (full_q && ((kd > 0 || nd) != (kt > 0 || nt) || nd || nt)) return TT_ERR_UNSUPPORTED;
  // a repetition penalty needs its family's top-k, and one-hot transfer
  const bool pd = from_logits && pen_draft(prm), pt = pen_target(prm);
  if ((pd && kd == 0) || (pt && kt == 0) || (full_q && (pd || pt))) return TT_ERR_UNSUPPORTED;
  if ((pd && !history_ok(batch->hist_off_d, batch->hist_cols_d, batch->n_hist_d)) ||
      (pt && !history_ok(batch->hist_off_t, batch->hist_cols_t, batch->n_hist_t)))
    return TT_ERR_INVALID_ARG;
  AlignArgs a;
  const tt_status st = fill_align_args(batch, vd, vt, prm, a);
  if (st != TT_OK) return st;
  *need = workspace_layout(nullptr, batch->B, batch->n_draft, batch->n_target,
                           from_logits ? draft->n_cols : 0, target->n_cols, kd, kt, nd, nt,
                           pen_sizes(batch, pd, pt))
              .bytes;
  return TT_OK;
}
}  // namespace tt

extern "C" {

size_t tt_workspace_bytes_for(const tt_batch* batch, int32_t V_d, int32_t V_t,
                              const tt_params* prm) {
  if (!batch || batch->B < 0 || batch->n_draft < 0 || batch->n_target < 0) return 0;
  const int kd = prm ? prm->top_k_draft : 0, kt = prm ? prm->top_k_target : 0;
  if (kd < 0 || kd > TT_MAX_TOP_K || kt < 0 || kt > TT_MAX_TOP_K) return 0;
  const bool nd = prm && nuc_draft(prm), nt = prm && nuc_target(prm);
  const bool pd = prm && pen_draft(prm), pt = prm && pen_target(prm);
  return workspace_layout(nullptr, batch->B, batch->n_draft, batch->n_target, V_d < 0 ? 0 : V_d,
                          V_t < 0 ? 0 : V_t, kd, kt, nd, nt, pen_sizes(batch, pd, pt))
      .bytes;
}

size_t tt_workspace_bytes(const tt_batch* batch, int32_t V_d, int32_t V_t) {
  if (!batch || batch->B < 0 || batch->n_draft < 0 || batch->n_target < 0) return 0;
  return workspace_layout(nullptr, batch->B, batch->n_draft, batch->n_target, V_d < 0 ? 0 : V_d,
                          V_t < 0 ? 0 : V_t)
      .bytes;
}

tt_status tt_align(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                   const tt_params* prm, int32_t* path, int32_t* path_len, int32_t* cost,
                   int32_t* map, int32_t* status, void* stream) {
  if (!batch_ok(batch) || !params_ok(prm)) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!vocab_ok(vd) || !vocab_ok(vt) || !status) return TT_ERR_INVALID_ARG;
  if ((batch->n_draft > 0 && !batch->draft_ids) || (batch->n_target > 0 && !batch->target_ids))
    return TT_ERR_INVALID_ARG;
  AlignArgs a;
  tt_status st = fill_align_args(batch, vd, vt, prm, a);
  if (st != TT_OK) return st;
  a.path = path;
  a.path_len = path_len;
  a.cost = cost;
  a.map = map;
  a.status = status;
  cudaError_t e = ensure_loaded();
  if (e == cudaSuccess) e = launch_align(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TT_OK : cuda_fail(e);
}

tt_status tt_transfer(const tt_batch* batch, const int32_t* map, const tt_logits* draft,
                      const float* draft_probs, const tt_params* prm, void* workspace,
                      size_t workspace_bytes, float* q_hat, int32_t* status, void* stream) {
  if (!batch_ok(batch) || !params_ok(prm)) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!q_hat || !status || (batch->n_target > 0 && !map)) return TT_ERR_INVALID_ARG;
  const bool from_logits = draft_probs == nullptr;
  if (from_logits && !logits_ok(draft, batch->n_draft)) return TT_ERR_INVALID_ARG;
  const int32_t* cols = batch->draft_cols ? batch->draft_cols : batch->draft_ids;
  if (from_logits && batch->n_draft > 0 && !cols) return TT_ERR_INVALID_ARG;
  const int kd = from_logits ? k_draft(prm) : 0;  // given probabilities are taken as they are
  const bool nd = from_logits && nuc_draft(prm);
  const bool pd = from_logits && pen_draft(prm);
  if (pd && kd == 0) return TT_ERR_UNSUPPORTED;
  if (pd && !history_ok(batch->hist_off_d, batch->hist_cols_d, batch->n_hist_d))
    return TT_ERR_INVALID_ARG;
  const int V_d = from_logits ? draft->n_cols : 0;
  const size_t need = workspace_layout(nullptr, batch->B, batch->n_draft, batch->n_target, V_d,
                                       0, kd, 0, nd, false, pen_sizes(batch, pd, false))
                          .bytes;
  if (from_logits && (!workspace || workspace_bytes < need ||
                      (reinterpret_cast<uintptr_t>(workspace) & 255) != 0))
    return TT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Workspace ws = workspace_layout(workspace, batch->B, batch->n_draft, batch->n_target, V_d, 0,
                                  kd, 0, nd, false, pen_sizes(batch, pd, false));

  DecideArgs d;
  std::memset(&d, 0, sizeof d);
  d.sm_count = sm_count_current();
  d.B = batch->B;
  d.n_draft = batch->n_draft;
  d.n_target = batch->n_target;
  d.max_k = batch->max_k;
  d.max_m = batch->max_m;
  d.mode_transfer_only = 1;
  d.draft_off = batch->draft_off;
  d.draft_cols = cols;
  d.target_off = batch->target_off;
  d.map = map;
  d.draft_probs = draft_probs;
  d.d = from_logits ? rowset(draft, ws.part_d, ws.need_d, prm->temp_draft) : no_rows();
  d.d.top_k = kd;
  d.d.cand = ws.cand_d;
  attach_nucleus(d.d, nd);
  attach_pen(d.d, pd, prm->rep_penalty_draft, ws.pen_d, ws.pbase_d, ws.pcnt_d, ws.pstart_d);
  d.status_p = pd ? ws.pstatus : nullptr;
  d.top_p_d = prm->top_p_draft;
  d.t = no_rows();
  d.dt_d = from_logits ? draft->dtype : TT_F32;
  d.status = status;
  d.q_hat_out = q_hat;
  cudaError_t e = ensure_loaded();
  if (e != cudaSuccess) return cuda_fail(e);
  if (from_logits) {
    PrepArgs p;
    std::memset(&p, 0, sizeof p);
    p.B = batch->B;
    p.n_draft = batch->n_draft;
    p.n_target = batch->n_target;
    p.draft_off = batch->draft_off;
    p.target_off = batch->target_off;
    p.map = map;
    p.need = ws.need_d;
    p.work = ws.work;
    if ((e = launch_prep(p, s)) != cudaSuccess) return cuda_fail(e);
    if (pd && (e = launch_pen_sets(batch, d.d, no_rows(), true, false, cols, nullptr, ws, s)) !=
                  cudaSuccess)
      return cuda_fail(e);
    RowPassArgs r;
    std::memset(&r, 0, sizeof r);
    r.d = d.d;
    r.t = no_rows();
    r.rows_d = batch->n_draft;
    r.rows_t = 0;
    r.B = batch->B;
    r.n_draft = batch->n_draft;
    r.draft_off = batch->draft_off;
    r.err = ws.err;
    r.epoch = next_epoch();
    r.work = ws.work;
    r.pre_eighths = 4;
    d.err = ws.err;
    d.epoch = r.epoch;
    // (the absent family's type is a placeholder: the draft's, one kernel variant)
    if ((e = launch_rowpass(r, draft->dtype, draft->dtype, s, sm_count_current(), true)) !=
        cudaSuccess)
      return cuda_fail(e);
  }
  if (kd > 0 || nd) {
    attach_kept(d, ws);
    if (kd > 0 && (e = launch_kept_sets(d.d, batch->n_draft, no_rows(), 0, prm, ws, s, true,
                                        batch, draft->dtype, draft->dtype)) != cudaSuccess)
      return cuda_fail(e);
    if (nd && (e = launch_nucleus_sets(d.d, batch->n_draft, no_rows(), 0, prm, ws, draft->dtype,
                                       draft->dtype, batch, nullptr, s, true)) != cudaSuccess)
      return cuda_fail(e);
    if ((e = launch_filter_q(d, s, true)) != cudaSuccess) return cuda_fail(e);
  } else if ((e = launch_decide(d, s, from_logits)) != cudaSuccess) {
    return cuda_fail(e);
  }
  return TT_OK;
}

tt_status tt_verify(const tt_batch* batch, const float* q_hat, const tt_logits* target,
                    const tt_logits* draft, const int32_t* map, const tt_params* prm,
                    void* workspace, size_t workspace_bytes, int32_t* accepted,
                    int32_t* next_token, float* p_hat, float* lse, int32_t* status,
                    void* stream) {
  if (!batch_ok(batch) || !params_ok(prm)) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!accepted || !next_token || !status) return TT_ERR_INVALID_ARG;
  if (batch->n_target > 0 && !q_hat) return TT_ERR_INVALID_ARG;
  const int32_t* tcols = batch->target_cols ? batch->target_cols : batch->target_ids;
  if (batch->n_target > 0 && !tcols) return TT_ERR_INVALID_ARG;
  if (!logits_ok(target, int64_t(batch->n_target) + batch->B)) return TT_ERR_INVALID_ARG;
  const bool full_q = prm->full_q != 0;
  if (full_q) {
    if (!logits_ok(draft, batch->n_draft) || draft->n_cols != target->n_cols) return TT_ERR_INVALID_ARG;
    if (batch->n_target > 0 && !map) return TT_ERR_INVALID_ARG;
  }
  // q_hat is given; the draft rows' filter matters only to the full-q residual
  const int kt = k_target(prm), kd = full_q ? k_draft(prm) : 0;
  const bool nt = nuc_target(prm), nd = full_q && nuc_draft(prm);
  // full-q: both families filtered or neither, and no nucleus family
  if (full_q && ((kd > 0 || nd) != (kt > 0 || nt) || nd || nt)) return TT_ERR_UNSUPPORTED;
  // a target penalty needs the target's top-k, and one-hot transfer
  const bool pt = pen_target(prm);
  if ((pt && kt == 0) || (full_q && (pt || pen_draft(prm)))) return TT_ERR_UNSUPPORTED;
  if (pt && !history_ok(batch->hist_off_t, batch->hist_cols_t, batch->n_hist_t))
    return TT_ERR_INVALID_ARG;
  const int V_d = full_q ? draft->n_cols : 0;
  const size_t need = workspace_layout(nullptr, batch->B, batch->n_draft, batch->n_target, V_d,
                                       target->n_cols, kd, kt, false, nt,
                                       pen_sizes(batch, false, pt)).bytes;
  if (!workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return TT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Workspace ws = workspace_layout(workspace, batch->B, batch->n_draft, batch->n_target, V_d,
                                  target->n_cols, kd, kt, false, nt, pen_sizes(batch, false, pt));
  cudaError_t e = ensure_loaded();
  if (e != cudaSuccess) return cuda_fail(e);
  if (full_q) {  // the residual needs the mapped draft rows' normalisers
    PrepArgs p;
    std::memset(&p, 0, sizeof p);
    p.B = batch->B;
    p.n_draft = batch->n_draft;
    p.n_target = batch->n_target;
    p.draft_off = batch->draft_off;
    p.target_off = batch->target_off;
    p.map = map;
    p.need = ws.need_d;
    p.work = ws.work;
    if ((e = launch_prep(p, s)) != cudaSuccess) return cuda_fail(e);
  }
  RowPassArgs r;
  std::memset(&r, 0, sizeof r);
  r.t = rowset(target, ws.part_t, nullptr, prm->temp_target);
  r.t.top_k = kt;
  r.t.cand = ws.cand_t;
  attach_nucleus(r.t, nt);
  attach_pen(r.t, pt, prm->rep_penalty_target, ws.pen_t, ws.pbase_t, ws.pcnt_t, ws.pstart_t);
  if (pt && (e = launch_pen_sets(batch, no_rows(), r.t, false, true, nullptr, tcols, ws, s)) !=
                cudaSuccess)
    return cuda_fail(e);
  r.rows_t = int64_t(batch->n_target) + batch->B;
  r.d = full_q ? rowset(draft, ws.part_d, ws.need_d, prm->temp_draft) : no_rows();
  r.d.top_k = kd;
  r.d.cand = ws.cand_d;
  r.rows_d = full_q ? batch->n_draft : 0;
  r.B = batch->B;
  r.n_target = batch->n_target;
  r.target_off = batch->target_off;
  r.target_cols = tcols;
  r.err = ws.err;
  r.epoch = next_epoch();
  r.work = full_q ? ws.work : nullptr;  // zeroed by the prep kernel
  r.pre_eighths = 4;
  // the first kernel of the chain starts only after the caller's work is
  // complete: it reads the logits before its grid-dependency wait
  if ((e = launch_rowpass(r, full_q ? draft->dtype : target->dtype, target->dtype, s,
                          sm_count_current(), full_q)) != cudaSuccess)
    return cuda_fail(e);

  DecideArgs d;
  std::memset(&d, 0, sizeof d);
  d.sm_count = sm_count_current();
  d.B = batch->B;
  d.n_draft = batch->n_draft;
  d.n_target = batch->n_target;
  d.max_k = batch->max_k;
  d.max_m = batch->max_m;
  d.full_q = full_q ? 1 : 0;
  d.draft_off = batch->draft_off;
  d.target_off = batch->target_off;
  d.target_cols = tcols;
  d.map = map;
  d.q_hat_in = q_hat;
  d.d = r.d;
  d.t = r.t;
  d.dt_d = full_q ? draft->dtype : TT_F32;
  d.dt_t = target->dtype;
  d.seed = prm->seed;
  d.request_base = prm->request_base;
  d.accepted = accepted;
  d.next_token = next_token;
  d.status = status;
  d.p_hat = p_hat;
  d.lse = lse;
  d.err = ws.err;
  d.epoch = r.epoch;
  d.top_p_d = prm->top_p_draft;
  d.top_p_t = prm->top_p_target;
  d.status_p = pt ? ws.pstatus : nullptr;
  if (kt > 0) {
    attach_kept(d, ws);
    if ((e = launch_kept_sets(r.d, r.rows_d, r.t, r.rows_t, prm, ws, s, true, batch, d.dt_d,
                              d.dt_t)) != cudaSuccess)
      return cuda_fail(e);
    if ((e = launch_decide_filtered(d, s, true)) != cudaSuccess) return cuda_fail(e);
  } else if (nt) {
    attach_kept(d, ws);
    if ((e = launch_nucleus_sets(no_rows(), 0, r.t, r.rows_t, prm, ws, target->dtype,
                                 target->dtype, batch, tcols, s, true)) != cudaSuccess)
      return cuda_fail(e);
    if ((e = launch_decide_nucleus(d, s, true)) != cudaSuccess) return cuda_fail(e);
  } else if ((e = launch_decide(d, s, true)) != cudaSuccess) {
    return cuda_fail(e);
  }
  return TT_OK;
}

tt_status tt_step(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                  const tt_logits* draft, const float* draft_probs, const tt_logits* target,
                  const tt_params* prm, void* workspace, size_t workspace_bytes,
                  const tt_step_out* out, void* stream) {
  size_t need = 0;
  const tt_status chk = step_check(batch, vd, vt, draft, draft_probs, target, prm, out, &need);
  if (chk != TT_OK || batch->B == 0) return chk;
  if (!workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return TT_ERR_INVALID_ARG;
  const bool full_q = prm->full_q != 0;
  const bool from_logits = draft_probs == nullptr || full_q;
  const int kd = from_logits ? k_draft(prm) : 0, kt = k_target(prm);
  const bool nd = from_logits && nuc_draft(prm), nt = nuc_target(prm);
  const bool pd = from_logits && pen_draft(prm), pt = pen_target(prm);
  const bool filtered = kd > 0 || kt > 0 || nd || nt;
  const int V_d = from_logits ? draft->n_cols : 0;
  const int32_t* dcols = batch->draft_cols ? batch->draft_cols : batch->draft_ids;
  const int32_t* tcols = batch->target_cols ? batch->target_cols : batch->target_ids;
  AlignArgs a;
  tt_status st = fill_align_args(batch, vd, vt, prm, a);
  if (st != TT_OK) return st;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Workspace ws = workspace_layout(workspace, batch->B, batch->n_draft, batch->n_target, V_d,
                                  target->n_cols, kd, kt, nd, nt, pen_sizes(batch, pd, pt));
  int32_t* map = out->map ? out->map : ws.map;
  a.path = out->path;
  a.path_len = out->path_len;
  a.cost = out->cost;
  a.map = map;
  a.status = out->status;
  a.need = from_logits ? ws.need_d : nullptr;
  a.work = ws.work;
  a.target_cols = tcols;
  a.excl = ws.excl;

  RowPassArgs r;
  std::memset(&r, 0, sizeof r);
  r.t = rowset(target, ws.part_t, nullptr, prm->temp_target);
  r.rows_t = int64_t(batch->n_target) + batch->B;
  r.d = from_logits ? rowset(draft, ws.part_d, ws.need_d, prm->temp_draft) : no_rows();
  r.rows_d = from_logits ? batch->n_draft : 0;
  r.t.top_k = kt;
  r.t.cand = ws.cand_t;
  attach_nucleus(r.t, nt);
  r.d.top_k = kd;
  r.d.cand = ws.cand_d;
  attach_nucleus(r.d, nd);
  attach_pen(r.d, pd, prm->rep_penalty_draft, ws.pen_d, ws.pbase_d, ws.pcnt_d, ws.pstart_d);
  attach_pen(r.t, pt, prm->rep_penalty_target, ws.pen_t, ws.pbase_t, ws.pcnt_t, ws.pstart_t);
  r.B = batch->B;
  r.n_target = batch->n_target;
  r.n_draft = batch->n_draft;
  r.target_off = batch->target_off;
  r.target_cols = tcols;
  r.draft_off = batch->draft_off;

  cudaError_t e = ensure_loaded();
  if (e != cudaSuccess) return cuda_fail(e);
  // the penalty's per-request sets, complete before the alignment (launched
  // without a dependent-launch attribute) and so before the row pass starts
  if ((pd || pt) &&
      (e = launch_pen_sets(batch, r.d, r.t, pd, pt, dcols, tcols, ws, s)) != cudaSuccess)
    return cuda_fail(e);
  record(prm, 0, s);
  if ((e = launch_align(a, s)) != cudaSuccess) return cuda_fail(e);
  record(prm, 1, s);

  r.err = ws.err;
  r.epoch = next_epoch();
  r.work = ws.work;       // zeroed by the alignment kernel
  r.pre_eighths = pre_wait_eighths(batch);
  r.excl_late = ws.excl;  // written by the alignment kernel
  // programmatic dependent launch: target rows stream while the alignment runs
  // (unless stage events sit between the kernels)
  const bool pdl = prm->events == nullptr;
  if ((e = launch_rowpass(r, from_logits ? draft->dtype : target->dtype, target->dtype, s,
                          sm_count_current(), pdl)) != cudaSuccess)
    return cuda_fail(e);
  record(prm, 2, s);

  DecideArgs d;
  std::memset(&d, 0, sizeof d);
  d.sm_count = sm_count_current();
  d.B = batch->B;
  d.n_draft = batch->n_draft;
  d.n_target = batch->n_target;
  d.max_k = batch->max_k;
  d.max_m = batch->max_m;
  d.full_q = full_q ? 1 : 0;
  d.draft_off = batch->draft_off;
  d.draft_cols = dcols;
  d.target_off = batch->target_off;
  d.target_cols = tcols;
  d.map = map;
  d.q_hat_in = nullptr;
  d.draft_probs = full_q ? nullptr : draft_probs;
  d.d = r.d;
  d.t = r.t;
  d.dt_d = from_logits ? draft->dtype : TT_F32;
  d.dt_t = target->dtype;
  d.status_in = out->status;
  d.seed = prm->seed;
  d.request_base = prm->request_base;
  d.accepted = out->accepted;
  d.next_token = out->next_token;
  d.status = out->status;
  d.q_hat_out = out->q_hat;
  d.p_hat = out->p_hat;
  d.lse = out->lse;
  d.err = ws.err;
  d.epoch = r.epoch;
  d.top_p_d = prm->top_p_draft;
  d.top_p_t = prm->top_p_target;
  d.status_p = (pd || pt) ? ws.pstatus : nullptr;
  if (!filtered) {
    d.warm_ctas = sm_count_current();  // the first CTA on each SM
    if ((e = launch_decide(d, s, pdl)) != cudaSuccess) return cuda_fail(e);
    record(prm, 3, s);
    return TT_OK;
  }
  // Filtered: the kept sets (top-k families from their lists, nucleus families
  // from their partials and logits); q_hat (from the draft rows' kept sets, or
  // as without filters), into out->q_hat or the workspace with its own status;
  // then the decision over the target rows (their kept sets, or the partials).
  float* qbuf = out->q_hat ? out->q_hat : ws.q_hat;
  attach_kept(d, ws);
  if ((kd > 0 || kt > 0) &&
      (e = launch_kept_sets(r.d, r.rows_d, r.t, r.rows_t, prm, ws, s, pdl, batch, d.dt_d,
                            d.dt_t)) != cudaSuccess)
    return cuda_fail(e);
  if ((nd || nt) &&
      (e = launch_nucleus_sets(r.d, r.rows_d, r.t, r.rows_t, prm, ws, d.dt_d, d.dt_t, batch, tcols,
                               s, pdl)) != cudaSuccess)
    return cuda_fail(e);
  DecideArgs q = d;
  q.mode_transfer_only = 1;
  q.status = ws.status;
  q.q_hat_out = qbuf;
  q.draft_probs = full_q ? nullptr : draft_probs;
  if (kd > 0 || nd) {
    if ((e = launch_filter_q(q, s, pdl)) != cudaSuccess) return cuda_fail(e);
  } else if ((e = launch_decide(q, s, pdl)) != cudaSuccess) {
    return cuda_fail(e);
  }
  d.q_hat_in = qbuf;
  d.q_hat_out = nullptr;
  d.draft_probs = nullptr;
  d.status_q = ws.status;
  if (kt > 0) {
    if ((e = launch_decide_filtered(d, s, pdl)) != cudaSuccess) return cuda_fail(e);
  } else if (nt) {
    if ((e = launch_decide_nucleus(d, s, pdl)) != cudaSuccess) return cuda_fail(e);
  } else if ((e = launch_decide(d, s, false)) != cudaSuccess) {
    // (this decision kernel reads q_hat before its grid-dependency wait)
    return cuda_fail(e);
  }
  record(prm, 3, s);
  return TT_OK;
}

size_t tt_sharded_workspace_bytes(const tt_batch* batch, const tt_shards* target) {
  if (!batch_ok(batch)) return 0;
  int32_t V = 0;
  if (!shards_ok(target, int64_t(batch->n_target) + batch->B, &V)) return 0;
  return shard_workspace(nullptr, batch, target).bytes;
}

tt_status tt_verify_sharded(const tt_batch* batch, const float* q_hat, const tt_shards* target,
                            const tt_params* prm, void* workspace, size_t workspace_bytes,
                            int32_t* accepted, int32_t* next_token, float* p_hat, float* lse,
                            float* summaries, int32_t* status, void* stream) {
  if (!batch_ok(batch) || !params_ok(prm)) return TT_ERR_INVALID_ARG;
  if (batch->B == 0) return TT_OK;
  if (!accepted || !next_token || !status) return TT_ERR_INVALID_ARG;
  if (batch->n_target > 0 && !q_hat) return TT_ERR_INVALID_ARG;
  const int32_t* tcols = batch->target_cols ? batch->target_cols : batch->target_ids;
  if (batch->n_target > 0 && !tcols) return TT_ERR_INVALID_ARG;
  const int64_t rows = int64_t(batch->n_target) + batch->B;
  int32_t V = 0;
  if (!shards_ok(target, rows, &V)) return TT_ERR_INVALID_ARG;
  // one-hot transfer, no filters
  if (prm->full_q != 0 || prm->top_k_target != 0 || prm->top_p_target < 1.f ||
      pen_target(prm))
    return TT_ERR_UNSUPPORTED;
  const ShardWorkspace ws0 = shard_workspace(nullptr, batch, target);
  if (!workspace || workspace_bytes < ws0.bytes ||
      (reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return TT_ERR_INVALID_ARG;
  const ShardWorkspace ws = shard_workspace(workspace, batch, target);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = ensure_loaded();
  if (e != cudaSuccess) return cuda_fail(e);

  ShardArgs a;
  std::memset(&a, 0, sizeof a);
  a.B = batch->B;
  a.n_target = batch->n_target;
  a.S = target->S;
  a.V = V;
  a.max_m = batch->max_m;
  a.rows = rows;
  a.target_off = batch->target_off;
  a.target_cols = tcols;
  a.excl = ws.excl;
  a.rec = ws.rec;
  a.work = ws.work;
  a.scale = log2e_over(prm->temp_target);
  a.q_hat = q_hat;
  a.seed = prm->seed;
  a.request_base = prm->request_base;
  a.err = ws.err;
  a.epoch = next_epoch();
  a.accepted = accepted;
  a.next_token = next_token;
  a.status = status;
  a.p_hat = p_hat;
  a.lse = lse;
  for (int k = 0; k < target->S; ++k) {
    const tt_logits& L = target->shards[k];
    ShardDesc& d = a.sh[k];
    d.data = static_cast<const char*>(L.data);
    d.stride_bytes = L.row_stride * (L.dtype == TT_F32 ? 4 : 2);
    d.V = L.n_cols;
    d.col0 = target->col0[k];
    d.nch = n_chunks(L.n_cols);
    d.dtype = L.dtype;
    d.part = ws.part[k];
  }
  if ((e = launch_shard_excl(a, s)) != cudaSuccess) return cuda_fail(e);
  // each shard's slice reduced by its own row pass (what one rank does). Passes
  // after the first start while the one before drains (programmatic dependent
  // launch): what they read before their grid-dependency wait -- the scored
  // columns and their zeroed work counters -- was written by the excl kernel,
  // which finished before the first pass, launched without the attribute, began.
  for (int k = 0; k < target->S; ++k) {
    RowPassArgs r;
    std::memset(&r, 0, sizeof r);
    r.t = rowset(&target->shards[k], ws.part[k], nullptr, prm->temp_target);
    r.rows_t = rows;
    r.d = no_rows();
    r.rows_d = 0;
    r.excl = ws.excl + int64_t(k) * rows;
    r.B = batch->B;
    r.n_target = batch->n_target;
    r.target_off = batch->target_off;
    r.target_cols = tcols;
    r.err = ws.err;
    r.epoch = a.epoch;
    r.pre_eighths = 4;
    r.work = reinterpret_cast<unsigned long long*>(reinterpret_cast<char*>(ws.work) +
                                                   size_t(k) * kWorkShards * kWorkStride *
                                                       sizeof(unsigned long long));
    if ((e = launch_rowpass(r, target->shards[k].dtype, target->shards[k].dtype, s,
                            sm_count_current(), k > 0)) != cudaSuccess)
      return cuda_fail(e);
  }
  if ((e = launch_shard_summary(a, s, sm_count_current())) != cudaSuccess) return cuda_fail(e);
  if (summaries &&
      (e = cudaMemcpyAsync(summaries, ws.rec, sizeof(ShardRec) * size_t(target->S) * rows,
                           cudaMemcpyDeviceToDevice, s)) != cudaSuccess)
    return cuda_fail(e);
  if ((e = launch_decide_sharded(a, s)) != cudaSuccess) return cuda_fail(e);
  return TT_OK;
}

const char* tt_status_string(tt_status s) {
  switch (s) {
    case TT_OK: return "ok";
    case TT_ERR_INVALID_ARG: return "invalid argument";
    case TT_ERR_UNSUPPORTED: return "unsupported configuration";
    case TT_ERR_CUDA: return "CUDA launch failure";
  }
  return "unknown status";
}

int32_t tt_last_cuda_error(void) { return g_last_cuda_error.load(); }

int32_t tt_version(void) { return 110; }

}  // extern "C"
