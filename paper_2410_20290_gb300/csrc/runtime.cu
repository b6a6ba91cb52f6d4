// libsr runtime: model loading, workspace, the generator / reward-model forward passes, and the
// Speculative Rejection controller (Algorithm 1, Section 4.2) behind the C ABI of sr.h.
//
// Host code here only enqueues kernels and reads a handful of control words (live count, free pages) to size
// launches; between page boundaries, where no memory trigger can fire, decode steps are enqueued back to back
// and the words are read once per boundary.  Every step of the method runs on the device: embedding, norms,
// GEMMs, RoPE + paged KV append, attention, sampling, partial-reward scoring (with the reward model's K/V kept
// across rounds when sr_set_rm_cache gives it a pool), the r_cut radix select, compaction and page release.
#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <cstdlib>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"

namespace sr {

static thread_local std::string g_msg;

// NVTX range on the host timeline around one phase of the controller (prompt prefill, a decode step, a scoring
// pass, a rejection round, the final scoring); a no-op unless a profiler such as Nsight Systems is attached.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

sr_status set_err(sr_status s, const char* fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_msg = buf;
  return s;
}

int* gemm_error_word();
void gemm_release_workspace(cudaStream_t st);

// LM head and sampling fused (16-bit models), only with SR_FUSED_SAMPLE=1: on GB300 the fused epilogue's Gumbel
// scan (a Philox call per 4 ids, one epilogue warp per SMSP) outlasts the GEMM's main loop, 1.63 against 1.10 ms
// for the LM head plus the separate sampling pass at 1024 rows, so by default the logits are stored and sampled
// in a pass of their own.
bool fused_sample_enabled() {
  static const bool on = [] {
    const char* e = getenv("SR_FUSED_SAMPLE");
    return e && e[0] == '1';
  }();
  return on;
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* e = getenv("SR_PDL");
    return !(e && e[0] == '0');
  }();
  return on;
}

namespace {

template <typename T>
sr_status grow(T*& p, size_t& cap, size_t n) {
  if (n <= cap && p) return SR_OK;
  if (p) cudaFree(p);
  p = nullptr;
  cap = 0;
  SR_CUDA(cudaMalloc(reinterpret_cast<void**>(&p), std::max<size_t>(n, 1) * sizeof(T)));
  cap = n;
  return SR_OK;
}

template <typename T>
sr_status grow_host(T*& p, size_t& cap, size_t n) {
  if (n <= cap && p) return SR_OK;
  if (p) cudaFreeHost(p);
  p = nullptr;
  cap = 0;
  SR_CUDA(cudaMallocHost(reinterpret_cast<void**>(&p), std::max<size_t>(n, 1) * sizeof(T)));
  cap = n;
  return SR_OK;
}

double now_ms() {
  return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now().time_since_epoch()).count();
}

// -------------------------------------------------------------------------------------------------
// per-kernel-class timing: CUDA events recorded on the launching stream around one launch in
// `period` of each class (chosen by a hash of the class's launch counter, so repeating launch patterns
// are sampled evenly), read back after the stream synchronises; every launch's work is counted
// -------------------------------------------------------------------------------------------------
struct Prof {
  bool on = false;
  int period = 1;
  std::vector<cudaEvent_t> ev;
  size_t used = 0;
  struct Rec {
    int cls;
    size_t a, b;
    double fl, by;
  };
  std::vector<Rec> recs;
  double ms[SR_KC_N] = {}, fl[SR_KC_N] = {}, by[SR_KC_N] = {};     // timed launches
  double fl_all[SR_KC_N] = {}, by_all[SR_KC_N] = {};                 // every launch
  long long n[SR_KC_N] = {}, n_all[SR_KC_N] = {};
  unsigned cnt[SR_KC_N] = {};

  cudaEvent_t take() {
    if (used == ev.size()) {
      cudaEvent_t e;
      cudaEventCreate(&e);
      ev.push_back(e);
    }
    return ev[used++];
  }
  long long begin(int cls, cudaStream_t st) {
    if (!on) return -1;
    const unsigned h = (cnt[cls]++ * 2654435761u) >> 16;
    if (period > 1 && h % (unsigned)period != 0) return -2;  // counted, not timed
    const size_t i = used;
    cudaEventRecord(take(), st);
    return (long long)i;
  }
  void end(long long i, int cls, cudaStream_t st, double f, double b) {
    if (i == -1) return;
    n_all[cls] += 1;
    fl_all[cls] += f;
    by_all[cls] += b;
    if (i < 0) return;
    const size_t j = used;
    cudaEventRecord(take(), st);
    recs.push_back({cls, (size_t)i, j, f, b});
  }
  void harvest() {  // every recorded event has completed (the stream was synchronised)
    for (const Rec& r : recs) {
      float t = 0.f;
      if (cudaEventElapsedTime(&t, ev[r.a], ev[r.b]) == cudaSuccess) ms[r.cls] += t;
      n[r.cls] += 1;
      fl[r.cls] += r.fl;
      by[r.cls] += r.by;
    }
    recs.clear();
    used = 0;
  }
  void reset() {
    recs.clear();
    used = 0;
    for (int c = 0; c < SR_KC_N; ++c) ms[c] = fl[c] = by[c] = fl_all[c] = by_all[c] = 0, n[c] = n_all[c] = 0, cnt[c] = 0;
  }
  ~Prof() {
    for (cudaEvent_t e : ev) cudaEventDestroy(e);
  }
};

// RAII timing scope for one launch (a no-op when profiling is off or pf is null)
struct Scope {
  Prof* p;
  long long i;
  int cls;
  cudaStream_t st;
  double f, b;
  Scope(Prof* p_, int cls_, cudaStream_t st_, double f_ = 0, double b_ = 0)
      : p(p_), i(p_ ? p_->begin(cls_, st_) : -1), cls(cls_), st(st_), f(f_), b(b_) {}
  ~Scope() {
    if (p) p->end(i, cls, st, f, b);
  }
};

// -------------------------------------------------------------------------------------------------
// model
// -------------------------------------------------------------------------------------------------
struct LayerW {
  void *attn_w, *attn_b, *wqkv, *wo, *mlp_w, *mlp_b, *wgu, *wdown;
};

struct Model {
  sr_model_desc d{};
  int esz = 2;
  int et = SR_DT_F16;  // device element type: SR_DT_F32 or SR_DT_F16
  char* blob = nullptr;
  void *tok_emb = nullptr, *pos_emb = nullptr, *final_w = nullptr, *final_b = nullptr, *lm_head = nullptr,
       *score_head = nullptr;
  std::vector<LayerW> L;
  float2* rope = nullptr;
  bool gated() const { return d.act != SR_ACT_GELU; }
  int qkv_dim() const { return (d.n_heads + 2 * d.n_kv_heads) * d.head_dim; }
  size_t kv_tok_elems() const { return (size_t)d.n_kv_heads * d.head_dim; }
};

sr_status check_desc(const sr_model_desc* m, const char* who) {
  if (!m) return set_err(SR_ERR_INVALID_ARG, "%s: null descriptor", who);
  if (m->n_layers < 1 || m->d_model < 1 || m->n_heads < 1 || m->n_kv_heads < 1 || m->head_dim < 2 ||
      m->ffn_dim < 1 || m->vocab < 1 || m->max_pos < 1 || m->window < 0)
    return set_err(SR_ERR_INVALID_ARG, "%s: non-positive dimension", who);
  if (m->norm != SR_NORM_RMS && m->norm != SR_NORM_LAYER) return set_err(SR_ERR_INVALID_ARG, "%s: norm", who);
  if (m->act < SR_ACT_SWIGLU || m->act > SR_ACT_GEGLU) return set_err(SR_ERR_INVALID_ARG, "%s: act", who);
  if (m->pos != SR_POS_ROPE && m->pos != SR_POS_LEARNED) return set_err(SR_ERR_INVALID_ARG, "%s: pos", who);
  if (m->dtype != SR_DT_F32 && m->dtype != SR_DT_BF16 && m->dtype != SR_DT_F16)
    return set_err(SR_ERR_INVALID_ARG, "%s: dtype", who);
  if (m->n_heads % m->n_kv_heads) return set_err(SR_ERR_UNSUPPORTED, "%s: n_heads %% n_kv_heads != 0", who);
  if (m->head_dim % 2) return set_err(SR_ERR_UNSUPPORTED, "%s: odd head_dim", who);
  if (m->ffn_dim % 32) return set_err(SR_ERR_UNSUPPORTED, "%s: ffn_dim %% 32 != 0", who);
  if (m->dtype != SR_DT_F32) {
    if (m->d_model % 64 || m->ffn_dim % 64 || m->vocab % 32 || (m->n_heads * m->head_dim) % 64)
      return set_err(SR_ERR_UNSUPPORTED,
                     "%s: 16-bit models need d_model, ffn_dim, n_heads*head_dim %% 64 == 0 and vocab %% 32 == 0", who);
    if (m->head_dim != 32 && m->head_dim != 64 && m->head_dim != 128 && m->head_dim != 256)
      return set_err(SR_ERR_UNSUPPORTED, "%s: head_dim %d (16-bit models need 32/64/128/256)", who, m->head_dim);
  }
  return SR_OK;
}

// Copy one model's blob (host or device; densely packed in the sr.h order) into an aligned
// device allocation; gate/up rows are interleaved in blocks of 16 for the fused GLU epilogues.
sr_status load_model(Model& M, const sr_model_desc* d, const void* src) {
  M.d = *d;
  M.esz = d->dtype == SR_DT_F32 ? 4 : 2;
  M.et = d->dtype == SR_DT_F32 ? SR_DT_F32 : SR_DT_F16;
  const size_t D = d->d_model, F = d->ffn_dim, V = d->vocab, E = M.esz;
  const bool ln = d->norm == SR_NORM_LAYER;
  struct T {
    size_t elems;
    void** dst;
    int kind;  // 0 plain, 1 gate (interleave into wgu), 2 up
  };
  std::vector<T> ts;
  M.L.assign(d->n_layers, LayerW{});
  ts.push_back({V * D, &M.tok_emb, 0});
  if (d->pos == SR_POS_LEARNED) ts.push_back({(size_t)d->max_pos * D, &M.pos_emb, 0});
  for (auto& l : M.L) {
    ts.push_back({D, &l.attn_w, 0});
    if (ln) ts.push_back({D, &l.attn_b, 0});
    ts.push_back({(size_t)((d->n_heads + 2 * d->n_kv_heads) * d->head_dim) * D, &l.wqkv, 0});
    ts.push_back({D * (size_t)(d->n_heads * d->head_dim), &l.wo, 0});
    ts.push_back({D, &l.mlp_w, 0});
    if (ln) ts.push_back({D, &l.mlp_b, 0});
    if (d->act != SR_ACT_GELU) {
      ts.push_back({F * D, &l.wgu, 1});
      ts.push_back({F * D, &l.wgu, 2});
    } else {
      ts.push_back({F * D, &l.wgu, 0});
    }
    ts.push_back({D * F, &l.wdown, 0});
  }
  ts.push_back({D, &M.final_w, 0});
  if (ln) ts.push_back({D, &M.final_b, 0});
  if (d->has_lm_head) ts.push_back({V * D, &M.lm_head, 0});
  if (d->has_scalar_head) ts.push_back({D, &M.score_head, 0});

  // destination layout: every tensor 256-byte aligned; a gated layer's gate+up share one [2F][D] slot
  size_t total = 0;
  std::vector<size_t> dst_off(ts.size());
  for (size_t i = 0; i < ts.size(); ++i) {
    if (ts[i].kind == 2) {
      dst_off[i] = dst_off[i - 1];
      continue;
    }
    total = (total + 255) & ~size_t(255);
    dst_off[i] = total;
    total += ts[i].elems * (ts[i].kind == 1 ? 2 : 1) * E;
  }
  SR_CUDA(cudaMalloc(&M.blob, total));
  size_t soff = 0;
  const char* s = static_cast<const char*>(src);
  for (size_t i = 0; i < ts.size(); ++i) {
    char* dst = M.blob + dst_off[i];
    *ts[i].dst = dst;
    const size_t bytes = ts[i].elems * E;
    if (ts[i].kind == 0) {
      SR_CUDA(cudaMemcpy(dst, s + soff, bytes, cudaMemcpyDefault));
    } else {
      // rows of block j (16 rows of D) land at rows 32j (gate) or 32j + 16 (up)
      const size_t row_bytes = D * E;
      char* base = dst + (ts[i].kind == 2 ? 16 * row_bytes : 0);
      SR_CUDA(cudaMemcpy2D(base, 32 * row_bytes, s + soff, 16 * row_bytes, 16 * row_bytes, F / 16,
                           cudaMemcpyDefault));
    }
    soff += bytes;
  }
  if (d->dtype == SR_DT_BF16) SR_TRY(launch_bf16_to_f16(M.blob, total / 2, 0));  // fp16 operands on the device
  if (d->pos == SR_POS_ROPE) {
    SR_CUDA(cudaMalloc(&M.rope, (size_t)d->max_pos * (d->head_dim / 2) * sizeof(float2)));
    SR_TRY(launch_rope_table(M.rope, d->max_pos, d->head_dim, (double)d->rope_theta, 0));
  }
  SR_CUDA(cudaDeviceSynchronize());
  return SR_OK;
}

void free_model(Model& M) {
  if (M.blob) cudaFree(M.blob);
  if (M.rope) cudaFree(M.rope);
  M.blob = nullptr;
  M.rope = nullptr;
}

// -------------------------------------------------------------------------------------------------
// per-model workspace (rows = tokens processed together)
// -------------------------------------------------------------------------------------------------
struct Work {
  size_t c_x = 0, c_xn = 0, c_qkv = 0, c_q = 0, c_k = 0, c_v = 0, c_att = 0, c_h = 0, c_gu = 0, c_part = 0;
  float* x = nullptr;
  char* xn = nullptr;
  float* qkv = nullptr;
  char *q = nullptr, *k = nullptr, *v = nullptr, *att = nullptr, *h = nullptr;
  float* gu = nullptr;
  float* part = nullptr;
  float* sseg = nullptr;  // streaming decode attention: segment partials and per-(row, kv head) counters
  int* scnt = nullptr;
  size_t c_sseg = 0, c_scnt = 0;
  int rows = 0;

  sr_status ensure(const Model& m, int n) {
    if (n <= rows) return SR_OK;
    const size_t R = n, D = m.d.d_model, E = m.esz, F = m.d.ffn_dim;
    const size_t HD = (size_t)m.d.n_heads * m.d.head_dim;
    SR_TRY(grow(x, c_x, R * D));
    SR_TRY(grow(xn, c_xn, R * D * E));
    SR_TRY(grow(qkv, c_qkv, R * m.qkv_dim()));
    SR_TRY(grow(q, c_q, R * HD * E));
    SR_TRY(grow(k, c_k, R * m.kv_tok_elems() * E));
    SR_TRY(grow(v, c_v, R * m.kv_tok_elems() * E));
    SR_TRY(grow(att, c_att, R * HD * E));
    SR_TRY(grow(h, c_h, R * F * E));
    if (m.et == SR_DT_F32) SR_TRY(grow(gu, c_gu, R * F * (m.gated() ? 2 : 1)));
    rows = n;
    return SR_OK;
  }
  void release() {
    void* ps[] = {x, xn, qkv, q, k, v, att, h, gu, part, sseg, scnt};
    for (void* p : ps)
      if (p) cudaFree(p);
    *this = Work();
  }
};

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

// Workspace of the streaming decode-attention kernel for b rows of Hq query heads (counters zeroed when
// they are first allocated; every launch leaves them zero).
sr_status stream_ws(Work& w, int b, int Hq, int pool_pages, cudaStream_t st, DecodeStreamWs* ws) {
  const int grid = num_sms();
  SR_TRY(grow(w.sseg, w.c_sseg, decode_stream_part_floats(grid, Hq)));
  if (w.c_scnt < (size_t)b * 8) {
    SR_TRY(grow(w.scnt, w.c_scnt, (size_t)b * 8));
    SR_CUDA(cudaMemsetAsync(w.scnt, 0, w.c_scnt * sizeof(int), st));
  }
  ws->seg_part = w.sseg;
  ws->seg_cnt = w.scnt;
  ws->grid = grid;
  ws->pool_pages = pool_pages;
  ws->err = tc_error_word();
  return SR_OK;
}

// Attention layout of one prefill call (packed sequences, optional shared prefix per layer).
struct PrefillPlan {
  const int* seq_off = nullptr;   // device [n_seq + 1]
  int n_seq = 1;
  const int* tile_seq = nullptr;  // device, bf16 path
  const int* tile_q0 = nullptr;
  int n_tiles = 0;
  int pos0 = 0;
  int n_pre = 0;
  const char* pre_k = nullptr;    // per-layer prefix K / V stores: base + l * layer_stride
  const char* pre_v = nullptr;
  size_t pre_layer_bytes = 0;
  // cached keys between the prefix and each sequence's own rows (reward-model KV kept across rounds)
  const char* cache_pool = nullptr;  // layer 0 page 0; layer l at + l * cache_layer_bytes
  size_t cache_layer_bytes = 0;
  const int* cache_pt = nullptr;
  int cache_pt_stride = 0;
  const int* seq_cand = nullptr;     // device [n_seq]
  const int* seq_cached = nullptr;   // device [n_seq]
  int max_cached = 0;
  int cache_pages = 0;               // pages per layer of the cache pool
};
// Where a prefill's per-layer K/V goes.
struct PrefillKv {
  char* store_k = nullptr;        // contiguous [rows][Hkv][dh] per layer at + l * store_layer_bytes
  char* store_v = nullptr;
  size_t store_layer_bytes = 0;
  void* pool = nullptr;           // paged pool (layer 0 page 0) or nullptr
  size_t pool_layer_bytes = 0;
  const int* page_row = nullptr;  // page table: one row for every input row (row_seq = null) ...
  int pt_stride = 0;
  const int* row_seq = nullptr;   // ... or row row_seq[r] for input row r (< 0: not stored)
  int pos_base = 0;               // positions held by the pages start here
};

sr_status linear(const Model& m, const void* A, const void* W, void* C, int M, int N, int K, int epi,
                 cudaStream_t st, Prof* pf = nullptr, int cls = SR_KC_GEMM_DECODE) {
  const double E = m.esz;
  const double out_b = (epi == EPI_F32) ? 4.0 * M * N : (epi == EPI_ADD_F32) ? 8.0 * M * N
                       : (epi == EPI_SWIGLU || epi == EPI_GEGLU) ? E * M * N / 2 : E * M * N;
  Scope sc(pf, cls, st, 2.0 * M * N * K, E * ((double)M * K + (double)N * K) + out_b);
  if (m.et == SR_DT_F16) return gemm_tc(SR_DT_F16, A, W, C, M, N, K, epi, st);
  return gemm_f32((const float*)A, (const float*)W, (float*)C, M, N, K, epi, st);
}

// MLP block: x += W_down act(W_gate h, W_up h) (or GELU(W_fc h)), h = Norm(x) already in w.xn
sr_status mlp(const Model& m, Work& w, const LayerW& lw, int M, cudaStream_t st, Prof* pf, int cls) {
  const int D = m.d.d_model, F = m.d.ffn_dim;
  if (m.et == SR_DT_F16) {
    const int epi = m.d.act == SR_ACT_SWIGLU ? EPI_SWIGLU : (m.d.act == SR_ACT_GEGLU ? EPI_GEGLU : EPI_GELU);
    SR_TRY(linear(m, w.xn, lw.wgu, w.h, M, m.gated() ? 2 * F : F, D, epi, st, pf, cls));
  } else {
    SR_TRY(linear(m, w.xn, lw.wgu, w.gu, M, m.gated() ? 2 * F : F, D, EPI_F32, st, pf, cls));
    Scope sc(pf, SR_KC_ELEMENTWISE, st);
    SR_TRY(launch_act(m.et, m.d.act, w.gu, M, F, w.h, st));
  }
  return linear(m, w.h, lw.wdown, w.x, M, D, F, EPI_ADD_F32, st, pf, cls);
}

// Prefill `M` rows (tokens / positions already on the device) through all layers; leaves the
// residual stream in w.x.
sr_status forward_prefill(const Model& m, Work& w, int M, const int* tok, const int* pos, const PrefillPlan& plan,
                          const PrefillKv& kv, cudaStream_t st, Prof* pf, int gcls, double attn_flops) {
  const sr_model_desc& d = m.d;
  const int D = d.d_model, Hq = d.n_heads, Hkv = d.n_kv_heads, dh = d.head_dim;
  SR_TRY(w.ensure(m, M));
  {
    Scope sc(pf, SR_KC_ELEMENTWISE, st);
    SR_TRY(launch_embed(m.et, m.tok_emb, m.pos_emb, tok, pos, M, D, w.x, st));
  }
  for (int l = 0; l < d.n_layers; ++l) {
    const LayerW& lw = m.L[l];
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_norm(m.et, d.norm, w.x, lw.attn_w, lw.attn_b, d.norm_eps, M, D, w.xn, st));
    }
    SR_TRY(linear(m, w.xn, lw.wqkv, w.qkv, M, m.qkv_dim(), D, EPI_F32, st, pf, gcls));
    char* kout = kv.store_k ? kv.store_k + l * kv.store_layer_bytes : w.k;
    char* vout = kv.store_v ? kv.store_v + l * kv.store_layer_bytes : w.v;
    KvSink sink{nullptr, nullptr, 0, nullptr};
    if (kv.pool)
      sink = KvSink{static_cast<char*>(kv.pool) + l * kv.pool_layer_bytes, kv.page_row, kv.pt_stride, kv.row_seq,
                    kv.pos_base};
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_rope_store(m.et, w.qkv, M, pos, m.rope, Hq, Hkv, dh, w.q, kout, vout, sink, st));
    }
    const char* pk = plan.n_pre ? plan.pre_k + l * plan.pre_layer_bytes : nullptr;
    const char* pv = plan.n_pre ? plan.pre_v + l * plan.pre_layer_bytes : nullptr;
    CachedKeys ck;
    if (plan.cache_pool) {
      ck.pool = plan.cache_pool + l * plan.cache_layer_bytes;
      ck.page_table = plan.cache_pt;
      ck.pt_stride = plan.cache_pt_stride;
      ck.seq_cand = plan.seq_cand;
      ck.seq_cached = plan.seq_cached;
      ck.pool_pages = plan.cache_pages;
    }
    const double kvb = (double)m.kv_tok_elems() * m.esz;
    {
      Scope sa(pf, SR_KC_ATTN_PREFILL, st, attn_flops,
               2.0 * M * (double)Hq * dh * m.esz + 2.0 * kvb * (M + (double)plan.n_pre));
      if (m.et == SR_DT_F16)
        SR_TRY(launch_prefill_attention(m.et, w.q, kout, vout, pk, pv, plan.n_pre, plan.seq_off, plan.n_seq,
                                        plan.tile_seq, plan.tile_q0, plan.n_tiles, plan.pos0, Hq, Hkv, dh, d.window,
                                        w.att, st, ck, M));
      else
        SR_TRY(launch_prefill_attention_f32((const float*)w.q, (const float*)kout, (const float*)vout,
                                            (const float*)pk, (const float*)pv, plan.n_pre, plan.seq_off, plan.n_seq,
                                            M, plan.pos0, Hq, Hkv, dh, d.window, (float*)w.att, st, ck,
                                            plan.max_cached));
    }
    SR_TRY(linear(m, w.att, lw.wo, w.x, M, D, Hq * dh, EPI_ADD_F32, st, pf, gcls));
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_norm(m.et, d.norm, w.x, lw.mlp_w, lw.mlp_b, d.norm_eps, M, D, w.xn, st));
    }
    SR_TRY(mlp(m, w, lw, M, st, pf, gcls));
  }
  return SR_OK;
}

// algorithmic flops of causal prefill attention: new row i of a sequence with c cached positions sees
// n_pre + c + i + 1 keys (c = 0 without a cache)
double prefill_attn_flops(const Model& m, const std::vector<int>& taus, size_t s0, size_t n, int n_pre,
                          const std::vector<int>* cached = nullptr) {
  double keys = 0;
  for (size_t j = s0; j < s0 + n; ++j) {
    const double c = cached ? (*cached)[j] : 0;
    const double t = taus[j] - c;  // new rows
    keys += t * (n_pre + c) + t * (t + 1) / 2;
  }
  return 4.0 * m.d.n_heads * m.d.head_dim * keys;  // per layer
}

}  // namespace
}  // namespace sr

// =================================================================================================
// context and batch state
// =================================================================================================
struct sr_ctx {
  int device = 0;
  cudaStream_t own = nullptr, st = nullptr;
  sr::Model gen, rm;
  sr::Work wg, wr;
  // KV pool of the generator: [layer][page][2][Hkv][16][dh]; the last physical page is the
  // prompt-tail template and never enters the free stack
  size_t pool_bytes_req = 0;
  char* pool = nullptr;
  int pool_cap_pages = 0;  // physical pages including the template page
  size_t page_elems = 0, page_bytes = 0;
  // reward-model prompt KV store [layer][P][Hkv][dh] (K and V)
  char *rm_pk = nullptr, *rm_pv = nullptr;
  size_t c_rm_pk = 0, c_rm_pv = 0;
  // reward-model KV of response positions kept across rounds: [layer][page][2][Hkv][16][dh], page table
  // rm_pt [N][rm_max_pages] (device; host mirror and free stack in the batch)
  size_t rm_cache_bytes_req = 0;
  char* rm_pool = nullptr;
  int rm_pool_cap = 0;          // pages allocated
  size_t rm_page_bytes = 0;
  int* rm_pt = nullptr;
  size_t c_rm_pt = 0;
  int* row_cand = nullptr;      // scoring rows -> candidate whose cache receives the row (-1: not stored)
  size_t c_row_cand = 0;
  // candidate state
  size_t c_len = 0, c_status = 0, c_tok = 0, c_pt = 0, c_live = 0, c_rset = 0, c_free = 0, c_tokin = 0, c_posin = 0,
         c_kvlen = 0, c_tail = 0, c_prow = 0, c_ids = 0, c_reward = 0, c_rr = 0, c_logits = 0, c_mask = 0, c_prompt = 0,
         c_iota = 0, c_meta = 0, c_hmeta = 0, c_out = 0, c_lastrow = 0, c_logits0 = 0;
  int *len = nullptr, *status = nullptr, *tok = nullptr, *pt = nullptr, *live = nullptr, *rset = nullptr,
      *free_stack = nullptr, *tok_in = nullptr, *pos_in = nullptr, *kv_len = nullptr, *tail_dst = nullptr,
      *prompt_row = nullptr, *ids = nullptr, *prompt = nullptr, *iota = nullptr, *meta = nullptr, *out_tok = nullptr,
      *last_row = nullptr;
  float *reward = nullptr, *rr = nullptr, *logits = nullptr, *logits0 = nullptr;
  sr::SampleRec* srec = nullptr;  // records of the LM head's sampling epilogue, [live rows][vocab / 64]
  size_t c_srec = 0;
  // self-likelihood reward (Section 5.3): running ln p(Y | X) per candidate id
  int reward_kind = SR_REWARD_MODEL;
  double* lp_sum = nullptr;
  size_t c_lpsum = 0;
  uint8_t* mask = nullptr;
  int* ctrl = nullptr;       // C_N ints
  float* ctrlf = nullptr;    // 4 floats (r_cut, score)
  int* h_ctrl = nullptr;     // pinned mirror
  float* h_ctrlf = nullptr;
  int* h_meta = nullptr;     // pinned staging for scoring plans
  float* d_score = nullptr;
  int* d_outlen = nullptr;
  sr::Prof prof;
};

// Host bookkeeping of the reward-model KV cache of one batch: which response positions of each
// candidate have their reward-model K/V in the cache pool, and the pages that hold them.
struct RmCache {
  bool on = false;
  int pages = 0, max_pages = 0;     // pool pages; pages per candidate (ceil(max_new / 16))
  std::vector<int> free_stack;      // LIFO, top at the back
  std::vector<int> cached;          // [N] positions 0 .. cached - 1 are in the cache
  std::vector<int> held;            // [N] pages held
  std::vector<int> pt;              // [N][max_pages] host mirror of the device page table
  long long reused = 0;             // positions read from the cache instead of recomputed
};

struct sr_batch {
  int P = 0, N = 0, max_new = 0, eos_id = -1, n_sh = 0, has_tail = 0, max_pages = 0, n_pages = 0;
  float temperature = 1.f, eos_bias = 0.f;
  uint64_t seed = 0;
  int n_live = 0, n_rset = 0, g = 0;  // g: tokens generated by every live candidate
  bool active = false;
  int reward_kind = SR_REWARD_MODEL;  // the context's reward kind when the batch started
  RmCache rmc;
};

namespace sr {
namespace {

sr_status read_ctrl(sr_ctx* c) {
  SR_CUDA(cudaMemcpyAsync(c->h_ctrl, c->ctrl, C_N * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaMemcpyAsync(c->h_ctrlf, c->ctrlf, 4 * sizeof(float), cudaMemcpyDeviceToHost, c->st));
  int* gerr = gemm_error_word();
  if (gerr) SR_CUDA(cudaMemcpyAsync(c->h_ctrl + C_N, gerr, sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaStreamSynchronize(c->st));
  if (gerr && c->h_ctrl[C_N] != 0)
    return set_err(SR_ERR_TIMEOUT, "a bounded device wait expired (code %d: 1-3 tensor-core GEMM, 10 decode attention)",
                   c->h_ctrl[C_N]);
  c->prof.harvest();
  if (c->h_ctrl[C_ERR] == E_POOL_EMPTY) return set_err(SR_ERR_OOM, "KV page pool exhausted");
  if (c->h_ctrl[C_ERR] == E_STATE) return set_err(SR_ERR_STATE, "no completed candidate");
  return SR_OK;
}

size_t kv_bytes_per_token(const Model& m) { return (size_t)m.d.n_layers * 2 * m.kv_tok_elems() * m.esz; }

int private_pages_full(int P, int max_new) { return (P + max_new - 2) / PAGE + 1 - P / PAGE; }

// Size the pool for this call: the caller's byte budget, or everything that N candidates need.
sr_status prepare_pool(sr_ctx* c, sr_batch& b) {
  const Model& g = c->gen;
  const size_t kvt = kv_bytes_per_token(g);
  long long pages;
  if (c->pool_bytes_req)
    pages = (long long)(c->pool_bytes_req / (PAGE * kvt));
  else
    pages = b.P / PAGE + (long long)b.N * private_pages_full(b.P, b.max_new);
  if (pages < 1) return set_err(SR_ERR_OOM, "KV pool smaller than one page");
  if (pages > (1ll << 30)) return set_err(SR_ERR_INVALID_ARG, "KV pool too large");
  b.n_pages = (int)pages;
  c->page_elems = (size_t)2 * g.d.n_kv_heads * PAGE * g.d.head_dim;
  c->page_bytes = c->page_elems * g.esz;
  if (c->pool_cap_pages < b.n_pages + 1) {
    if (c->pool) cudaFree(c->pool);
    c->pool = nullptr;
    c->pool_cap_pages = 0;
    SR_CUDA(cudaMalloc(&c->pool, (size_t)(b.n_pages + 1) * c->page_bytes * g.d.n_layers));
    c->pool_cap_pages = b.n_pages + 1;
  }
  return SR_OK;
}

size_t pool_layer_bytes(const sr_ctx* c) { return (size_t)c->pool_cap_pages * c->page_bytes; }

sr_status prepare_state(sr_ctx* c, sr_batch& b) {
  const size_t N = b.N;
  SR_TRY(grow(c->len, c->c_len, N));
  SR_TRY(grow(c->status, c->c_status, N));
  SR_TRY(grow(c->tok, c->c_tok, N * b.max_new));
  SR_TRY(grow(c->pt, c->c_pt, N * b.max_pages));
  SR_TRY(grow(c->live, c->c_live, N));
  SR_TRY(grow(c->rset, c->c_rset, N));
  SR_TRY(grow(c->free_stack, c->c_free, (size_t)b.n_pages));
  SR_TRY(grow(c->tok_in, c->c_tokin, N));
  SR_TRY(grow(c->pos_in, c->c_posin, N));
  SR_TRY(grow(c->kv_len, c->c_kvlen, N));
  SR_TRY(grow(c->tail_dst, c->c_tail, N));
  SR_TRY(grow(c->prompt_row, c->c_prow, (size_t)b.max_pages));
  SR_TRY(grow(c->ids, c->c_ids, N));
  SR_TRY(grow(c->reward, c->c_reward, N));
  SR_TRY(grow(c->lp_sum, c->c_lpsum, N));
  SR_TRY(grow(c->rr, c->c_rr, N));
  SR_TRY(grow(c->mask, c->c_mask, N));
  SR_TRY(grow(c->last_row, c->c_lastrow, N));
  SR_TRY(grow(c->out_tok, c->c_out, (size_t)b.max_new));
  SR_TRY(grow(c->logits0, c->c_logits0, (size_t)c->gen.d.vocab));
  SR_TRY(c->wg.ensure(c->gen, std::max<int>(b.N, b.P)));
  const int iota_n = std::max(c->gen.d.max_pos, c->rm.d.max_pos);
  if (c->c_iota < (size_t)iota_n) {
    std::vector<int> h(iota_n);
    for (int i = 0; i < iota_n; ++i) h[i] = i;
    SR_TRY(grow(c->iota, c->c_iota, (size_t)iota_n));
    SR_CUDA(cudaMemcpy(c->iota, h.data(), iota_n * sizeof(int), cudaMemcpyHostToDevice));
  }
  SR_CUDA(cudaMemsetAsync(c->status, 0xff, N * sizeof(int), c->st));
  SR_CUDA(cudaMemsetAsync(c->len, 0, N * sizeof(int), c->st));
  SR_CUDA(cudaMemsetAsync(c->lp_sum, 0, N * sizeof(double), c->st));
  SR_CUDA(cudaMemsetAsync(c->pt, 0, N * b.max_pages * sizeof(int), c->st));
  return SR_OK;
}

// single-sequence prefill plan over [0, P): seq_off = {0, P}, tiles of 64 rows
sr_status upload_single_plan(sr_ctx* c, int P, PrefillPlan& plan) {
  const int n_tiles = (P + 63) / 64;
  const size_t need = 2 + 2 * (size_t)n_tiles;
  SR_TRY(grow_host(c->h_meta, c->c_hmeta, need));
  SR_TRY(grow(c->meta, c->c_meta, need));
  SR_CUDA(cudaStreamSynchronize(c->st));  // staging may still feed an earlier copy
  c->h_meta[0] = 0;
  c->h_meta[1] = P;
  for (int t = 0; t < n_tiles; ++t) c->h_meta[2 + t] = 0, c->h_meta[2 + n_tiles + t] = t * 64;
  SR_CUDA(cudaMemcpyAsync(c->meta, c->h_meta, need * sizeof(int), cudaMemcpyHostToDevice, c->st));
  plan.seq_off = c->meta;
  plan.n_seq = 1;
  plan.tile_seq = c->meta + 2;
  plan.tile_q0 = c->meta + 2 + n_tiles;
  plan.n_tiles = n_tiles;
  plan.pos0 = 0;
  plan.n_pre = 0;
  return SR_OK;
}

// Prompt through the reward model (KV kept for every later scoring chunk) and through the
// generator (KV into the shared pages + tail template page; logits of the last position).
sr_status prefill_prompt(sr_ctx* c, sr_batch& b) {
  NvtxRange nv("sr prefill");
  const Model& g = c->gen;
  const Model& r = c->rm;
  const int P = b.P;
  PrefillPlan plan;
  SR_TRY(upload_single_plan(c, P, plan));
  Prof* pf = &c->prof;
  const std::vector<int> ptau(1, P);
  // reward model: prompt KV stored for the scoring passes (the self-likelihood reward needs none)
  if (b.reward_kind == SR_REWARD_MODEL) {
    const size_t rm_layer = (size_t)P * r.kv_tok_elems() * r.esz;
    SR_TRY(grow(c->rm_pk, c->c_rm_pk, rm_layer * r.d.n_layers));
    SR_TRY(grow(c->rm_pv, c->c_rm_pv, rm_layer * r.d.n_layers));
    PrefillKv kv;
    kv.store_k = c->rm_pk;
    kv.store_v = c->rm_pv;
    kv.store_layer_bytes = rm_layer;
    SR_TRY(forward_prefill(r, c->wr, P, c->prompt, c->iota, plan, kv, c->st, pf, SR_KC_GEMM_PROMPT,
                           prefill_attn_flops(r, ptau, 0, 1, 0)));
  }
  // generator: pages for the prompt, KV into them
  {
    Scope sc(pf, SR_KC_CONTROL, c->st);
    SR_TRY(ctl_prompt_pages(c->free_stack, c->ctrl, b.n_sh, b.has_tail, c->pool_cap_pages - 1, c->prompt_row,
                            c->st));
  }
  // the prompt's page ids are used by the KV writes below: stop with SR_ERR_OOM if the pool could not give them
  SR_TRY(read_ctrl(c));
  PrefillKv gkv;
  gkv.pool = c->pool;
  gkv.pool_layer_bytes = pool_layer_bytes(c);
  gkv.page_row = c->prompt_row;
  SR_TRY(forward_prefill(g, c->wg, P, c->prompt, c->iota, plan, gkv, c->st, pf, SR_KC_GEMM_PROMPT,
                         prefill_attn_flops(g, ptau, 0, 1, 0)));
  // logits of the last prompt position (the distribution of token 0 of every candidate)
  {
    Scope sc(pf, SR_KC_ELEMENTWISE, c->st);
    SR_TRY(launch_norm(g.et, g.d.norm, c->wg.x + (size_t)(P - 1) * g.d.d_model, g.final_w, g.final_b,
                       g.d.norm_eps, 1, g.d.d_model, c->wg.xn, c->st));
  }
  SR_TRY(linear(g, c->wg.xn, g.lm_head, c->logits0, 1, g.d.vocab, g.d.d_model, EPI_F32, c->st, pf,
                SR_KC_GEMM_PROMPT));
  return SR_OK;
}

// Admit candidates [start, start + count): pages, tail copy, token 0 from the prompt logits.
sr_status admit(sr_ctx* c, sr_batch& b, int start, int count) {
  const Model& g = c->gen;
  Prof* pf = &c->prof;
  {
    Scope sc(pf, SR_KC_CONTROL, c->st);
    SR_TRY(ctl_admit(start, count, b.n_sh, b.has_tail, c->prompt_row, c->pt, b.max_pages, c->len, c->status,
                     c->live, c->rset, c->free_stack, c->ctrl, c->tail_dst, c->st));
  }
  // the tail pages the admission popped are copied into below: stop with SR_ERR_OOM if it could not pop them
  if (b.has_tail) SR_TRY(read_ctrl(c));
  if (b.has_tail) {
    Scope sc(pf, SR_KC_ELEMENTWISE, c->st);
    SR_TRY(launch_copy_page(g.et, c->pool, (long long)(pool_layer_bytes(c) / g.esz), g.d.n_layers,
                            (int)c->page_elems, c->pool_cap_pages - 1, c->tail_dst, count, c->st));
  }
  {
    Scope sc(pf, SR_KC_SAMPLE, c->st, 0, 4.0 * g.d.vocab);
    SR_TRY(launch_sample(c->logits0, 0, count, g.d.vocab, c->live, nullptr, b.seed, b.temperature, b.eos_bias,
                         b.eos_id, nullptr, c->tok, b.max_new, c->len, c->status, c->st,
                         b.reward_kind == SR_REWARD_LOGPROB ? c->lp_sum : nullptr));
  }
  {
    Scope sc(pf, SR_KC_CONTROL, c->st);
    SR_TRY(ctl_step_end(b.P, b.n_sh, c->live, c->ctrl, c->len, c->status, c->pt, b.max_pages, c->free_stack,
                        c->st));
  }
  SR_TRY(read_ctrl(c));
  b.n_live = c->h_ctrl[C_NLIVE];
  b.n_rset = c->h_ctrl[C_NRSET];
  b.g = 1;
  return SR_OK;
}

// One batched decode step of every live candidate (positions P + g - 1), Eq. auto-regressive.
// sync = false enqueues the step without reading the control words back: the launches are sized for
// b.n_live, an upper bound of the live count (candidates only complete between rounds), and the kernels
// that write candidate state skip the slots past the device's live count.
sr_status decode_step(sr_ctx* c, sr_batch& b, float* logits_host, bool sync = true) {
  NvtxRange nv("sr decode step");
  const Model& m = c->gen;
  const sr_model_desc& d = m.d;
  Work& w = c->wg;
  const int n = b.n_live;
  const int D = d.d_model, Hq = d.n_heads, Hkv = d.n_kv_heads, dh = d.head_dim;
  SR_TRY(w.ensure(m, n));
  Prof* pf = &c->prof;
  cudaStream_t st = c->st;
  {
    Scope sc(pf, SR_KC_CONTROL, st);
    SR_TRY(ctl_step_begin(b.P, c->live, c->ctrl, c->len, c->pt, b.max_pages, c->free_stack, c->tok, b.max_new,
                          c->tok_in, c->pos_in, c->kv_len, st));
  }
  const int max_len = b.P + b.g;
  const int eff_len = d.window > 0 ? std::min(max_len, d.window) : max_len;
  // the prompt's full pages are shared by every candidate: a tensor-core prefix pass reads them once per 64
  // candidates (16-bit KV only)
  const int shared_pos = (m.et == SR_DT_F16 && b.n_sh > 0) ? PAGE * b.n_sh : 0;
  const int splits = decode_attention_slots(max_len, d.window, shared_pos);
  if (splits > 1) SR_TRY(grow(w.part, w.c_part, decode_attention_part_floats(n, Hq, dh, splits)));
  DecodeStreamWs sws;
  SR_TRY(stream_ws(w, n, Hq, c->pool_cap_pages, st, &sws));
  // algorithmic work of one decode-attention launch: the shared prompt KV once, each candidate's own KV,
  // q in and the output out
  const double kvb = 2.0 * Hkv * dh * m.esz;
  const double shared = (eff_len == max_len) ? (double)PAGE * b.n_sh : 0.0;
  const double attn_bytes = kvb * (shared + (double)n * (eff_len - shared)) + 2.0 * n * Hq * dh * m.esz;
  const double attn_flops = 4.0 * n * Hq * dh * (double)eff_len;
  {
    Scope sc(pf, SR_KC_ELEMENTWISE, st);
    SR_TRY(launch_embed(m.et, m.tok_emb, m.pos_emb, c->tok_in, c->pos_in, n, D, w.x, st));
  }
  for (int l = 0; l < d.n_layers; ++l) {
    const LayerW& lw = m.L[l];
    char* pool_l = c->pool + l * pool_layer_bytes(c);
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_norm(m.et, d.norm, w.x, lw.attn_w, lw.attn_b, d.norm_eps, n, D, w.xn, st));
    }
    SR_TRY(linear(m, w.xn, lw.wqkv, w.qkv, n, m.qkv_dim(), D, EPI_F32, st, pf, SR_KC_GEMM_DECODE));
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_rope_store(m.et, w.qkv, n, c->pos_in, m.rope, Hq, Hkv, dh, w.q, nullptr, nullptr,
                               KvSink{pool_l, c->pt, b.max_pages, c->live, 0, c->ctrl + C_NLIVE}, st));
    }
    {
      Scope sc(pf, SR_KC_ATTN_DECODE, st, attn_flops, attn_bytes);
      SR_TRY(launch_decode_attention(m.et, w.q, pool_l, c->pt, b.max_pages, c->live, c->kv_len, n, Hq, Hkv, dh,
                                     d.window, w.att, w.part, splits, st, shared_pos, max_len, nullptr, &sws));
    }
    SR_TRY(linear(m, w.att, lw.wo, w.x, n, D, Hq * dh, EPI_ADD_F32, st, pf, SR_KC_GEMM_DECODE));
    {
      Scope sc(pf, SR_KC_ELEMENTWISE, st);
      SR_TRY(launch_norm(m.et, d.norm, w.x, lw.mlp_w, lw.mlp_b, d.norm_eps, n, D, w.xn, st));
    }
    SR_TRY(mlp(m, w, lw, n, st, pf, SR_KC_GEMM_DECODE));
  }
  {
    Scope sc(pf, SR_KC_ELEMENTWISE, st);
    SR_TRY(launch_norm(m.et, d.norm, w.x, m.final_w, m.final_b, d.norm_eps, n, D, w.xn, st));
  }
  double* lp = b.reward_kind == SR_REWARD_LOGPROB ? c->lp_sum : nullptr;
  if (m.et == SR_DT_F16 && !logits_host && fused_sample_enabled()) {
    // LM head fused with sampling: the GEMM epilogue reduces each row's logits to one record per 64 ids
    const int nch = (d.vocab + SAMPLE_CHUNK - 1) / SAMPLE_CHUNK;
    SR_TRY(grow(c->srec, c->c_srec, (size_t)n * nch));
    {
      Scope sc(pf, SR_KC_GEMM_DECODE, st, 2.0 * n * d.vocab * D,
               m.esz * ((double)n * D + (double)d.vocab * D) + sizeof(SampleRec) * (double)n * nch);
      SR_TRY(lm_head_sample(false, w.xn, m.lm_head, n, d.vocab, D, c->live, c->len, b.seed, b.temperature,
                            b.eos_bias, b.eos_id, lp ? 1 : 0, c->srec, st));
    }
    Scope sc(pf, SR_KC_SAMPLE, st, 0, sizeof(SampleRec) * (double)n * nch);
    SR_TRY(launch_sample_reduce(c->srec, nch, n, c->live, b.eos_id, nullptr, c->tok, b.max_new, c->len, c->status,
                                st, lp, c->ctrl + C_NLIVE));
  } else {
    SR_TRY(grow(c->logits, c->c_logits, (size_t)n * d.vocab));
    SR_TRY(linear(m, w.xn, m.lm_head, c->logits, n, d.vocab, D, EPI_F32, st, pf, SR_KC_GEMM_DECODE));
    if (logits_host)
      SR_CUDA(cudaMemcpyAsync(logits_host, c->logits, (size_t)n * d.vocab * sizeof(float), cudaMemcpyDeviceToHost,
                              st));
    Scope sc(pf, SR_KC_SAMPLE, st, 0, 4.0 * n * d.vocab);
    SR_TRY(launch_sample(c->logits, d.vocab, n, d.vocab, c->live, nullptr, b.seed, b.temperature, b.eos_bias,
                         b.eos_id, nullptr, c->tok, b.max_new, c->len, c->status, st, lp, c->ctrl + C_NLIVE));
  }
  {
    Scope sc(pf, SR_KC_CONTROL, st);
    SR_TRY(ctl_step_end(b.P, b.n_sh, c->live, c->ctrl, c->len, c->status, c->pt, b.max_pages, c->free_stack, st));
  }
  b.g += 1;
  if (!sync) return SR_OK;
  SR_TRY(read_ctrl(c));
  b.n_live = c->h_ctrl[C_NLIVE];
  return SR_OK;
}

// Reward-model input rows of one scoring chunk: sequence j (candidate ids[j]) contributes its response
// tokens cached[j] .. cached[j] + n - 1 at positions P + cached[j] + i; row_cand receives the candidate id
// where the rows' K/V go to the cache (store[j] != 0), else -1.
__global__ void k_gather_rows(const int* __restrict__ ids, const int* __restrict__ off, const int* __restrict__ cached,
                              const int* __restrict__ store, const int* __restrict__ tok, int max_new, int P,
                              int* tok_rows, int* pos_rows, int* row_cand, int* last_row) {
  pdl_entry();
  const int j = blockIdx.x;
  const int id = ids[j], r0 = off[j], n = off[j + 1] - off[j];
  const int c = cached ? cached[j] : 0;
  const int rc = (row_cand && store[j]) ? id : -1;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    tok_rows[r0 + i] = tok[(size_t)id * max_new + c + i];
    pos_rows[r0 + i] = P + c + i;
    if (row_cand) row_cand[r0 + i] = rc;
  }
  if (threadIdx.x == 0) last_row[j] = r0 + n - 1;
}

// Self-likelihood reward of Section 5.3: s = ln p(Y^{<=tau} | X) / tau from the running sums the sampler
// keeps per candidate (tau = the tokens the candidate has, as for the reward model).
__global__ void k_mean_logprob(const int* __restrict__ ids_taus, int n, const double* __restrict__ lp_sum,
                               float* __restrict__ out) {
  pdl_entry();
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j < n) out[j] = (float)(lp_sum[ids_taus[j]] / (double)ids_taus[n + j]);
}

constexpr int CHUNK_ROWS = 16384;  // reward-model rows (response tokens) per scoring pass

// Give back the cache pages of every candidate that may not keep them (not in `keep`), in ascending
// (candidate id, page index) order.
void rm_cache_release(RmCache& rc, const std::vector<char>& keep) {
  for (size_t id = 0; id < rc.held.size(); ++id) {
    if (keep[id] || rc.held[id] == 0) continue;
    for (int p = 0; p < rc.held[id]; ++p) rc.free_stack.push_back(rc.pt[id * rc.max_pages + p]);
    rc.held[id] = 0;
    rc.cached[id] = 0;
  }
}

// Rewards s(X ++ Y_k^{<= tau_k}) for candidates ids_h[0..n) with tau_k = taus[k] (Eq.
// partial.reward.set); results into rewards_dev[0..n).  Each chunk runs the reward model over the
// packed response tokens, attending to the prompt KV computed once at prefill.  With the reward-model
// cache on, positions already in the cache are not run again: a candidate's new rows start at its cached
// length (one row at least) and attend to the prompt, its cached pages and each other; when `store` is
// set (a rejection round), the new rows' K/V are added to the cache for every candidate the free pages
// can serve, in ascending id order, so that a later round or the final scoring reads them.
sr_status score(sr_ctx* c, sr_batch& b, const std::vector<int>& ids_h, const std::vector<int>& taus,
                float* rewards_dev, bool store, long long* rm_rows = nullptr) {
  NvtxRange nv("sr score");
  const Model& r = c->rm;
  const int n = (int)ids_h.size();
  if (n == 0) return SR_OK;
  if (b.reward_kind == SR_REWARD_LOGPROB) {
    SR_CUDA(cudaStreamSynchronize(c->st));  // the pinned staging buffer may still feed an earlier copy
    SR_TRY(grow_host(c->h_meta, c->c_hmeta, 2 * (size_t)n));
    SR_TRY(grow(c->meta, c->c_meta, 2 * (size_t)n));
    for (int j = 0; j < n; ++j) c->h_meta[j] = ids_h[j], c->h_meta[n + j] = taus[j];
    SR_CUDA(cudaMemcpyAsync(c->meta, c->h_meta, 2 * (size_t)n * sizeof(int), cudaMemcpyHostToDevice, c->st));
    Scope sc(&c->prof, SR_KC_CONTROL, c->st);
    launch_k(k_mean_logprob, (n + 255) / 256, 256, 0, c->st, (const int*)c->meta, n, (const double*)c->lp_sum,
             rewards_dev);
    SR_LAUNCH();
    return SR_OK;
  }
  const size_t rm_layer = (size_t)b.P * r.kv_tok_elems() * r.esz;
  RmCache& rc = b.rmc;
  SR_CUDA(cudaStreamSynchronize(c->st));  // host staging and the page-table mirror may feed earlier copies
  // new rows per candidate, and where their K/V go
  std::vector<int> cached(n, 0), newr(n), st_flag(n, 0);
  if (rc.on) {
    std::vector<char> keep(rc.held.size(), 0);
    for (int id : ids_h) keep[id] = 1;
    rm_cache_release(rc, keep);
    for (int j = 0; j < n; ++j) cached[j] = std::min(rc.cached[ids_h[j]], taus[j] - 1);
    if (store) {
      for (int j = 0; j < n; ++j) {
        const int id = ids_h[j];
        const int need = std::max(0, (taus[j] + PAGE - 1) / PAGE - rc.held[id]);
        if (need > (int)rc.free_stack.size()) continue;
        for (int p = 0; p < need; ++p) {
          rc.pt[(size_t)id * rc.max_pages + rc.held[id] + p] = rc.free_stack.back();
          rc.free_stack.pop_back();
        }
        rc.held[id] += need;
        st_flag[j] = 1;
      }
      SR_CUDA(cudaMemcpyAsync(c->rm_pt, rc.pt.data(), rc.pt.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
    }
  }
  long long rows_total = 0;
  int max_cached = 0;
  for (int j = 0; j < n; ++j) {
    newr[j] = taus[j] - cached[j];
    rows_total += newr[j];
    rc.reused += cached[j];
    max_cached = std::max(max_cached, cached[j]);
  }
  if (rm_rows) *rm_rows += rows_total;
  // plan chunks on the host: [ids | off | cached | store | tiles_seq | tiles_q0] per chunk in one pinned buffer
  struct Chunk {
    int s0, ns, rows, n_tiles;
    size_t meta;
  };
  std::vector<Chunk> chunks;
  size_t meta_len = 0;
  for (int s = 0; s < n;) {
    Chunk ch{s, 0, 0, 0, meta_len};
    while (s < n && (ch.ns == 0 || ch.rows + newr[s] <= CHUNK_ROWS)) {
      ch.rows += newr[s];
      ch.n_tiles += (newr[s] + 63) / 64;
      ++ch.ns;
      ++s;
    }
    meta_len += 3 * (size_t)ch.ns + (ch.ns + 1) + 2 * (size_t)ch.n_tiles;
    chunks.push_back(ch);
  }
  SR_TRY(grow_host(c->h_meta, c->c_hmeta, meta_len));
  SR_TRY(grow(c->meta, c->c_meta, meta_len));
  int max_rows = 0;
  for (const Chunk& ch : chunks) {
    int* h = c->h_meta + ch.meta;
    int* hid = h;
    int* hoff = h + ch.ns;
    int* hc = hoff + ch.ns + 1;
    int* hst = hc + ch.ns;
    int* hts = hst + ch.ns;
    int* htq = hts + ch.n_tiles;
    int o = 0, t = 0;
    for (int j = 0; j < ch.ns; ++j) {
      hid[j] = ids_h[ch.s0 + j];
      hoff[j] = o;
      hc[j] = cached[ch.s0 + j];
      hst[j] = st_flag[ch.s0 + j];
      const int nr = newr[ch.s0 + j];
      for (int q0 = 0; q0 < nr; q0 += 64) hts[t] = j, htq[t] = q0, ++t;
      o += nr;
    }
    hoff[ch.ns] = o;
    max_rows = std::max(max_rows, ch.rows);
  }
  SR_CUDA(cudaMemcpyAsync(c->meta, c->h_meta, meta_len * sizeof(int), cudaMemcpyHostToDevice, c->st));
  SR_TRY(c->wr.ensure(r, max_rows));
  if (rc.on) SR_TRY(grow(c->row_cand, c->c_row_cand, (size_t)max_rows));
  // token / position rows for the largest chunk
  int *tok_rows = nullptr, *pos_rows = nullptr;
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&tok_rows), (size_t)max_rows * sizeof(int), c->st));
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&pos_rows), (size_t)max_rows * sizeof(int), c->st));
  const size_t cache_layer = (size_t)rc.pages * c->rm_page_bytes;
  sr_status status = SR_OK;
  for (const Chunk& ch : chunks) {
    const int* did = c->meta + ch.meta;
    const int* doff = did + ch.ns;
    const int* dc = doff + ch.ns + 1;
    const int* dst = dc + ch.ns;
    const int* dts = dst + ch.ns;
    const int* dtq = dts + ch.n_tiles;
    {
      Scope sc(&c->prof, SR_KC_ELEMENTWISE, c->st);
      launch_k(k_gather_rows, ch.ns, 128, 0, c->st, did, doff, rc.on ? dc : (const int*)nullptr, dst, c->tok,
               b.max_new, b.P, tok_rows, pos_rows, rc.on ? c->row_cand : (int*)nullptr, c->last_row);
    }
    if ((status = [&]() -> sr_status { SR_LAUNCH(); return SR_OK; }()) != SR_OK) break;
    PrefillPlan plan;
    plan.seq_off = doff;
    plan.n_seq = ch.ns;
    plan.tile_seq = dts;
    plan.tile_q0 = dtq;
    plan.n_tiles = ch.n_tiles;
    plan.pos0 = b.P;
    plan.n_pre = b.P;
    plan.pre_k = c->rm_pk;
    plan.pre_v = c->rm_pv;
    plan.pre_layer_bytes = rm_layer;
    PrefillKv kv;
    if (rc.on) {
      plan.cache_pool = c->rm_pool;
      plan.cache_layer_bytes = cache_layer;
      plan.cache_pt = c->rm_pt;
      plan.cache_pt_stride = rc.max_pages;
      plan.seq_cand = did;
      plan.seq_cached = dc;
      plan.max_cached = max_cached;
      plan.cache_pages = rc.pages;
      if (store) {
        kv.pool = c->rm_pool;
        kv.pool_layer_bytes = cache_layer;
        kv.page_row = c->rm_pt;
        kv.pt_stride = rc.max_pages;
        kv.row_seq = c->row_cand;
        kv.pos_base = b.P;
      }
    }
    if ((status = forward_prefill(r, c->wr, ch.rows, tok_rows, pos_rows, plan, kv, c->st, &c->prof, SR_KC_GEMM_SCORE,
                                  prefill_attn_flops(r, taus, ch.s0, ch.ns, b.P, &cached))) != SR_OK)
      break;
    Scope sc(&c->prof, SR_KC_ELEMENTWISE, c->st);
    if ((status = launch_score_head(r.et, r.d.norm, c->wr.x, c->last_row, ch.ns, r.final_w, r.final_b,
                                    r.d.norm_eps, r.score_head, r.d.d_model, rewards_dev + ch.s0, c->st)) != SR_OK)
      break;
  }
  cudaFreeAsync(tok_rows, c->st);
  cudaFreeAsync(pos_rows, c->st);
  if (status == SR_OK && rc.on && store)
    for (int j = 0; j < n; ++j)
      if (st_flag[j]) rc.cached[ids_h[j]] = taus[j];
  return status;
}

// ids and lengths of the round batch (host copies), plus their status
sr_status read_rset(sr_ctx* c, sr_batch& b, std::vector<int>& ids, std::vector<int>& taus, std::vector<int>* st) {
  ids.resize(b.n_rset);
  taus.resize(b.n_rset);
  std::vector<int> lens(b.N), stat(b.N);
  SR_CUDA(cudaMemcpyAsync(ids.data(), c->rset, b.n_rset * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaMemcpyAsync(lens.data(), c->len, b.N * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaMemcpyAsync(stat.data(), c->status, b.N * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaStreamSynchronize(c->st));
  for (int i = 0; i < b.n_rset; ++i) taus[i] = lens[ids[i]];
  if (st) {
    st->resize(b.n_rset);
    for (int i = 0; i < b.n_rset; ++i) (*st)[i] = stat[ids[i]];
  }
  return SR_OK;
}

sr_status validate_common(const sr_ctx* c, int P, int N, int max_new, float temperature, int eos_id) {
  if (!c) return set_err(SR_ERR_INVALID_ARG, "null context");
  if (P < 1 || N < 1 || N > MAX_BATCH || max_new < 1)
    return set_err(SR_ERR_INVALID_ARG, "need P >= 1, 1 <= N <= %d, max_new >= 1", MAX_BATCH);
  if (P + max_new > c->gen.d.max_pos || P + max_new > c->rm.d.max_pos)
    return set_err(SR_ERR_INVALID_ARG, "P + max_new exceeds max_pos");
  if (!(temperature > 0.f) || !std::isfinite(temperature)) return set_err(SR_ERR_INVALID_ARG, "temperature must be > 0");
  if (eos_id < -1 || eos_id >= c->gen.d.vocab) return set_err(SR_ERR_INVALID_ARG, "eos_id out of range");
  return SR_OK;
}

// The reward-model KV cache of this batch (off unless sr_set_rm_cache gave it bytes and the reward model
// scores): pages = floor(bytes / (16 positions x the reward model's KV bytes per position)).
sr_status prepare_rm_cache(sr_ctx* c, sr_batch& b) {
  RmCache& rc = b.rmc;
  rc = RmCache();
  if (c->rm_cache_bytes_req == 0 || b.reward_kind != SR_REWARD_MODEL) return SR_OK;
  const Model& r = c->rm;
  c->rm_page_bytes = (size_t)2 * r.d.n_kv_heads * PAGE * r.d.head_dim * r.esz;
  const size_t per_page = c->rm_page_bytes * r.d.n_layers;
  const long long pages = (long long)(c->rm_cache_bytes_req / per_page);
  if (pages < 1) return SR_OK;  // too small for one page: no cache
  if (pages > (1ll << 30)) return set_err(SR_ERR_INVALID_ARG, "reward-model cache too large");
  if (c->rm_pool_cap != (int)pages) {
    if (c->rm_pool) cudaFree(c->rm_pool);
    c->rm_pool = nullptr;
    c->rm_pool_cap = 0;
    SR_CUDA(cudaMalloc(&c->rm_pool, (size_t)pages * per_page));
    c->rm_pool_cap = (int)pages;
  }
  rc.on = true;
  rc.pages = (int)pages;
  rc.max_pages = (b.max_new + PAGE - 1) / PAGE;
  rc.free_stack.resize(rc.pages);
  for (int i = 0; i < rc.pages; ++i) rc.free_stack[i] = i;  // LIFO: the first page taken is the highest
  rc.cached.assign(b.N, 0);
  rc.held.assign(b.N, 0);
  rc.pt.assign((size_t)b.N * rc.max_pages, 0);
  SR_TRY(grow(c->rm_pt, c->c_rm_pt, rc.pt.size()));
  return SR_OK;
}

sr_status begin(sr_ctx* c, sr_batch& b, const int32_t* prompt, bool prompt_on_device, int P, int N, int max_new,
                float temperature, float eos_bias, int eos_id, uint64_t seed) {
  SR_TRY(validate_common(c, P, N, max_new, temperature, eos_id));
  c->prof.reset();
  b = sr_batch();
  b.reward_kind = c->reward_kind;
  b.P = P, b.N = N, b.max_new = max_new, b.temperature = temperature, b.eos_bias = eos_bias, b.eos_id = eos_id;
  b.seed = seed;
  b.n_sh = P / PAGE;
  b.has_tail = P % PAGE != 0;
  b.max_pages = (P + max_new - 1) / PAGE + 1;
  SR_TRY(prepare_pool(c, b));
  SR_TRY(prepare_state(c, b));
  SR_TRY(prepare_rm_cache(c, b));
  SR_TRY(grow(c->prompt, c->c_prompt, (size_t)P));
  SR_CUDA(cudaMemcpyAsync(c->prompt, prompt, P * sizeof(int), prompt_on_device ? cudaMemcpyDeviceToDevice
                                                                              : cudaMemcpyHostToDevice, c->st));
  SR_TRY(ctl_pool_init(c->free_stack, b.n_pages, c->ctrl, c->st));
  SR_TRY(prefill_prompt(c, b));
  b.active = true;
  return SR_OK;
}

// Algorithm 1 for a prepared batch; outputs stay on the device (c->out_tok, d_outlen, d_score).
sr_status run_sr(sr_ctx* c, sr_batch& b, float alpha, const sr_schedule* sched, sr_stats* st) {
  NvtxRange nv("sr generate");
  const bool pool_mode = sched->kind == SR_SCHED_POOL_FULL;
  std::vector<int> taus_sched(sched->tau, sched->tau + (sched->kind == SR_SCHED_FIXED ? sched->n_tau : 0));
  sr_stats S;
  memset(&S, 0, sizeof S);
  S.pool_pages = b.n_pages;
  double t0 = now_ms();
  SR_CUDA(cudaStreamSynchronize(c->st));
  S.ms_prefill = now_ms() - t0;
  // waves: alpha = 0 under a memory trigger is Best-of-N in pool-sized waves
  std::vector<std::pair<int, int>> waves;
  if (pool_mode && alpha == 0.f) {
    SR_TRY(read_ctrl(c));
    const int per = private_pages_full(b.P, b.max_new);
    const int free_pages = c->h_ctrl[C_TOP];
    const int w = per == 0 ? b.N : std::min(b.N, free_pages / per);
    if (w <= 0) return set_err(SR_ERR_OOM, "KV pool cannot hold one candidate to max_new");
    for (int s = 0; s < b.N; s += w) waves.push_back({s, std::min(w, b.N - s)});
  } else {
    waves.push_back({0, b.N});
  }
  S.waves = (int)waves.size();
  std::vector<int> ids, taus, stat;
  for (auto& wv : waves) {
    double ta = now_ms();
    SR_TRY(admit(c, b, wv.first, wv.second));
    S.ms_decode += now_ms() - ta;
    while (b.n_live > 0) {
      const bool need = (b.P + b.g - 1) % PAGE == 0;
      if (alpha > 0.f) {
        bool trig;
        if (pool_mode) {
          trig = need && c->h_ctrl[C_TOP] < b.n_live;
        } else {
          trig = std::find(taus_sched.begin(), taus_sched.end(), b.g) != taus_sched.end();
        }
        if (trig) {
          double ts = now_ms();
          SR_TRY(read_rset(c, b, ids, taus, nullptr));
          SR_TRY(score(c, b, ids, taus, c->rr, true, &S.rm_tokens));
          SR_CUDA(cudaStreamSynchronize(c->st));
          double tsel = now_ms();
          S.ms_score += tsel - ts;
          {
            NvtxRange nv("sr reject and compact");
            Scope sc(&c->prof, SR_KC_CONTROL, c->st);
            SR_TRY(ctl_round(b.P, b.n_sh, alpha, pool_mode && need ? 1 : 0, c->rr, c->rset, c->live, c->ctrl,
                             c->ctrlf, c->status, c->len, c->reward, c->pt, b.max_pages, c->free_stack, nullptr,
                             c->st));
          }
          SR_TRY(read_ctrl(c));
          S.ms_select += now_ms() - tsel;
          if (S.rounds < SR_MAX_ROUNDS) {
            S.b_per_round[S.rounds] = b.n_rset;
            S.step_per_round[S.rounds] = b.g;
            S.k_per_round[S.rounds] = c->h_ctrl[C_K];
            S.accepted_per_round[S.rounds] = c->h_ctrl[C_NACC];
            S.r_cut_per_round[S.rounds] = c->h_ctrlf[0];
          }
          S.k_raised += c->h_ctrl[C_KRAISED];
          S.rounds++;
          b.n_live = c->h_ctrl[C_NLIVE];
          b.n_rset = c->h_ctrl[C_NRSET];
          if (b.n_live == 0) break;
        }
      }
      if (need && c->h_ctrl[C_TOP] < b.n_live) return set_err(SR_ERR_OOM, "KV pool cannot hold the next decode step");
      // Between page boundaries no memory trigger can fire and no step needs a page, so the next steps are
      // enqueued without reading the live count back; the host syncs before a step that opens a page and
      // when the candidates reach max_new.
      const bool sync = (b.P + b.g) % PAGE == 0 || b.g + 1 >= b.max_new;
      double td = now_ms();
      SR_TRY(decode_step(c, b, nullptr, sync));
      S.ms_decode += now_ms() - td;
      S.decode_steps++;
    }
    // completed candidates not scored in a round: final rewards
    double tf = now_ms();
    SR_TRY(read_rset(c, b, ids, taus, &stat));
    std::vector<int> pid, ptau;
    for (size_t i = 0; i < ids.size(); ++i)
      if (stat[i] == ST_PENDING) pid.push_back(ids[i]), ptau.push_back(taus[i]);
    if (!pid.empty()) {
      SR_TRY(score(c, b, pid, ptau, c->rr, false, &S.rm_tokens));
      SR_CUDA(cudaMemcpyAsync(c->ids, pid.data(), pid.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
      SR_TRY(ctl_mark_done(c->ids, c->rr, (int)pid.size(), c->status, c->reward, c->st));
      SR_CUDA(cudaStreamSynchronize(c->st));
    }
    S.ms_score += now_ms() - tf;
  }
  S.rm_tokens += b.P;
  if (b.reward_kind != SR_REWARD_MODEL) S.rm_tokens = 0;  // the generator scored itself
  S.rm_tokens_cached = b.rmc.reused;
  SR_TRY(ctl_final(b.N, c->status, c->reward, c->tok, b.max_new, c->len, c->out_tok, c->d_outlen, c->ctrlf + 1,
                   c->ctrl, c->st));
  SR_TRY(read_ctrl(c));
  std::vector<int> lens(b.N), stv(b.N);
  SR_CUDA(cudaMemcpy(lens.data(), c->len, b.N * sizeof(int), cudaMemcpyDeviceToHost));
  SR_CUDA(cudaMemcpy(stv.data(), c->status, b.N * sizeof(int), cudaMemcpyDeviceToHost));
  for (int i = 0; i < b.N; ++i) {
    S.gen_tokens += lens[i];
    S.n_completed += stv[i] == ST_DONE;
  }
  c->prof.harvest();
  for (int k = 0; k < SR_KC_N; ++k) {
    S.kern_ms[k] = c->prof.ms[k];
    S.kern_timed[k] = c->prof.n[k];
    S.kern_timed_flops[k] = c->prof.fl[k];
    S.kern_timed_bytes[k] = c->prof.by[k];
    S.kern_launches[k] = c->prof.n_all[k];
    S.kern_flops[k] = c->prof.fl_all[k];
    S.kern_bytes[k] = c->prof.by_all[k];
  }
  S.best_id = c->h_ctrl[C_BEST];
  S.peak_pages_in_use = c->h_ctrl[C_PEAK];
  S.ms_total = now_ms() - t0 + S.ms_prefill;
  if (st) *st = S;
  b.active = false;
  return SR_OK;
}

}  // namespace
}  // namespace sr

using namespace sr;

// =================================================================================================
// C ABI
// =================================================================================================
extern "C" {

const char* sr_last_error(void) { return g_msg.c_str(); }

sr_status sr_init(sr_ctx** out, const sr_model_desc* gen, const void* gen_w, const sr_model_desc* rm,
                  const void* rm_w, size_t kv_pool_bytes, int page_tokens, int device) {
  if (!out) return set_err(SR_ERR_INVALID_ARG, "null output pointer");
  *out = nullptr;
  SR_TRY(check_desc(gen, "generator"));
  SR_TRY(check_desc(rm, "reward model"));
  if (!gen_w || !rm_w) return set_err(SR_ERR_INVALID_ARG, "null weights");
  if (!gen->has_lm_head) return set_err(SR_ERR_INVALID_ARG, "generator needs an LM head");
  if (!rm->has_scalar_head) return set_err(SR_ERR_INVALID_ARG, "reward model needs a scalar head");
  if ((gen->dtype == SR_DT_F32) != (rm->dtype == SR_DT_F32))
    return set_err(SR_ERR_INVALID_ARG, "generator and reward model must both be fp32 or both 16-bit");
  if (gen->vocab != rm->vocab) return set_err(SR_ERR_INVALID_ARG, "generator and reward model vocabularies differ");
  if (page_tokens != PAGE) return set_err(SR_ERR_INVALID_ARG, "page_tokens must be 16");
  int ndev = 0;
  SR_CUDA(cudaGetDeviceCount(&ndev));
  if (device < 0 || device >= ndev) return set_err(SR_ERR_INVALID_ARG, "device %d not present", device);
  SR_CUDA(cudaSetDevice(device));
  sr_ctx* c = new sr_ctx();
  c->device = device;
  c->pool_bytes_req = kv_pool_bytes;
  auto fail = [&](sr_status s) {
    sr_destroy(c);
    return s;
  };
  if (cudaStreamCreateWithFlags(&c->own, cudaStreamNonBlocking) != cudaSuccess)
    return fail(set_err(SR_ERR_CUDA, "stream creation failed"));
  c->st = c->own;
  sr_status s;
  if ((s = load_model(c->gen, gen, gen_w)) != SR_OK) return fail(s);
  if ((s = load_model(c->rm, rm, rm_w)) != SR_OK) return fail(s);
  if (cudaMalloc(&c->ctrl, C_N * sizeof(int)) != cudaSuccess || cudaMalloc(&c->ctrlf, 4 * sizeof(float)) ||
      cudaMallocHost(&c->h_ctrl, (C_N + 1) * sizeof(int)) || cudaMallocHost(&c->h_ctrlf, 4 * sizeof(float)) ||
      cudaMalloc(&c->d_score, sizeof(float)) || cudaMalloc(&c->d_outlen, sizeof(int)))
    return fail(set_err(SR_ERR_OOM, "control buffers"));
  cudaMemset(c->ctrl, 0, C_N * sizeof(int));
  *out = c;
  return SR_OK;
}

void sr_destroy(sr_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->device);
  if (c->st) cudaStreamSynchronize(c->st);
  if (c->own) cudaStreamSynchronize(c->own);
  // the GEMM's split-K buffers of this context's streams
  if (c->own) gemm_release_workspace(c->own);
  if (c->st && c->st != c->own) gemm_release_workspace(c->st);
  free_model(c->gen);
  free_model(c->rm);
  c->wg.release();
  c->wr.release();
  void* dev[] = {c->pool, c->rm_pk, c->rm_pv, c->rm_pool, c->rm_pt, c->row_cand, c->len, c->status, c->tok, c->pt, c->live, c->rset, c->free_stack,
                 c->tok_in, c->pos_in, c->kv_len, c->tail_dst, c->prompt_row, c->ids, c->prompt, c->iota, c->meta,
                 c->out_tok, c->last_row, c->reward, c->rr, c->logits, c->logits0, c->mask, c->ctrl, c->ctrlf, c->d_score,
                 c->d_outlen, c->srec};
  for (void* p : dev)
    if (p) cudaFree(p);
  if (c->h_ctrl) cudaFreeHost(c->h_ctrl);
  if (c->h_ctrlf) cudaFreeHost(c->h_ctrlf);
  if (c->h_meta) cudaFreeHost(c->h_meta);
  if (c->own) cudaStreamDestroy(c->own);
  delete c;
}

sr_status sr_auto_b_init(const sr_model_desc* gen, size_t kv_pool_bytes, int P, int tau_min, int n_max,
                         int* n_out) {
  if (!gen || !n_out) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (P < 1 || tau_min < 1 || n_max < 1 || gen->n_layers < 1 || gen->n_kv_heads < 1 || gen->head_dim < 1)
    return set_err(SR_ERR_INVALID_ARG, "sr_auto_b_init: bad argument");
  const size_t esz = gen->dtype == SR_DT_F32 ? 4 : 2;
  const size_t kvt = (size_t)gen->n_layers * 2 * gen->n_kv_heads * gen->head_dim * esz;
  const long long pages = (long long)(kv_pool_bytes / (PAGE * kvt));
  const long long avail = pages - P / PAGE;
  const int per = private_pages_full(P, tau_min);
  long long n = avail < 0 ? 0 : (per == 0 ? n_max : std::min<long long>(n_max, avail / per));
  *n_out = (int)n;
  if (n < 1) return set_err(SR_ERR_OOM, "sr_auto_b_init: the pool cannot hold one candidate to tau_min tokens");
  return SR_OK;
}

sr_status sr_set_rm_cache(sr_ctx* c, size_t bytes) {
  if (!c) return set_err(SR_ERR_INVALID_ARG, "null context");
  c->rm_cache_bytes_req = bytes;
  if (bytes == 0 && c->rm_pool) {
    SR_CUDA(cudaSetDevice(c->device));
    SR_CUDA(cudaStreamSynchronize(c->st));
    cudaFree(c->rm_pool);
    c->rm_pool = nullptr;
    c->rm_pool_cap = 0;
  }
  return SR_OK;
}

sr_status sr_set_reward(sr_ctx* c, int kind) {
  if (!c) return set_err(SR_ERR_INVALID_ARG, "null context");
  if (kind != SR_REWARD_MODEL && kind != SR_REWARD_LOGPROB) return set_err(SR_ERR_INVALID_ARG, "unknown reward kind");
  c->reward_kind = kind;
  return SR_OK;
}

sr_status sr_set_profiling(sr_ctx* c, int enable) {
  if (!c) return set_err(SR_ERR_INVALID_ARG, "null context");
  if (enable < 0) return set_err(SR_ERR_INVALID_ARG, "profiling period must be >= 0");
  c->prof.on = enable != 0;
  c->prof.period = enable > 0 ? enable : 1;
  c->prof.reset();
  return SR_OK;
}

sr_status sr_set_stream(sr_ctx* c, void* stream) {
  if (!c) return set_err(SR_ERR_INVALID_ARG, "null context");
  c->st = stream ? static_cast<cudaStream_t>(stream) : c->own;
  return SR_OK;
}

static sr_status check_sched(const sr_schedule* sched, float alpha) {
  if (!sched) return set_err(SR_ERR_INVALID_ARG, "null schedule");
  if (!(alpha >= 0.f && alpha <= 1.f)) return set_err(SR_ERR_INVALID_ARG, "alpha must be in [0, 1]");
  if (sched->kind == SR_SCHED_FIXED) {
    if (sched->n_tau < 0 || (sched->n_tau > 0 && !sched->tau)) return set_err(SR_ERR_INVALID_ARG, "bad tau list");
    for (int i = 0; i < sched->n_tau; ++i)
      if (sched->tau[i] < 1 || (i && sched->tau[i] <= sched->tau[i - 1]))
        return set_err(SR_ERR_INVALID_ARG, "tau values must be ascending and >= 1");
  } else if (sched->kind != SR_SCHED_POOL_FULL) {
    return set_err(SR_ERR_INVALID_ARG, "unknown schedule kind");
  }
  return SR_OK;
}

static sr_status generate_impl(sr_ctx* c, const int32_t* prompt, bool dev, int P, int N, float alpha,
                               const sr_schedule* sched, int max_new, float temperature, float eos_bias, int eos_id,
                               uint64_t seed, sr_stats* st) {
  SR_TRY(check_sched(sched, alpha));
  SR_CUDA(cudaSetDevice(c->device));
  sr_batch b;
  SR_TRY(begin(c, b, prompt, dev, P, N, max_new, temperature, eos_bias, eos_id, seed));
  return run_sr(c, b, alpha, sched, st);
}

sr_status sr_generate(sr_ctx* c, const int32_t* prompt, int P, int N, float alpha, const sr_schedule* sched,
                      int max_new, float temperature, float eos_bias, int eos_id, uint64_t seed, int32_t* out_tokens,
                      int* out_len, float* out_score, sr_stats* st) {
  if (!c || !prompt || !out_tokens || !out_len || !out_score) return set_err(SR_ERR_INVALID_ARG, "null argument");
  SR_TRY(generate_impl(c, prompt, false, P, N, alpha, sched, max_new, temperature, eos_bias, eos_id, seed, st));
  int L = 0;
  SR_CUDA(cudaMemcpyAsync(&L, c->d_outlen, sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaMemcpyAsync(out_score, c->ctrlf + 1, sizeof(float), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaStreamSynchronize(c->st));
  SR_CUDA(cudaMemcpyAsync(out_tokens, c->out_tok, L * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaStreamSynchronize(c->st));
  *out_len = L;
  return SR_OK;
}

sr_status sr_generate_dev(sr_ctx* c, const int32_t* prompt_dev, int P, int N, float alpha, const sr_schedule* sched,
                          int max_new, float temperature, float eos_bias, int eos_id, uint64_t seed,
                          int32_t* out_tokens_dev, int* out_len_dev, float* out_score_dev, sr_stats* st,
                          void* stream) {
  if (!c || !prompt_dev || !out_tokens_dev || !out_len_dev || !out_score_dev)
    return set_err(SR_ERR_INVALID_ARG, "null argument");
  cudaStream_t prev = c->st;
  if (stream) c->st = static_cast<cudaStream_t>(stream);
  sr_status s = generate_impl(c, prompt_dev, true, P, N, alpha, sched, max_new, temperature, eos_bias, eos_id, seed, st);
  if (s == SR_OK) {
    cudaMemcpyAsync(out_tokens_dev, c->out_tok, (size_t)max_new * sizeof(int), cudaMemcpyDeviceToDevice, c->st);
    cudaMemcpyAsync(out_len_dev, c->d_outlen, sizeof(int), cudaMemcpyDeviceToDevice, c->st);
    cudaMemcpyAsync(out_score_dev, c->ctrlf + 1, sizeof(float), cudaMemcpyDeviceToDevice, c->st);
    if (cudaStreamSynchronize(c->st) != cudaSuccess) s = set_err(SR_ERR_CUDA, "output copy failed");
  }
  c->st = prev;
  return s;
}

// ---- component calls ----
sr_status sr_batch_begin(sr_ctx* c, const int32_t* prompt, int P, int N, int max_new, float temperature,
                         float eos_bias, int eos_id, uint64_t seed, sr_batch** out) {
  if (!c || !prompt || !out) return set_err(SR_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  SR_CUDA(cudaSetDevice(c->device));
  sr_batch* b = new sr_batch();
  sr_status s = begin(c, *b, prompt, false, P, N, max_new, temperature, eos_bias, eos_id, seed);
  if (s == SR_OK) s = admit(c, *b, 0, N);
  if (s != SR_OK) {
    delete b;
    return s;
  }
  *out = b;
  return SR_OK;
}

sr_status sr_decode_step(sr_ctx* c, sr_batch* b, float* logits_out) {
  if (!c || !b) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (!b->active || b->n_live == 0) return set_err(SR_ERR_STATE, "no live candidate");
  const bool need = (b->P + b->g - 1) % PAGE == 0;
  if (need && c->h_ctrl[C_TOP] < b->n_live) return set_err(SR_ERR_OOM, "KV pool cannot hold the next decode step");
  return decode_step(c, *b, logits_out);
}

sr_status sr_score_partial(sr_ctx* c, sr_batch* b, float* rewards, int* b_out) {
  if (!c || !b || !rewards) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (!b->active) return set_err(SR_ERR_STATE, "batch not active");
  std::vector<int> ids, taus;
  SR_TRY(read_rset(c, *b, ids, taus, nullptr));
  SR_TRY(score(c, *b, ids, taus, c->rr, true));
  SR_CUDA(cudaMemcpyAsync(rewards, c->rr, ids.size() * sizeof(float), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaStreamSynchronize(c->st));
  if (b_out) *b_out = (int)ids.size();
  return SR_OK;
}

sr_status sr_reject_compact(sr_ctx* c, sr_batch* b, const float* rewards, float alpha, float* r_cut_out,
                            int32_t* accepted_ids_out, int* b_out, int* b_live_out) {
  if (!c || !b || !rewards) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (!b->active || b->n_rset == 0) return set_err(SR_ERR_STATE, "empty round batch");
  if (!(alpha >= 0.f && alpha <= 1.f)) return set_err(SR_ERR_INVALID_ARG, "alpha must be in [0, 1]");
  std::vector<int> ids(b->n_rset);
  SR_CUDA(cudaMemcpyAsync(ids.data(), c->rset, b->n_rset * sizeof(int), cudaMemcpyDeviceToHost, c->st));
  SR_CUDA(cudaMemcpyAsync(c->rr, rewards, b->n_rset * sizeof(float), cudaMemcpyHostToDevice, c->st));
  SR_TRY(ctl_round(b->P, b->n_sh, alpha, 0, c->rr, c->rset, c->live, c->ctrl, c->ctrlf, c->status, c->len, c->reward,
                   c->pt, b->max_pages, c->free_stack, c->mask, c->st));
  std::vector<uint8_t> mask(b->n_rset);
  SR_CUDA(cudaMemcpyAsync(mask.data(), c->mask, b->n_rset, cudaMemcpyDeviceToHost, c->st));
  SR_TRY(read_ctrl(c));
  int na = 0;
  for (int i = 0; i < b->n_rset; ++i)
    if (mask[i]) {
      if (accepted_ids_out) accepted_ids_out[na] = ids[i];
      ++na;
    }
  if (r_cut_out) *r_cut_out = c->h_ctrlf[0];
  if (b_out) *b_out = na;
  b->n_live = c->h_ctrl[C_NLIVE];
  b->n_rset = c->h_ctrl[C_NRSET];
  if (b_live_out) *b_live_out = b->n_live;
  return SR_OK;
}

sr_status sr_batch_query(sr_ctx* c, const sr_batch* b, int32_t* ids_live, int32_t* lengths, int32_t* status,
                         int32_t* tokens, int32_t* page_table, int32_t* free_stack, int* n_live, int* free_top,
                         int* max_pages) {
  if (!c || !b) return set_err(SR_ERR_INVALID_ARG, "null argument");
  SR_TRY(read_ctrl(c));
  const size_t N = b->N;
  if (ids_live) SR_CUDA(cudaMemcpy(ids_live, c->live, b->n_live * sizeof(int), cudaMemcpyDeviceToHost));
  if (lengths) SR_CUDA(cudaMemcpy(lengths, c->len, N * sizeof(int), cudaMemcpyDeviceToHost));
  if (status) SR_CUDA(cudaMemcpy(status, c->status, N * sizeof(int), cudaMemcpyDeviceToHost));
  if (tokens) SR_CUDA(cudaMemcpy(tokens, c->tok, N * b->max_new * sizeof(int), cudaMemcpyDeviceToHost));
  if (page_table) SR_CUDA(cudaMemcpy(page_table, c->pt, N * b->max_pages * sizeof(int), cudaMemcpyDeviceToHost));
  if (free_stack) SR_CUDA(cudaMemcpy(free_stack, c->free_stack, c->h_ctrl[C_TOP] * sizeof(int), cudaMemcpyDeviceToHost));
  if (n_live) *n_live = c->h_ctrl[C_NLIVE];
  if (free_top) *free_top = c->h_ctrl[C_TOP];
  if (max_pages) *max_pages = b->max_pages;
  return SR_OK;
}

void sr_batch_end(sr_ctx* c, sr_batch* b) {
  (void)c;
  delete b;
}

// ---- kernel-level entry points ----
sr_status sr_k_sample(const float* logits, long long ld, int b, int vocab, const int32_t* orig_ids,
                      const int32_t* steps, uint64_t seed, float temperature, float eos_bias, int eos_id,
                      int32_t* tokens_out, void* stream, double* logprob_sum) {
  if (!logits || !orig_ids || !steps || !tokens_out || b < 0 || vocab < 1)
    return set_err(SR_ERR_INVALID_ARG, "sr_k_sample: bad argument");
  return launch_sample(logits, ld, b, vocab, orig_ids, steps, seed, temperature, eos_bias, eos_id, tokens_out,
                       nullptr, 0, nullptr, nullptr, static_cast<cudaStream_t>(stream), logprob_sum);
}

sr_status sr_k_lm_head_sample(int dtype, const void* x, const void* W, int M, int vocab, int K,
                              const int32_t* orig_ids, const int32_t* lens, uint64_t seed, float temperature,
                              float eos_bias, int eos_id, int32_t* tokens_out, void* stream) {
  if (!x || !W || !orig_ids || !lens || !tokens_out || M < 0 || vocab < 1)
    return set_err(SR_ERR_INVALID_ARG, "sr_k_lm_head_sample: bad argument");
  if (dtype != SR_DT_F16 && dtype != SR_DT_BF16)
    return set_err(SR_ERR_INVALID_ARG, "sr_k_lm_head_sample: dtype must be SR_DT_F16 or SR_DT_BF16");
  if (M == 0) return SR_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int nch = (vocab + SAMPLE_CHUNK - 1) / SAMPLE_CHUNK;
  SampleRec* rec = nullptr;
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&rec), (size_t)M * nch * sizeof(SampleRec), st));
  sr_status s = lm_head_sample(dtype == SR_DT_BF16, x, W, M, vocab, K, orig_ids, lens, seed, temperature, eos_bias,
                               eos_id, 0, rec, st);
  if (s == SR_OK)
    s = launch_sample_reduce(rec, nch, M, orig_ids, eos_id, tokens_out, nullptr, 0, const_cast<int*>(lens), nullptr,
                             st);
  cudaFreeAsync(rec, st);
  return s;
}

sr_status sr_k_rcut(const float* rewards, int b, float alpha, int k_override, float* r_cut_out, uint8_t* mask_out,
                    void* stream) {
  if (!rewards || !r_cut_out || !mask_out) return set_err(SR_ERR_INVALID_ARG, "sr_k_rcut: null argument");
  if (!(alpha >= 0.f && alpha <= 1.f)) return set_err(SR_ERR_INVALID_ARG, "alpha must be in [0, 1]");
  return launch_rcut(rewards, b, alpha, k_override, r_cut_out, mask_out, static_cast<cudaStream_t>(stream));
}

sr_status sr_k_gemm(int dtype, const void* A, const void* W, void* C, int M, int N, int K, int epilogue,
                    void* stream) {
  if (!A || !W || !C) return set_err(SR_ERR_INVALID_ARG, "sr_k_gemm: null argument");
  if (epilogue < 0 || epilogue > EPI_GELU) return set_err(SR_ERR_INVALID_ARG, "sr_k_gemm: bad epilogue");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (dtype == SR_DT_BF16 || dtype == SR_DT_F16) return gemm_tc(dtype, A, W, C, M, N, K, epilogue, st);
  if (dtype == SR_DT_F32) return gemm_f32((const float*)A, (const float*)W, (float*)C, M, N, K, epilogue, st);
  return set_err(SR_ERR_INVALID_ARG, "sr_k_gemm: bad dtype");
}

sr_status sr_k_decode_attention(int dtype, const void* q, const void* pool, const int32_t* page_table, int pt_stride,
                                const int32_t* orig_ids, const int32_t* lens, int b, int n_heads, int n_kv_heads,
                                int head_dim, int window, int shared_pos, void* out, void* stream) {
  if (!q || !pool || !page_table || !orig_ids || !lens || !out) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (b < 0 || n_kv_heads < 1 || n_heads < 1 || head_dim < 1) return set_err(SR_ERR_INVALID_ARG, "bad shape");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // partials for sequences longer than one split: sized for the longest possible context
  std::vector<int> h(b);
  if (b) SR_CUDA(cudaMemcpy(h.data(), lens, b * sizeof(int), cudaMemcpyDeviceToHost));
  int mx = 1;
  for (int x : h) mx = std::max(mx, x);
  if (shared_pos < 0 || shared_pos % PAGE) return set_err(SR_ERR_INVALID_ARG, "shared_pos must be a multiple of 16");
  for (int x : h)
    if (x <= shared_pos) return set_err(SR_ERR_INVALID_ARG, "every length must exceed shared_pos");
  const int splits = decode_attention_slots(mx, window, shared_pos);
  float* part = nullptr;
  if (splits > 1) SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&part),
                                          decode_attention_part_floats(b, n_heads, head_dim, splits) * sizeof(float), st));
  // the streaming kernel's workspace.  The pool's size is not an argument here, so its tensor map spans the
  // largest page count a 2D map can address; the kernel reads only the pages the page table names, as the
  // per-row kernels do.
  DecodeStreamWs ws;
  ws.grid = num_sms();
  ws.err = tc_error_word();
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&ws.seg_part),
                          decode_stream_part_floats(ws.grid, n_heads) * sizeof(float), st));
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&ws.seg_cnt), (size_t)std::max(b, 1) * 8 * sizeof(int), st));
  SR_CUDA(cudaMemsetAsync(ws.seg_cnt, 0, (size_t)std::max(b, 1) * 8 * sizeof(int), st));
  ws.pool_pages = (int)(((1u << 31) - 1) / (2u * 8u * PAGE));
  sr_status s = launch_decode_attention(dtype, q, pool, page_table, pt_stride, orig_ids, lens, b, n_heads, n_kv_heads,
                                        head_dim, window, out, part, splits, st, shared_pos, mx, nullptr, &ws);
  if (part) cudaFreeAsync(part, st);
  cudaFreeAsync(ws.seg_part, st);
  cudaFreeAsync(ws.seg_cnt, st);
  return s;
}

sr_status sr_k_prefill_attention(int dtype, const void* q, const void* k, const void* v, const void* k_pre,
                                 const void* v_pre, int n_pre, const int32_t* seq_off, int n_seq, int pos0,
                                 int n_heads, int n_kv_heads, int head_dim, int window, void* out, void* stream) {
  if (!q || !k || !v || !seq_off || !out || n_seq < 1) return set_err(SR_ERR_INVALID_ARG, "null argument");
  if (n_pre > 0 && (!k_pre || !v_pre)) return set_err(SR_ERR_INVALID_ARG, "prefix pointers missing");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  std::vector<int> off(n_seq + 1);
  SR_CUDA(cudaMemcpy(off.data(), seq_off, (n_seq + 1) * sizeof(int), cudaMemcpyDeviceToHost));
  std::vector<int> ts, tq;
  for (int j = 0; j < n_seq; ++j)
    for (int q0 = 0; q0 < off[j + 1] - off[j]; q0 += 64) ts.push_back(j), tq.push_back(q0);
  const int nt = (int)ts.size();
  if (nt == 0) return SR_OK;
  int* d = nullptr;
  SR_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&d), 2 * nt * sizeof(int), st));
  std::vector<int> hcat(ts);
  hcat.insert(hcat.end(), tq.begin(), tq.end());
  SR_CUDA(cudaMemcpyAsync(d, hcat.data(), 2 * nt * sizeof(int), cudaMemcpyHostToDevice, st));
  sr_status s = launch_prefill_attention(dtype, q, k, v, k_pre, v_pre, n_pre, seq_off, n_seq, d, d + nt, nt, pos0,
                                         n_heads, n_kv_heads, head_dim, window, out, st, CachedKeys(), off[n_seq]);
  cudaStreamSynchronize(st);  // the host copy of the tile list must outlive the upload
  cudaFreeAsync(d, st);
  return s;
}

}  // extern "C"
