// C ABI of the FastMTP speculative decode step (include/fastmtp.h): context, workspace,
// TMA descriptors and the launch sequence of draft_step / verify_step / accept_commit.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <string>
#include <vector>

#include "../../include/fastmtp.h"
#include "internal.h"

using namespace fm;

namespace {

thread_local std::string g_tls_err;

struct LayerMaps {
  CUtensorMap wqkv, wo, gu_routed, gu_shared, dn_routed, dn_shared;
};

struct ActMaps {
  CUtensorMap m[5];
};

typedef std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>> Mark;

// One captured call: the key of everything its kernels bake in (sizes and caller pointers),
// the instantiated graph, its launch counts per kernel class and, for profiled graphs, the
// event pairs recorded around each launch group.
struct GraphKey {
  int kind, B, K, prof;
  const void* p[4];
  bool operator==(const GraphKey& o) const {
    return kind == o.kind && B == o.B && K == o.K && prof == o.prof && p[0] == o.p[0] && p[1] == o.p[1] &&
           p[2] == o.p[2] && p[3] == o.p[3];
  }
};
struct CallGraph {
  GraphKey key;
  cudaGraphExec_t exec = nullptr;
  std::vector<std::pair<int, int>> counts;
  std::vector<Mark> marks;
};

}  // namespace

struct spec_ctx {
  spec_config cfg{};
  cudaStream_t stream = nullptr;
  int device = 0;
  std::string err;

  spec_weights w{};
  std::vector<spec_layer_weights> layers;
  bf16* kv_pool = nullptr;
  bf16* dkv_pool = nullptr;
  // attention: the pools as TMA tensors (per verifier layer, and the draft pool), when the
  // page size allows whole-chunk boxes
  bool attn_tma = false;
  std::vector<CUtensorMap> kv_maps;
  CUtensorMap dkv_map;

  std::vector<LayerMaps> lmaps;
  CUtensorMap lm{}, eh{}, mqkv{}, mwo{}, mgu{}, mdn{};
  ActMaps a_xn{}, a_attn{}, a_xs{}, a_act{}, a_b{}, a_dcat{}, a_dxn{}, a_dattn{}, a_dact{}, a_u{};

  int Bmax = 0, Rmax = 0, Tmax = 0, Tcap = 0, n_chunks = 0, lm_tiles = 0, dstage_rows = 0;
  size_t sk_floats = 0;

  // workspace (one allocation)
  void* ws = nullptr;
  size_t ws_bytes = 0;
  float* h = nullptr;
  bf16* xn = nullptr;
  bf16* q = nullptr;
  bf16* stage = nullptr;
  float* attn_part = nullptr;
  int* attn_tickets = nullptr;
  int* commit_tickets = nullptr;
  int* rowmap = nullptr;        // [n_experts][Tmax] (token << 3 | rank) of each routed expert row
  bf16* attn_out = nullptr;
  int* route_idx = nullptr;
  float* route_gate = nullptr;
  int* counts = nullptr;
  int* moe_dep = nullptr;       // [L][n_experts + n_shared][dep_stride] gate/up tiles done per row tile
  int dep_stride = 0;
  bf16* x_sorted = nullptr;
  bf16* act = nullptr;
  // fp8 experts: e4m3 copies of the expert inputs and SwiGLU activations (else NULL)
  bool fp8 = false;
  uint8_t* x_sorted8 = nullptr;   // [n_experts][Tcap][d]
  uint8_t* xn8 = nullptr;         // [Tmax][d]
  uint8_t* act8 = nullptr;        // [n_experts + n_shared][Tcap][I]
  ActMaps a_xs8{}, a_xn8{}, a_act8{};
  float* y = nullptr;
  bf16* b_ws = nullptr;
  unsigned long long* am_key = nullptr;   // packed (logit, token) per row of the LM head
  int* am_done = nullptr;                 // CTA ticket of the verify LM head
  int* vtok = nullptr;
  int* m_ws = nullptr;
  int* cand_ws = nullptr;
  int* pos = nullptr;
  long long* kv_rowoff = nullptr;
  int* seq_len = nullptr;
  int* pending = nullptr;
  int* block_table = nullptr;
  int* draft_n = nullptr;
  bf16* draft_b = nullptr;
  int* draft_tok = nullptr;
  bf16* dcat = nullptr;
  float* z = nullptr;
  float* dres = nullptr;
  bf16* dxn = nullptr;
  bf16* dattn = nullptr;
  bf16* dact = nullptr;
  bf16* u = nullptr;
  bf16* dstage = nullptr;
  int* last_row = nullptr;
  float* sk_ws = nullptr;
  int* sk_tickets = nullptr;
  float2* rope = nullptr;
  int* d_err = nullptr;

  // measurement: event pairs per kernel class, launch counts, expert counters (device int64[2])
  bool prof_on = false;
  std::vector<cudaEvent_t> ev_free;
  std::vector<Mark> marks;
  // CUDA graphs: one per distinct call key, replayed on later calls with the same key
  bool use_graphs = true;
  // FASTMTP_CHECK_LAUNCHES: no graphs, and the stream is synchronised after every launch group
  // so that a fault or a guard flag is reported with the kernel class that raised it
  bool check_launches = false;
  int64_t launch_seq = 0;
  std::vector<CallGraph*> graphs;
  CallGraph* capturing = nullptr;
  int64_t launches[SPEC_K_COUNT] = {};
  double prof_ms[SPEC_K_COUNT] = {};
  unsigned long long* d_expert_ctr = nullptr;

  // host-side state machine
  bool verified = false;
  int last_B = 0, last_K = 0;
  const int* last_slots = nullptr;
  int last_draft_K = 0, last_draft_B = 0;
};

namespace {

spec_status fail(spec_ctx* c, spec_status s, const std::string& msg) {
  if (c) c->err = msg;
  else g_tls_err = msg;
  return s;
}

#define CK(call)                                                                      \
  do {                                                                                \
    cudaError_t e_ = (call);                                                          \
    if (e_ != cudaSuccess)                                                            \
      return fail(ctx, SPEC_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// A GemmArgs with the context-wide fields filled in.
GemmArgs base_args(spec_ctx* ctx) {
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.split_k = 1;
  g.n_routed = 1 << 30;
  g.rope = ctx->rope;
  g.max_pos = ctx->cfg.max_position;
  g.sk_ws = ctx->sk_ws;
  g.sk_tickets = ctx->sk_tickets;
  g.err = ctx->d_err;
  return g;
}

// A GemmArgs of a draft-block projection: the block's weights (54 MB with P) are loaded with the
// L2 evict-last policy, so that they stay resident across the depths of a step while the LM
// head streams through L2 with evict-first.
GemmArgs draft_args(spec_ctx* ctx) {
  GemmArgs g = base_args(ctx);
  g.a_keep = 1;
  return g;
}

int box_log_for(int rows) {
  int bl = 0;
  while ((16 << bl) < rows && bl < 4) ++bl;
  return bl;
}

// Dense GEMM over M activation rows (starting at row b_row_off of the activation buffer).
cudaError_t run_dense(spec_ctx* ctx, GemmArgs g, int epi, const CUtensorMap& wmap, const ActMaps& amap, int N,
                      int K, int M, bool split, bool paired = false, int half_rows = 0) {
  g.a_map[0] = wmap;
  for (int b = 0; b < 5; ++b) g.b_map[0][b] = amap.m[b];
  g.N = N;
  g.K = K;
  g.M = M;
  g.paired = paired ? 1 : 0;
  g.half_rows = half_rows;
  g.box_log = box_log_for(M < 256 ? M : 256);
  g.n_tiles = paired ? (N / 128) : (N + 127) / 128;
  g.split_k = split ? dense_split_k(N, K) : 1;
  if (g.split_k > 1 && M >= kSeqSplitRows) {
    // many rows: one CTA per (weight tile, 64 rows) computes every split into its own TMEM
    // accumulator and adds them in split order -- the same sums as the cross-CTA split
    g.seq_split = 1;
    g.box_log = 2;
  } else if (g.split_k > 1) {
    // few rows: one CTA per split, the splits of a tile form a cluster and add their partial
    // tiles through distributed shared memory, in split order
    g.cluster = g.split_k;
  }
  const int box = 16 << g.box_log;
  g.m_tiles = (M + box - 1) / box;
  g.n_items = g.n_tiles * (g.seq_split ? 1 : g.split_k) * g.m_tiles;
  const int grid = g.cluster ? g.n_items : (g.n_items < num_sms() ? g.n_items : num_sms());
  return gemm_launch(epi, box <= 64 ? 64 : 256, g, grid, ctx->stream);
}

size_t align_up(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

cudaEvent_t take_event(spec_ctx* ctx) {
  if (!ctx->ev_free.empty()) {
    cudaEvent_t e = ctx->ev_free.back();
    ctx->ev_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Brackets one launch group of kernel class `cls` (n_kernels kernels): counts its launches
// and, when profiling, records an event pair around it (as external event nodes while a
// profiled graph is being captured).
struct ProfScope {
  spec_ctx* ctx;
  int cls;
  cudaEvent_t e0 = nullptr;
  ProfScope(spec_ctx* c, int k) : ctx(c), cls(k) {
    if (ctx->capturing != nullptr) {
      if (ctx->capturing->key.prof) {
        cudaEventCreate(&e0);
        cudaEventRecordWithFlags(e0, ctx->stream, cudaEventRecordExternal);
      }
    } else if (ctx->prof_on) {
      e0 = take_event(ctx);
      cudaEventRecord(e0, ctx->stream);
    }
  }
  void done(int n_kernels) {
    if (ctx->capturing != nullptr) {
      ctx->capturing->counts.push_back({cls, n_kernels});
      if (ctx->capturing->key.prof) {
        cudaEvent_t e1 = nullptr;
        cudaEventCreate(&e1);
        cudaEventRecordWithFlags(e1, ctx->stream, cudaEventRecordExternal);
        ctx->capturing->marks.push_back({cls, {e0, e1}});
      }
      return;
    }
    ctx->launches[cls] += n_kernels;
    if (ctx->prof_on) {
      cudaEvent_t e1 = take_event(ctx);
      cudaEventRecord(e1, ctx->stream);
      ctx->marks.push_back({cls, {e0, e1}});
    }
  }
};

void destroy_graph(CallGraph* g) {
  if (g->exec) cudaGraphExecDestroy(g->exec);
  for (auto& m : g->marks) {
    cudaEventDestroy(m.second.first);
    cudaEventDestroy(m.second.second);
  }
  delete g;
}

// Runs `body` (the launch sequence of one call) through a CUDA graph: captured the first
// time a key is seen, replayed afterwards.  Profiled graphs are synchronised after each replay
// so that their event pairs can be read before the next replay records them again.
template <class F>
spec_status run_graphed(spec_ctx* ctx, GraphKey key, F body) {
  key.prof = ctx->prof_on ? 1 : 0;
  if (!ctx->use_graphs || ctx->stream == nullptr) return body();
  CallGraph* g = nullptr;
  for (CallGraph* c : ctx->graphs)
    if (c->key == key) g = c;
  if (g == nullptr) {
    g = new CallGraph();
    g->key = key;
    cudaError_t e = cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) {
      delete g;
      return fail(ctx, SPEC_ECUDA, std::string("cudaStreamBeginCapture: ") + cudaGetErrorString(e));
    }
    ctx->capturing = g;
    spec_status st = body();
    ctx->capturing = nullptr;
    cudaGraph_t graph = nullptr;
    e = cudaStreamEndCapture(ctx->stream, &graph);
    if (st != SPEC_OK || e != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      destroy_graph(g);
      if (st != SPEC_OK) return st;
      return fail(ctx, SPEC_ECUDA, std::string("cudaStreamEndCapture: ") + cudaGetErrorString(e));
    }
    e = cudaGraphInstantiate(&g->exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
      destroy_graph(g);
      return fail(ctx, SPEC_ECUDA, std::string("cudaGraphInstantiate: ") + cudaGetErrorString(e));
    }
    ctx->graphs.push_back(g);
  }
  cudaError_t e = cudaGraphLaunch(g->exec, ctx->stream);
  if (e != cudaSuccess) return fail(ctx, SPEC_ECUDA, std::string("cudaGraphLaunch: ") + cudaGetErrorString(e));
  for (auto& c : g->counts) ctx->launches[c.first] += c.second;
  if (key.prof) {
    e = cudaStreamSynchronize(ctx->stream);
    if (e != cudaSuccess) return fail(ctx, SPEC_ECUDA, std::string("profiled graph: ") + cudaGetErrorString(e));
    for (auto& m : g->marks) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, m.second.first, m.second.second) == cudaSuccess) ctx->prof_ms[m.first] += ms;
    }
  }
  return SPEC_OK;
}

}  // namespace

// Synchronises after one launch group in checking mode and names the group in the error.
spec_status check_launch(spec_ctx* ctx, int cls, const char* what) {
  ++ctx->launch_seq;
  if (!ctx->check_launches || ctx->capturing != nullptr) return SPEC_OK;
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  int flag = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&flag, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess || flag != 0) {
    char buf[256];
    snprintf(buf, sizeof(buf), "launch %lld (class %d: %s): %s, guard flag 0x%x",
             static_cast<long long>(ctx->launch_seq), cls, what, cudaGetErrorString(e), flag);
    return fail(ctx, e != cudaSuccess ? SPEC_ECUDA : SPEC_EDEVICE, buf);
  }
  return SPEC_OK;
}

#define LAUNCH(cls, nk, call)                             \
  do {                                                    \
    ProfScope ps_(ctx, cls);                              \
    CK(call);                                             \
    ps_.done(nk);                                         \
    spec_status cs_ = check_launch(ctx, cls, #call);      \
    if (cs_ != SPEC_OK) return cs_;                       \
  } while (0)

// ============================================================================ init / destroy
extern "C" spec_status spec_init(const spec_config* cfg, const spec_weights* w, void* kv_pool, void* draft_kv_pool,
                                 void* stream, spec_ctx** out) {
  spec_ctx* ctx = nullptr;
  if (out == nullptr) return fail(nullptr, SPEC_EINVAL, "out is NULL");
  *out = nullptr;
  if (cfg == nullptr || w == nullptr || kv_pool == nullptr || draft_kv_pool == nullptr)
    return fail(nullptr, SPEC_EINVAL, "null argument");
  const spec_config& c = *cfg;
  if (c.hidden != kD || c.n_heads != kH || c.head_dim != kHD || c.n_experts != kE || c.top_k != kTopK ||
      c.n_shared != kShared || c.expert_inter != kI || c.draft_inter != kId)
    return fail(nullptr, SPEC_EINVAL, "shape contract: kernels are built for d=1280, 10x128 heads, 64 experts top-6, "
                                      "2 shared, expert inter 896, draft inter 3584");
  if (c.n_layers < 1 || c.vocab < 2 || c.page_size < 16 || c.page_size % 16 || c.max_batch < 1 ||
      c.max_pages_per_seq < 1 || c.n_pages_total < 1 || c.K_max < 0 || c.K_max + 1 > kMaxR || c.max_position < 1 ||
      !(c.rms_eps >= 0.f) || !(c.rope_theta > 0.f))
    return fail(nullptr, SPEC_EINVAL, "config field out of range");
  if (c.max_batch * (c.K_max + 1) > 2048)
    return fail(nullptr, SPEC_EINVAL, "max_batch * (K_max + 1) must be <= 2048");
  if (c.expert_fp8 != 0 && c.expert_fp8 != 1) return fail(nullptr, SPEC_EINVAL, "expert_fp8 must be 0 or 1");
  if (w->layers == nullptr || w->embed == nullptr || w->lm_head == nullptr || w->final_norm == nullptr ||
      w->enorm == nullptr || w->hnorm == nullptr || w->eh_proj == nullptr || w->mtp_attn_norm == nullptr ||
      w->mtp_wqkv == nullptr || w->mtp_wo == nullptr || w->mtp_ffn_norm == nullptr || w->mtp_w_gate_up == nullptr ||
      w->mtp_w_down == nullptr)
    return fail(nullptr, SPEC_EINVAL, "null weight pointer");
  for (int l = 0; l < c.n_layers; ++l) {
    const spec_layer_weights& L = w->layers[l];
    const void* ps[] = {L.attn_norm, L.wqkv, L.wo, L.moe_norm, L.router, L.w_gate_up, L.w_down,
                        L.shared_gate_up, L.shared_down};
    for (const void* p : ps)
      if (p == nullptr || !aligned16(p)) return fail(nullptr, SPEC_EINVAL, "layer weight NULL or not 16-byte aligned");
    if (c.expert_fp8 && (L.gate_up_scale == nullptr || L.down_scale == nullptr || L.shared_gate_up_scale == nullptr ||
                         L.shared_down_scale == nullptr))
      return fail(nullptr, SPEC_EINVAL, "expert_fp8: a layer's expert scales are NULL");
  }
  const void* top[] = {w->embed, w->lm_head, w->eh_proj, w->mtp_wqkv, w->mtp_wo, w->mtp_w_gate_up, w->mtp_w_down,
                       kv_pool, draft_kv_pool};
  for (const void* p : top)
    if (!aligned16(p)) return fail(nullptr, SPEC_EINVAL, "matrix or pool not 16-byte aligned");

  {
    cudaError_t e = gemm_prepare();
    if (e == cudaSuccess) e = attention_prepare();
    if (e == cudaSuccess) e = router_prepare();
    if (e != cudaSuccess) return fail(nullptr, SPEC_ECUDA, std::string("kernel attributes: ") + cudaGetErrorString(e));
  }
  ctx = new spec_ctx();
  ctx->cfg = c;
  ctx->stream = static_cast<cudaStream_t>(stream);
  cudaGetDevice(&ctx->device);
  ctx->w = *w;
  ctx->layers.assign(w->layers, w->layers + c.n_layers);
  ctx->w.layers = ctx->layers.data();
  ctx->kv_pool = static_cast<bf16*>(kv_pool);
  ctx->dkv_pool = static_cast<bf16*>(draft_kv_pool);
  ctx->check_launches = getenv("FASTMTP_CHECK_LAUNCHES") != nullptr;
  ctx->use_graphs = getenv("FASTMTP_NO_GRAPHS") == nullptr && !ctx->check_launches;

  const int L = c.n_layers;
  ctx->Bmax = c.max_batch;
  ctx->Rmax = c.K_max + 1;
  ctx->Tmax = ctx->Bmax * ctx->Rmax;
  const int Tmax = ctx->Tmax, Bmax = ctx->Bmax, Rmax = ctx->Rmax;
  ctx->n_chunks = (c.max_pages_per_seq * c.page_size + Rmax + kAttnChunk - 1) / kAttnChunk;
  ctx->lm_tiles = (c.vocab + 127) / 128;
  ctx->dstage_rows = c.K_max > 1 ? c.K_max - 1 : 1;
  {
    // split-K partials: per split, a tile's rows are padded to the row box (< 2 * rows + 16)
    const int shapes[][2] = {{3 * kD, kD}, {kD, kD}, {kD, 2 * kD}, {kD, kId}, {2 * kId, kD}};
    size_t mx = 0;
    for (auto& sh : shapes) {
      const size_t v = static_cast<size_t>(dense_split_k(sh[0], sh[1])) * ((sh[0] + 127) / 128) * 128;
      if (v > mx) mx = v;
    }
    ctx->sk_floats = mx * (2 * static_cast<size_t>(Tmax) + 256) + 16;
  }
  // ---- workspace layout
  struct Sub {
    void** p;
    size_t bytes;
  };
  std::vector<Sub> subs;
  auto add = [&](void* pp, size_t bytes) { subs.push_back({reinterpret_cast<void**>(pp), bytes}); };
  const size_t d = kD;
  add(&ctx->h, sizeof(float) * Tmax * d);
  add(&ctx->xn, sizeof(bf16) * Tmax * d);
  add(&ctx->q, sizeof(bf16) * Tmax * d);
  add(&ctx->stage, sizeof(bf16) * L * Bmax * Rmax * 2 * d);
  add(&ctx->attn_part, sizeof(float) * static_cast<size_t>(Bmax) * kH * ((ctx->n_chunks + kAttnSuper - 1) / kAttnSuper) *
                           Rmax * kAttnPartStride);
  add(&ctx->attn_tickets, sizeof(int) * Bmax * kH);
  add(&ctx->commit_tickets, sizeof(int) * Bmax);
  ctx->Tcap = (Tmax + kExpertTileRows - 1) / kExpertTileRows * kExpertTileRows;
  add(&ctx->rowmap, sizeof(int) * kE * ctx->Tcap);
  add(&ctx->attn_out, sizeof(bf16) * Tmax * d);
  add(&ctx->route_idx, sizeof(int) * L * Tmax * kTopK);
  add(&ctx->route_gate, sizeof(float) * L * Tmax * kTopK);
  add(&ctx->counts, sizeof(int) * L * kE);
  ctx->dep_stride = ctx->Tcap / kExpertTileRows;
  add(&ctx->moe_dep, sizeof(int) * L * (kE + kShared) * ctx->dep_stride);
  add(&ctx->x_sorted, sizeof(bf16) * kE * ctx->Tcap * d);
  add(&ctx->act, sizeof(bf16) * (kE + kShared) * ctx->Tcap * kI);
  ctx->fp8 = c.expert_fp8 != 0;
  if (ctx->fp8) {
    add(&ctx->x_sorted8, static_cast<size_t>(kE) * ctx->Tcap * d);
    add(&ctx->xn8, static_cast<size_t>(Tmax) * d);
    add(&ctx->act8, static_cast<size_t>(kE + kShared) * ctx->Tcap * kI);
  }
  add(&ctx->y, sizeof(float) * Tmax * kSlots * d);
  add(&ctx->b_ws, sizeof(bf16) * Tmax * d);
  add(&ctx->am_key, sizeof(unsigned long long) * Tmax);
  add(&ctx->am_done, sizeof(int));
  add(&ctx->vtok, sizeof(int) * Tmax);
  add(&ctx->m_ws, sizeof(int) * Bmax);
  add(&ctx->cand_ws, sizeof(int) * Tmax);
  add(&ctx->pos, sizeof(int) * Tmax);
  add(&ctx->kv_rowoff, sizeof(long long) * Tmax);
  add(&ctx->seq_len, sizeof(int) * Bmax);
  add(&ctx->pending, sizeof(int) * Bmax);
  add(&ctx->block_table, sizeof(int) * Bmax * c.max_pages_per_seq);
  add(&ctx->draft_n, sizeof(int) * Bmax);
  add(&ctx->draft_b, sizeof(bf16) * Bmax * kMaxR * d);
  add(&ctx->draft_tok, sizeof(int) * Bmax * kMaxR);
  add(&ctx->dcat, sizeof(bf16) * Tmax * 2 * d);
  add(&ctx->z, sizeof(float) * Tmax * d);
  add(&ctx->dres, sizeof(float) * Bmax * d);
  add(&ctx->dxn, sizeof(bf16) * Tmax * d);
  add(&ctx->dattn, sizeof(bf16) * Bmax * d);
  add(&ctx->dact, sizeof(bf16) * Bmax * kId);
  add(&ctx->u, sizeof(bf16) * (c.K_max > 0 ? c.K_max : 1) * Bmax * d);
  add(&ctx->dstage, sizeof(bf16) * Bmax * ctx->dstage_rows * 2 * d);
  add(&ctx->last_row, sizeof(int) * Bmax);
  add(&ctx->sk_ws, sizeof(float) * ctx->sk_floats);
  add(&ctx->sk_tickets, sizeof(int) * 8192);
  add(&ctx->rope, sizeof(float2) * static_cast<size_t>(c.max_position) * (kHD / 2));
  add(&ctx->d_err, sizeof(int) * 4);
  add(&ctx->d_expert_ctr, sizeof(unsigned long long) * 2);
  size_t total = 0;
  for (auto& s : subs) total += align_up(s.bytes);
  if (cudaMalloc(&ctx->ws, total) != cudaSuccess) {
    cudaGetLastError();
    delete ctx;
    return fail(nullptr, SPEC_ENOMEM, "workspace allocation of " + std::to_string(total) + " bytes failed");
  }
  ctx->ws_bytes = total;
  size_t off = 0;
  for (auto& s : subs) {
    *s.p = static_cast<char*>(ctx->ws) + off;
    off += align_up(s.bytes);
  }
  auto bail = [&](spec_status st, const std::string& m) {
    cudaFree(ctx->ws);
    delete ctx;
    return fail(nullptr, st, m);
  };
  if (cudaMemsetAsync(ctx->ws, 0, total, ctx->stream) != cudaSuccess) return bail(SPEC_ECUDA, "workspace memset failed");

  // ---- RoPE table: cos/sin of p * theta^(-2i/hd) in double, stored fp32
  {
    std::vector<float2> tab(static_cast<size_t>(c.max_position) * (kHD / 2));
    for (int p = 0; p < c.max_position; ++p)
      for (int i = 0; i < kHD / 2; ++i) {
        const double inv = pow(static_cast<double>(c.rope_theta), -2.0 * i / kHD);
        const double ang = static_cast<double>(p) * inv;
        tab[static_cast<size_t>(p) * (kHD / 2) + i] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
      }
    if (cudaMemcpyAsync(ctx->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice, ctx->stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(ctx->stream) != cudaSuccess)
      return bail(SPEC_ECUDA, "RoPE table upload failed");
  }

  // ---- tensor maps
  std::string e;
  bool ok = true;
  ctx->lmaps.resize(L);
  for (int l = 0; l < L && ok; ++l) {
    const spec_layer_weights& W = ctx->layers[l];
    LayerMaps& m = ctx->lmaps[l];
    ok = ok && encode_map_2d(&m.wqkv, W.wqkv, kD, 3 * kD, 128, &e);
    ok = ok && encode_map_2d(&m.wo, W.wo, kD, kD, 128, &e);
    const int eb = ctx->fp8 ? 1 : 2;   // expert matrices: e4m3 bytes or bf16
    ok = ok && encode_map_3d(&m.gu_routed, W.w_gate_up, kD, 2 * kI, kE, 64, &e, eb);
    ok = ok && encode_map_3d(&m.gu_shared, W.shared_gate_up, kD, 2 * kI, kShared, 64, &e, eb);
    ok = ok && encode_map_3d(&m.dn_routed, W.w_down, kI, kD, kE, 128, &e, eb);
    ok = ok && encode_map_3d(&m.dn_shared, W.shared_down, kI, kD, kShared, 128, &e, eb);
  }
  ok = ok && encode_map_2d(&ctx->lm, w->lm_head, kD, c.vocab, 128, &e);
  ok = ok && encode_map_2d(&ctx->eh, w->eh_proj, 2 * kD, kD, 128, &e);
  ok = ok && encode_map_2d(&ctx->mqkv, w->mtp_wqkv, kD, 3 * kD, 128, &e);
  ok = ok && encode_map_2d(&ctx->mwo, w->mtp_wo, kD, kD, 128, &e);
  ok = ok && encode_map_2d(&ctx->mgu, w->mtp_w_gate_up, kD, 2 * kId, 64, &e);
  ok = ok && encode_map_2d(&ctx->mdn, w->mtp_w_down, kId, kD, 128, &e);
  ok = ok && encode_act_maps(ctx->a_xn.m, ctx->xn, kD, Tmax, &e);
  ok = ok && encode_act_maps(ctx->a_attn.m, ctx->attn_out, kD, Tmax, &e);
  ok = ok && encode_act_maps(ctx->a_xs.m, ctx->x_sorted, kD, static_cast<uint64_t>(kE) * ctx->Tcap, &e);
  if (ctx->fp8) {
    ok = ok && encode_act_maps(ctx->a_xs8.m, ctx->x_sorted8, kD, static_cast<uint64_t>(kE) * ctx->Tcap, &e, 1);
    ok = ok && encode_act_maps(ctx->a_xn8.m, ctx->xn8, kD, Tmax, &e, 1);
    ok = ok && encode_act_maps(ctx->a_act8.m, ctx->act8, kI, static_cast<uint64_t>(kE + kShared) * ctx->Tcap, &e, 1);
  }
  ok = ok && encode_act_maps(ctx->a_act.m, ctx->act, kI, static_cast<uint64_t>(kE + kShared) * ctx->Tcap, &e);
  ok = ok && encode_act_maps(ctx->a_b.m, ctx->b_ws, kD, Tmax, &e);
  ok = ok && encode_act_maps(ctx->a_dcat.m, ctx->dcat, 2 * kD, Tmax, &e);
  ok = ok && encode_act_maps(ctx->a_dxn.m, ctx->dxn, kD, Tmax, &e);
  ok = ok && encode_act_maps(ctx->a_dattn.m, ctx->dattn, kD, Bmax, &e);
  ok = ok && encode_act_maps(ctx->a_dact.m, ctx->dact, kId, Bmax, &e);
  ok = ok && encode_act_maps(ctx->a_u.m, ctx->u, kD, static_cast<uint64_t>(c.K_max > 0 ? c.K_max : 1) * Bmax, &e);
  {
    const long long pool_rows = static_cast<long long>(c.n_pages_total) * 2 * kH * c.page_size;
    ctx->attn_tma = (c.page_size % kAttnChunk == 0) && pool_rows < (1ll << 31);
    if (ctx->attn_tma) {
      const size_t pool_layer = static_cast<size_t>(pool_rows) * kHD;
      ctx->kv_maps.resize(L);
      for (int l = 0; l < L && ok; ++l)
        ok = encode_map_2d(&ctx->kv_maps[l], ctx->kv_pool + l * pool_layer, kHD, pool_rows, kAttnChunk, &e);
      ok = ok && encode_map_2d(&ctx->dkv_map, ctx->dkv_pool, kHD, pool_rows, kAttnChunk, &e);
    }
  }
  if (!ok) return bail(SPEC_EINVAL, "tensor map: " + e);
  if (cudaStreamSynchronize(ctx->stream) != cudaSuccess) return bail(SPEC_ECUDA, "stream synchronize failed");
  *out = ctx;
  return SPEC_OK;
}

extern "C" void spec_destroy(spec_ctx* ctx) {
  if (ctx == nullptr) return;
  if (ctx->stream != nullptr) cudaStreamSynchronize(ctx->stream);
  else cudaDeviceSynchronize();
  for (auto& m : ctx->marks) {
    cudaEventDestroy(m.second.first);
    cudaEventDestroy(m.second.second);
  }
  for (cudaEvent_t e : ctx->ev_free) cudaEventDestroy(e);
  for (CallGraph* g : ctx->graphs) destroy_graph(g);
  cudaFree(ctx->ws);
  delete ctx;
}

void fm::set_thread_error(const std::string& msg) { g_tls_err = msg; }

extern "C" const char* spec_last_error(const spec_ctx* ctx) {
  return ctx ? ctx->err.c_str() : g_tls_err.c_str();
}

// ============================================================================ sequence state
extern "C" spec_status spec_seq_reset(spec_ctx* ctx, int32_t slot, int32_t ctx_len, const int32_t* block_table,
                                      int32_t pending) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  const spec_config& c = ctx->cfg;
  if (slot < 0 || slot >= ctx->Bmax) return fail(ctx, SPEC_EINVAL, "slot out of range");
  if (ctx_len < 0 || ctx_len >= c.max_pages_per_seq * c.page_size || ctx_len + 1 > c.max_position)
    return fail(ctx, SPEC_EINVAL, "ctx_len out of range");
  if (pending < 0 || pending >= c.vocab) return fail(ctx, SPEC_EINVAL, "pending token out of range");
  if (block_table == nullptr) return fail(ctx, SPEC_EINVAL, "block_table is NULL");
  const int need = (ctx_len + c.page_size - 1) / c.page_size;
  for (int i = 0; i < c.max_pages_per_seq; ++i) {
    const int p = block_table[i];
    if (p < -1 || p >= c.n_pages_total) return fail(ctx, SPEC_EINVAL, "page id out of range");
    if (i < need && p < 0) return fail(ctx, SPEC_EINVAL, "prefix position without a page");
  }
  CK(cudaMemcpyAsync(ctx->block_table + static_cast<size_t>(slot) * c.max_pages_per_seq, block_table,
                     sizeof(int) * c.max_pages_per_seq, cudaMemcpyHostToDevice, ctx->stream));
  const int zero = 0;
  CK(cudaMemcpyAsync(ctx->seq_len + slot, &ctx_len, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaMemcpyAsync(ctx->pending + slot, &pending, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaMemcpyAsync(ctx->draft_n + slot, &zero, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  return SPEC_OK;
}

extern "C" spec_status spec_seq_set_draft_rows(spec_ctx* ctx, int32_t slot, int32_t n_rows, const void* b_rows,
                                               const int32_t* next_tokens) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (slot < 0 || slot >= ctx->Bmax) return fail(ctx, SPEC_EINVAL, "slot out of range");
  if (n_rows < 1 || n_rows > ctx->Rmax) return fail(ctx, SPEC_EINVAL, "n_rows out of range");
  if (b_rows == nullptr || next_tokens == nullptr) return fail(ctx, SPEC_EINVAL, "null argument");
  for (int i = 0; i < n_rows; ++i)
    if (next_tokens[i] < 0 || next_tokens[i] >= ctx->cfg.vocab) return fail(ctx, SPEC_EINVAL, "token out of range");
  int len = 0, pend = 0;
  CK(cudaMemcpyAsync(&len, ctx->seq_len + slot, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaMemcpyAsync(&pend, ctx->pending + slot, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  if (len < n_rows) return fail(ctx, SPEC_EINVAL, "more draft rows than committed positions");
  if (next_tokens[n_rows - 1] != pend) return fail(ctx, SPEC_EINVAL, "last next token must be the pending token");
  CK(cudaMemcpyAsync(ctx->draft_b + static_cast<size_t>(slot) * kMaxR * kD, b_rows, sizeof(bf16) * n_rows * kD,
                     cudaMemcpyDeviceToDevice, ctx->stream));
  CK(cudaMemcpyAsync(ctx->draft_tok + slot * kMaxR, next_tokens, sizeof(int) * n_rows, cudaMemcpyHostToDevice,
                     ctx->stream));
  CK(cudaMemcpyAsync(ctx->draft_n + slot, &n_rows, sizeof(int), cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  return SPEC_OK;
}

extern "C" spec_status spec_seq_state(spec_ctx* ctx, int32_t slot, int32_t* ctx_len, int32_t* pending) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (slot < 0 || slot >= ctx->Bmax || ctx_len == nullptr || pending == nullptr)
    return fail(ctx, SPEC_EINVAL, "bad argument");
  CK(cudaMemcpyAsync(ctx_len, ctx->seq_len + slot, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaMemcpyAsync(pending, ctx->pending + slot, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  return SPEC_OK;
}

// ============================================================================ verify
extern "C" spec_status verify_step(spec_ctx* ctx, int32_t B, int32_t K, const int32_t* slots, const int32_t* cand,
                                   int32_t* verifier_tokens, int32_t* accept_len) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  const spec_config& c = ctx->cfg;
  if (B < 1 || B > ctx->Bmax) return fail(ctx, SPEC_EINVAL, "B out of range");
  if (K < 0 || K > c.K_max) return fail(ctx, SPEC_EINVAL, "K out of range");
  if (slots == nullptr || cand == nullptr || verifier_tokens == nullptr || accept_len == nullptr)
    return fail(ctx, SPEC_EINVAL, "null argument");
  if (ctx->verified) return fail(ctx, SPEC_ESTATE, "the previous verify_step has not been committed");
  const int R = K + 1, T = B * R, L = c.n_layers;
  const float eps = c.rms_eps;
  cudaStream_t s = ctx->stream;
  const size_t stage_layer = static_cast<size_t>(ctx->Bmax) * ctx->Rmax * 2 * kD;
  const size_t pool_layer = static_cast<size_t>(c.n_pages_total) * 2 * kH * c.page_size * kHD;

  GraphKey key{1, B, K, 0, {slots, cand, verifier_tokens, accept_len}};
  spec_status st = run_graphed(ctx, key, [&]() -> spec_status {
  CK(cudaMemcpyAsync(ctx->cand_ws, cand, sizeof(int) * T, cudaMemcpyDeviceToDevice, s));
  LAUNCH(SPEC_K_EMBED, 1, embed_norm_launch(ctx->cand_ws, B, R, slots, ctx->pending, ctx->seq_len, static_cast<const bf16*>(ctx->w.embed),
                       c.vocab, static_cast<const bf16*>(ctx->layers[0].attn_norm), eps, ctx->h, ctx->xn, ctx->pos,
                       ctx->kv_rowoff, ctx->Rmax, ctx->Bmax, ctx->d_err, ctx->counts, L * kE, ctx->moe_dep,
                       L * (kE + kShared) * ctx->dep_stride, s));
  for (int l = 0; l < L; ++l) {
    const spec_layer_weights& W = ctx->layers[l];
    const LayerMaps& M = ctx->lmaps[l];
    // QKV + RoPE, K/V staged
    {
      GemmArgs g = base_args(ctx);
      g.q_out = ctx->q;
      g.kv_base = ctx->stage + l * stage_layer;
      g.kv_rowoff = ctx->kv_rowoff;
      g.head_stride = kHD;
      g.v_off = static_cast<long long>(kH) * kHD;
      g.pos = ctx->pos;
      LAUNCH(SPEC_K_QKV, 1, run_dense(ctx, g, EPI_QKV, M.wqkv, ctx->a_xn, 3 * kD, kD, T, true));
    }
    // attention over committed pages + staged candidates
    {
      AttnArgs a{};
      a.q = ctx->q;
      a.q_row0 = nullptr;
      a.R = R;
      a.qoff = 0;
      a.slots = slots;
      a.seq_len = ctx->seq_len;
      a.n_slots = ctx->Bmax;
      a.pool = ctx->kv_pool + l * pool_layer;
      if (ctx->attn_tma) {
        a.kv_map = ctx->kv_maps[l];
        a.use_tma = 1;
      }
      a.page_size = c.page_size;
      a.n_pages = c.n_pages_total;
      a.block_table = ctx->block_table;
      a.max_pages = c.max_pages_per_seq;
      a.stage = ctx->stage + l * stage_layer;
      a.stage_seq_stride = static_cast<long long>(ctx->Rmax) * 2 * kD;
      a.stage_row_stride = 2 * kD;
      a.stage_kv_stride = kD;
      a.part = ctx->attn_part;
      a.tickets = ctx->attn_tickets;
      a.n_chunks = ctx->n_chunks;
      a.out = ctx->attn_out;
      a.out_row_stride_seq = R;
      a.err = ctx->d_err;
      a.prewait = 1;   // pages, block table, slots and lengths change only in accept_commit / seq_reset
      LAUNCH(SPEC_K_ATTN, 1, attention_launch(a, B, s));
    }
    // O-proj + residual
    {
      GemmArgs g = base_args(ctx);
      g.out = ctx->h;
      g.ldo = kD;
      LAUNCH(SPEC_K_OPROJ, 1, run_dense(ctx, g, EPI_RESID, M.wo, ctx->a_attn, kD, kD, T, true));
    }
    int* ridx = ctx->route_idx + static_cast<size_t>(l) * ctx->Tmax * kTopK;
    float* rgate = ctx->route_gate + static_cast<size_t>(l) * ctx->Tmax * kTopK;
    {
      RouteArgs ra;
      ra.h = ctx->h;
      ra.gain = static_cast<const bf16*>(W.moe_norm);
      ra.eps = eps;
      ra.wr = static_cast<const bf16*>(W.router);
      ra.bias = W.router_bias;
      ra.xn = ctx->xn;
      ra.idx = ridx;
      ra.gate = rgate;
      ra.err = ctx->d_err;
      ra.T = T;
      ra.counts = ctx->counts + l * kE;
      ra.rowmap = ctx->rowmap;
      ra.x_sorted = ctx->x_sorted;
      ra.map_stride = ctx->Tcap;
      ra.xn8 = ctx->xn8;               // NULL unless fp8 experts
      ra.x_sorted8 = ctx->x_sorted8;
      LAUNCH(SPEC_K_ROUTER, 1, router_launch(ra, s));
    }
    // routed + shared experts: gate/up + SwiGLU, then down scattered to (token, slot), in one
    // cooperative launch (a down tile starts as soon as the gate/up tiles of its rows are done)
    {
      GemmArgs g = base_args(ctx);
      g.a_map[0] = M.gu_routed;
      g.a_map[1] = M.gu_shared;
      for (int b = 0; b < 5; ++b) {
        g.b_map[0][b] = ctx->fp8 ? ctx->a_xs8.m[b] : ctx->a_xs.m[b];
        g.b_map[1][b] = ctx->fp8 ? ctx->a_xn8.m[b] : ctx->a_xn.m[b];
      }
      g.N = 2 * kI;
      g.K = kD;
      g.a3d = 1;
      g.paired = 1;
      g.half_rows = kI;
      g.n_routed = kE;
      g.grp_cnt = ctx->counts + l * kE;
      g.grp_T = T;
      g.grp_rows = (T >= kExpertLargeFromRows) ? kExpertTileRowsLarge : kExpertTileRows;
      const bool dual = g.grp_rows == kExpertTileRowsLarge;   // gate/up item: 128 gate + 128 up features
      g.grp_tiles = dual ? kI / 128 : 2 * kI / 128;
      g.grp_b_direct = 1;   // shared experts read the normalised rows directly
      g.map_stride = ctx->Tcap;
      g.expert_ctr = ctx->d_expert_ctr;
      g.act = ctx->act;
      g.ld_act = kI;
      if (ctx->fp8) {
        g.f8 = 1;
        g.act8 = ctx->act8;
        g.w_scale[0] = W.gate_up_scale;
        g.w_scale[1] = W.shared_gate_up_scale;
        g.scale_rows = 2 * kI;
      }
      g.dep = ctx->moe_dep + static_cast<size_t>(l) * (kE + kShared) * ctx->dep_stride;
      g.dep_stride = ctx->dep_stride;
      GemmArgs d = base_args(ctx);
      d.a_map[0] = M.dn_routed;
      d.a_map[1] = M.dn_shared;
      for (int b = 0; b < 5; ++b) {
        d.b_map[0][b] = ctx->fp8 ? ctx->a_act8.m[b] : ctx->a_act.m[b];
        d.b_map[1][b] = d.b_map[0][b];
      }
      d.N = kD;
      d.K = kI;
      d.a3d = 1;
      d.n_routed = kE;
      d.grp_cnt = ctx->counts + l * kE;
      d.grp_T = T;
      d.grp_tiles = dual ? kD / 256 : kD / 128;   // down item: 256 or 128 outputs
      d.grp_rows = g.grp_rows;
      d.rowmap = ctx->rowmap;
      d.map_stride = ctx->Tcap;
      d.y = ctx->y;
      if (ctx->fp8) {
        d.f8 = 1;
        d.w_scale[0] = W.down_scale;
        d.w_scale[1] = W.shared_down_scale;
        d.scale_rows = kD;
      }
      LAUNCH(SPEC_K_EXPERT_GU, 1, moe_launch(g, d, s));
    }
    const bf16* next_gain =
        static_cast<const bf16*>(l + 1 < L ? ctx->layers[l + 1].attn_norm : ctx->w.final_norm);
    LAUNCH(SPEC_K_COMBINE, 1, combine_launch(ctx->h, ctx->y, rgate, T, next_gain, eps, l + 1 < L ? ctx->xn : ctx->b_ws, s));
  }
  // LM head + argmax (logits never leave the SM) + greedy accept
  {
    GemmArgs g = base_args(ctx);
    g.am_key = ctx->am_key;
    g.am_done = ctx->am_done;
    g.fin_B = B;
    g.fin_R = R;
    g.fin_cand = ctx->cand_ws;
    g.fin_vtok_out = verifier_tokens;
    g.fin_vtok_ws = ctx->vtok;
    g.fin_accept_out = accept_len;
    g.fin_m_ws = ctx->m_ws;
    LAUNCH(SPEC_K_LMHEAD, 1, run_dense(ctx, g, EPI_ARGMAX, ctx->lm, ctx->a_b, c.vocab, kD, T, false));
  }
    return SPEC_OK;
  });
  if (st != SPEC_OK) return st;
  ctx->verified = true;
  ctx->last_B = B;
  ctx->last_K = K;
  ctx->last_slots = slots;
  return SPEC_OK;
}

// ============================================================================ commit
extern "C" spec_status accept_commit(spec_ctx* ctx, int32_t B, const int32_t* slots, int32_t* committed,
                                     int32_t* n_committed) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (!ctx->verified) return fail(ctx, SPEC_ESTATE, "accept_commit without a verify_step");
  if (B != ctx->last_B || slots != ctx->last_slots)
    return fail(ctx, SPEC_EINVAL, "B and slots must be those of the last verify_step");
  if (committed == nullptr || n_committed == nullptr) return fail(ctx, SPEC_EINVAL, "null argument");
  const spec_config& c = ctx->cfg;
  GraphKey key{2, B, ctx->last_K, 0, {slots, committed, n_committed, nullptr}};
  spec_status st = run_graphed(ctx, key, [&]() -> spec_status {
  LAUNCH(SPEC_K_COMMIT, 1, commit_launch(B, ctx->last_K + 1, ctx->Rmax, ctx->Bmax, slots, ctx->m_ws, ctx->vtok, ctx->cand_ws, ctx->stage,
                   ctx->kv_pool, c.n_layers, c.n_pages_total, c.page_size, ctx->block_table, c.max_pages_per_seq,
                   ctx->seq_len, ctx->pending, ctx->b_ws, ctx->draft_b, ctx->draft_tok, ctx->draft_n, committed,
                   n_committed, ctx->commit_tickets, ctx->d_err, ctx->stream));
    return SPEC_OK;
  });
  if (st != SPEC_OK) return st;
  ctx->verified = false;
  return SPEC_OK;
}

// ============================================================================ draft
extern "C" spec_status draft_step(spec_ctx* ctx, int32_t B, int32_t K, const int32_t* slots, int32_t* cand) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  const spec_config& c = ctx->cfg;
  if (B < 1 || B > ctx->Bmax) return fail(ctx, SPEC_EINVAL, "B out of range");
  if (K < 1 || K > c.K_max) return fail(ctx, SPEC_EINVAL, "K out of range");
  if (slots == nullptr || cand == nullptr) return fail(ctx, SPEC_EINVAL, "null argument");
  if (ctx->verified) return fail(ctx, SPEC_ESTATE, "a verify_step is waiting for accept_commit");
  cudaStream_t s = ctx->stream;
  const float eps = c.rms_eps;
  const int Rm = ctx->Rmax, T1 = B * Rm, ld = K + 1;
  const long long dstage_seq = static_cast<long long>(ctx->dstage_rows) * 2 * kD;

  GraphKey key{3, B, K, 0, {slots, cand, nullptr, nullptr}};
  spec_status st = run_graphed(ctx, key, [&]() -> spec_status {
  // depth 1: the rows committed by the last step enter the draft cache with their base states
  LAUNCH(SPEC_K_DRAFT_MISC, 1, draft_prep_launch(B, Rm, slots, ctx->seq_len, ctx->pending, ctx->draft_n, ctx->draft_b, ctx->draft_tok,
                       static_cast<const bf16*>(ctx->w.embed), c.vocab, static_cast<const bf16*>(ctx->w.enorm),
                       static_cast<const bf16*>(ctx->w.hnorm), eps, ctx->dcat, ctx->pos, ctx->kv_rowoff, ctx->last_row,
                       c.page_size, ctx->block_table, c.max_pages_per_seq, c.n_pages_total, cand, ld, ctx->Bmax,
                       ctx->d_err, s));
  {
    GemmArgs g = draft_args(ctx);
    g.out = ctx->z;
    g.ldo = kD;
    LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_F32, ctx->eh, ctx->a_dcat, kD, 2 * kD, T1, true));
  }
  LAUNCH(SPEC_K_DRAFT_MISC, 1, rmsnorm_launch(ctx->z, T1, static_cast<const bf16*>(ctx->w.mtp_attn_norm), eps, ctx->dxn, s));
  {
    GemmArgs g = draft_args(ctx);
    g.q_out = ctx->q;
    g.kv_base = ctx->dkv_pool;
    g.kv_rowoff = ctx->kv_rowoff;
    g.head_stride = static_cast<long long>(c.page_size) * kHD;
    g.v_off = static_cast<long long>(kH) * c.page_size * kHD;
    g.pos = ctx->pos;
    LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_QKV, ctx->mqkv, ctx->a_dxn, 3 * kD, kD, T1, true));
  }
  LAUNCH(SPEC_K_DRAFT_MISC, 1, gather_rows_launch(ctx->z, ctx->last_row, B, ctx->dres, s));

  for (int k = 1; k <= K; ++k) {
    if (k > 1) {
      GemmArgs g = draft_args(ctx);
      g.out = ctx->dres;
      g.ldo = kD;
      LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_F32, ctx->eh, ctx->a_dcat, kD, 2 * kD, B, true));
      LAUNCH(SPEC_K_DRAFT_MISC, 1, rmsnorm_launch(ctx->dres, B, static_cast<const bf16*>(ctx->w.mtp_attn_norm), eps, ctx->dxn, s));
      GemmArgs q = draft_args(ctx);
      q.q_out = ctx->q;
      q.kv_base = ctx->dstage;
      q.kv_rowoff = ctx->kv_rowoff;
      q.head_stride = kHD;
      q.v_off = static_cast<long long>(kH) * kHD;
      q.pos = ctx->pos;
      LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, q, EPI_QKV, ctx->mqkv, ctx->a_dxn, 3 * kD, kD, B, true));
    }
    {
      AttnArgs a{};
      a.q = ctx->q;
      a.q_row0 = (k == 1) ? ctx->last_row : nullptr;
      a.R = 1;
      a.qoff = (k == 1) ? -1 : k - 2;
      a.slots = slots;
      a.seq_len = ctx->seq_len;
      a.n_slots = ctx->Bmax;
      a.pool = ctx->dkv_pool;
      if (ctx->attn_tma) {
        a.kv_map = ctx->dkv_map;
        a.use_tma = 1;
      }
      a.page_size = c.page_size;
      a.n_pages = c.n_pages_total;
      a.block_table = ctx->block_table;
      a.max_pages = c.max_pages_per_seq;
      a.stage = ctx->dstage;
      a.stage_seq_stride = dstage_seq;
      a.stage_row_stride = 2 * kD;
      a.stage_kv_stride = kD;
      a.part = ctx->attn_part;
      a.tickets = ctx->attn_tickets;
      a.n_chunks = ctx->n_chunks;
      a.out = ctx->dattn;
      a.out_row_stride_seq = 1;
      a.err = ctx->d_err;
      // committed draft rows older than the last Rmax positions were written by earlier steps
      // (draft_prep / accept_commit / seq_reset, other graphs): fetched before the wait
      a.prewait = 1;
      a.prewait_guard = ctx->Rmax;
      LAUNCH(SPEC_K_ATTN, 1, attention_launch(a, B, s));
    }
    {
      GemmArgs g = draft_args(ctx);
      g.out = ctx->dres;
      g.ldo = kD;
      LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_RESID, ctx->mwo, ctx->a_dattn, kD, kD, B, true));
    }
    LAUNCH(SPEC_K_DRAFT_MISC, 1, rmsnorm_launch(ctx->dres, B, static_cast<const bf16*>(ctx->w.mtp_ffn_norm), eps, ctx->dxn, s));
    {
      GemmArgs g = draft_args(ctx);
      g.act = ctx->dact;
      g.ld_act = kId;
      LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_SWIGLU, ctx->mgu, ctx->a_dxn, 2 * kId, kD, B, true, true, kId));
    }
    {
      GemmArgs g = draft_args(ctx);
      g.out = ctx->dres;
      g.ldo = kD;
      LAUNCH(SPEC_K_DRAFT_GEMM, 1, run_dense(ctx, g, EPI_RESID, ctx->mdn, ctx->a_dact, kD, kId, B, true));
    }
    bf16* uk = ctx->u + static_cast<size_t>(k - 1) * ctx->Bmax * kD;
    LAUNCH(SPEC_K_DRAFT_MISC, 1, rmsnorm_launch(ctx->dres, B, static_cast<const bf16*>(ctx->w.final_norm), eps, uk, s));
    {
      GemmArgs g = base_args(ctx);
      g.am_key = ctx->am_key;
      // rows of depth k start at (k-1) * Bmax in the u buffer
      g.a_map[0] = ctx->lm;
      for (int b = 0; b < 5; ++b) g.b_map[0][b] = ctx->a_u.m[b];
      g.N = c.vocab;
      g.K = kD;
      g.M = B;
      g.box_log = box_log_for(B < 256 ? B : 256);
      const int box = 16 << g.box_log;
      g.m_tiles = (B + box - 1) / box;
      g.n_tiles = (c.vocab + 127) / 128;
      g.split_k = 1;
      g.n_items = g.n_tiles * g.m_tiles;
      g.b_row_off = (k - 1) * ctx->Bmax;
      const int grid = g.n_items < num_sms() ? g.n_items : num_sms();
      LAUNCH(SPEC_K_LMHEAD, 1, gemm_launch(EPI_ARGMAX, box <= 64 ? 64 : 256, g, grid, s));
    }
    LAUNCH(SPEC_K_ARGMAX, 1, draft_next_launch(ctx->am_key, c.vocab, ctx->d_err, B, k, K, slots, ctx->Bmax, ctx->seq_len, uk,
                         static_cast<const bf16*>(ctx->w.embed), static_cast<const bf16*>(ctx->w.enorm),
                         static_cast<const bf16*>(ctx->w.hnorm), eps, ctx->dcat, ctx->pos, ctx->kv_rowoff, dstage_seq,
                         cand, ld, s));
  }
    return SPEC_OK;
  });
  if (st != SPEC_OK) return st;
  ctx->last_draft_K = K;
  ctx->last_draft_B = B;
  return SPEC_OK;
}

// ============================================================================ sync / introspection
namespace {
__device__ int g_gemm_err;   // guard flag of spec_gemm_bf16's kernels
}

// spec_sync(NULL): waits for the current device and reports the guard flags of the
// context-free entry points spec_gemm_bf16, spec_gemm_bf16_noalloc and spec_draft_loss.
static spec_status sync_device_flags() {
  spec_ctx* ctx = nullptr;
  CK(cudaDeviceSynchronize());
  int gemm_flag = 0, na_flag = 0;
  CK(cudaMemcpyFromSymbol(&gemm_flag, g_gemm_err, sizeof(int)));
  if (gemm_flag != 0) {
    const int zero = 0;
    CK(cudaMemcpyToSymbol(g_gemm_err, &zero, sizeof(int)));
  }
  int loss_flag = 0;
  CK(noalloc_take_flag(&na_flag));
  CK(loss_take_flag(&loss_flag));
  if (gemm_flag != 0 || na_flag != 0 || loss_flag != 0) {
    char buf[256];
    snprintf(buf, sizeof(buf), "device guard flag: spec_gemm_bf16 0x%x, spec_gemm_bf16_noalloc 0x%x, spec_draft_loss "
             "0x%x (1 wait timeout, 32 position)", gemm_flag, na_flag, loss_flag);
    return fail(nullptr, SPEC_EDEVICE, buf);
  }
  return SPEC_OK;
}

extern "C" spec_status spec_sync(spec_ctx* ctx) {
  if (ctx == nullptr) return sync_device_flags();
  CK(cudaStreamSynchronize(ctx->stream));
  int flag = 0;
  CK(cudaMemcpy(&flag, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost));
  if (flag != 0) {
    const int zero = 0;
    CK(cudaMemcpy(ctx->d_err, &zero, sizeof(int), cudaMemcpyHostToDevice));
    char buf[256];
    snprintf(buf, sizeof(buf), "device guard flag 0x%x (1 wait timeout, 2 token range, 4 page range, 8 pending "
             "mismatch, 16 no draft rows, 32 position, 64 slot range, 128 non-finite router row)", flag);
    return fail(ctx, SPEC_EDEVICE, buf);
  }
  return SPEC_OK;
}

extern "C" spec_status spec_trace_read(void* host_records, int32_t cap, int32_t reset, int32_t* n_records) {
  if (n_records == nullptr || cap < 0 || (cap > 0 && host_records == nullptr))
    return fail(nullptr, SPEC_EINVAL, "spec_trace_read: n_records NULL, cap < 0 or NULL buffer");
  *n_records = 0;
#ifdef FM_TRACE
  unsigned long long* out = static_cast<unsigned long long*>(host_records);
  int n = 0;
  for (auto rd : {fm::trace_read_gemm, fm::trace_read_attn, fm::trace_read_small}) {
    const int got = rd(out + 4 * static_cast<size_t>(n), cap - n, reset != 0);
    if (got < 0) return fail(nullptr, SPEC_ECUDA, "spec_trace_read: copy of the trace buffers failed");
    n += got;
  }
  *n_records = n;
  return SPEC_OK;
#else
  (void)reset;
  return fail(nullptr, SPEC_EINVAL, "spec_trace_read: the library was built without the device timeline (FASTMTP_TRACE=1)");
#endif
}

extern "C" spec_status spec_profile(spec_ctx* ctx, int32_t mode) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (mode < 0 || mode > 2) return fail(ctx, SPEC_EINVAL, "mode must be 0, 1 or 2");
  if (mode != 0) {
    CK(cudaStreamSynchronize(ctx->stream));
    for (auto& m : ctx->marks) {
      ctx->ev_free.push_back(m.second.first);
      ctx->ev_free.push_back(m.second.second);
    }
    ctx->marks.clear();
    for (int i = 0; i < SPEC_K_COUNT; ++i) {
      ctx->launches[i] = 0;
      ctx->prof_ms[i] = 0.0;
    }
    CK(cudaMemsetAsync(ctx->d_expert_ctr, 0, 2 * sizeof(unsigned long long), ctx->stream));
  }
  ctx->prof_on = mode == 1;
  return SPEC_OK;
}

extern "C" spec_status spec_profile_read(spec_ctx* ctx, spec_profile_t* out) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (out == nullptr) return fail(ctx, SPEC_EINVAL, "out is NULL");
  CK(cudaStreamSynchronize(ctx->stream));
  for (auto& m : ctx->marks) {
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, m.second.first, m.second.second));
    ctx->prof_ms[m.first] += ms;
    ctx->ev_free.push_back(m.second.first);
    ctx->ev_free.push_back(m.second.second);
  }
  ctx->marks.clear();
  unsigned long long ctr[2] = {0, 0};
  CK(cudaMemcpy(ctr, ctx->d_expert_ctr, sizeof(ctr), cudaMemcpyDeviceToHost));
  for (int i = 0; i < SPEC_K_COUNT; ++i) {
    out->launches[i] = ctx->launches[i];
    out->ms[i] = ctx->prof_ms[i];
  }
  out->experts_touched = static_cast<int64_t>(ctr[0]);
  out->expert_rows = static_cast<int64_t>(ctr[1]);
  return SPEC_OK;
}

extern "C" spec_status spec_read_workspace(spec_ctx* ctx, int32_t id, void* dst, size_t bytes) {
  if (ctx == nullptr) return fail(nullptr, SPEC_EINVAL, "ctx is NULL");
  if (dst == nullptr) return fail(ctx, SPEC_EINVAL, "dst is NULL");
  const void* src = nullptr;
  size_t cap = 0;
  const size_t L = ctx->cfg.n_layers, Tm = ctx->Tmax;
  switch (id) {
    case SPEC_WS_B: src = ctx->b_ws; cap = sizeof(bf16) * Tm * kD; break;
    case SPEC_WS_ROUTE_IDX: src = ctx->route_idx; cap = sizeof(int) * L * Tm * kTopK; break;
    case SPEC_WS_ROUTE_GATE: src = ctx->route_gate; cap = sizeof(float) * L * Tm * kTopK; break;
    case SPEC_WS_EXPERT_CNT: src = ctx->counts; cap = sizeof(int) * L * kE; break;
    case SPEC_WS_DRAFT_U: src = ctx->u; cap = sizeof(bf16) * (ctx->cfg.K_max > 0 ? ctx->cfg.K_max : 1) * ctx->Bmax * kD; break;
    case SPEC_WS_HIDDEN: src = ctx->h; cap = sizeof(float) * Tm * kD; break;
    default: return fail(ctx, SPEC_EINVAL, "unknown workspace id");
  }
  if (bytes > cap) return fail(ctx, SPEC_EINVAL, "bytes larger than the workspace tensor");
  CK(cudaStreamSynchronize(ctx->stream));
  CK(cudaMemcpy(dst, src, bytes, cudaMemcpyDeviceToHost));
  return SPEC_OK;
}

// ============================================================================ standalone GEMM
extern "C" spec_status spec_gemm_e4m3(const void* X, const void* W, const float* w_scale, float* Y, int32_t M,
                                      int32_t N, int32_t Kdim, void* stream) {
  spec_ctx* ctx = nullptr;
  if (X == nullptr || W == nullptr || w_scale == nullptr || Y == nullptr)
    return fail(nullptr, SPEC_EINVAL, "null argument");
  if (M < 1 || N < 1 || Kdim < 128 || Kdim % 128) return fail(nullptr, SPEC_EINVAL, "bad sizes (Kdim a multiple of 128)");
  if (!aligned16(X) || !aligned16(W)) return fail(nullptr, SPEC_EINVAL, "X and W must be 16-byte aligned");
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  std::string e;
  if (!encode_map_2d(&g.a_map[0], W, Kdim, N, 128, &e, 1)) return fail(nullptr, SPEC_EINVAL, e);
  if (!encode_act_maps(g.b_map[0], X, Kdim, M, &e, 1)) return fail(nullptr, SPEC_EINVAL, e);
  int* err = nullptr;
  CK(gemm_prepare());
  CK(cudaGetSymbolAddress(reinterpret_cast<void**>(&err), g_gemm_err));
  g.err = err;
  g.f8 = 1;
  g.w_scale[0] = w_scale;
  g.n_routed = 1 << 30;
  g.N = N;
  g.K = Kdim;
  g.M = M;
  g.box_log = box_log_for(M < 256 ? M : 256);
  const int box = 16 << g.box_log;
  g.m_tiles = (M + box - 1) / box;
  g.n_tiles = (N + 127) / 128;
  g.split_k = 1;
  g.n_items = g.n_tiles * g.m_tiles;
  g.out = Y;
  g.ldo = N;
  const int grid = g.n_items < num_sms() ? g.n_items : num_sms();
  CK(gemm_launch(EPI_F32, box <= 64 ? 64 : 256, g, grid, static_cast<cudaStream_t>(stream), false));
  return SPEC_OK;
}


extern "C" spec_status spec_gemm_bf16(const void* X, const void* W, float* Y, int32_t M, int32_t N, int32_t Kdim,
                                      void* stream) {
  spec_ctx* ctx = nullptr;
  if (X == nullptr || W == nullptr || Y == nullptr) return fail(nullptr, SPEC_EINVAL, "null argument");
  if (M < 1 || N < 1 || Kdim < 64 || Kdim % 64) return fail(nullptr, SPEC_EINVAL, "bad sizes");
  if (!aligned16(X) || !aligned16(W)) return fail(nullptr, SPEC_EINVAL, "X and W must be 16-byte aligned");
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  std::string e;
  if (!encode_map_2d(&g.a_map[0], W, Kdim, N, 128, &e)) return fail(nullptr, SPEC_EINVAL, e);
  if (!encode_act_maps(g.b_map[0], X, Kdim, M, &e)) return fail(nullptr, SPEC_EINVAL, e);
  int* err = nullptr;
  CK(gemm_prepare());
  CK(cudaGetSymbolAddress(reinterpret_cast<void**>(&err), g_gemm_err));
  g.err = err;
  g.n_routed = 1 << 30;
  g.N = N;
  g.K = Kdim;
  g.M = M;
  g.box_log = box_log_for(M < 256 ? M : 256);
  const int box = 16 << g.box_log;
  g.m_tiles = (M + box - 1) / box;
  g.n_tiles = (N + 127) / 128;
  g.split_k = 1;
  g.n_items = g.n_tiles * g.m_tiles;
  g.out = Y;
  g.ldo = N;
  const int grid = g.n_items < num_sms() ? g.n_items : num_sms();
  CK(gemm_launch(EPI_F32, box <= 64 ? 64 : 256, g, grid, static_cast<cudaStream_t>(stream), false));
  return SPEC_OK;
}
