// Host-side interfaces between the FastMTP translation units: the GEMM engine's argument
// block and the launchers of every kernel.  Not part of the public ABI (include/fastmtp.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <utility>

namespace fm {

// Launches `kernel` with programmatic stream serialization: it may start while the previous
// kernel of the stream finishes; the kernel itself waits (griddepcontrol.wait) before it
// touches memory that earlier kernels write.
template <typename... KArgs, typename... Args>
cudaError_t launch_k(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  return launch_k(true, kernel, grid, block, smem, s, std::forward<Args>(args)...);
}

typedef __nv_bfloat16 bf16;

// Fixed widths of the decoder the kernels are built for.
constexpr int kD = 1280;        // hidden
constexpr int kH = 10;          // heads
constexpr int kHD = 128;        // head dim
constexpr int kE = 64;          // routed experts
constexpr int kTopK = 6;
constexpr int kShared = 2;
constexpr int kI = 896;         // expert intermediate
constexpr int kId = 3584;       // draft-block intermediate
constexpr int kSlots = kTopK + kShared;   // per-token expert outputs combined
constexpr int kAttnChunk = 64;            // split-KV chunk (keys), fixed by absolute position
constexpr int kAttnSuper = 4;             // chunks per attention super-chunk (one partial each)
constexpr int kAttnPartStride = 132;      // floats per (super-chunk, query) partial: O[128], M, L, pad
constexpr int kMaxR = 8;                  // K_max + 1 <= 8 candidate rows per sequence
constexpr int kMaxSplit = 8;              // split-K ways of a dense GEMM (a portable cluster)

// ------------------------------------------------------------------------- GEMM engine
enum EpiKind : int {
  EPI_F32 = 0,      // out[row][n] = acc
  EPI_RESID = 1,    // out[row][n] += acc (fp32 residual stream)
  EPI_QKV = 2,      // RoPE on q/k, q -> fp32 buffer, k/v -> bf16 cache rows
  EPI_SWIGLU = 3,   // tile = 64 gate rows + 64 up rows -> bf16 silu(g)*u
  EPI_SCATTER = 4,  // expert down: out row (token, slot) from the sorted index
  EPI_ARGMAX = 5,   // running (max, argmax) of each column in a packed key (LM head)
  EPI_MOE = 6,      // grouped gate/up (SWIGLU) items, then the down (SCATTER) items, one launch
  EPI_LOSS = 7      // draft-head objective: per (vocab tile, activation row) softmax statistics
};

// One work item: weight tile x activation rows.  x = expert | n_tile << 16, y = TMA row of
// the activation source, z = output row (row index of the epilogue), w = number of rows.
// Dense launches generate items from the shape; grouped launches from the per-expert row counts.
struct GemmArgs {
  CUtensorMap a_map[2];        // weights: [0] main / routed experts, [1] shared experts
  CUtensorMap b_map[2][5];     // activations: [source][box height 16,32,64,128,256]
  int N;                       // output features of the weight matrix (bounds of the last tile)
  int K;                       // reduction length, multiple of 64
  int a3d;                     // weight maps are 3-D [experts][rows][K]
  int paired;                  // SwiGLU: tile rows 0..63 gate, 64..127 up (offset half_rows)
  int half_rows;
  int n_routed;                // experts with id >= n_routed read a_map[1] and source 1
  int split_k;                 // >= 1, fixed per matrix shape
  int seq_split;               // dense, split_k > 1: one CTA computes every split of a tile into
                               // its own TMEM accumulator (64-row boxes), no partials in memory
  int cluster;                 // dense, split_k > 1, one item per CTA: the split_k CTAs of a tile
                               // are a cluster and add their partials through shared memory
  // Grouped launches (grp_cnt != NULL): the work is every (expert, 64-row tile, weight tile),
  // experts in order, routed experts e < n_routed with grp_cnt[e] rows, then the shared ones
  // with grp_T rows each; expert e's rows are rows e * map_stride + 0.. of its input and output.
  const int* grp_cnt;          // [n_routed] rows of each routed expert
  int grp_T;                   // rows of each shared expert (the step's tokens)
  int grp_tiles;               // weight tiles per expert
  int grp_b_direct;            // shared experts read activation rows 0..T-1 directly
  int grp_rows;                // row tile of the grouped items: kExpertTileRows or kExpertTileRowsLarge
  const int* rowmap;           // SCATTER: [n_routed][map_stride] (token << 3 | rank) of each row
  int map_stride;
  unsigned long long* expert_ctr;   // if set, CTA 0 adds (experts with rows, rows) of the launch
  // EPI_MOE: this struct describes the gate/up items, a second one (the kernel's second
  // argument) the down items.  The gate/up epilogue of (expert e, row tile m) adds one to
  // dep[e * dep_stride + m] after its SwiGLU rows are stored; a down item of (e, m) waits until
  // all grp_tiles gate/up tiles of (e, m) have.
  int* dep;
  int dep_stride;
  int n_items;                 // dense: number of items
  int M;                       // dense: activation rows
  int m_tiles, box_log;        // dense: row tiles of 16 << box_log rows
  int b_row_off;               // dense: first activation row read by TMA
  int n_tiles;                 // dense: weight tiles
  // epilogue operands
  float* out; int ldo;                                        // F32 / RESID
  bf16* q_out; bf16* kv_base; const long long* kv_rowoff;    // QKV (q stored bf16)
  long long head_stride, v_off; const int* pos; const float2* rope; int max_pos;
  bf16* act; int ld_act;                                      // SWIGLU
  float* y;                                                   // SCATTER: [T][8 slots][d]
  // ARGMAX: am_key[row] = max over tiles of (ordered logit << 32 | ~token) (atomicMax; zero =
  // empty).  fin_B > 0: the last CTA (ticket am_done) decodes the tokens of fin_B x fin_R rows,
  // computes the greedy accept lengths and clears the keys.
  unsigned long long* am_key; int* am_done;
  int fin_B, fin_R; const int* fin_cand; int* fin_vtok_out; int* fin_vtok_ws; int* fin_accept_out; int* fin_m_ws;
  float* sk_ws; int* sk_tickets;                              // split-K partials / per-tile tickets
  // LOSS (operands swapped: a_map = the packed activations, tiles of 128 rows, N their count;
  // b_map = W_lm, 256-row vocabulary tiles, M the vocabulary size): activation rows come in
  // groups of loss_G (a power of two, 2..8), row 0 of a group a verifier state b, rows 1.. draft
  // states u.  loss_part[vocab tile * ldo + row] = (max, sum of exp(x - max), sum of
  // exp(q - max_q) (q - x) with q the group's b-row logit, max_q) over the tile's vocabulary.
  // loss_G != 0 also makes dense items run through the A tiles first.
  float4* loss_part; int loss_G;
  int a_keep;                  // weight tiles loaded with the L2 evict-last policy (kept resident)
  // fp8 experts: both operands e4m3 bytes (k-chunks of 128 elements, tcgen05 kind::f8f6f4); the
  // SWIGLU / SCATTER epilogues multiply each weight row's accumulator by its fp32 scale
  // (w_scale[0]: routed experts [E][scale_rows], w_scale[1]: shared experts), and SWIGLU writes
  // its rows as e4m3 to act8.
  int f8;
  const float* w_scale[2];
  int scale_rows;
  uint8_t* act8;
  int* err;
};

// Encodes a 2-D or 3-D tensor map with the 128-byte swizzle: bf16 elements (elem_bytes 2, box
// inner dim 64) or e4m3 bytes (elem_bytes 1, box inner dim 128); `inner` counts elements.
bool encode_map_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                   std::string* err, int elem_bytes = 2);
bool encode_map_3d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t depth,
                   uint32_t box_rows, std::string* err, int elem_bytes = 2);
// Fills b_map[src][*] for an activation buffer of `rows` x `inner` elements.
bool encode_act_maps(CUtensorMap (&maps)[5], const void* base, uint64_t inner, uint64_t rows, std::string* err,
                     int elem_bytes = 2);

// Launches the persistent tcgen05 GEMM; nmax = 64 or 256 (largest row box of any item).
// pdl = false launches without programmatic serialization (for streams whose earlier kernels
// may still be writing the weights).
cudaError_t gemm_launch(int epi, int nmax, const GemmArgs& a, int grid, cudaStream_t s, bool pdl = true);
// The routed + shared experts' gate/up and down in one cooperative launch (EPI_MOE).
cudaError_t moe_launch(const GemmArgs& gate_up, const GemmArgs& down, cudaStream_t s);
int num_sms();
// Sets the message spec_last_error(NULL) returns in this thread.
void set_thread_error(const std::string& msg);
// Reads and clears the device guard flag of spec_gemm_bf16_noalloc's kernels on the current
// device (0 if that entry point never ran there); the caller has synchronised the device.
cudaError_t noalloc_take_flag(int* flag);
// The same for the GEMM of spec_draft_loss.
cudaError_t loss_take_flag(int* flag);
#ifdef FM_TRACE
// Device-timeline buffers of the three kernel translation units (FM_TRACE builds): copy up to
// `cap` records (4 x u64 each) to host memory, return the count (-1 on a CUDA error).
int trace_read_gemm(unsigned long long* host, int cap, bool reset);
int trace_read_attn(unsigned long long* host, int cap, bool reset);
int trace_read_small(unsigned long long* host, int cap, bool reset);
#endif
// Kernel attributes (dynamic shared memory limits) set once, before any launch or capture.
cudaError_t gemm_prepare();
cudaError_t attention_prepare();
cudaError_t router_prepare();

// Split-K count of a dense matrix: depends on (N, K) only, never on M, so every row's sum
// order is the same at any batch size.  From kSeqSplitRows activation rows on, the splits of
// a tile are computed by one CTA (GemmArgs::seq_split) instead of one CTA each.
int dense_split_k(int N, int K);
constexpr int kSeqSplitRows = 128;
// Row tile of the grouped expert launches (work-list items cover at most this many rows): 64
// rows (the 8-stage, 64-column kernel; a gate/up item is 64 gate + 64 up features, a down item
// 128 outputs) below kExpertLargeFromRows candidate rows, 128 rows from there on (the 4-stage
// dual kernel: an item is two 128-row weight tiles against one activation tile -- 128 gate and
// the 128 up features of the same outputs, or 256 down outputs -- so each activation tile is
// read once per 256 weight rows, and half as many items carry the per-item costs).  Below 16
// rows (B = 1 at K = 3: about 3.6 of the smaller items per CTA) the coarser items leave a
// longer tail than they save (measured).  The tile height only groups rows into items; every
// row's sums are the same at either height.
constexpr int kExpertTileRows = 64;
constexpr int kExpertTileRowsLarge = 128;
constexpr int kExpertLargeFromRows = 16;

// ------------------------------------------------------------------------- other kernels
struct AttnArgs {
  // The pool of this launch as a 2-D bf16 tensor [n_pages * 2 * H * page_size][hd], box 64 x
  // 64 with the 128-byte swizzle; used for chunks whose 64 keys are all committed when
  // use_tma is set (page_size a multiple of 64).
  CUtensorMap kv_map;
  int use_tma;
  const bf16* q;               // [rows][H][hd] bf16
  const int* q_row0;           // per sequence first query row (NULL: b * R)
  int R;                       // queries per sequence
  int qoff;                    // query r of sequence b sits at seq_len[slot] + qoff + r
  const int* slots; const int* seq_len;   // keys at positions < seq_len[slot] are in pages
  int n_slots;                 // valid slot ids are 0..n_slots-1
  const bf16* pool; int page_size; int n_pages; const int* block_table; int max_pages;
  const bf16* stage;           // keys at positions >= seq_len[slot]: staged row (pos - seq_len)
  long long stage_seq_stride, stage_row_stride, stage_kv_stride;
  float* part;                 // [B][H][ceil(n_chunks / 4)][R][132] super-chunk partials
  int* tickets;                // [B][H] super-chunk counters, zero between launches
  int n_chunks;                // most chunks a sequence may span (pool capacity + staged rows)
  int B;                       // sequences of this launch (set by attention_launch)
  // Set when no kernel of the same graph writes the pages, the block table, the slots or the
  // lengths (the verify step): the K/V of the first committed chunks is then fetched before
  // the wait for the previous kernel.
  int prewait;
  // With prewait: only chunks whose keys all sit below seq_len - prewait_guard are fetched before
  // the wait (the draft step writes the draft pool's last K_max + 1 committed rows itself).
  int prewait_guard;
  bf16* out;                   // [B*R][H*hd]
  int out_row_stride_seq;      // rows of out per sequence (R)
  int* err;
};
cudaError_t attention_launch(const AttnArgs& a, int B, cudaStream_t s);

cudaError_t embed_norm_launch(const int* cand, int B, int R, const int* slots, const int* pending,
                              const int* seq_len, const bf16* embed, int vocab, const bf16* gain, float eps,
                              float* h, bf16* xn, int* pos, long long* kv_rowoff, int stage_R, int n_slots,
                              int* err, int* zero, int n_zero, int* zero2, int n_zero2, cudaStream_t s);
// Router: RMSNorm, logits, softmax, top-6; each selection claims the next row of its expert
// (atomic add on counts) and copies the token's rounded row into the expert's input region.
struct RouteArgs {
  const float* h; const bf16* gain; float eps; const bf16* wr; const float* bias;
  bf16* xn; int* idx; float* gate; int* err; int T;
  int* counts;     // [64] rows routed to each expert so far (zero before the layer's router)
  int* rowmap;     // [64][map_stride] per expert: (token << 3 | rank) of each of its rows
  bf16* x_sorted;  // [64][map_stride][d] per expert: its input rows (the rounded xn rows)
  int map_stride;  // >= T
  // fp8 experts (else NULL): the rows rounded to e4m3 -- every token row into xn8 [T][d] (the
  // shared experts' input) and each selection into x_sorted8 [64][map_stride][d] instead of x_sorted
  uint8_t* xn8;
  uint8_t* x_sorted8;
};
cudaError_t router_launch(const RouteArgs& a, cudaStream_t s);
cudaError_t combine_launch(float* h, const float* y, const float* gate, int T, const bf16* gain, float eps,
                           bf16* out, cudaStream_t s);
cudaError_t commit_launch(int B, int R, int stage_R, int Bmax, const int* slots, const int* m_ws, const int* vtok_ws,
                          const int* cand_ws, const bf16* stage, bf16* pool, int L, int n_pages,
                          int page_size, const int* block_table, int max_pages, int* seq_len, int* pending,
                          const bf16* b_ws, bf16* draft_b, int* draft_tok, int* draft_n, int* committed,
                          int* n_committed, int* tickets, int* err, cudaStream_t s);
cudaError_t draft_prep_launch(int B, int R, const int* slots, const int* seq_len, const int* pending,
                              const int* draft_n, const bf16* draft_b, const int* draft_tok,
                              const bf16* embed, int vocab, const bf16* enorm, const bf16* hnorm, float eps,
                              bf16* dcat, int* pos, long long* kv_rowoff, int* last_row, int page_size,
                              const int* block_table, int max_pages, int n_pages, int* cand, int cand_ld,
                              int n_slots, int* err, cudaStream_t s);
cudaError_t rmsnorm_launch(const float* x, int rows, const bf16* gain, float eps, bf16* out, cudaStream_t s);
cudaError_t gather_rows_launch(const float* src, const int* rows, int B, float* dst, cudaStream_t s);
cudaError_t draft_next_launch(unsigned long long* am_key, int vocab, int* err, int B, int k, int K, const int* slots,
                              int n_slots, const int* seq_len, const bf16* u, const bf16* embed,
                              const bf16* enorm, const bf16* hnorm, float eps, bf16* dcat, int* pos,
                              long long* kv_rowoff, long long dstage_seq_stride, int* cand, int cand_ld,
                              cudaStream_t s);

}  // namespace fm
