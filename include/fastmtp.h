/*
 * fastmtp.h -- C ABI of the GB300 (sm_103a) FastMTP speculative decode step.
 *
 * The operation is the speculative greedy decode step of arXiv 2609.03181 ("Jina-OCR-v1"),
 * Sec. 3 "Model Architecture" and Sec. 3.1 "Draft-head architecture":
 *   draft_step   -- the FastMTP draft head (draft-head equation of Sec. 3.1): one shared
 *                   dense block B_theta applied recursively K times along the diagonal
 *                   p = j+k-1 (Fig. "FastMTP state-shift alignment"), with the embedding E,
 *                   output norm N_o and LM head W_lm tied to the verifier;
 *   verify_step  -- the verifier forward of the DeepSeekMoE decoder (Table "Model
 *                   specification": 12 layers, d=1280, 64 routed + 2 shared experts, top-6,
 *                   vocabulary 129,280, RoPE theta=1e6) over the K+1 candidates of every
 *                   sequence against its paged bf16 KV cache, then greedy acceptance: per-row
 *                   argmax v_r and the longest equality prefix m (acceptance equation of
 *                   Sec. 3.1);
 *   accept_commit-- commit x^_{1:m} then v_{m+1} (the bonus token when m = K), append the
 *                   K/V of the accepted candidates to the cache, drop the rejected tail.
 * The committed stream equals plain greedy decoding (K = 0) for any drafts (Sec. 3.1).
 *
 * Conventions (all entry points):
 *  - Pointers marked "dev" are CUDA device pointers on the device that was current at
 *    spec_init; "host" pointers are host memory.  Sizes are element counts.
 *  - Weights and KV pools are owned by the caller and borrowed for the context's lifetime.
 *    The context owns only its workspace (allocated once in spec_init, freed in
 *    spec_destroy); no step allocates memory.
 *  - Every step is asynchronous on the stream given to spec_init.  Arguments are validated
 *    on the host before any launch; a rejected call launches nothing and leaves the state
 *    unchanged.  Data-dependent faults found on the device (a token id out of range, a page
 *    index outside the pool, a slot id in a device array outside [0, max_batch), a
 *    candidate 0 that is not the pending token, a non-finite router row, a wait that ran
 *    out) set a device guard flag instead of trapping, and the affected work is skipped or
 *    clamped to a valid index; spec_sync() reports it as SPEC_EDEVICE.  Kernels never trap
 *    and never spin without a time limit.
 *  - bf16 tensors are row-major with the last dimension contiguous; matrices are stored
 *    [out_features][in_features].
 *  - Layout of the verifier KV pool (bf16): [n_layers][n_pages_total][2 (K,V)][n_heads]
 *    [page_size][head_dim]; keys are stored after RoPE.  The draft-block pool has the same
 *    layout with one layer.  Both caches of a sequence use the same block table.
 */
#ifndef FASTMTP_H
#define FASTMTP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct spec_ctx spec_ctx;  /* opaque */

typedef enum {
  SPEC_OK = 0,
  SPEC_EINVAL = 1,   /* bad argument (host-side check); nothing launched */
  SPEC_ENOMEM = 2,   /* workspace allocation failed in spec_init */
  SPEC_ECUDA = 3,    /* a CUDA runtime call failed; message in spec_last_error */
  SPEC_ESTATE = 4,   /* call out of order (e.g. accept_commit without a verify_step) */
  SPEC_EDEVICE = 5   /* the device guard flag is set (see spec_sync) */
} spec_status;

/* Shape contract.  The kernels are built for hidden = 1280, n_heads = 10, head_dim = 128,
 * n_experts = 64, top_k = 6, n_shared = 2, expert_inter = 896, draft_inter = 3584 (the
 * paper's decoder with the widths the paper leaves open); spec_init rejects other values of
 * those fields.  vocab, n_layers, page_size and the capacity fields are free. */
typedef struct spec_config {
  int32_t hidden, n_heads, head_dim, n_layers;
  int32_t n_experts, top_k, n_shared, expert_inter, draft_inter, vocab;
  int32_t page_size;          /* tokens per KV page, a multiple of 16 */
  int32_t max_batch;          /* largest B of any step; also the number of sequence slots */
  int32_t max_pages_per_seq;  /* block-table width */
  int32_t n_pages_total;      /* pages in each pool */
  int32_t K_max;              /* largest draft depth K, 0..7 */
  int32_t max_position;       /* RoPE table length (position limit, e.g. 32768) */
  float rms_eps, rope_theta;  /* 1e-6, 1e6 */
  /* 0: bf16 expert weights (the paper's model).  1: fp8 experts, a precision option with no
   * counterpart in the paper: the routed and shared expert matrices are e4m3 byte codes (1 sign,
   * 4 exponent bits with bias 7, 3 mantissa bits) with one fp32 scale per output row (the
   * *_scale pointers of spec_layer_weights), and the rows entering the expert products (the
   * normalised token rows and the SwiGLU activations) are rounded to e4m3 (ties to even,
   * saturating at 448); products in fp32 (tcgen05 kind::f8f6f4). */
  int32_t expert_fp8;
} spec_config;

/* One verifier layer (all dev, bf16 unless noted). */
typedef struct spec_layer_weights {
  const void* attn_norm;       /* [d] */
  const void* wqkv;            /* [3*H*hd][d]: q rows, then k rows, then v rows */
  const void* wo;              /* [d][H*hd] */
  const void* moe_norm;        /* [d] */
  const void* router;          /* [E][d] */
  const void* w_gate_up;       /* [E][2I][d]: gate rows 0..I-1, up rows I..2I-1 */
  const void* w_down;          /* [E][d][I] */
  const void* shared_gate_up;  /* [n_shared][2I][d] */
  const void* shared_down;     /* [n_shared][d][I] */
  const float* router_bias;    /* fp32 [E] added to the router logits, or NULL */
  /* expert_fp8 only (else ignored): fp32 scale of every row of w_gate_up [E][2I], w_down [E][d],
   * shared_gate_up [n_shared][2I], shared_down [n_shared][d]; the four expert matrices above
   * are then e4m3 codes (1 byte per element, same shapes). */
  const float* gate_up_scale;
  const float* down_scale;
  const float* shared_gate_up_scale;
  const float* shared_down_scale;
} spec_layer_weights;

/* All weights (dev, bf16).  E, N_o and W_lm are shared by the verifier and the draft head
 * (Sec. 3.1: tied); the mtp_* block is B_theta, enorm/hnorm are N_e/N_h, eh_proj is P. */
typedef struct spec_weights {
  const void* embed;            /* [V][d] */
  const void* lm_head;          /* [V][d] */
  const void* final_norm;       /* [d] (N_o) */
  const spec_layer_weights* layers;  /* host array of n_layers */
  const void* enorm;            /* [d] */
  const void* hnorm;            /* [d] */
  const void* eh_proj;          /* [d][2d]: input [N_e(e); N_h(a)] */
  const void* mtp_attn_norm;    /* [d] */
  const void* mtp_wqkv;         /* [3*H*hd][d] */
  const void* mtp_wo;           /* [d][H*hd] */
  const void* mtp_ffn_norm;     /* [d] */
  const void* mtp_w_gate_up;    /* [2*Id][d]: gate rows, then up rows */
  const void* mtp_w_down;       /* [d][Id] */
} spec_weights;

/* Creates a context on the current device.  kv_pool / draft_kv_pool: dev, layouts above,
 * n_pages_total pages each.  stream: a cudaStream_t (NULL = legacy default stream).  Builds
 * the TMA descriptors of every weight matrix and the RoPE table, allocates the workspace
 * (sized for max_batch x (K_max+1) rows) and zeroes all sequence slots.
 * Errors: SPEC_EINVAL (shape contract, null pointer, misaligned matrix), SPEC_ENOMEM,
 * SPEC_ECUDA.  On error *out is NULL. */
spec_status spec_init(const spec_config* cfg, const spec_weights* w, void* kv_pool,
                      void* draft_kv_pool, void* stream, spec_ctx** out);

/* Sets sequence slot `slot` to a committed prefix: ctx_len KV positions already in both
 * pools (positions 0..ctx_len-1 of the verifier cache and rows 0..ctx_len-1 of the draft
 * cache), pending token `pending` (committed, not yet consumed, at position ctx_len), and
 * its block table (host int32 [max_pages_per_seq], page ids into both pools; entries the
 * sequence will never reach may be -1).  The slot has no queued draft rows: the first step
 * on it must be verify_step with K = 0.  Synchronous with the stream.  Errors: SPEC_EINVAL
 * (slot, ctx_len, token or page id out of range). */
spec_status spec_seq_reset(spec_ctx* ctx, int32_t slot, int32_t ctx_len,
                           const int32_t* block_table, int32_t pending);

/* Queues n_rows (1..K_max+1) draft rows on slot `slot` as if a commit had just made them:
 * base states b_p (dev bf16 [n_rows][d]) of rows p = ctx_len-n_rows .. ctx_len-1 and the
 * tokens x_{p+1} that follow them (host int32 [n_rows]; the last one must equal the
 * pending token).  Lets a caller start the draft head from states computed elsewhere.
 * Synchronous.  Errors: SPEC_EINVAL. */
spec_status spec_seq_set_draft_rows(spec_ctx* ctx, int32_t slot, int32_t n_rows,
                                    const void* b_rows, const int32_t* next_tokens);

/* FastMTP draft step (Sec. 3.1) for B sequences (dev int32 slots[B], distinct).  For each
 * sequence the rows queued by the last commit enter the draft cache at depth 1 (committed,
 * base states), then the chain from the last of them drafts x^_1..x^_K.  Writes
 * cand (dev int32 [B][K+1]) = [pending token, x^_1, .., x^_K], the candidate layout
 * verify_step takes.  1 <= K <= K_max.  Errors: SPEC_EINVAL, SPEC_ESTATE (a verify is
 * waiting for its accept_commit). */
spec_status draft_step(spec_ctx* ctx, int32_t B, int32_t K, const int32_t* slots,
                       int32_t* cand);

/* Verifier forward + greedy acceptance for B sequences.  cand: dev int32 [B][K+1] with
 * cand[b][0] the pending token of slots[b] and cand[b][1..K] its drafts; candidate r sits at
 * position ctx_len + r.  Writes verifier_tokens (dev int32 [B][K+1], v_{r+1} = argmax of row
 * r, lowest id on ties) and accept_len (dev int32 [B], m in 0..K).  The K/V of the
 * candidates are staged in the workspace, not yet in the pools.  0 <= K <= K_max; K = 0 is
 * one step of plain greedy decoding.  Errors: SPEC_EINVAL, SPEC_ESTATE (previous verify not
 * committed). */
spec_status verify_step(spec_ctx* ctx, int32_t B, int32_t K, const int32_t* slots,
                        const int32_t* cand, int32_t* verifier_tokens, int32_t* accept_len);

/* Commits the last verify_step (same B and slots): copies the staged K/V of candidates
 * 0..m into the verifier pool, advances ctx_len by m+1, makes v_{m+1} the pending token and
 * queues the m+1 new rows for the next draft_step.  Writes committed (dev int32 [B][K+1]:
 * x^_1..x^_m, v_{m+1}; entries past m+1 are -1) and n_committed (dev int32 [B] = m+1).
 * Errors: SPEC_EINVAL, SPEC_ESTATE (no verify to commit). */
spec_status accept_commit(spec_ctx* ctx, int32_t B, const int32_t* slots, int32_t* committed,
                          int32_t* n_committed);

/* Waits for the context's stream and reports the device guard flag: SPEC_OK, or
 * SPEC_EDEVICE with the flag bits in spec_last_error (the flag is then cleared).  Also
 * SPEC_ECUDA if the stream reports an error.
 * With ctx NULL: waits for the whole current device (cudaDeviceSynchronize) and reports the
 * guard flags of the context-free entry points spec_gemm_bf16, spec_gemm_bf16_noalloc and
 * spec_draft_loss on that device (1 = a pipeline wait ran out and the tiles it covers were
 * left unwritten), with
 * the bits in spec_last_error(NULL); the flags are then cleared.  Allocates nothing. */
spec_status spec_sync(spec_ctx* ctx);

/* Reads one slot's state (synchronous): committed KV length and pending token. */
spec_status spec_seq_state(spec_ctx* ctx, int32_t slot, int32_t* ctx_len, int32_t* pending);

/* Workspace views for tests and statistics.  Copies (synchronously) `bytes` bytes of the
 * named workspace tensor into host memory `dst`.  Valid after the step that writes it:
 *   SPEC_WS_B          bf16 [B][K+1][d]    post-norm verifier states b = N_o(h_L)
 *   SPEC_WS_ROUTE_IDX  int32 [L][B*(K+1)][top_k] selected experts per layer (row b*(K+1)+r)
 *   SPEC_WS_ROUTE_GATE fp32 [L][B*(K+1)][top_k] their router probabilities
 *   SPEC_WS_EXPERT_CNT int32 [L][n_experts] tokens routed to each expert
 *   SPEC_WS_DRAFT_U    bf16 [K][B][d]      draft states u^(k) of the last draft_step
 *   SPEC_WS_HIDDEN     fp32 [B*(K+1)][d]   residual stream after the last layer
 * Errors: SPEC_EINVAL (unknown id or bytes larger than the tensor). */
enum { SPEC_WS_B = 0, SPEC_WS_ROUTE_IDX = 1, SPEC_WS_ROUTE_GATE = 2, SPEC_WS_EXPERT_CNT = 3,
       SPEC_WS_DRAFT_U = 4, SPEC_WS_HIDDEN = 5 };
spec_status spec_read_workspace(spec_ctx* ctx, int32_t id, void* dst, size_t bytes);

/* Dense projection Y = X W^T on the tcgen05 GEMM engine every projection of the step runs
 * on (X dev bf16 [M][Kdim], W dev bf16 [N][Kdim], Y dev fp32 [M][N]); M >= 1, N a multiple
 * of 128 or any N >= 1 (a ragged last tile is masked), Kdim a multiple of 64, both base
 * pointers 16-byte aligned.  Asynchronous on `stream`; needs no context.  Errors:
 * SPEC_EINVAL, SPEC_ECUDA. */
spec_status spec_gemm_bf16(const void* X, const void* W, float* Y, int32_t M, int32_t N,
                           int32_t Kdim, void* stream);

/* Dense e4m3 projection Y = (X W^T) * scale on the same tcgen05 engine as the fp8 experts
 * (kind::f8f6f4): X dev e4m3 codes [M][Kdim], W dev e4m3 codes [N][Kdim] (1 sign, 4 exponent
 * bits with bias 7, 3 mantissa bits), w_scale dev fp32 [N] (one per row of W), Y dev fp32
 * [M][N]; Kdim a multiple of 128, both code pointers 16-byte aligned.  A precision option with
 * no counterpart in the paper.  Asynchronous on `stream`; needs no context.  Errors:
 * SPEC_EINVAL, SPEC_ECUDA; device-side faults via spec_sync(NULL). */
spec_status spec_gemm_e4m3(const void* X, const void* W, const float* w_scale, float* Y, int32_t M, int32_t N,
                           int32_t Kdim, void* stream);

/* Kernel-class timing for measurement.  spec_profile(ctx, mode): mode 1 zeroes the counters
 * and starts recording a CUDA event pair around every launch group (inside the captured CUDA
 * graph of each call, as external event nodes; a profiled call then waits for its graph to
 * finish); mode 2 zeroes the counters without recording events; mode 0 stops recording.
 * Launch counts and the expert counters are kept in every mode.  spec_profile_read waits for
 * the stream and fills *out:
 *   launches[c], ms[c]  kernel launches and summed event time of class c (SPEC_K_*);
 *   experts_touched     routed + shared experts with at least one row, summed over the
 *                       grouped gate/up launches (the expert weight bytes actually read);
 *   expert_rows         (token, expert) rows processed by those launches.
 * SPEC_K_PERMUTE stays in the numbering but no longer launches: the router writes each
 * expert's input rows itself. */
enum { SPEC_K_EMBED = 0, SPEC_K_QKV = 1, SPEC_K_ATTN = 2, SPEC_K_OPROJ = 3, SPEC_K_ROUTER = 4,
       SPEC_K_PERMUTE = 5, SPEC_K_EXPERT_GU = 6, SPEC_K_EXPERT_DN = 7, SPEC_K_COMBINE = 8,
       SPEC_K_LMHEAD = 9, SPEC_K_ARGMAX = 10, SPEC_K_COMMIT = 11, SPEC_K_DRAFT_GEMM = 12,
       SPEC_K_DRAFT_MISC = 13, SPEC_K_COUNT = 14 };
typedef struct spec_profile_t {
  int64_t launches[SPEC_K_COUNT];
  double ms[SPEC_K_COUNT];
  int64_t experts_touched;
  int64_t expert_rows;
} spec_profile_t;
spec_status spec_profile(spec_ctx* ctx, int32_t mode);
spec_status spec_profile_read(spec_ctx* ctx, spec_profile_t* out);

/* Device timeline for measurement (no counterpart in the paper; it backs the per-kernel time
 * breakdown of the step).  A library built with FASTMTP_TRACE=1 (a separate build, see the
 * package's build script) records, for thread 0 of every CTA of every kernel, the global timer at
 * entry, when its first wait for the previous kernel returns and, for the GEMM, attention, router
 * and combine kernels, at exit.  spec_trace_read waits for the device, copies up to `cap`
 * records to `host_records` (host memory, 4 x uint64 each: signature, block index, t_a, t_b;
 * signature = kernel id << 48 | gridDim.x << 32 | gridDim.y << 16 | blockDim.x, bit 63 set on
 * exit records, whose t_a is the exit time; other records carry entry time and wait-return
 * time in nanoseconds), stores the count in *n_records and, if `reset`, empties the device
 * buffers (65,536 records per kernel source file; later records are dropped).  Kernel ids:
 * 1 + GEMM epilogue (1 plain fp32, 2 residual, 3 QKV, 4 SwiGLU, 5 scatter, 6 argmax, 7 fused
 * experts), 16 attention, 17 router, 18 combine, 19 embedding, 20 RMSNorm, 21 commit, 22-24
 * draft glue.  Errors: SPEC_EINVAL for a NULL n_records, cap < 0, a NULL buffer with cap > 0,
 * or a library built without the timeline (then *n_records = 0); SPEC_ECUDA if a copy fails.
 * Messages via spec_last_error(NULL). */
spec_status spec_trace_read(void* host_records, int32_t cap, int32_t reset, int32_t* n_records);

/* Y = X W^T like spec_gemm_bf16, computed split-K, for callers that cannot allocate device
 * memory: code running while a stream is captured into a CUDA graph (an allocation there is
 * rejected or breaks the capture), runtimes that give out device memory only from their own
 * fixed pool, serving loops where a hidden cudaMalloc would stall the device.  (The paper has
 * no counterpart; this is an interface for such callers.)  The split-K partial tiles and
 * tickets live in a fixed file-scope device array of 4 MiB + 4 KiB that every GPU loading the
 * library holds until the process exits; the call allocates and frees nothing.  The first call
 * on a device looks the array up on that device (it must be current) and should come before
 * any stream capture; host threads may make first calls concurrently (the lookup is locked).
 * Every call shares the array and leaves its last contents there; the call clears the tickets
 * it uses before its kernel runs.  Calls whose kernels overlap on the GPU race on the array:
 * keep them on one stream.  Splits: min(SM count / ceil(N/128), Kdim/128, 8), at least 1.
 * Limits: ceil(N/128) * ceil(M/box) * splits * box * 128 floats <= 2^20, box the row tile
 * (16, 32, 64, 128 or 256: the smallest power of two >= min(M, 256), at least 16); e.g. M <= 64
 * with N <= 4096 at Kdim = 1280, or M = 256 with N <= 512 on a 152-SM GPU.  Larger problems get
 * SPEC_EINVAL with the reason in spec_last_error(NULL).  Device-side faults (a pipeline wait
 * that ran out) are not returned by this call, which does not wait for its kernel: they set a
 * guard flag that spec_sync(NULL) reports.  Same argument rules and errors as spec_gemm_bf16
 * otherwise; asynchronous on `stream`. */
spec_status spec_gemm_bf16_noalloc(const void* X, const void* W, float* Y, int32_t M, int32_t N,
                                   int32_t Kdim, void* stream);

/* Draft-head training objective (Sec. 5.6 "Draft-head objective": the CE, KL and MSE terms per
 * recursive depth and their alpha-weighted sum).  For rows p = 0..n_rows-1 and depths
 * k = 1..K (1 <= K <= 7):
 *   CE_k  = mean_p -log softmax(W_lm u_p^(k))[x_{p+2}]
 *   KL_k  = mean_p KL(Q_p || softmax(W_lm u_p^(k))),  Q_p = softmax(W_lm b_{p+1})
 *   MSE_k = mean_p ||u_p^(k) - b_{p+1}||^2
 *   L     = w_ce sum_k alpha_k CE_k + w_kl sum_k alpha_k KL_k + w_mse sum_k alpha_k MSE_k,
 *           alpha_k = beta^(k-1) / sum_{r=1..K} beta^(r-1)   (the paper: beta 0.6, w 0.85/0.45/0.45)
 * the means taken over the rows with valid[p] != 0.  Arguments (dev unless noted):
 *   u        bf16 [K][n_rows][d]   draft states u_p^(k) (d = 1280, 16-byte aligned)
 *   b_next   bf16 [n_rows][d]      verifier states b_{p+1} (the detached targets)
 *   target   int32 [n_rows]        tokens x_{p+2}; an id outside [0, vocab) makes that row's CE NaN
 *   valid    int32 [n_rows] or NULL (every row counted)
 *   lm_head  bf16 [vocab][d]       the tied LM head (16-byte aligned)
 *   out      fp32 [1 + 3K]         L, CE_1..CE_K, KL_1..KL_K, MSE_1..MSE_K
 *   row_out  fp32 [K][n_rows][3] or NULL: per row (CE, KL, MSE), valid or not
 *   workspace, workspace_bytes: caller-owned device memory (256-byte aligned) of at least the
 *            size spec_draft_loss_workspace returns; the call allocates nothing.
 * One pass over W_lm: the logits are reduced on chip to per-row softmax statistics and never
 * written.  Asynchronous on `stream`; calls sharing a workspace must not overlap.  Device-side
 * faults (a pipeline wait that ran out) set a guard flag that spec_sync(NULL) reports.
 * Errors: SPEC_EINVAL (null pointer, sizes, alignment, workspace too small, beta <= 0 or a
 * non-finite weight), SPEC_ECUDA. */
spec_status spec_draft_loss_workspace(int32_t K, int32_t n_rows, int32_t vocab, size_t* bytes);
spec_status spec_draft_loss(const void* u, const void* b_next, const int32_t* target, const int32_t* valid,
                            const void* lm_head, int32_t K, int32_t n_rows, int32_t vocab, float beta,
                            float w_ce, float w_kl, float w_mse, float* out, float* row_out,
                            void* workspace, size_t workspace_bytes, void* stream);

/* Frees the workspace.  Borrowed weights and pools are untouched.  NULL is ignored. */
void spec_destroy(spec_ctx* ctx);

/* Last error message of the context ("" if none); NULL ctx gives the last error of
 * spec_init / spec_gemm_bf16 in this thread. */
const char* spec_last_error(const spec_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* FASTMTP_H */
