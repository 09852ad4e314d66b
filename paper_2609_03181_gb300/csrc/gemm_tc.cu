// Persistent tcgen05 GEMM engine for the decode regime (few activation rows, weight bytes
// dominate).  Every projection of the verify and draft steps runs here: QKV (+RoPE, KV
// staging), O-proj (+residual), the grouped routed/shared expert SwiGLU FFNs, the draft
// block's projections and the LM head (+argmax, logits never written).
//
// Swap-AB tiling: the weight matrix W [N][K] is the MMA's A operand (M = 128 weight rows
// per tile), the activations X [rows][K] are the B operand (N = 16..256 rows), so a tile
// D^T[128][rows] = W_tile X^T accumulates in TMEM.  Both operands are K-major bf16 tiles of
// 64 columns loaded by TMA with the 128-byte swizzle.  One CTA per SM; warp 0 issues TMA,
// warp 1 owns TMEM and issues tcgen05.mma from one thread, warps 2-5 drain the
// double-buffered accumulator through tcgen05.ld and run the fused epilogue.
//
// Determinism: each output element is the fp32 sum of its K range in the fixed k-chunk
// order; split-K partials are reduced by the last-arriving CTA of a tile in split order (an
// atomic ticket, no spin-wait).  Split counts depend on the matrix shape only, so a row's
// result never depends on how many other rows share the launch.
#include <cuda_fp8.h>
#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

// NMAX: most activation rows of a tile; ST: pipeline stages (8 for the long weight streams, 4
// for the short per-split streams of the dense cluster schedule, which leaves room on the SM
// for the CTAs of the next kernel to start early).
// DUAL (the expert launch's large-row items, NMAX = 128): every stage holds two 128-row weight
// tiles multiplied by the same activation tile into two accumulators (gate and up features of
// the same outputs, or two output tiles of the down projection).
template <int NMAX, int ST = (NMAX <= 64) ? 8 : 4, bool DUAL = false>
struct Cfg {
  static constexpr int A_BYTES = (DUAL ? 2 : 1) * 128 * 128;   // 128 rows x 64 bf16, per weight tile
  static constexpr int B_BYTES = NMAX * 128;           // NMAX rows x 64 bf16
  static constexpr int STAGES = ST;
  static constexpr int TMEM_COLS = (DUAL ? 4 : 2) * NMAX;   // two accumulator buffers (of two with DUAL)
  static constexpr int XCHG_FLOATS = 128 * 17;
  static constexpr int AM_BYTES = 128 * 8;             // argmax partials of 8 row groups x 16 columns
  static constexpr int META_BYTES = 256 * 16;          // per-row metadata of an item (QKV, SCATTER)
  static constexpr int ROPE_BYTES = 2 * 16 * 64 * 8;   // QKV: RoPE factors of two 16-row chunks
  static constexpr int SMEM_BYTES =
      1024 + STAGES * (A_BYTES + B_BYTES) + 256 + XCHG_FLOATS * 4 + AM_BYTES + META_BYTES + ROPE_BYTES;
};

constexpr int kShallowStages = 4;   // stages of the dense cluster schedule

// The configuration of an instantiation: the expert launch with 128-row items is the DUAL one.
template <int NMAX, int EPI, int ST>
using KCfg = Cfg<NMAX, ST, EPI == EPI_MOE && NMAX == 128>;

struct Item {
  int e, n_tile, b_row, out_row, rows, split, box_log;
  int grow;   // grouped: first row of the item within its expert
  int phase;  // EPI_MOE: 0 gate/up item, 1 down item
};

// Per-expert tables of a grouped launch in shared memory, built by every CTA from the counts,
// indexed by list position p (the shared experts first -- they have the most rows, so their
// down items are free to start early -- then the routed experts in order): grp[p] first item
// of the expert at p (grp[66] = items), grp[67 + p] its rows, and for EPI_MOE grp[134 + p] its
// first down item counted from the first down item.
constexpr int kGrpItem = 0, kGrpCnt = kE + kShared + 1, kGrpDn = 2 * (kE + kShared + 1);
__device__ __forceinline__ int grp_expert(int p) { return p < kShared ? kE + p : p - kShared; }

template <int EPI>
__device__ __forceinline__ void get_item(const GemmArgs& a, const GemmArgs& a2, int i, Item& it, const int* grp) {
  it.phase = 0;
  if (a.grp_cnt != nullptr) {
    const int* pre = grp + kGrpItem;
    const GemmArgs* P = &a;
    if (i >= grp[kGrpItem + kE + kShared]) {   // past the gate/up items: an EPI_MOE down item
      i -= grp[kGrpItem + kE + kShared];
      pre = grp + kGrpDn;
      P = &a2;
      it.phase = 1;
    }
    int lo = 0, hi = kE + kShared - 1;   // the last position whose first item is <= i has items
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (pre[mid] <= i) lo = mid;
      else hi = mid - 1;
    }
    const int j = i - pre[lo], m = j / P->grp_tiles;
    it.e = grp_expert(lo);
    it.n_tile = j - m * P->grp_tiles;
    it.grow = a.grp_rows * m;
    it.rows = min(a.grp_rows, grp[kGrpCnt + lo] - it.grow);
    it.out_row = it.e * a.map_stride + it.grow;
    it.b_row = (P->grp_b_direct && it.e >= a.n_routed) ? it.grow : it.out_row;
    it.split = 0;
    int bl = 0;
    while ((16 << bl) < it.rows) ++bl;
    it.box_log = bl;
  } else {
    it.grow = 0;
    // items run through the activation tiles first, or (EPI_LOSS: the two operands swapped, A =
    // activations) through the A tiles first, so that the CTAs reading one B tile run together
    constexpr bool swapped = (EPI == EPI_LOSS);
    const int mt = swapped ? i / a.n_tiles : i % a.m_tiles;
    const int t = swapped ? i % a.n_tiles : i / a.m_tiles;
    const int ns = a.seq_split ? 1 : a.split_k;   // in-CTA splits: one item covers every split
    it.split = t % ns;
    it.n_tile = t / ns;
    it.e = 0;
    const int box = 16 << a.box_log;
    it.out_row = mt * box;
    it.b_row = a.b_row_off + it.out_row;
    it.rows = min(box, a.M - it.out_row);
    it.box_log = a.box_log;
  }
}

// ------------------------------------------------------------------ epilogues
// v: 16 accumulator columns (activation rows j0..j0+15 of the item) of tile row `row`.
// epi_pre issues the global loads a chunk needs (the old residuals, the scatter targets, the
// RoPE factors) into registers; the chunk loops call it one chunk ahead, so a chunk's loads
// are in flight while the previous chunk computes and stores.  epi_post computes and
// stores.  Shared scratch: xchg [128][17] floats, am_val/am_idx [128], s_pos/s_off [256].
struct EpiPre {
  float old[16];
};

struct EpiSmem {
  float* xchg;
  float* xchg2;       // SWIGLU: the second exchange buffer (in the RoPE region, past the grouped tables)
  float* am_val;
  int* am_idx;
  int* s_pos;         // QKV: position of each row of the item; SCATTER: token
  int* s_aux;         // SCATTER: slot
  long long* s_off;   // QKV: staging offset
  float2* rope;       // QKV: [2][16 rows][64] cos/sin of a chunk's positions (double-buffered)
};

template <int EPI>
__device__ __forceinline__ void epi_pre(const GemmArgs& a, const Item& it, int row, int j0, const EpiSmem& sm,
                                        EpiPre& p) {
  if constexpr (EPI == EPI_RESID) {
    const int n = it.n_tile * 128 + row;
    if (n < a.N) {
      const float* base = a.out + static_cast<size_t>(it.out_row + j0) * a.ldo + n;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) p.old[jj] = (j0 + jj < it.rows) ? base[static_cast<size_t>(jj) * a.ldo] : 0.f;
    }
  }
}

// Rotate-half RoPE of the pair (x_i, x_{i+64}) with (cos, sin) = f, rounded the same way in
// every epilogue: lo' = x_i cos - x_{i+64} sin, hi' = x_{i+64} cos + x_i sin.
__device__ __forceinline__ float rope_lo(float lo, float hi, float2 f) { return __fmaf_rn(lo, f.x, -__fmul_rn(hi, f.y)); }
__device__ __forceinline__ float rope_hi(float hi, float lo, float2 f) { return __fmaf_rn(hi, f.x, __fmul_rn(lo, f.y)); }

// QKV with RoPE (q and k tiles): the cos/sin rows of a chunk's 16 positions, fetched by all
// 128 epilogue threads as 16-byte pieces (rope_load, issued a chunk ahead) and put into one of
// two shared buffers (rope_store) before the barrier that precedes their use.
struct RopeRegs {
  float4 r[4];
};
__device__ __forceinline__ void rope_load(const GemmArgs& a, const Item& it, int j0, const EpiSmem& sm, RopeRegs& rr) {
  const int t = threadIdx.x - 64;
  bool bad = false;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int idx = t + 128 * k, r = idx >> 5, piece = idx & 31;   // 16 rows x 32 pieces of 16 bytes
    int q = (j0 + r < it.rows) ? sm.s_pos[j0 + r] : 0;
    if (q < 0 || q >= a.max_pos) {
      bad = true;
      q = 0;
    }
    rr.r[k] = *reinterpret_cast<const float4*>(a.rope + static_cast<size_t>(q) * (kHD / 2) + piece * 2);
  }
  if (bad) atomicOr(a.err, ERR_POSITION);
}
__device__ __forceinline__ void rope_store(const EpiSmem& sm, int buf, const RopeRegs& rr) {
  const int t = threadIdx.x - 64;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int idx = t + 128 * k, r = idx >> 5, piece = idx & 31;
    *reinterpret_cast<float4*>(sm.rope + (buf * 16 + r) * 64 + piece * 2) = rr.r[k];
  }
}

// The per-row metadata of an item into shared memory, loaded once by all 128 epilogue
// threads (QKV: positions and staging offsets; SCATTER: token and slot of each sorted row).
// The barriers keep the previous item's readers and this item's readers apart.
template <int EPI>
__device__ __forceinline__ void stage_meta(const GemmArgs& a, const Item& it, const EpiSmem& sm) {
  if constexpr (EPI == EPI_QKV || EPI == EPI_SCATTER) {
    const int t = threadIdx.x - 64;
    named_bar_sync(1, 128);
    for (int r = t; r < it.rows; r += 128) {
      if constexpr (EPI == EPI_QKV) {
        sm.s_pos[r] = a.pos[it.out_row + r];
        sm.s_off[r] = a.kv_rowoff[it.out_row + r];
      } else {
        if (it.e < a.n_routed) {
          const int v = a.rowmap[static_cast<size_t>(it.e) * a.map_stride + it.grow + r];
          sm.s_pos[r] = v >> 3;
          sm.s_aux[r] = v & 7;
        } else {   // shared expert j: every token in order, slot top_k + j
          sm.s_pos[r] = it.grow + r;
          sm.s_aux[r] = kTopK + it.e - a.n_routed;
        }
      }
    }
    named_bar_sync(1, 128);
  }
}

template <int EPI, bool F8 = false>
__device__ __forceinline__ void epi_post(const GemmArgs& a, const Item& it, int row, int j0, float (&v)[16],
                                         const EpiPre& p, const EpiSmem& sm, int rope_buf) {
  if constexpr (EPI == EPI_F32 || EPI == EPI_RESID) {
    const int n = it.n_tile * 128 + row;
    if (EPI == EPI_F32 && F8 && n < a.N) {   // e4m3 GEMM: each weight row's scale
      const float sc = a.w_scale[0][n];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) v[jj] *= sc;
    }
    if (n < a.N) {
      float* base = a.out + static_cast<size_t>(it.out_row + j0) * a.ldo + n;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj)
        if (j0 + jj < it.rows) base[static_cast<size_t>(jj) * a.ldo] = (EPI == EPI_RESID) ? p.old[jj] + v[jj] : v[jj];
    }
  } else if constexpr (EPI == EPI_SCATTER) {
    const int n = it.n_tile * 128 + row;
    if constexpr (F8) {   // fp8 experts: the scale of output feature n's weight row
      const float sc = ((it.e < a.n_routed) ? a.w_scale[0] + static_cast<size_t>(it.e) * a.scale_rows
                                            : a.w_scale[1] + static_cast<size_t>(it.e - a.n_routed) * a.scale_rows)[n];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) v[jj] *= sc;
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
      if (j0 + jj < it.rows)
        a.y[(static_cast<size_t>(sm.s_pos[j0 + jj]) * kSlots + sm.s_aux[j0 + jj]) * kD + n] = v[jj];
  } else if constexpr (EPI == EPI_SWIGLU) {
    // Tile rows 0..63 are gate features, 64..127 the up features of the same 64 outputs.  The
    // gate thread of output p computes activation rows j0..j0+7 of it, the up thread rows
    // j0+8..j0+15: each passes the other the 8 values it lacks through one of two exchange
    // buffers (by chunk parity), so one barrier per chunk suffices: a buffer is written again
    // two chunks later, after a barrier that every thread reaches only once it has read this
    // chunk's values (between items, the barriers at the start of each item do the same).
    float* xchg = (rope_buf & 1) ? sm.xchg2 : sm.xchg;
    if constexpr (F8) {   // fp8 experts: this weight row's scale (tile rows 0..63 gate, 64..127 up)
      const int wr = (row < 64) ? it.n_tile * 64 + row : a.half_rows + it.n_tile * 64 + (row - 64);
      const float* ws = (it.e < a.n_routed) ? a.w_scale[0] + static_cast<size_t>(it.e) * a.scale_rows
                                            : a.w_scale[1] + static_cast<size_t>(it.e - a.n_routed) * a.scale_rows;
      const float sc = ws[wr];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) v[jj] *= sc;
    }
    const int up = row >> 6, pr = row & 63, mine = up * 8;   // mine: first of this thread's 8 rows
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) xchg[row * 17 + (8 - mine) + jj] = up ? v[jj] : v[8 + jj];
    named_bar_sync(1, 128);
    const float* other = xchg + (row ^ 64) * 17 + mine;
    const int f = it.n_tile * 64 + pr;
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const int r = j0 + mine + jj;
      const float o = other[jj];
      const float own = up ? v[8 + jj] : v[jj];
      const float g = up ? o : own;
      const float u = up ? own : o;
      if (r < it.rows) {
        const size_t at = static_cast<size_t>(it.out_row + r) * a.ld_act + f;
        if constexpr (F8) a.act8[at] = __nv_cvt_float_to_fp8(silu_f(g) * u, __NV_SATFINITE, __NV_E4M3);
        else a.act[at] = __float2bfloat16(silu_f(g) * u);
      }
    }
  } else if constexpr (EPI == EPI_QKV) {
    const int which = it.n_tile / kH;   // 0 q, 1 k, 2 v
    const int head = it.n_tile % kH;
    if (which < 2) {
      float* xchg = sm.xchg;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) xchg[row * 17 + jj] = v[jj];
      named_bar_sync(1, 128);
      float partner[16];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) partner[jj] = xchg[(row ^ 64) * 17 + jj];
      named_bar_sync(1, 128);
      const float2* cs = sm.rope + rope_buf * 16 * 64 + (row & 63);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const float2 f = cs[jj * 64];
        v[jj] = (row < 64) ? rope_lo(v[jj], partner[jj], f) : rope_hi(v[jj], partner[jj], f);
      }
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int r = j0 + jj;
      if (r >= it.rows) continue;
      const int m = it.out_row + r;
      if (which == 0) {
        a.q_out[static_cast<size_t>(m) * (kH * kHD) + head * kHD + row] = __float2bfloat16(v[jj]);
      } else {
        const long long off = sm.s_off[r];
        if (off >= 0) a.kv_base[off + (which == 2 ? a.v_off : 0) + head * a.head_stride + row] = __float2bfloat16(v[jj]);
      }
    }
  } else if constexpr (EPI == EPI_ARGMAX) {
    // per activation row: max over the tile's 128 logits (lower id on ties), through a
    // transpose in shared memory: 8 groups of 16 tile rows per column, then the 8 groups
    const int n = it.n_tile * 128 + row;
    float* xchg = sm.xchg;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) xchg[row * 17 + jj] = (n < a.N) ? v[jj] : -INFINITY;
    named_bar_sync(1, 128);
    const int t = threadIdx.x - 64, j = t & 15, grp = t >> 4;
    {
      float bv = xchg[(grp * 16) * 17 + j];
      int bi = grp * 16;
#pragma unroll
      for (int rr = 1; rr < 16; ++rr) {
        const float x = xchg[(grp * 16 + rr) * 17 + j];
        if (x > bv) {
          bv = x;
          bi = grp * 16 + rr;
        }
      }
      sm.am_val[grp * 16 + j] = bv;
      sm.am_idx[grp * 16 + j] = bi;
    }
    named_bar_sync(1, 128);
    if (t < 16 && j0 + t < it.rows) {
      float bv = sm.am_val[t];
      int bi = sm.am_idx[t];
#pragma unroll
      for (int g2 = 1; g2 < 8; ++g2) {
        const float x = sm.am_val[g2 * 16 + t];
        if (x > bv) {
          bv = x;
          bi = sm.am_idx[g2 * 16 + t];
        }
      }
      atomicMax(a.am_key + it.out_row + j0 + t, argmax_key(bv, it.n_tile * 128 + bi));
    }
    named_bar_sync(1, 128);
  }
}


// SwiGLU of two adjacent 16-column chunks (activation rows j0..j0+31) with one exchange: the
// gate thread of output p computes rows j0..j0+15 of it, the up thread rows j0+16..j0+31; each
// passes the other its 16 values of the other half through exchange buffer `buf` (alternating,
// as in epi_post<EPI_SWIGLU>).  The same arithmetic per element as epi_post<EPI_SWIGLU>.
template <bool F8>
__device__ __forceinline__ void epi_swiglu32(const GemmArgs& a, const Item& it, int row, int j0, float (&v)[16],
                                             float (&w)[16], const EpiSmem& sm, int buf) {
  float* xchg = (buf & 1) ? sm.xchg2 : sm.xchg;
  if constexpr (F8) {
    const int wr = (row < 64) ? it.n_tile * 64 + row : a.half_rows + it.n_tile * 64 + (row - 64);
    const float* ws = (it.e < a.n_routed) ? a.w_scale[0] + static_cast<size_t>(it.e) * a.scale_rows
                                          : a.w_scale[1] + static_cast<size_t>(it.e - a.n_routed) * a.scale_rows;
    const float sc = ws[wr];
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      v[jj] *= sc;
      w[jj] *= sc;
    }
  }
  const int up = row >> 6, pr = row & 63;
#pragma unroll
  for (int jj = 0; jj < 16; ++jj) xchg[row * 17 + jj] = up ? v[jj] : w[jj];
  named_bar_sync(1, 128);
  const float* other = xchg + (row ^ 64) * 17;
  const int f = it.n_tile * 64 + pr, r0 = j0 + up * 16;
#pragma unroll
  for (int jj = 0; jj < 16; ++jj) {
    const int r = r0 + jj;
    const float o = other[jj];
    const float own = up ? w[jj] : v[jj];
    const float g = up ? o : own;
    const float u = up ? own : o;
    if (r < it.rows) {
      const size_t at = static_cast<size_t>(it.out_row + r) * a.ld_act + f;
      if constexpr (F8) a.act8[at] = __nv_cvt_float_to_fp8(silu_f(g) * u, __NV_SATFINITE, __NV_E4M3);
      else a.act[at] = __float2bfloat16(silu_f(g) * u);
    }
  }
}

// Draft-head objective (EPI_LOSS): the operands are swapped for this launch -- A is the packed
// activation matrix (tile row = activation row, one per epilogue thread), B a tile of 256
// vocabulary rows of W_lm (the accumulator columns) -- so each thread folds its own row's logits
// with an online softmax, chunk by chunk: running max m and sum z of exp(x - m), and for the KL
// term the verifier logits q of its row group (lane (lane & ~(G-1)): row 0 of the group holds
// b_{p+1}) with running max mq and a = sum exp(q - mq) (q - x).  No shared memory, no barrier.
struct LossState {
  float m, z, mq, a;
};
__device__ __forceinline__ void loss_chunk(const GemmArgs& a, const Item& it, int j0, const float (&v)[16], LossState& st) {
  const int lane = threadIdx.x & 31;
  const int src = lane & ~(a.loss_G - 1);
  const int nv = min(16, it.rows - j0);   // valid vocabulary columns of this chunk
  float q[16];
#pragma unroll
  for (int jj = 0; jj < 16; ++jj) q[jj] = __shfl_sync(0xffffffffu, v[jj], src);
  if (nv <= 0) return;
  float xm = -INFINITY, qm = -INFINITY;
#pragma unroll
  for (int jj = 0; jj < 16; ++jj)
    if (jj < nv) {
      xm = fmaxf(xm, v[jj]);
      qm = fmaxf(qm, q[jj]);
    }
  const float m1 = fmaxf(st.m, xm), q1 = fmaxf(st.mq, qm);
  float z = (st.m == -INFINITY) ? 0.f : st.z * __expf(st.m - m1);
  float acc = (st.mq == -INFINITY) ? 0.f : st.a * __expf(st.mq - q1);
#pragma unroll
  for (int jj = 0; jj < 16; ++jj)
    if (jj < nv) {
      z += __expf(v[jj] - m1);
      acc += __expf(q[jj] - q1) * (q[jj] - v[jj]);
    }
  st.m = m1;
  st.z = z;
  st.mq = q1;
  st.a = acc;
}

// Cluster split-K reduction by whole chunks (the epilogues without a quad form below; the dense
// launches use the quad form), run by the 128 epilogue threads of every CTA of the cluster after
// the first cluster barrier: CTA `rank` takes chunks rank, rank + S, ..., adds the S partial
// tiles of each (read from the cluster's shared memory) in split order -- the same sums as the
// other schedules -- and runs the epilogue on them.  The epilogue operands of its first chunk
// (`first`, and its RoPE factors in rope buffer 0) were fetched while the MMAs ran.  The CTA
// arrives on the cluster barrier as soon as its last read of another CTA's shared memory is
// done; the caller waits on it before the CTA exits.
template <int EPI>
__device__ __forceinline__ void cluster_reduce(const GemmArgs& a, const EpiSmem& esm, uint32_t part_saddr, int row,
                                               const EpiPre& first) {
  Item it;
  get_item<EPI>(a, a, blockIdx.x, it, nullptr);
  const int S = a.cluster;
  const int rank = static_cast<int>(cluster_ctarank());
  const int nchunks = (it.rows + 15) >> 4;
  const bool rope = (EPI == EPI_QKV) && it.n_tile < 2 * kH;
  if (rank >= nchunks) cluster_arrive();
  int k = 0;
  for (int c = rank; c < nchunks; c += S, ++k) {
    EpiPre cur = first;
    if (k > 0) {
      if (rope) {
        RopeRegs rr;
        rope_load(a, it, c * 16, esm, rr);
        rope_store(esm, k & 1, rr);
        named_bar_sync(1, 128);
      }
      epi_pre<EPI>(a, it, row, c * 16, esm, cur);
    }
    float v[16];
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      float4 p[kMaxSplit][2];
#pragma unroll
      for (int sp = 0; sp < kMaxSplit; ++sp)
        if (sp < S)
#pragma unroll
          for (int q2 = 0; q2 < 2; ++q2)
            p[sp][q2] = ld_dsmem_f4(part_saddr + ((c * 4 + 2 * hf + q2) * 128 + row) * 16, sp);
#pragma unroll
      for (int q2 = 0; q2 < 2; ++q2) {
        float4 t = p[0][q2];
#pragma unroll
        for (int sp = 1; sp < kMaxSplit; ++sp)
          if (sp < S) {
            t.x += p[sp][q2].x;
            t.y += p[sp][q2].y;
            t.z += p[sp][q2].z;
            t.w += p[sp][q2].w;
          }
        const int q4 = 2 * hf + q2;
        v[4 * q4] = t.x;
        v[4 * q4 + 1] = t.y;
        v[4 * q4 + 2] = t.z;
        v[4 * q4 + 3] = t.w;
      }
    }
    if (c + S >= nchunks) cluster_arrive();   // no more reads of the other CTAs' partial tiles
    epi_post<EPI>(a, it, row, c * 16, v, cur, esm, k & 1);
  }
}

// Cluster split-K reduction in quad units, for the epilogues whose row pairs need no more than
// one warp (F32, RESID, QKV, SWIGLU).  A unit is 4 activation rows (one float4 column of the
// partial tiles) x 32 tile rows: row group g of the tile is rows 16g..16g+15 (lanes 0..15) and
// their rotate-half / gate-up partners 64+16g..64+16g+15 (lanes 16..31), so a pair meets by one
// shuffle.  Units are dealt over the cluster's CTAs first, then over their 4 epilogue warps:
// a tile of 4 activation rows is reduced by 4 warps on 4 SMs, each reading the S partials of
// its unit at once (one round trip through distributed shared memory), instead of by all 128
// threads of one CTA in two.  The sums and the epilogue arithmetic are those of cluster_reduce.
template <int EPI>
__device__ __forceinline__ constexpr bool quad_epi() {
  return EPI == EPI_F32 || EPI == EPI_RESID || EPI == EPI_QKV || EPI == EPI_SWIGLU;
}
__device__ __forceinline__ int quad_row(int g, int lane) { return (lane < 16) ? 16 * g + lane : 48 + 16 * g + lane; }
// the k-th unit of epilogue warp `slot` of cluster rank `rank`: units go round the cluster's
// CTAs first, then their warps
__device__ __forceinline__ int quad_unit(int k, int slot, int rank, int S) { return (k * 4 + slot) * S + rank; }

// Epilogue operands of one unit, read before the reduction: the old residuals (RESID) or the
// cos/sin of the 4 rows' positions at this lane's feature (QKV q and k tiles).
struct QuadOps {
  float old[4];
  float2 rope[4];
};
struct QuadPre {
  QuadOps u[2];   // the first two units of the warp
};

template <int EPI>
__device__ __forceinline__ void quad_ops(const GemmArgs& a, const Item& it, const EpiSmem& sm, int u, int lane,
                                         QuadOps& o) {
  const int r = quad_row(u & 3, lane), j0 = 4 * (u >> 2);
  if constexpr (EPI == EPI_RESID) {
    const int n = it.n_tile * 128 + r;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj)
      o.old[jj] = (n < a.N && j0 + jj < it.rows) ? a.out[static_cast<size_t>(it.out_row + j0 + jj) * a.ldo + n] : 0.f;
  } else if constexpr (EPI == EPI_QKV) {
    if (it.n_tile < 2 * kH) {
      bool bad = false;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        int q = (j0 + jj < it.rows) ? sm.s_pos[j0 + jj] : 0;
        if (q < 0 || q >= a.max_pos) {
          bad = true;
          q = 0;
        }
        o.rope[jj] = a.rope[static_cast<size_t>(q) * (kHD / 2) + (r & 63)];
      }
      if (bad) atomicOr(a.err, ERR_POSITION);
    }
  }
}

template <int EPI>
__device__ __forceinline__ void quad_post(const GemmArgs& a, const Item& it, const EpiSmem& sm, int u, int lane,
                                          float (&v)[4], const QuadOps& o) {
  const int r = quad_row(u & 3, lane), j0 = 4 * (u >> 2);
  if constexpr (EPI == EPI_F32 || EPI == EPI_RESID) {
    const int n = it.n_tile * 128 + r;
    if (n < a.N) {
#pragma unroll
      for (int jj = 0; jj < 4; ++jj)
        if (j0 + jj < it.rows)
          a.out[static_cast<size_t>(it.out_row + j0 + jj) * a.ldo + n] = (EPI == EPI_RESID) ? o.old[jj] + v[jj] : v[jj];
    }
  } else if constexpr (EPI == EPI_QKV) {
    const int which = it.n_tile / kH;   // 0 q, 1 k, 2 v
    const int head = it.n_tile % kH;
    if (which < 2) {
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const float partner = __shfl_xor_sync(0xffffffffu, v[jj], 16);
        v[jj] = (r < 64) ? rope_lo(v[jj], partner, o.rope[jj]) : rope_hi(v[jj], partner, o.rope[jj]);
      }
    }
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int j = j0 + jj;
      if (j >= it.rows) continue;
      const int m = it.out_row + j;
      if (which == 0) {
        a.q_out[static_cast<size_t>(m) * (kH * kHD) + head * kHD + r] = __float2bfloat16(v[jj]);
      } else {
        const long long off = sm.s_off[j];
        if (off >= 0) a.kv_base[off + (which == 2 ? a.v_off : 0) + head * a.head_stride + r] = __float2bfloat16(v[jj]);
      }
    }
  } else if constexpr (EPI == EPI_SWIGLU) {
    // lanes 0..15 hold gate features, lanes 16..31 the up features of the same outputs; the
    // gate lane computes rows 0 and 1 of the unit, the up lane rows 2 and 3
    const int up = lane >> 4;
    float other[4];
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) other[jj] = __shfl_xor_sync(0xffffffffu, v[jj], 16);
    const int f = it.n_tile * 64 + (r & 63);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int jj = 2 * up + h, j = j0 + jj;
      const float g = up ? other[jj] : v[jj];
      const float uu = up ? v[jj] : other[jj];
      if (j < it.rows) a.act[static_cast<size_t>(it.out_row + j) * a.ld_act + f] = __float2bfloat16(silu_f(g) * uu);
    }
  }
}

// Epilogue warp `slot` (0..3) of cluster rank `rank` takes units (k * 4 + slot) * S + rank,
// k = 0, 1, ..., two at a time with every split's loads of both in flight.
template <int EPI>
__device__ __forceinline__ void quad_prefetch(const GemmArgs& a, const Item& it, const EpiSmem& sm, int slot, int lane,
                                              QuadPre& qp) {
  const int S = a.cluster, rank = static_cast<int>(cluster_ctarank());
  const int U = 4 * ((it.rows + 3) >> 2);
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int u = quad_unit(k, slot, rank, S);
    if (u < U) quad_ops<EPI>(a, it, sm, u, lane, qp.u[k]);
  }
}

template <int EPI>
__device__ __forceinline__ void cluster_reduce_quads(const GemmArgs& a, const EpiSmem& sm, uint32_t part_saddr,
                                                     int slot, int lane, const QuadPre& qp) {
  Item it;
  get_item<EPI>(a, a, blockIdx.x, it, nullptr);
  const int S = a.cluster, rank = static_cast<int>(cluster_ctarank());
  const int U = 4 * ((it.rows + 3) >> 2);
  int n_mine = 0;
  while (quad_unit(n_mine, slot, rank, S) < U) ++n_mine;
  if (n_mine == 0) cluster_arrive();
  for (int k0 = 0; k0 < n_mine; k0 += 2) {
    float4 p[2][kMaxSplit];
    QuadOps o[2];
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      if (k0 + kk >= n_mine) break;
      const int u = quad_unit(k0 + kk, slot, rank, S);
      const int r = quad_row(u & 3, lane);
      const uint32_t at = part_saddr + static_cast<uint32_t>(((u >> 2) * 128 + r) * 16);
#pragma unroll
      for (int sp = 0; sp < kMaxSplit; ++sp)
        if (sp < S) p[kk][sp] = ld_dsmem_f4(at, sp);
      if (k0 == 0) o[kk] = qp.u[kk];
      else quad_ops<EPI>(a, it, sm, u, lane, o[kk]);
    }
    float v[2][4];
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      if (k0 + kk >= n_mine) break;
      float4 t = p[kk][0];
#pragma unroll
      for (int sp = 1; sp < kMaxSplit; ++sp)
        if (sp < S) {
          t.x += p[kk][sp].x;
          t.y += p[kk][sp].y;
          t.z += p[kk][sp].z;
          t.w += p[kk][sp].w;
        }
      v[kk][0] = t.x;
      v[kk][1] = t.y;
      v[kk][2] = t.z;
      v[kk][3] = t.w;
    }
    if (k0 + 2 >= n_mine) cluster_arrive();   // no more reads of the other CTAs' partial tiles
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      if (k0 + kk >= n_mine) break;
      quad_post<EPI>(a, it, sm, quad_unit(k0 + kk, slot, rank, S), lane, v[kk], o[kk]);
    }
  }
}

// ------------------------------------------------------------------ kernel
template <int NMAX, int EPI, int ST, bool F8 = false>
__global__ void __launch_bounds__(192, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a,
                                                         const __grid_constant__ GemmArgs a2) {
  using C = KCfg<NMAX, EPI, ST>;
  constexpr bool DUAL = (EPI == EPI_MOE && NMAX == 128);
  extern __shared__ uint8_t smem_raw[];
  const uint32_t base_u32 = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((base_u32 + 1023u) & ~1023u) - base_u32);
  uint8_t* smA = smem;
  uint8_t* smB = smA + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smB + C::STAGES * C::B_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::STAGES;
  uint64_t* tfull = bars + 2 * C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* fin = tempty + 2;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(fin + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  int* s_vote = const_cast<int*>(s_abort) + 1;   // [4]
  int* s_last = s_vote + 4;
  EpiSmem esm;
  EpiPre first_pre;   // cluster split-K: the epilogue operands of the first chunk this CTA reduces
  QuadPre quad_pre;   // cluster split-K in quad units: those of the warp's first two units
  esm.xchg = reinterpret_cast<float*>(smem + C::STAGES * (C::A_BYTES + C::B_BYTES) + 256);
  esm.am_val = esm.xchg + C::XCHG_FLOATS;
  esm.am_idx = reinterpret_cast<int*>(esm.am_val + 128);
  esm.s_off = reinterpret_cast<long long*>(esm.am_idx + 128);
  esm.s_pos = reinterpret_cast<int*>(esm.s_off + 256);
  esm.s_aux = esm.s_pos + 256;
  esm.rope = reinterpret_cast<float2*>(esm.s_aux + 256);
  esm.xchg2 = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(esm.rope) + 1024);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  pdl_trigger(kTrGemm + EPI);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&tfull[s], 1);
      mbar_init(&tempty[s], 4);
    }
    mbar_init(fin, 1);
    *s_abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&a.a_map[0]);
    tma_prefetch_desc(&a.a_map[1]);
  }
  // accumulator buffers: two of NMAX columns, or with in-CTA splits one (split_k > 4) or two
  // groups of split_k x 64 columns
  const uint32_t tmem_cols = a.seq_split ? 512u : static_cast<uint32_t>(C::TMEM_COLS);
  const int nbuf = (a.seq_split && a.split_k > 4) ? 1 : 2;
  const uint32_t acc_stride =
      a.seq_split ? static_cast<uint32_t>(a.split_k) * 64u : static_cast<uint32_t>((DUAL ? 2 : 1) * NMAX);
  if (warp == 1) {
    tmem_alloc(s_tmem, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;

  // Dense launches know their items from the arguments: the producer streams its first weight
  // tiles (never written by earlier kernels) before it waits for the previous kernel; every
  // other thread waits before its first global access.  The producer's warp skips this wait
  // as a whole: its other lanes read nothing an earlier kernel writes, and a blocking wait on
  // them would hold the producer lane too, so the weights would only be requested after it.
  const bool dense = (a.grp_cnt == nullptr);
  if (!(dense && warp == 0)) pdl_wait();
  // grouped launches: the per-expert tables (in the RoPE buffer, which only QKV uses)
  int* grp = reinterpret_cast<int*>(esm.rope);
  int n_items = a.n_items;
  if (!dense) {
    if (threadIdx.x < 32) {   // three experts per lane, prefix sums by warp scan
      int c[3], ni[3], nd[3], sc = 0, si = 0, sd = 0, touched = 0;
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        const int p = 3 * static_cast<int>(threadIdx.x) + k, e = grp_expert(p);
        c[k] = (p < kE + kShared) ? ((e < a.n_routed) ? a.grp_cnt[e] : a.grp_T) : 0;
        const int mt = (c[k] + a.grp_rows - 1) / a.grp_rows;
        ni[k] = mt * a.grp_tiles;
        nd[k] = (EPI == EPI_MOE) ? mt * a2.grp_tiles : 0;
        sc += c[k];
        si += ni[k];
        sd += nd[k];
        touched += (c[k] > 0) ? 1 : 0;
      }
      int ic = sc, ii = si, id = sd;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int yc = __shfl_up_sync(0xffffffffu, ic, o), yi = __shfl_up_sync(0xffffffffu, ii, o);
        const int yd = __shfl_up_sync(0xffffffffu, id, o);
        if (static_cast<int>(threadIdx.x) >= o) {
          ic += yc;
          ii += yi;
          id += yd;
        }
      }
      int ri = ii - si, rd = id - sd;
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        const int p = 3 * static_cast<int>(threadIdx.x) + k;
        if (p < kE + kShared) {
          grp[kGrpCnt + p] = c[k];
          grp[kGrpItem + p] = ri;
          grp[kGrpDn + p] = rd;
        }
        ri += ni[k];
        rd += nd[k];
      }
      if (threadIdx.x == 31) {
        grp[kGrpItem + kE + kShared] = ii;
        grp[kGrpDn + kE + kShared] = id;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) touched += __shfl_xor_sync(0xffffffffu, touched, o);
      if (a.expert_ctr != nullptr && blockIdx.x == 0 && threadIdx.x == 31) {
        atomicAdd(&a.expert_ctr[0], static_cast<unsigned long long>(touched));
        atomicAdd(&a.expert_ctr[1], static_cast<unsigned long long>(ic));
      }
    }
    __syncthreads();
    n_items = grp[kGrpItem + kE + kShared] + ((EPI == EPI_MOE) ? grp[kGrpDn + kE + kShared] : 0);
  }

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t pol_w = a.a_keep ? l2_policy_evict_last() : l2_policy_evict_first();
      // (operands swapped for the objective: the streamed W_lm tiles are the B side)
      const uint64_t pol_x = (EPI == EPI_LOSS) ? l2_policy_evict_first() : l2_policy_evict_last();
      uint32_t g = 0;   // loads issued
      bool failed = false;
      bool waited = !dense;
      for (int i = blockIdx.x; i < n_items && !failed; i += gridDim.x) {
        Item it;
        get_item<EPI>(a, a2, i, it, grp);
        const GemmArgs& P = it.phase ? a2 : a;   // the item's operands (EPI_MOE down items: a2)
        constexpr int kw = F8 ? 128 : 64;         // elements of a 128-byte k-chunk
        const int kc_total = P.K / kw;
        const int src = (!dense && it.e >= a.n_routed) ? 1 : 0;
        const int el = it.e - (src ? a.n_routed : 0);
        const CUtensorMap* amap = &P.a_map[src];
        const CUtensorMap* bmap = &P.b_map[src][it.box_log];
        const uint32_t bytes = C::A_BYTES + (16u << it.box_log) * 128u;
        const int kc0 = a.seq_split ? 0 : it.split * kc_total / a.split_k;
        const int kc1 = a.seq_split ? kc_total : (it.split + 1) * kc_total / a.split_k;
        auto load_a = [&](int st, int kc) {
          uint8_t* sa = smA + st * C::A_BYTES;
          const int k = kc * kw;
          if constexpr (DUAL) {
            // two 128-row weight tiles: gate rows 128 t.. and up rows half_rows + 128 t.. (64-row
            // boxes of the paired map), or down rows 256 t.. and 256 t + 128.. (128-row boxes)
            if (P.paired) {
              const int r0 = it.n_tile * 128;
              tma_load_3d(sa, amap, &full[st], k, r0, el, pol_w);
              tma_load_3d(sa + 8192, amap, &full[st], k, r0 + 64, el, pol_w);
              tma_load_3d(sa + 16384, amap, &full[st], k, P.half_rows + r0, el, pol_w);
              tma_load_3d(sa + 16384 + 8192, amap, &full[st], k, P.half_rows + r0 + 64, el, pol_w);
            } else {
              const int r0 = it.n_tile * 256;
              tma_load_3d(sa, amap, &full[st], k, r0, el, pol_w);
              tma_load_3d(sa + 16384, amap, &full[st], k, r0 + 128, el, pol_w);
            }
            return;
          }
          if (P.paired) {
            const int r0 = it.n_tile * 64;
            if (P.a3d) {
              tma_load_3d(sa, amap, &full[st], k, r0, el, pol_w);
              tma_load_3d(sa + 8192, amap, &full[st], k, P.half_rows + r0, el, pol_w);
            } else {
              tma_load_2d(sa, amap, &full[st], k, r0, pol_w);
              tma_load_2d(sa + 8192, amap, &full[st], k, P.half_rows + r0, pol_w);
            }
          } else {
            const int r0 = it.n_tile * 128;
            if (P.a3d) tma_load_3d(sa, amap, &full[st], k, r0, el, pol_w);
            else tma_load_2d(sa, amap, &full[st], k, r0, pol_w);
          }
        };
        int kc = kc0;
        if (EPI == EPI_MOE && it.phase == 1) {
          // a down item reads the SwiGLU rows of its (expert, row tile): wait until all gate/up
          // tiles of them are stored (they come earlier in the item order, so they always end)
          const int* d = a.dep + it.e * a.dep_stride + it.grow / a.grp_rows;
          if (ld_acquire_gpu(d) < a.grp_tiles) {
            const uint64_t t0 = globaltimer();
            while (ld_acquire_gpu(d) < a.grp_tiles) {
              if (*s_abort || globaltimer() - t0 > kWaitLimitNs) {
                failed = true;
                break;
              }
              __nanosleep(64);
            }
            if (failed) break;
          }
          fence_proxy_async_global();   // the rows were stored by other CTAs' generic stores
        }
        if (!waited) {
          // first item: the stages are all free (g == 0); weights first, activations after the wait
          const int npre = min(C::STAGES, kc1 - kc0);
          for (int q = 0; q < npre; ++q) {
            mbar_arrive_expect_tx(&full[q], bytes);
            load_a(q, kc0 + q);
          }
          pdl_wait();
          waited = true;
          for (int q = 0; q < npre; ++q)
            tma_load_2d(smB + q * C::B_BYTES, bmap, &full[q], (kc0 + q) * kw, it.b_row, pol_x);
          g = npre;
          kc = kc0 + npre;
        }
        for (; kc < kc1; ++kc, ++g) {
          const int st = g % C::STAGES;
          const uint32_t ph = (g / C::STAGES) & 1u;
          if (!mbar_wait(&empty[st], ph ^ 1u, s_abort)) {
            failed = true;
            break;
          }
          mbar_arrive_expect_tx(&full[st], bytes);
          load_a(st, kc);
          tma_load_2d(smB + st * C::B_BYTES, bmap, &full[st], kc * kw, it.b_row, pol_x);
        }
      }
      if (!waited) pdl_wait();
      if (failed) {
        *s_abort = 1;
        atomicOr(a.err, ERR_WAIT_TIMEOUT);
        // let the copies still in flight land before the CTA's shared memory is released
        volatile int never = 0;
        const uint32_t back = g < C::STAGES ? g : C::STAGES;
        for (uint32_t b = 1; b <= back; ++b) {
          const uint32_t gg = g - b;
          mbar_wait(&full[gg % C::STAGES], (gg / C::STAGES) & 1u, &never, 100000000ull);
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t g = 0;
      int local = 0;
      bool failed = false;
      for (int i = blockIdx.x; i < n_items && !failed; i += gridDim.x, ++local) {
        Item it;
        get_item<EPI>(a, a2, i, it, grp);
        const int kc_total = (it.phase ? a2.K : a.K) / (F8 ? 128 : 64);
        const int acc = local % nbuf;
        const uint32_t acc_ph = static_cast<uint32_t>(local / nbuf) & 1u;
        if (!mbar_wait(&tempty[acc], acc_ph ^ 1u, s_abort)) {
          failed = true;
          break;
        }
        tc_fence_after();
        const uint32_t idesc = F8 ? idesc_e4m3(128, 16 << it.box_log) : idesc_bf16(128, 16 << it.box_log);
        const int kc0 = a.seq_split ? 0 : it.split * kc_total / a.split_k;
        const int kc1 = a.seq_split ? kc_total : (it.split + 1) * kc_total / a.split_k;
        // with in-CTA splits, split sp accumulates k-chunks [sp*kc/S, (sp+1)*kc/S) into its own
        // 64 columns, starting from zero, exactly as a separate CTA would
        int sp = 0, sp_begin = kc0, sp_end = a.seq_split ? kc_total / a.split_k : kc1;
        for (int kc = kc0; kc < kc1; ++kc, ++g) {
          if (kc == sp_end) {
            ++sp;
            sp_begin = kc;
            sp_end = (sp + 1) * kc_total / a.split_k;
          }
          const uint32_t d_tmem = tmem_base + acc * acc_stride + sp * 64;
          const int st = g % C::STAGES;
          const uint32_t ph = (g / C::STAGES) & 1u;
          if (!mbar_wait(&full[st], ph, s_abort)) {
            failed = true;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sw128_kmajor_desc(smem_u32(smA + st * C::A_BYTES));
          const uint64_t bd = sw128_kmajor_desc(smem_u32(smB + st * C::B_BYTES));
          // 4 MMAs per 128-byte k-chunk (K=16 bf16 or K=32 e4m3 each): +32 B in the swizzled row
#pragma unroll
          for (int s = 0; s < 4; ++s) {
            if constexpr (F8) tc_mma_e4m3(d_tmem, ad + 2 * s, bd + 2 * s, idesc, (kc > sp_begin || s > 0) ? 1u : 0u);
            else tc_mma_bf16(d_tmem, ad + 2 * s, bd + 2 * s, idesc, (kc > sp_begin || s > 0) ? 1u : 0u);
          }
          if constexpr (DUAL) {
            // the second weight tile against the same activation tile, into the second accumulator
            const uint64_t ad1 = sw128_kmajor_desc(smem_u32(smA + st * C::A_BYTES + 16384));
#pragma unroll
            for (int s = 0; s < 4; ++s) {
              if constexpr (F8)
                tc_mma_e4m3(d_tmem + NMAX, ad1 + 2 * s, bd + 2 * s, idesc, (kc > sp_begin || s > 0) ? 1u : 0u);
              else tc_mma_bf16(d_tmem + NMAX, ad1 + 2 * s, bd + 2 * s, idesc, (kc > sp_begin || s > 0) ? 1u : 0u);
            }
          }
          tc_commit(&empty[st]);
        }
        if (failed) break;
        tc_commit(&tfull[acc]);
      }
      if (failed) {
        *s_abort = 1;
        atomicOr(a.err, ERR_WAIT_TIMEOUT);
        if (g > 0) {
          // every MMA issued so far has completed once `fin` flips
          tc_commit(fin);
          volatile int never = 0;
          mbar_wait(fin, 0, &never, 100000000ull);
        }
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (warps 2..5)
    const int q = warp & 3;                // TMEM lane quadrant of this warp
    const int row = q * 32 + lane;         // tile row = weight row within the tile
    const int ew = warp - 2;
    int local = 0;
    for (int i = blockIdx.x; i < n_items; i += gridDim.x, ++local) {
      Item it;
      get_item<EPI>(a, a2, i, it, grp);
      const int acc = local % nbuf;
      const uint32_t acc_ph = static_cast<uint32_t>(local / nbuf) & 1u;
      // the item's metadata, RoPE factors and first old residuals are fetched while its MMAs
      // run (in a cluster, those of the first chunk this CTA reduces)
      if constexpr (EPI == EPI_MOE) {
        if (it.phase) stage_meta<EPI_SCATTER>(a2, it, esm);
      } else {
        stage_meta<EPI>(a, it, esm);
      }
      const bool rope = (EPI == EPI_QKV) && it.n_tile < 2 * kH;
      RopeRegs rr;
      EpiPre cur, nxt;
      if (quad_epi<EPI>() && a.cluster > 1) {
        quad_prefetch<EPI>(a, it, esm, ew, lane, quad_pre);
      } else {
        const int c_first = (a.cluster > 1) ? static_cast<int>(cluster_ctarank()) : 0;
        if (rope) {
          rope_load(a, it, c_first * 16, esm, rr);
          rope_store(esm, 0, rr);
          named_bar_sync(1, 128);
        }
        epi_pre<EPI>(a, it, row, c_first * 16, esm, cur);
        first_pre = cur;
      }
      bool ok = mbar_wait(&tfull[acc], acc_ph, s_abort);
      ok = __all_sync(0xffffffffu, ok);
      if (lane == 0) s_vote[ew] = ok ? 1 : 0;
      named_bar_sync(1, 128);
      const bool all_ok = s_vote[0] && s_vote[1] && s_vote[2] && s_vote[3];
      named_bar_sync(1, 128);
      if (!all_ok) {
        *s_abort = 1;
        atomicOr(a.err, ERR_WAIT_TIMEOUT);
        break;
      }
      tc_fence_after();
      const uint32_t tb = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * acc_stride;
      const int nchunks = (it.rows + 15) >> 4;
      float v[16];
      LossState ls = {-INFINITY, 0.f, -INFINITY, 0.f};
      if constexpr (DUAL) {
        // 128-row items: accumulator 0 at tb, accumulator 1 at tb + NMAX (same lanes, same rows)
        const bool routed = it.e < a.n_routed;
        if (it.phase == 0) {
          // gate feature f in accumulator 0, up feature f in accumulator 1: SwiGLU in registers
          const int f = it.n_tile * 128 + row;
          float sg = 1.f, su = 1.f;
          if constexpr (F8) {
            const float* ws = routed ? a.w_scale[0] + static_cast<size_t>(it.e) * a.scale_rows
                                     : a.w_scale[1] + static_cast<size_t>(it.e - a.n_routed) * a.scale_rows;
            sg = ws[f];
            su = ws[a.half_rows + f];
          }
          for (int c = 0; c < nchunks; ++c) {
            float g[16], u[16];
            tc_ld16x2(tb + c * 16, tb + NMAX + c * 16, g, u);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) {
              const int r = c * 16 + jj;
              if (r < it.rows) {
                float gv = g[jj], uv = u[jj];
                if constexpr (F8) {
                  gv *= sg;
                  uv *= su;
                }
                const size_t at = static_cast<size_t>(it.out_row + r) * a.ld_act + f;
                if constexpr (F8) a.act8[at] = __nv_cvt_float_to_fp8(silu_f(gv) * uv, __NV_SATFINITE, __NV_E4M3);
                else a.act[at] = __float2bfloat16(silu_f(gv) * uv);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[acc]);
          fence_proxy_async_global();   // the SwiGLU rows are stored: count the tile for (e, m)
          __threadfence();
          named_bar_sync(1, 128);
          if (threadIdx.x == 64) atomicAdd(a.dep + it.e * a.dep_stride + it.grow / a.grp_rows, 1);
        } else {
          // output features n0 (accumulator 0) and n0 + 128 (accumulator 1), scattered to
          // (token, slot)
          const int n0 = it.n_tile * 256 + row;
          float s0 = 1.f, s1 = 1.f;
          if constexpr (F8) {
            const float* ws = routed ? a2.w_scale[0] + static_cast<size_t>(it.e) * a2.scale_rows
                                     : a2.w_scale[1] + static_cast<size_t>(it.e - a2.n_routed) * a2.scale_rows;
            s0 = ws[n0];
            s1 = ws[n0 + 128];
          }
          for (int c = 0; c < nchunks; ++c) {
            float v0[16], v1[16];
            tc_ld16x2(tb + c * 16, tb + NMAX + c * 16, v0, v1);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) {
              const int r = c * 16 + jj;
              if (r < it.rows) {
                float* dst = a2.y + (static_cast<size_t>(esm.s_pos[r]) * kSlots + esm.s_aux[r]) * kD + n0;
                if constexpr (F8) {
                  dst[0] = v0[jj] * s0;
                  dst[128] = v1[jj] * s1;
                } else {
                  dst[0] = v0[jj];
                  dst[128] = v1[jj];
                }
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[acc]);
        }
        continue;
      }
      if (EPI == EPI_MOE && it.phase == 0) {
        // gate/up items: two chunks per exchange
        for (int c = 0, x = 0; c < nchunks; c += 2, ++x) {
          if (c + 1 < nchunks) {
            float w[16];
            tc_ld16x2(tb + c * 16, tb + (c + 1) * 16, v, w);
            epi_swiglu32<F8>(a, it, row, c * 16, v, w, esm, x & 1);
          } else {
            tc_ld16(tb + c * 16, v);
            epi_post<EPI_SWIGLU, F8>(a, it, row, c * 16, v, cur, esm, x & 1);
          }
        }
        tc_fence_before();   // the accumulator is read: the next item's MMAs may use it
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        // this gate/up tile's SwiGLU rows are stored: count it for the down items of (e, m)
        fence_proxy_async_global();
        __threadfence();
        named_bar_sync(1, 128);
        if (threadIdx.x == 64) atomicAdd(a.dep + it.e * a.dep_stride + it.grow / a.grp_rows, 1);
      } else if (a.split_k == 1 || a.seq_split) {
        for (int c = 0; c < nchunks; ++c) {
          if (c + 1 < nchunks) {
            epi_pre<EPI>(a, it, row, (c + 1) * 16, esm, nxt);
            if (rope) rope_load(a, it, (c + 1) * 16, esm, rr);
          }
          tc_ld16(tb + c * 16, v);
          for (int sp = 1; sp < (a.seq_split ? a.split_k : 1); ++sp) {
            // in-CTA splits: partial sums added in split order, as the cross-CTA reduction does
            float w[16];
            tc_ld16(tb + sp * 64 + c * 16, w);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] += w[jj];
          }
          if constexpr (EPI == EPI_MOE) {
            epi_post<EPI_SCATTER, F8>(a2, it, row, c * 16, v, cur, esm, c & 1);   // down items
          } else if constexpr (EPI == EPI_LOSS) {
            loss_chunk(a, it, c * 16, v, ls);
          } else {
            epi_post<EPI, F8>(a, it, row, c * 16, v, cur, esm, c & 1);
          }
          cur = nxt;
          if (rope && c + 1 < nchunks) {
            rope_store(esm, (c + 1) & 1, rr);
            named_bar_sync(1, 128);
          }
        }
        if constexpr (EPI == EPI_LOSS) {
          // this activation row's statistics over the item's vocabulary tile
          const int arow = it.n_tile * 128 + row;
          if (arow < a.N)
            a.loss_part[static_cast<size_t>(it.out_row / 256) * a.ldo + arow] = make_float4(ls.m, ls.z, ls.a, ls.mq);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
      } else if (a.cluster > 1) {
        // cluster split-K: the partial tile goes to this CTA's shared memory (the pipeline
        // stages are free once the tile's MMAs have completed), laid out [chunk][quad][row];
        // the reduction follows the cluster barrier at the end of the kernel
        float4* part = reinterpret_cast<float4*>(smA);
        for (int c = 0; c < nchunks; ++c) {
          tc_ld16(tb + c * 16, v);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4)
            part[(c * 4 + q4) * 128 + row] = make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
      } else {
        // split-K: each split writes its fp32 partial tile thread-major (a thread's 16 values
        // of a chunk are 64 contiguous bytes); the last split of the tile to arrive (atomic
        // ticket, no wait) sums the partials in split order and runs the epilogue.
        const int box = 16 << it.box_log;
        const int tile = it.n_tile * a.m_tiles + it.out_row / box;
        const size_t tstride = static_cast<size_t>(box / 16) * 128 * 16;    // floats per split of a tile
        float* mine = a.sk_ws + (static_cast<size_t>(tile) * a.split_k + it.split) * tstride;
        for (int c = 0; c < nchunks; ++c) {
          tc_ld16(tb + c * 16, v);
          float4* dst = reinterpret_cast<float4*>(mine + (static_cast<size_t>(c) * 128 + row) * 16);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) dst[q4] = make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        __threadfence();
        named_bar_sync(1, 128);
        if (threadIdx.x == 64) {
          const int old = atomicAdd(&a.sk_tickets[tile], 1);
          *s_last = (old == a.split_k - 1) ? 1 : 0;
          if (old == a.split_k - 1) a.sk_tickets[tile] = 0;
        }
        named_bar_sync(1, 128);
        if (*s_last) {
          __threadfence();
          const float* base = a.sk_ws + static_cast<size_t>(tile) * a.split_k * tstride;
          for (int c = 0; c < nchunks; ++c) {
            if (c + 1 < nchunks) {
              epi_pre<EPI>(a, it, row, (c + 1) * 16, esm, nxt);
              if (rope) rope_load(a, it, (c + 1) * 16, esm, rr);
            }
            // two halves of the 16 values, each with all splits' loads in flight
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
              float4 p[kMaxSplit][2];
#pragma unroll
              for (int sp = 0; sp < kMaxSplit; ++sp)
                if (sp < a.split_k) {
                  const float4* src = reinterpret_cast<const float4*>(
                      base + sp * tstride + (static_cast<size_t>(c) * 128 + row) * 16) + 2 * hf;
                  p[sp][0] = __ldcg(src);
                  p[sp][1] = __ldcg(src + 1);
                }
#pragma unroll
              for (int q2 = 0; q2 < 2; ++q2) {
                float4 t = p[0][q2];
#pragma unroll
                for (int sp = 1; sp < kMaxSplit; ++sp)
                  if (sp < a.split_k) {
                    t.x += p[sp][q2].x;
                    t.y += p[sp][q2].y;
                    t.z += p[sp][q2].z;
                    t.w += p[sp][q2].w;
                  }
                const int q4 = 2 * hf + q2;
                v[4 * q4] = t.x;
                v[4 * q4 + 1] = t.y;
                v[4 * q4 + 2] = t.z;
                v[4 * q4 + 3] = t.w;
              }
            }
            epi_post<EPI>(a, it, row, c * 16, v, cur, esm, c & 1);
            cur = nxt;
            if (rope && c + 1 < nchunks) {
              rope_store(esm, (c + 1) & 1, rr);
              named_bar_sync(1, 128);
            }
          }
        }
      }
    }
    if constexpr (EPI == EPI_ARGMAX) {
      if (a.fin_B > 0) {
        // every CTA's keys are final once the last CTA takes the ticket: it decodes the tokens,
        // then m = longest prefix r with cand[b][r+1] == v[b][r] (acceptance rule of Sec. 3.1)
        __threadfence();
        named_bar_sync(1, 128);
        const int et = threadIdx.x - 64;
        if (et == 0) {
          const int old = atomicAdd(a.am_done, 1);
          *s_last = (old == static_cast<int>(gridDim.x) - 1) ? 1 : 0;
          if (*s_last) *a.am_done = 0;
        }
        named_bar_sync(1, 128);
        if (*s_last) {
          __threadfence();
          const int T = a.fin_B * a.fin_R;
          for (int t = et; t < T; t += 128) {
            const int tok = argmax_key_index(__ldcg(a.am_key + t));
            a.am_key[t] = 0ull;
            a.fin_vtok_out[t] = tok;
            a.fin_vtok_ws[t] = tok;
          }
          named_bar_sync(1, 128);
          for (int b = et; b < a.fin_B; b += 128) {
            int m = 0;
            for (int r = 1; r < a.fin_R; ++r) {
              if (a.fin_cand[b * a.fin_R + r] == a.fin_vtok_ws[b * a.fin_R + r - 1]) m = r;
              else break;
            }
            a.fin_accept_out[b] = m;
            a.fin_m_ws[b] = m;
          }
        }
      }
    }
  }

  if (a.cluster > 1) {
    cluster_sync_all();   // every split's partial tile is in its CTA's shared memory
    if (warp >= 2) {
      if (quad_epi<EPI>() && a.cluster > 1) cluster_reduce_quads<EPI>(a, esm, smem_u32(smA), warp - 2, lane, quad_pre);
      else cluster_reduce<EPI>(a, esm, smem_u32(smA), (warp & 3) * 32 + lane, first_pre);
    } else {
      cluster_arrive();
    }
    cluster_wait();       // no CTA leaves while the others still read its shared memory
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, tmem_cols);
  }
  trace_exit();
}

// ------------------------------------------------------------------ host side
namespace {
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

template <int NMAX, int EPI, int ST = Cfg<NMAX>::STAGES, bool F8 = false>
cudaError_t set_smem_attr() {
  return cudaFuncSetAttribute(gemm_tc_kernel<NMAX, EPI, ST, F8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              KCfg<NMAX, EPI, ST>::SMEM_BYTES);
}

template <int NMAX, int EPI, int ST = Cfg<NMAX>::STAGES, bool F8 = false>
cudaError_t launch_one(const GemmArgs& a, int grid, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = KCfg<NMAX, EPI, ST>::SMEM_BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (a.cluster > 1) {   // the split_k CTAs of a tile form one thread-block cluster
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = a.cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<NMAX, EPI, ST, F8>, a, a);
}
}  // namespace

bool encode_map_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                   std::string* err, int elem_bytes) {
  auto fn = get_encode();
  if (fn == nullptr) {
    *err = "cuTensorMapEncodeTiled not available from the driver";
    return false;
  }
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * static_cast<cuuint64_t>(elem_bytes)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(128 / elem_bytes), box_rows};
  cuuint32_t es[2] = {1, 1};
  const CUtensorMapDataType dt = elem_bytes == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUresult r = fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *err = "cuTensorMapEncodeTiled (2-D) failed with code " + std::to_string(static_cast<int>(r));
    return false;
  }
  return true;
}

bool encode_map_3d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t depth,
                   uint32_t box_rows, std::string* err, int elem_bytes) {
  auto fn = get_encode();
  if (fn == nullptr) {
    *err = "cuTensorMapEncodeTiled not available from the driver";
    return false;
  }
  const cuuint64_t eb = static_cast<cuuint64_t>(elem_bytes);
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {inner * eb, inner * rows * eb};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(128 / elem_bytes), box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  const CUtensorMapDataType dt = elem_bytes == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUresult r = fn(m, dt, 3, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *err = "cuTensorMapEncodeTiled (3-D) failed with code " + std::to_string(static_cast<int>(r));
    return false;
  }
  return true;
}

bool encode_act_maps(CUtensorMap (&maps)[5], const void* base, uint64_t inner, uint64_t rows, std::string* err,
                     int elem_bytes) {
  for (int b = 0; b < 5; ++b)
    if (!encode_map_2d(&maps[b], base, inner, rows, 16u << b, err, elem_bytes)) return false;
  return true;
}

cudaError_t gemm_prepare() {
  cudaError_t e = cudaSuccess;
#define FM_ATTR(E)                                                  \
  if (e == cudaSuccess) e = set_smem_attr<64, E>();                 \
  if (e == cudaSuccess) e = set_smem_attr<256, E>();
  FM_ATTR(EPI_F32)
  FM_ATTR(EPI_RESID)
  FM_ATTR(EPI_QKV)
  FM_ATTR(EPI_SWIGLU)
  FM_ATTR(EPI_SCATTER)
  FM_ATTR(EPI_ARGMAX)
  FM_ATTR(EPI_LOSS)
#undef FM_ATTR
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_MOE>();
  if (e == cudaSuccess) e = set_smem_attr<128, EPI_MOE, 4>();
  // fp8 experts and the dense e4m3 GEMM: separate instantiations, so that the bf16 kernels carry
  // no fp8 code
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_MOE, Cfg<64>::STAGES, true>();
  if (e == cudaSuccess) e = set_smem_attr<128, EPI_MOE, 4, true>();
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_F32, Cfg<64>::STAGES, true>();
  if (e == cudaSuccess) e = set_smem_attr<256, EPI_F32, Cfg<256>::STAGES, true>();
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_F32, kShallowStages>();
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_RESID, kShallowStages>();
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_QKV, kShallowStages>();
  if (e == cudaSuccess) e = set_smem_attr<64, EPI_SWIGLU, kShallowStages>();
  num_sms();
  return e;
}

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

// Most clusters of s CTAs of the dense cluster GEMM kernel (one CTA per SM) resident at once.
static int max_resident_clusters(int s) {
  static int cache[kMaxSplit + 1] = {};
  if (cache[s] == 0) {
    set_smem_attr<64, EPI_F32, kShallowStages>();
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(s * num_sms()));
    cfg.blockDim = dim3(192);
    cfg.dynamicSmemBytes = Cfg<64, kShallowStages>::SMEM_BYTES;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = static_cast<unsigned>(s);
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<64, EPI_F32, kShallowStages>, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = 1;
    }
    cache[s] = n;
  }
  return cache[s];
}

int dense_split_k(int N, int K) {
  // Splits per weight tile: about one CTA per SM over the whole matrix, at least two k-chunks
  // (16 KB of weights) per split, at most kMaxSplit, and no more than lets every tile's cluster
  // of splits be resident at once.  A function of the shape (and the GPU) only.
  const int n_tiles = (N + 127) / 128;
  const int kc = K / 64;
  int s = num_sms() / n_tiles;
  if (s > kc / 2) s = kc / 2;
  if (s > kMaxSplit) s = kMaxSplit;
  while (s > 1 && n_tiles > max_resident_clusters(s)) --s;
  if (s < 1) s = 1;
  return s;
}

cudaError_t moe_launch(const GemmArgs& gate_up, const GemmArgs& down, cudaStream_t s) {
  // one persistent CTA per SM; its down items wait on gate/up tiles of other CTAs, so the
  // launch is cooperative (every CTA resident at once).  Items of up to 64 rows run the
  // 8-stage 64-column kernel, items of up to 128 rows the 4-stage dual kernel.
  const bool large = gate_up.grp_rows > kExpertTileRows;
  if (gate_up.grp_rows != down.grp_rows || (gate_up.grp_rows != kExpertTileRows && gate_up.grp_rows != kExpertTileRowsLarge))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(num_sms());
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = large ? KCfg<128, EPI_MOE, 4>::SMEM_BYTES : Cfg<64>::SMEM_BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (gate_up.f8) {
    if (large) return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<128, EPI_MOE, 4, true>, gate_up, down);
    return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<64, EPI_MOE, Cfg<64>::STAGES, true>, gate_up, down);
  }
  if (large) return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<128, EPI_MOE, 4>, gate_up, down);
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<64, EPI_MOE, Cfg<64>::STAGES>, gate_up, down);
}

cudaError_t gemm_launch(int epi, int nmax, const GemmArgs& a, int grid, cudaStream_t s, bool pdl) {
  if (grid <= 0) return cudaSuccess;
  if (a.f8) {   // the dense e4m3 GEMM (plain fp32 output with row scales)
    if (epi != EPI_F32 || a.cluster > 1 || a.split_k != 1) return cudaErrorInvalidValue;
    return nmax <= 64 ? launch_one<64, EPI_F32, Cfg<64>::STAGES, true>(a, grid, s, pdl)
                      : launch_one<256, EPI_F32, Cfg<256>::STAGES, true>(a, grid, s, pdl);
  }
  if (a.cluster > 1 && nmax <= 64) {   // the dense cluster schedule: short per-split streams
    switch (epi) {
      case EPI_F32:
        return launch_one<64, EPI_F32, kShallowStages>(a, grid, s, pdl);
      case EPI_RESID:
        return launch_one<64, EPI_RESID, kShallowStages>(a, grid, s, pdl);
      case EPI_QKV:
        return launch_one<64, EPI_QKV, kShallowStages>(a, grid, s, pdl);
      case EPI_SWIGLU:
        return launch_one<64, EPI_SWIGLU, kShallowStages>(a, grid, s, pdl);
      default:
        return cudaErrorInvalidValue;
    }
  }
#define FM_CASE(E)                                                                      \
  case E:                                                                               \
    return nmax <= 64 ? launch_one<64, E>(a, grid, s, pdl) : launch_one<256, E>(a, grid, s, pdl);
  switch (epi) {
    FM_CASE(EPI_F32)
    FM_CASE(EPI_RESID)
    FM_CASE(EPI_QKV)
    FM_CASE(EPI_SWIGLU)
    FM_CASE(EPI_SCATTER)
    FM_CASE(EPI_ARGMAX)
    FM_CASE(EPI_LOSS)
    default:
      return cudaErrorInvalidValue;
  }
#undef FM_CASE
}

#ifdef FM_TRACE
FM_TRACE_READER(trace_read_gemm)
#endif

}  // namespace fm
