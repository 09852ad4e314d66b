// Split-KV decode attention over a paged bf16 KV cache plus staged candidate rows.
//
// Each sequence has R queries at consecutive positions p0..p0+R-1 (the K+1 verify
// candidates, or one draft row).  Keys at positions < ctx_len live in the sequence's pages,
// keys at positions >= ctx_len in a staging buffer (candidates not yet committed).  The key
// range is cut into chunks of 64 positions and super-chunks of 4 chunks (256 positions), both
// fixed by absolute position.
//
// Arithmetic (fixed by position, never by the launch shape): a super-chunk's chunks are
// folded in chunk order by the online softmax (running max M, sum L and unnormalised output O
// per query, rescaled by 2^(M_old - M_new) when the max grows); a query's result is the merge
// of its super-chunks, O = sum_s w_s O_s / sum_s w_s L_s with w_s = 2^(M_s - max M), the
// outputs added in position order and the sums over a fixed tree.
// Scores K q^T and outputs V^T p^T run on bf16 tensor cores (mma.sync m16n8k16, fp32
// accumulation, queries padded to 8); a score sums its even and its odd 16-dim steps
// separately, then adds the two; p enters the product as two bf16 terms (hi + lo, about 16
// bits) whose products accumulate separately over a super-chunk and are added at its end; the
// transposes between the score and the product layouts stay in registers (movmatrix).  Masked
// keys contribute exact zeros, so a query's result is the same whether its keys sit in pages
// or in staging and however many queries or sequences share the launch: greedy decoding
// (K = 0) and speculative verification see identical rows.
//
// Scheduling: the launch's work is the list of (sequence, head, super-chunk) items, sequences
// in order, then heads, then super-chunks.  Every CTA builds the list's per-sequence prefix
// from the lengths and takes one contiguous share of ceil(W / grid) items, so that it streams
// many chunks back to back whatever the mix of lengths, and all shares but the last are equal.
// One producer warp fetches up to two chunks ahead: a chunk whose 64 keys are all committed
// is one page segment per head, its K and V rows two contiguous 16 KB blocks fetched as four
// TMA boxes (64 rows x 128 bytes, 128-byte swizzle); a chunk holding the newest keys (staged
// candidates, masked positions) is gathered row by row with 16-byte cp.async into the same
// swizzled layout, zero-filled where there is no key; the queries of each (sequence, head)
// go to one of two query slots.  Four consumer warps each recompute a chunk's 64 x 8 scores
// (cheap) and own 32 of the 128 output dims.  Each super-chunk's (M, L, O) goes to global
// memory; the CTA whose atomic count completes the super-chunks of a (sequence, head) merges
// them (no wait on other CTAs).  In the verify step, where nothing in the step writes the
// pages, the producer fetches the first committed chunks before it waits for the previous
// kernel.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

constexpr int kCH = kAttnChunk;                  // keys per chunk (64)
constexpr int kSuper = kAttnSuper;               // chunks per super-chunk
constexpr int kHalfBytes = kCH * 128;            // 64 rows x 64 dims of K or V: 8 KB
constexpr int kTileBytes = 2 * kHalfBytes;       // K (or V) of a chunk: 16 KB
constexpr int kStageBytes = 2 * kTileBytes;      // K and V of a chunk: 32 KB
constexpr int kQBytes = kMaxR * kHD * 2;         // the queries of one (sequence, head): 2 KB
// Chunks in flight per CTA: two stages keep a CTA at 64 KB of shared memory and 128 registers
// a thread, three CTAs per SM (192 KB in flight per SM, as three stages at two CTAs would) --
// more CTAs, so that a launch spreads over more of them.  Launches over one or two sequences
// (at most a few items per SM) take four stages, one CTA per SM: a super-chunk's four chunks
// are then all fetched before the wait for the previous kernel.
constexpr int kAttnStages = 2;
constexpr int kAttnStagesSmall = 4;
// Launches whose items fit two CTAs per SM at once take three stages: three of a super-chunk's
// four chunks are fetched before the wait.
constexpr int kAttnStagesMid = 3;
constexpr int kConsumers = 128;                  // four warps, each owning 32 of the 128 dims
constexpr int kAttnThreads = kConsumers + 32;    // plus the producer warp
constexpr int kPartStride = kAttnPartStride;     // floats per (super-chunk, query): O[128], M, L, pad

// Shared memory of a CTA of a launch over B sequences: 1 KB alignment slack, the stages, two
// query slots, the barriers, the flags, and the per-sequence tables (first query position,
// slot, item prefix).
constexpr int kXchgBytes = 4 * 32 * 16 + 2 * 4 * kMaxR * 4;   // P fragments of the 4 key tiles, max / sum partials
constexpr size_t attn_smem(int stages, int B) {
  return 1024 + stages * kStageBytes + 2 * kQBytes + kXchgBytes + (2 * stages + 4) * 8 + 8 * 4 +
         (3 * static_cast<size_t>(B) + 1) * 4;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}

// ---- warp-level tensor-core helpers (bf16 m16n8k16, fp32 accumulation)
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t (&r)[2]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "r"(addr));
}
// Transpose of an 8x8 b16 matrix held in the warp's fragment layout (lane 4i+j: row i,
// columns 2j, 2j+1).
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Byte offset of 16-byte chunk `ch` of row `row` in a tile of 256-byte rows (the 8 query rows
// of 128 bf16), chunks swizzled by row: conflict-free for ldmatrix.
__device__ __forceinline__ uint32_t swz(int row, int ch) { return row * 256 + ((ch ^ (row & 7)) << 4); }
// Byte offset of 16-byte chunk `ch` (dims 8ch..8ch+7) of key row `row` in a K or V tile: two
// halves of 64 dims, each 64 rows of 128 bytes in the 128-byte swizzle a TMA box writes (chunk
// index XOR row mod 8, from a 1024-byte aligned base).  Conflict-free for ldmatrix.
__device__ __forceinline__ uint32_t swt(int row, int ch) {
  return (ch >> 3) * kHalfBytes + row * 128 + (((ch & 7) ^ (row & 7)) << 4);
}

// Arrives on the mbarrier when every cp.async this thread issued before has landed; the
// arrival counts against the barrier's expected count.
__device__ __forceinline__ void cp_async_mbar_arrive(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}
// Orders this thread's earlier generic-proxy shared-memory accesses before its later TMA writes.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// A position in a CTA's share of the item list: item i is super-chunk s of head h of
// sequence b, which has nsup super-chunks.  pref[b] is the index of sequence b's first item
// (pref[B] = the launch's item count).
struct Walk {
  int i, b, h, s, nsup;
  __device__ __forceinline__ void seek(const int* pref, int B, int item) {
    int lo = 0, hi = B - 1;   // the last sequence whose first item is <= item has items
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (pref[mid] <= item) lo = mid;
      else hi = mid - 1;
    }
    i = item;
    b = lo;
    nsup = (pref[b + 1] - pref[b]) / kH;
    const int r = item - pref[b];
    h = r / nsup;
    s = r - h * nsup;
  }
  // the next item (the caller has checked that there is one)
  __device__ __forceinline__ void next(const int* pref) {
    ++i;
    if (++s < nsup) return;
    s = 0;
    if (++h < kH) return;
    h = 0;
    do ++b;
    while (pref[b + 1] == pref[b]);
    nsup = (pref[b + 1] - pref[b]) / kH;
  }
};

__device__ __forceinline__ int chunks_live(int p0, int R) { return (p0 + R - 1) / kCH + 1; }

// Merge of the super-chunks of every query of (sequence b, head h), run by the 128 consumer
// threads of the CTA that completed its count: query r combines super-chunks 0..floor(p_r/256).
// Warp w takes queries w, w + 4, each lane four output dims.  Every load a query needs is
// issued before its first use (one round trip to L2 for up to 8 super-chunks): lane l holds the
// maximum and the sum of super-chunk l (l + 32, ...), the maximum M is the warp's maximum, the
// weighted sum L = sum_s w_s L_s is added per lane and then over a fixed tree of lanes, and the
// output O = sum_s w_s O_s is added in position order, with w_s = 2^(M_s - M) taken from lane s
// by a shuffle.  The order of every sum depends on the query's position only.
__device__ __forceinline__ void merge_seq_head(const AttnArgs& a, int b, int h, int R, int p0, int n_super, int tid) {
  const int lane = tid & 31, warp = tid >> 5;
  const float* part = a.part + (static_cast<size_t>(b) * kH + h) * n_super * R * kPartStride;
  const size_t sst = static_cast<size_t>(R) * kPartStride;   // floats between super-chunks of a query
  const int d = lane * 4;
  for (int r = warp; r < R; r += kConsumers / 32) {
    const int ns = (p0 + r) / (kCH * kSuper) + 1;
    const float* pr = part + static_cast<size_t>(r) * kPartStride;
    // the first group's statistics and the first eight outputs, all in flight together
    float ms0 = -INFINITY, ls0 = 0.f;
    if (lane < ns) {
      ms0 = __ldcg(pr + lane * sst + kHD);
      ls0 = __ldcg(pr + lane * sst + kHD + 1);
    }
    float4 x[8];
#pragma unroll
    for (int t = 0; t < 8; ++t)
      if (t < ns) x[t] = __ldcg(reinterpret_cast<const float4*>(pr + t * sst + d));
    float m = ms0;
    for (int s = lane + 32; s < ns; s += 32) m = fmaxf(m, __ldcg(pr + s * sst + kHD));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    const float M = m;
    float w0 = (ms0 == -INFINITY) ? 0.f : exp2f(ms0 - M);
    float l = ls0 * w0;
    for (int s = lane + 32; s < ns; s += 32) {
      const float ms = __ldcg(pr + s * sst + kHD);
      l += __ldcg(pr + s * sst + kHD + 1) * ((ms == -INFINITY) ? 0.f : exp2f(ms - M));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = 0; s0 < ns; s0 += 32) {
      float w = w0;   // weight of super-chunk s0 + lane
      if (s0 > 0) {
        const int s = s0 + lane;
        const float ms = (s < ns) ? __ldcg(pr + s * sst + kHD) : -INFINITY;
        w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
      }
      const int n = min(32, ns - s0);
      for (int j = 0; j < n; j += 8) {
        if (s0 > 0 || j > 0) {
#pragma unroll
          for (int t = 0; t < 8; ++t)
            if (j + t < n) x[t] = __ldcg(reinterpret_cast<const float4*>(pr + (s0 + j + t) * sst + d));
        }
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const float wt = __shfl_sync(0xffffffffu, w, (j + t) & 31);
          if (j + t < n) {
            O.x += x[t].x * wt;
            O.y += x[t].y * wt;
            O.z += x[t].z * wt;
            O.w += x[t].w * wt;
          }
        }
      }
    }
    const float inv = 1.f / l;
    bf16* o = a.out + (static_cast<size_t>(b) * a.out_row_stride_seq + r) * (kH * kHD) + h * kHD + d;
    *reinterpret_cast<__nv_bfloat162*>(o) = __floats2bfloat162_rn(O.x * inv, O.y * inv);
    *reinterpret_cast<__nv_bfloat162*>(o + 2) = __floats2bfloat162_rn(O.z * inv, O.w * inv);
  }
}

template <int kStages>
__global__ void __launch_bounds__(kAttnThreads, kStages == 2 ? 3 : (kStages == 3 ? 2 : 1)) attn_kernel(const __grid_constant__ AttnArgs a) {
  extern __shared__ uint8_t asmem_raw[];
  const uint32_t raw_u32 = smem_u32(asmem_raw);
  uint8_t* stages = asmem_raw + (((raw_u32 + 1023u) & ~1023u) - raw_u32);   // [S][K 16 KB | V 16 KB]
  uint8_t* sQ = stages + kStages * kStageBytes;                             // [2][8 queries][128] bf16
  uint4* sP = reinterpret_cast<uint4*>(sQ + 2 * kQBytes);                  // [4 key tiles][32 lanes] P^T frags
  float* s_cmax = reinterpret_cast<float*>(sP + 4 * 32);                    // [4 warps][8 queries] chunk max
  float* s_csum = s_cmax + 4 * kMaxR;                                       // [4 warps][8 queries] chunk sum
  uint64_t* full = reinterpret_cast<uint64_t*>(s_csum + 4 * kMaxR);         // [S] chunk landed
  uint64_t* empty = full + kStages;                                         // [S] chunk consumed
  uint64_t* qfull = empty + kStages;                                        // [2] queries landed
  uint64_t* qempty = qfull + 2;                                             // [2] queries loaded
  int* s_flag = reinterpret_cast<int*>(qempty + 2);                         // abort, last, err, warp sums[5]
  volatile int* s_abort = s_flag;
  int* s_p0 = s_flag + 8;                                                   // [B] first query position
  int* s_slot = s_p0 + a.B;                                                 // [B] slot
  int* s_pref = s_slot + a.B;                                               // [B + 1] first item
  pdl_trigger(kTrAttn);
  if (!a.prewait) pdl_wait();

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int B = a.B, R = a.R;
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) {
      mbar_init(&full[st], 32);
      mbar_init(&empty[st], kConsumers / 32);
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(&qfull[q], 32);
      mbar_init(&qempty[q], kConsumers / 32);
    }
    s_flag[0] = 0;
    s_flag[2] = 0;
    fence_mbar_init();
  }
  if (tid == kConsumers && a.use_tma) tma_prefetch_desc(&a.kv_map);

  // ---- per-sequence tables: slot, first query position and super-chunk count, then the
  // exclusive prefix of the item counts (thread t scans a contiguous block of sequences)
  for (int bb = tid; bb < B; bb += kAttnThreads) s_slot[bb] = a.slots[bb];
  __syncthreads();
  int errbits = 0;
  for (int bb = tid; bb < B; bb += kAttnThreads) {
    const int slot = s_slot[bb];
    int p0 = -1, nsup = 0;
    if (slot < 0 || slot >= a.n_slots) {
      errbits |= ERR_SLOT_RANGE;
    } else {
      p0 = a.seq_len[slot] + a.qoff;
      if (p0 >= 0) {
        const int n_live = chunks_live(p0, R);
        if (n_live > a.n_chunks) errbits |= ERR_PAGE_RANGE;
        else nsup = (n_live + kSuper - 1) / kSuper;
      }
    }
    s_p0[bb] = p0;
    s_pref[bb] = nsup * kH;
  }
  if (errbits) atomicOr(&s_flag[2], errbits);
  __syncthreads();
  {
    const int per = (B + kAttnThreads - 1) / kAttnThreads;
    const int b0 = min(B, tid * per), b1 = min(B, b0 + per);
    int own = 0;
    for (int bb = b0; bb < b1; ++bb) own += s_pref[bb];
    int incl = own;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_flag[3 + warp] = incl;
    __syncthreads();
    int acc = incl - own;
    for (int w = 0; w < warp; ++w) acc += s_flag[3 + w];
    for (int bb = b0; bb < b1; ++bb) {
      const int n = s_pref[bb];
      s_pref[bb] = acc;
      acc += n;
    }
    if (tid == kAttnThreads - 1) s_pref[B] = acc;
  }
  __syncthreads();
  if (blockIdx.x == 0 && tid == 0 && s_flag[2]) {
    pdl_wait();
    atomicOr(a.err, s_flag[2]);
  }
  const int W = s_pref[B];
  const int per_cta = (W + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x);
  const int i_begin = static_cast<int>(blockIdx.x) * per_cta;
  const int i_end = min(W, i_begin + per_cta);
  if (i_begin >= i_end) return;
  const int n_super = (a.n_chunks + kSuper - 1) / kSuper;

  if (warp == kConsumers / 32) {
    // ------------------------------------------------------------------ producer warp
    const uint64_t pol = l2_policy_evict_first();
    int perr = 0;
    // lanes 0..3: the page of chunk 4 s + lane of item w if it can come by TMA (its 64 keys
    // all committed), -1 if it is gathered, -2 if its page is outside the table or the pool
    auto lookup = [&](const Walk& w) -> int {
      int pg = -1;
      if (lane < kSuper && a.use_tma) {
        const int p0 = s_p0[w.b], c = kSuper * w.s + lane;
        if (c < chunks_live(p0, R) && (c + 1) * kCH <= p0 - a.qoff) {
          const int pi = c * kCH / a.page_size;
          pg = (pi < a.max_pages) ? a.block_table[s_slot[w.b] * a.max_pages + pi] : -2;
          if (pg < 0 || pg >= a.n_pages) pg = -2;
        }
      }
      return pg;
    };
    auto issue_tma = [&](int st, int page, int h, int c) {
      if (lane == 0) {
        if (page < 0) {   // completes the stage without data; the guard flag reports it
          perr |= ERR_PAGE_RANGE;
          mbar_arrive(&full[st]);
        } else {
          uint8_t* dst = stages + st * kStageBytes;
          const int row_k = (page * 2 * kH + h) * a.page_size + (c * kCH) % a.page_size;
          const int row_v = row_k + kH * a.page_size;
          fence_proxy_async_smem();
          mbar_arrive_expect_tx(&full[st], kStageBytes);
          tma_load_2d(dst, &a.kv_map, &full[st], 0, row_k, pol);
          tma_load_2d(dst + kHalfBytes, &a.kv_map, &full[st], 64, row_k, pol);
          tma_load_2d(dst + kTileBytes, &a.kv_map, &full[st], 0, row_v, pol);
          tma_load_2d(dst + kTileBytes + kHalfBytes, &a.kv_map, &full[st], 64, row_v, pol);
        }
      } else {
        mbar_arrive(&full[st]);
      }
    };
    // keys lane and lane + 32 of chunk c, K and V, eight... sixteen 16-byte pieces each
    auto issue_gather = [&](int st, int b, int h, int c) {
      uint8_t* stage = stages + st * kStageBytes;
      const int slot = s_slot[b], p0 = s_p0[b];
      const int sl = p0 - a.qoff, last = p0 + R - 1;
#pragma unroll
      for (int k2 = 0; k2 < 2; ++k2) {
        const int key = lane + 32 * k2, pos = c * kCH + key;
        const bf16* srck = a.pool;
        const bf16* srcv = a.pool;
        int bytes = 0;
        if (pos <= last) {
          if (pos < sl) {
            const int pi = pos / a.page_size;
            const int page = (pi < a.max_pages) ? a.block_table[slot * a.max_pages + pi] : -1;
            if (page >= 0 && page < a.n_pages) {
              srck = a.pool + ((static_cast<long long>(page) * 2 * kH + h) * a.page_size + pos % a.page_size) * kHD;
              srcv = srck + static_cast<long long>(kH) * a.page_size * kHD;
              bytes = 16;
            } else {
              perr |= ERR_PAGE_RANGE;
            }
          } else {
            srck = a.stage + b * a.stage_seq_stride + static_cast<long long>(pos - sl) * a.stage_row_stride +
                   static_cast<long long>(h) * kHD;
            srcv = srck + a.stage_kv_stride;
            bytes = 16;
          }
        }
#pragma unroll
        for (int ch = 0; ch < 16; ++ch) {
          const int o = bytes ? ch * 8 : 0;
          cp_async16(stage + swt(key, ch), srck + o, bytes);
          cp_async16(stage + kTileBytes + swt(key, ch), srcv + o, bytes);
        }
      }
      cp_async_mbar_arrive(&full[st]);
    };
    // the queries of run r (rows R..7 zero) into slot r & 1, four 16-byte pieces per lane
    auto issue_q = [&](int r, int b, int h) -> bool {
      const int qs = r & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&qempty[qs], ((r >> 1) & 1) ^ 1u, s_abort));
      if (!ok) return false;
      const int qrow0 = a.q_row0 ? a.q_row0[b] : b * R;
      const int row = lane >> 2;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int ch = (lane & 3) * 4 + k;
        const bool has = row < R;
        const bf16* src = has ? a.q + (static_cast<size_t>(qrow0 + row) * kH + h) * kHD + ch * 8 : a.q;
        cp_async16(sQ + qs * kQBytes + swz(row, ch), src, has ? 16 : 0);
      }
      cp_async_mbar_arrive(&qfull[qs]);
      return true;
    };

    Walk w;
    w.seek(s_pref, B, i_begin);
    // pass 1 (verify step): the K/V of the leading committed chunks, before the wait
    int j_pre = 0;
    if (a.prewait) {
      Walk v = w;
      bool go = true;
      while (go) {
        const int pg = lookup(v);
        const int c0 = kSuper * v.s, c1 = min(c0 + kSuper, chunks_live(s_p0[v.b], R));
        const int safe = s_p0[v.b] - a.qoff - a.prewait_guard;   // keys below this are not written by this graph
        for (int c = c0; c < c1 && go; ++c) {
          const int page = __shfl_sync(0xffffffffu, pg, c - c0);
          if (page == -1 || j_pre == kStages || (c + 1) * kCH > safe) {
            go = false;
          } else {
            issue_tma(j_pre, page, v.h, c);
            ++j_pre;
          }
        }
        if (go && v.i + 1 < i_end) v.next(s_pref);
        else go = false;
      }
      pdl_wait();
    }
    // pass 2: every chunk in order -- the queries at the start of each (sequence, head) run,
    // the K/V of the chunks pass 1 did not fetch; page lookups one item ahead
    int j = 0, r = -1;
    bool failed = false;
    int pg = lookup(w);
    Walk wn = w;
    bool has_next = w.i + 1 < i_end;
    int pg_next = -1;
    if (has_next) {
      wn.next(s_pref);
      pg_next = lookup(wn);
    }
    while (true) {
      if (w.i == i_begin || w.s == 0) {
        ++r;
        if (!issue_q(r, w.b, w.h)) {
          failed = true;
          break;
        }
      }
      const int c0 = kSuper * w.s, c1 = min(c0 + kSuper, chunks_live(s_p0[w.b], R));
      for (int c = c0; c < c1; ++c, ++j) {
        if (j < j_pre) continue;
        const int st = j % kStages;
        if (!__all_sync(0xffffffffu, mbar_wait(&empty[st], ((j / kStages) & 1) ^ 1u, s_abort))) {
          failed = true;
          break;
        }
        const int page = __shfl_sync(0xffffffffu, pg, c - c0);
        if (page == -1) issue_gather(st, w.b, w.h, c);
        else issue_tma(st, page, w.h, c);
      }
      if (failed || !has_next) break;
      w = wn;
      pg = pg_next;
      has_next = w.i + 1 < i_end;
      if (has_next) {
        wn.next(s_pref);
        pg_next = lookup(wn);
      }
    }
    if (failed) {
      if (lane == 0) *s_abort = 1;
      perr |= ERR_WAIT_TIMEOUT;
    }
    // let every copy still in flight land before the CTA's shared memory is released
    asm volatile("cp.async.wait_all;" ::: "memory");
    if (lane == 0) {
      volatile int never = 0;
      const int issued = max(j, j_pre);
      for (int jj = max(0, issued - kStages); jj < issued; ++jj)
        mbar_wait(&full[jj % kStages], static_cast<uint32_t>(jj / kStages) & 1u, &never, 100000000ull);
    }
    perr = __reduce_or_sync(0xffffffffu, perr);
    if (lane == 0 && perr) atomicOr(a.err, perr);
    return;
  }

  // -------------------------------------------------------------------- consumer warps
  if (a.prewait) pdl_wait();
  const int g = lane >> 2, t4 = lane & 3, mi = lane >> 3, ri = lane & 7;
  const int qa = 2 * t4, qb = 2 * t4 + 1;                    // the two queries of this lane
  const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(kHD));   // log2(e) / sqrt(hd)
  Walk w;
  w.seek(s_pref, B, i_begin);
  int j = 0, r = -1, run_items = 0;
  bool ok = true;            // false once a wait has run out: the rest is walked without compute
  uint32_t qf[8][2];         // Q^T fragments (B operand of S^T = K Q^T) of the current run
  while (true) {
    if (w.i == i_begin || w.s == 0) {
      ++r;
      run_items = 0;
      const int qs = r & 1;
      if (ok && !__all_sync(0xffffffffu, mbar_wait(&qfull[qs], (r >> 1) & 1, s_abort))) ok = false;
      const uint32_t qbase = smem_u32(sQ + qs * kQBytes);
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) ldsm_x2(qbase + swz(ri, 2 * ks + (mi & 1)), qf[ks]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&qempty[qs]);
    }
    const int b = w.b, h = w.h;
    const int p0 = s_p0[b];
    const int c0 = kSuper * w.s, c1 = min(c0 + kSuper, chunks_live(p0, R));
    float M_a = -INFINITY, M_b = -INFINITY, L_a = 0.f, L_b = 0.f;
    float O[2][4], Ol[2][4];   // hi and lo parts of the unnormalised output, dims 32 warp + 16 j
#pragma unroll
    for (int jj = 0; jj < 2; ++jj)
#pragma unroll
      for (int e = 0; e < 4; ++e) O[jj][e] = Ol[jj][e] = 0.f;
    for (int c = c0; c < c1; ++c, ++j) {
      const int st = j % kStages;
      if (ok && !__all_sync(0xffffffffu, mbar_wait(&full[st], (j / kStages) & 1, s_abort))) {
        ok = false;
        if (lane == 0) {
          *s_abort = 1;
          atomicOr(a.err, ERR_WAIT_TIMEOUT);
        }
      }
      {
        // Warp w scores the chunk's keys 16w..16w+15 (S^T = K Q^T over 8 k-steps of 16 dims,
        // even and odd k-steps in separate accumulators, added at the end); the chunk's max and
        // sum per query and its P^T fragments (bf16 hi + lo) go through shared memory, so that
        // each warp can then multiply all 64 keys of V^T for its 32 output dims.  Waits and
        // barriers run even after a wait has run out (then on stale data) so that the four
        // warps always meet at the same barriers.
        const uint32_t kbase = smem_u32(stages + st * kStageBytes);
        const uint32_t vbase = kbase + kTileBytes;
        float sc[4] = {0.f, 0.f, 0.f, 0.f}, sc1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 8; ks += 2) {
          uint32_t ak[4], ak1[4];
          ldsm_x4(kbase + swt(16 * warp + ri + ((mi & 1) ? 8 : 0), 2 * ks + (mi >> 1)), ak);
          ldsm_x4(kbase + swt(16 * warp + ri + ((mi & 1) ? 8 : 0), 2 * ks + 2 + (mi >> 1)), ak1);
          mma_bf16_16816(sc, ak, qf[ks]);
          mma_bf16_16816(sc1, ak1, qf[ks + 1]);
        }
        // visibility and this warp's max per query (lanes sharing t4 hold the same two queries)
        const int kb = c * kCH + 16 * warp;
        float m_a = -INFINITY, m_b = -INFINITY;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kb + g + ((e >> 1) ? 8 : 0);
          const int q = (e & 1) ? qb : qa;
          const float x = (q < R && key <= p0 + q) ? (sc[e] + sc1[e]) * scale : -INFINITY;
          sc[e] = x;
          if (e & 1) m_b = fmaxf(m_b, x);
          else m_a = fmaxf(m_a, x);
        }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          m_a = fmaxf(m_a, __shfl_xor_sync(0xffffffffu, m_a, o));
          m_b = fmaxf(m_b, __shfl_xor_sync(0xffffffffu, m_b, o));
        }
        if (g == 0) {
          s_cmax[warp * kMaxR + qa] = m_a;
          s_cmax[warp * kMaxR + qb] = m_b;
        }
        named_bar_sync(2, kConsumers);
        m_a = fmaxf(fmaxf(s_cmax[qa], s_cmax[kMaxR + qa]), fmaxf(s_cmax[2 * kMaxR + qa], s_cmax[3 * kMaxR + qa]));
        m_b = fmaxf(fmaxf(s_cmax[qb], s_cmax[kMaxR + qb]), fmaxf(s_cmax[2 * kMaxR + qb], s_cmax[3 * kMaxR + qb]));
        const float Mn_a = fmaxf(M_a, m_a), Mn_b = fmaxf(M_b, m_b);
        const float al_a = (M_a == -INFINITY) ? 0.f : exp2f(M_a - Mn_a);
        const float al_b = (M_b == -INFINITY) ? 0.f : exp2f(M_b - Mn_b);
        M_a = Mn_a;
        M_b = Mn_b;
        // p = 2^(x - M) (exact zeros where masked), this warp's sums, and its P^T fragments
        float l_a = 0.f, l_b = 0.f, p[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float Mq = (e & 1) ? M_b : M_a;
          p[e] = (sc[e] == -INFINITY) ? 0.f : exp2f(sc[e] - Mq);
          if (e & 1) l_b += p[e];
          else l_a += p[e];
          lo[e] = p[e] - __bfloat162float(__float2bfloat16(p[e]));
        }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          l_a += __shfl_xor_sync(0xffffffffu, l_a, o);
          l_b += __shfl_xor_sync(0xffffffffu, l_b, o);
        }
        if (g == 0) {
          s_csum[warp * kMaxR + qa] = l_a;
          s_csum[warp * kMaxR + qb] = l_b;
        }
        sP[warp * 32 + lane] = make_uint4(movmatrix_t(pack_bf16(p[0], p[1])),    // keys 16w+0..7
                                          movmatrix_t(pack_bf16(p[2], p[3])),    // keys 16w+8..15
                                          movmatrix_t(pack_bf16(lo[0], lo[1])),
                                          movmatrix_t(pack_bf16(lo[2], lo[3])));
        named_bar_sync(2, kConsumers);
        L_a = L_a * al_a + (((s_csum[qa] + s_csum[kMaxR + qa]) + s_csum[2 * kMaxR + qa]) + s_csum[3 * kMaxR + qa]);
        L_b = L_b * al_b + (((s_csum[qb] + s_csum[kMaxR + qb]) + s_csum[2 * kMaxR + qb]) + s_csum[3 * kMaxR + qb]);
        // O^T[dim][query] = al * O^T + V^T P^T for this warp's two 16-dim tiles (dims
        // 32w..32w+31), 4 k-steps of 16 keys; hi and lo products in separate accumulators
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          O[jj][0] *= al_a;
          O[jj][1] *= al_b;
          O[jj][2] *= al_a;
          O[jj][3] *= al_b;
          Ol[jj][0] *= al_a;
          Ol[jj][1] *= al_b;
          Ol[jj][2] *= al_a;
          Ol[jj][3] *= al_b;
        }
#pragma unroll
        for (int kt = 0; kt < 4; ++kt) {
          const uint4 pf = sP[kt * 32 + lane];
          const uint32_t ph[2] = {pf.x, pf.y}, pl[2] = {pf.z, pf.w};
#pragma unroll
          for (int jj = 0; jj < 2; ++jj) {
            uint32_t av[4];
            ldsm_x4_t(vbase + swt(16 * kt + ri + ((mi >> 1) ? 8 : 0), 2 * (2 * warp + jj) + (mi & 1)), av);
            mma_bf16_16816(O[jj], av, ph);
            mma_bf16_16816(Ol[jj], av, pl);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);   // this warp is done with the stage
    }
    // end of the super-chunk: its (M, L, O) per query (each warp its 32 dims)
    {
      float* ps = a.part + ((static_cast<size_t>(b) * kH + h) * n_super + w.s) * R * kPartStride;
#pragma unroll
      for (int jj = 0; jj < 2; ++jj) {
        const int d = 16 * (2 * warp + jj) + g;
        if (qa < R) {
          ps[qa * kPartStride + d] = O[jj][0] + Ol[jj][0];
          ps[qa * kPartStride + d + 8] = O[jj][2] + Ol[jj][2];
        }
        if (qb < R) {
          ps[qb * kPartStride + d] = O[jj][1] + Ol[jj][1];
          ps[qb * kPartStride + d + 8] = O[jj][3] + Ol[jj][3];
        }
      }
      if (warp == 0 && g == 0) {
        if (qa < R) {
          ps[qa * kPartStride + kHD] = M_a;
          ps[qa * kPartStride + kHD + 1] = L_a;
        }
        if (qb < R) {
          ps[qb * kPartStride + kHD] = M_b;
          ps[qb * kPartStride + kHD + 1] = L_b;
        }
      }
    }
    ++run_items;
    const bool more = w.i + 1 < i_end;
    if (!more || w.s == w.nsup - 1) {
      // this CTA's super-chunks of (b, h) are written: count them; the CTA that completes the
      // count merges every super-chunk of (b, h).  The barrier orders the four warps' partial
      // stores before thread 0's device-scope fence and count (fences are cumulative).
      named_bar_sync(1, kConsumers);
      if (tid == 0) {
        __threadfence();
        int* ticket = a.tickets + b * kH + h;
        const int old = atomicAdd(ticket, run_items);
        const int last = (old + run_items == w.nsup) ? 1 : 0;
        if (last) *ticket = 0;
        s_flag[1] = last;
      }
      named_bar_sync(1, kConsumers);
      if (s_flag[1]) {
        __threadfence();
        merge_seq_head(a, b, h, R, p0, n_super, tid);
      }
    }
    if (!more) break;
    w.next(s_pref);
  }
  trace_exit();
}

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<kAttnStages>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(attn_smem(kAttnStages, 2048)));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<kAttnStagesSmall>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(attn_smem(kAttnStagesSmall, 2048)));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<kAttnStagesMid>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(attn_smem(kAttnStagesMid, 2048)));
  return e;
}

template <int kStages>
static cudaError_t attention_launch_s(const AttnArgs& a, int B, cudaStream_t s) {
  const size_t smem = attn_smem(kStages, B);
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attn_kernel<kStages>, kAttnThreads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  const long long most = static_cast<long long>(B) * kH * ((a.n_chunks + kSuper - 1) / kSuper);
  long long grid = static_cast<long long>(per_sm) * num_sms();
  if (grid > most) grid = most;
  if (grid < 1) grid = 1;
  return launch_pdl(attn_kernel<kStages>, dim3(static_cast<unsigned>(grid)), dim3(kAttnThreads), smem, s, a);
}

cudaError_t attention_launch(const AttnArgs& a_in, int B, cudaStream_t s) {
  // As many CTAs as fit at once (at most one per item).  Pure scheduling: the arithmetic of
  // every super-chunk and of the merge is the same for any grid and stage count.
  AttnArgs a = a_in;
  a.B = B;
  if (B <= 2) return attention_launch_s<kAttnStagesSmall>(a, B, s);
  const long long items = static_cast<long long>(B) * kH * ((a.n_chunks + kSuper - 1) / kSuper);
  if (items <= 2LL * num_sms()) return attention_launch_s<kAttnStagesMid>(a, B, s);
  return attention_launch_s<kAttnStages>(a, B, s);
}

#ifdef FM_TRACE
FM_TRACE_READER(trace_read_attn)
#endif

}  // namespace fm
