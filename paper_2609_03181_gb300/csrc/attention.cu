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
// of its super-chunks in order, O = sum_s w_s O_s / sum_s w_s L_s with w_s = 2^(M_s - max M).
// Scores K q^T and outputs V^T p^T run on bf16 tensor cores (mma.sync m16n8k16, fp32
// accumulation, queries padded to 8); a score sums its even and its odd 16-dim steps
// separately, then adds the two; p enters the product as two bf16 terms (hi + lo, about 16
// bits) whose products accumulate separately over a super-chunk and are added at its end; the
// transposes between the score and the product layouts stay in registers (movmatrix).  Masked
// keys contribute exact zeros, so a query's result is the same whether its keys sit in pages
// or in staging and however many queries or sequences share the launch: greedy decoding
// (K = 0) and speculative verification see identical rows.
//
// Scheduling: four warps per CTA, each recomputing a chunk's 64 x 8 scores and owning 32 of
// the 128 output dims; two stages per CTA (three CTAs per SM) for launches of about two waves
// or fewer, three stages (two per SM) above.  The CTAs of one (sequence, head) take its
// super-chunks in turn (CTA u: super-chunks u, u + n, u + 2n, ...).  A chunk whose 64 keys are
// all committed is one page segment per head: its K and V rows are two contiguous 16 KB
// blocks, fetched as four TMA boxes (64 rows x 128 bytes, 128-byte swizzle) onto the stage's
// mbarrier, issued ahead of the compute.  The chunk holding the newest keys (staged candidates,
// masked positions) is gathered row by row with 16-byte cp.async into the same swizzled layout,
// zero-filled where there is no key.  Each super-chunk's (M, L, O) goes to global memory; the
// CTA that finishes last for a (sequence, head) merges them (atomic ticket, no wait).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

constexpr int kCH = kAttnChunk;                  // keys per chunk (64)
constexpr int kSuper = kAttnSuper;               // chunks per super-chunk
constexpr int kUnitMaxSuper = 4;                 // most super-chunks one CTA streams
constexpr int kUnitMaxChunks = kSuper * kUnitMaxSuper;
constexpr int kHalfBytes = kCH * 128;            // 64 rows x 64 dims of K or V: 8 KB
constexpr int kTileBytes = 2 * kHalfBytes;       // K (or V) of a chunk: 16 KB
constexpr int kStageBytes = 2 * kTileBytes;      // K and V of a chunk: 32 KB
constexpr int kAttnThreads = 128;                // four warps, each owning 32 of the 128 dims
constexpr int kPartStride = kAttnPartStride;     // floats per (super-chunk, query): O[128], M, L, pad
// shared memory of a CTA with `stages` stages: 1 KB alignment slack, the stages, Q, barriers
constexpr int attn_smem(int stages) { return 1024 + stages * kStageBytes + kMaxR * kHD * 2 + stages * 8; }

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
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
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

// Merge of the super-chunks of every query of (sequence b, head h), run by the CTA that
// finishes last for it: query r combines super-chunks 0..floor(p_r/256) in order.  Warp w
// writes queries w, w + 4; each lane four dims.
__device__ __forceinline__ void merge_all(const AttnArgs& a, int b, int h, int R, int p0, int n_sup, float* smem) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_super = (a.n_chunks + kSuper - 1) / kSuper;
  const float* part = a.part + (static_cast<size_t>(b) * kH + h) * n_super * R * kPartStride;
  float* sm = smem;                      // [n_sup * R] super-chunk max, then weight
  float* sl = smem + n_sup * R;          // [n_sup * R] super-chunk sum
  float* sL = sl + n_sup * R;            // [R] total weight
  for (int i = tid; i < n_sup * R; i += kAttnThreads) {
    const float* pc = part + static_cast<size_t>(i) * kPartStride;
    sm[i] = __ldcg(&pc[kHD]);
    sl[i] = __ldcg(&pc[kHD + 1]);
  }
  __syncthreads();
  if (tid < R) {
    const int r = tid, lasts = (p0 + r) / (kCH * kSuper);
    float M = -INFINITY;
    for (int s = 0; s <= lasts; ++s) M = fmaxf(M, sm[s * R + r]);
    float L = 0.f;
    for (int s = 0; s <= lasts; ++s) {
      const float ms = sm[s * R + r];
      const float w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
      sm[s * R + r] = w;
      L += sl[s * R + r] * w;
    }
    sL[r] = L;
  }
  __syncthreads();
  const int d = lane * 4;   // four dims per lane
  for (int r = warp; r < R; r += kAttnThreads / 32) {
    const int lasts = (p0 + r) / (kCH * kSuper);
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    int s = 0;
    for (; s + 4 <= lasts + 1; s += 4) {
      float4 x[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        x[u] = __ldcg(reinterpret_cast<const float4*>(part + (static_cast<size_t>(s + u) * R + r) * kPartStride + d));
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float w = sm[(s + u) * R + r];
        O.x += x[u].x * w;
        O.y += x[u].y * w;
        O.z += x[u].z * w;
        O.w += x[u].w * w;
      }
    }
    for (; s <= lasts; ++s) {
      const float4 x =
          __ldcg(reinterpret_cast<const float4*>(part + (static_cast<size_t>(s) * R + r) * kPartStride + d));
      const float w = sm[s * R + r];
      O.x += x.x * w;
      O.y += x.y * w;
      O.z += x.z * w;
      O.w += x.w * w;
    }
    const float inv = 1.f / sL[r];
    bf16* o = a.out + (static_cast<size_t>(b) * a.out_row_stride_seq + r) * (kH * kHD) + h * kHD + d;
    *reinterpret_cast<__nv_bfloat162*>(o) = __floats2bfloat162_rn(O.x * inv, O.y * inv);
    *reinterpret_cast<__nv_bfloat162*>(o + 2) = __floats2bfloat162_rn(O.z * inv, O.w * inv);
  }
}

// Gathers the K and V rows of chunk c into a stage with 16-byte cp.async (two threads per key,
// eight 16-byte pieces of K and of V each); rows without a visible key are zero-filled.  Used
// for the chunk that holds staged candidates or masked positions, and for every chunk when the
// pool has no TMA map.
__device__ __forceinline__ void gather_chunk(const AttnArgs& a, int b, int h, int slot, int sl, int last, int c,
                                             uint8_t* stage) {
  const int key = threadIdx.x >> 1, half = threadIdx.x & 1;
  const int pos = c * kCH + key;
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
        atomicOr(a.err, ERR_PAGE_RANGE);
      }
    } else {
      srck = a.stage + b * a.stage_seq_stride + static_cast<long long>(pos - sl) * a.stage_row_stride +
             static_cast<long long>(h) * kHD;
      srcv = srck + a.stage_kv_stride;
      bytes = 16;
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int ch = half * 8 + i;
    const int o = bytes ? ch * 8 : 0;
    cp_async16(stage + swt(key, ch), srck + o, bytes);
    cp_async16(stage + kTileBytes + swt(key, ch), srcv + o, bytes);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// kStages stages per CTA: 3 (two CTAs per SM) when the launch spans many waves, 2 (three CTAs
// per SM) when it fits in about two.  Four warps: each recomputes the chunk's 64 x 8 scores
// (cheap) and owns 32 of the 128 output dims, so its dependent MMA chain is short.
template <int kStages>
__global__ void __launch_bounds__(kAttnThreads) attn_chunk_kernel(const __grid_constant__ AttnArgs a) {
  extern __shared__ uint8_t asmem_raw[];
  const uint32_t raw_u32 = smem_u32(asmem_raw);
  uint8_t* stages = asmem_raw + (((raw_u32 + 1023u) & ~1023u) - raw_u32);   // [S][K 16 KB | V 16 KB]
  uint8_t* sQ = stages + kStages * kStageBytes;              // [8 queries][128 dims] bf16
  uint64_t* full = reinterpret_cast<uint64_t*>(sQ + kMaxR * kHD * 2);   // [S] TMA stage barriers
  __shared__ int s_page[kUnitMaxChunks];                     // page of each TMA chunk of the unit
  __shared__ int s_abort;
  __shared__ int s_last;
  pdl_trigger();
  pdl_wait();

  const int u = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, t4 = lane & 3, mi = lane >> 3, ri = lane & 7;
  const int R = a.R;
  // the queries first (bf16, as the QKV epilogue stored them; rows R..7 zero): their loads need
  // no slot and overlap the slot -> length -> page lookups
  uint4 qv = make_uint4(0, 0, 0, 0);
  {
    const int qrow0 = a.q_row0 ? a.q_row0[b] : b * R;
    const int q = tid >> 4, ch = tid & 15;   // 8 queries x 16 pieces of 16 bytes
    if (q < R) qv = *reinterpret_cast<const uint4*>(a.q + (static_cast<size_t>(qrow0 + q) * kH + h) * kHD + ch * 8);
  }
  const int slot = a.slots[b];
  if (slot < 0 || slot >= a.n_slots) {   // every CTA of the sequence leaves; no ticket, no merge
    if (u == 0 && h == 0 && tid == 0) atomicOr(a.err, ERR_SLOT_RANGE);
    return;
  }
  // this CTA's super-chunks: u, u + n_units, u + 2 n_units, ... (strided, so that short contexts
  // spread over the CTAs of the (sequence, head) as evenly as long ones); its chunk list, in
  // increasing order, is chunk_of(i)
  const int n_units = gridDim.x;
  auto chunk_of = [&](int i) { return (u + (i / kSuper) * n_units) * kSuper + i % kSuper; };
  // the pages of every chunk the CTA may own are looked up now, alongside the length
  int spec_page = -1;
  if (tid < a.unit * kSuper) {
    const int pi = chunk_of(tid) * kCH / a.page_size;
    if (pi < a.max_pages) spec_page = a.block_table[slot * a.max_pages + pi];
  }
  const int sl = a.seq_len[slot];
  const int p0 = sl + a.qoff;
  const int last = p0 + R - 1;
  if (p0 < 0) return;
  const int n_live = last / kCH + 1;                         // chunks holding keys 0..last
  const int n_sup_live = (n_live + kSuper - 1) / kSuper;
  if (u >= n_sup_live) return;
  const int n_mine = (n_sup_live - 1 - u) / n_units + 1;            // super-chunks of this CTA
  const int last_sup = u + (n_mine - 1) * n_units;
  const int n = (n_mine - 1) * kSuper + (min(n_live, (last_sup + 1) * kSuper) - last_sup * kSuper);
  // a prefix of the list holds committed keys only and comes by TMA; the rest are gathered
  int n_tma = 0;
  if (a.use_tma)
    while (n_tma < n && (chunk_of(n_tma) + 1) * kCH <= sl) ++n_tma;

  if (tid < n_tma) {
    int page = spec_page;
    if (page < 0 || page >= a.n_pages) {
      atomicOr(a.err, ERR_PAGE_RANGE);
      page = -1;
    }
    s_page[tid] = page;
  }
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(&full[st], 1);
    s_abort = 0;
    fence_mbar_init();
  }
  *reinterpret_cast<uint4*>(sQ + swz(tid >> 4, tid & 15)) = qv;
  __syncthreads();

  // TMA of chunk i of the unit into stage i % S; a chunk whose page is invalid completes its
  // barrier without data (the guard flag is already set)
  const uint64_t pol = l2_policy_evict_first();
  auto issue = [&](int i) {
    const int st = i % kStages;
    uint8_t* dst = stages + st * kStageBytes;
    const int page = s_page[i];
    if (page < 0) {
      mbar_arrive(&full[st]);
      return;
    }
    const int c = chunk_of(i);
    const int row_k = (page * 2 * kH + h) * a.page_size + (c * kCH) % a.page_size;
    const int row_v = row_k + kH * a.page_size;
    mbar_arrive_expect_tx(&full[st], kStageBytes);
    tma_load_2d(dst, &a.kv_map, &full[st], 0, row_k, pol);
    tma_load_2d(dst + kHalfBytes, &a.kv_map, &full[st], 64, row_k, pol);
    tma_load_2d(dst + kTileBytes, &a.kv_map, &full[st], 0, row_v, pol);
    tma_load_2d(dst + kTileBytes + kHalfBytes, &a.kv_map, &full[st], 64, row_v, pol);
  };
  if (tid == 0) {
    if (n_tma > 0) tma_prefetch_desc(&a.kv_map);
    for (int i = 0; i < min(n_tma, kStages); ++i) issue(i);
  }

  // Q^T fragments (B operand of S^T = K Q^T), the same for every chunk
  const uint32_t qbase = smem_u32(sQ);
  uint32_t qf[8][2];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) ldsm_x2(qbase + swz(ri, 2 * ks + (mi & 1)), qf[ks]);

  const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(kHD));   // log2(e) / sqrt(hd)
  const int qa = 2 * t4, qb = 2 * t4 + 1;                    // the two queries of this lane
  float* part = a.part + (static_cast<size_t>(b) * kH + h) * ((a.n_chunks + kSuper - 1) / kSuper) * R * kPartStride;
  float M_a = -INFINITY, M_b = -INFINITY, L_a = 0.f, L_b = 0.f;
  float O[2][4], Ol[2][4];   // hi and lo parts of the unnormalised output, dims 32 warp + 16 j
  int consumed = 0;          // TMA chunks waited for
  bool aborted = false;
  for (int i = 0; i < n; ++i) {
    const int c = chunk_of(i);
    const int st = i % kStages;
    uint8_t* stage = stages + st * kStageBytes;
    if (c % kSuper == 0 || i == 0) {
      M_a = M_b = -INFINITY;
      L_a = L_b = 0.f;
#pragma unroll
      for (int j = 0; j < 2; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) O[j][e] = Ol[j][e] = 0.f;
    }
    if (i < n_tma) {
      const bool ok = mbar_wait(&full[st], static_cast<uint32_t>(i / kStages) & 1u, &s_abort);
      if (__syncthreads_or(!ok)) {
        aborted = true;
        break;
      }
      consumed = i + 1;
    } else {
      gather_chunk(a, b, h, slot, sl, last, c, stage);
      asm volatile("cp.async.wait_group 0;" ::: "memory");
      __syncthreads();
    }
    const uint32_t kbase = smem_u32(stage);
    const uint32_t vbase = kbase + kTileBytes;

    // S^T[key][query] = K Q^T over four 16-key tiles, 8 k-steps of 16 dims: even and odd
    // k-steps in separate accumulators (eight independent MMA chains), added at the end
    float s[4][4], s1[4][4];
#pragma unroll
    for (int kt = 0; kt < 4; ++kt)
#pragma unroll
      for (int e = 0; e < 4; ++e) s[kt][e] = s1[kt][e] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 8; ks += 2) {
#pragma unroll
      for (int kt = 0; kt < 4; ++kt) {
        uint32_t ak[4], ak1[4];
        ldsm_x4(kbase + swt(16 * kt + ri + ((mi & 1) ? 8 : 0), 2 * ks + (mi >> 1)), ak);
        ldsm_x4(kbase + swt(16 * kt + ri + ((mi & 1) ? 8 : 0), 2 * ks + 2 + (mi >> 1)), ak1);
        mma_bf16_16816(s[kt], ak, qf[ks]);
        mma_bf16_16816(s1[kt], ak1, qf[ks + 1]);
      }
    }
#pragma unroll
    for (int kt = 0; kt < 4; ++kt)
#pragma unroll
      for (int e = 0; e < 4; ++e) s[kt][e] += s1[kt][e];
    // visibility, chunk max per query (lanes sharing t4 hold the same two queries)
    const int kb = c * kCH;
    float m_a = -INFINITY, m_b = -INFINITY;
#pragma unroll
    for (int kt = 0; kt < 4; ++kt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kb + 16 * kt + g + ((e >> 1) ? 8 : 0);
        const int q = (e & 1) ? qb : qa;
        const float x = (q < R && key <= p0 + q) ? s[kt][e] * scale : -INFINITY;
        s[kt][e] = x;
        if (e & 1) m_b = fmaxf(m_b, x);
        else m_a = fmaxf(m_a, x);
      }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      m_a = fmaxf(m_a, __shfl_xor_sync(0xffffffffu, m_a, o));
      m_b = fmaxf(m_b, __shfl_xor_sync(0xffffffffu, m_b, o));
    }
    const float Mn_a = fmaxf(M_a, m_a), Mn_b = fmaxf(M_b, m_b);
    const float al_a = (M_a == -INFINITY) ? 0.f : exp2f(M_a - Mn_a);
    const float al_b = (M_b == -INFINITY) ? 0.f : exp2f(M_b - Mn_b);
    M_a = Mn_a;
    M_b = Mn_b;
    // p = 2^(x - M) (exact zeros where masked), row sums, and P^T as bf16 hi + lo fragments
    float l_a = 0.f, l_b = 0.f;
    uint32_t ph[4][2], pl[4][2];
#pragma unroll
    for (int kt = 0; kt < 4; ++kt) {
      float p[4], lo[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float Mq = (e & 1) ? M_b : M_a;
        p[e] = (s[kt][e] == -INFINITY) ? 0.f : exp2f(s[kt][e] - Mq);
        if (e & 1) l_b += p[e];
        else l_a += p[e];
        lo[e] = p[e] - __bfloat162float(__float2bfloat16(p[e]));
      }
      ph[kt][0] = movmatrix_t(pack_bf16(p[0], p[1]));     // keys 16kt+0..7
      ph[kt][1] = movmatrix_t(pack_bf16(p[2], p[3]));     // keys 16kt+8..15
      pl[kt][0] = movmatrix_t(pack_bf16(lo[0], lo[1]));
      pl[kt][1] = movmatrix_t(pack_bf16(lo[2], lo[3]));
    }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      l_a += __shfl_xor_sync(0xffffffffu, l_a, o);
      l_b += __shfl_xor_sync(0xffffffffu, l_b, o);
    }
    L_a = L_a * al_a + l_a;
    L_b = L_b * al_b + l_b;
    // O^T[dim][query] = al * O^T + V^T P^T for this warp's two 16-dim tiles (dims 32w..32w+31),
    // 4 k-steps of 16 keys; hi and lo products in separate accumulators, summed per super-chunk
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      O[j][0] *= al_a;
      O[j][1] *= al_b;
      O[j][2] *= al_a;
      O[j][3] *= al_b;
      Ol[j][0] *= al_a;
      Ol[j][1] *= al_b;
      Ol[j][2] *= al_a;
      Ol[j][3] *= al_b;
    }
#pragma unroll
    for (int kt = 0; kt < 4; ++kt) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        uint32_t av[4];
        ldsm_x4_t(vbase + swt(16 * kt + ri + ((mi >> 1) ? 8 : 0), 2 * (2 * warp + j) + (mi & 1)), av);
        mma_bf16_16816(O[j], av, ph[kt]);
        mma_bf16_16816(Ol[j], av, pl[kt]);
      }
    }
    __syncthreads();   // every warp is done with this stage
    if (tid == 0 && i + kStages < n_tma) issue(i + kStages);

    // end of a super-chunk: its (M, L, O) per query (each warp its 32 dims)
    if ((c + 1) % kSuper == 0 || c + 1 == n_live) {
      float* ps = part + static_cast<size_t>(c / kSuper) * R * kPartStride;
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int d = 16 * (2 * warp + j) + g;
        if (qa < R) {
          ps[qa * kPartStride + d] = O[j][0] + Ol[j][0];
          ps[qa * kPartStride + d + 8] = O[j][2] + Ol[j][2];
        }
        if (qb < R) {
          ps[qb * kPartStride + d] = O[j][1] + Ol[j][1];
          ps[qb * kPartStride + d + 8] = O[j][3] + Ol[j][3];
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
  }
  if (aborted) {
    // a stage wait ran out: flag it and let the copies still in flight land, then take the
    // ticket as usual so that the counters stay consistent (the merged result is invalid)
    if (tid == 0) {
      atomicOr(a.err, ERR_WAIT_TIMEOUT);
      const int issued = min(n_tma, consumed + kStages);
      int never = 0;
      for (int i = consumed; i < issued; ++i)
        mbar_wait(&full[i % kStages], static_cast<uint32_t>(i / kStages) & 1u, &never, 100000000ull);
    }
    __syncthreads();
  }

  // the CTA that finishes last for (sequence, head) merges every query
  __threadfence();
  __syncthreads();
  const int n_busy = min(n_units, n_sup_live);   // CTAs of this (sequence, head) with work
  if (tid == 0) {
    int* ticket = a.tickets + b * kH + h;
    const int old = atomicAdd(ticket, 1);
    s_last = (old == n_busy - 1) ? 1 : 0;
    if (s_last) *ticket = 0;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    merge_all(a, b, h, R, p0, (n_live + kSuper - 1) / kSuper, reinterpret_cast<float*>(stages));
  }
}

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_chunk_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, attn_smem(2));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_chunk_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize, attn_smem(3));
  return e;
}

cudaError_t attention_launch(const AttnArgs& a_in, int B, cudaStream_t s) {
  // At most `unit` super-chunks per CTA: enough CTAs for about two waves of two per SM over the
  // largest context the pools allow.  Pure scheduling: the arithmetic of every super-chunk and
  // of the merge is the same for any assignment.
  AttnArgs a = a_in;
  const int n_super = (a.n_chunks + kSuper - 1) / kSuper;
  const long long target = 4ll * num_sms();
  const long long per_unit = static_cast<long long>(B) * kH;
  int unit = static_cast<int>((per_unit * n_super + target - 1) / target);
  if (unit < 1) unit = 1;
  if (unit > kUnitMaxSuper) unit = kUnitMaxSuper;
  a.unit = unit;
  const int n_units = (n_super + unit - 1) / unit;
  const long long ctas = static_cast<long long>(n_units) * kH * B;
  if (ctas <= 6ll * num_sms())
    return launch_pdl(attn_chunk_kernel<2>, dim3(n_units, kH, B), dim3(kAttnThreads), attn_smem(2), s, a);
  return launch_pdl(attn_chunk_kernel<3>, dim3(n_units, kH, B), dim3(kAttnThreads), attn_smem(3), s, a);
}

}  // namespace fm
