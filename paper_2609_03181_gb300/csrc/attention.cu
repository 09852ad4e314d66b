// Split-KV decode attention over a paged bf16 KV cache plus staged candidate rows.
//
// Each sequence has R queries at consecutive positions p0..p0+R-1 (the K+1 verify
// candidates, or one draft row).  Keys at positions < ctx_len live in the sequence's pages,
// keys at positions >= ctx_len in a staging buffer (candidates not yet committed).  The key
// range is cut into chunks of 64 positions fixed by absolute position.  For each chunk and
// query the kernel forms (max, sum, unnormalised output) of the chunk's softmax terms; a query's
// result is the chunk-ordered merge of its chunks.  Scores K q^T and outputs V^T p^T run on
// bf16 tensor cores (mma.sync m16n8k16, fp32 accumulation, queries padded to 8; p enters as a
// sum of two bf16 terms so the product keeps about 16 bits of it).
//
// Scheduling: one CTA per (unit of consecutive chunks, head, sequence); it resolves the
// page offsets of all its keys at once, then streams its chunks through two shared-memory
// stages (16-byte cp.async), computing one chunk while the next is in flight.  The CTA that
// finishes the last unit of a (sequence, head) merges (atomic ticket, no wait).  Masked keys
// contribute exact zeros and the chunk grouping does not enter the arithmetic, so a query's
// result is the same whether its keys sit in pages or in staging and however many queries or
// sequences share the launch: greedy decoding (K = 0) and speculative verification see
// identical rows.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

constexpr int kCH = kAttnChunk;                  // keys per chunk (64)
constexpr int kUnitMax = 16;                     // most chunks one CTA streams
constexpr int kAttnThreads = 128;
constexpr int kStageBytes = 2 * kCH * kHD * 2;   // K and V of one chunk: 32 KB
constexpr int kAttnSmem = 2 * kStageBytes + kMaxR * kHD * 2 + 2 * kMaxR * kCH * 2 + kMaxR * kCH * 4;
constexpr long long kStagedBit = 1ll << 62;

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
// Byte offset of 16-byte chunk `ch` of row `row` in a tile of 256-byte rows (a K or V row of
// 128 bf16), chunks swizzled by row: conflict-free for ldmatrix and for row-wise cp.async.
__device__ __forceinline__ uint32_t swz(int row, int ch) { return row * 256 + ((ch ^ (row & 7)) << 4); }
// Same for the 128-byte rows of the probability tiles (64 keys per query).
__device__ __forceinline__ uint32_t swz_p(int row, int ch) { return row * 128 + ((ch ^ (row & 7)) << 4); }

// Merge of the chunks of every query of (sequence b, head h), run by the CTA that finishes the
// last unit: query r combines chunks 0..floor(p_r/64) in chunk order,
// O = sum_c w_c acc_c / sum_c w_c l_c with w_c = 2^(m_c - max_c m_c).  The (m, l) pairs are
// staged in shared memory by all threads at once; the accumulator loads are independent.
__device__ __forceinline__ void merge_all(const AttnArgs& a, int b, int h, int R, int p0, int n_live, float* smem) {
  const float* part = a.part + (static_cast<size_t>(b) * kH + h) * a.n_chunks * R * (kHD + 2);
  float* sm = smem;                      // [n_live * R] chunk max, then weight
  float* sl = smem + n_live * R;         // [n_live * R] chunk sum
  float* sL = sl + n_live * R;           // [R] total weight
  for (int i = threadIdx.x; i < n_live * R; i += blockDim.x) {
    const float* pc = part + static_cast<size_t>(i) * (kHD + 2);
    sm[i] = __ldcg(&pc[kHD]);
    sl[i] = __ldcg(&pc[kHD + 1]);
  }
  __syncthreads();
  if (threadIdx.x < R) {
    const int r = threadIdx.x, lastc = (p0 + r) / kCH;
    float M = -INFINITY;
    for (int c = 0; c <= lastc; ++c) M = fmaxf(M, sm[c * R + r]);
    float L = 0.f;
    for (int c = 0; c <= lastc; ++c) {
      const float mc = sm[c * R + r];
      const float w = (mc == -INFINITY) ? 0.f : exp2f(mc - M);
      sm[c * R + r] = w;
      L += sl[c * R + r] * w;
    }
    sL[r] = L;
  }
  __syncthreads();
  const int d = threadIdx.x;
  if (d < kHD) {
    for (int r = 0; r < R; ++r) {
      const int lastc = (p0 + r) / kCH;
      float O = 0.f;
      int c = 0;
      for (; c + 4 <= lastc + 1; c += 4) {
        float x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) x[u] = __ldcg(&part[(static_cast<size_t>(c + u) * R + r) * (kHD + 2) + d]);
#pragma unroll
        for (int u = 0; u < 4; ++u) O += x[u] * sm[(c + u) * R + r];
      }
      for (; c <= lastc; ++c) O += __ldcg(&part[(static_cast<size_t>(c) * R + r) * (kHD + 2) + d]) * sm[c * R + r];
      a.out[(static_cast<size_t>(b) * a.out_row_stride_seq + r) * (kH * kHD) + h * kHD + d] =
          __float2bfloat16(O / sL[r]);
    }
  }
}

// Copies the K and V rows j0..j0+63 of the unit into a stage as one cp.async group; rows
// without a key are zero-filled.
__device__ __forceinline__ void issue_chunk(const AttnArgs& a, const long long* s_base, int j0, uint8_t* stage) {
  const long long v_pool = static_cast<long long>(kH) * a.page_size * kHD;
  uint8_t* sK = stage;
  uint8_t* sV = stage + kCH * kHD * 2;
#pragma unroll 4
  for (int v = threadIdx.x; v < kCH * 16; v += kAttnThreads) {
    const int j = v >> 4, ch = v & 15;
    const long long off = s_base[j0 + j];
    const bf16* srck = a.pool;
    const bf16* srcv = a.pool;
    int bytes = 0;
    if (off >= 0) {
      if (off & kStagedBit) {
        srck = a.stage + (off & (kStagedBit - 1)) + ch * 8;
        srcv = srck + a.stage_kv_stride;
      } else {
        srck = a.pool + off + ch * 8;
        srcv = srck + v_pool;
      }
      bytes = 16;
    }
    cp_async16(sK + swz(j, ch), srck, bytes);
    cp_async16(sV + swz(j, ch), srcv, bytes);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

__global__ void __launch_bounds__(kAttnThreads) attn_chunk_kernel(const AttnArgs a) {
  extern __shared__ __align__(128) uint8_t asmem[];
  uint8_t* stages = asmem;                                   // [2][K 16 KB | V 16 KB]
  uint8_t* sQ = asmem + 2 * kStageBytes;                     // [8 queries][128 dims] bf16
  uint8_t* sP = sQ + kMaxR * kHD * 2;                        // [8][64 keys] bf16 p, high part
  uint8_t* sPl = sP + kMaxR * kCH * 2;                       // [8][64 keys] bf16 p - high part
  float* sS = reinterpret_cast<float*>(sPl + kMaxR * kCH * 2);   // [8][64] fp32 scores
  __shared__ long long s_base[kUnitMax * kCH];               // element offset of every key row of the unit
  __shared__ int s_last;
  pdl_trigger();
  pdl_wait();

  const int u = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int R = a.R;
  const int slot = a.slots[b];
  if (slot < 0 || slot >= a.n_slots) {   // every CTA of the sequence leaves; no ticket, no merge
    if (u == 0 && h == 0 && threadIdx.x == 0) atomicOr(a.err, ERR_SLOT_RANGE);
    return;
  }
  const int sl = a.seq_len[slot];
  const int p0 = sl + a.qoff;
  const int last = p0 + R - 1;
  if (p0 < 0) return;
  const int n_live = last / kCH + 1;                         // chunks holding keys 0..last
  const int c0 = u * a.unit;
  if (c0 >= n_live) return;
  const int c1 = min(c0 + a.unit, n_live);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t4 = lane & 3, mi = lane >> 3, ri = lane & 7;

  // page offsets of every key of the unit, all lookups in flight at once
  for (int j = tid; j < (c1 - c0) * kCH; j += kAttnThreads) {
    const int pos = c0 * kCH + j;
    long long off = -1;
    if (pos <= last) {
      if (pos < sl) {
        const int pi = pos / a.page_size;
        const int page = (pi < a.max_pages) ? a.block_table[slot * a.max_pages + pi] : -1;
        if (page >= 0 && page < a.n_pages)
          off = ((static_cast<long long>(page) * 2 * kH + h) * a.page_size + pos % a.page_size) * kHD;
        else
          atomicOr(a.err, ERR_PAGE_RANGE);
      } else {
        off = kStagedBit | (b * a.stage_seq_stride + static_cast<long long>(pos - sl) * a.stage_row_stride +
                            static_cast<long long>(h) * kHD);
      }
    }
    s_base[j] = off;
  }
  // queries (bf16, as the QKV epilogue stored them); rows R..7 are zero
  const int qrow0 = a.q_row0 ? a.q_row0[b] : b * R;
  {
    const int q = tid >> 4, ch = tid & 15;   // 8 queries x 16 chunks of 16 bytes
    uint4 val = make_uint4(0, 0, 0, 0);
    if (q < R) val = *reinterpret_cast<const uint4*>(a.q + (static_cast<size_t>(qrow0 + q) * kH + h) * kHD + ch * 8);
    *reinterpret_cast<uint4*>(sQ + swz(q, ch)) = val;
  }
  __syncthreads();
  issue_chunk(a, s_base, 0, stages);

  const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(kHD));   // log2(e) / sqrt(hd)
  const uint32_t qbase = smem_u32(sQ), pbase = smem_u32(sP), plbase = smem_u32(sPl);
  int st = 0;
  for (int c = c0; c < c1; ++c) {
    const bool has_next = c + 1 < c1;
    if (has_next) {
      issue_chunk(a, s_base, (c + 1 - c0) * kCH, stages + (st ^ 1) * kStageBytes);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    const uint32_t kbase = smem_u32(stages + st * kStageBytes);
    const uint32_t vbase = kbase + kCH * kHD * 2;
    const int start = c * kCH;
    const int nk = min(kCH, last + 1 - start);

    // S^T[key][query] = K Q^T: warp w owns keys 16w..16w+15, 8 k-steps of 16 dims
    {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        uint32_t bq[2], ak[4];
        ldsm_x2(qbase + swz(ri, 2 * ks + (mi & 1)), bq);
        const int key = warp * 16 + ri + ((mi & 1) ? 8 : 0);
        ldsm_x4(kbase + swz(key, 2 * ks + (mi >> 1)), ak);
        mma_bf16_16816(acc, ak, bq);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = warp * 16 + g + ((e >> 1) ? 8 : 0);
        const int q = 2 * t4 + (e & 1);
        const bool vis = q < R && key < nk && start + key <= p0 + q;
        sS[q * kCH + key] = vis ? acc[e] * scale : -INFINITY;
      }
    }
    __syncthreads();

    // per query: chunk max, p = hi + lo (exact zeros where masked), sum
    float* part = a.part + ((static_cast<size_t>(b) * kH + h) * a.n_chunks + c) * R * (kHD + 2);
    for (int q = warp; q < kMaxR; q += 4) {
      const float x0 = sS[q * kCH + lane], x1 = sS[q * kCH + lane + 32];
      const float m = warp_max(fmaxf(x0, x1));
      float l = 0.f;
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int key = lane + 32 * i;
        const float x = i ? x1 : x0;
        const float p = (m == -INFINITY || x == -INFINITY) ? 0.f : exp2f(x - m);
        const bf16 hi = __float2bfloat16(p);
        const bf16 lo = __float2bfloat16(p - __bfloat162float(hi));
        *reinterpret_cast<bf16*>(sP + swz_p(q, key >> 3) + (key & 7) * 2) = hi;
        *reinterpret_cast<bf16*>(sPl + swz_p(q, key >> 3) + (key & 7) * 2) = lo;
        l += p;
      }
      l = warp_sum(l);
      if (lane == 0 && q < R) {
        part[q * (kHD + 2) + kHD] = m;
        part[q * (kHD + 2) + kHD + 1] = l;
      }
    }
    __syncthreads();

    // O^T[dim][query] = V^T P^T: warp w owns dims 32w..32w+31 (two tiles), 4 k-steps of 16 keys
    {
      float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int ks = 0; ks < kCH / 16; ++ks) {
        uint32_t bp[2], bl[2];
        ldsm_x2(pbase + swz_p(ri, 2 * ks + (mi & 1)), bp);
        ldsm_x2(plbase + swz_p(ri, 2 * ks + (mi & 1)), bl);
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          uint32_t av[4];
          const int key = ks * 16 + ri + ((mi >> 1) ? 8 : 0);
          ldsm_x4_t(vbase + swz(key, (warp * 32 + mt * 16) / 8 + (mi & 1)), av);
          mma_bf16_16816(acc[mt], av, bp);
          mma_bf16_16816(acc[mt], av, bl);
        }
      }
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int d = warp * 32 + mt * 16 + g + ((e >> 1) ? 8 : 0);
          const int q = 2 * t4 + (e & 1);
          if (q < R) part[q * (kHD + 2) + d] = acc[mt][e];
        }
    }
    __syncthreads();   // this stage and the score/probability tiles are reused next
    st ^= 1;
  }

  // the CTA that finishes the last unit of (sequence, head) merges every query
  __threadfence();
  __syncthreads();
  const int n_units = (n_live + a.unit - 1) / a.unit;
  if (tid == 0) {
    int* ticket = a.tickets + b * kH + h;
    const int old = atomicAdd(ticket, 1);
    s_last = (old == n_units - 1) ? 1 : 0;
    if (s_last) *ticket = 0;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    merge_all(a, b, h, R, p0, n_live, reinterpret_cast<float*>(stages));   // the K/V stages are free
  }
}

cudaError_t attention_prepare() {
  return cudaFuncSetAttribute(attn_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
}

cudaError_t attention_launch(const AttnArgs& a_in, int B, cudaStream_t s) {
  // Chunks per CTA: enough CTAs for about three resident per SM over the largest context the
  // pools allow.  Pure scheduling: the arithmetic of every chunk and of the merge is the same
  // for any grouping.
  AttnArgs a = a_in;
  const long long target = 3ll * num_sms();
  const long long per_unit = static_cast<long long>(B) * kH;
  int unit = static_cast<int>((per_unit * a.n_chunks + target - 1) / target);
  if (unit < 1) unit = 1;
  if (unit > kUnitMax) unit = kUnitMax;
  a.unit = unit;
  const int n_units = (a.n_chunks + unit - 1) / unit;
  return launch_pdl(attn_chunk_kernel, dim3(n_units, kH, B), dim3(kAttnThreads), kAttnSmem, s, a);
}

}  // namespace fm
