// Split-KV decode attention over a paged bf16 KV cache plus staged candidate rows.
//
// Each sequence has R queries at consecutive positions p0..p0+R-1 (the K+1 verify
// candidates, or one draft row).  Keys at positions < ctx_len live in the sequence's pages,
// keys at positions >= ctx_len in a staging buffer (candidates not yet committed).  The key
// range is cut into chunks of 128 positions fixed by absolute position; one CTA per
// (chunk, head, sequence) stages the chunk's K and V in shared memory with 16-byte
// cp.async copies, scores every (query, key) pair in fp32, and writes the chunk's
// (max, sum, unnormalised output) per query; the last chunk of a (sequence, head) to finish
// merges the chunks of each query in chunk order.  Masked keys contribute exact zeros, so a
// query's result is the same whether its key sits in a page or in staging and however many
// other queries share the chunk: greedy decoding (K = 0) and speculative verification see
// identical rows.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

constexpr int kCH = kAttnChunk;
constexpr int kAttnSmem = 2 * kCH * kHD * 2 + kMaxR * kHD * 4 + kMaxR * kCH * 4;
constexpr long long kStagedBit = 1ll << 62;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}

// Merge of the chunks of every query of (sequence b, head h), run by the last chunk CTA:
// query r combines chunks 0..floor(p_r/128) in chunk order, O = sum_c w_c acc_c / sum_c w_c l_c
// with w_c = 2^(m_c - max_c m_c).  The (m, l) pairs are staged in shared memory by all threads
// at once; the accumulator loads of the weighted sum are independent of each other.
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

__global__ void __launch_bounds__(128) attn_chunk_kernel(const AttnArgs a) {
  extern __shared__ __align__(16) uint8_t asmem[];
  bf16* sK = reinterpret_cast<bf16*>(asmem);               // [kCH][kHD], 16-byte chunks swizzled by row
  bf16* sV = sK + kCH * kHD;
  float* sq = reinterpret_cast<float*>(sV + kCH * kHD);    // [R][kHD]
  float* sp = sq + kMaxR * kHD;                           // [R][kCH] scores, then probabilities
  __shared__ long long s_base[kCH];                       // element offset of each key row (-1: none)
  __shared__ int s_last;

  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int R = a.R;
  const int slot = a.slots[b];
  const int sl = a.seq_len[slot];
  const int p0 = sl + a.qoff;
  const int last = p0 + R - 1;
  const int start = c * kCH;
  if (start > last || p0 < 0) return;
  const int nk = min(kCH, last + 1 - start);
  const int tid = threadIdx.x;

  // where each key row lives: a page of the pool (positions < ctx_len) or a staging row
  {
    const int j = tid;
    const int pos = start + j;
    long long off = -1;
    if (j < nk) {
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
  __syncthreads();

  // K, then V, rows of the chunk -> shared memory (zero-filled where there is no key)
  const long long v_pool = static_cast<long long>(kH) * a.page_size * kHD;
#pragma unroll 4
  for (int v = tid; v < kCH * 16; v += 128) {
    const int j = v >> 4, ch = v & 15;
    const long long off = s_base[j];
    const bf16* src = a.pool;
    int bytes = 0;
    if (off >= 0) {
      src = ((off & kStagedBit) ? a.stage + (off & (kStagedBit - 1)) : a.pool + off) + ch * 8;
      bytes = 16;
    }
    cp_async16(sK + j * kHD + ((ch ^ (j & 7)) * 8), src, bytes);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
#pragma unroll 4
  for (int v = tid; v < kCH * 16; v += 128) {
    const int j = v >> 4, ch = v & 15;
    const long long off = s_base[j];
    const bf16* src = a.pool;
    int bytes = 0;
    if (off >= 0) {
      src = ((off & kStagedBit) ? a.stage + (off & (kStagedBit - 1)) + a.stage_kv_stride : a.pool + off + v_pool) +
            ch * 8;
      bytes = 16;
    }
    cp_async16(sV + j * kHD + ((ch ^ (j & 7)) * 8), src, bytes);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");

  // queries, pre-scaled by log2(e) / sqrt(hd) so that softmax uses exp2
  const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(kHD));
  const int qrow0 = a.q_row0 ? a.q_row0[b] : b * R;
  for (int v = tid; v < R * kHD; v += 128) {
    const int r = v / kHD, d = v % kHD;
    sq[v] = a.q[(static_cast<size_t>(qrow0 + r) * kH + h) * kHD + d] * qscale;
  }
  asm volatile("cp.async.wait_group 1;" ::: "memory");   // K has landed; V may still be in flight
  __syncthreads();

  // scores: thread j owns key j of the chunk
  {
    const int j = tid;
    float s[kMaxR];
#pragma unroll
    for (int r = 0; r < kMaxR; ++r) s[r] = 0.f;
#pragma unroll 4
    for (int ch = 0; ch < 16; ++ch) {
      const uint4 raw = *reinterpret_cast<const uint4*>(sK + j * kHD + ((ch ^ (j & 7)) * 8));
      const bf16* kv = reinterpret_cast<const bf16*>(&raw);
      float kf[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) kf[u] = __bfloat162float(kv[u]);
#pragma unroll
      for (int r = 0; r < kMaxR; ++r) {
        if (r < R) {
          const float* qr = sq + r * kHD + ch * 8;
#pragma unroll
          for (int u = 0; u < 8; ++u) s[r] += qr[u] * kf[u];
        }
      }
    }
    const int pos = start + j;
#pragma unroll
    for (int r = 0; r < kMaxR; ++r)
      if (r < R) sp[r * kCH + j] = (j < nk && pos <= p0 + r) ? s[r] : -INFINITY;
  }
  __syncthreads();

  // per query: chunk max, probabilities (exact zeros where masked), sum
  const int warp = tid >> 5, lane = tid & 31;
  float* part = a.part + ((static_cast<size_t>(b) * kH + h) * a.n_chunks + c) * R * (kHD + 2);
  for (int r = warp; r < R; r += 4) {
    float x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = sp[r * kCH + lane + 32 * i];
    const float m = warp_max(fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])));
    float l = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float p = (m == -INFINITY || x[i] == -INFINITY) ? 0.f : exp2f(x[i] - m);
      sp[r * kCH + lane + 32 * i] = p;
      l += p;
    }
    l = warp_sum(l);
    if (lane == 0) {
      part[r * (kHD + 2) + kHD] = m;
      part[r * (kHD + 2) + kHD + 1] = l;
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();

  // P V: thread d owns output dim d
  {
    const int d = tid;
    float acc[kMaxR];
#pragma unroll
    for (int r = 0; r < kMaxR; ++r) acc[r] = 0.f;
    for (int j = 0; j < nk; ++j) {
      const float vv = __bfloat162float(sV[j * kHD + (((d >> 3) ^ (j & 7)) * 8) + (d & 7)]);
#pragma unroll
      for (int r = 0; r < kMaxR; ++r)
        if (r < R) acc[r] += sp[r * kCH + j] * vv;
    }
#pragma unroll
    for (int r = 0; r < kMaxR; ++r)
      if (r < R) part[r * (kHD + 2) + d] = acc[r];
  }

  // the last chunk of (sequence, head) to finish merges every query (atomic ticket, no wait)
  __threadfence();
  __syncthreads();
  const int n_live = last / kCH + 1;
  if (tid == 0) {
    int* ticket = a.tickets + b * kH + h;
    const int old = atomicAdd(ticket, 1);
    s_last = (old == n_live - 1) ? 1 : 0;
    if (s_last) *ticket = 0;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    merge_all(a, b, h, R, p0, n_live, reinterpret_cast<float*>(asmem));   // K/V tiles are no longer needed
  }
}

cudaError_t attention_prepare() {
  return cudaFuncSetAttribute(attn_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
}

cudaError_t attention_launch(const AttnArgs& a, int B, cudaStream_t s) {
  attn_chunk_kernel<<<dim3(a.n_chunks, kH, B), 128, kAttnSmem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace fm
