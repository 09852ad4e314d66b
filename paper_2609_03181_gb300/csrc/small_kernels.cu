// Latency-bound kernels of the FastMTP step: embedding + RMSNorm, RMSNorm, router
// (norm, logits, softmax, top-6), token permute/scatter by expert, MoE combine (+ the next
// RMSNorm), the KV commit, and the glue of the draft chain.  Every reduction runs in a fixed
// order, so a row's result never depends on the other rows of the batch.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace fm {

// Sum over an NT-thread block in a fixed order (warp trees, then warps in index order).
template <int NT>
__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float s = red[0];
#pragma unroll
  for (int i = 1; i < NT / 32; ++i) s += red[i];
  __syncthreads();
  return s;
}
__device__ __forceinline__ float block128_sum(float v, float* red) { return block_sum<128>(v, red); }

// x (kD/NT values per thread, element i = tid + NT*k) -> bf16 x * rsqrt(mean(x^2) + eps) * gain
template <int NT>
__device__ __forceinline__ void norm_row_store_t(const float (&x)[kD / NT], const bf16* gain, float eps, bf16* out,
                                                 float* red) {
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kD / NT; ++k) ss += x[k] * x[k];
  ss = block_sum<NT>(ss, red);
  const float inv = rsqrtf(ss / kD + eps);
#pragma unroll
  for (int k = 0; k < kD / NT; ++k) {
    const int i = threadIdx.x + NT * k;
    out[i] = __float2bfloat16(x[k] * inv * __bfloat162float(gain[i]));
  }
}
__device__ __forceinline__ void norm_row_store(const float (&x)[10], const bf16* gain, float eps, bf16* out,
                                               float* red) {
  norm_row_store_t<128>(x, gain, eps, out, red);
}

// ---------------------------------------------------------------- embedding + norm
__global__ void __launch_bounds__(128) embed_norm_kernel(const int* cand, int R, const int* slots, const int* pending,
                                                         const int* seq_len, const bf16* embed, int vocab,
                                                         const bf16* gain, float eps, float* h, bf16* xn, int* pos,
                                                         long long* kv_rowoff, int stage_R, int n_slots, int* err) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[4];
  const int row = blockIdx.x, b = row / R, r = row % R;
  const int slot = slots[b];
  const bool slot_ok = slot >= 0 && slot < n_slots;
  if (!slot_ok && r == 0 && threadIdx.x == 0) atomicOr(err, ERR_SLOT_RANGE);
  int tok = cand[row];
  if (tok < 0 || tok >= vocab) {
    if (threadIdx.x == 0) atomicOr(err, ERR_TOKEN_RANGE);
    tok = 0;
  }
  if (slot_ok && r == 0 && tok != pending[slot] && threadIdx.x == 0) atomicOr(err, ERR_PENDING);
  const bf16* e = embed + static_cast<size_t>(tok) * kD;
  float x[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) {
    const int i = threadIdx.x + 128 * k;
    x[k] = __bfloat162float(e[i]);
    h[static_cast<size_t>(row) * kD + i] = x[k];
  }
  norm_row_store(x, gain, eps, xn + static_cast<size_t>(row) * kD, red);
  if (threadIdx.x == 0) {
    pos[row] = (slot_ok ? seq_len[slot] : 0) + r;
    kv_rowoff[row] = static_cast<long long>(b * stage_R + r) * 2 * kH * kHD;
  }
}

cudaError_t embed_norm_launch(const int* cand, int B, int R, const int* slots, const int* pending,
                              const int* seq_len, const bf16* embed, int vocab, const bf16* gain, float eps,
                              float* h, bf16* xn, int* pos, long long* kv_rowoff, int stage_R, int n_slots,
                              int* err, cudaStream_t s) {
  return launch_pdl(embed_norm_kernel, dim3(B * R), dim3(128), 0, s, cand, R, slots, pending, seq_len, embed, vocab, gain,
                    eps, h, xn, pos, kv_rowoff, stage_R, n_slots, err);
}

// ---------------------------------------------------------------- RMSNorm
__global__ void __launch_bounds__(128) rmsnorm_kernel(const float* x, const bf16* gain, float eps, bf16* out) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[4];
  const size_t row = blockIdx.x;
  float v[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) v[k] = x[row * kD + threadIdx.x + 128 * k];
  norm_row_store(v, gain, eps, out + row * kD, red);
}

cudaError_t rmsnorm_launch(const float* x, int rows, const bf16* gain, float eps, bf16* out, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(128), 0, s, x, gain, eps, out);
}

// ---------------------------------------------------------------- router + expert grouping
// RR rows per CTA: 1 for small batches (latency), 4 above 128 rows (the 64 x 1280 router
// matrix is then read once per four rows).  Per row:
// RMSNorm of the residual row -> xn (bf16, also the experts' input); logits of the 64 experts
// from the bf16 row, fp32 softmax, top-6 by probability (lower id on ties).  Every row's
// arithmetic is the same whatever rows share its CTA.
//
// Then the CTA that finishes last (atomic ticket, no wait) groups the (token, slot) pairs of
// the layer by expert: routed rows of expert e take act rows offs[e] .. offs[e+1]-1 in token
// order (rank from a per-expert token bitmap and its prefix popcounts); the two shared experts
// follow with all T tokens each.  It writes the destination row of every pair, the sorted
// token/slot lists, the GEMM work lists (row tiles of at most 64 rows, so every grouped launch
// runs the deep 8-stage weight pipeline) and the expert counters.
constexpr int kRouterRows = 4;
constexpr int kMaxT = 2048;
constexpr int kMaxW = kMaxT / 32;

__device__ __forceinline__ void group_by_expert(const RouteArgs& a, int* gsm) {
  const int T = a.T, W = (T + 31) / 32, T6 = T * kTopK, tid = threadIdx.x;
  int* s_idx = gsm;                       // [T*6]
  unsigned* bits = reinterpret_cast<unsigned*>(s_idx + T6);   // [64][W]
  int* pre = reinterpret_cast<int*>(bits + kE * W);          // [64][W]
  int* cnt = pre + kE * W;                // [66]
  int* offs = cnt + kE + kShared;         // [67]
  int* ibase = offs + kE + kShared + 1;   // [67] gate_up item offsets
  int* dbase = ibase + kE + kShared + 1;  // [67]
  for (int p = tid; p < T6; p += blockDim.x) s_idx[p] = __ldcg(a.idx + p);
  for (int p = tid; p < kE * W; p += blockDim.x) bits[p] = 0u;
  __syncthreads();
  for (int p = tid; p < T6; p += blockDim.x) {
    const int t = p / kTopK, e = s_idx[p];
    atomicOr(&bits[e * W + (t >> 5)], 1u << (t & 31));
  }
  __syncthreads();
  if (tid < kE) {
    int run = 0;
    for (int w = 0; w < W; ++w) {
      pre[tid * W + w] = run;
      run += __popc(bits[tid * W + w]);
    }
    cnt[tid] = run;
  } else if (tid < kE + kShared) {
    cnt[tid] = T;
  }
  __syncthreads();
  if (tid < 32) {
    // exclusive prefix sums over the 66 experts (three per lane, lanes in order)
    int c3[3], m3[3];
    int sc = 0, sm = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const int e = tid * 3 + k;
      c3[k] = (e < kE + kShared) ? cnt[e] : 0;
      m3[k] = (c3[k] + kExpertTileRows - 1) / kExpertTileRows;
      sc += c3[k];
      sm += m3[k];
    }
    int ic = sc, im = sm;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int xc = __shfl_up_sync(0xffffffffu, ic, o), xm = __shfl_up_sync(0xffffffffu, im, o);
      if (tid >= o) {
        ic += xc;
        im += xm;
      }
    }
    int rc = ic - sc, rm = im - sm;   // exclusive
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const int e = tid * 3 + k;
      if (e <= kE + kShared) {
        offs[e] = rc;
        ibase[e] = rm * (kI / 64);
        dbase[e] = rm * (kD / 128);
      }
      rc += c3[k];
      rm += m3[k];
    }
    if (tid == 31) {
      a.n_items[0] = im * (kI / 64);
      a.n_items[1] = im * (kD / 128);
    }
  }
  __syncthreads();
  for (int p = tid; p < T6; p += blockDim.x) {
    const int t = p / kTopK, sl = p % kTopK, e = s_idx[p];
    const int dst = offs[e] + pre[e * W + (t >> 5)] + __popc(bits[e * W + (t >> 5)] & ((1u << (t & 31)) - 1u));
    a.dst_row[p] = dst;
    a.sorted_tok[dst] = t;
    a.sorted_slot[dst] = sl;
  }
  for (int p = tid; p < kShared * T; p += blockDim.x) {
    const int j = p / T, t = p % T;
    a.sorted_tok[offs[kE + j] + t] = t;
    a.sorted_slot[offs[kE + j] + t] = kTopK + j;
  }
  if (tid < kE + kShared) {
    const int e = tid, n = cnt[e];
    if (e < kE) a.counts[e] = n;
    if (n > 0) {
      atomicAdd(&a.expert_ctr[0], 1ull);
      atomicAdd(&a.expert_ctr[1], static_cast<unsigned long long>(n));
    }
    const int mt = (n + kExpertTileRows - 1) / kExpertTileRows;
    for (int m = 0; m < mt; ++m) {
      const int rows = min(kExpertTileRows, n - kExpertTileRows * m);
      const int out_row = offs[e] + kExpertTileRows * m;
      const int b_row_gu = (e < kE) ? out_row : kExpertTileRows * m;   // shared experts read xn rows directly
      for (int nt = 0; nt < kI / 64; ++nt)
        a.items_gu[ibase[e] + m * (kI / 64) + nt] = make_int4(e | (nt << 16), b_row_gu, out_row, rows);
      for (int nt = 0; nt < kD / 128; ++nt)
        a.items_dn[dbase[e] + m * (kD / 128) + nt] = make_int4(e | (nt << 16), out_row, out_row, rows);
    }
  }
}

template <int RR>
__global__ void __launch_bounds__(256) router_kernel(const __grid_constant__ RouteArgs a) {
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the first four experts of this warp's eight: router weights are never written by earlier
  // kernels, so their loads go out before the wait for the previous kernel
  uint4 raw[4][5];
  auto load_group = [&](int e0) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int c = 0; c < 5; ++c)
        raw[q][c] = *reinterpret_cast<const uint4*>(a.wr + static_cast<size_t>(e0 + q) * kD + c * 256 + lane * 8);
  };
  load_group(warp * 8);
  pdl_wait();
  constexpr int NT = 256, EPT = kD / NT;
  __shared__ float red[NT / 32][RR];
  __shared__ __align__(16) float xs[RR][kD];
  __shared__ float lg[RR][kE];
  __shared__ float sp[RR][kE];
  __shared__ int s_last;
  extern __shared__ int gsm[];
  const int t0 = blockIdx.x * RR;
  const int nr = min(RR, a.T - t0);
  {
    float v[RR][EPT];
    float ss[RR];
#pragma unroll
    for (int r = 0; r < RR; ++r) {
#pragma unroll
      for (int k = 0; k < EPT; ++k) v[r][k] = (r < nr) ? a.h[static_cast<size_t>(t0 + r) * kD + threadIdx.x + NT * k] : 0.f;
      ss[r] = 0.f;
#pragma unroll
      for (int k = 0; k < EPT; ++k) ss[r] += v[r][k] * v[r][k];
      ss[r] = warp_sum(ss[r]);
    }
    if (lane == 0)
#pragma unroll
      for (int r = 0; r < RR; ++r) red[warp][r] = ss[r];
    __syncthreads();
#pragma unroll
    for (int r = 0; r < RR; ++r) {
      if (r >= nr) break;
      float tot = red[0][r];
#pragma unroll
      for (int w = 1; w < NT / 32; ++w) tot += red[w][r];
      const float inv = rsqrtf(tot / kD + a.eps);
      bf16* xo = a.xn + static_cast<size_t>(t0 + r) * kD;
#pragma unroll
      for (int k = 0; k < EPT; ++k) {
        const int i = threadIdx.x + NT * k;
        const bf16 rb = __float2bfloat16(v[r][k] * inv * __bfloat162float(a.gain[i]));
        xo[i] = rb;
        xs[r][i] = __bfloat162float(rb);   // the rounded row, as the experts see it
      }
    }
  }
  __syncthreads();
  for (int e0 = warp * 8; e0 < warp * 8 + 8; e0 += 4) {
    // four experts at a time: 20 independent 16-byte weight loads in flight per lane, each
    // weight used for every row of the CTA
    if (e0 != warp * 8) load_group(e0);
#pragma unroll
    for (int r = 0; r < RR; ++r) {
      if (r >= nr) break;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float acc = 0.f;
#pragma unroll
        for (int c = 0; c < 5; ++c) {
          const int i0 = c * 256 + lane * 8;
          const bf16* wv = reinterpret_cast<const bf16*>(&raw[q][c]);
#pragma unroll
          for (int u = 0; u < 8; ++u) acc += __bfloat162float(wv[u]) * xs[r][i0 + u];
        }
        acc = warp_sum(acc);
        if (lane == 0) lg[r][e0 + q] = acc + (a.bias ? a.bias[e0 + q] : 0.f);
      }
    }
  }
  __syncthreads();
  if (warp < nr) {
    const int r = warp;
    const size_t t = t0 + r;
    const float l0 = lg[r][lane], l1 = lg[r][lane + 32];
    const float m = warp_max(fmaxf(l0, l1));
    const float e0 = expf(l0 - m), e1 = expf(l1 - m);
    const float sum = warp_sum(e0 + e1);
    float p0 = e0 / sum, p1 = e1 / sum;
    // a non-finite row still selects six distinct valid experts (NaN ranks below every number)
    const bool bad = __any_sync(0xffffffffu, !(p0 == p0) || !(p1 == p1));
    if (bad) {
      if (lane == 0) atomicOr(a.err, ERR_NONFINITE);
      if (!(p0 == p0)) p0 = -1.f;
      if (!(p1 == p1)) p1 = -1.f;
    }
    // top-6: the rank of each expert among the 64 (a higher probability, or an equal one with a
    // lower id, ranks ahead) -- the experts of rank 0..5 are the selection, in that order
    sp[r][lane] = p0;
    sp[r][lane + 32] = p1;
    __syncwarp();
    int rk0 = 0, rk1 = 0;
#pragma unroll 16
    for (int j = 0; j < kE; ++j) {
      const float pj = sp[r][j];
      rk0 += better(pj, j, p0, lane) ? 1 : 0;
      rk1 += better(pj, j, p1, lane + 32) ? 1 : 0;
    }
    if (rk0 < kTopK) {
      a.idx[t * kTopK + rk0] = lane;
      a.gate[t * kTopK + rk0] = p0;
    }
    if (rk1 < kTopK) {
      a.idx[t * kTopK + rk1] = lane + 32;
      a.gate[t * kTopK + rk1] = p1;
    }
  }
  // the last CTA to finish groups the layer's pairs by expert
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int old = atomicAdd(a.ticket, 1);
    s_last = (old == static_cast<int>(gridDim.x) - 1) ? 1 : 0;
    if (s_last) *a.ticket = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  group_by_expert(a, gsm);
}

cudaError_t router_prepare() {
  const int smem = static_cast<int>(sizeof(int) * (kMaxT * kTopK + 2 * kE * kMaxW + 4 * 67));
  cudaError_t e = cudaFuncSetAttribute(router_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(router_kernel<kRouterRows>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return e;
}

cudaError_t router_launch(const RouteArgs& a, cudaStream_t s) {
  if (a.T > kMaxT || a.T < 1) return cudaErrorInvalidValue;
  const int W = (a.T + 31) / 32;
  const size_t smem = sizeof(int) * (static_cast<size_t>(a.T) * kTopK + 2 * kE * W + 4 * (kE + kShared + 1));
  if (a.T <= 128) return launch_pdl(router_kernel<1>, dim3(a.T), dim3(256), smem, s, a);
  return launch_pdl(router_kernel<kRouterRows>, dim3((a.T + kRouterRows - 1) / kRouterRows), dim3(256), smem, s, a);
}

// ---------------------------------------------------------------- permute (row gather)
// Copies the normalised row of every routed (token, slot) pair to its expert-sorted row of
// the experts' input, one warp per pair, all of a row's loads issued before its stores.
__global__ void __launch_bounds__(256) permute_kernel(const int* dst_row, int T6, const bf16* xn, bf16* xs) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * 8 + warp, nw = gridDim.x * 8;
  for (int p = gw; p < T6; p += nw) {
    const int t = p / kTopK, dst = dst_row[p];
    const uint4* src = reinterpret_cast<const uint4*>(xn + static_cast<size_t>(t) * kD);
    uint4* d = reinterpret_cast<uint4*>(xs + static_cast<size_t>(dst) * kD);
    uint4 v[kD / 8 / 32];
#pragma unroll
    for (int c = 0; c < kD / 8 / 32; ++c) v[c] = src[lane + 32 * c];
#pragma unroll
    for (int c = 0; c < kD / 8 / 32; ++c) d[lane + 32 * c] = v[c];
  }
}

cudaError_t permute_launch(const int* dst_row, int T, const bf16* xn, bf16* x_sorted, cudaStream_t s) {
  const int pairs = T * kTopK;
  int grid = (pairs + 7) / 8;     // one warp per (token, slot) row copy
  if (grid > 1024) grid = 1024;
  if (grid < 1) grid = 1;
  return launch_pdl(permute_kernel, dim3(grid), dim3(256), 0, s, dst_row, pairs, xn, x_sorted);
}

// ---------------------------------------------------------------- combine
// h += sum_{s<6} gate_s * y_s + y_shared0 + y_shared1 (fixed slot order), then RMSNorm -> out.
__global__ void __launch_bounds__(256) combine_kernel(float* h, const float* y, const float* gate, const bf16* gain,
                                                      float eps, bf16* out) {
  pdl_trigger();
  pdl_wait();
  constexpr int NT = 256, EPT = kD / NT;
  __shared__ float red[NT / 32];
  const size_t t = blockIdx.x;
  float g[kTopK];
#pragma unroll
  for (int s = 0; s < kTopK; ++s) g[s] = gate[t * kTopK + s];
  float ys[EPT][kSlots];
#pragma unroll
  for (int k = 0; k < EPT; ++k)
#pragma unroll
    for (int s = 0; s < kSlots; ++s) ys[k][s] = y[(t * kSlots + s) * kD + threadIdx.x + NT * k];
  float x[EPT];
#pragma unroll
  for (int k = 0; k < EPT; ++k) x[k] = h[t * kD + threadIdx.x + NT * k];   // all loads before any store
#pragma unroll
  for (int k = 0; k < EPT; ++k) {
    float acc = 0.f;
#pragma unroll
    for (int s = 0; s < kTopK; ++s) acc += g[s] * ys[k][s];
    acc += ys[k][kTopK];
    acc += ys[k][kTopK + 1];
    x[k] += acc;
    h[t * kD + threadIdx.x + NT * k] = x[k];
  }
  norm_row_store_t<NT>(x, gain, eps, out + t * kD, red);
}

cudaError_t combine_launch(float* h, const float* y, const float* gate, int T, const bf16* gain, float eps,
                           bf16* out, cudaStream_t s) {
  return launch_pdl(combine_kernel, dim3(T), dim3(256), 0, s, h, y, gate, gain, eps, out);
}

// ---------------------------------------------------------------- KV commit
// Appends the staged K/V of candidates 0..m of each sequence to its pages (16-byte
// vectors), advances the slot, writes the committed tokens and queues the m+1 new rows
// (base states b and next tokens) for the draft head.  The rejected tail stays in the
// staging buffer and is overwritten by the next verify.  One CTA per (sequence, layer); the
// last CTA of a sequence to finish its copies (atomic ticket) updates the sequence's state,
// after every CTA of that sequence has read the old length.
__global__ void __launch_bounds__(256) commit_kernel(int R, int stage_R, int Bmax, const int* slots, const int* m_ws,
                                                     const int* vtok, const int* cand, const bf16* stage, bf16* pool,
                                                     int L, int n_pages, int page_size, const int* block_table,
                                                     int max_pages, int* seq_len, int* pending, const bf16* b_ws,
                                                     bf16* draft_b, int* draft_tok, int* draft_n, int* committed,
                                                     int* n_committed, int* tickets, int* err) {
  pdl_trigger();
  pdl_wait();
  __shared__ int s_last;
  const int b = blockIdx.x, l = blockIdx.y, slot = slots[b];
  if (slot < 0 || slot >= Bmax) {   // every CTA of the sequence skips it, none takes the ticket
    if (threadIdx.x == 0 && l == 0) atomicOr(err, ERR_SLOT_RANGE);
    return;
  }
  int m = m_ws[b];
  if (m < 0 || m >= R) {   // an accept length the verify cannot produce: flag it, commit the bonus only
    if (threadIdx.x == 0 && l == 0) atomicOr(err, ERR_TOKEN_RANGE);
    m = 0;
  }
  const int c = seq_len[slot];
  constexpr int kVec = kHD / 8;   // 16-byte vectors per head row
  constexpr int kBatch = 8;       // copies whose loads are issued before their stores
  const int total = (m + 1) * 2 * kH * kVec;
  for (int v0 = threadIdx.x; v0 < total; v0 += blockDim.x * kBatch) {
    uint4 val[kBatch];
    uint4* dst[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      dst[u] = nullptr;
      const int v = v0 + u * blockDim.x;
      if (v >= total) continue;
      int t = v;
      const int vec = t % kVec; t /= kVec;
      const int h = t % kH; t /= kH;
      const int kv = t % 2;
      const int r = t / 2;
      const int pos = c + r;
      const int pi = pos / page_size;
      const int page = (pi < max_pages) ? block_table[slot * max_pages + pi] : -1;
      if (page < 0 || page >= n_pages) {
        atomicOr(err, ERR_PAGE_RANGE);
        continue;
      }
      val[u] = reinterpret_cast<const uint4*>(
          stage + ((((static_cast<size_t>(l) * Bmax + b) * stage_R + r) * 2 + kv) * kH + h) * kHD)[vec];
      dst[u] = reinterpret_cast<uint4*>(
                   pool + ((((static_cast<size_t>(l) * n_pages + page) * 2 + kv) * kH + h) * page_size + pos % page_size) *
                              kHD) + vec;
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u)
      if (dst[u] != nullptr) *dst[u] = val[u];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&tickets[b], 1) == L - 1;
  }
  __syncthreads();
  if (!s_last) return;
  // queue the new rows for the draft head: b_p and x_{p+1}
  for (int v = threadIdx.x; v < (m + 1) * (kD / 8); v += blockDim.x) {
    const int r = v / (kD / 8), c8 = v % (kD / 8);
    reinterpret_cast<uint4*>(draft_b + (static_cast<size_t>(slot) * kMaxR + r) * kD)[c8] =
        reinterpret_cast<const uint4*>(b_ws + static_cast<size_t>(b * R + r) * kD)[c8];
  }
  if (threadIdx.x < R) {
    const int r = threadIdx.x;
    const int tok = (r < m) ? cand[b * R + r + 1] : (r == m ? vtok[b * R + m] : -1);
    committed[b * R + r] = tok;
    if (r <= m) draft_tok[slot * kMaxR + r] = tok;
  }
  if (threadIdx.x == 0) {
    tickets[b] = 0;
    n_committed[b] = m + 1;
    pending[slot] = vtok[b * R + m];
    seq_len[slot] = c + m + 1;
    draft_n[slot] = m + 1;
  }
}

cudaError_t commit_launch(int B, int R, int stage_R, int Bmax, const int* slots, const int* m_ws,
                          const int* vtok_ws, const int* cand_ws, const bf16* stage, bf16* pool, int L, int n_pages,
                          int page_size, const int* block_table, int max_pages, int* seq_len, int* pending,
                          const bf16* b_ws, bf16* draft_b, int* draft_tok, int* draft_n, int* committed,
                          int* n_committed, int* tickets, int* err, cudaStream_t s) {
  return launch_pdl(commit_kernel, dim3(B, L), dim3(256), 0, s, R, stage_R, Bmax, slots, m_ws, vtok_ws, cand_ws, stage,
                    pool, L, n_pages, page_size, block_table, max_pages, seq_len, pending, b_ws, draft_b, draft_tok,
                    draft_n, committed, n_committed, tickets, err);
}

// ---------------------------------------------------------------- draft glue
// Depth-1 rows of the draft step: for the rows queued by the last commit, dcat =
// [N_e(E x_{p+1}); N_h(b_p)] (bf16), positions p and page offsets of their committed draft
// K/V; padding rows are zero and write no K/V.  Also cand[b][0] = pending token.
__global__ void __launch_bounds__(128) draft_prep_kernel(int R, const int* slots, const int* seq_len,
                                                         const int* pending, const int* draft_n, const bf16* draft_b,
                                                         const int* draft_tok, const bf16* embed, int vocab,
                                                         const bf16* enorm, const bf16* hnorm, float eps, bf16* dcat,
                                                         int* pos, long long* kv_rowoff, int* last_row, int page_size,
                                                         const int* block_table, int max_pages, int n_pages, int* cand,
                                                         int cand_ld, int n_slots, int* err) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[4];
  const int b = blockIdx.x / R, i = blockIdx.x % R, row = blockIdx.x;
  int slot = slots[b];
  if (slot < 0 || slot >= n_slots) {   // treated as a slot with no queued rows
    if (threadIdx.x == 0 && i == 0) atomicOr(err, ERR_SLOT_RANGE);
    slot = -1;
  }
  int n = slot >= 0 ? draft_n[slot] : 0;
  if (slot >= 0 && (n < 1 || n > kMaxR)) {
    if (threadIdx.x == 0 && i == 0) atomicOr(err, ERR_NO_DRAFT_ROWS);
    n = 0;
  }
  if (i == 0 && threadIdx.x == 0) {
    cand[b * cand_ld] = slot >= 0 ? pending[slot] : 0;
    last_row[b] = b * R + (n > 0 ? n - 1 : 0);
  }
  bf16* out = dcat + static_cast<size_t>(row) * 2 * kD;
  if (i >= n) {
    for (int k = threadIdx.x; k < 2 * kD; k += 128) out[k] = __float2bfloat16(0.f);
    if (threadIdx.x == 0) {
      pos[row] = 0;
      kv_rowoff[row] = -1;
    }
    return;
  }
  int tok = draft_tok[slot * kMaxR + i];
  if (tok < 0 || tok >= vocab) {
    if (threadIdx.x == 0) atomicOr(err, ERR_TOKEN_RANGE);
    tok = 0;
  }
  float x[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) x[k] = __bfloat162float(embed[static_cast<size_t>(tok) * kD + threadIdx.x + 128 * k]);
  norm_row_store(x, enorm, eps, out, red);
#pragma unroll
  for (int k = 0; k < 10; ++k)
    x[k] = __bfloat162float(draft_b[(static_cast<size_t>(slot) * kMaxR + i) * kD + threadIdx.x + 128 * k]);
  norm_row_store(x, hnorm, eps, out + kD, red);
  if (threadIdx.x == 0) {
    const int p = seq_len[slot] - n + i;
    pos[row] = p;
    const int pi = p / page_size;
    const int page = (p >= 0 && pi < max_pages) ? block_table[slot * max_pages + pi] : -1;
    if (page < 0 || page >= n_pages) {
      atomicOr(err, ERR_PAGE_RANGE);
      kv_rowoff[row] = -1;
    } else {
      kv_rowoff[row] = (static_cast<long long>(page) * 2 * kH * page_size + (p % page_size)) * kHD;
    }
  }
}

cudaError_t draft_prep_launch(int B, int R, const int* slots, const int* seq_len, const int* pending,
                              const int* draft_n, const bf16* draft_b, const int* draft_tok, const bf16* embed,
                              int vocab, const bf16* enorm, const bf16* hnorm, float eps, bf16* dcat, int* pos,
                              long long* kv_rowoff, int* last_row, int page_size, const int* block_table,
                              int max_pages, int n_pages, int* cand, int cand_ld, int n_slots, int* err,
                              cudaStream_t s) {
  return launch_pdl(draft_prep_kernel, dim3(B * R), dim3(128), 0, s, R, slots, seq_len, pending, draft_n, draft_b,
                    draft_tok, embed, vocab, enorm, hnorm, eps, dcat, pos, kv_rowoff, last_row, page_size, block_table,
                    max_pages, n_pages, cand, cand_ld, n_slots, err);
}

__global__ void gather_rows_kernel(const float* src, const int* rows, float* dst) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const float4* s = reinterpret_cast<const float4*>(src + static_cast<size_t>(rows[b]) * kD);
  float4* d = reinterpret_cast<float4*>(dst + static_cast<size_t>(b) * kD);
  for (int i = threadIdx.x; i < kD / 4; i += blockDim.x) d[i] = s[i];
}

cudaError_t gather_rows_launch(const float* src, const int* rows, int B, float* dst, cudaStream_t s) {
  return launch_pdl(gather_rows_kernel, dim3(B), dim3(128), 0, s, src, rows, dst);
}

// After the LM head of depth k: x^_k = argmax (decoded from the LM head's packed key, which
// is cleared for the next use); for k < K the inputs of depth k+1: dcat = [N_e(E x^_k);
// N_h(u^(k))], position p = j + k (j = ctx_len - 1) and the staging row k-1 of its tentative
// draft K/V.
__global__ void __launch_bounds__(128) draft_next_kernel(unsigned long long* am_key, int vocab, int* err, int k, int K,
                                                         const int* slots, int n_slots,
                                                         const int* seq_len, const bf16* u, const bf16* embed,
                                                         const bf16* enorm, const bf16* hnorm, float eps, bf16* dcat,
                                                         int* pos, long long* kv_rowoff, long long dstage_seq_stride,
                                                         int* cand, int cand_ld) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[4];
  __shared__ int s_tok;
  const int b = blockIdx.x;
  if (threadIdx.x == 0) {
    int tok = argmax_key_index(am_key[b]);
    am_key[b] = 0ull;
    if (tok < 0 || tok >= vocab) {   // no logit reached this row
      atomicOr(err, ERR_TOKEN_RANGE);
      tok = 0;
    }
    s_tok = tok;
    cand[b * cand_ld + k] = tok;
  }
  __syncthreads();
  if (k >= K) return;
  const int tok = s_tok;
  bf16* out = dcat + static_cast<size_t>(b) * 2 * kD;
  float x[10];
#pragma unroll
  for (int q = 0; q < 10; ++q) x[q] = __bfloat162float(embed[static_cast<size_t>(tok) * kD + threadIdx.x + 128 * q]);
  norm_row_store(x, enorm, eps, out, red);
#pragma unroll
  for (int q = 0; q < 10; ++q) x[q] = __bfloat162float(u[static_cast<size_t>(b) * kD + threadIdx.x + 128 * q]);
  norm_row_store(x, hnorm, eps, out + kD, red);
  if (threadIdx.x == 0) {
    const int slot = slots[b];
    const bool slot_ok = slot >= 0 && slot < n_slots;
    if (!slot_ok) atomicOr(err, ERR_SLOT_RANGE);
    pos[b] = (slot_ok ? seq_len[slot] : 0) + k - 1;
    kv_rowoff[b] = b * dstage_seq_stride + static_cast<long long>(k - 1) * 2 * kH * kHD;
  }
}

cudaError_t draft_next_launch(unsigned long long* am_key, int vocab, int* err, int B, int k, int K, const int* slots,
                              int n_slots, const int* seq_len,
                              const bf16* u, const bf16* embed, const bf16* enorm, const bf16* hnorm, float eps,
                              bf16* dcat, int* pos, long long* kv_rowoff, long long dstage_seq_stride, int* cand,
                              int cand_ld, cudaStream_t s) {
  return launch_pdl(draft_next_kernel, dim3(B), dim3(128), 0, s, am_key, vocab, err, k, K, slots, n_slots, seq_len, u, embed, enorm, hnorm,
                    eps, dcat, pos, kv_rowoff, dstage_seq_stride, cand, cand_ld);
}

}  // namespace fm
