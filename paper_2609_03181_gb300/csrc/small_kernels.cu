// Latency-bound kernels of the FastMTP step: embedding + RMSNorm, RMSNorm, router
// (norm, logits, softmax, top-6, per-expert row lists and input rows), MoE combine (+ the next
// RMSNorm), the KV commit, and the glue of the draft chain.  Every reduction runs in a fixed
// order, so a row's result never depends on the other rows of the batch.
#include <cuda_fp8.h>
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

// The norm gain of this thread's elements i = tid + NT*k as floats.  A gain is a weight, never
// written by an earlier kernel, so every kernel below reads it before its wait.
template <int NT>
__device__ __forceinline__ void load_gain_t(const bf16* gain, float (&gv)[kD / NT]) {
#pragma unroll
  for (int k = 0; k < kD / NT; ++k) gv[k] = __bfloat162float(gain[threadIdx.x + NT * k]);
}
// x (kD/NT values per thread, element i = tid + NT*k) -> bf16 x * rsqrt(mean(x^2) + eps) * gain
template <int NT>
__device__ __forceinline__ void norm_row_store_t(const float (&x)[kD / NT], const float (&gv)[kD / NT], float eps,
                                                 bf16* out, float* red) {
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kD / NT; ++k) ss += x[k] * x[k];
  ss = block_sum<NT>(ss, red);
  const float inv = rsqrtf(ss / kD + eps);
#pragma unroll
  for (int k = 0; k < kD / NT; ++k) out[threadIdx.x + NT * k] = __float2bfloat16(x[k] * inv * gv[k]);
}
__device__ __forceinline__ void norm_row_store(const float (&x)[10], const float (&gv)[10], float eps, bf16* out,
                                               float* red) {
  norm_row_store_t<128>(x, gv, eps, out, red);
}

// ---------------------------------------------------------------- embedding + norm
__global__ void __launch_bounds__(128) embed_norm_kernel(const int* cand, int R, const int* slots, const int* pending,
                                                         const int* seq_len, const bf16* embed, int vocab,
                                                         const bf16* gain, float eps, float* h, bf16* xn, int* pos,
                                                         long long* kv_rowoff, int stage_R, int n_slots, int* err,
                                                         int* zero, int n_zero, int* zero2, int n_zero2) {
  pdl_trigger(kTrEmbed);
  float gv[10];
  load_gain_t<128>(gain, gv);
  pdl_wait();
  if (blockIdx.x == 0) {   // the step's per-expert row counters and tile counters start from zero
    for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero[i] = 0;
    for (int i = threadIdx.x; i < n_zero2; i += blockDim.x) zero2[i] = 0;
  }
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
  if (threadIdx.x == 32) {   // the position, while the embedding row is fetched
    pos[row] = (slot_ok ? seq_len[slot] : 0) + r;
    kv_rowoff[row] = static_cast<long long>(b * stage_R + r) * 2 * kH * kHD;
  }
  const bf16* e = embed + static_cast<size_t>(tok) * kD;
  float x[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) {
    const int i = threadIdx.x + 128 * k;
    x[k] = __bfloat162float(e[i]);
    h[static_cast<size_t>(row) * kD + i] = x[k];
  }
  norm_row_store(x, gv, eps, xn + static_cast<size_t>(row) * kD, red);
}

cudaError_t embed_norm_launch(const int* cand, int B, int R, const int* slots, const int* pending,
                              const int* seq_len, const bf16* embed, int vocab, const bf16* gain, float eps,
                              float* h, bf16* xn, int* pos, long long* kv_rowoff, int stage_R, int n_slots,
                              int* err, int* zero, int n_zero, int* zero2, int n_zero2, cudaStream_t s) {
  return launch_pdl(embed_norm_kernel, dim3(B * R), dim3(128), 0, s, cand, R, slots, pending, seq_len, embed, vocab, gain,
                    eps, h, xn, pos, kv_rowoff, stage_R, n_slots, err, zero, n_zero, zero2, n_zero2);
}

// ---------------------------------------------------------------- RMSNorm
__global__ void __launch_bounds__(128) rmsnorm_kernel(const float* x, const bf16* gain, float eps, bf16* out) {
  pdl_trigger(kTrNorm);
  float gv[10];
  load_gain_t<128>(gain, gv);
  pdl_wait();
  __shared__ float red[4];
  const size_t row = blockIdx.x;
  float v[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) v[k] = x[row * kD + threadIdx.x + 128 * k];
  norm_row_store(v, gv, eps, out + row * kD, red);
}

cudaError_t rmsnorm_launch(const float* x, int rows, const bf16* gain, float eps, bf16* out, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(128), 0, s, x, gain, eps, out);
}

// ---------------------------------------------------------------- router
// 4 token rows per CTA (8 or 16 when that many CTAs would not fit on the GPU at once), in the
// first rows of a 16-row MMA tile (the router matrix is read from L2 once per CTA; more CTAs
// spread the copies of the selected rows).  Per row: RMSNorm of the residual row -> xn (bf16, also the experts' input); the 64 logits of the
// rounded row on bf16 tensor cores (mma.sync m16n8k16, fp32 accumulation; warp w computes
// experts 8w..8w+7 of all 16 rows, each lane streaming 16-byte pieces of its expert's row);
// fp32 softmax; top-6 by probability (lower id on ties).  Each selected (token, rank, expert)
// takes the next row of its expert with one atomic add on the layer's per-expert counter,
// records (token << 3 | rank) in that row of the expert's list and copies the rounded row to
// that row of the expert's input region (map_stride rows per expert), so neither a grouping
// pass nor a row gather follows.  A row's arithmetic is the same whatever rows share its CTA,
// and a (token, expert) row's result does not depend on its position among the expert's rows.
constexpr int kRouteRows = 16;      // rows of the MMA tile
constexpr int kRouteCtaRows = 4;    // token rows of a CTA while one such CTA per SM covers T
constexpr int kRouteStride = kD + 32;   // bf16 per staged row: rows 64 bytes apart in the banks
constexpr int kMaxT = 2048;

__global__ void __launch_bounds__(256) router_kernel(const __grid_constant__ RouteArgs a, int cta_rows) {
  pdl_trigger(kTrRouter);
  __shared__ __align__(16) bf16 xs[kRouteRows * kRouteStride];   // the rounded rows
  __shared__ float lg[kRouteRows][kE];                           // logits, then probabilities
  __shared__ int dst[kRouteRows][kTopK];                         // input row of each selection
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  // The router matrix is never written by earlier kernels: this lane's share of its expert's
  // row (expert 8 warp + g, columns 32 c + 8 t4 .. + 7) is loaded before the wait.
  constexpr int kSteps = kD / 32;
  const uint4* wrow = reinterpret_cast<const uint4*>(a.wr + static_cast<size_t>(warp * 8 + g) * kD) + t4;
  uint4 wq[kSteps];
#pragma unroll
  for (int c = 0; c < kSteps; ++c) wq[c] = wrow[4 * c];
  uint2 gq[kD / 128];   // norm gain (bf16, also a weight), lane's columns 4 (lane + 32 k) .. + 3
#pragma unroll
  for (int k = 0; k < kD / 128; ++k) gq[k] = *reinterpret_cast<const uint2*>(a.gain + 4 * (lane + 32 * k));
  pdl_wait();
  const int t0 = blockIdx.x * cta_rows;
  const int nr = min(cta_rows, a.T - t0);
  // RMSNorm: warp w takes rows w and w + 8 of the 16-row MMA tile, of which the first nr are
  // token rows and the rest zeros; a lane sums its 40 squares of a row in order, then a warp tree
  {
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int r = warp + 8 * h2;
      bf16* xr = xs + r * kRouteStride;
      if (r >= nr) {   // a padding row of the MMA tile (warp-uniform): zeros, no load
#pragma unroll
        for (int k = 0; k < kD / 128; ++k) *reinterpret_cast<uint2*>(xr + 4 * (lane + 32 * k)) = make_uint2(0u, 0u);
        continue;
      }
      const float4* hr = reinterpret_cast<const float4*>(a.h + static_cast<size_t>(t0 + r) * kD);
      float4 v[kD / 128];
#pragma unroll
      for (int k = 0; k < kD / 128; ++k) v[k] = hr[lane + 32 * k];
      float ss = 0.f;
#pragma unroll
      for (int k = 0; k < kD / 128; ++k) ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
      ss = warp_sum(ss);
      const float inv = rsqrtf(ss / kD + a.eps);
      bf16* xo = a.xn + static_cast<size_t>(t0 + r) * kD;
#pragma unroll
      for (int k = 0; k < kD / 128; ++k) {
        const int i = 4 * (lane + 32 * k);
        const __nv_bfloat162 g01 = *reinterpret_cast<const __nv_bfloat162*>(&gq[k].x);
        const __nv_bfloat162 g23 = *reinterpret_cast<const __nv_bfloat162*>(&gq[k].y);
        __align__(8) bf16 o4[4];
        o4[0] = __float2bfloat16(v[k].x * inv * __low2float(g01));
        o4[1] = __float2bfloat16(v[k].y * inv * __high2float(g01));
        o4[2] = __float2bfloat16(v[k].z * inv * __low2float(g23));
        o4[3] = __float2bfloat16(v[k].w * inv * __high2float(g23));
        *reinterpret_cast<uint2*>(xo + i) = *reinterpret_cast<const uint2*>(o4);
        *reinterpret_cast<uint2*>(xr + i) = *reinterpret_cast<const uint2*>(o4);
        if (a.xn8 != nullptr) {   // fp8 experts: the shared experts' input row, rounded to e4m3
          uint32_t q = 0;
#pragma unroll
          for (int e = 0; e < 4; ++e)
            q |= static_cast<uint32_t>(__nv_cvt_float_to_fp8(__bfloat162float(o4[e]), __NV_SATFINITE, __NV_E4M3))
                 << (8 * e);
          *reinterpret_cast<uint32_t*>(a.xn8 + static_cast<size_t>(t0 + r) * kD + i) = q;
        }
      }
    }
  }
  __syncthreads();
  // logits D[row][expert] = xs W^T: 40 steps of 32 columns, two k16 MMAs each.  Within a step
  // the columns enter the MMA in a fixed permuted order (lane t4's four pairs 32c + 8t4 + 2j,
  // j = 0..3, as k pairs 2t4 and 2t4 + 8 of the first MMA and of the second), the same for the
  // rows and the weights.
  // two independent accumulator chains (even and odd steps), added at the end
  float dq[2][4] = {};
#pragma unroll
  for (int c = 0; c < kSteps; ++c) {
    const uint4 w = wq[c];
    const uint4 x0 = *reinterpret_cast<const uint4*>(xs + g * kRouteStride + 32 * c + 8 * t4);
    const uint4 x1 = *reinterpret_cast<const uint4*>(xs + (g + 8) * kRouteStride + 32 * c + 8 * t4);
    const uint32_t a0[4] = {x0.x, x1.x, x0.y, x1.y}, b0[2] = {w.x, w.y};
    const uint32_t a1[4] = {x0.z, x1.z, x0.w, x1.w}, b1[2] = {w.z, w.w};
    mma_bf16_16816(dq[c & 1], a0, b0);
    mma_bf16_16816(dq[c & 1], a1, b1);
  }
  float d[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) d[u] = dq[0][u] + dq[1][u];
  {
    const int e = warp * 8 + 2 * t4;
    const float b0 = a.bias ? a.bias[e] : 0.f, b1 = a.bias ? a.bias[e + 1] : 0.f;
    lg[g][e] = d[0] + b0;
    lg[g][e + 1] = d[1] + b1;
    lg[g + 8][e] = d[2] + b0;
    lg[g + 8][e + 1] = d[3] + b1;
  }
  __syncthreads();
  // softmax of rows warp and warp + 8 (lane l holds experts l and l + 32); lg then holds each
  // probability p as the 32-bit order key of p + 0 (a larger key = a larger p)
  unsigned* ok = reinterpret_cast<unsigned*>(&lg[0][0]);
#pragma unroll
  for (int h2 = 0; h2 < 2; ++h2) {
    const int r = warp + 8 * h2;
    if (r >= nr) break;
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
    ok[r * kE + lane] = static_cast<unsigned>(argmax_key(p0, lane) >> 32);
    ok[r * kE + lane + 32] = static_cast<unsigned>(argmax_key(p1, lane + 32) >> 32);
  }
  __syncthreads();
  // top-6: the thread of (row r, expert e) counts the experts whose (probability, lower id
  // first) key beats its own -- its rank, the place six argmax rounds would give it -- and,
  // ranked among the first six, takes the next row of expert e
  for (int pr = threadIdx.x; pr < nr * kE; pr += 256) {
    const int r = pr >> 6, e = pr & 63;
    // the full keys (order key << 32 | ~id), as argmax_key builds them
    const unsigned pk = ok[r * kE + e];
    const unsigned long long mine = (static_cast<unsigned long long>(pk) << 32) | static_cast<unsigned>(~e);
    int rank = 0;
#pragma unroll
    for (int o = 0; o < kE; ++o)
      rank += ((static_cast<unsigned long long>(ok[r * kE + o]) << 32 | static_cast<unsigned>(~o)) > mine) ? 1 : 0;
    if (rank < kTopK) {
      // the probability back from its key (the key of p + 0 maps one to one onto p)
      const float pe = __uint_as_float((pk & 0x80000000u) ? (pk & 0x7fffffffu) : ~pk);
      const int t = t0 + r;
      const int pos = atomicAdd(a.counts + e, 1);
      a.idx[static_cast<size_t>(t) * kTopK + rank] = e;
      a.gate[static_cast<size_t>(t) * kTopK + rank] = pe;
      a.rowmap[static_cast<size_t>(e) * a.map_stride + pos] = (t << 3) | rank;
      dst[r][rank] = e * a.map_stride + pos;
    }
  }
  __syncthreads();
  // the rounded rows into their experts' input rows, 8 elements per thread and step (16 bytes
  // of bf16, or with fp8 experts 8 bytes of e4m3)
  constexpr int kVec = kD / 8;
  for (int i = threadIdx.x; i < nr * kTopK * kVec; i += 256) {
    const int v = i % kVec, sel = i / kVec, r = sel / kTopK;
    const uint4 x = *reinterpret_cast<const uint4*>(xs + r * kRouteStride + 8 * v);
    const size_t row = static_cast<size_t>(dst[r][sel % kTopK]);
    if (a.x_sorted8 != nullptr) {
      const bf16* xe = reinterpret_cast<const bf16*>(&x);
      uint32_t lo = 0, hi = 0;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        lo |= static_cast<uint32_t>(__nv_cvt_float_to_fp8(__bfloat162float(xe[e]), __NV_SATFINITE, __NV_E4M3)) << (8 * e);
        hi |= static_cast<uint32_t>(__nv_cvt_float_to_fp8(__bfloat162float(xe[4 + e]), __NV_SATFINITE, __NV_E4M3))
              << (8 * e);
      }
      *reinterpret_cast<uint2*>(a.x_sorted8 + row * kD + 8 * v) = make_uint2(lo, hi);
    } else {
      *reinterpret_cast<uint4*>(a.x_sorted + row * kD + 8 * v) = x;
    }
  }
  trace_exit();
}

cudaError_t router_prepare() { return cudaSuccess; }

cudaError_t router_launch(const RouteArgs& a, cudaStream_t s) {
  if (a.T > kMaxT || a.T < 1 || a.T > a.map_stride) return cudaErrorInvalidValue;
  // 4 rows a CTA while that fits one wave of one CTA per SM, else 8 or 16 (the router is one CTA
  // per SM: 240 registers a thread); a row's arithmetic does not depend on the rows beside it
  int rows = kRouteCtaRows;
  while (rows < kRouteRows && (a.T + rows - 1) / rows > num_sms()) rows *= 2;
  return launch_pdl(router_kernel, dim3((a.T + rows - 1) / rows), dim3(256), 0, s, a, rows);
}

// ---------------------------------------------------------------- combine
// h += sum_{s<6} gate_s * y_s + y_shared0 + y_shared1 (fixed slot order), then RMSNorm -> out.
__global__ void __launch_bounds__(256) combine_kernel(float* h, const float* y, const float* gate, const bf16* gain,
                                                      float eps, bf16* out) {
  pdl_trigger(kTrCombine);
  constexpr int NT = 256, EPT = kD / NT;
  float gv[EPT];
  load_gain_t<NT>(gain, gv);
  pdl_wait();
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
  norm_row_store_t<NT>(x, gv, eps, out + t * kD, red);
  trace_exit();
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
  pdl_trigger(kTrCommit);
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
  pdl_trigger(kTrDraftPrep);
  float ge[10], gh[10];
  load_gain_t<128>(enorm, ge);
  load_gain_t<128>(hnorm, gh);
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
  // three independent chains go out together: the token (then its embedding row), the base
  // state row, and the position (then its page)
  __shared__ int s_tok;
  float xb[10];
#pragma unroll
  for (int k = 0; k < 10; ++k)
    xb[k] = __bfloat162float(draft_b[(static_cast<size_t>(slot) * kMaxR + i) * kD + threadIdx.x + 128 * k]);
  if (threadIdx.x == 0) {
    int tok = draft_tok[slot * kMaxR + i];
    if (tok < 0 || tok >= vocab) {
      atomicOr(err, ERR_TOKEN_RANGE);
      tok = 0;
    }
    s_tok = tok;
  } else if (threadIdx.x == 32) {
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
  __syncthreads();
  const int tok = s_tok;
  float x[10];
#pragma unroll
  for (int k = 0; k < 10; ++k) x[k] = __bfloat162float(embed[static_cast<size_t>(tok) * kD + threadIdx.x + 128 * k]);
  norm_row_store(xb, gh, eps, out + kD, red);   // while the embedding row is on its way
  norm_row_store(x, ge, eps, out, red);
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
  pdl_trigger(kTrGather);
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
  pdl_trigger(kTrDraftNext);
  float ge[10], gh[10];
  load_gain_t<128>(enorm, ge);
  load_gain_t<128>(hnorm, gh);
  pdl_wait();
  __shared__ float red[4];
  __shared__ int s_tok;
  const int b = blockIdx.x;
  // the loads that do not depend on the drafted token go out together with the key: the
  // token's state row u and the sequence's position
  float xu[10];
  if (k < K) {
#pragma unroll
    for (int q = 0; q < 10; ++q) xu[q] = __bfloat162float(u[static_cast<size_t>(b) * kD + threadIdx.x + 128 * q]);
  }
  if (threadIdx.x == 0) {
    int tok = argmax_key_index(am_key[b]);
    am_key[b] = 0ull;
    if (tok < 0 || tok >= vocab) {   // no logit reached this row
      atomicOr(err, ERR_TOKEN_RANGE);
      tok = 0;
    }
    s_tok = tok;
    cand[b * cand_ld + k] = tok;
  } else if (threadIdx.x == 32 && k < K) {
    const int slot = slots[b];
    const bool slot_ok = slot >= 0 && slot < n_slots;
    if (!slot_ok) atomicOr(err, ERR_SLOT_RANGE);
    pos[b] = (slot_ok ? seq_len[slot] : 0) + k - 1;
    kv_rowoff[b] = b * dstage_seq_stride + static_cast<long long>(k - 1) * 2 * kH * kHD;
  }
  __syncthreads();
  if (k >= K) return;
  const int tok = s_tok;
  bf16* out = dcat + static_cast<size_t>(b) * 2 * kD;
  float x[10];
#pragma unroll
  for (int q = 0; q < 10; ++q) x[q] = __bfloat162float(embed[static_cast<size_t>(tok) * kD + threadIdx.x + 128 * q]);
  norm_row_store(xu, gh, eps, out + kD, red);   // while the embedding row is on its way
  norm_row_store(x, ge, eps, out, red);
}

cudaError_t draft_next_launch(unsigned long long* am_key, int vocab, int* err, int B, int k, int K, const int* slots,
                              int n_slots, const int* seq_len,
                              const bf16* u, const bf16* embed, const bf16* enorm, const bf16* hnorm, float eps,
                              bf16* dcat, int* pos, long long* kv_rowoff, long long dstage_seq_stride, int* cand,
                              int cand_ld, cudaStream_t s) {
  return launch_pdl(draft_next_kernel, dim3(B), dim3(128), 0, s, am_key, vocab, err, k, K, slots, n_slots, seq_len, u, embed, enorm, hnorm,
                    eps, dcat, pos, kv_rowoff, dstage_seq_stride, cand, cand_ld);
}

#ifdef FM_TRACE
FM_TRACE_READER(trace_read_small)
#endif

}  // namespace fm
