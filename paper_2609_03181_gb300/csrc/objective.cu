// The FastMTP draft-head training objective (Sec. 5.6, "Draft-head objective"): for every valid
// response row p and recursive depth k, the cross-entropy of the draft distribution
// P_p^(k) = softmax(W_lm u_p^(k)) at the token x_{p+2}, the KL divergence KL(Q_p || P_p^(k)) from
// the detached verifier distribution Q_p = softmax(W_lm b_{p+1}), and the squared distance
// ||u_p^(k) - b_{p+1}||^2, averaged over the valid rows and combined with the depth weights
// alpha_k = beta^(k-1) / sum_r beta^(r-1) as 0.85 CE + 0.45 KL + 0.45 MSE.
//
// One pass over the tied LM head, logits never written: the rows [b_{p+1}; u_p^(1); ..; u_p^(K)]
// of every p are packed into one activation matrix (groups of G = the power of two >= K+1 rows,
// spare rows zero); the tcgen05 GEMM engine, with the activations as the 128-row A operand and a
// 256-token vocabulary tile of W_lm as the B operand, leaves each activation row's logits in one
// thread's TMEM lane, and its LOSS epilogue folds them into per-row softmax statistics (max, sum
// of exp(x - max), and the KL cross term sum exp(q - max_q) (q - x) against the verifier logits
// q of the row's group, taken from the group's first lane); a finishing kernel folds the tiles of
// each row in tile order, adds the target logit (one dot product) and the squared distance, and a
// last kernel averages over the valid rows.
// KL(Q || P) = sum_v Q(v) (q_v - x_v) - lse(q) + lse(x), the sum being A / Z_q.
#include <math.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>

#include "../../include/fastmtp.h"
#include "common.cuh"
#include "internal.h"

namespace fm {
namespace {

constexpr int kLossMaxK = 7;
constexpr int kLossMaxRows = 1 << 16;   // packed activation rows (n_rows * G)

static __device__ int g_loss_err;

struct LossLayout {
  int G, M, M_pad, a_tiles, v_tiles;   // packed rows, padded to 128-row A tiles; 256-token vocabulary tiles
  size_t x_off, part_off, rows_off, total;
};

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

LossLayout loss_layout(int K, int n_rows, int vocab) {
  LossLayout L;
  L.G = 2;
  while (L.G < K + 1) L.G <<= 1;
  L.M = n_rows * L.G;
  L.M_pad = (L.M + 127) / 128 * 128;
  L.a_tiles = L.M_pad / 128;
  L.v_tiles = (vocab + 255) / 256;
  L.x_off = 0;
  L.part_off = align256(static_cast<size_t>(L.M_pad) * kD * sizeof(bf16));
  L.rows_off = L.part_off + align256(static_cast<size_t>(L.v_tiles) * L.M_pad * sizeof(float4));
  L.total = L.rows_off + align256(static_cast<size_t>(K) * n_rows * 3 * sizeof(float));
  return L;
}

// Row r = p * G + c of the activation matrix: c = 0 the verifier state b_{p+1}, c = 1..K the
// draft states u_p^(c), other rows zero.  160 threads, 16 bytes each.
__global__ void __launch_bounds__(160) loss_pack_kernel(const bf16* u, const bf16* b_next, int K, int n_rows, int G,
                                                        bf16* X) {
  const int r = blockIdx.x, p = r / G, c = r % G;
  const int i = threadIdx.x;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (p < n_rows && c <= K) {
    const bf16* src = (c == 0) ? b_next + static_cast<size_t>(p) * kD
                               : u + (static_cast<size_t>(c - 1) * n_rows + p) * kD;
    v = reinterpret_cast<const uint4*>(src)[i];
  }
  reinterpret_cast<uint4*>(X + static_cast<size_t>(r) * kD)[i] = v;
}

// (m, z) of a softmax partial merged with another; exp(-inf) = 0 leaves an empty side out.
__device__ __forceinline__ void merge_mz(float& m, float& z, float m2, float z2) {
  const float mm = fmaxf(m, m2);
  if (mm == -INFINITY) return;
  z = z * expf(m - mm) + z2 * expf(m2 - mm);
  m = mm;
}

// One CTA per row p, one warp per packed column c = 0..K.  Lane l folds the tiles l, l + 32, ...
// in order, then the warp merges its lanes in a fixed xor tree (a + b == b + a in IEEE
// arithmetic, so every lane ends with the same value).
__global__ void loss_finish_kernel(const float4* part, int ld, int n_tiles, int G, int K, int n_rows, const bf16* u,
                                   const bf16* b_next, const int* target, const bf16* lm_head, int vocab,
                                   float* rows_out) {
  __shared__ float s_q[2];   // verifier column: lse(q) and Z_q (relative to the global max of q)
  const int p = blockIdx.x, c = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int col = p * G + c;
  float m = -INFINITY, z = 0.f, mq = -INFINITY, A = 0.f;
  for (int t = lane; t < n_tiles; t += 32) {
    const float4 v = __ldcg(part + static_cast<size_t>(t) * ld + col);
    merge_mz(m, z, v.x, v.y);
    merge_mz(mq, A, v.w, v.z);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), z2 = __shfl_xor_sync(0xffffffffu, z, o);
    const float q2 = __shfl_xor_sync(0xffffffffu, mq, o), a2 = __shfl_xor_sync(0xffffffffu, A, o);
    merge_mz(m, z, m2, z2);
    merge_mz(mq, A, q2, a2);
  }
  if (c == 0 && lane == 0) {
    s_q[0] = m + logf(z);
    s_q[1] = z;
  }
  __syncthreads();
  if (c == 0) return;
  // the draft logit of the target token and the squared distance to the verifier state
  const bf16* uk = u + (static_cast<size_t>(c - 1) * n_rows + p) * kD;
  const bf16* bp = b_next + static_cast<size_t>(p) * kD;
  int x = target[p];
  const bool bad = x < 0 || x >= vocab;
  if (bad) x = 0;
  const bf16* w = lm_head + static_cast<size_t>(x) * kD;
  float dot = 0.f, sq = 0.f;
  for (int i = lane; i < kD / 8; i += 32) {
    const uint4 uw = reinterpret_cast<const uint4*>(uk)[i];
    const uint4 ww = reinterpret_cast<const uint4*>(w)[i];
    const uint4 bw = reinterpret_cast<const uint4*>(bp)[i];
    const bf16* ue = reinterpret_cast<const bf16*>(&uw);
    const bf16* we = reinterpret_cast<const bf16*>(&ww);
    const bf16* be = reinterpret_cast<const bf16*>(&bw);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float uf = __bfloat162float(ue[e]);
      dot = fmaf(uf, __bfloat162float(we[e]), dot);
      const float df = uf - __bfloat162float(be[e]);
      sq = fmaf(df, df, sq);
    }
  }
  dot = warp_sum(dot);
  sq = warp_sum(sq);
  if (lane == 0) {
    const float lse = m + logf(z);
    float* o = rows_out + (static_cast<size_t>(c - 1) * n_rows + p) * 3;
    o[0] = bad ? NAN : lse - dot;                 // -log P(x_{p+2})
    o[1] = A / s_q[1] - s_q[0] + lse;             // KL(Q || P)
    o[2] = sq;                                    // ||u - b||^2
  }
}

// Means over the valid rows (thread-strided sums, then a fixed block tree) and the weighted total:
// out = [L, CE_1..CE_K, KL_1..KL_K, MSE_1..MSE_K].
struct LossAlpha {
  float a[kLossMaxK];
};

__global__ void __launch_bounds__(256) loss_reduce_kernel(const float* rows, const int* valid, int K, int n_rows,
                                                          LossAlpha alpha, float w_ce, float w_kl, float w_mse,
                                                          float* out) {
  __shared__ float red[8];
  __shared__ float s_mean[3 * kLossMaxK];
  float cnt = 0.f;
  for (int p = threadIdx.x; p < n_rows; p += 256) cnt += (valid == nullptr || valid[p] != 0) ? 1.f : 0.f;
  auto block_total = [&](float v) {
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) s += red[i];
    __syncthreads();
    return s;
  };
  const float n = block_total(cnt);
  for (int k = 0; k < K; ++k)
    for (int term = 0; term < 3; ++term) {
      float s = 0.f;
      for (int p = threadIdx.x; p < n_rows; p += 256)
        if (valid == nullptr || valid[p] != 0) s += rows[(static_cast<size_t>(k) * n_rows + p) * 3 + term];
      s = block_total(s);
      if (threadIdx.x == 0) s_mean[term * kLossMaxK + k] = n > 0.f ? s / n : 0.f;
    }
  __syncthreads();
  if (threadIdx.x == 0) {
    float L = 0.f;
    for (int k = 0; k < K; ++k) {
      const float ce = s_mean[k], kl = s_mean[kLossMaxK + k], mse = s_mean[2 * kLossMaxK + k];
      out[1 + k] = ce;
      out[1 + K + k] = kl;
      out[1 + 2 * K + k] = mse;
      L += w_ce * alpha.a[k] * ce + w_kl * alpha.a[k] * kl + w_mse * alpha.a[k] * mse;
    }
    out[0] = L;
  }
}

std::atomic<bool> g_ready[64];
int* g_err_ptr[64];
std::mutex g_ready_lock;

spec_status fail(spec_status s, const std::string& m) {
  set_thread_error(m);
  return s;
}

}  // namespace
}  // namespace fm

using namespace fm;

extern "C" spec_status spec_draft_loss_workspace(int32_t K, int32_t n_rows, int32_t vocab, size_t* bytes) {
  if (bytes == nullptr) return fail(SPEC_EINVAL, "bytes is NULL");
  *bytes = 0;
  if (K < 1 || K > kLossMaxK || n_rows < 1 || vocab < 1) return fail(SPEC_EINVAL, "K, n_rows or vocab out of range");
  const LossLayout L = loss_layout(K, n_rows, vocab);
  if (L.M_pad > kLossMaxRows) return fail(SPEC_EINVAL, "n_rows * (power of two >= K + 1) above 65536");
  *bytes = L.total;
  return SPEC_OK;
}

extern "C" spec_status spec_draft_loss(const void* u, const void* b_next, const int32_t* target, const int32_t* valid,
                                       const void* lm_head, int32_t K, int32_t n_rows, int32_t vocab, float beta,
                                       float w_ce, float w_kl, float w_mse, float* out, float* row_out,
                                       void* workspace, size_t workspace_bytes, void* stream) {
  if (u == nullptr || b_next == nullptr || target == nullptr || lm_head == nullptr || out == nullptr ||
      workspace == nullptr)
    return fail(SPEC_EINVAL, "null argument");
  size_t need = 0;
  spec_status st = spec_draft_loss_workspace(K, n_rows, vocab, &need);
  if (st != SPEC_OK) return st;
  if (workspace_bytes < need)
    return fail(SPEC_EINVAL, "workspace too small: " + std::to_string(need) + " bytes needed");
  auto misaligned = [](const void* ptr, uintptr_t a) { return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0; };
  if (misaligned(u, 16) || misaligned(b_next, 16) || misaligned(lm_head, 16) || misaligned(workspace, 256))
    return fail(SPEC_EINVAL, "u, b_next and lm_head must be 16-byte aligned, the workspace 256-byte aligned");
  if (!(beta > 0.f) || !isfinite(beta) || !isfinite(w_ce) || !isfinite(w_kl) || !isfinite(w_mse))
    return fail(SPEC_EINVAL, "beta must be positive and finite, the weights finite");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) return fail(SPEC_ECUDA, "cudaGetDevice failed or device above 63");
  if (!g_ready[dev].load(std::memory_order_acquire)) {
    std::lock_guard<std::mutex> hold(g_ready_lock);
    if (!g_ready[dev].load(std::memory_order_relaxed)) {
      int* ep = nullptr;
      e = gemm_prepare();
      if (e == cudaSuccess) e = cudaGetSymbolAddress(reinterpret_cast<void**>(&ep), g_loss_err);
      if (e != cudaSuccess) return fail(SPEC_ECUDA, std::string("set-up: ") + cudaGetErrorString(e));
      g_err_ptr[dev] = ep;
      g_ready[dev].store(true, std::memory_order_release);
    }
  }
  const LossLayout L = loss_layout(K, n_rows, vocab);
  char* ws = static_cast<char*>(workspace);
  bf16* X = reinterpret_cast<bf16*>(ws + L.x_off);
  float4* part = reinterpret_cast<float4*>(ws + L.part_off);
  float* rows = row_out != nullptr ? row_out : reinterpret_cast<float*>(ws + L.rows_off);
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  std::string err;
  // operands swapped: A = the packed activation rows (128-row tiles), B = W_lm (256-row boxes)
  if (!encode_map_2d(&g.a_map[0], X, kD, L.M_pad, 128, &err)) return fail(SPEC_EINVAL, err);
  if (!encode_act_maps(g.b_map[0], lm_head, kD, vocab, &err)) return fail(SPEC_EINVAL, err);
  g.n_routed = 1 << 30;
  g.N = L.M_pad;
  g.K = kD;
  g.M = vocab;
  g.box_log = 4;
  g.m_tiles = L.v_tiles;
  g.n_tiles = L.a_tiles;
  g.split_k = 1;
  g.n_items = L.v_tiles * L.a_tiles;
  g.ldo = L.M_pad;
  g.a_keep = 1;   // the packed rows are read once per vocabulary tile: keep them in L2
  g.loss_part = part;
  g.loss_G = L.G;
  g.err = g_err_ptr[dev];
  // alpha_k = beta^(k-1) / sum_r beta^(r-1), k = 1..K (computed in double, passed as fp32)
  LossAlpha alpha = {};
  {
    double zs = 0.0;
    for (int r = 0; r < K; ++r) zs += pow(static_cast<double>(beta), r);
    for (int k = 0; k < K; ++k) alpha.a[k] = static_cast<float>(pow(static_cast<double>(beta), k) / zs);
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  loss_pack_kernel<<<L.M_pad, 160, 0, s>>>(static_cast<const bf16*>(u), static_cast<const bf16*>(b_next), K, n_rows,
                                           L.G, X);
  e = cudaGetLastError();
  if (e == cudaSuccess) {
    const int grid = g.n_items < num_sms() ? g.n_items : num_sms();
    e = gemm_launch(EPI_LOSS, 256, g, grid, s, false);
  }
  if (e == cudaSuccess) {
    loss_finish_kernel<<<n_rows, 32 * (K + 1), 0, s>>>(part, L.M_pad, L.v_tiles, L.G, K, n_rows,
                                                      static_cast<const bf16*>(u), static_cast<const bf16*>(b_next),
                                                      target, static_cast<const bf16*>(lm_head), vocab, rows);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    loss_reduce_kernel<<<1, 256, 0, s>>>(rows, valid, K, n_rows, alpha, w_ce, w_kl, w_mse, out);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) return fail(SPEC_ECUDA, std::string("launch: ") + cudaGetErrorString(e));
  return SPEC_OK;
}

// The guard flag of the objective's GEMM on the current device (0 if it never ran there),
// cleared after reading; spec_sync(NULL) reports it.
cudaError_t fm::loss_take_flag(int* flag) {
  *flag = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64 || !g_ready[dev].load(std::memory_order_acquire)) return e;
  e = cudaMemcpyFromSymbol(flag, g_loss_err, sizeof(int));
  if (e == cudaSuccess && *flag != 0) {
    const int zero = 0;
    e = cudaMemcpyToSymbol(g_loss_err, &zero, sizeof(int));
  }
  return e;
}
