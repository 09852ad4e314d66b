// spec_gemm_bf16_noalloc: the split-K form of the dense projection for callers that cannot
// allocate device memory.
//
// Who needs it: code that runs while a CUDA stream is being captured into a graph (an
// allocation there is either rejected or breaks the capture), runtimes that hand out device
// memory only from their own fixed pool and forbid hidden allocations, and latency-critical
// serving loops where an implicit cudaMalloc would synchronise the device.  The split-K GEMM
// needs scratch memory for its partial tiles and per-tile tickets; here that scratch is a
// file-scope device array, so the call allocates nothing.  The caller still passes X, W and Y.
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>

#include "../../include/fastmtp.h"
#include "internal.h"

using namespace fm;

namespace {

constexpr size_t kNoAllocScratchFloats = 1u << 20;   // 4 MiB of split-K partial tiles
constexpr int kNoAllocTickets = 1024;                // per-tile tickets

// Shared by every call on a device and held by every GPU that loads the library until the
// process exits.  Calls whose kernels overlap on the GPU race on it.
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];
static __device__ __align__(256) int g_noalloc_tickets[kNoAllocTickets];
static __device__ int g_noalloc_err;

// Device addresses of the arrays, per device.  `ready` is published with release order after
// the pointers are written and read with acquire order, and the first lookup on a device runs
// under a lock, so host threads making their first calls at the same time each see either no
// entry (and wait for the lock) or a complete one.
struct DevPtrs {
  std::atomic<bool> ready{false};
  float* scratch = nullptr;
  int* tickets = nullptr;
  int* err = nullptr;
};
DevPtrs g_dev[64];
std::mutex g_dev_lock;

spec_status fail(spec_status s, const std::string& m) {
  set_thread_error(m);   // reported by spec_last_error(NULL)
  return s;
}

// In host code the arrays' names are host-side stand-ins, not device addresses: the device
// addresses are looked up once per device, with that device current.
spec_status device_ptrs(DevPtrs** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(SPEC_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return fail(SPEC_EINVAL, "device index above 63");
  DevPtrs& p = g_dev[dev];
  if (!p.ready.load(std::memory_order_acquire)) {
    std::lock_guard<std::mutex> hold(g_dev_lock);
    if (!p.ready.load(std::memory_order_relaxed)) {
      float* scratch = nullptr;
      int* tickets = nullptr;
      int* err = nullptr;
      e = cudaGetSymbolAddress(reinterpret_cast<void**>(&scratch), g_noalloc_scratch);
      if (e == cudaSuccess) e = cudaGetSymbolAddress(reinterpret_cast<void**>(&tickets), g_noalloc_tickets);
      if (e == cudaSuccess) e = cudaGetSymbolAddress(reinterpret_cast<void**>(&err), g_noalloc_err);
      if (e == cudaSuccess) e = gemm_prepare();
      if (e != cudaSuccess)
        return fail(SPEC_ECUDA, std::string("scratch symbol lookup: ") + cudaGetErrorString(e));
      p.scratch = scratch;
      p.tickets = tickets;
      p.err = err;
      p.ready.store(true, std::memory_order_release);
    }
  }
  *out = &p;
  return SPEC_OK;
}

// Split count: a function of the SM count, N and K only (about one CTA per SM over the weight
// tiles, at least two 64-wide k-chunks per split, at most kMaxSplit), so the shapes that fit the
// fixed scratch do not depend on any occupancy query.
int noalloc_split_k(int N, int K) {
  const int n_tiles = (N + 127) / 128;
  int s = num_sms() / n_tiles;
  if (s > (K / 64) / 2) s = (K / 64) / 2;
  if (s > kMaxSplit) s = kMaxSplit;
  return s < 1 ? 1 : s;
}

}  // namespace

extern "C" spec_status spec_gemm_bf16_noalloc(const void* X, const void* W, float* Y, int32_t M, int32_t N,
                                              int32_t Kdim, void* stream) {
  if (X == nullptr || W == nullptr || Y == nullptr) return fail(SPEC_EINVAL, "null argument");
  if (M < 1 || N < 1 || Kdim < 64 || Kdim % 64) return fail(SPEC_EINVAL, "bad sizes");
  if ((reinterpret_cast<uintptr_t>(X) & 15u) || (reinterpret_cast<uintptr_t>(W) & 15u))
    return fail(SPEC_EINVAL, "X and W must be 16-byte aligned");
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.n_routed = 1 << 30;
  g.N = N;
  g.K = Kdim;
  g.M = M;
  int bl = 0;
  while ((16 << bl) < (M < 256 ? M : 256) && bl < 4) ++bl;
  g.box_log = bl;
  const int box = 16 << bl;
  g.m_tiles = (M + box - 1) / box;
  g.n_tiles = (N + 127) / 128;
  g.split_k = noalloc_split_k(N, Kdim);
  g.n_items = g.n_tiles * g.split_k * g.m_tiles;
  const size_t need = static_cast<size_t>(g.n_tiles) * g.m_tiles * g.split_k * box * 128;
  if (need > kNoAllocScratchFloats || g.n_tiles * g.m_tiles > kNoAllocTickets)
    return fail(SPEC_EINVAL, "problem too large for the fixed scratch of spec_gemm_bf16_noalloc: needs " +
                                 std::to_string(need * 4) + " bytes of partial tiles, the maximum is " +
                                 std::to_string(kNoAllocScratchFloats * 4));
  DevPtrs* p = nullptr;
  spec_status st = device_ptrs(&p);
  if (st != SPEC_OK) return st;
  std::string e;
  if (!encode_map_2d(&g.a_map[0], W, Kdim, N, 128, &e)) return fail(SPEC_EINVAL, e);
  if (!encode_act_maps(g.b_map[0], X, Kdim, M, &e)) return fail(SPEC_EINVAL, e);
  g.out = Y;
  g.ldo = N;
  g.sk_ws = p->scratch;
  g.sk_tickets = p->tickets;
  g.err = p->err;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // tickets start at zero (a completed call leaves them zero; an aborted one might not)
  cudaError_t ce = cudaMemsetAsync(p->tickets, 0, sizeof(int) * g.n_tiles * g.m_tiles, s);
  if (ce != cudaSuccess) return fail(SPEC_ECUDA, std::string("ticket reset: ") + cudaGetErrorString(ce));
  const int grid = g.n_items < num_sms() ? g.n_items : num_sms();
  ce = gemm_launch(EPI_F32, box <= 64 ? 64 : 256, g, grid, s, false);
  if (ce != cudaSuccess) return fail(SPEC_ECUDA, std::string("launch: ") + cudaGetErrorString(ce));
  return SPEC_OK;
}

// The guard flag of this entry point's kernels on the current device (0 if it never ran there),
// cleared after reading.  Called by spec_sync(NULL) after it has waited for the device.
cudaError_t fm::noalloc_take_flag(int* flag) {
  *flag = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64 || !g_dev[dev].ready.load(std::memory_order_acquire)) return e;
  e = cudaMemcpyFromSymbol(flag, g_noalloc_err, sizeof(int));
  if (e == cudaSuccess && *flag != 0) {
    const int zero = 0;
    e = cudaMemcpyToSymbol(g_noalloc_err, &zero, sizeof(int));
  }
  return e;
}
