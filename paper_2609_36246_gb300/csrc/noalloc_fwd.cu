// noalloc_fwd.cu -- olive_token_logprob_fwd_noalloc: the forward log-prob /
// loss call for callers that cannot hand the library any device memory of
// their own.
//
// Who needs it: code that runs inside a host framework whose allocator owns
// every byte of device memory and offers no way to borrow a scratch buffer
// (a plugin or custom operator loaded into another runtime), and callers on a
// latency budget that cannot afford cudaMalloc's implicit device
// synchronisation.  Such callers still pass their inputs and outputs; the
// scratch space the forward needs (compacted hidden rows and per-segment
// log-sum-exp partials) comes from one fixed array compiled into the library.
//
// The array is a file-scope __device__ object of OLIVE_NOALLOC_SCRATCH_BYTES,
// so every GPU that loads the library holds it until the process exits.  Its
// device address is looked up once per device with cudaGetSymbolAddress (the
// host-side name is only a stand-in for it); that lookup happens on the first
// call made on each device, which should therefore come before any stream
// capture.  All calls share the array and it keeps the last call's contents:
// calls whose kernels overlap on the GPU (different streams, or threads
// without ordering) race on it and must be serialised by the caller.  The
// forward writes every scratch byte it later reads (it zero-fills the padded
// rows itself), so nothing has to be cleared between calls.
#include <cmath>
#include <mutex>

#include "internal.h"

namespace olive {
namespace {

constexpr size_t kNoallocScratchBytes = OLIVE_NOALLOC_SCRATCH_BYTES;

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (set-up on the
// first call per device).
olive_status scratch_address(int device, void** out) {
  if (device < 0 || device >= kMaxDevices) return OLIVE_ERR_UNSUPPORTED_DEVICE;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[device] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return OLIVE_ERR_CUDA;
    }
    g_scratch_addr[device] = p;
  }
  *out = g_scratch_addr[device];
  return OLIVE_OK;
}

bool is_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace olive

extern "C" OLIVE_API olive_status olive_token_logprob_fwd_noalloc(
    const void* hidden, const void* W, const int32_t* targets, const int32_t* rows,
    const int32_t* n_rows, int32_t T, int32_t d, int32_t V, float inv_tau, int reduction,
    float* logp, float* lse, float* loss, int32_t* dev_status, void* stream) {
  using namespace olive;
  if (!hidden || !W || !targets || !rows || !n_rows || !logp || !lse || !loss || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (reduction != OLIVE_REDUCE_SUM && reduction != OLIVE_REDUCE_MEAN) return OLIVE_ERR_INVALID_ARG;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > (1 << 20)) return OLIVE_ERR_SHAPE;
  if (d % 8 != 0 || !is_aligned16(hidden) || !is_aligned16(W)) return OLIVE_ERR_ALIGNMENT;
  // the whole scratch of this call must fit the fixed array
  if (fwd_ws_bytes(T, d) > kNoallocScratchBytes) return OLIVE_ERR_SHAPE;
  Ctx c;
  olive_status st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  void* ws = nullptr;
  st = scratch_address(c.device, &ws);
  if (st != OLIVE_OK) return st;
  return launch_logprob_fwd(c, hidden, W, targets, rows, n_rows, T, d, V, inv_tau, reduction,
                            logp, lse, loss, ws, dev_status);
}
