// olive_api.cu -- the extern "C" entry points of libolive.so (include/olive.h):
// host-side argument checks, workspace layout, device checks and the
// tensor-map encoder.  All compute is in the kernels of the other files.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
#include <mutex>

#include "internal.h"

namespace olive {

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

uint64_t wait_limit_from_env() {
  // OLIVE_WAIT_LIMIT_MS bounds every internal wait of the GEMM kernels
  // (default 1000 ms; 0 makes the first unsatisfied wait give up, which the
  // tests use to exercise the timeout path).
  const char* s = std::getenv("OLIVE_WAIT_LIMIT_MS");
  if (!s || !*s) return 1000ull * 1000ull * 1000ull;
  char* end = nullptr;
  const unsigned long long ms = std::strtoull(s, &end, 10);
  if (end == s) return 1000ull * 1000ull * 1000ull;
  return static_cast<uint64_t>(ms) * 1000ull * 1000ull;
}

}  // namespace

olive_status make_ctx(void* stream, Ctx* ctx) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return OLIVE_ERR_CUDA;
  }
  int major = 0, minor = 0, sms = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return OLIVE_ERR_CUDA;
  }
  if (major != 10 || minor != 3) return OLIVE_ERR_UNSUPPORTED_DEVICE;
  if (!encode_fn()) return OLIVE_ERR_CUDA;
  ctx->stream = static_cast<cudaStream_t>(stream);
  ctx->device = dev;
  ctx->num_sms = sms;
  ctx->wait_limit_ns = wait_limit_from_env();
  return OLIVE_OK;
}

bool set_smem_once(const void* func, int smem, int device, std::atomic<int>* done) {
  const bool cached = device >= 0 && device < kMaxDevices;
  if (cached && done[device].load(std::memory_order_acquire) == smem) return true;
  if (cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return false;
  if (cached) done[device].store(smem, std::memory_order_release);
  return true;
}

static bool encode_bf16_2d_swz(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer,
                               CUtensorMapSwizzle swz) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                    uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return encode_bf16_2d_swz(map, base, inner, outer, row_bytes, box_inner, box_outer,
                            CU_TENSOR_MAP_SWIZZLE_128B);
}

bool encode_bf16_2d_plain(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return encode_bf16_2d_swz(map, base, inner, outer, row_bytes, box_inner, box_outer,
                            CU_TENSOR_MAP_SWIZZLE_NONE);
}

int64_t slab_rows(int64_t Tpad, int64_t V) {
  // G buffer of at most ~5.6 GB (bf16), in whole 128-row tiles, <= 32768 rows;
  // OLIVE_SLAB_ROWS (a multiple of 128) can lower the cap, e.g. to exercise
  // several slabs on small inputs
  const int64_t budget = 5600ll * 1000 * 1000;
  int64_t tc = budget / (2 * vpad(V)) / kRowAlign * kRowAlign;
  if (tc < kRowAlign) tc = kRowAlign;
  if (tc > 32768) tc = 32768;
  if (const char* e = std::getenv("OLIVE_SLAB_ROWS")) {
    const long long cap = std::atoll(e);
    if (cap >= kRowAlign && cap % kRowAlign == 0 && cap < tc) tc = cap;
  }
  if (tc > Tpad) tc = Tpad;
  return tc;
}

// ------------------------------------------------------------- workspace ---
namespace {
struct Carver {
  char* base;
  size_t off = 0;
  void* take(size_t bytes) {
    void* p = base ? base + off : nullptr;
    off = align_up(off + bytes, kWsAlign);
    return p;
  }
};
}  // namespace

static FwdWs carve_fwd_impl(void* ws, int64_t T, int64_t d, size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  Carver c{static_cast<char*>(ws)};
  FwdWs w;
  w.hc = c.take(2ull * Tpad * d);
  w.part_m = static_cast<float*>(c.take(4ull * kSvMax * Tpad));
  w.part_s = static_cast<float*>(c.take(4ull * kSvMax * Tpad));
  w.zy = static_cast<float*>(c.take(4ull * Tpad));
  w.nll = static_cast<float*>(c.take(4ull * Tpad));
  if (total) *total = c.off;
  return w;
}
size_t fwd_ws_bytes(int64_t T, int64_t d) {
  size_t n = 0;
  carve_fwd_impl(nullptr, T, d, &n);
  return n;
}
FwdWs carve_fwd(void* ws, int64_t T, int64_t d) { return carve_fwd_impl(ws, T, d, nullptr); }

static TopkWs carve_topk_impl(void* ws, int64_t T, int64_t d, size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  Carver c{static_cast<char*>(ws)};
  TopkWs w;
  w.hc = c.take(2ull * Tpad * d);
  w.part_m = static_cast<float*>(c.take(4ull * kSvMax * Tpad));
  w.part_s = static_cast<float*>(c.take(4ull * kSvMax * Tpad));
  w.part_a = static_cast<float*>(c.take(4ull * kSvMax * Tpad));
  w.part_tv = static_cast<float*>(c.take(4ull * 16 * kSvMax * Tpad));
  w.part_ti = static_cast<int32_t*>(c.take(4ull * 16 * kSvMax * Tpad));
  if (total) *total = c.off;
  return w;
}
size_t topk_ws_bytes(int64_t T, int64_t d) {
  size_t n = 0;
  carve_topk_impl(nullptr, T, d, &n);
  return n;
}
TopkWs carve_topk(void* ws, int64_t T, int64_t d) { return carve_topk_impl(ws, T, d, nullptr); }

static BwdWs carve_bwd_impl(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype,
                            size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  Carver c{static_cast<char*>(ws)};
  BwdWs w;
  w.tc = slab_rows(Tpad, V);
  w.hc = c.take(2ull * Tpad * d);
  w.g = c.take(2ull * w.tc * vpad(V));
  w.dw_acc = grad_dtype == OLIVE_DTYPE_BF16 ? static_cast<float*>(c.take(4ull * V * d)) : nullptr;
  w.counters = static_cast<uint32_t*>(c.take(4ull * bwd_counter_words(Tpad, w.tc)));
  if (total) *total = c.off;
  return w;
}
size_t bwd_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype) {
  size_t n = 0;
  carve_bwd_impl(nullptr, T, d, V, grad_dtype, &n);
  return n;
}
BwdWs carve_bwd(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype) {
  return carve_bwd_impl(ws, T, d, V, grad_dtype, nullptr);
}

static OpdWs carve_opd_impl(void* ws, int64_t T, int64_t ds, int64_t dt, size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const size_t lst = 4ull * 16 * kSvMax * Tpad;
  Carver c{static_cast<char*>(ws)};
  OpdWs w;
  w.hcs = c.take(2ull * Tpad * ds);
  w.hct = c.take(2ull * Tpad * dt);
  w.part = static_cast<float*>(c.take(4ull * 6 * kSvMax * Tpad));
  w.part_sv = static_cast<float*>(c.take(lst));
  w.part_si = static_cast<int32_t*>(c.take(lst));
  w.part_sx = static_cast<float*>(c.take(lst));
  w.part_tv = static_cast<float*>(c.take(lst));
  w.part_ti = static_cast<int32_t*>(c.take(lst));
  if (total) *total = c.off;
  return w;
}
size_t opd_ws_bytes(int64_t T, int64_t ds, int64_t dt) {
  size_t n = 0;
  carve_opd_impl(nullptr, T, ds, dt, &n);
  return n;
}
OpdWs carve_opd(void* ws, int64_t T, int64_t ds, int64_t dt) {
  return carve_opd_impl(ws, T, ds, dt, nullptr);
}

static FbWs carve_fb_impl(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype,
                          size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const int64_t vh = ceil_div(V, 128);  // partials per 128-column half tile
  Carver c{static_cast<char*>(ws)};
  FbWs w;
  w.tc = slab_rows(Tpad, V);
  w.hc = c.take(2ull * Tpad * d);
  w.g = c.take(2ull * w.tc * vpad(V));
  w.part_zm = static_cast<float*>(c.take(4ull * w.tc * vh));
  w.part_zs = static_cast<float*>(c.take(4ull * w.tc * vh));
  w.zy = static_cast<float*>(c.take(4ull * w.tc));
  w.nll = static_cast<float*>(c.take(4ull * Tpad));
  w.dw_acc = grad_dtype == OLIVE_DTYPE_BF16 ? static_cast<float*>(c.take(4ull * V * d)) : nullptr;
  w.zref = static_cast<float*>(c.take(8ull * w.tc));
  w.lam = static_cast<float*>(c.take(4ull * w.tc));
  w.hs = c.take(2ull * Tpad * d);
  if (total) *total = c.off;
  return w;
}
size_t fb_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype) {
  size_t n = 0;
  carve_fb_impl(nullptr, T, d, V, grad_dtype, &n);
  return n;
}
FbWs carve_fb(void* ws, int64_t T, int64_t d, int64_t V, int grad_dtype) {
  return carve_fb_impl(ws, T, d, V, grad_dtype, nullptr);
}

// the backward's regions, then coef [T] and val [T, 16] of the top-K KL gradient
size_t topk_kl_bwd_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype) {
  return bwd_ws_bytes(T, d, V, grad_dtype) + align_up(4ull * T, kWsAlign) +
         align_up(4ull * 16 * T, kWsAlign);
}

// the fused forward + backward's regions, then the true half-tile maxima
// [tc, ceil(V/128)] of the slab rows
size_t topk_kl_fb_ws_bytes(int64_t T, int64_t d, int64_t V, int grad_dtype) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  return fb_ws_bytes(T, d, V, grad_dtype) +
         align_up(4ull * slab_rows(Tpad, V) * ceil_div(V, 128), kWsAlign);
}

static GroupWs carve_group_impl(void* ws, int64_t T, int64_t d, int64_t V, size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const int64_t rt = Tpad / kRowAlign;
  const int gmax = group_g_max(d);
  Carver c{static_cast<char*>(ws)};
  GroupWs w;
  w.hc = c.take(2ull * Tpad * d);
  w.rref = static_cast<float*>(c.take(4ull * Tpad));
  w.rmax = static_cast<float*>(c.take(4ull * Tpad));
  w.zy = static_cast<float*>(c.take(4ull * Tpad));
  w.pyb = static_cast<float*>(c.take(4ull * Tpad));
  w.nll = static_cast<float*>(c.take(4ull * Tpad));
  w.part_s = static_cast<float*>(c.take(4ull * gmax * Tpad));
  w.part_m = static_cast<float*>(c.take(4ull * gmax * Tpad));
  w.ring = c.take(group_ring_bytes(T, d, V));
  // counters in one region, zeroed by one memset per column sweep: group
  // barriers [2 rt] (first and redo launch), the redo list [1 + rt], then the
  // ring counters of the three launches of a sweep
  const size_t rw = group_ctr_words(T, d, V);
  w.ctr_words = static_cast<size_t>(3 * rt + 1) + 3 * rw;
  uint32_t* ctr = static_cast<uint32_t*>(c.take(4ull * w.ctr_words));
  w.outer = ctr;
  w.redo = ctr ? ctr + 2 * rt : nullptr;
  w.ring_ctr = ctr ? ctr + 3 * rt + 1 : nullptr;
  if (total) *total = c.off;
  return w;
}
size_t group_ws_bytes(int64_t T, int64_t d, int64_t V) {
  size_t n = 0;
  carve_group_impl(nullptr, T, d, V, &n);
  return n;
}
GroupWs carve_group(void* ws, int64_t T, int64_t d, int64_t V) {
  return carve_group_impl(ws, T, d, V, nullptr);
}

static KlWs carve_kl_impl(void* ws, int64_t T, int64_t ds, int64_t dt, int64_t V, int grad,
                          size_t* total) {
  const int64_t Tpad = align_up(static_cast<size_t>(T), kRowAlign);
  const int64_t rt = Tpad / kRowAlign;
  Carver c{static_cast<char*>(ws)};
  KlWs w = {};
  w.hcs = c.take(2ull * Tpad * ds);
  w.hct = c.take(2ull * Tpad * dt);
  w.part = static_cast<float*>(c.take(4ull * 5 * kSvMax * Tpad));
  if (grad) {
    w.lse_p = static_cast<float*>(c.take(4ull * Tpad));
    w.lse_q = static_cast<float*>(c.take(4ull * Tpad));
    w.ring = c.take(group_ring_bytes(T, ds, V));
    // the same counter layout as the training step's (group barriers and
    // redo list unused here), so every sweep's launch has its ring counters
    w.ctr_words = static_cast<size_t>(3 * rt + 1) + 3 * group_ctr_words(T, ds, V);
    w.ctr = static_cast<uint32_t*>(c.take(4ull * w.ctr_words));
  }
  if (total) *total = c.off;
  return w;
}
size_t kl_ws_bytes(int64_t T, int64_t ds, int64_t dt, int64_t V, int grad) {
  size_t n = 0;
  carve_kl_impl(nullptr, T, ds, dt, V, grad, &n);
  return n;
}
KlWs carve_kl(void* ws, int64_t T, int64_t ds, int64_t dt, int64_t V, int grad) {
  return carve_kl_impl(ws, T, ds, dt, V, grad, nullptr);
}

}  // namespace olive

using namespace olive;

namespace {

constexpr int32_t kMaxDim = 1 << 20;  // widths above this are rejected

olive_status check_ws(void* ws, size_t have, size_t need) {
  if (need == 0) return OLIVE_ERR_SHAPE;
  if (!ws || have < need || (reinterpret_cast<uintptr_t>(ws) & (kWsAlign - 1)) != 0)
    return OLIVE_ERR_WORKSPACE;
  return OLIVE_OK;
}

bool width_ok(int32_t d) { return d >= 8 && d <= kMaxDim && (d % 8) == 0; }

}  // namespace

extern "C" {

int olive_abi_version(void) { return OLIVE_ABI_VERSION; }

int32_t olive_slab_rows(int32_t T, int32_t V) {
  if (T < 1 || V < 1) return 0;
  return static_cast<int32_t>(slab_rows(align_up(static_cast<size_t>(T), kRowAlign), V));
}

const char* olive_status_string(olive_status s) {
  switch (s) {
    case OLIVE_OK: return "ok";
    case OLIVE_ERR_INVALID_ARG: return "invalid argument (null pointer or bad enum)";
    case OLIVE_ERR_SHAPE: return "invalid shape";
    case OLIVE_ERR_ALIGNMENT: return "pointer or width breaks the 16-byte rule";
    case OLIVE_ERR_TOKEN_RANGE: return "token id or target outside [0, V)";
    case OLIVE_ERR_OFFSETS: return "malformed offsets or row list";
    case OLIVE_ERR_TIMEOUT: return "an internal wait ran out of time";
    case OLIVE_ERR_UNSUPPORTED_DEVICE: return "device is not compute capability 10.3";
    case OLIVE_ERR_CUDA: return "CUDA call failed";
    case OLIVE_ERR_WORKSPACE: return "workspace null, misaligned or too small";
    case OLIVE_ERR_BOUNDS: return "a device index check failed (OLIVE_DEBUG build)";
  }
  return "unknown status";
}

size_t olive_workspace_size(int op, int32_t T, int32_t d, int32_t d_t, int32_t V, int grad,
                            int grad_dtype) {
  if (op == OLIVE_OP_SPLICE_MASKED) return T < 1 ? 0 : splice_masked_ws_bytes(T);
  if (T < 1 || V < 1 || !width_ok(d)) return 0;
  switch (op) {
    case OLIVE_OP_LOGPROB_FWD: return fwd_ws_bytes(T, d);
    case OLIVE_OP_LOSS_BWD:
      if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return 0;
      return group_ws_bytes(T, d, V);
    case OLIVE_OP_DIVERGENCE:
      if (!width_ok(d_t)) return 0;
      return kl_ws_bytes(T, d, d_t, V, grad);
    case OLIVE_OP_TOPK_FWD: return topk_ws_bytes(T, d);
    case OLIVE_OP_LOSS_FWD_BWD:
      if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return 0;
      return group_ws_bytes(T, d, V);
    case OLIVE_OP_LOSS_FWD_BWD_SLAB:
      if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return 0;
      return fb_ws_bytes(T, d, V, grad_dtype);
    case OLIVE_OP_OPD_STATS:
      if (!width_ok(d_t)) return 0;
      return opd_ws_bytes(T, d, d_t);
    case OLIVE_OP_TOPK_KL_BWD:
      if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return 0;
      return topk_kl_bwd_ws_bytes(T, d, V, grad_dtype);
    case OLIVE_OP_TOPK_KL_FWD_BWD:
      if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return 0;
      return topk_kl_fb_ws_bytes(T, d, V, grad_dtype);
    default: return 0;
  }
}

olive_status olive_splice_pack(const int32_t* prefix_ids, const int32_t* prefix_off,
                               const int32_t* cont_ids, const int32_t* cont_off, int32_t S,
                               int32_t V, int32_t T_cap, int32_t* ids, int32_t* targets,
                               uint8_t* loss_mask, int32_t* cu_seqlens, int32_t* cut_offsets,
                               int32_t* rows, int32_t* n_rows, int32_t* dev_status, void* stream) {
  if (!prefix_ids || !prefix_off || !cont_ids || !cont_off || !ids || !targets || !loss_mask ||
      !cu_seqlens || !cut_offsets || !rows || !n_rows || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (S < 1 || V < 1 || T_cap < 1) return OLIVE_ERR_SHAPE;
  Ctx c;
  olive_status st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_splice_pack(c, prefix_ids, prefix_off, cont_ids, cont_off, S, V, T_cap, ids,
                            targets, loss_mask, cu_seqlens, cut_offsets, rows, n_rows, dev_status);
}

olive_status olive_splice_pack_masked(const int32_t* prefix_ids, const int32_t* prefix_off,
                                      const int32_t* cont_ids, const int32_t* cont_off,
                                      const uint8_t* cont_loss, int32_t S, int32_t V, int32_t T_cap,
                                      int32_t* ids, int32_t* targets, uint8_t* loss_mask,
                                      int32_t* cu_seqlens, int32_t* cut_offsets, int32_t* rows,
                                      int32_t* n_rows, void* workspace, size_t ws_bytes,
                                      int32_t* dev_status, void* stream) {
  if (!prefix_ids || !prefix_off || !cont_ids || !cont_off || !cont_loss || !ids || !targets ||
      !loss_mask || !cu_seqlens || !cut_offsets || !rows || !n_rows || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (S < 1 || V < 1 || T_cap < 1) return OLIVE_ERR_SHAPE;
  olive_status st = check_ws(workspace, ws_bytes, splice_masked_ws_bytes(T_cap));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_splice_pack_masked(c, prefix_ids, prefix_off, cont_ids, cont_off, cont_loss, S, V,
                                   T_cap, ids, targets, loss_mask, cu_seqlens, cut_offsets, rows,
                                   n_rows, workspace, dev_status);
}

olive_status olive_token_logprob_fwd(const void* hidden, const void* W, const int32_t* targets,
                                     const int32_t* rows, const int32_t* n_rows, int32_t T,
                                     int32_t d, int32_t V, float inv_tau, int reduction,
                                     float* logp, float* lse, float* loss, void* workspace,
                                     size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!hidden || !W || !targets || !rows || !n_rows || !logp || !lse || !loss || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (reduction != OLIVE_REDUCE_SUM && reduction != OLIVE_REDUCE_MEAN) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(hidden) || !aligned16(W)) return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, fwd_ws_bytes(T, d));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_logprob_fwd(c, hidden, W, targets, rows, n_rows, T, d, V, inv_tau, reduction, logp,
                            lse, loss, workspace, dev_status);
}

olive_status olive_token_topk_fwd(const void* hidden, const void* W, const int32_t* rows,
                                  const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                                  float inv_tau, int32_t K, float* lse, float* entropy,
                                  float* topk_logp, int32_t* topk_ids, void* workspace,
                                  size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!hidden || !W || !rows || !n_rows || !lse || !entropy || !topk_logp || !topk_ids ||
      !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim || K < 1 || K > 16 || K > V) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(hidden) || !aligned16(W)) return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, topk_ws_bytes(T, d));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_topk_fwd(c, hidden, W, rows, n_rows, T, d, V, inv_tau, K, lse, entropy, topk_logp,
                         topk_ids, workspace, dev_status);
}

olive_status olive_topk_compare(const void* h_t, const void* W_t, int32_t d_t,
                                const int32_t* rows, const int32_t* n_rows, int32_t T, int32_t V,
                                float inv_tau, int32_t K, const int32_t* s_ids,
                                const float* s_logp, const int32_t* t_ids, const float* t_lse,
                                float* overlap, float* kl_topk, float* t_logp_s,
                                int32_t* dev_status, void* stream) {
  if (!h_t || !W_t || !rows || !n_rows || !s_ids || !s_logp || !t_ids || !t_lse || !overlap ||
      !kl_topk || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d_t < 1 || d_t > kMaxDim || K < 1 || K > 16 || K > V) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d_t % 8 != 0 || !aligned16(h_t) || !aligned16(W_t)) return OLIVE_ERR_ALIGNMENT;
  Ctx c;
  olive_status st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_topk_compare(c, h_t, W_t, d_t, rows, n_rows, T, V, inv_tau, K, s_ids, s_logp,
                             t_ids, t_lse, overlap, kl_topk, t_logp_s, dev_status);
}

olive_status olive_topk_kl_bwd(const void* h_s, const void* W_s, const int32_t* rows,
                               const int32_t* n_rows, int32_t T, int32_t d, int32_t V,
                               float inv_tau, int32_t K, const float* s_lse, const int32_t* s_ids,
                               const float* s_logp, const float* t_logp_s, const float* kl_topk,
                               const float* grad_kl, void* d_h_s, void* d_W_s, int grad_dtype,
                               void* workspace, size_t ws_bytes, int32_t* dev_status,
                               void* stream) {
  if (!h_s || !W_s || !rows || !n_rows || !s_lse || !s_ids || !s_logp || !t_logp_s || !kl_topk ||
      !grad_kl || !d_h_s || !d_W_s || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim || K < 1 || K > 16 || K > V) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(h_s) || !aligned16(W_s) || !aligned16(d_h_s) || !aligned16(d_W_s))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, topk_kl_bwd_ws_bytes(T, d, V, grad_dtype));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  char* sparse = static_cast<char*>(workspace) + bwd_ws_bytes(T, d, V, grad_dtype);
  float* coef = reinterpret_cast<float*>(sparse);
  float* val = reinterpret_cast<float*>(sparse + align_up(4ull * T, kWsAlign));
  st = launch_topk_kl_prep(c, rows, n_rows, T, V, inv_tau, K, s_ids, s_logp, t_logp_s, kl_topk,
                           grad_kl, coef, val, dev_status);
  if (st != OLIVE_OK) return st;
  const SparseGrad sg{coef, val, s_ids, K};
  return launch_loss_bwd(c, h_s, W_s, nullptr, rows, n_rows, T, d, V, inv_tau, OLIVE_REDUCE_SUM,
                         s_lse, nullptr, d_h_s, d_W_s, grad_dtype, workspace, dev_status, &sg);
}

olive_status olive_topk_kl_fwd_bwd(const void* h_s, const void* W_s, int32_t d_s, const void* h_t,
                                   const void* W_t, int32_t d_t, const int32_t* rows,
                                   const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                                   int32_t K, const float* t_lse, const int32_t* t_ids,
                                   const float* grad_kl, float* s_lse, int32_t* s_ids,
                                   float* s_logp, float* t_logp_s, float* kl_topk, float* overlap,
                                   void* d_h_s, void* d_W_s, int grad_dtype, void* workspace,
                                   size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!h_s || !W_s || !h_t || !W_t || !rows || !n_rows || !t_lse || !grad_kl || !s_lse ||
      !s_ids || !s_logp || !t_logp_s || !kl_topk || (t_ids && !overlap) || !d_h_s || !d_W_s ||
      !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d_s < 1 || d_s > kMaxDim || d_t < 1 || d_t > kMaxDim || K < 1 ||
      K > 16 || K > V)
    return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d_s % 8 != 0 || d_t % 8 != 0 || !aligned16(h_s) || !aligned16(W_s) || !aligned16(h_t) ||
      !aligned16(W_t) || !aligned16(d_h_s) || !aligned16(d_W_s))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, topk_kl_fb_ws_bytes(T, d_s, V, grad_dtype));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_topk_kl_fwd_bwd(c, h_s, W_s, d_s, h_t, W_t, d_t, rows, n_rows, T, V, inv_tau, K,
                                t_lse, t_ids, grad_kl, s_lse, s_ids, s_logp, t_logp_s, kl_topk,
                                overlap, d_h_s, d_W_s, grad_dtype, workspace, dev_status);
}

olive_status olive_token_loss_bwd(const void* hidden, const void* W, const int32_t* targets,
                                  const int32_t* rows, const int32_t* n_rows, int32_t T, int32_t d,
                                  int32_t V, float inv_tau, int reduction, const float* lse,
                                  const float* grad_loss, void* d_hidden, void* d_W,
                                  int grad_dtype, void* workspace, size_t ws_bytes,
                                  int32_t* dev_status, void* stream) {
  if (!hidden || !W || !targets || !rows || !n_rows || !lse || !grad_loss || !d_hidden || !d_W ||
      !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (reduction != OLIVE_REDUCE_SUM && reduction != OLIVE_REDUCE_MEAN) return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(hidden) || !aligned16(W) || !aligned16(d_hidden) || !aligned16(d_W))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, group_ws_bytes(T, d, V));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_loss_group(c, hidden, W, targets, rows, n_rows, T, d, V, inv_tau, reduction,
                           grad_loss, lse, nullptr, nullptr, nullptr, d_hidden, d_W, grad_dtype,
                           workspace, dev_status);
}

olive_status olive_token_loss_fwd_bwd(const void* hidden, const void* W, const int32_t* targets,
                                      const int32_t* rows, const int32_t* n_rows, int32_t T,
                                      int32_t d, int32_t V, float inv_tau, int reduction,
                                      const float* grad_loss, float* logp, float* lse, float* loss,
                                      void* d_hidden, void* d_W, int grad_dtype, void* workspace,
                                      size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!hidden || !W || !targets || !rows || !n_rows || !grad_loss || !logp || !lse || !loss ||
      !d_hidden || !d_W || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (reduction != OLIVE_REDUCE_SUM && reduction != OLIVE_REDUCE_MEAN) return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(hidden) || !aligned16(W) || !aligned16(d_hidden) || !aligned16(d_W))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, group_ws_bytes(T, d, V));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_loss_group(c, hidden, W, targets, rows, n_rows, T, d, V, inv_tau, reduction,
                           grad_loss, nullptr, logp, lse, loss, d_hidden, d_W, grad_dtype,
                           workspace, dev_status);
}

olive_status olive_token_loss_fwd_bwd_slab(const void* hidden, const void* W, const int32_t* targets,
                                           const int32_t* rows, const int32_t* n_rows, int32_t T,
                                           int32_t d, int32_t V, float inv_tau, int reduction,
                                           const float* grad_loss, float* logp, float* lse, float* loss,
                                           void* d_hidden, void* d_W, int grad_dtype, void* workspace,
                                           size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!hidden || !W || !targets || !rows || !n_rows || !grad_loss || !logp || !lse || !loss ||
      !d_hidden || !d_W || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if (reduction != OLIVE_REDUCE_SUM && reduction != OLIVE_REDUCE_MEAN) return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d < 1 || d > kMaxDim) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d % 8 != 0 || !aligned16(hidden) || !aligned16(W) || !aligned16(d_hidden) || !aligned16(d_W))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, fb_ws_bytes(T, d, V, grad_dtype));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_loss_fwd_bwd(c, hidden, W, targets, rows, n_rows, T, d, V, inv_tau, reduction,
                             grad_loss, logp, lse, loss, d_hidden, d_W, grad_dtype, workspace,
                             dev_status);
}

olive_status olive_opd_token_stats(const void* h_s, const void* W_s, int32_t d_s, const void* h_t,
                                   const void* W_t, int32_t d_t, const int32_t* rows,
                                   const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                                   int direction, int32_t K, float* kl, float* s_lse, float* t_lse,
                                   float* s_entropy, float* s_topk_logp, int32_t* s_topk_ids,
                                   float* t_logp_s, float* overlap, float* kl_topk,
                                   void* workspace, size_t ws_bytes, int32_t* dev_status,
                                   void* stream) {
  if (!h_s || !W_s || !h_t || !W_t || !rows || !n_rows || !dev_status) return OLIVE_ERR_INVALID_ARG;
  if (!kl && !s_lse && !t_lse && !s_entropy && !s_topk_logp && !s_topk_ids && !t_logp_s &&
      !overlap && !kl_topk)
    return OLIVE_ERR_INVALID_ARG;
  if (direction != OLIVE_KL_REVERSE && direction != OLIVE_KL_FORWARD) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d_s < 1 || d_t < 1 || d_s > kMaxDim || d_t > kMaxDim || K < 1 || K > 16 ||
      K > V)
    return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d_s % 8 != 0 || d_t % 8 != 0 || !aligned16(h_s) || !aligned16(W_s) || !aligned16(h_t) ||
      !aligned16(W_t))
    return OLIVE_ERR_ALIGNMENT;
  olive_status st = check_ws(workspace, ws_bytes, opd_ws_bytes(T, d_s, d_t));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_opd_stats(c, h_s, W_s, d_s, h_t, W_t, d_t, rows, n_rows, T, V, inv_tau, direction,
                          K, kl, s_lse, t_lse, s_entropy, s_topk_logp, s_topk_ids, t_logp_s,
                          overlap, kl_topk, workspace, dev_status);
}

olive_status olive_scale(const void* x, void* y, size_t n, int dtype, const float* scale,
                         void* stream) {
  if (!x || !y || !scale) return OLIVE_ERR_INVALID_ARG;
  if (dtype != OLIVE_DTYPE_BF16 && dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (n < 1) return OLIVE_ERR_SHAPE;
  if (!aligned16(x) || !aligned16(y)) return OLIVE_ERR_ALIGNMENT;
  Ctx c;
  olive_status st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_scale(c, x, y, n, dtype, scale);
}

olive_status olive_token_divergence(const void* h_s, const void* W_s, int32_t d_s, const void* h_t,
                                    const void* W_t, int32_t d_t, const int32_t* rows,
                                    const int32_t* n_rows, int32_t T, int32_t V, float inv_tau,
                                    int direction, float* kl, const float* grad_kl, void* d_h_s,
                                    int grad_dtype, void* workspace, size_t ws_bytes,
                                    int32_t* dev_status, void* stream) {
  if (!h_s || !W_s || !h_t || !W_t || !rows || !n_rows || !kl || !dev_status)
    return OLIVE_ERR_INVALID_ARG;
  if ((grad_kl == nullptr) != (d_h_s == nullptr)) return OLIVE_ERR_INVALID_ARG;
  if (direction != OLIVE_KL_REVERSE && direction != OLIVE_KL_FORWARD) return OLIVE_ERR_INVALID_ARG;
  if (grad_dtype != OLIVE_DTYPE_BF16 && grad_dtype != OLIVE_DTYPE_F32) return OLIVE_ERR_INVALID_ARG;
  if (T < 1 || V < 1 || d_s < 1 || d_t < 1 || d_s > kMaxDim || d_t > kMaxDim) return OLIVE_ERR_SHAPE;
  if (!(inv_tau > 0.f) || !std::isfinite(inv_tau)) return OLIVE_ERR_INVALID_ARG;
  if (d_s % 8 != 0 || d_t % 8 != 0 || !aligned16(h_s) || !aligned16(W_s) || !aligned16(h_t) ||
      !aligned16(W_t) || (d_h_s && !aligned16(d_h_s)))
    return OLIVE_ERR_ALIGNMENT;
  const int grad = d_h_s != nullptr;
  olive_status st = check_ws(workspace, ws_bytes, kl_ws_bytes(T, d_s, d_t, V, grad));
  if (st != OLIVE_OK) return st;
  Ctx c;
  st = make_ctx(stream, &c);
  if (st != OLIVE_OK) return st;
  return launch_divergence(c, h_s, W_s, d_s, h_t, W_t, d_t, rows, n_rows, T, V, inv_tau, direction,
                           kl, grad_kl, d_h_s, grad_dtype, workspace, dev_status);
}

}  // extern "C"
