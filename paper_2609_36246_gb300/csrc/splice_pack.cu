// splice_pack.cu -- builds the packed student-update batch of Section 3.1:
// every sequence is prefix_s (prompt x and student prefix y_{1:k}) followed by
// the teacher continuation y~_{1:l}; row t predicts packed token t+1 of the
// same sequence, and only rows whose target is a continuation token carry a
// term of Eq. (osd-ce).
//
// Two launches, integer work only:
//   scan   one block: validates the CSR offsets, writes cu_seqlens,
//          cut_offsets and n_rows (= sum_s C_s); on malformed input it
//          zeroes them so the fill kernel clears every output.
//   fill   one thread per packed position t < T_cap: finds its sequence by
//          binary search over cu_seqlens and writes ids, targets, the loss
//          mask and, for masked rows, rows[cont_off[s] + j] = t (the j-th
//          continuation token of sequence s is predicted by row cut_s - 1 + j,
//          so rows come out ascending with no scan over the mask).
//
// Multi-turn variant (Section 3.2: the loss covers only the teacher's
// actions; student turns and environment observations stay as context): a
// flag per continuation token selects the rows, so the row list needs a scan
// over the packed stream.  It runs scan, then per 2048-position chunk a count,
// one block that turns the chunk counts into offsets, and a fill that writes
// each chunk's masked rows after a block-wide scan.
#include "internal.h"

namespace olive {
namespace {

constexpr int kScanThreads = 1024;

__device__ __forceinline__ long long block_excl_scan(long long v, long long* total, long long* sh) {
  // inclusive scan of one value per thread, 1024 threads
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  long long x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    long long w = sh[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;
  }
  __syncthreads();
  const long long before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[31];
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(kScanThreads)
    splice_scan_kernel(const int32_t* __restrict__ prefix_off, const int32_t* __restrict__ cont_off,
                       int S, int T_cap, int32_t* __restrict__ cu, int32_t* __restrict__ cut,
                       int32_t* __restrict__ n_rows, int32_t* dev_status) {
  __shared__ long long sh[32];
  __shared__ int bad;
  if (threadIdx.x == 0) bad = (prefix_off[0] != 0 || cont_off[0] != 0) ? 1 : 0;
  __syncthreads();
  // pass 1: validate lengths and totals
  long long tot_len = 0, tot_c = 0;
  for (int b = 0; b < S; b += kScanThreads) {
    const int s = b + threadIdx.x;
    long long L = 0, C = 0;
    if (s < S) {
      const long long P = static_cast<long long>(prefix_off[s + 1]) - prefix_off[s];
      C = static_cast<long long>(cont_off[s + 1]) - cont_off[s];
      if (P < 1 || C < 0) bad = 1;
      L = P + C;
    }
    long long t1, t2;
    block_excl_scan(L, &t1, sh);
    block_excl_scan(C, &t2, sh);
    tot_len += t1;
    tot_c += t2;
  }
  __syncthreads();
  if (tot_len > T_cap) bad = 1;
  __syncthreads();
  if (bad) {
    for (int s = threadIdx.x; s <= S; s += kScanThreads) {
      cu[s] = 0;
      if (s < S) cut[s] = 0;
    }
    if (threadIdx.x == 0) {
      *n_rows = 0;
      atomicOr(dev_status, 1 << OLIVE_ERR_OFFSETS);
    }
    return;
  }
  // pass 2: exclusive scan of L_s = P_s + C_s
  long long carry = 0;
  for (int b = 0; b < S; b += kScanThreads) {
    const int s = b + threadIdx.x;
    long long L = 0, P = 0;
    if (s < S) {
      P = static_cast<long long>(prefix_off[s + 1]) - prefix_off[s];
      L = P + (static_cast<long long>(cont_off[s + 1]) - cont_off[s]);
    }
    long long tot;
    const long long before = block_excl_scan(L, &tot, sh);
    if (s < S) {
      cu[s] = static_cast<int32_t>(carry + before);
      cut[s] = static_cast<int32_t>(carry + before + P);
    }
    carry += tot;
  }
  if (threadIdx.x == 0) {
    cu[S] = static_cast<int32_t>(carry);
    *n_rows = static_cast<int32_t>(tot_c);
  }
}

__global__ void splice_fill_kernel(const int32_t* __restrict__ prefix_ids,
                                   const int32_t* __restrict__ prefix_off,
                                   const int32_t* __restrict__ cont_ids,
                                   const int32_t* __restrict__ cont_off, int S, int V, int T_cap,
                                   const int32_t* __restrict__ cu, const int32_t* __restrict__ n_rows,
                                   int32_t* __restrict__ ids, int32_t* __restrict__ targets,
                                   uint8_t* __restrict__ loss_mask, int32_t* __restrict__ rows,
                                   int32_t* dev_status) {
  const int T = cu[S];
  const int nr = *n_rows;
  bool range_bad = false;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T_cap; t += gridDim.x * blockDim.x) {
    if (t >= nr) rows[t] = -1;
    if (t >= T) {
      ids[t] = 0;
      targets[t] = -1;
      loss_mask[t] = 0;
      continue;
    }
    // sequence s with cu[s] <= t < cu[s+1]
    int lo = 0, hi = S;  // invariant: cu[lo] <= t < cu[hi]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (cu[mid] <= t) lo = mid; else hi = mid;
    }
    const int s = lo;
    const int i = t - cu[s];
    const int L = cu[s + 1] - cu[s];
    const int P = prefix_off[s + 1] - prefix_off[s];
    const int id = i < P ? prefix_ids[prefix_off[s] + i] : cont_ids[cont_off[s] + (i - P)];
    ids[t] = id;
    if (id < 0 || id >= V) range_bad = true;
    int tgt = -1;
    uint8_t m = 0;
    if (i + 1 < L) {
      const int j = i + 1;
      tgt = j < P ? prefix_ids[prefix_off[s] + j] : cont_ids[cont_off[s] + (j - P)];
      if (j >= P) {
        m = 1;
        rows[cont_off[s] + (j - P)] = t;
      }
    }
    targets[t] = tgt;
    loss_mask[t] = m;
  }
  if (range_bad) atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
}

constexpr int kChunk = 2048;        // packed positions per block (masked variant)
constexpr int kChunkThreads = 256;  // 8 positions per thread

struct PosInfo {
  int id, tgt;
  bool masked;
};

// Id, target and multi-turn loss flag of packed position t < T.
__device__ __forceinline__ PosInfo position_info(int t, int S, const int32_t* __restrict__ cu,
                                                 const int32_t* __restrict__ prefix_ids,
                                                 const int32_t* __restrict__ prefix_off,
                                                 const int32_t* __restrict__ cont_ids,
                                                 const int32_t* __restrict__ cont_off,
                                                 const uint8_t* __restrict__ cont_loss) {
  int lo = 0, hi = S;  // cu[lo] <= t < cu[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (cu[mid] <= t) lo = mid; else hi = mid;
  }
  const int s = lo;
  const int i = t - cu[s];
  const int L = cu[s + 1] - cu[s];
  const int P = prefix_off[s + 1] - prefix_off[s];
  PosInfo r;
  r.id = i < P ? prefix_ids[prefix_off[s] + i] : cont_ids[cont_off[s] + (i - P)];
  r.tgt = -1;
  r.masked = false;
  if (i + 1 < L) {
    const int j = i + 1;
    r.tgt = j < P ? prefix_ids[prefix_off[s] + j] : cont_ids[cont_off[s] + (j - P)];
    r.masked = j >= P && cont_loss[cont_off[s] + (j - P)] != 0;
  }
  return r;
}

__device__ __forceinline__ int block_excl_scan_int(int v, int* total, int* sh) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int w = lane < nw ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;
  }
  __syncthreads();
  const int before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(kChunkThreads)
    turns_count_kernel(const int32_t* __restrict__ prefix_ids, const int32_t* __restrict__ prefix_off,
                       const int32_t* __restrict__ cont_ids, const int32_t* __restrict__ cont_off,
                       const uint8_t* __restrict__ cont_loss, int S, const int32_t* __restrict__ cu,
                       int32_t* __restrict__ chunk_count) {
  __shared__ int sh[32];
  const int T = cu[S];
  const int t0 = blockIdx.x * kChunk + threadIdx.x * (kChunk / kChunkThreads);
  int c = 0;
  for (int q = 0; q < kChunk / kChunkThreads; ++q) {
    const int t = t0 + q;
    if (t < T) c += position_info(t, S, cu, prefix_ids, prefix_off, cont_ids, cont_off, cont_loss).masked;
  }
  int total;
  block_excl_scan_int(c, &total, sh);
  if (threadIdx.x == 0) chunk_count[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanThreads)
    turns_offsets_kernel(int32_t* __restrict__ chunk_count, int n_chunks, int32_t* __restrict__ n_rows) {
  __shared__ int sh[32];
  int carry = 0;
  for (int b = 0; b < n_chunks; b += kScanThreads) {
    const int k = b + threadIdx.x;
    const int v = k < n_chunks ? chunk_count[k] : 0;
    int total;
    const int before = block_excl_scan_int(v, &total, sh);
    if (k < n_chunks) chunk_count[k] = carry + before;
    carry += total;
  }
  if (threadIdx.x == 0) *n_rows = carry;
}

__global__ void __launch_bounds__(kChunkThreads)
    turns_fill_kernel(const int32_t* __restrict__ prefix_ids, const int32_t* __restrict__ prefix_off,
                      const int32_t* __restrict__ cont_ids, const int32_t* __restrict__ cont_off,
                      const uint8_t* __restrict__ cont_loss, int S, int V, int T_cap,
                      const int32_t* __restrict__ cu, const int32_t* __restrict__ chunk_offset,
                      const int32_t* __restrict__ n_rows, int32_t* __restrict__ ids,
                      int32_t* __restrict__ targets, uint8_t* __restrict__ loss_mask,
                      int32_t* __restrict__ rows, int32_t* dev_status) {
  __shared__ int sh[32];
  constexpr int kPer = kChunk / kChunkThreads;
  const int T = cu[S];
  const int nr = *n_rows;
  const int t0 = blockIdx.x * kChunk + threadIdx.x * kPer;
  bool range_bad = false;
  uint32_t bits = 0;
  for (int q = 0; q < kPer; ++q) {
    const int t = t0 + q;
    if (t >= T_cap) break;
    if (t >= nr) rows[t] = -1;
    if (t >= T) {
      ids[t] = 0;
      targets[t] = -1;
      loss_mask[t] = 0;
      continue;
    }
    const PosInfo r = position_info(t, S, cu, prefix_ids, prefix_off, cont_ids, cont_off, cont_loss);
    ids[t] = r.id;
    if (r.id < 0 || r.id >= V) range_bad = true;
    targets[t] = r.tgt;
    loss_mask[t] = r.masked ? 1 : 0;
    if (r.masked) bits |= 1u << q;
  }
  int total;
  int at = chunk_offset[blockIdx.x] + block_excl_scan_int(__popc(bits), &total, sh);
  for (int q = 0; q < kPer; ++q)
    if (bits & (1u << q)) rows[at++] = t0 + q;
  if (range_bad) atomicOr(dev_status, 1 << OLIVE_ERR_TOKEN_RANGE);
}

}  // namespace

olive_status launch_splice_pack(const Ctx& c, const int32_t* prefix_ids, const int32_t* prefix_off,
                                const int32_t* cont_ids, const int32_t* cont_off, int32_t S,
                                int32_t V, int32_t T_cap, int32_t* ids, int32_t* targets,
                                uint8_t* loss_mask, int32_t* cu_seqlens, int32_t* cut_offsets,
                                int32_t* rows, int32_t* n_rows, int32_t* dev_status) {
  splice_scan_kernel<<<1, kScanThreads, 0, c.stream>>>(prefix_off, cont_off, S, T_cap, cu_seqlens,
                                                       cut_offsets, n_rows, dev_status);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  const int64_t want = ceil_div(T_cap, 256);
  const int blocks = static_cast<int>(want < c.num_sms * 16LL ? want : c.num_sms * 16LL);
  splice_fill_kernel<<<blocks, 256, 0, c.stream>>>(prefix_ids, prefix_off, cont_ids, cont_off, S, V,
                                                   T_cap, cu_seqlens, n_rows, ids, targets,
                                                   loss_mask, rows, dev_status);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  return OLIVE_OK;
}

}  // namespace olive

namespace olive {

size_t splice_masked_ws_bytes(int64_t T_cap) {
  return align_up(sizeof(int32_t) * static_cast<size_t>(ceil_div(T_cap, kChunk)), kWsAlign);
}

olive_status launch_splice_pack_masked(const Ctx& c, const int32_t* prefix_ids,
                                       const int32_t* prefix_off, const int32_t* cont_ids,
                                       const int32_t* cont_off, const uint8_t* cont_loss, int32_t S,
                                       int32_t V, int32_t T_cap, int32_t* ids, int32_t* targets,
                                       uint8_t* loss_mask, int32_t* cu_seqlens,
                                       int32_t* cut_offsets, int32_t* rows, int32_t* n_rows,
                                       void* ws, int32_t* dev_status) {
  int32_t* chunk = static_cast<int32_t*>(ws);
  const int n_chunks = static_cast<int>(ceil_div(T_cap, kChunk));
  splice_scan_kernel<<<1, kScanThreads, 0, c.stream>>>(prefix_off, cont_off, S, T_cap, cu_seqlens,
                                                       cut_offsets, n_rows, dev_status);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  turns_count_kernel<<<n_chunks, kChunkThreads, 0, c.stream>>>(prefix_ids, prefix_off, cont_ids,
                                                               cont_off, cont_loss, S, cu_seqlens,
                                                               chunk);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  turns_offsets_kernel<<<1, kScanThreads, 0, c.stream>>>(chunk, n_chunks, n_rows);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  turns_fill_kernel<<<n_chunks, kChunkThreads, 0, c.stream>>>(
      prefix_ids, prefix_off, cont_ids, cont_off, cont_loss, S, V, T_cap, cu_seqlens, chunk, n_rows,
      ids, targets, loss_mask, rows, dev_status);
  if (cudaGetLastError() != cudaSuccess) return OLIVE_ERR_CUDA;
  return OLIVE_OK;
}

}  // namespace olive
