// k_select.cu -- per-head top-k over materialised scores, and id-list <-> bitmap conversions.
//
// Selection (Sec. 4.1: keep the top rows of the archive plus sinks and the recent window; ties go to the
// smaller position): one CTA per (b, h) finds the k-th largest order-preserving key of the archive
// [n_sink, N-W) by a 4 x 8-bit radix select, then makes one ordered pass over all positions that keeps
// sinks, window, keys above the threshold and the first `need` keys equal to it, writing the ascending id
// list and the 32-bit bitmap words at once.
#include "vk_common.cuh"

namespace vk {

constexpr int SEL_THREADS = 512;

__global__ void __launch_bounds__(SEL_THREADS) k_select_dense(
    int H, int N, const float* __restrict__ scores, const long long* __restrict__ k_per_head, long long k_all,
    int W, int n_sink, int32_t* __restrict__ idx, int32_t* __restrict__ count, int cap, int append,
    float* __restrict__ kth, uint32_t* __restrict__ bitmap, long long nw, int* status) {
  __shared__ unsigned int hist[256];
  __shared__ unsigned int s_prefix, s_need;
  __shared__ int scan_scratch[33];
  const int64_t bh = blockIdx.x;
  const float* a = scores + bh * (int64_t)N;
  const int lo = n_sink, hi = N - W;
  long long k = k_all;
  if (k_per_head) k = min(k, k_per_head[bh]);
  if (k > (long long)max(0, hi - lo)) k = max(0, hi - lo);

  unsigned int prefix = 0, mask = 0, need = (unsigned int)k;
  if (k > 0) {
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
      __syncthreads();
      for (int u = lo + threadIdx.x; u < hi; u += blockDim.x) {
        const uint32_t key = fkey(a[u]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        unsigned int above = 0;
        int d = 255;
        for (; d > 0; --d) {
          if (above + hist[d] >= need) break;
          above += hist[d];
        }
        s_prefix = prefix | ((unsigned int)d << shift);
        s_need = need - above;
      }
      __syncthreads();
      prefix = s_prefix;
      need = s_need;
      mask |= 255u << shift;
      __syncthreads();
    }
  }
  const uint32_t tau = prefix;   // the k-th largest key; `need` of the keys equal to it are kept

  int base = append ? count[bh] : 0;
  const int start_base = base;
  int ties_seen = 0;
  int32_t* out = idx + bh * (int64_t)cap;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int c = 0; c < N; c += blockDim.x) {
    const int u = c + threadIdx.x;
    bool in = false, tie = false;
    if (u < N) {
      if (u < lo || u >= hi) {
        in = !append;      // sinks and window are part of S_h, not of an appended list
      } else if (k > 0) {
        const uint32_t key = fkey(a[u]);
        if (key > tau) in = true;
        else if (key == tau) tie = true;
      }
    }
    int tot;
    const int tie_rank = ties_seen + block_exclusive_scan(tie ? 1 : 0, scan_scratch, &tot);
    ties_seen += tot;
    if (tie && tie_rank < (int)need) in = true;
    const int pos = base + block_exclusive_scan(in ? 1 : 0, scan_scratch, &tot);
    if (in && pos < cap) out[pos] = u;
    base += tot;
    if (bitmap) {
      const uint32_t word = __ballot_sync(0xffffffffu, in);
      const int w = (c >> 5) + warp;
      if (lane == 0 && (long long)w < nw) bitmap[bh * nw + w] = word;
    }
  }
  if (threadIdx.x == 0) {
    count[bh] = base;
    if (kth && !append) kth[bh] = k > 0 ? funkey(tau) : INFINITY;
    if (base > cap) raise_status(status, VK_ERR_CAPACITY);
    (void)start_base;
  }
}

cudaError_t launch_select_dense(int B, int H, int N, const float* scores, const int64_t* k_per_head, int64_t k,
                                int W, int n_sink, int32_t* idx, int32_t* count, int cap, int append, float* kth,
                                uint32_t* bitmap, int64_t nw, int* status, cudaStream_t st) {
  k_select_dense<<<B * H, SEL_THREADS, 0, st>>>(H, N, scores, reinterpret_cast<const long long*>(k_per_head),
                                                (long long)k, W, n_sink, idx, count, cap, append, kth, bitmap,
                                                (long long)nw, status);
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- lists
// Ascending list from a bitmap, appended after count[b,h] entries (count grows by the popcount).
__global__ void __launch_bounds__(SEL_THREADS) k_bitmap_to_list(int N, const uint32_t* __restrict__ bitmap,
                                                                long long nw, int32_t* __restrict__ idx,
                                                                int32_t* __restrict__ count, int cap, int* status) {
  __shared__ int scan_scratch[33];
  const int64_t bh = blockIdx.x;
  int base = count[bh];
  int32_t* out = idx + bh * (int64_t)cap;
  for (long long c = 0; c < nw; c += blockDim.x) {
    const long long w = c + threadIdx.x;
    const uint32_t word = (w < nw) ? bitmap[bh * nw + w] : 0u;
    int tot;
    int pos = base + block_exclusive_scan(__popc(word), scan_scratch, &tot);
    uint32_t bits = word;
    while (bits) {
      const int i = __ffs(bits) - 1;
      bits &= bits - 1;
      if (pos < cap) out[pos] = (int32_t)(w * 32 + i);
      ++pos;
    }
    base += tot;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (base > cap) raise_status(status, VK_ERR_CAPACITY);
    count[bh] = base;
  }
}

cudaError_t launch_bitmap_to_list(int B, int H, int N, const uint32_t* bitmap, int64_t nw, int32_t* idx,
                                  int32_t* count, int cap, int* status, cudaStream_t st) {
  k_bitmap_to_list<<<B * H, SEL_THREADS, 0, st>>>(N, bitmap, (long long)nw, idx, count, cap, status);
  count_launches(1);
  return cudaGetLastError();
}

// Bitmap from caller-given id lists; ids outside [0, N) are skipped and flag VK_ERR_INVALID_ARG.
__global__ void k_list_to_bitmap(int N, const int32_t* __restrict__ idx, const int32_t* __restrict__ count,
                                 int cap, uint32_t* __restrict__ bitmap, long long nw, int* status) {
  const int64_t bh = blockIdx.y;
  const int n = min(count[bh], cap);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const int u = idx[bh * (int64_t)cap + i];
    if (u < 0 || u >= N) { raise_status(status, VK_ERR_INVALID_ARG); continue; }
    atomicOr(&bitmap[bh * nw + (u >> 5)], 1u << (u & 31));
  }
}

cudaError_t launch_list_to_bitmap(int B, int H, int N, const int32_t* idx, const int32_t* count, int cap,
                                  uint32_t* bitmap, int64_t nw, int* status, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(bitmap, 0, sizeof(uint32_t) * nw * B * H, st);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)(cap > 64 * 256 ? 64 : (cap + 255) / 256 + 1), B * H);
  k_list_to_bitmap<<<grid, 256, 0, st>>>(N, idx, count, cap, bitmap, (long long)nw, status);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
