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
constexpr int CAND_THREADS = 256;
constexpr long long SEL_SMEM_BITMAP_WORDS = 8192;   // positions up to 262,144: bitmap built in shared memory

// Radix-select step over a 256-bin histogram, run by one full warp: the largest digit d with
// (count of bins above d) < need <= (count of bins at or above d). Lane l owns bins 255 - 8l .. 248 - 8l.
// Writes d and the count above it to *d_out / *above_out (digit 0 if fewer than `need` keys remain).
__device__ __forceinline__ void pick_digit_desc(const unsigned int* hist, unsigned int need, unsigned int* d_out,
                                                unsigned int* above_out, unsigned int* count_out) {
  const int lane = threadIdx.x & 31;
  unsigned int v[8], sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) { v[i] = hist[255 - 8 * lane - i]; sum += v[i]; }
  unsigned int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  const unsigned int excl = incl - sum;
  const unsigned int hit = __ballot_sync(0xffffffffu, excl < need && need <= incl);
  const int src = hit ? __ffs(hit) - 1 : 31;
  if (lane == src) {
    unsigned int acc = excl, d = 255 - 8 * lane - 7, cnt = v[7];
    if (hit) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (acc + v[i] >= need) { d = 255 - 8 * lane - i; cnt = v[i]; break; }
        acc += v[i];
      }
    } else {
      acc = incl - v[7];
    }
    *d_out = d;
    *above_out = acc;
    if (count_out) *count_out = cnt;
  }
}

// Same, ascending: the smallest digit d with (count below d) < need <= (count at or below d).
__device__ __forceinline__ void pick_digit_asc(const unsigned int* hist, unsigned int need, unsigned int* d_out,
                                               unsigned int* below_out) {
  const int lane = threadIdx.x & 31;
  unsigned int v[8], sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) { v[i] = hist[8 * lane + i]; sum += v[i]; }
  unsigned int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  const unsigned int excl = incl - sum;
  const unsigned int hit = __ballot_sync(0xffffffffu, excl < need && need <= incl);
  const int src = hit ? __ffs(hit) - 1 : 0;
  if (lane == src) {
    unsigned int acc = excl, d = 8 * lane;
    if (hit) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (acc + v[i] >= need) { d = 8 * lane + i; break; }
        acc += v[i];
      }
    }
    *d_out = d;
    *below_out = acc;
  }
}

// Key sources for the ordered selection: scores stored in memory, or recomputed from the RoPE columns or the digest
// (the exact fallback of the fused path: a[u] = qt[0:r] . key_u[0:r] in fp32, qt already in shared memory).
struct StoredKeys {
  const float* a;
  __device__ __forceinline__ float operator()(int u) const { return a[u]; }
};
struct RecomputedKeys {
  const __nv_bfloat16* rows;    // this sequence's RoPE rows (r = 64) or digest rows
  int64_t ld;
  const float* qt;              // 64 floats in shared memory
  int r;                        // key width, a multiple of 8
  __device__ __forceinline__ float operator()(int u) const {
    const uint4* rp = reinterpret_cast<const uint4*>(rows + (int64_t)u * ld);
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (8 * i >= r) break;
      const uint4 w = rp[i];
      acc = fmaf(qt[8 * i + 0], bf_lo(w.x), acc); acc = fmaf(qt[8 * i + 1], bf_hi(w.x), acc);
      acc = fmaf(qt[8 * i + 2], bf_lo(w.y), acc); acc = fmaf(qt[8 * i + 3], bf_hi(w.y), acc);
      acc = fmaf(qt[8 * i + 4], bf_lo(w.z), acc); acc = fmaf(qt[8 * i + 5], bf_hi(w.z), acc);
      acc = fmaf(qt[8 * i + 6], bf_lo(w.w), acc); acc = fmaf(qt[8 * i + 7], bf_hi(w.w), acc);
    }
    return acc;
  }
};

// Ascending ids of the set bits of wbm[0, nw), written to out[base ...] (entries past cap are dropped). Each warp
// takes a contiguous range of words, counts its bits, one barrier shares the warps' totals, then every warp
// writes its ids in groups of eight 32-word chunks: the eight chunks' warp prefix sums run interleaved (one scan
// latency per group, not per chunk), then each lane writes the ids of its word in every chunk -- a sparse word bit
// by bit, a full word (the window, sinks) by the whole warp, one id per lane. Returns base + the number of set
// bits. Called by the whole block (blockDim a multiple of 32, at most 1024); scratch holds 32 ints.
__device__ __forceinline__ int bitmap_to_ids(const uint32_t* wbm, long long nw, int32_t* out, int base, int cap,
                                             int* scratch) {
  constexpr int GC = 8;                              // chunks per group
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
  const long long per = ((nw + nwarp - 1) / nwarp + 31) / 32 * 32;   // words per warp, whole chunks
  const long long w0 = (long long)w * per, w1 = min(nw, w0 + per);
  int cnt = 0;
  for (long long i = w0 + lane; i < w1; i += 32) cnt += __popc(wbm[i]);
  cnt = __reduce_add_sync(0xffffffffu, cnt);
  __syncthreads();                                   // scratch may still be read by an earlier caller
  if (lane == 0) scratch[w] = cnt;
  __syncthreads();
  int pos = base, total = 0;
  for (int i = 0; i < nwarp; ++i) {
    const int c = scratch[i];
    if (i < w) pos += c;
    total += c;
  }
  for (long long g0 = w0; g0 < w1; g0 += 32 * GC) {
    uint32_t wv[GC];
    int n[GC], inc[GC];
#pragma unroll
    for (int j = 0; j < GC; ++j) {
      const long long i = g0 + 32 * j + lane;
      wv[j] = i < w1 ? wbm[i] : 0u;
      n[j] = __popc(wv[j]);
      inc[j] = n[j];
    }
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
#pragma unroll
      for (int j = 0; j < GC; ++j) {
        const int y = __shfl_up_sync(0xffffffffu, inc[j], d);
        if (lane >= d) inc[j] += y;
      }
    }
#pragma unroll
    for (int j = 0; j < GC; ++j) {
      const long long c0 = g0 + 32 * j;
      const int p0 = pos + inc[j] - n[j];
      const bool full = wv[j] == 0xffffffffu;
      int p = p0;
      uint32_t bits = full ? 0u : wv[j];
      while (bits) {
        const int b = __ffs(bits) - 1;
        bits &= bits - 1;
        if (p < cap) out[p] = (int32_t)((c0 + lane) * 32 + b);
        ++p;
      }
      uint32_t fl = __ballot_sync(0xffffffffu, full);
      while (fl) {
        const int src = __ffs(fl) - 1;
        fl &= fl - 1;
        const int ps = __shfl_sync(0xffffffffu, p0, src) + lane;
        if (ps < cap) out[ps] = (int32_t)((c0 + src) * 32 + lane);
      }
      pos += __shfl_sync(0xffffffffu, inc[j], 31);
    }
  }
  return base + total;
}

// Block-wide AND and OR of one value per thread (scratch: 2 x 32 words). Every thread gets both.
__device__ __forceinline__ void block_and_or(uint32_t& a, uint32_t& o, uint32_t* scratch) {
  a = __reduce_and_sync(0xffffffffu, a);
  o = __reduce_or_sync(0xffffffffu, o);
  const int w = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) { scratch[w] = a; scratch[32 + w] = o; }
  __syncthreads();
  a = 0xffffffffu;
  o = 0u;
  for (int i = 0; i < nwarp; ++i) { a &= scratch[i]; o |= scratch[32 + i]; }
}

// The k-th largest of n keys (1 <= k <= n) by radix select in 8-bit digits that start at the keys' highest
// differing bit (bits above it are common to all keys, so they take no pass and pile into no single bin).
// With max_passes < 4 the result is the lower bound of the bucket reached (a key <= the k-th largest).
// Returns the key; *need_out = how many keys equal to it are among the k (exact result only); *ties_out = how
// many keys fall in its final bucket. Called by the whole block; each_key(f) calls f(key) for every key this
// thread holds (in registers, shared or global memory). With mask_out, the select stops as soon as the bucket
// holding the k-th largest key holds exactly the keys still needed: the k largest are then the keys whose bits
// under *mask_out are >= the returned prefix (*need_out == *ties_out).
template <class EachKey>
__device__ uint32_t radix_kth_desc(const EachKey& each_key, int n, unsigned int k, unsigned int* hist,
                                   uint32_t* scratch, unsigned int* need_out, unsigned int* ties_out,
                                   int max_passes = 8, uint32_t* mask_out = nullptr) {
  __shared__ unsigned int s_digit, s_above, s_cnt;
  uint32_t kand = 0xffffffffu, kor = 0u;
  each_key([&](uint32_t key) { kand &= key; kor |= key; });
  block_and_or(kand, kor, scratch);
  const uint32_t diff = kand ^ kor;
  if (diff == 0u) {                                   // all keys equal
    *need_out = k;
    *ties_out = (unsigned int)n;
    if (mask_out) *mask_out = 0xffffffffu;
    return kand;
  }
  int hb = 31 - __clz(diff);                          // highest differing bit
  uint32_t prefix = hb == 31 ? 0u : (kand & ~((2u << hb) - 1u));
  uint32_t mask = hb == 31 ? 0u : ~((2u << hb) - 1u);
  unsigned int need = k, ties = 0;
  for (int pass = 0;; ++pass) {
    const int shift = max(hb - 7, 0);
    const uint32_t dmask = (2u << (hb - shift)) - 1u;   // digit of hb - shift + 1 <= 8 bits
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    each_key([&](uint32_t key) {
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & dmask], 1u);
    });
    __syncthreads();
    if (threadIdx.x < 32) pick_digit_desc(hist, need, &s_digit, &s_above, &s_cnt);
    __syncthreads();
    prefix |= s_digit << shift;
    mask |= dmask << shift;
    need -= s_above;
    ties = s_cnt;
    __syncthreads();
    if (shift == 0 || pass + 1 >= max_passes || (mask_out && ties == need)) break;
    hb = shift - 1;
  }
  *need_out = need;
  *ties_out = ties;
  if (mask_out) *mask_out = mask;
  return prefix;
}

// Ordered per-head selection over positions [0, N) (one CTA): the k largest keys of the archive [lo, hi) by
// (key desc, position asc), plus -- unless `append` -- every position outside the archive (sinks, window).
// Writes the ascending id list (after count[bh] entries when appending), the bitmap words, count and kth.
template <class Keys>
__device__ void select_ordered(const Keys& key_of, int N, int lo, int hi, long long k, int32_t* out, int32_t* count_bh,
                               int cap, int append, float* kth_bh, uint32_t* bitmap_bh, long long nw, int* status) {
  __shared__ unsigned int hist[256];
  __shared__ unsigned int s_prefix, s_need, s_digit, s_above;
  __shared__ int scan_scratch[33];
  unsigned int prefix = 0, mask = 0, need = (unsigned int)k;
  if (k > 0) {
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
      __syncthreads();
      for (int u = lo + threadIdx.x; u < hi; u += blockDim.x) {
        const uint32_t key = fkey(key_of(u));
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x < 32) pick_digit_desc(hist, need, &s_digit, &s_above, nullptr);
      __syncthreads();
      if (threadIdx.x == 0) {
        s_prefix = prefix | (s_digit << shift);
        s_need = need - s_above;
      }
      __syncthreads();
      prefix = s_prefix;
      need = s_need;
      mask |= 255u << shift;
      __syncthreads();
    }
  }
  const uint32_t tau = prefix;   // the k-th largest key; `need` of the keys equal to it are kept (smallest u first)

  int base = append ? *count_bh : 0;
  int ties_seen = 0;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int c = 0; c < N; c += blockDim.x) {
    const int u = c + threadIdx.x;
    bool in = false, tie = false;
    if (u < N) {
      if (u < lo || u >= hi) {
        in = !append;
      } else if (k > 0) {
        const uint32_t key = fkey(key_of(u));
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
    if (bitmap_bh) {
      const uint32_t word = __ballot_sync(0xffffffffu, in);
      const int w = (c >> 5) + warp;
      if (lane == 0 && (long long)w < nw) bitmap_bh[w] = word;
    }
  }
  if (threadIdx.x == 0) {
    *count_bh = base;
    if (kth_bh && !append) *kth_bh = k > 0 ? funkey(tau) : INFINITY;
    if (base > cap) raise_status(status, VK_ERR_CAPACITY);
  }
}

__global__ void __launch_bounds__(SEL_THREADS) k_select_dense(
    int H, int N, const float* __restrict__ scores, const long long* __restrict__ k_per_head, long long k_all,
    int W, int n_sink, int32_t* __restrict__ idx, int32_t* __restrict__ count, int cap, int append,
    float* __restrict__ kth, uint32_t* __restrict__ bitmap, long long nw, int* status) {
  const int64_t bh = blockIdx.x;
  const int lo = n_sink, hi = N - W;
  long long k = k_all;
  if (k_per_head) k = min(k, k_per_head[bh]);
  if (k > (long long)max(0, hi - lo)) k = max(0, hi - lo);
  StoredKeys keys{scores + bh * (int64_t)N};
  select_ordered(keys, N, lo, hi, k, idx + bh * (int64_t)cap, count + bh, cap, append, kth ? kth + bh : nullptr,
                 bitmap ? bitmap + bh * nw : nullptr, nw, status);
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

// ---------------------------------------------------------------------------------------------- fused path
// Threshold from a strided sample of the archive: theta[b,h] = the j-th largest sampled score, so that about
// j * stride archive rows score >= theta (chosen well above k). The candidate pass then emits only those rows.
// sample[(b*H + h) * ns + i] is the score of position off + stride * i, in bf16 (theta only steers how many
// candidates pass; the candidates themselves carry fp32 scores). Up to THETA_R x NT archive samples are held in
// registers (THETA_R per thread, loaded together); more go through shared memory (ns x 4 bytes). NT = 128 (four
// warps per head, about ten blocks resident per SM) while the samples fit, else 256: at B = 64, N = 65536, H = 64
// the pass takes 21 us with four warps per head against 34 us with eight (the blocks are latency-bound, so more of
// them in flight pays). Measured slower: one warp per head with exact two-pass 8-bit histograms of the 16-bit bf16 keys
// (43-47 us: a head's scores share a few exponents, so the first pass's shared-memory atomics pile onto a few
// buckets), the same with the lanes of a bucket aggregated by match_any (102 us), match_any aggregation in the
// eight-warp block (48 us), and a binary search over the keys with a block-wide count per step (45 us).
constexpr int THETA_R = 16;
template <int NT>
__global__ void __launch_bounds__(NT) k_theta(int ns, int ld, int off, int stride, int lo, int hi, int j,
                                                        const __nv_bfloat16* __restrict__ sample,
                                                        float* __restrict__ theta, int* __restrict__ zero_cnt) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ unsigned int hist[256];
  __shared__ uint32_t scratch[64];
  const int64_t bh = blockIdx.x;
  if (zero_cnt && threadIdx.x == 0) zero_cnt[bh] = 0;  // the candidate pass that follows counts from zero
  const __nv_bfloat16* a = sample + bh * (int64_t)ld;
  // sampled positions off + stride * i inside [lo, hi) are a contiguous index range [i0, i1)
  const int i0 = lo > off ? (lo - off + stride - 1) / stride : 0;
  const int i1 = min(ns, hi > off ? (hi - off + stride - 1) / stride : 0);
  const int na = max(0, i1 - i0);
  if (j <= 0 || j > na) {
    if (threadIdx.x == 0) theta[bh] = -INFINITY;      // emit every archive row
    return;
  }
  unsigned int need_eq, ties;
  // two digits below the samples' first differing bit pin the j-th largest to a bucket of 2^-16 of their key
  // range; its lower bound is theta (a little below the exact order statistic: a few more candidates pass)
  uint32_t prefix;
  if (na <= THETA_R * NT) {
    uint32_t kr[THETA_R];
#pragma unroll
    for (int r = 0; r < THETA_R; ++r) {
      const int e = threadIdx.x + r * NT;
      kr[r] = fkey(e < na ? __bfloat162float(a[i0 + e]) : 0.f);
    }
    auto each_key = [&](auto f) {
#pragma unroll
      for (int r = 0; r < THETA_R; ++r)
        if (threadIdx.x + r * NT < na) f(kr[r]);
    };
    prefix = radix_kth_desc(each_key, na, (unsigned int)j, hist, scratch, &need_eq, &ties, 2);
  } else {
    uint32_t* keys = reinterpret_cast<uint32_t*>(smem);         // the archive samples' keys
    for (int i = threadIdx.x; i < na; i += 16 * NT) {
      float v[16];
#pragma unroll
      for (int r = 0; r < 16; ++r) {
        const int e = i + r * NT;
        v[r] = e < na ? __bfloat162float(a[i0 + e]) : 0.f;
      }
#pragma unroll
      for (int r = 0; r < 16; ++r) {
        const int e = i + r * NT;
        if (e < na) keys[e] = fkey(v[r]);
      }
    }
    __syncthreads();
    auto each_key = [&](auto f) {
      for (int i = threadIdx.x; i < na; i += NT) f(keys[i]);
    };
    prefix = radix_kth_desc(each_key, na, (unsigned int)j, hist, scratch, &need_eq, &ties, 2);
  }
  if (threadIdx.x == 0) theta[bh] = funkey(prefix);
}

cudaError_t launch_theta(int B, int H, int ns, int ld, int off, int stride, int lo, int hi, int j, const void* sample,
                         float* theta, cudaStream_t st, int* zero_cnt) {
  // four warps per head while the samples fit their registers (2048), else eight (4096); past that, shared memory
  const bool small = ns <= THETA_R * 128;
  const int nt = small ? 128 : 256;
  const size_t smem = ns > THETA_R * nt ? (size_t)ns * 4 : 0;
  auto kern = small ? k_theta<128> : k_theta<256>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<B * H, nt, smem, st>>>(ns, ld, off, stride, lo, hi, j, static_cast<const __nv_bfloat16*>(sample), theta,
                                zero_cnt);
  count_launches(1);
  return cudaGetLastError();
}

// The selection proper from a head's candidates: the k-th largest key tau by radix select, then -- when more
// keys equal tau than are needed -- the `need` smallest positions among the tied ones by a second radix select
// on positions; the selected rows (plus sinks and window unless appending) become the head's bitmap and its
// ascending id list. each_kp(f) calls f(key, position) for every candidate this thread holds.
template <class EachKP>
__device__ void select_from_candidates(const EachKP& each_kp, int c, long long k, int N, int lo, int hi, int append,
                                       uint32_t* sbm, uint32_t* bm, long long nw, int32_t* out, int32_t* count_bh,
                                       int cap, float* kth_bh, int* status) {
  __shared__ unsigned int hist[256];
  __shared__ uint32_t scratch[64];
  __shared__ unsigned int s_digit, s_above;
  __shared__ int scan_scratch[33];
  auto each_key = [&](auto f) { each_kp([&](uint32_t key, uint32_t) { f(key); }); };
  unsigned int prefix = 0, need = (unsigned int)k, ties = 0;
  uint32_t pos_cut = 0xffffffffu;
  uint32_t kmask = 0xffffffffu;   // the bits of a key compared with the threshold
  if (k > 0) {
    // without a k-th key to report, stop once the bucket of the k-th key is taken whole
    prefix = radix_kth_desc(each_key, c, (unsigned int)k, hist, scratch, &need, &ties, 8, kth_bh ? nullptr : &kmask);
    if (ties > need) {
      // among keys equal to tau keep the `need` smallest positions: find the need-th smallest of them
      unsigned int pprefix = 0, pmask = 0, pneed = need;
      for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
        __syncthreads();
        each_kp([&](uint32_t key, uint32_t p) {
          if (key == prefix && (p & pmask) == pprefix) atomicAdd(&hist[(p >> shift) & 255u], 1u);
        });
        __syncthreads();
        if (threadIdx.x < 32) pick_digit_asc(hist, pneed, &s_digit, &s_above);
        __syncthreads();
        pprefix |= s_digit << shift;
        pneed -= s_above;
        pmask |= 255u << shift;
        __syncthreads();
      }
      pos_cut = pprefix;
    }
  }
  const uint32_t tau = prefix;
  // bitmap (built in shared memory when it fits): clear, then set sinks and window (tier 1) and the selected
  // candidates, then write it out
  uint32_t* wbm = sbm ? sbm : bm;
  for (long long w = threadIdx.x; w < nw; w += blockDim.x) wbm[w] = 0u;
  __syncthreads();
  if (!append) {
    for (int u = threadIdx.x; u < lo; u += blockDim.x) atomicOr(&wbm[u >> 5], 1u << (u & 31));
    for (int u = hi + threadIdx.x; u < N; u += blockDim.x) atomicOr(&wbm[u >> 5], 1u << (u & 31));
  }
  if (k > 0) {
    each_kp([&](uint32_t key, uint32_t p) {
      const uint32_t km = key & kmask;
      if (km > tau || (km == tau && p <= pos_cut)) atomicOr(&wbm[p >> 5], 1u << (p & 31));
    });
  }
  __syncthreads();
  if (wbm != bm)
    for (long long w = threadIdx.x; w < nw; w += blockDim.x) bm[w] = wbm[w];
  // ascending ids from the bitmap
  const int base = bitmap_to_ids(wbm, nw, out, append ? *count_bh : 0, cap, scan_scratch);
  if (threadIdx.x == 0) {
    *count_bh = base;
    if (kth_bh && !append) *kth_bh = k > 0 ? funkey(tau) : INFINITY;
    if (base > cap) raise_status(status, VK_ERR_CAPACITY);
  }
}

// Selection from a head's candidate list (every archive row with score >= theta, in arbitrary order). When the
// list holds at least k and at most capc entries it contains the whole top-k (select_from_candidates). The keys
// of lists of up to CAND_R x 256 entries are loaded once into registers (CAND_R per thread, all loads in flight
// together) and every radix pass runs on them; longer lists are re-read from memory (L2-resident after the
// scoring pass) on every pass. The block is latency-bound, so the launch bounds ask for 8 resident blocks per SM
// even though the compiler then keeps part of the state in local memory: for 4096 heads of ~3.2k candidates
// that measured 0.097 ms, against 0.106 ms at 4 blocks per SM without spills and 0.105 ms with the keys in
// shared memory instead. When the list is too short or too long (theta landed too high or too low) or with
// VK_FLAG_FORCE_FALLBACK, the head takes the exact ordered selection over scores recomputed from the RoPE
// columns. With `append` (the top_j of the fired rows, whose list can never overflow) only candidates are
// selected, no sinks or window, and the ids are appended after count[b,h].
constexpr int CAND_R = 16;
__global__ void __launch_bounds__(CAND_THREADS, 8) k_select_cand(
    int H, int N, int lo, int hi, long long k_all, const long long* __restrict__ k_per_head,
    const int* __restrict__ cand_cnt, const int2* __restrict__ cand, int capc, int force_fallback,
    const __nv_bfloat16* __restrict__ rope, int64_t rld, int64_t rbs, int r, const float* __restrict__ qt,
    const __nv_bfloat16* __restrict__ qrope,
    int32_t* __restrict__ idx, int32_t* __restrict__ count, int cap, int append, float* __restrict__ kth,
    uint32_t* __restrict__ bitmap, long long nw, int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  uint32_t* sbm = nw <= SEL_SMEM_BITMAP_WORDS ? reinterpret_cast<uint32_t*>(smem) : nullptr;   // bitmap words
  __shared__ float qts[D_ROPE];
  const int64_t bh = blockIdx.x;
  const int b = (int)(bh / H);
  long long k = k_all;
  if (k_per_head) k = min(k, k_per_head[bh]);
  const int c = cand_cnt[bh];
  if (append) k = min(k, (long long)c);
  uint32_t* bm = bitmap + bh * nw;
  int32_t* out = idx + bh * (int64_t)cap;
  float* kth_bh = kth ? kth + bh : nullptr;

  if (force_fallback || c < k || c > capc) {
    if (append) {                       // cannot happen: the fired list has room for the whole archive
      if (threadIdx.x == 0) raise_status(status, VK_ERR_CAPACITY);
      return;
    }
    // the scoring query: qt from the query prep when it ran, else (r = 64: no rotation) the RoPE query itself
    for (int i = threadIdx.x; i < D_ROPE; i += blockDim.x)
      qts[i] = qt ? qt[bh * D_ROPE + i] : __bfloat162float(qrope[bh * D_ROPE + i]);
    __syncthreads();
    RecomputedKeys keys{rope + (int64_t)b * rbs, rld, qts, r};
    select_ordered(keys, N, lo, hi, k, out, count + bh, cap, 0, kth_bh, bm, nw, status);
    return;
  }

  const int2* g = cand + bh * (int64_t)capc;
  if (c <= CAND_R * CAND_THREADS) {
    // keys in registers; a position is read back from the list only where a pass needs it (ties, marking)
    uint32_t kr[CAND_R];
#pragma unroll
    for (int r = 0; r < CAND_R; ++r) {
      const int i = threadIdx.x + r * CAND_THREADS;
      kr[r] = fkey(i < c ? __int_as_float(g[i].y) : 0.f);
    }
    auto each_kp = [&](auto f) {
#pragma unroll
      for (int r = 0; r < CAND_R; ++r) {
        const int i = threadIdx.x + r * CAND_THREADS;
        if (i < c) f(kr[r], (uint32_t)g[i].x);
      }
    };
    select_from_candidates(each_kp, c, k, N, lo, hi, append, sbm, bm, nw, out, count + bh, cap, kth_bh, status);
  } else {
    auto each_kp = [&](auto f) {
      for (int i = threadIdx.x; i < c; i += CAND_THREADS) {
        const int2 e = g[i];
        f(fkey(__int_as_float(e.y)), (uint32_t)e.x);
      }
    };
    select_from_candidates(each_kp, c, k, N, lo, hi, append, sbm, bm, nw, out, count + bh, cap, kth_bh, status);
  }
}

cudaError_t launch_select_cand(int B, int H, int N, int lo, int hi, int64_t k, const int64_t* k_per_head,
                               const int* cand_cnt, const int2* cand, int capc, int force_fallback, const vk_view& v,
                               int r, const void* digest, const float* qt, int32_t* idx, int32_t* count, int cap,
                               int append, float* kth, uint32_t* bitmap, int64_t nw, int* status, cudaStream_t st) {
  const size_t smem = nw <= SEL_SMEM_BITMAP_WORDS ? (size_t)nw * 4 : 0;
  cudaError_t e = cudaFuncSetAttribute(k_select_cand, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_select_cand<<<B * H, CAND_THREADS, smem, st>>>(
      H, N, lo, hi, (long long)k, reinterpret_cast<const long long*>(k_per_head), cand_cnt, cand, capc,
      force_fallback,
      r == D_ROPE ? static_cast<const __nv_bfloat16*>(v.rope) : static_cast<const __nv_bfloat16*>(digest),
      r == D_ROPE ? v.rope_ld : (int64_t)r, r == D_ROPE ? v.rope_bstride : (int64_t)v.N * r, r, qt,
      static_cast<const __nv_bfloat16*>(v.q_rope), idx, count, cap,
      append, kth, bitmap, (long long)nw, status);
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
  int32_t* out = idx + bh * (int64_t)cap;
  const int base = bitmap_to_ids(bitmap + bh * nw, nw, out, count[bh], cap, scan_scratch);
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
