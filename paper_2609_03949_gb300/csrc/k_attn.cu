// k_attn.cu -- gather + absorbed-MLA attention over per-head selected rows, split over positions, and the
// log-sum-exp merge of the splits (flash-decoding style).
//
// Attention (Eq. 1 with the absorbed query; Lemma 1: the output depends only on the attended multiset):
//   s[h,u] = lambda (Qc_h . L_u + Qr_h . K_u),  out_h = sum_u softmax_u(s) L_u,  lse_h,  s*_h = max_u s.
// Each CTA owns one sequence b, one range of positions and up to 64 heads. It ORs the heads' bitmaps over
// its range into the union of selected rows, copies each union row from HBM once (cp.async, 16-byte
// pieces), and every head that selected the row consumes it from shared memory. Each warp owns a fixed set of
// heads and keeps their running (max, sum, 512-wide accumulator) in registers.
// Splits of the fired rows (two-tier mode) write further partial slots; the combine merges all slots with
// their LSE weights, which is exact because the fired rows are disjoint from the tier-1 rows.
#include "vk_common.cuh"

namespace vk {

constexpr int AT_THREADS = 512;
constexpr int AT_WARPS = AT_THREADS / 32;
constexpr int AT_CHUNK = 16;                       // union rows per pipeline stage
constexpr int AT_HPW = HG / AT_WARPS;              // heads per warp (4)

template <typename T> struct Elem;
template <> struct Elem<__nv_bfloat16> { static constexpr int bytes = 2; };
template <> struct Elem<float> { static constexpr int bytes = 4; };

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// The 18 coordinates lane `lane` owns of a 576-wide row in shared memory: latent [16 lane, 16 lane + 16)
// and RoPE coordinates 2 lane, 2 lane + 1 (stored after the 512 latent values).
__device__ __forceinline__ void load_slice(const __nv_bfloat16* row, int lane, float* x) {
  const uint4 a = *reinterpret_cast<const uint4*>(row + lane * 16);
  const uint4 b = *reinterpret_cast<const uint4*>(row + lane * 16 + 8);
  const uint32_t c = *reinterpret_cast<const uint32_t*>(row + D_LAT + lane * 2);
  x[0] = bf_lo(a.x); x[1] = bf_hi(a.x); x[2] = bf_lo(a.y); x[3] = bf_hi(a.y);
  x[4] = bf_lo(a.z); x[5] = bf_hi(a.z); x[6] = bf_lo(a.w); x[7] = bf_hi(a.w);
  x[8] = bf_lo(b.x); x[9] = bf_hi(b.x); x[10] = bf_lo(b.y); x[11] = bf_hi(b.y);
  x[12] = bf_lo(b.z); x[13] = bf_hi(b.z); x[14] = bf_lo(b.w); x[15] = bf_hi(b.w);
  x[16] = bf_lo(c); x[17] = bf_hi(c);
}
__device__ __forceinline__ void load_slice(const float* row, int lane, float* x) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 v = *reinterpret_cast<const float4*>(row + lane * 16 + 4 * i);
    x[4 * i] = v.x; x[4 * i + 1] = v.y; x[4 * i + 2] = v.z; x[4 * i + 3] = v.w;
  }
  const float2 r = *reinterpret_cast<const float2*>(row + D_LAT + lane * 2);
  x[16] = r.x; x[17] = r.y;
}

template <typename T>
__global__ void __launch_bounds__(AT_THREADS, 1) k_attn_simt(
    const T* __restrict__ latent, int64_t lld, int64_t lbs, const T* __restrict__ rope, int64_t rld, int64_t rbs,
    const T* __restrict__ q_latent, const T* __restrict__ q_rope, int H, int N, float lam,
    const uint32_t* __restrict__ bitmap, int64_t nw, int split_len, int slot0, int nslot, int qrows,
    float* __restrict__ part_o, float* __restrict__ part_ml) {
  constexpr int ROWE = D_LAT + D_ROPE;                     // elements per staged row
  extern __shared__ __align__(16) unsigned char smem_raw[];
  T* qs = reinterpret_cast<T*>(smem_raw);                  // [qrows][576]
  T* rows = qs + qrows * ROWE;                             // [2][AT_CHUNK][576]
  unsigned long long* umask = reinterpret_cast<unsigned long long*>(rows + 2 * AT_CHUNK * ROWE);  // [split_len]
  int32_t* ulist = reinterpret_cast<int32_t*>(umask + split_len);                                // [split_len]
  __shared__ int scan_scratch[33];

  const int split = blockIdx.x, hg = blockIdx.y, b = blockIdx.z;
  const int h0 = hg * HG, nh = min(HG, H - h0);
  const int p0 = split * split_len, p1 = min(N, p0 + split_len);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  // queries of this head group -> shared memory
  for (int i = threadIdx.x; i < nh * (ROWE * Elem<T>::bytes / 16); i += blockDim.x) {
    const int h = i / (ROWE * Elem<T>::bytes / 16), piece = i % (ROWE * Elem<T>::bytes / 16);
    const int e0 = piece * 16 / Elem<T>::bytes;
    const T* src = (e0 < D_LAT) ? q_latent + ((int64_t)b * H + h0 + h) * D_LAT + e0
                                : q_rope + ((int64_t)b * H + h0 + h) * D_ROPE + (e0 - D_LAT);
    *reinterpret_cast<uint4*>(qs + h * ROWE + e0) = *reinterpret_cast<const uint4*>(src);
  }

  // union of the heads' selections over [p0, p1), with each row's 64-bit head mask, in ascending order
  int nU = 0;
  const uint32_t* bm = bitmap + ((int64_t)b * H + h0) * nw;
  for (int c = p0; c < p1; c += blockDim.x) {
    const int u = c + threadIdx.x;
    unsigned long long m = 0ull;
    if (u < p1) {
      const int w = u >> 5, bit = u & 31;
      for (int h = 0; h < nh; ++h) m |= (unsigned long long)((bm[(int64_t)h * nw + w] >> bit) & 1u) << h;
    }
    int tot;
    const int pos = nU + block_exclusive_scan(m ? 1 : 0, scan_scratch, &tot);
    if (m) { ulist[pos] = u; umask[pos] = m; }
    nU += tot;
  }
  __syncthreads();

  // per-warp heads and running softmax state
  float o[AT_HPW][16];
  float mrun[AT_HPW], lrun[AT_HPW];
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) {
    mrun[i] = -INFINITY; lrun[i] = 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j) o[i][j] = 0.f;
  }

  const int nchunks = (nU + AT_CHUNK - 1) / AT_CHUNK;
  constexpr int PIECES_LAT = D_LAT * Elem<T>::bytes / 16, PIECES_ROPE = D_ROPE * Elem<T>::bytes / 16;
  constexpr int PIECES = PIECES_LAT + PIECES_ROPE;
  auto issue = [&](int ch) {
    T* dst = rows + (ch & 1) * AT_CHUNK * ROWE;
    const int r0 = ch * AT_CHUNK, nr = min(AT_CHUNK, nU - r0);
    for (int i = threadIdx.x; i < nr * PIECES; i += blockDim.x) {
      const int j = i / PIECES, piece = i % PIECES;
      const int u = ulist[r0 + j];
      const T* src = (piece < PIECES_LAT)
                         ? latent + (int64_t)b * lbs + (int64_t)u * lld + piece * (16 / Elem<T>::bytes)
                         : rope + (int64_t)b * rbs + (int64_t)u * rld + (piece - PIECES_LAT) * (16 / Elem<T>::bytes);
      cp_async16(dst + j * ROWE + piece * (16 / Elem<T>::bytes), src);
    }
    cp_async_commit();
  };

  if (nchunks > 0) issue(0);
  for (int ch = 0; ch < nchunks; ++ch) {
    if (ch + 1 < nchunks) { issue(ch + 1); cp_async_wait<1>(); } else { cp_async_wait<0>(); }
    __syncthreads();
    const T* buf = rows + (ch & 1) * AT_CHUNK * ROWE;
    const int r0 = ch * AT_CHUNK, nr = min(AT_CHUNK, nU - r0);
    const unsigned long long rmask = (lane < nr) ? umask[r0 + lane] : 0ull;
#pragma unroll
    for (int i = 0; i < AT_HPW; ++i) {
      const int hl = warp + AT_WARPS * i;                   // local head index
      if (hl >= nh) break;
      uint32_t todo = __ballot_sync(0xffffffffu, (rmask >> hl) & 1ull);
      if (!todo) continue;
      float q[18];
      load_slice(qs + hl * ROWE, lane, q);
      while (todo) {
        const int j = __ffs(todo) - 1;
        todo &= todo - 1;
        float x[18];
        load_slice(buf + j * ROWE, lane, x);
        float d = 0.f;
#pragma unroll
        for (int t = 0; t < 18; ++t) d = fmaf(q[t], x[t], d);
#pragma unroll
        for (int off = 16; off; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off);
        const float s = d * lam;
        if (s > mrun[i]) {
          const float sc = __expf(mrun[i] - s);
          lrun[i] *= sc;
#pragma unroll
          for (int t = 0; t < 16; ++t) o[i][t] *= sc;
          mrun[i] = s;
        }
        const float p = __expf(s - mrun[i]);
        lrun[i] += p;
#pragma unroll
        for (int t = 0; t < 16; ++t) o[i][t] = fmaf(p, x[t], o[i][t]);
      }
    }
    __syncthreads();
  }

  // partials: part_o [B][nslot][H][512], part_ml [B][nslot][H][2]
  const int slot = slot0 + split;
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) {
    const int hl = warp + AT_WARPS * i;
    if (hl >= nh) break;
    const int64_t base = (((int64_t)b * nslot + slot) * H + h0 + hl);
    float4* dst = reinterpret_cast<float4*>(part_o + base * D_LAT + lane * 16);
#pragma unroll
    for (int t = 0; t < 4; ++t) dst[t] = make_float4(o[i][4 * t], o[i][4 * t + 1], o[i][4 * t + 2], o[i][4 * t + 3]);
    if (lane == 0) { part_ml[base * 2] = mrun[i]; part_ml[base * 2 + 1] = lrun[i]; }
  }
}

// Dynamic shared memory of one attention CTA: queries, two row stages, the union list and its head masks.
size_t attn_smem_bytes(int dtype, int H, int split_len) {
  const int esz = dtype == VK_BF16 ? 2 : 4;
  return (size_t)(min(H, HG) + 2 * AT_CHUNK) * (D_LAT + D_ROPE) * esz + (size_t)split_len * (4 + 8);
}

cudaError_t launch_attn(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, int nsplit, int split_len,
                        int slot0, int nslot, float* part_o, float* part_ml, cudaStream_t st) {
  dim3 grid(nsplit, (v.H + HG - 1) / HG, v.B);
  const size_t smem = attn_smem_bytes(v.dtype, v.H, split_len);
  const int qrows = min(v.H, HG);
  if (v.dtype == VK_BF16) {
    using T = __nv_bfloat16;
    cudaError_t e = cudaFuncSetAttribute(k_attn_simt<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_attn_simt<T><<<grid, AT_THREADS, smem, st>>>(
        reinterpret_cast<const T*>(v.latent), v.latent_ld, v.latent_bstride, reinterpret_cast<const T*>(v.rope),
        v.rope_ld, v.rope_bstride, reinterpret_cast<const T*>(v.q_latent), reinterpret_cast<const T*>(v.q_rope), v.H,
        v.N, lam, bitmap, nw, split_len, slot0, nslot, qrows, part_o, part_ml);
  } else {
    using T = float;
    cudaError_t e = cudaFuncSetAttribute(k_attn_simt<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_attn_simt<T><<<grid, AT_THREADS, smem, st>>>(
        reinterpret_cast<const T*>(v.latent), v.latent_ld, v.latent_bstride, reinterpret_cast<const T*>(v.rope),
        v.rope_ld, v.rope_bstride, reinterpret_cast<const T*>(v.q_latent), reinterpret_cast<const T*>(v.q_rope), v.H,
        v.N, lam, bitmap, nw, split_len, slot0, nslot, qrows, part_o, part_ml);
  }
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- s* and merge
__global__ void k_smax_reduce(int BH, int H, int nsplit, int nslot, const float* __restrict__ part_ml,
                              float* __restrict__ smax) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH) return;
  const int b = i / H, h = i % H;
  float m = -INFINITY;
  for (int s = 0; s < nsplit; ++s) m = fmaxf(m, part_ml[(((int64_t)b * nslot + s) * H + h) * 2]);
  smax[i] = m;
}

cudaError_t launch_smax_reduce(int B, int H, int nsplit, int nslot, const float* part_ml, float* smax,
                               cudaStream_t st) {
  k_smax_reduce<<<(B * H + 255) / 256, 256, 0, st>>>(B * H, H, nsplit, nslot, part_ml, smax);
  count_launches(1);
  return cudaGetLastError();
}

// One warp per (b, h): o = sum_s e^{m_s - m} o_s / sum_s e^{m_s - m} l_s, lse = m + log(sum), and s* = the
// max over the first nslot_tier1 slots.
__global__ void k_combine(int BH, int H, int nslot, int nslot_tier1, const float* __restrict__ part_o,
                          const float* __restrict__ part_ml, float* __restrict__ out, float* __restrict__ lse,
                          float* __restrict__ smax) {
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= BH) return;
  const int b = wid / H, h = wid % H;
  float m = -INFINITY, m1 = -INFINITY;
  for (int s = 0; s < nslot; ++s) {
    const float ms = part_ml[(((int64_t)b * nslot + s) * H + h) * 2];
    m = fmaxf(m, ms);
    if (s < nslot_tier1) m1 = fmaxf(m1, ms);
  }
  float acc[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) acc[t] = 0.f;
  float l = 0.f;
  if (m > -INFINITY) {
    for (int s = 0; s < nslot; ++s) {
      const int64_t base = ((int64_t)b * nslot + s) * H + h;
      const float ms = part_ml[base * 2], ls = part_ml[base * 2 + 1];
      if (!(ls > 0.f)) continue;
      const float w = __expf(ms - m);
      l = fmaf(w, ls, l);
      const float4* src = reinterpret_cast<const float4*>(part_o + base * D_LAT + lane * 16);
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const float4 x = src[t];
        acc[4 * t] = fmaf(w, x.x, acc[4 * t]);
        acc[4 * t + 1] = fmaf(w, x.y, acc[4 * t + 1]);
        acc[4 * t + 2] = fmaf(w, x.z, acc[4 * t + 2]);
        acc[4 * t + 3] = fmaf(w, x.w, acc[4 * t + 3]);
      }
    }
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
  float4* dst = reinterpret_cast<float4*>(out + (int64_t)wid * D_LAT + lane * 16);
#pragma unroll
  for (int t = 0; t < 4; ++t)
    dst[t] = make_float4(acc[4 * t] * inv, acc[4 * t + 1] * inv, acc[4 * t + 2] * inv, acc[4 * t + 3] * inv);
  if (lane == 0) {
    if (lse) lse[wid] = l > 0.f ? m + logf(l) : -INFINITY;
    if (smax) smax[wid] = m1;
  }
}

cudaError_t launch_combine(int B, int H, int nslot, int nslot_tier1, const float* part_o, const float* part_ml,
                           float* out, float* lse, float* smax, cudaStream_t st) {
  const int BH = B * H, threads = 256;
  k_combine<<<(BH * 32 + threads - 1) / threads, threads, 0, st>>>(BH, H, nslot, nslot_tier1, part_o, part_ml, out,
                                                                  lse, smax);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
