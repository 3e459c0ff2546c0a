// k_attn_list.cu -- attention of each head over its fired rows: the recall tier's fetched rows (Sec. 4.2), marked in
// the head's fired bitmap, join that head's softmax as exact copies (Lemma 1). The bitmap, not the output list, is
// the source, so a list cut by its capacity does not change the outputs.
//
// The tier exists to fetch the few archived rows that could still beat the attended set's best, so the sets are
// small (empty when every query is well served). One CTA per (b, h) walks its own bitmap, each warp 32 words at a
// time (one coalesced load, a ballot of the non-empty ones), and takes each fired row with the whole warp: lane l
// holds latent dims [16 l, 16 l + 16) and RoPE dims 2 l, 2 l + 1 of the row and of the query, the logit
// lambda (Qc . L_u + Qr . K_u) is a warp sum, each warp keeps an online softmax, and the eight warps' (max, sum,
// output) are merged in shared memory into one partial (max logit, sum of e^(s - max), unnormalised output) in the
// fired slot that the LSE combine reads. Work and bytes scale with the fired rows, not with the cache.
#include "vk_common.cuh"

namespace vk {

namespace {

constexpr int AL_WARPS = 8;

__device__ __forceinline__ void load16(const __nv_bfloat16* p, float (&x)[16]) {
  const uint4 a = reinterpret_cast<const uint4*>(p)[0], b = reinterpret_cast<const uint4*>(p)[1];
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void load16(const float* p, float (&x)[16]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 f = reinterpret_cast<const float4*>(p)[i];
    x[4 * i] = f.x;
    x[4 * i + 1] = f.y;
    x[4 * i + 2] = f.z;
    x[4 * i + 3] = f.w;
  }
}
__device__ __forceinline__ float2 load2(const __nv_bfloat16* p) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
}
__device__ __forceinline__ float2 load2(const float* p) { return *reinterpret_cast<const float2*>(p); }

template <typename T>
__global__ void __launch_bounds__(AL_WARPS * 32) k_attn_list(int H, int N, const T* __restrict__ latent, int64_t lld,
                                                            int64_t lbs, const T* __restrict__ rope, int64_t rld,
                                                            int64_t rbs, const T* __restrict__ q_latent,
                                                            const T* __restrict__ q_rope, float lam,
                                                            const uint32_t* __restrict__ bitmap, int64_t nw,
                                                            int nslot, int slot, float* __restrict__ part_o,
                                                            float* __restrict__ part_ml, int* __restrict__ status,
                                                            const int* __restrict__ mode) {
  __shared__ float sm_m[AL_WARPS], sm_l[AL_WARPS];
  __shared__ float sm_o[AL_WARPS][D_LAT];
  if (mode && *mode == 0) return;                    // the tile pass takes the fired rows this step
  const int64_t bh = blockIdx.x;
  const int64_t b = bh / H, h = bh - b * H;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float qc[16];
  load16(q_latent + bh * D_LAT + 16 * lane, qc);
  const float2 qr = load2(q_rope + bh * D_ROPE + 2 * lane);
  float m = -INFINITY, l = 0.f, acc[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i] = 0.f;
  // this warp's fired rows in ascending order (warp-uniform state): chunks of 32 bitmap words, one per lane
  const uint32_t* bm = bitmap + bh * nw;
  int64_t w0 = (int64_t)w * 32 - AL_WARPS * 32;
  uint32_t word = 0u, live = 0u, bits = 0u;
  int src = 0;
  auto next = [&]() -> int64_t {
    while (true) {
      if (bits) {
        const int64_t u = (w0 + src) * 32 + (__ffs(bits) - 1);
        bits &= bits - 1;
        return u;
      }
      if (live) {
        src = __ffs(live) - 1;
        live &= live - 1;
        bits = __shfl_sync(0xffffffffu, word, src);
        continue;
      }
      w0 += AL_WARPS * 32;
      if (w0 >= nw) return -1;
      word = w0 + lane < nw ? bm[w0 + lane] : 0u;
      live = __ballot_sync(0xffffffffu, word != 0u);
    }
  };
  auto update = [&](float s, const float (&x)[16]) {
    if (s > m) {
      const float sc = __expf(m - s);                // 0 for the first row (m = -inf)
      l *= sc;
#pragma unroll
      for (int i = 0; i < 16; ++i) acc[i] *= sc;
      m = s;
    }
    const float p = __expf(s - m);
    l += p;
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = fmaf(p, x[i], acc[i]);
  };
  // rows two at a time, so that two rows' loads are in flight per warp
  for (int64_t u0 = next(); u0 >= 0;) {
    int64_t u1 = next();
    const bool ok0 = u0 < N, two = u1 >= 0, ok1 = two && u1 < N;
    if ((!ok0 || (two && !ok1)) && lane == 0) raise_status(status, VK_ERR_INVALID_ARG);   // never set by the library
    const int64_t r0 = ok0 ? u0 : 0, r1 = ok1 ? u1 : r0;
    float x0[16], x1[16];
    load16(latent + b * lbs + r0 * lld + 16 * lane, x0);
    load16(latent + b * lbs + r1 * lld + 16 * lane, x1);
    const float2 k0 = load2(rope + b * rbs + r0 * rld + 2 * lane);
    const float2 k1 = load2(rope + b * rbs + r1 * rld + 2 * lane);
    float d0 = fmaf(qr.x, k0.x, qr.y * k0.y), d1 = fmaf(qr.x, k1.x, qr.y * k1.y);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      d0 = fmaf(qc[i], x0[i], d0);
      d1 = fmaf(qc[i], x1[i], d1);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      d0 += __shfl_xor_sync(0xffffffffu, d0, o);
      d1 += __shfl_xor_sync(0xffffffffu, d1, o);
    }
    if (ok0) update(lam * d0, x0);
    if (ok1) update(lam * d1, x1);
    u0 = two ? next() : -1;
  }
  if (lane == 0) { sm_m[w] = m; sm_l[w] = l; }
#pragma unroll
  for (int i = 0; i < 16; ++i) sm_o[w][16 * lane + i] = acc[i];
  __syncthreads();
  float M = sm_m[0];
#pragma unroll
  for (int i = 1; i < AL_WARPS; ++i) M = fmaxf(M, sm_m[i]);
  float fw[AL_WARPS], L = 0.f;
#pragma unroll
  for (int i = 0; i < AL_WARPS; ++i) {
    fw[i] = sm_m[i] == -INFINITY ? 0.f : __expf(sm_m[i] - M);
    L = fmaf(fw[i], sm_l[i], L);
  }
  const int64_t base = ((int64_t)b * nslot + slot) * H + h;
  for (int d = threadIdx.x; d < D_LAT; d += blockDim.x) {
    float o = 0.f;
#pragma unroll
    for (int i = 0; i < AL_WARPS; ++i) o = fmaf(fw[i], sm_o[i][d], o);
    part_o[base * D_LAT + d] = o;
  }
  if (threadIdx.x == 0) {
    part_ml[base * 2] = M;
    part_ml[base * 2 + 1] = L;
  }
}

// mode[0] = 1 when every head fired at most `limit` rows (this kernel takes the pass), else 0 (the tile pass does).
__global__ void __launch_bounds__(1024) k_fired_mode(int64_t BH, const int32_t* __restrict__ count, int n0, int limit,
                                                     int* __restrict__ mode) {
  __shared__ int big;
  if (threadIdx.x == 0) big = 0;
  __syncthreads();
  int mine = 0;
  for (int64_t i = threadIdx.x; i < BH; i += blockDim.x) mine |= (count[i] - n0) > limit;
  if (mine) big = 1;
  __syncthreads();
  if (threadIdx.x == 0) mode[0] = big ? 0 : 1;
}

}  // namespace

cudaError_t launch_fired_mode(int64_t BH, const int32_t* count, int n0, int limit, int* mode, cudaStream_t st) {
  k_fired_mode<<<1, 1024, 0, st>>>(BH, count, n0, limit, mode);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_attn_list(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, int nslot, int slot,
                             float* part_o, float* part_ml, int* status, const int* mode, cudaStream_t st) {
  const unsigned grid = (unsigned)((int64_t)v.B * v.H);
  if (v.dtype == VK_BF16) {
    using T = __nv_bfloat16;
    k_attn_list<T><<<grid, AL_WARPS * 32, 0, st>>>(v.H, v.N, static_cast<const T*>(v.latent), v.latent_ld,
                                                   v.latent_bstride, static_cast<const T*>(v.rope), v.rope_ld,
                                                   v.rope_bstride, static_cast<const T*>(v.q_latent),
                                                   static_cast<const T*>(v.q_rope), lam, bitmap, nw, nslot, slot,
                                                   part_o, part_ml, status, mode);
  } else {
    k_attn_list<float><<<grid, AL_WARPS * 32, 0, st>>>(v.H, v.N, static_cast<const float*>(v.latent), v.latent_ld,
                                                       v.latent_bstride, static_cast<const float*>(v.rope), v.rope_ld,
                                                       v.rope_bstride, static_cast<const float*>(v.q_latent),
                                                       static_cast<const float*>(v.q_rope), lam, bitmap, nw, nslot,
                                                       slot, part_o, part_ml, status, mode);
  }
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
