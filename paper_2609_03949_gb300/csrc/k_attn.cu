// k_attn.cu -- gather + absorbed-MLA attention over per-head selected rows, split over positions, and the
// log-sum-exp merge of the splits (flash-decoding style).
//
// Attention (Eq. 1 with the absorbed query; Lemma 1: the output depends only on the attended multiset):
//   s[h,u] = lambda (Qc_h . L_u + Qr_h . K_u),  out_h = sum_u softmax_u(s) L_u,  lse_h,  s*_h = max_u s.
// Each CTA owns one sequence b, one range of positions and up to 64 heads. A producer warp bulk-copies each
// row selected by at least one of the CTA's heads (the union) from HBM once into a shared-memory ring; every
// head that selected the row consumes it from there. The work per (head, row) pair is a 576-wide dot product
// and a 512-wide axpy on the SIMT pipes (bf16 x bf16 -> fp32 mixed-precision FMAs): at ~4% density per head a
// dense tensor-core formulation would do ~25x the arithmetic for the same bytes.
// Splits of the fired rows (two-tier mode) write further partial slots; the combine merges all slots with
// their LSE weights, which is exact because the fired rows are disjoint from the tier-1 rows.
#include "vk_common.cuh"
#include "vk_ptx.cuh"

namespace vk {

constexpr int AT_CONS = 16;                          // consumer warps (each owns HG / AT_CONS heads)
constexpr int AT_THREADS = (AT_CONS + 1) * 32;       // + one producer warp
constexpr int AT_BLK = 16;                           // positions per pipeline stage
constexpr int AT_HPW = HG / AT_CONS;                 // heads per consumer warp (4)
constexpr int AT_MAX_STAGES = 8;

template <typename T> struct Elem;
template <> struct Elem<__nv_bfloat16> { static constexpr int bytes = 2; };
template <> struct Elem<float> { static constexpr int bytes = 4; };

__device__ __forceinline__ uint16_t lo16(uint32_t w) { return static_cast<uint16_t>(w & 0xffffu); }
__device__ __forceinline__ uint16_t hi16(uint32_t w) { return static_cast<uint16_t>(w >> 16); }

// The 18 coordinates a lane owns of a 576-wide row: latent [8 lane, 8 lane + 8) and [256 + 8 lane, 256 + 8 lane + 8),
// RoPE 2 lane and 2 lane + 1. With this mapping a warp's 16-byte loads cover contiguous 512-byte runs, so
// shared-memory reads are free of bank conflicts.
struct SliceBF16 {
  uint4 a, b;
  uint32_t c;
  __device__ __forceinline__ void load(const __nv_bfloat16* row, int lane) {
    a = *reinterpret_cast<const uint4*>(row + lane * 8);
    b = *reinterpret_cast<const uint4*>(row + 256 + lane * 8);
    c = *reinterpret_cast<const uint32_t*>(row + D_LAT + lane * 2);
  }
};
struct SliceF32 {
  float x[18];
  __device__ __forceinline__ void load(const float* row, int lane) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float4 v = *reinterpret_cast<const float4*>(row + lane * 8 + 4 * i);
      const float4 w = *reinterpret_cast<const float4*>(row + 256 + lane * 8 + 4 * i);
      x[4 * i] = v.x; x[4 * i + 1] = v.y; x[4 * i + 2] = v.z; x[4 * i + 3] = v.w;
      x[8 + 4 * i] = w.x; x[8 + 4 * i + 1] = w.y; x[8 + 4 * i + 2] = w.z; x[8 + 4 * i + 3] = w.w;
    }
    const float2 r = *reinterpret_cast<const float2*>(row + D_LAT + lane * 2);
    x[16] = r.x; x[17] = r.y;
  }
};

// Partial dot product of a lane's 18 coordinates (two accumulators for instruction-level parallelism).
__device__ __forceinline__ float slice_dot(const SliceBF16& q, const SliceBF16& x) {
  float d0 = 0.f, d1 = 0.f;
  const uint32_t qa[4] = {q.a.x, q.a.y, q.a.z, q.a.w}, qb[4] = {q.b.x, q.b.y, q.b.z, q.b.w};
  const uint32_t xa[4] = {x.a.x, x.a.y, x.a.z, x.a.w}, xb[4] = {x.b.x, x.b.y, x.b.z, x.b.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    d0 = fma_bf16(lo16(qa[i]), lo16(xa[i]), d0);
    d1 = fma_bf16(hi16(qa[i]), hi16(xa[i]), d1);
    d0 = fma_bf16(lo16(qb[i]), lo16(xb[i]), d0);
    d1 = fma_bf16(hi16(qb[i]), hi16(xb[i]), d1);
  }
  d0 = fma_bf16(lo16(q.c), lo16(x.c), d0);
  d1 = fma_bf16(hi16(q.c), hi16(x.c), d1);
  return d0 + d1;
}
__device__ __forceinline__ float slice_dot(const SliceF32& q, const SliceF32& x) {
  float d0 = 0.f, d1 = 0.f;
#pragma unroll
  for (int i = 0; i < 18; i += 2) { d0 = fmaf(q.x[i], x.x[i], d0); d1 = fmaf(q.x[i + 1], x.x[i + 1], d1); }
  return d0 + d1;
}

// o[0:16] = o * scale_unused + p * latent slice (p rounded to bf16 for the mixed FMA; the same rounded p
// enters the softmax denominator, so the normalisation matches the weights used).
__device__ __forceinline__ float slice_axpy(float p, const SliceBF16& x, float* o) {
  const __nv_bfloat16 pb = __float2bfloat16_rn(p);
  const uint16_t p16 = __bfloat16_as_ushort(pb);
  const uint32_t xa[4] = {x.a.x, x.a.y, x.a.z, x.a.w}, xb[4] = {x.b.x, x.b.y, x.b.z, x.b.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[2 * i] = fma_bf16(p16, lo16(xa[i]), o[2 * i]);
    o[2 * i + 1] = fma_bf16(p16, hi16(xa[i]), o[2 * i + 1]);
    o[8 + 2 * i] = fma_bf16(p16, lo16(xb[i]), o[8 + 2 * i]);
    o[8 + 2 * i + 1] = fma_bf16(p16, hi16(xb[i]), o[8 + 2 * i + 1]);
  }
  return __bfloat162float(pb);
}
__device__ __forceinline__ float slice_axpy(float p, const SliceF32& x, float* o) {
#pragma unroll
  for (int i = 0; i < 16; ++i) o[i] = fmaf(p, x.x[i], o[i]);
  return p;
}

template <typename T> struct SliceOf;
template <> struct SliceOf<__nv_bfloat16> { using type = SliceBF16; };
template <> struct SliceOf<float> { using type = SliceF32; };

// Shared-memory layout of one attention CTA (bytes), shared by the kernel and the launcher.
struct AttnSmem {
  uint32_t q, rows, heads, uni, bars, total;
  __host__ __device__ AttnSmem(int esz, int qrows, int nst) {
    const uint32_t rowb = (D_LAT + D_ROPE) * esz;
    q = 0;
    rows = q + qrows * rowb;
    heads = rows + nst * AT_BLK * rowb;
    uni = heads + nst * HG * 2;
    bars = (uni + nst * 4 + 7) & ~7u;
    total = bars + 2 * nst * 8;
  }
};

// One CTA = (split of positions, head group of <= 64 heads, sequence). Warp AT_CONS produces: for each
// 16-position block it reads the heads' bitmap bits, stages them and their union in shared memory, and bulk-
// copies every union row (1152 B in bf16) into the block's ring slot, completing on the slot's `full`
// mbarrier. Consumer warp w owns heads w, w + 16, w + 32, w + 48 and, for every set bit of those heads,
// computes the logit, updates its online softmax and accumulates the latent row; it then arrives on the slot's
// `empty` mbarrier. No block-wide barrier is taken after the prologue, so warps with more selected pairs in a
// block do not hold the others back (the ring absorbs the imbalance).
template <typename T>
__global__ void __launch_bounds__(AT_THREADS, 1) k_attn(
    const T* __restrict__ latent, int64_t lld, int64_t lbs, const T* __restrict__ rope, int64_t rld, int64_t rbs,
    const T* __restrict__ q_latent, const T* __restrict__ q_rope, int H, int N, float lam_log2e,
    const uint32_t* __restrict__ bitmap, int64_t nw, int split_len, int slot0, int nslot, int qrows, int nst,
    float* __restrict__ part_o, float* __restrict__ part_ml, int* status, const int* __restrict__ skip) {
  if (skip && *skip) return;                         // another kernel took this pass (the whole block leaves)
  using Slice = typename SliceOf<T>::type;
  constexpr int ROWE = D_LAT + D_ROPE;
  constexpr int ESZ = Elem<T>::bytes;
  extern __shared__ __align__(128) unsigned char smem[];
  const AttnSmem L(ESZ, qrows, nst);
  T* qs = reinterpret_cast<T*>(smem + L.q);
  T* rows = reinterpret_cast<T*>(smem + L.rows);
  uint16_t* hdr_heads = reinterpret_cast<uint16_t*>(smem + L.heads);
  uint32_t* hdr_union = reinterpret_cast<uint32_t*>(smem + L.uni);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty = full + nst;
  __shared__ int abort_flag;
  __shared__ uint32_t tmem_base;

  const int split = blockIdx.x, hg = blockIdx.y, b = blockIdx.z;
  const int h0 = hg * HG, nh = min(HG, H - h0);
  const int p0 = split * split_len, p1 = min(N, p0 + split_len);
  const int nb = (p1 - p0 + AT_BLK - 1) / AT_BLK;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool contiguous = (rope == latent + D_LAT) && lld == ROWE && rld == ROWE && rbs == lbs;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < nst; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], AT_CONS); }
    mbar_fence_init();
  }
  // queries of this head group -> shared memory (16-byte pieces)
  constexpr int QPIECES = ROWE * ESZ / 16;
  for (int i = threadIdx.x; i < nh * QPIECES; i += blockDim.x) {
    const int h = i / QPIECES, e0 = (i % QPIECES) * (16 / ESZ);
    const T* src = (e0 < D_LAT) ? q_latent + ((int64_t)b * H + h0 + h) * D_LAT + e0
                                : q_rope + ((int64_t)b * H + h0 + h) * D_ROPE + (e0 - D_LAT);
    *reinterpret_cast<uint4*>(qs + h * ROWE + e0) = *reinterpret_cast<const uint4*>(src);
  }
  if (warp == 0) tmem_alloc(&tmem_base, 256);       // 16 heads x 16 columns per TMEM lane quarter
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();

  if (warp == AT_CONS) {
    // ------------------------------------------------------------------ producer
    const uint32_t* bm = bitmap + ((int64_t)b * H + h0) * nw;
    const int64_t w_base = p0 >> 5;                   // p0 is a multiple of 32
    uint32_t cur0[8], cur1[8];                        // 8 bitmap words (256 positions) of heads lane, lane + 32
    auto load_chunk = [&](int c, uint32_t* d0, uint32_t* d1) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int64_t w = w_base + 8 * c + j;
        d0[j] = (lane < nh && w < nw) ? bm[(int64_t)lane * nw + w] : 0u;
        d1[j] = (lane + 32 < nh && w < nw) ? bm[(int64_t)(lane + 32) * nw + w] : 0u;
      }
    };
    const int nchunks = (nb + 15) / 16;
    load_chunk(0, cur0, cur1);
    bool ok = true;
    for (int c = 0; c < nchunks && ok; ++c) {
      uint32_t nxt0[8], nxt1[8];
      if (c + 1 < nchunks) load_chunk(c + 1, nxt0, nxt1);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int blk = 16 * c + j;
        if (blk >= nb || !ok) break;
        const int s = blk % nst;
        const int use = blk / nst;
        if (use > 0 && !mbar_wait(&empty[s], (use - 1) & 1, &abort_flag)) {
          raise_status(status, VK_ERR_TIMEOUT);
          abort_flag = 1;
          ok = false;
          break;
        }
        if (abort_flag) { ok = false; break; }
        const int pos0 = p0 + blk * AT_BLK;
        const int left = p1 - pos0;
        const uint32_t vmask = left >= AT_BLK ? 0xffffu : ((1u << left) - 1u);
        const uint32_t ha = (cur0[j >> 1] >> (16 * (j & 1))) & vmask;
        const uint32_t hb = (cur1[j >> 1] >> (16 * (j & 1))) & vmask;
        hdr_heads[s * HG + lane] = static_cast<uint16_t>(ha);
        hdr_heads[s * HG + lane + 32] = static_cast<uint16_t>(hb);
        const uint32_t uni = __reduce_or_sync(0xffffffffu, ha | hb);
        if (lane == 0) hdr_union[s] = uni;
        __syncwarp();
        // every union row goes to the stage slot of its position in the block; with the interleaved row layout
        // (RoPE right after the latent, 576-wide rows) a run of consecutive union rows is one contiguous range
        // and one bulk copy, otherwise each row takes two (latent, RoPE)
        if (contiguous) {
          if (lane == 0) {
            uint32_t bytes = 0;
            for (uint32_t m = uni; m; ) {
              const int j0 = __ffs(m) - 1;
              const int len = __ffs(~(m >> j0)) - 1;       // length of the run of set bits starting at j0
              bytes += (uint32_t)len * (uint32_t)(ROWE * ESZ);
              m &= ~(((len >= 32) ? 0xffffffffu : ((1u << len) - 1u)) << j0);
            }
            mbar_arrive_expect_tx(&full[s], bytes);
          }
          __syncwarp();
          if (lane < AT_BLK && ((uni >> lane) & 1u) && (lane == 0 || !((uni >> (lane - 1)) & 1u))) {
            const int len = __ffs(~(uni >> lane)) - 1;
            const int64_t u = pos0 + lane;
            bulk_g2s(rows + ((int64_t)s * AT_BLK + lane) * ROWE, latent + (int64_t)b * lbs + u * lld,
                     (uint32_t)len * (uint32_t)(ROWE * ESZ), &full[s]);
          }
        } else {
          if (lane == 0) mbar_arrive_expect_tx(&full[s], __popc(uni) * (uint32_t)(ROWE * ESZ));
          __syncwarp();
          if (lane < AT_BLK && ((uni >> lane) & 1u)) {
            const int64_t u = pos0 + lane;
            T* dst = rows + ((int64_t)s * AT_BLK + lane) * ROWE;
            bulk_g2s(dst, latent + (int64_t)b * lbs + u * lld, D_LAT * ESZ, &full[s]);
            bulk_g2s(dst + D_LAT, rope + (int64_t)b * rbs + u * rld, D_ROPE * ESZ, &full[s]);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) { cur0[j] = nxt0[j]; cur1[j] = nxt1[j]; }
    }
    // never leave while bulk copies may still write into this CTA's shared memory
    if (lane == 0) {
      for (int s = 0; s < nst && s < nb; ++s) {
        const int last_use = (nb - 1 - s) / nst;      // the last block that used slot s
        mbar_wait(&full[s], last_use & 1, nullptr);
      }
    }
    return;
  }

  // -------------------------------------------------------------------- consumers
  // Each consumer warp keeps its heads' query slices in registers and their 512-wide running sums in tensor
  // memory: lane t of warp w holds head (w + 16 i)'s 16 accumulators in TMEM lane 32 (w % 4) + t, columns
  // 16 (4 (w / 4) + i) .. + 15.
  Slice q[AT_HPW];
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) {
    const int hl = warp + AT_CONS * i;
    if (hl < nh) q[i].load(qs + hl * ROWE, lane);
  }
  const uint32_t tacc = tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)((warp >> 2) * AT_HPW * 16);
  float o[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) o[t] = 0.f;
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) tmem_st16(tacc + 16 * i, o);
  float m2[AT_HPW], l[AT_HPW];
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) { m2[i] = -INFINITY; l[i] = 0.f; }

  for (int blk = 0; blk < nb; ++blk) {
    const int s = blk % nst;
    if (!mbar_wait(&full[s], (blk / nst) & 1, &abort_flag)) {
      if (lane == 0) { raise_status(status, VK_ERR_TIMEOUT); abort_flag = 1; }
      break;
    }
    const T* stage = rows + (int64_t)s * AT_BLK * ROWE;
#pragma unroll
    for (int i = 0; i < AT_HPW; ++i) {
      const int hl = warp + AT_CONS * i;
      if (hl >= nh) break;
      uint32_t bits = hdr_heads[s * HG + hl];
      while (bits) {
        const int j = __ffs(bits) - 1;
        bits &= bits - 1;
        Slice x;
        x.load(stage + j * ROWE, lane);                   // rows sit at their position's slot
        tmem_wait_st();
        tmem_ld16(tacc + 16 * i, o);                    // overlaps with the dot product below
        float d = slice_dot(q[i], x);
#pragma unroll
        for (int off = 16; off; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off);
        const float s2 = d * lam_log2e;                 // logit in log2 units
        tmem_wait_ld();
        if (s2 > m2[i]) {
          const float sc = ex2(m2[i] - s2);
          l[i] *= sc;
#pragma unroll
          for (int t = 0; t < 16; ++t) o[t] *= sc;
          m2[i] = s2;
        }
        l[i] += slice_axpy(ex2(s2 - m2[i]), x, o);
        tmem_st16(tacc + 16 * i, o);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
  }
  tmem_wait_st();

  // partials: part_o [B][nslot][H][512] (unnormalised), part_ml [B][nslot][H][2] = (max logit, sum)
  const int slot = slot0 + split;
  constexpr float LN2 = 0.6931471805599453f;
#pragma unroll
  for (int i = 0; i < AT_HPW; ++i) {
    const int hl = warp + AT_CONS * i;
    if (hl >= nh) break;
    tmem_ld16(tacc + 16 * i, o);
    tmem_wait_ld();
    const int64_t base = (((int64_t)b * nslot + slot) * H + h0 + hl);
    float4* d0 = reinterpret_cast<float4*>(part_o + base * D_LAT + lane * 8);
    float4* d1 = reinterpret_cast<float4*>(part_o + base * D_LAT + 256 + lane * 8);
    d0[0] = make_float4(o[0], o[1], o[2], o[3]);
    d0[1] = make_float4(o[4], o[5], o[6], o[7]);
    d1[0] = make_float4(o[8], o[9], o[10], o[11]);
    d1[1] = make_float4(o[12], o[13], o[14], o[15]);
    if (lane == 0) { part_ml[base * 2] = m2[i] * LN2; part_ml[base * 2 + 1] = l[i]; }
  }
  // every consumer is done with tensor memory: release it
  tmem_fence_before();
  named_barrier(1, AT_CONS * 32);
  if (warp == 0) {
    tmem_fence_after();
    tmem_dealloc(tmem_base, 256);
  }
}

int attn_stages(int dtype, int H) {
  const int esz = dtype == VK_BF16 ? 2 : 4;
  const int qrows = min(H, HG);
  for (int nst = AT_MAX_STAGES; nst >= 2; --nst)
    if (AttnSmem(esz, qrows, nst).total <= (uint32_t)SMEM_BUDGET) return nst;
  return 2;
}

size_t attn_smem_bytes(int dtype, int H, int split_len) {
  (void)split_len;
  return AttnSmem(dtype == VK_BF16 ? 2 : 4, min(H, HG), attn_stages(dtype, H)).total;
}

cudaError_t launch_attn(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, const AttnGeom& g, int slot0,
                        int nslot, float* part_o, float* part_ml, uint32_t flags, int* status, cudaStream_t st,
                        const int* skip) {
  // bf16 caches: both contractions on the tensor cores, persistent layout (k_attn_tc.cu); fp32 caches: the SIMT
  // kernel below, split layout
  if (g.G > 0) return launch_attn_tc(v, lam, bitmap, nw, g, slot0, nslot, part_o, part_ml, flags, status, st, nullptr, skip);
  const int nsplit = g.nsplit, split_len = g.split_len;
  dim3 grid(nsplit, (v.H + HG - 1) / HG, v.B);
  const int nst = attn_stages(v.dtype, v.H);
  const size_t smem = attn_smem_bytes(v.dtype, v.H, split_len);
  const int qrows = min(v.H, HG);
  const float lam_log2e = lam * 1.4426950408889634f;
  if (v.dtype == VK_BF16) {
    using T = __nv_bfloat16;
    cudaError_t e = cudaFuncSetAttribute(k_attn<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_attn<T><<<grid, AT_THREADS, smem, st>>>(
        reinterpret_cast<const T*>(v.latent), v.latent_ld, v.latent_bstride, reinterpret_cast<const T*>(v.rope),
        v.rope_ld, v.rope_bstride, reinterpret_cast<const T*>(v.q_latent), reinterpret_cast<const T*>(v.q_rope), v.H,
        v.N, lam_log2e, bitmap, nw, split_len, slot0, nslot, qrows, nst, part_o, part_ml, status, skip);
  } else {
    using T = float;
    cudaError_t e = cudaFuncSetAttribute(k_attn<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_attn<T><<<grid, AT_THREADS, smem, st>>>(
        reinterpret_cast<const T*>(v.latent), v.latent_ld, v.latent_bstride, reinterpret_cast<const T*>(v.rope),
        v.rope_ld, v.rope_bstride, reinterpret_cast<const T*>(v.q_latent), reinterpret_cast<const T*>(v.q_rope), v.H,
        v.N, lam_log2e, bitmap, nw, split_len, slot0, nslot, qrows, nst, part_o, part_ml, status, skip);
  }
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- s* and merge
// s*_h of the tier-1 set: the max over the written tier-1 slots of (b, h).
__global__ void k_smax_reduce(int BH, int H, const AttnGeom g, int nslot, const float* __restrict__ part_ml,
                              float* __restrict__ smax) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH) return;
  const int b = i / H, h = i % H;
  const int nv = attn_nvalid(g, (long long)b * g.n_hg + h / HG);
  float m = -INFINITY;
  for (int s = 0; s < nv; ++s) m = fmaxf(m, part_ml[(((int64_t)b * nslot + s) * H + h) * 2]);
  smax[i] = m;
}

cudaError_t launch_smax_reduce(int B, int H, const AttnGeom& g, int nslot, const float* part_ml, float* smax,
                               cudaStream_t st) {
  k_smax_reduce<<<(B * H + 255) / 256, 256, 0, st>>>(B * H, H, g, nslot, part_ml, smax);
  count_launches(1);
  return cudaGetLastError();
}

// One warp per (b, h): o = sum_s e^{m_s - m} o_s / sum_s e^{m_s - m} l_s over the written slots of both tiers,
// lse = m + log(sum), and s* = the max over the tier-1 slots. Slot s of the list is tier-1 slot s for s < nv, else
// fired slot g.nslot + s - nv (only when nslot covers two tiers): nf of them (the per-head fired pass writes one), or
// nv when nf < 0; with `mode` given, *mode != 0 says the per-head pass ran (nf = 1), else the tile pass (nf = nv).
__global__ void k_combine(int BH, int H, const AttnGeom g, int nslot, int nf, const int* __restrict__ mode,
                          const float* __restrict__ part_o,
                          const float* __restrict__ part_ml, float* __restrict__ out, float* __restrict__ lse,
                          float* __restrict__ smax) {
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= BH) return;
  const int b = wid / H, h = wid % H;
  const int nv = attn_nvalid(g, (long long)b * g.n_hg + h / HG);
  const int nfe = mode ? (*mode ? 1 : -1) : nf;
  const int nlist = nslot > g.nslot ? nv + (nfe < 0 ? nv : nfe) : nv;
  auto slot_of = [&](int s) { return s < nv ? s : g.nslot + s - nv; };
  float m = -INFINITY, m1 = -INFINITY;
  for (int s = 0; s < nlist; ++s) {
    const float ms = part_ml[(((int64_t)b * nslot + slot_of(s)) * H + h) * 2];
    m = fmaxf(m, ms);
    if (s < nv) m1 = fmaxf(m1, ms);
  }
  float acc[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) acc[t] = 0.f;
  float l = 0.f;
  if (m > -INFINITY) {
    for (int s = 0; s < nlist; ++s) {
      const int64_t base = ((int64_t)b * nslot + slot_of(s)) * H + h;
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

// The same merge for many slots per (b, h) (small batches: one sequence's tiles spread over up to 152 CTAs): one
// block of CMB_WARPS warps per (b, h). The block finds the max over the slots, each warp sums every CMB_WARPS-th
// slot (lanes over the 512 dims), and the warps' sums are added through shared memory -- the slots' loads run
// CMB_WARPS wide instead of one slot after another.
constexpr int CMB_WARPS = 8;
__global__ void __launch_bounds__(CMB_WARPS * 32) k_combine_wide(int H, const AttnGeom g, int nslot, int nf,
                                                                 const int* __restrict__ mode,
                                                                 const float* __restrict__ part_o,
                                                                 const float* __restrict__ part_ml,
                                                                 float* __restrict__ out, float* __restrict__ lse,
                                                                 float* __restrict__ smax) {
  __shared__ float red_m[CMB_WARPS], red_m1[CMB_WARPS], red_l[CMB_WARPS];
  __shared__ float4 red_acc[CMB_WARPS][32][4];
  const int bh = blockIdx.x, b = bh / H, h = bh % H;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nv = attn_nvalid(g, (long long)b * g.n_hg + h / HG);
  const int nfe = mode ? (*mode ? 1 : -1) : nf;
  const int nlist = nslot > g.nslot ? nv + (nfe < 0 ? nv : nfe) : nv;
  auto slot_of = [&](int s) { return s < nv ? s : g.nslot + s - nv; };
  float m = -INFINITY, m1 = -INFINITY;
  for (int s = threadIdx.x; s < nlist; s += blockDim.x) {
    const float ms = part_ml[(((int64_t)b * nslot + slot_of(s)) * H + h) * 2];
    m = fmaxf(m, ms);
    if (s < nv) m1 = fmaxf(m1, ms);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
  }
  if (lane == 0) { red_m[w] = m; red_m1[w] = m1; }
  __syncthreads();
  m = red_m[0];
  m1 = red_m1[0];
#pragma unroll
  for (int i = 1; i < CMB_WARPS; ++i) { m = fmaxf(m, red_m[i]); m1 = fmaxf(m1, red_m1[i]); }
  float acc[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) acc[t] = 0.f;
  float l = 0.f;
  if (m > -INFINITY) {
    for (int s = w; s < nlist; s += CMB_WARPS) {
      const int64_t base = ((int64_t)b * nslot + slot_of(s)) * H + h;
      const float ms = part_ml[base * 2], ls = part_ml[base * 2 + 1];
      if (!(ls > 0.f)) continue;
      const float wt = __expf(ms - m);
      l = fmaf(wt, ls, l);
      const float4* src = reinterpret_cast<const float4*>(part_o + base * D_LAT + lane * 16);
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const float4 x = src[t];
        acc[4 * t] = fmaf(wt, x.x, acc[4 * t]);
        acc[4 * t + 1] = fmaf(wt, x.y, acc[4 * t + 1]);
        acc[4 * t + 2] = fmaf(wt, x.z, acc[4 * t + 2]);
        acc[4 * t + 3] = fmaf(wt, x.w, acc[4 * t + 3]);
      }
    }
  }
#pragma unroll
  for (int t = 0; t < 4; ++t) red_acc[w][lane][t] = make_float4(acc[4 * t], acc[4 * t + 1], acc[4 * t + 2], acc[4 * t + 3]);
  if (lane == 0) red_l[w] = l;
  __syncthreads();
  if (w != 0) return;
  float lt = 0.f;
#pragma unroll
  for (int i = 0; i < CMB_WARPS; ++i) lt += red_l[i];
  const float inv = lt > 0.f ? 1.f / lt : 0.f;
  float4* dst = reinterpret_cast<float4*>(out + (int64_t)bh * D_LAT + lane * 16);
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    float4 a = red_acc[0][lane][t];
#pragma unroll
    for (int i = 1; i < CMB_WARPS; ++i) {
      const float4 x = red_acc[i][lane][t];
      a.x += x.x; a.y += x.y; a.z += x.z; a.w += x.w;
    }
    dst[t] = make_float4(a.x * inv, a.y * inv, a.z * inv, a.w * inv);
  }
  if (lane == 0) {
    if (lse) lse[bh] = lt > 0.f ? m + logf(lt) : -INFINITY;
    if (smax) smax[bh] = m1;
  }
}

cudaError_t launch_combine(int B, int H, const AttnGeom& g, int nslot, const float* part_o, const float* part_ml,
                           float* out, float* lse, float* smax, cudaStream_t st, int nf, const int* mode) {
  const int BH = B * H, threads = 256;
  if (nslot > CMB_WARPS)
    k_combine_wide<<<BH, CMB_WARPS * 32, 0, st>>>(H, g, nslot, nf, mode, part_o, part_ml, out, lse, smax);
  else
    k_combine<<<(BH * 32 + threads - 1) / threads, threads, 0, st>>>(BH, H, g, nslot, nf, mode, part_o, part_ml, out, lse,
                                                                     smax);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
