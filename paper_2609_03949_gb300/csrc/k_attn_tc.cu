// k_attn_tc.cu -- gather + absorbed-MLA attention with the logits on the tensor cores (bf16 caches).
//
// Per CTA: one sequence b, one range of positions, one group of <= 64 heads. Positions are walked in tiles of
// 32 (one bitmap word per head). For each tile:
//   warp 0 (producer)   stages the heads' 32-bit selection words and issues nine TMA loads (128-byte swizzle,
//                       K-major) of the tile's 32 rows x 576 columns into a 4-slot ring (tiles without any
//                       selected row are not loaded);
//   warp 1 (MMA)        S = Q . X^T on tcgen05: M = 64 heads, N = 32 rows, K = 576 (36 x K=16) into tensor
//                       memory; with M = 64 the logit of head 16g + t and row j sits in TMEM lane 32g + t,
//                       column j of the tile's slot;
//   warps 2..17         16 consumers, warp w owning heads 16 (w % 4) + 4 sub + i (sub = (w - 2) / 4, i < 4)
//                       so that their logits are in the warp's own TMEM lane quarter. For every selected
//                       (head, row) pair: read the logit (one tcgen05.ld), update the head's online softmax
//                       and accumulate p * latent row (bf16 x bf16 -> fp32 mixed FMAs) into the head's
//                       512-wide running sum, kept in registers (16 values per lane per head).
// The dense S tile costs ~35% of the tensor time the HBM stream leaves; the sparse part (softmax and the
// 512-wide axpy over ~4% of the (head, row) pairs) stays on the SIMT pipes. Partial (max, sum, out) per split
// are merged by the same LSE combine as the SIMT kernel (Lemma 1). All mbarrier waits are bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"

namespace vk {

constexpr int AT2_T = 32;                              // positions (rows) per tile
constexpr int AT2_NT = 4;                              // tile slots
constexpr int AT2_CONS = 16;                           // consumer warps
constexpr int AT2_THREADS = (2 + AT2_CONS) * 32;
constexpr uint32_t AT2_KBLK_Q = 64 * 128;              // one 64-column block of Q: 64 heads x 128 B
constexpr uint32_t AT2_KBLK_X = AT2_T * 128;           // one 64-column block of a tile: 32 rows x 128 B
constexpr uint32_t AT2_Q_BYTES = 9 * AT2_KBLK_Q;       // 73,728
constexpr uint32_t AT2_X_BYTES = 9 * AT2_KBLK_X;       // 36,864 per slot
constexpr uint32_t AT2_TMEM_COLS = 128;                // 4 x 32 logit columns
constexpr uint32_t AT2_S_COL0 = 0;

struct Attn2Smem {
  uint32_t q, x, words, uni, logit, bars, total;
  __host__ __device__ Attn2Smem() {
    q = 0;
    x = q + AT2_Q_BYTES;
    words = x + AT2_NT * AT2_X_BYTES;                  // [NT][64] selection words
    uni = words + AT2_NT * 64 * 4;                     // [NT] union words
    logit = uni;
    bars = (uni + AT2_NT * 4 + 7) & ~7u;               // x_full[NT], x_empty[NT], s_full[NT], q_full
    total = bars + (3 * AT2_NT + 1) * 8 + 1024;        // + slack to align the base to 1024
  }
};

__device__ __forceinline__ void tma_load_3d_(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ uint64_t sw128_desc_(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}
__device__ __forceinline__ void mma_bf16_(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit_(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ float tmem_ld1(uint32_t taddr) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];\n" : "=r"(r) : "r"(taddr) : "memory");
  return __uint_as_float(r);
}

__device__ __forceinline__ void tmem_ld32_(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

__device__ __forceinline__ uint16_t lo16_(uint32_t w) { return static_cast<uint16_t>(w & 0xffffu); }
__device__ __forceinline__ uint16_t hi16_(uint32_t w) { return static_cast<uint16_t>(w >> 16); }

struct Attn2Args {
  int H, N, nh_total;
  int split_len, slot0, nslot;
  int64_t nw;
  float lam_log2e;
  const uint32_t* bitmap;
  float* part_o;
  float* part_ml;
  int* status;
};

__global__ void __launch_bounds__(AT2_THREADS, 1) k_attn_tc(const __grid_constant__ CUtensorMap lmap,
                                                          const __grid_constant__ CUtensorMap rmap,
                                                          const __grid_constant__ CUtensorMap qlmap,
                                                          const __grid_constant__ CUtensorMap qrmap,
                                                          const Attn2Args args) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Attn2Smem L;
  unsigned char* sq = smem + L.q;
  unsigned char* sx = smem + L.x;
  uint32_t* words = reinterpret_cast<uint32_t*>(smem + L.words);
  uint32_t* unis = reinterpret_cast<uint32_t*>(smem + L.uni);
  uint64_t* x_full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* x_empty = x_full + AT2_NT;
  uint64_t* s_full = x_empty + AT2_NT;
  uint64_t* q_full = s_full + AT2_NT;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int split = blockIdx.x, hg = blockIdx.y, b = blockIdx.z;
  const int H = args.H;
  const int h0 = hg * 64, nh = min(64, H - h0);
  const int p0 = split * args.split_len, p1 = min(args.N, p0 + args.split_len);
  const int ntile = (p1 - p0 + AT2_T - 1) / AT2_T;         // p0 is a multiple of 32
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < AT2_NT; ++s) { mbar_init(&x_full[s], 1); mbar_init(&x_empty[s], AT2_CONS); mbar_init(&s_full[s], 1); }
    mbar_init(q_full, 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, AT2_TMEM_COLS);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    const uint32_t* bm = args.bitmap + ((int64_t)b * H + h0) * args.nw;
    if (lane == 0) {
      // the head group's queries: nine 64-column blocks of 64 rows (rows past nh read the next heads or zero fill;
      // their logits are never used)
      mbar_arrive_expect_tx(q_full, AT2_Q_BYTES);
      const int qrow = b * H + h0;
      for (int k = 0; k < 8; ++k) tma_load_3d_(sq + k * AT2_KBLK_Q, &qlmap, 64 * k, qrow, 0, q_full);
      tma_load_3d_(sq + 8 * AT2_KBLK_Q, &qrmap, 0, qrow, 0, q_full);
    }
    // the heads' selection words of tile t (lanes hold heads lane and lane + 32), fetched two tiles ahead
    auto fetch = [&](int t, uint32_t& wa, uint32_t& wb) {
      wa = wb = 0u;
      if (t >= ntile) return;
      const int pos0 = p0 + t * AT2_T;
      const int64_t w = pos0 >> 5;
      const int left = p1 - pos0;
      const uint32_t vmask = left >= 32 ? 0xffffffffu : ((1u << left) - 1u);
      if (lane < nh) wa = bm[(int64_t)lane * args.nw + w] & vmask;
      if (lane + 32 < nh) wb = bm[(int64_t)(lane + 32) * args.nw + w] & vmask;
    };
    uint32_t a0, b0, a1, b1, a2, b2;
    fetch(0, a0, b0);
    fetch(1, a1, b1);
    for (int t = 0; t < ntile; ++t) {
      fetch(t + 2, a2, b2);
      const int s = t % AT2_NT, use = t / AT2_NT;
      if (use > 0 && !mbar_wait(&x_empty[s], (use - 1) & 1, &abort_flag)) {
        if (lane == 0) { raise_status(args.status, VK_ERR_TIMEOUT); abort_flag = 1; }
        break;
      }
      if (abort_flag) break;
      const int pos0 = p0 + t * AT2_T;
      words[s * 64 + lane] = a0;
      words[s * 64 + lane + 32] = b0;
      const uint32_t uni = __reduce_or_sync(0xffffffffu, a0 | b0);
      if (lane == 0) unis[s] = uni;
      __syncwarp();
      if (lane == 0) {
        if (uni) {
          mbar_arrive_expect_tx(&x_full[s], AT2_X_BYTES);
          for (int k = 0; k < 8; ++k) tma_load_3d_(sx + s * AT2_X_BYTES + k * AT2_KBLK_X, &lmap, 64 * k, pos0, b, &x_full[s]);
          tma_load_3d_(sx + s * AT2_X_BYTES + 8 * AT2_KBLK_X, &rmap, 0, pos0, b, &x_full[s]);
        } else {
          mbar_arrive(&x_full[s]);                      // nothing selected: no load, no work
        }
      }
      a0 = a1; b0 = b1; a1 = a2; b1 = b2;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(AT2_T >> 3) << 17) | ((uint32_t)(64 >> 4) << 24);
      bool ok = mbar_wait(q_full, 0, &abort_flag);
      for (int t = 0; t < ntile && ok; ++t) {
        const int s = t % AT2_NT, use = t / AT2_NT;
        if (!mbar_wait(&x_full[s], use & 1, &abort_flag)) { ok = false; break; }
        if (unis[s]) {
          tmem_fence_after();
          const uint32_t xa = smem_addr(sx + s * AT2_X_BYTES), qa = smem_addr(sq);
          const uint32_t d = tmem_base + AT2_S_COL0 + s * AT2_T;
#pragma unroll 1
          for (int k = 0; k < 9; ++k)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16_(d, sw128_desc_(qa + k * AT2_KBLK_Q + 32 * kk), sw128_desc_(xa + k * AT2_KBLK_X + 32 * kk), idesc,
                        (k | kk) != 0);
          mma_commit_(&s_full[s]);
        } else {
          mbar_arrive(&s_full[s]);
        }
      }
      if (!ok) { raise_status(args.status, VK_ERR_TIMEOUT); abort_flag = 1; }
    }
  } else {
    // ------------------------------------------------------------------ consumers
    const int c = warp - 2;                              // 0..15
    const int q = warp & 3;                              // TMEM lane quarter this warp may access
    const int sub = c >> 2;                              // which 4 heads of the quarter's 16
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    float o[4][16];                                      // the 4 heads' running sums: dims 8 lane + t, 256 + 8 lane + t
    float m2[4], lsum[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      m2[i] = -INFINITY;
      lsum[i] = 0.f;
#pragma unroll
      for (int t = 0; t < 16; ++t) o[i][t] = 0.f;
    }
    const int hq0 = 16 * q + 4 * sub;                    // local heads hq0 .. hq0 + 3

    for (int t = 0; t < ntile; ++t) {
      const int s = t % AT2_NT, use = t / AT2_NT;
      if (!mbar_wait(&s_full[s], use & 1, &abort_flag) || !mbar_wait(&x_full[s], use & 1, &abort_flag)) {
        if (lane == 0) { raise_status(args.status, VK_ERR_TIMEOUT); abort_flag = 1; }
        break;
      }
      tmem_fence_after();
      const unsigned char* xs = sx + s * AT2_X_BYTES;
      const uint32_t scol = tmem_base + lane_base + AT2_S_COL0 + s * AT2_T;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int hl = hq0 + i;
        if (hl >= nh) break;
        uint32_t bits = words[s * 64 + hl];
        while (bits) {
          const int j = __ffs(bits) - 1;
          bits &= bits - 1;
          // logit of (head hl, row j): TMEM lane 32 q + (4 sub + i), column j of the slot
          const float sv = tmem_ld1(scol + j);
          // this lane's 16 latent values of row j: dims 8 lane .. + 7 and 256 + 8 lane .. + 7, un-swizzled
          const int ch = (lane & 7) ^ (j & 7);
          const uint4 xa = *reinterpret_cast<const uint4*>(xs + (lane >> 3) * AT2_KBLK_X + j * 128 + ch * 16);
          const uint4 xb = *reinterpret_cast<const uint4*>(xs + (4 + (lane >> 3)) * AT2_KBLK_X + j * 128 + ch * 16);
          tmem_wait_ld();
          const float s2 = __shfl_sync(0xffffffffu, sv, 4 * sub + i) * args.lam_log2e;
          if (s2 > m2[i]) {
            const float sc = ex2(m2[i] - s2);
            lsum[i] *= sc;
#pragma unroll
            for (int tt = 0; tt < 16; ++tt) o[i][tt] *= sc;
            m2[i] = s2;
          }
          const __nv_bfloat16 pb = __float2bfloat16_rn(ex2(s2 - m2[i]));
          const uint16_t p16 = __bfloat16_as_ushort(pb);
          lsum[i] += __bfloat162float(pb);
          const uint32_t wa[4] = {xa.x, xa.y, xa.z, xa.w}, wb[4] = {xb.x, xb.y, xb.z, xb.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            o[i][2 * k] = fma_bf16(p16, lo16_(wa[k]), o[i][2 * k]);
            o[i][2 * k + 1] = fma_bf16(p16, hi16_(wa[k]), o[i][2 * k + 1]);
            o[i][8 + 2 * k] = fma_bf16(p16, lo16_(wb[k]), o[i][8 + 2 * k]);
            o[i][8 + 2 * k + 1] = fma_bf16(p16, hi16_(wb[k]), o[i][8 + 2 * k + 1]);
          }
        }
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&x_empty[s]);
    }
    // partials: part_o [B][nslot][H][512] (unnormalised), part_ml [B][nslot][H][2] = (max logit, sum)
    const int slot = args.slot0 + split;
    constexpr float LN2 = 0.6931471805599453f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int hl = hq0 + i;
      if (hl >= nh) break;
      const int64_t base = (((int64_t)b * args.nslot + slot) * H + h0 + hl);
      float4* d0 = reinterpret_cast<float4*>(args.part_o + base * D_LAT + lane * 8);
      float4* d1 = reinterpret_cast<float4*>(args.part_o + base * D_LAT + 256 + lane * 8);
      d0[0] = make_float4(o[i][0], o[i][1], o[i][2], o[i][3]);
      d0[1] = make_float4(o[i][4], o[i][5], o[i][6], o[i][7]);
      d1[0] = make_float4(o[i][8], o[i][9], o[i][10], o[i][11]);
      d1[1] = make_float4(o[i][12], o[i][13], o[i][14], o[i][15]);
      if (lane == 0) { args.part_ml[base * 2] = m2[i] * LN2; args.part_ml[base * 2 + 1] = lsum[i]; }
    }
  }

  // wind down: nothing may still write this CTA's shared or tensor memory
  tmem_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0) {
    // drain tile loads that were issued but never consumed (only after an abort)
    for (int s = 0; s < AT2_NT && s < ntile; ++s) {
      const int last = (ntile - 1 - s) / AT2_NT;
      mbar_wait(&x_full[s], last & 1, nullptr);
    }
  }
  __syncthreads();
  tmem_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, AT2_TMEM_COLS);
}

// ---------------------------------------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 encode2() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult qr;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool attn_tc_supported(const vk_view& v) {
  return v.dtype == VK_BF16 && (v.latent_ld * 2) % 16 == 0 && (v.rope_ld * 2) % 16 == 0 &&
         (v.latent_bstride * 2) % 16 == 0 && (v.rope_bstride * 2) % 16 == 0 && encode2() != nullptr;
}

static bool make_map3(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint64_t batches, int64_t ld,
                      int64_t bstride, uint32_t box_rows) {
  cuuint64_t dims[3] = {cols, rows, batches};
  cuuint64_t str[2] = {(cuuint64_t)(ld * 2), (cuuint64_t)(bstride * 2)};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return encode2()(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, str, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t launch_attn_tc(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, int nsplit, int split_len,
                           int slot0, int nslot, float* part_o, float* part_ml, int* status, cudaStream_t st) {
  if (!encode2()) return cudaErrorNotSupported;
  CUtensorMap lmap, rmap, qlmap, qrmap;
  // cache rows: latent [B][N][512] and RoPE [B][N][64], 32-row boxes; queries: [B*H][512] and [B*H][64], 64-row boxes
  if (!make_map3(&lmap, v.latent, D_LAT, v.N, v.B, v.latent_ld, v.latent_bstride, AT2_T) ||
      !make_map3(&rmap, v.rope, D_ROPE, v.N, v.B, v.rope_ld, v.rope_bstride, AT2_T) ||
      !make_map3(&qlmap, v.q_latent, D_LAT, (uint64_t)v.B * v.H, 1, D_LAT, (int64_t)v.B * v.H * D_LAT, 64) ||
      !make_map3(&qrmap, v.q_rope, D_ROPE, (uint64_t)v.B * v.H, 1, D_ROPE, (int64_t)v.B * v.H * D_ROPE, 64))
    return cudaErrorInvalidValue;
  Attn2Args a{};
  a.H = v.H;
  a.N = v.N;
  a.split_len = split_len;
  a.slot0 = slot0;
  a.nslot = nslot;
  a.nw = nw;
  a.lam_log2e = lam * 1.4426950408889634f;
  a.bitmap = bitmap;
  a.part_o = part_o;
  a.part_ml = part_ml;
  a.status = status;
  const size_t smem = Attn2Smem().total;
  cudaError_t e = cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(nsplit, (v.H + 63) / 64, v.B);
  k_attn_tc<<<grid, AT2_THREADS, smem, st>>>(lmap, rmap, qlmap, qrmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
