// k_score_tc.cu -- RoPE-branch scoring on the 5th-generation tensor cores (tcgen05), bf16, r = 64.
//
// a[h,u] = Qr_h . K_u for every cached row (Eq. 4's exact summand): per sequence the [N x 64] RoPE slice times
// the [64 x H] query, a dense contraction at H flop per byte. One CTA per SM walks a contiguous range of
// 128-row tiles:
//   warp 0 (one thread)  TMA: the tile's 128 x 64 bf16 slice (128 B of every 1152-B row, 128-byte swizzle)
//                        into an 8-stage ring, and the sequence's H x 64 query when the sequence changes;
//   warp 1 (one thread)  tcgen05.mma M=128, N=H, K=16 (x4) into one of G fp32 accumulators in tensor memory
//                        (128 lanes = rows, H columns = heads); tcgen05.commit frees the ring slot and hands the
//                        accumulator to the epilogue group that owns it;
//   G groups of 4 warps  epilogue, group g taking tiles i = g (mod G), so G tiles are in flight at once (the
//                        candidate epilogue waits on global atomics): tcgen05.ld of 32 heads at a time, one
//                        thread per row, then
//                        mode 0  write fp32 scores [B][H][ld] (also used on a strided row sample),
//                        mode 1  emit (u, a) for archive rows with a >= theta[b,h] into per-head candidate lists,
//                        mode 2  trigger: T = lambda (a + |(O Qr)[r:]| page_res + z |Qc| eta) > s*_h for archive
//                                rows outside S_h -> 32-row words of the fired bitmap (or candidates for top_j).
// Every mbarrier wait is bounded; a wait that gives up raises VK_ERR_TIMEOUT and the CTA winds down.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"
#include "vk_score_tc.h"

namespace vk {

constexpr int TC_M = 128;                    // rows per tile (MMA M)
constexpr int TC_STAGES = 8;
constexpr uint32_t TC_TILE_BYTES = TC_M * 128;   // 128 rows x 64 bf16
constexpr int TC_MAX_G = 4;                  // epilogue groups (accumulator buffers)

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::
          "r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte swizzle layout: rows of 128 B (64 bf16),
// 8-row atoms of 1024 B stacked at stride 1024 B. Fields: start address >> 4 (bits 0-13), leading-byte offset
// >> 4 (16-29, unused for this layout: 1), stride-byte offset >> 4 (32-45), descriptor version 1 (46-47),
// swizzle mode 2 = 128B (61-63).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulate (bits 4-5 = 1), A and B bf16 (7-9, 10-12 = 1),
// both K-major, N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t mma_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_addr(bar))
               : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
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

struct TcSmem {
  uint32_t a, q, bars, params, total;
  __host__ __device__ TcSmem(int H) {
    a = 0;                                              // TC_STAGES x 16 KB (1024-aligned)
    q = a + TC_STAGES * TC_TILE_BYTES;                  // 2 x H x 128 B
    bars = q + 2 * H * 128;                             // 8-byte barriers
    params = bars + (2 * TC_STAGES + 4 + 2 * TC_MAX_G) * 8;   // per group: 4 x H floats of per-sequence params
    total = params + TC_MAX_G * 4 * H * 4 + 1024;       // + slack to align the base to 1024
  }
};

template <int G, int MODE>
__global__ void __launch_bounds__((2 + 4 * G) * 32, 1) k_score_tc(const __grid_constant__ CUtensorMap kmap,
                                                                const __grid_constant__ CUtensorMap qmap,
                                                                const ScoreTcArgs args) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int H = args.H;
  const TcSmem Ls(H);
  unsigned char* sa = smem + Ls.a;
  unsigned char* sq = smem + Ls.q;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Ls.bars);
  uint64_t* a_full = bars;
  uint64_t* a_empty = bars + TC_STAGES;
  uint64_t* q_full = bars + 2 * TC_STAGES;              // [2]
  uint64_t* q_empty = q_full + 2;                        // [2]
  uint64_t* d_full = q_empty + 2;                        // [G]
  uint64_t* d_empty = d_full + G;                        // [G]
  float* sparams = reinterpret_cast<float*>(smem + Ls.params);   // [G groups][4][H]
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t total = args.total_tiles;
  const int64_t t0 = total * blockIdx.x / gridDim.x, t1 = total * (blockIdx.x + 1) / gridDim.x;
  const int n = (int)(t1 - t0);
  const int tps = args.tiles_per_seq;
  const int b_first = (int)(t0 / tps);
  const uint32_t dcols = (uint32_t)H;                   // columns per accumulator buffer
  const uint32_t idesc = mma_idesc_bf16(TC_M, H);

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < TC_STAGES; ++s) { mbar_init(&a_full[s], 1); mbar_init(&a_empty[s], 1); }
    for (int i = 0; i < 2; ++i) { mbar_init(&q_full[i], 1); mbar_init(&q_empty[i], 1); }
    for (int i = 0; i < G; ++i) { mbar_init(&d_full[i], 1); mbar_init(&d_empty[i], 4); }
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, args.tmem_cols);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0 && n > 0) {
      int prev_b = -1;
      for (int i = 0; i < n; ++i) {
        const int64_t t = t0 + i;
        const int b = (int)(t / tps), row0 = (int)(t % tps) * TC_M;
        if (b != prev_b) {
          const int qi = (b - b_first) & 1, quse = (b - b_first) >> 1;
          if (quse > 0 && !mbar_wait(&q_empty[qi], (quse - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
          mbar_arrive_expect_tx(&q_full[qi], (uint32_t)H * 128u);
          tma_load_2d(sq + qi * H * 128, &qmap, 0, b * H, &q_full[qi]);
          prev_b = b;
        }
        const int s = i % TC_STAGES, use = i / TC_STAGES;
        if (use > 0 && !mbar_wait(&a_empty[s], (use - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
        if (abort_flag) break;
        mbar_arrive_expect_tx(&a_full[s], TC_TILE_BYTES);
        tma_load_3d(sa + s * TC_TILE_BYTES, &kmap, 0, row0, b, &a_full[s]);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0 && n > 0) {
      int prev_b = -1;
      for (int i = 0; i < n; ++i) {
        const int64_t t = t0 + i;
        const int b = (int)(t / tps);
        const int qi = (b - b_first) & 1;
        if (b != prev_b) {
          if (!mbar_wait(&q_full[qi], ((b - b_first) >> 1) & 1, &abort_flag)) { abort_flag = 1; break; }
          prev_b = b;
        }
        const int s = i % TC_STAGES, use = i / TC_STAGES;
        const int ds = i % G, duse = i / G;
        if (!mbar_wait(&a_full[s], use & 1, &abort_flag)) { abort_flag = 1; break; }
        if (duse > 0 && !mbar_wait(&d_empty[ds], (duse - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
        tmem_fence_after();
        const uint32_t a0 = smem_addr(sa + s * TC_TILE_BYTES), b0 = smem_addr(sq + qi * H * 128);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16(tmem_base + ds * dcols, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc, k > 0);
        mma_commit(&a_empty[s]);
        mma_commit(&d_full[ds]);
        const bool last_of_seq = (i + 1 == n) || ((t + 1) / tps != b);
        if (last_of_seq) mma_commit(&q_empty[qi]);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int ew = warp - 2;                              // 0 .. 4G-1
    const int g = ew >> 2;                                // group: tiles i = g (mod G), accumulator g
    const int quarter = warp & 3;                         // TMEM lane quarter = the warp's 32 rows of the tile
    float* prm = sparams + g * 4 * H;
    int prev_b = -1;
    for (int i = g; i < n; i += G) {
      const int64_t t = t0 + i;
      const int b = (int)(t / tps), row0 = (int)(t % tps) * TC_M;
      if (b != prev_b) {
        // per-sequence parameters -> this group's shared-memory slot (the group's 4 warps, then a barrier)
        named_barrier(2 + g, 128);
        for (int h = (ew & 3) * 32 + lane; h < H; h += 128) {
          if (MODE == 1) {
            prm[h] = args.theta[(int64_t)b * H + h];
          } else if (MODE == 2) {
            prm[h] = args.smax1[(int64_t)b * H + h];
            prm[H + h] = args.qcn[(int64_t)b * H + h] * args.z;
            prm[2 * H + h] = args.qrn[(int64_t)b * H + h];
          }
        }
        named_barrier(2 + g, 128);
        prev_b = b;
      }
      const int duse = i / G;
      if (!mbar_wait(&d_full[g], duse & 1, &abort_flag)) {
        if (lane == 0) { raise_status(args.status, VK_ERR_TIMEOUT); abort_flag = 1; }
        break;
      }
      tmem_fence_after();
      const int row = row0 + quarter * 32 + lane;          // row of the tensor map (position, or sample index)
      const bool in_rows = row < args.n_rows;
      const int64_t bh0 = (int64_t)b * H;
      const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) + g * dcols;
      bool arch = false;
      float row_add = 0.f, row_eta = 0.f;
      if (MODE >= 1) arch = in_rows && row >= args.arch_lo && row < args.arch_hi;
      if (MODE == 2 && in_rows) {
        row_add = args.page_res[(int64_t)b * args.n_pages + row / PAGE];
        row_eta = args.eta[(int64_t)b * args.N + row];
      }
      const int64_t word = (row0 + quarter * 32) / 32;      // this warp's 32 rows = one bitmap word
      const bool word_ok = word < args.nw;
      const bool emit = MODE == 1 || (MODE == 2 && args.top_j > 0);
      constexpr int NCH = G == 4 ? 4 : 8;                  // 32-head chunks (H <= 128 when G = 4)
      uint32_t mine[NCH];                                  // ballot of head c + lane, per 32-head chunk
      int base[NCH];
#pragma unroll
      for (int cc = 0; cc < NCH; ++cc) {
        const int c = cc * 32;
        if (c >= H) break;
        const int hn = min(32, H - c);                     // 32, or 16 for the last chunk when H % 32 == 16
        uint32_t sel_word = 0;
        if (MODE == 2 && lane < hn && word_ok) sel_word = args.selbm[(bh0 + c + lane) * args.nw + word];
        uint32_t m_lane = 0;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          if (16 * half >= hn) break;
          float v[16];
          tmem_ld16(tbase + c + 16 * half, v);
          tmem_wait_ld();
          if (MODE == 0) {
            if (in_rows) {
#pragma unroll
              for (int j = 0; j < 16; ++j) args.scores[(bh0 + c + 16 * half + j) * args.scores_ld + row] = v[j];
            }
            continue;
          }
#pragma unroll
          for (int jj = 0; jj < 16; ++jj) {
            const int j = 16 * half + jj;
            bool pass = false;
            if (MODE == 1) {
              pass = arch && v[jj] >= prm[c + j];
            } else {
              const uint32_t sw = __shfl_sync(0xffffffffu, sel_word, j);
              const float T = args.lam * (v[jj] + prm[2 * H + c + j] * row_add + prm[H + c + j] * row_eta);
              pass = arch && !((sw >> lane) & 1u) && T > prm[c + j];
            }
            const uint32_t m = __ballot_sync(0xffffffffu, pass);
            if (lane == j) m_lane = m;
          }
        }
        mine[cc] = m_lane;
        if (MODE == 2 && !emit && lane < hn && word_ok) args.firebm[(bh0 + c + lane) * args.nw + word] = m_lane;
      }
      if (emit) {
        // reserve room for every chunk first (the atomics overlap), then read the scores again and scatter
#pragma unroll
        for (int cc = 0; cc < NCH; ++cc) {
          if (cc * 32 >= H) break;
          const int cnt = __popc(mine[cc]);
          base[cc] = cnt ? atomicAdd(&args.cand_cnt[bh0 + cc * 32 + lane], cnt) : 0;
        }
#pragma unroll
        for (int cc = 0; cc < NCH; ++cc) {
          const int c = cc * 32;
          if (c >= H) break;
          const int hn = min(32, H - c);
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            if (16 * half >= hn) break;
            float v[16];
            tmem_ld16(tbase + c + 16 * half, v);
            tmem_wait_ld();
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) {
              const int j = 16 * half + jj;
              const uint32_t m = __shfl_sync(0xffffffffu, mine[cc], j);
              const int bj = __shfl_sync(0xffffffffu, base[cc], j);
              if ((m >> lane) & 1u) {
                const int pos = bj + __popc(m & ((1u << lane) - 1u));
                float val = v[jj];
                if (MODE == 2) val = args.lam * (v[jj] + prm[2 * H + c + j] * row_add + prm[H + c + j] * row_eta);
                if (pos < args.capc) args.cand[(bh0 + c + j) * args.capc + pos] = make_int2(row, __float_as_int(val));
              }
            }
          }
        }
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&d_empty[g]);
    }
  }

  // wind down: every warp is done with tensor memory once all epilogue arrivals happened
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, args.tmem_cols);
  if (threadIdx.x == 0 && abort_flag) raise_status(args.status, VK_ERR_TIMEOUT);
}

// ---------------------------------------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool score_tc_supported(const vk_view& v, int r) {
  return v.dtype == VK_BF16 && r == D_ROPE && v.H % 16 == 0 && v.H >= 16 && v.H <= 256 &&
         (v.rope_ld * 2) % 16 == 0 && (v.rope_bstride * 2) % 16 == 0 && encode_fn() != nullptr;
}

cudaError_t launch_score_tc(const vk_view& v, int row_offset, int row_stride, int n_rows, ScoreTcArgs args,
                            cudaStream_t st) {
  auto encode = encode_fn();
  if (!encode) return cudaErrorNotSupported;
  CUtensorMap kmap, qmap;
  const auto* rope = static_cast<const __nv_bfloat16*>(v.rope) + (int64_t)row_offset * v.rope_ld;
  cuuint64_t kdims[3] = {(cuuint64_t)D_ROPE, (cuuint64_t)n_rows, (cuuint64_t)v.B};
  cuuint64_t kstr[2] = {(cuuint64_t)(v.rope_ld * row_stride * 2), (cuuint64_t)(v.rope_bstride * 2)};
  cuuint32_t kbox[3] = {D_ROPE, TC_M, 1};
  cuuint32_t es3[3] = {1, 1, 1};
  // each row contributes one 128-byte segment 1152 bytes apart: no L2 promotion, so DRAM reads only those bytes
  if (encode(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(rope), kdims, kstr, kbox, es3,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  cuuint64_t qdims[2] = {(cuuint64_t)D_ROPE, (cuuint64_t)v.B * v.H};
  cuuint64_t qstr[1] = {(cuuint64_t)D_ROPE * 2};
  cuuint32_t qbox[2] = {D_ROPE, (cuuint32_t)v.H};
  cuuint32_t es2[2] = {1, 1};
  if (encode(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(v.q_rope), qdims, qstr, qbox, es2,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  args.B = v.B;
  args.H = v.H;
  args.N = v.N;
  args.n_rows = n_rows;
  args.tiles_per_seq = (n_rows + TC_M - 1) / TC_M;
  args.total_tiles = (int64_t)args.tiles_per_seq * v.B;
  args.n_pages = (v.N + PAGE - 1) / PAGE;
  const int G = v.H <= 128 ? 4 : 2;                   // G accumulators of H columns fit in 512 TMEM columns
  uint32_t cols = 32;
  while (cols < (uint32_t)(G * v.H)) cols <<= 1;
  args.tmem_cols = cols;
  const int grid = (int)std::min<int64_t>(args.total_tiles, 152);
  const size_t smem = TcSmem(v.H).total;
  auto pick = [&](auto kernel, int g) -> cudaError_t {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (grid > 0) kernel<<<grid, (2 + 4 * g) * 32, smem, st>>>(kmap, qmap, args);
    return cudaSuccess;
  };
  cudaError_t e;
  const int m = args.mode;
  if (G == 4) e = m == 0 ? pick(k_score_tc<4, 0>, 4) : m == 1 ? pick(k_score_tc<4, 1>, 4) : pick(k_score_tc<4, 2>, 4);
  else e = m == 0 ? pick(k_score_tc<2, 0>, 2) : m == 1 ? pick(k_score_tc<2, 1>, 2) : pick(k_score_tc<2, 2>, 2);
  if (e != cudaSuccess) return e;
  if (grid > 0) count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
