// k_sigma.cu -- the sigma selector of tier 1 (Sec. 4.1, Eq. 3) on the tensor cores, bf16 caches.
//
// For each closed block of T cached rows (T a multiple of 128) with R = the block's 64 RoPE-branch columns,
//   sigma_u = | R_u - (Phi Phi^T R)_u |,
// Phi [T x m] the orthonormal basis of the sequence-axis DFT bins 0 .. kappa-1: the constant, the cosine and sine of
// every bin that stands for a conjugate pair, and the alternation (-1)^u when kappa reaches T/2. The low-pass
// reconstruction of Eq. 3 (inverse DFT of the kept bins) is exactly this projection: a paired bin's weight 2 is the
// square of its basis norm sqrt(2/T). Two thin contractions per block on tcgen05, one CTA per SM walking a range of
// (sequence, block) items:
//   phase 1  C^T [64 dims x mp] = R^T Phi, accumulated over the block's 128-row chunks: A = the R chunk read
//            MN-major straight from its TMA tile, B = the Phi^T chunk; M = 64, N = mp, K = 128 per chunk;
//   phase 2  low [128 rows x 64 dims] = Phi_chunk C: A = the Phi chunk, B = C rounded to bf16 by the epilogue into
//            shared memory; M = 128, N = 64, K = mp, into one of four tensor-memory buffers. The R chunk is loaded
//            again (mostly from L2) into a ring of its own, and the epilogue (one thread per row) takes the row's low
//            part from tensor memory and the row from shared memory, and writes sigma.
// Phase 2 of an item needs the item's whole C, so the items are software-pipelined: in round r every role takes phase
// 1 of the CTA's item r and phase 2 of item r - 1, chunk by chunk, and the R stream from HBM (phase 1, a ring of its
// own) goes on while the item before takes its phase 2. C is double-buffered in shared memory (item r's is written
// while item r - 1's phase 2 products may still read the other).
// Roles: warp 0 TMA producer, warp 1 MMA issuer, warps 2..9 epilogue in two groups of four (one warp per
// tensor-memory lane quarter each): group 0 writes C and takes the even phase 2 chunks, group 1 the odd ones.
// Phi is built in the workspace in bf16 twice: Phi^T [mp][T] and Phi [T][mp] (mp = 32 for kappa <= 16, 64 for
// kappa <= 32, else 128). At mp = 32 the phase 2 operands (the Phi chunk and C) have 64-byte rows and the 64-byte
// swizzle.
// Rows past the last closed block (the open tail) get sigma = -1. Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"

namespace vk {

namespace {

constexpr int SG_CH = 128;                 // rows per chunk
constexpr int SG_THREADS = 10 * 32;
constexpr uint32_t SG_RBYTES = SG_CH * 128;  // one chunk of R: 128 rows x 64 bf16

template <int MP>
struct SgCfg {
  static constexpr uint32_t PHT = 2 * MP * 128;          // Phi^T chunk: two 64-row boxes of MP x 128 B
  static constexpr uint32_t STAGE1 = SG_RBYTES + PHT;    // a stage: an R chunk and its Phi^T chunk
  static constexpr int S1 = MP == 32 ? 6 : MP == 64 ? 5 : 3;   // the stage ring (the HBM stream)
  static constexpr int R2 = MP == 32 ? 4 : 3;                  // phase 2 ring of R chunks for the epilogue
  static constexpr uint32_t ROW2 = MP == 32 ? 64 : 128;  // row bytes of C, the phase 2 B operand
  static constexpr int NL = 4;                           // tensor-memory buffers of the phase 2 product
  static constexpr uint32_t CB = 64 * MP * 2;            // C as the phase 2 B operand: MP / 64 blocks of 64 x 128 B
  static constexpr uint32_t cbuf = S1 * STAGE1;          // two C buffers: one block's C while the next is written
  static constexpr uint32_t r2 = cbuf + 2 * CB;
  static constexpr uint32_t bars = r2 + R2 * SG_RBYTES;
  static constexpr uint32_t total = bars + (2 * S1 + 2 * R2 + 2 + 2 * NL) * 8 + 1024;
  static_assert(total <= 232448, "sigma shared memory exceeds the 227 KB opt-in limit");
};

__device__ __forceinline__ void sg_tma_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ void sg_tma_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::
          "r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}
// Shared-memory matrix descriptor, 128-byte swizzle, 8-row groups 1024 B apart; lbo only matters for an MN-major
// operand wider than one 64-element atom (not used here).
__device__ __forceinline__ uint64_t sg_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}
// MN-major operand, 128-byte swizzle: 64-element atoms along M/N `lbo` bytes apart, 8-row K groups 1024 B apart.
__device__ __forceinline__ uint64_t sg_desc_mn(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024u >> 4) << 32) | ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}
// K-major operand with 64-byte rows, 64-byte swizzle: 8-row groups 512 B apart.
__device__ __forceinline__ uint64_t sg_desc64(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(512u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)4u << 61);
}
// The phase 2 descriptor for the operand width of MP.
template <int MP>
__device__ __forceinline__ uint64_t sg_desc2(uint32_t saddr) {
  return MP == 32 ? sg_desc64(saddr) : sg_desc(saddr);
}
__device__ __forceinline__ void sg_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void sg_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ void sg_ld32(uint32_t taddr, float* v) {   // 32 columns of this thread's lane
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
// M = 64 accumulator: lanes 0..15 of the warp get columns [c, c + 32), lanes 16..31 columns [c + 32, c + 64) of the
// same 16 tensor-memory lanes.
__device__ __forceinline__ void sg_ld16x2(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], 32;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

__device__ __forceinline__ void fence_async_smem_sg() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }
// Warp-uniform bounded wait: lane 0 polls, the warp takes its verdict.
__device__ __forceinline__ bool warp_wait_sg(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int lane) {
  bool w = true;
  if (lane == 0) w = mbar_wait(bar, parity, abort_flag);
  return __shfl_sync(0xffffffffu, w, 0);
}

struct SigmaArgs {
  int B, N, T, nb;           // nb = closed blocks per sequence
  long long items;           // B * nb
  const __nv_bfloat16* rope;
  int64_t rld, rbs;
  float* sigma;              // [B, N]
  int* status;
};

template <int MP>
__global__ void __launch_bounds__(SG_THREADS, 1) k_sigma(const __grid_constant__ CUtensorMap rmap,
                                                       const __grid_constant__ CUtensorMap ptmap, const SigmaArgs args) {
  using L = SgCfg<MP>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* cb = smem + L::cbuf;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::bars);
  uint64_t* full1 = bars;                  // [S1] a stage has landed
  uint64_t* empty1 = full1 + L::S1;        // [S1] its products (both phases) are done
  uint64_t* c_full = empty1 + L::S1;       // phase 1 of an item is complete
  uint64_t* c_ready = c_full + 1;          // the epilogue has written C (bf16) for phase 2
  uint64_t* l_full = c_ready + 1;          // [NL] a phase 2 chunk's low part is in tensor memory
  uint64_t* l_empty = l_full + L::NL;      // [NL] the epilogue has read it
  uint64_t* r_full = l_empty + L::NL;      // [R2] a phase 2 R chunk has landed
  uint64_t* r_empty = r_full + L::R2;      // [R2] the epilogue is done with it
  unsigned char* rbuf = smem + L::r2;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long i0 = args.items * blockIdx.x / gridDim.x, i1 = args.items * (blockIdx.x + 1) / gridDim.x;
  const int nchunk = args.T / SG_CH;
  constexpr uint32_t C_COL = 0, L_COL = 128;               // tensor memory: C^T, then four 64-column low buffers

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < L::S1; ++s) { mbar_init(&full1[s], 1); mbar_init(&empty1[s], 1); }
    mbar_init(c_full, 1);
    mbar_init(c_ready, 4);
    for (int i = 0; i < L::NL; ++i) { mbar_init(&l_full[i], 1); mbar_init(&l_empty[i], 4); }
    for (int i = 0; i < L::R2; ++i) { mbar_init(&r_full[i], 1); mbar_init(&r_empty[i], 4); }
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, 512);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    // Round r loads phase 1 of the CTA's item r and phase 2 of item r - 1, chunk by chunk, so that the phase 1 stream
    // from HBM goes on while the item before takes its phase 2 (whose R chunks come again, mostly from L2).
    if (lane == 0) {
      int n1 = 0, n2 = 0;                                 // phase 1 stages and phase 2 chunks issued
      bool ok = true;
      const long long nitems = i1 - i0;
      for (long long r = 0; r <= nitems && ok; ++r) {
        const bool has1 = r < nitems, has2 = r >= 1;
        const long long it1 = i0 + r, it2 = i0 + r - 1;
        const int b1 = has1 ? (int)(it1 / args.nb) : 0, blk1 = has1 ? (int)(it1 - (long long)b1 * args.nb) : 0;
        const int b2 = has2 ? (int)(it2 / args.nb) : 0, blk2 = has2 ? (int)(it2 - (long long)b2 * args.nb) : 0;
        for (int c = 0; c < nchunk; ++c) {
          const int u0 = c * SG_CH;
          // the stage: chunk c of Phi^T (phase 1's B operand and phase 2's A operand: both phases of the round use
          // the same rows of the basis) and, with a phase 1, item r's R chunk
          const int s = n1 % L::S1, use = n1 / L::S1;
          if (use > 0 && !mbar_wait(&empty1[s], (use - 1) & 1, &abort_flag)) { ok = false; break; }
          unsigned char* st = smem + s * L::STAGE1;
          mbar_arrive_expect_tx(&full1[s], L::PHT + (has1 ? SG_RBYTES : 0u));
          if (has1) sg_tma_3d(st, &rmap, 0, blk1 * args.T + u0, b1, &full1[s]);
          sg_tma_2d(st + SG_RBYTES, &ptmap, u0, 0, &full1[s]);
          sg_tma_2d(st + SG_RBYTES + MP * 128, &ptmap, u0 + 64, 0, &full1[s]);
          ++n1;
          if (has2) {
            const int s2 = n2 % L::R2, use2 = n2 / L::R2;
            if (use2 > 0 && !mbar_wait(&r_empty[s2], (use2 - 1) & 1, &abort_flag)) { ok = false; break; }
            mbar_arrive_expect_tx(&r_full[s2], SG_RBYTES);
            sg_tma_3d(rbuf + s2 * SG_RBYTES, &rmap, 0, blk2 * args.T + u0, b2, &r_full[s2]);
            ++n2;
          }
        }
      }
      if (!ok) abort_flag = 1;
      // drain: the last load of every stage has landed before the CTA may leave (already true unless it aborted)
      for (int k = std::max(0, n1 - L::S1); k < n1; ++k) mbar_wait(&full1[k % L::S1], (k / L::S1) & 1, nullptr);
      for (int k = std::max(0, n2 - L::R2); k < n2; ++k) mbar_wait(&r_full[k % L::R2], (k / L::R2) & 1, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      // phase 1: D = C^T (M = 64 dims, N = MP), A = R^T MN-major (bit 15), B = Phi^T K-major
      constexpr uint32_t idesc1 = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | ((uint32_t)(MP >> 3) << 17) |
                                  ((uint32_t)(64 >> 4) << 24);
      // phase 2: D = low (M = 128 rows, N = 64 dims), A = Phi MN-major (bit 15: the Phi^T chunk), B = C K-major
      constexpr uint32_t idesc2 = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | ((uint32_t)(64 >> 3) << 17) |
                                  ((uint32_t)(128 >> 4) << 24);
      // round r: phase 1 of item r (into C^T) and phase 2 of item r - 1 (from C in shared memory), chunk by chunk
      int n1 = 0, n2 = 0, ncf = 0;                        // ncf: commits of c_full
      bool ok = true;
      const long long nitems = i1 - i0;
      for (long long r = 0; r <= nitems && ok; ++r) {
        const bool has1 = r < nitems, has2 = r >= 1;
        if (has2) {
          // item r - 1's C is in shared memory and its C^T has left tensor memory (item r may accumulate there)
          if (!mbar_wait(c_ready, (uint32_t)((r - 1) & 1), &abort_flag)) { ok = false; break; }
          tmem_fence_after();
        }
        const uint32_t cba = smem_addr(cb + (uint32_t)((r - 1) & 1) * L::CB);
        for (int c = 0; c < nchunk; ++c) {
          const int s = n1 % L::S1, use = n1 / L::S1;
          if (!mbar_wait(&full1[s], use & 1, &abort_flag)) { ok = false; break; }
          const int lb = n2 % L::NL, luse = n2 / L::NL;
          if (has2 && luse > 0 && !mbar_wait(&l_empty[lb], (luse - 1) & 1, &abort_flag)) { ok = false; break; }
          tmem_fence_after();
          const uint32_t st = smem_addr(smem + s * L::STAGE1);
          if (has1) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {                 // 16 rows per instruction
              const uint64_t ad = sg_desc(st + j * 2048);
              const uint64_t bd = sg_desc(st + SG_RBYTES + (j >> 2) * (MP * 128) + (j & 3) * 32);
              sg_mma(tmem + C_COL, ad, bd, idesc1, (c > 0 || j > 0) ? 1u : 0u);
            }
          }
          if (has2) {
            // A = the Phi^T chunk read MN-major (the chunk's 128 rows in two 64-row atoms MP x 128 B apart, 16 bins
            // per instruction), B = item r - 1's C
#pragma unroll
            for (int j = 0; j < MP / 16; ++j) {
              const uint64_t ad = sg_desc_mn(st + SG_RBYTES + j * 2048, MP * 128);
              const uint64_t bd = sg_desc2<MP>(cba + (j >> 2) * 8192 + (j & 3) * 32);
              sg_mma(tmem + L_COL + 64 * lb, ad, bd, idesc2, j > 0 ? 1u : 0u);
            }
          }
          sg_commit(&empty1[s]);
          ++n1;
          if (has2) {
            sg_commit(&l_full[lb]);
            ++n2;
          }
        }
        if (ok && has1) {
          sg_commit(c_full);
          ++ncf;
        }
      }
      if (!ok) {
        abort_flag = 1;
        raise_status(args.status, VK_ERR_TIMEOUT);
      }
      // nothing this thread issued may outlive the CTA
      sg_commit(c_full);
      mbar_wait(c_full, ncf & 1, nullptr);
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int q = warp & 3;                               // tensor-memory lane quarter
    const int eg = (warp - 2) >> 2;                       // epilogue group: 0 writes C, the groups split the chunks
    const uint32_t lq = (uint32_t)(32 * q) << 16;
    // round r: phase 2 of item r - 1 (the groups take alternate chunks), then group 0 turns item r's C^T into C
    bool ok = true;
    const long long nitems = i1 - i0;
    for (long long r = 0; r <= nitems && ok; ++r) {
      if (r >= 1) {
        const long long it = i0 + r - 1;
        const int b = (int)(it / args.nb), blk = (int)(it - (long long)b * args.nb);
        // phase 2: one row per thread; the row from the R ring (128-byte swizzle: chunk k of row x sits at k ^ (x & 7));
        // chunk c of this item is the ((r - 1) nchunk + c)-th phase 2 chunk of the CTA, taken by group c % 2
        for (int c = eg; c < nchunk; c += 2) {
          const int nl = (int)(r - 1) * nchunk + c;
          const int lb = nl % L::NL, luse = nl / L::NL;
          const int s2 = nl % L::R2, use2 = nl / L::R2;
          if (!warp_wait_sg(&l_full[lb], luse & 1, &abort_flag, lane) ||
              !warp_wait_sg(&r_full[s2], use2 & 1, &abort_flag, lane)) {
            ok = false;
            break;
          }
          tmem_fence_after();
          float lo[64];
          sg_ld32(tmem + lq + L_COL + 64 * lb, lo);
          sg_ld32(tmem + lq + L_COL + 64 * lb + 32, lo + 32);
          tmem_wait_ld();
          tmem_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&l_empty[lb]);
          const int x = 32 * q + lane;                      // row within the chunk
          const int u = blk * args.T + c * SG_CH + x;
          const unsigned char* rrow = rbuf + s2 * SG_RBYTES + x * 128;
          uint4 rv[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) rv[k] = *reinterpret_cast<const uint4*>(rrow + ((k ^ (x & 7)) * 16));
          __syncwarp();
          if (lane == 0) mbar_arrive(&r_empty[s2]);
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint4 w = rv[k];
            const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float d0 = bf_lo(ww[e]) - lo[8 * k + 2 * e], d1 = bf_hi(ww[e]) - lo[8 * k + 2 * e + 1];
              acc = fmaf(d0, d0, acc);
              acc = fmaf(d1, d1, acc);
            }
          }
          args.sigma[(int64_t)b * args.N + u] = sqrtf(acc);
        }
        if (!ok) break;
      }
      if (r < nitems && eg == 0) {
        if (!warp_wait_sg(c_full, (uint32_t)(r & 1), &abort_flag, lane)) { ok = false; break; }
        tmem_fence_after();
        {
          // C^T row d = 16 q + (lane % 16) (M = 64 layout), bins 32 (lane / 16) + 64 kb .. + 31 -> bf16 into the B
          // operand of phase 2: row d of K block kb, 16-byte chunks 4 (lane / 16) .. + 3, 128-byte swizzle (at MP = 32:
          // 64-byte rows of the 32 bins, 64-byte swizzle, written by the lanes of the first half)
          const int d = 16 * q + (lane & 15), half = lane >> 4;
#pragma unroll
          for (int kb = 0; kb < (MP + 63) / 64; ++kb) {
            float v[32];
            sg_ld16x2(tmem + lq + C_COL + 64 * kb, v);
            tmem_wait_ld();
            if (MP == 32 && half) continue;               // columns past the 32 bins
            unsigned char* row = cb + (uint32_t)(r & 1) * L::CB + kb * 8192 + d * L::ROW2;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const __nv_bfloat162 pb = __floats2bfloat162_rn(v[8 * k + 2 * e], v[8 * k + 2 * e + 1]);
                w[e] = *reinterpret_cast<const uint32_t*>(&pb);
              }
              const int chunk = MP == 32 ? (k ^ ((d >> 1) & 3)) : ((4 * half + k) ^ (d & 7));
              *reinterpret_cast<uint4*>(row + chunk * 16) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        }
        fence_async_smem_sg();
        tmem_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(c_ready);
      }
    }
    if (!ok && lane == 0) {
      abort_flag = 1;
      raise_status(args.status, VK_ERR_TIMEOUT);
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Phi^T [mp][T] in bf16 (the orthonormal low-pass basis, column n of Phi = row n here): 0 the constant 1/sqrt(T);
// 2 k - 1 and 2 k the cosine and sine of bin k = 1 .. npair times sqrt(2/T); then the alternation (-1)^u / sqrt(T)
// when kappa > T/2; zero up to mp. The angle is reduced exactly (k u mod T, in integers) before cospif / sinpif: fp32
// is ample for values rounded to bf16. Consecutive threads take consecutive positions u of one row.
__global__ void k_sigma_basis(int T, int kappa, int mp, __nv_bfloat16* phit) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)T * mp) return;
  const int n = (int)(i / T), u = (int)(i - (int64_t)n * T);
  const int npair = max(0, min(kappa - 1, T / 2 - 1));     // bins 1 .. npair (T is even)
  const int m = 1 + 2 * npair + (kappa > T / 2 ? 1 : 0);
  const float inv_sqrt_t = rsqrtf((float)T);
  float v = 0.f;
  if (n == 0) {
    v = inv_sqrt_t;
  } else if (n < 1 + 2 * npair) {
    const int k = (n + 1) / 2;
    const float x = 2.f * (float)(((int64_t)k * u) % T) / (float)T;
    v = sqrtf(2.f) * inv_sqrt_t * ((n & 1) ? cospif(x) : sinpif(x));
  } else if (n < m) {
    v = ((u & 1) ? -1.f : 1.f) * inv_sqrt_t;
  }
  phit[i] = __float2bfloat16_rn(v);
}

__global__ void k_sigma_tail(int N, int closed, float* sigma) {
  const int b = blockIdx.y;
  for (int u = closed + blockIdx.x * blockDim.x + threadIdx.x; u < N; u += gridDim.x * blockDim.x)
    sigma[(int64_t)b * N + u] = -1.f;
}

PFN_cuTensorMapEncodeTiled_v12000 sg_encode() {
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

template <int MP>
cudaError_t launch_sigma_mp(const vk_view& v, int T, int kappa, float* sigma, void* ws, int* status, cudaStream_t st) {
  auto encode = sg_encode();
  if (!encode) return cudaErrorNotSupported;
  __nv_bfloat16* phit = static_cast<__nv_bfloat16*>(ws);
  const int64_t ne = (int64_t)T * MP;
  k_sigma_basis<<<(unsigned)((ne + 255) / 256), 256, 0, st>>>(T, kappa, MP, phit);
  count_launches(1);
  const int nb = v.N / T, closed = nb * T;
  if (closed < v.N) {
    dim3 g((unsigned)std::min<int64_t>((v.N - closed + 255) / 256, 64), v.B);
    k_sigma_tail<<<g, 256, 0, st>>>(v.N, closed, sigma);
    count_launches(1);
  }
  if (nb == 0) return cudaGetLastError();
  CUtensorMap rmap, ptmap;
  {
    cuuint64_t dims[3] = {(cuuint64_t)D_ROPE, (cuuint64_t)v.N, (cuuint64_t)v.B};
    cuuint64_t str[2] = {(cuuint64_t)(v.rope_ld * 2), (cuuint64_t)(v.rope_bstride * 2)};
    cuuint32_t box[3] = {64, (cuuint32_t)SG_CH, 1};
    cuuint32_t es[3] = {1, 1, 1};
    if (encode(&rmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(v.rope), dims, str, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    cuuint64_t dims[2] = {(cuuint64_t)T, (cuuint64_t)MP};
    cuuint64_t str[1] = {(cuuint64_t)T * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)MP};
    cuuint32_t es[2] = {1, 1};
    if (encode(&ptmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, phit, dims, str, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  SigmaArgs a{};
  a.B = v.B;
  a.N = v.N;
  a.T = T;
  a.nb = nb;
  a.items = (long long)v.B * nb;
  a.rope = static_cast<const __nv_bfloat16*>(v.rope);
  a.rld = v.rope_ld;
  a.rbs = v.rope_bstride;
  a.sigma = sigma;
  a.status = status;
  const int grid = (int)std::min<long long>(a.items, sm_count());
  const size_t smem = SgCfg<MP>::total;
  cudaError_t e = cudaFuncSetAttribute(k_sigma<MP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_sigma<MP><<<grid, SG_THREADS, smem, st>>>(rmap, ptmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace

int sigma_basis_cols(int kappa) { return kappa <= 16 ? 32 : kappa <= 32 ? 64 : 128; }

size_t sigma_workspace_bytes(int T, int kappa) {
  return 256 + (size_t)2 * sigma_basis_cols(kappa) * (size_t)T;   // status word, Phi^T (bf16)
}

cudaError_t launch_sigma(const vk_view& v, int T, int kappa, float* sigma, void* ws, cudaStream_t st) {
  int* status = static_cast<int*>(ws);
  void* tables = static_cast<char*>(ws) + 256;
  const int mp = sigma_basis_cols(kappa);
  return mp == 32   ? launch_sigma_mp<32>(v, T, kappa, sigma, tables, status, st)
         : mp == 64 ? launch_sigma_mp<64>(v, T, kappa, sigma, tables, status, st)
                    : launch_sigma_mp<128>(v, T, kappa, sigma, tables, status, st);
}

}  // namespace vk
