// k_score_tc.cu -- RoPE-branch scoring on the 5th-generation tensor cores (tcgen05), bf16, r in {8, 16, 32, 64}.
//
// a[h,u] = Qr_h . K_u for every cached row (Eq. 4's exact summand): per sequence the [H x 64] query times the
// [64 x N] RoPE slice, a dense contraction at H flop per byte. For a width-r digest D_u (r = 32, 16, 8) it is
// (O Qr_h)[0:r] . D_u: the rotated query is fp32, so it enters as two bf16 parts (high and the rounding rest),
// two products accumulated in fp32, and the digest tile is read with the swizzle its row width allows (64, 32 or
// 16 bytes; at r = 8 the second 8 columns of the K = 16 product are the query's zero padding). One CTA per SM
// walks a contiguous range of 128-row tiles:
//   warp 0 (one thread)  TMA: the tile's 128 x 64 bf16 slice (128 B of every 1152-B row, 128-byte swizzle) into a
//                        7-stage ring, and the sequence's H x 64 query when the sequence changes;
//   warp 1 (one thread)  D = Q . K^T on tcgen05: M = 64 heads (H <= 64) or 128 per head group, N = 128 rows,
//                        K = 16 (x4), issued as one burst into one of G accumulators in tensor memory (TMEM lane =
//                        head, column = row); tcgen05.commit frees the ring slot and hands the accumulator on;
//   G groups of 4 warps  epilogue, group g taking tiles i = g (mod G). The thread of head h reads its logits in
//                        32-row chunks (tcgen05.ld 16x32bx2 for M = 64, 32x32b for M = 128), so a chunk's
//                        threshold test is directly the head's 32-bit bitmap word of those rows:
//                        mode 0  write scores [B][H][ld], fp32 (or bf16 for the strided row sample that only
//                                feeds the threshold estimate),
//                        mode 1  emit (u, a) for archive rows with a >= theta[b,h] into per-head candidate lists:
//                                one atomic per thread and tile reserves the room, then the chunk is staged in
//                                shared memory and only its set bits are visited,
//                        mode 2  trigger: T = lambda (a + |(O Qr)[r:]| page_res + z |Qc| eta) > s*_h for archive
//                                rows outside S_h -> 32-row words of the fired bitmap (or candidates for top_j).
//                                With a rank-SK content sketch (Eq. 4), each stage also holds the tile's sketch
//                                rows s_u (TMA, [TM x SK] bf16) and the query buffer the bf16 high and low parts of
//                                p_h = V^T Qc_h, so that p_h . s_u accumulates into the same tensor-memory
//                                accumulator as a (SK/16 x 2 more instructions); the certificate's |Qc| is then the
//                                sketch residual norm, passed in its place.
//                                With the page norm maxima given, a tile in which no head's page bound can reach
//                                s*_h (page_may_fire) is skipped: the producer warp decides per tile, loads nothing
//                                and tells the MMA issuer to issue nothing; the epilogue, applying the same test per
//                                head and page, writes empty words without reading the accumulator.
// Every mbarrier wait is bounded; a wait that gives up raises VK_ERR_TIMEOUT and the CTA winds down.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"
#include "vk_score_tc.h"

namespace vk {


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

// K-major operand descriptor for rows of ROWB bytes: 128, 64 and 32 take the matching swizzle (8-row atoms of
// 8 x ROWB bytes, the next 8 rows ROWB x 8 bytes on); 16 is the unswizzled layout of 8-row x 16-byte core matrices
// 128 bytes apart, whose leading offset (the next 8 columns along K) is 0: the r = 8 digest's K = 16 product reads
// its 8 columns twice, against the query's 8 values and its 8 zeros.
template <int ROWB>
__device__ __forceinline__ uint64_t kmajor_desc(uint32_t saddr) {
  constexpr uint64_t layout = ROWB == 128 ? 2 : ROWB == 64 ? 4 : ROWB == 32 ? 6 : 0;
  constexpr uint64_t lbo = ROWB == 16 ? 0 : 1;
  constexpr uint64_t sbo = (uint64_t)(8 * ROWB) >> 4;
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | (lbo << 16) | (sbo << 32) | ((uint64_t)1u << 46) | (layout << 61);
}

// Instruction descriptor of tcgen05.mma kind::f16// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulate (bits 4-5 = 1), A and B bf16 (7-9, 10-12 = 1),
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

// One 32-row chunk of this thread's head: M = 128 (lane = head) reads 32 columns of its own lane; M = 64 (16 heads
// per lane quarter) reads with 16x32bx2, lanes 0..15 columns [col, col + 32) and lanes 16..31 [col + 32, col + 64).
template <int MH>
__device__ __forceinline__ void tmem_ld_chunk(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  if (MH == 128) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
        "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
  } else {
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,"
        "%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], 32;\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
  }
}

// Whether a row of a 64-row page can fire for a head: its trigger score lambda (a + z |Qc| eta_u) is at most the page
// bound lambda (|Qr| max|K_u| + z |Qc| max eta_u) (Cauchy-Schwarz, a = Qr . K_u); the bound is inflated by 2^-10 so
// that the fp32 rounding of the scores and norms cannot turn a skip into a missed row. Rounded operations are
// explicit so that the producer and the epilogue reach the same decision bit for bit.
__device__ __forceinline__ bool page_may_fire(float lam, float qrf, float zqc, float sstar, float pk, float pe) {
  const float bound = __fmul_rn(__fmul_rn(lam, __fadd_rn(__fmul_rn(qrf, pk), __fmul_rn(zqc, pe))), 1.0f + 0x1p-10f);
  return !(bound <= sstar);
}

// Bits of the rows [lo, hi) within the 32 rows starting at r0.
__device__ __forceinline__ uint32_t range_mask(int r0, int lo, int hi) {
  const int a = max(lo - r0, 0), e = min(hi - r0, 32);
  if (e <= a) return 0u;
  const uint32_t upto = e >= 32 ? 0xffffffffu : ((1u << e) - 1u);
  return upto & ~((1u << a) - 1u);
}

// One configuration of the kernel: TM rows per tile (the MMA's N: 64 or 128), G epilogue groups of WPQ warps per
// tensor-memory lane quarter (a tile's 32-row chunks of a head are split among them), NACC accumulators of
// NHG x TM tensor-memory columns (all 512 columns), a ring of STAGES tiles (96 to 112 KB). Shared memory from a
// 1024-aligned base: the ring, two query buffers of NHG x MH rows (one with a sketch, whose query parts take the
// room), 128 B of staging per epilogue thread (modes 1, 2), barriers. SK: the content sketch width (mode 2), or 0.
template <int MH, int NHG, int TM_, int G_, int WPQ_ = 1, int RW_ = 64, int SK_ = 0, int MODE_ = 0>
struct TcCfg {
  static constexpr int TM = TM_;
  static constexpr int G = G_;
  static constexpr int WPQ = WPQ_;
  static constexpr int RW = RW_;                         // score width: the RoPE columns (64) or a digest width
  static constexpr int KP = RW < 16 ? 16 : RW;           // the product's K (r = 8 padded to 16 on the query side)
  static constexpr int QPARTS = RW == 64 ? 1 : 2;        // bf16 query parts: the RoPE query, or high + low
  static constexpr uint32_t QROW = KP * 2;               // bytes per query row
  static constexpr uint32_t QPART = NHG * MH * QROW;     // one query part
  static constexpr uint32_t DCOLS = NHG * TM;            // columns per accumulator
  static constexpr int NACC = 512 / DCOLS;
  static constexpr int SK = SK_;
  static constexpr uint32_t KTILE = TM * RW * 2;         // TM rows x RW bf16
  static constexpr uint32_t TILE = KTILE + TM * SK * 2;  // ... then TM rows x SK bf16 of sketch
  static constexpr uint32_t SQPART = NHG * MH * SK * 2;  // one bf16 part of the sketch query p
  static constexpr int NC = MH == 128 ? TM / 32 : TM / 64;   // 32-row chunks per lane and tile
  static constexpr int NCT = NC / WPQ;                   // of which one epilogue thread takes
  static constexpr int EW = 4 * G * WPQ;                 // epilogue warps
  static constexpr int THREADS = (2 + EW) * 32;
  static constexpr int QB = SK > 0 ? 1 : 2;              // query buffers
  static constexpr uint32_t qbuf = QPARTS * QPART + 2 * SQPART;
  static constexpr uint32_t STG = EW * 32 * 128;
  // as many ring stages as fit beside the queries and the staging rows, up to 112 KB of tiles (160 KB with the
  // sketch's wider stages; 28 at most)
  static constexpr uint32_t RING_CAP = (SK > 0 ? 160u : 112u) * 1024u;
  static constexpr int STAGES_FIT = (int)((224u * 1024u - QB * qbuf - STG) / TILE);
  static constexpr int STAGES_CAP = (int)(RING_CAP / TILE) < 28 ? (int)(RING_CAP / TILE) : 28;
  static constexpr int STAGES = STAGES_FIT < STAGES_CAP ? STAGES_FIT : STAGES_CAP;
  static constexpr uint32_t a = 0;
  static constexpr uint32_t q = a + STAGES * TILE;
  static constexpr uint32_t stg = q + QB * qbuf;
  // mode 2: a ring of the tiles' eta rows (TM fp32 each), filled by the producer and released by the epilogue; it
  // holds the tiles that sit in the stage ring and in the accumulators at once
  static constexpr int E = MODE_ == 2 ? STAGES + NACC : 0;
  static constexpr uint32_t eta = stg + STG;
  static constexpr uint32_t bars = eta + E * TM * 4;
  static constexpr uint32_t total = bars + (2 * STAGES + 4 + 2 * NACC + 2 * E) * 8 + 1024;
  static_assert(G <= NACC, "every epilogue group needs an accumulator of its own");
  static_assert(NC % WPQ == 0 && STAGES >= 4, "configuration");
  static_assert(TILE % 1024 == 0 && qbuf % 1024 == 0 && (SK == 0 || SK == 16 || SK == 32 || SK == 64), "alignment");
  static_assert(total <= 232448, "scoring shared memory exceeds the 227 KB opt-in limit");
};

template <int MH, int NHG, int MODE, int TM_, int G_, int WPQ_, int RW_, int SK_>
__global__ void __launch_bounds__(TcCfg<MH, NHG, TM_, G_, WPQ_, RW_, SK_, MODE>::THREADS, 1)
    k_score_tc(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
               const __grid_constant__ CUtensorMap smap, const __grid_constant__ CUtensorMap sqmap,
               const __grid_constant__ CUtensorMap emap, const ScoreTcArgs args) {
  using L = TcCfg<MH, NHG, TM_, G_, WPQ_, RW_, SK_, MODE>;
  static_assert(SK_ == 0 || MODE == 2, "the sketch belongs to the trigger");
  constexpr int G = L::G, TC_M = L::TM, TC_STAGES = L::STAGES, NACC = L::NACC;
  constexpr uint32_t TC_TILE_BYTES = L::TILE;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int H = args.H;
  unsigned char* sa = smem + L::a;
  unsigned char* sq = smem + L::q;
  float* stg = reinterpret_cast<float*>(smem + L::stg);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::bars);
  uint64_t* a_full = bars;
  uint64_t* a_empty = bars + TC_STAGES;
  uint64_t* q_full = bars + 2 * TC_STAGES;              // [2]
  uint64_t* q_empty = q_full + 2;                        // [2]
  uint64_t* d_full = q_empty + 2;                        // [NACC]
  uint64_t* d_empty = d_full + NACC;                     // [NACC]
  uint64_t* e_full = d_empty + NACC;                     // [E] mode 2: a tile's eta rows landed
  uint64_t* e_empty = e_full + L::E;                     // [E] the epilogue is done with them
  float* eta_s = reinterpret_cast<float*>(smem + L::eta);
  const bool eta_tma = MODE == 2 && args.eta_tma;       // else the epilogue reads eta from global memory
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  __shared__ int skip_stage[TC_STAGES];                  // mode 2 page skip: the ring stage's tile was not loaded
  const bool page_skip = MODE == 2 && L::RW == 64 && L::SK == 0 && args.page_knorm != nullptr;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t total = args.total_tiles;
  const int64_t t0 = total * blockIdx.x / gridDim.x, t1 = total * (blockIdx.x + 1) / gridDim.x;
  const int n = (int)(t1 - t0);
  const int tps = args.tiles_per_seq;
  const int b_first = (int)(t0 / tps);
  const int kt_first = (int)(t0 - (int64_t)b_first * tps);
  // (sequence, tile within it) of the range's tiles, stepped without divisions: a 64-bit division per tile on
  // the producer's or the MMA issuer's thread is slower than the tile's whole TMA + MMA work
  constexpr uint32_t DCOLS = L::DCOLS;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < TC_STAGES; ++s) { mbar_init(&a_full[s], 1); mbar_init(&a_empty[s], 1); }
    for (int i = 0; i < 2; ++i) { mbar_init(&q_full[i], 1); mbar_init(&q_empty[i], 1); }
    for (int i = 0; i < NACC; ++i) { mbar_init(&d_full[i], 1); mbar_init(&d_empty[i], 4 * L::WPQ); }
    for (int i = 0; i < L::E; ++i) { mbar_init(&e_full[i], 1); mbar_init(&e_empty[i], 4 * L::WPQ); }
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, 512);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();

  if (warp == 0 && page_skip) {
    // ------------------------------------------------------------------ TMA producer with the page skip
    // The whole warp walks the tiles: lane l holds heads l + 32 j (their |Qr|, z |Qc| and s*), the tile is skipped
    // when no head may fire on either of its two pages; lane 0 issues the copies.
    constexpr int NJ = NHG * MH / 32;
    float hq[NJ], hz[NJ], hs[NJ];
    bool ok = n > 0;
    int prev_b = -1, b = b_first, kt = kt_first;
    for (int i = 0; i < n && ok; ++i, kt = kt + 1 == tps ? (++b, 0) : kt + 1) {
      const int row0 = kt * TC_M;
      bool lok = true;
      if (b != prev_b) {
        if (lane == 0) {
          const int qi = (b - b_first) % L::QB, quse = (b - b_first) / L::QB;
          if (quse > 0 && !mbar_wait(&q_empty[qi], (quse - 1) & 1, &abort_flag)) {
            lok = false;
          } else {
            mbar_arrive_expect_tx(&q_full[qi], (uint32_t)H * L::QROW * L::QPARTS);
            for (int part = 0; part < L::QPARTS; ++part)
              tma_load_2d(sq + qi * L::qbuf + part * L::QPART, &qmap, 0, (b * L::QPARTS + part) * H, &q_full[qi]);
          }
        }
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
          const int hh = lane + 32 * j;
          hq[j] = hz[j] = 0.f;
          hs[j] = INFINITY;                              // a head past H never fires
          if (hh < H) {
            const int64_t bh = (int64_t)b * H + hh;
            hq[j] = args.qrf[bh];
            hz[j] = args.qcn[bh] * args.z;
            hs[j] = args.smax1[bh];
          }
        }
        prev_b = b;
      }
      const int64_t pg = (int64_t)b * args.n_pages + row0 / PAGE;
      const bool two = TC_M > PAGE && row0 + PAGE < args.n_rows;
      const float pk0 = args.page_knorm[pg], pe0 = args.page_eta[pg];
      const float pk1 = two ? args.page_knorm[pg + 1] : 0.f, pe1 = two ? args.page_eta[pg + 1] : 0.f;
      bool may = false;
#pragma unroll
      for (int j = 0; j < NJ; ++j)
        may = may || page_may_fire(args.lam, hq[j], hz[j], hs[j], pk0, pe0) ||
              (two && page_may_fire(args.lam, hq[j], hz[j], hs[j], pk1, pe1));
      const bool skip = !__any_sync(0xffffffffu, may);
      if (lane == 0 && lok) {
        const int s = i % TC_STAGES, use = i / TC_STAGES;
        if ((use > 0 && !mbar_wait(&a_empty[s], (use - 1) & 1, &abort_flag)) || abort_flag) {
          lok = false;
        } else {
          skip_stage[s] = skip ? 1 : 0;                  // published by the arrive below (release)
          if (skip) {
            mbar_arrive(&a_full[s]);
          } else {
            mbar_arrive_expect_tx(&a_full[s], TC_TILE_BYTES);
            tma_load_3d(sa + s * TC_TILE_BYTES, &kmap, 0, row0, b, &a_full[s]);
          }
          // the tile's eta rows (nothing to load for a skipped tile: its epilogue reads none)
          const int e = i % L::E, euse = i / L::E;
          if (euse > 0 && !mbar_wait(&e_empty[e], (euse - 1) & 1, &abort_flag)) {
            lok = false;
          } else if (eta_tma && !skip) {
            mbar_arrive_expect_tx(&e_full[e], (uint32_t)TC_M * 4u);
            tma_load_2d(eta_s + e * TC_M, &emap, row0, b, &e_full[e]);
          } else {
            mbar_arrive(&e_full[e]);
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, lok, 0);
    }
    if (n > 0 && !ok && lane == 0) abort_flag = 1;
  } else if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0 && n > 0) {
      int prev_b = -1, b = b_first, kt = kt_first;
      for (int i = 0; i < n; ++i, kt = kt + 1 == tps ? (++b, 0) : kt + 1) {
        const int row0 = kt * TC_M;
        if (b != prev_b) {
          const int qi = (b - b_first) % L::QB, quse = (b - b_first) / L::QB;
          if (quse > 0 && !mbar_wait(&q_empty[qi], (quse - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
          mbar_arrive_expect_tx(&q_full[qi], (uint32_t)H * (L::QROW * L::QPARTS + 4u * L::SK));
          for (int part = 0; part < L::QPARTS; ++part)
            tma_load_2d(sq + qi * L::qbuf + part * L::QPART, &qmap, 0, (b * L::QPARTS + part) * H, &q_full[qi]);
          if constexpr (L::SK > 0) {
            for (int part = 0; part < 2; ++part)
              tma_load_2d(sq + qi * L::qbuf + L::QPARTS * L::QPART + part * L::SQPART, &sqmap, 0, (b * 2 + part) * H,
                          &q_full[qi]);
          }
          prev_b = b;
        }
        const int s = i % TC_STAGES, use = i / TC_STAGES;
        if (use > 0 && !mbar_wait(&a_empty[s], (use - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
        if (abort_flag) break;
        mbar_arrive_expect_tx(&a_full[s], TC_TILE_BYTES);
        tma_load_3d(sa + s * TC_TILE_BYTES, &kmap, 0, row0, b, &a_full[s]);
        if constexpr (L::SK > 0) tma_load_3d(sa + s * TC_TILE_BYTES + L::KTILE, &smap, 0, row0, b, &a_full[s]);
        if constexpr (MODE == 2) {
          // the tile's eta rows, into a ring that the epilogue releases
          const int e = i % L::E, euse = i / L::E;
          if (euse > 0 && !mbar_wait(&e_empty[e], (euse - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
          if (eta_tma) {
            mbar_arrive_expect_tx(&e_full[e], (uint32_t)TC_M * 4u);
            tma_load_2d(eta_s + e * TC_M, &emap, row0, b, &e_full[e]);
          } else {
            mbar_arrive(&e_full[e]);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0 && n > 0) {
      constexpr uint32_t idesc = mma_idesc_bf16(MH, TC_M);
      int prev_b = -1, b = b_first, kt = kt_first;
      for (int i = 0; i < n; ++i, kt = kt + 1 == tps ? (++b, 0) : kt + 1) {
        const int qi = (b - b_first) % L::QB;
        if (b != prev_b) {
          if (!mbar_wait(&q_full[qi], ((b - b_first) / L::QB) & 1, &abort_flag)) { abort_flag = 1; break; }
          prev_b = b;
        }
        const int s = i % TC_STAGES, use = i / TC_STAGES;
        const int ds = i % NACC, duse = i / NACC;
        if (!mbar_wait(&a_full[s], use & 1, &abort_flag)) { abort_flag = 1; break; }
        if (duse > 0 && !mbar_wait(&d_empty[ds], (duse - 1) & 1, &abort_flag)) { abort_flag = 1; break; }
        tmem_fence_after();                              // the epilogue's reads of this accumulator came first
        const uint64_t bd = kmajor_desc<L::RW * 2>(smem_addr(sa + s * TC_TILE_BYTES));
        if (!(page_skip && skip_stage[s])) {             // a skipped tile: no product (the epilogue ignores it)
#pragma unroll
          for (int hg = 0; hg < NHG; ++hg)
#pragma unroll
            for (int part = 0; part < L::QPARTS; ++part) {
              const uint64_t ad =
                  kmajor_desc<L::QROW>(smem_addr(sq + qi * L::qbuf + part * L::QPART + hg * MH * L::QROW));
#pragma unroll
              for (int k = 0; k < L::KP / 16; ++k)
                mma_bf16(tmem_base + ds * DCOLS + hg * TC_M, ad + (uint64_t)((32 * k) >> 4),
                         bd + (uint64_t)(L::RW >= 16 ? (32 * k) >> 4 : 0), idesc, (part > 0 || k > 0) ? 1u : 0u);
            }
          if constexpr (L::SK > 0) {
            // + p_h . s_u: the sketch rows after the key tile, the query's high and low parts after its key parts
            const uint64_t sd = kmajor_desc<L::SK * 2>(smem_addr(sa + s * TC_TILE_BYTES + L::KTILE));
#pragma unroll
            for (int hg = 0; hg < NHG; ++hg)
#pragma unroll
              for (int part = 0; part < 2; ++part) {
                const uint64_t ad = kmajor_desc<L::SK * 2>(smem_addr(sq + qi * L::qbuf + L::QPARTS * L::QPART +
                                                                     part * L::SQPART + hg * MH * L::SK * 2));
#pragma unroll
                for (int k = 0; k < L::SK / 16; ++k)
                  mma_bf16(tmem_base + ds * DCOLS + hg * TC_M, ad + (uint64_t)((32 * k) >> 4),
                           sd + (uint64_t)((32 * k) >> 4), idesc, 1u);
              }
          }
        }
        mma_commit(&a_empty[s]);
        mma_commit(&d_full[ds]);
        const bool last_of_seq = (i + 1 == n) || kt + 1 == tps;
        if (last_of_seq) mma_commit(&q_empty[qi]);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int ew = warp - 2;                              // 0 .. EW-1
    const int g = ew / (4 * L::WPQ);                      // group: tiles i = g (mod G), accumulator i mod NACC
    const int sub = (ew % (4 * L::WPQ)) >> 2;             // which of the group's warps on this lane quarter
    const int quarter = warp & 3;                         // TMEM lane quarter this warp may read
    constexpr int NCT = L::NCT;                           // 32-row chunks per thread and tile: sub + WPQ j
    float* my_stg = stg + (ew * 32 + lane) * 32;          // this thread's staging row (128 B, 16-byte swizzled)
    int prev_b = -1;
    float th[NHG], p1[NHG], p2[NHG], p3[NHG];             // per head: theta, or (s*, |(O Qr)[r:]|, z |Qc|, |Qr|)
    int b = b_first, kt = kt_first + g;
    for (int i = g; i < n; i += G, kt += G) {
      while (kt >= tps) { kt -= tps; ++b; }
      const int row0 = kt * TC_M;
      if (b != prev_b) {
#pragma unroll
        for (int hg = 0; hg < NHG; ++hg) {
          const int hh = hg * 128 + (MH == 128 ? 32 * quarter + lane : 16 * quarter + (lane & 15));
          th[hg] = p1[hg] = p2[hg] = p3[hg] = 0.f;
          if (hh < H) {
            const int64_t bh = (int64_t)b * H + hh;
            if (MODE == 1) th[hg] = args.theta[bh];
            if (MODE == 2) {
              th[hg] = args.smax1[bh];
              p1[hg] = args.qrn[bh];
              p2[hg] = args.qcn[bh] * args.z;
              if (page_skip) p3[hg] = args.qrf[bh];
            }
          }
        }
        prev_b = b;
      }
      const int ds = i % NACC, duse = i / NACC;
      if (!mbar_wait(&d_full[ds], duse & 1, &abort_flag) ||
          (MODE == 2 && !mbar_wait(&e_full[i % L::E], (i / L::E) & 1, &abort_flag))) {
        if (lane == 0) { raise_status(args.status, VK_ERR_TIMEOUT); abort_flag = 1; }
        break;
      }
      // mode 2: the tile's eta rows in shared memory (zero past the last row), or in global memory
      const float* eta_tile = eta_tma ? eta_s + (i % L::E) * TC_M : nullptr;
      tmem_fence_after();
#pragma unroll
      for (int hg = 0; hg < NHG; ++hg) {
        const int hh = hg * 128 + (MH == 128 ? 32 * quarter + lane : 16 * quarter + (lane & 15));
        const bool valid = hh < H;
        const int64_t bh = (int64_t)b * H + hh;
        const uint32_t taddr = tmem_base + ((uint32_t)(32 * quarter) << 16) + ds * DCOLS + hg * TC_M;
        const bool emit = MODE == 1 || (MODE == 2 && args.top_j > 0);
        uint32_t msk[NCT];
        float keep[NCT == 1 ? 32 : 1];                    // one chunk per thread: its values, kept for the emission
        int cnt = 0;
#pragma unroll
        for (int j = 0; j < NCT; ++j) {
          const int c = sub + L::WPQ * j;
          float v[32];
          tmem_ld_chunk<MH>(taddr + (MH == 128 ? 32 * c : 64 * c), v);
          tmem_wait_ld();
          const int rc = row0 + (MH == 128 ? 32 * c : 64 * c + 32 * (lane >> 4));   // first row of the chunk
          uint32_t m = 0u;
          if (MODE == 0 && args.scores_bf16) {
            if (valid) {
              __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(args.scores) + bh * args.scores_ld + rc;
              if (rc + 32 <= args.n_rows && ((bh * args.scores_ld + rc) & 7) == 0) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  uint32_t w[4];
#pragma unroll
                  for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 pb = __floats2bfloat162_rn(v[8 * k + 2 * e], v[8 * k + 2 * e + 1]);
                    w[e] = *reinterpret_cast<const uint32_t*>(&pb);
                  }
                  reinterpret_cast<uint4*>(dst)[k] = make_uint4(w[0], w[1], w[2], w[3]);
                }
              } else {
#pragma unroll
                for (int k = 0; k < 32; ++k)
                  if (rc + k < args.n_rows) dst[k] = __float2bfloat16_rn(v[k]);
              }
            }
          } else if (MODE == 0) {
            if (valid) {
              float* dst = args.scores + bh * args.scores_ld + rc;
              if (rc + 32 <= args.n_rows && ((bh * args.scores_ld + rc) & 3) == 0) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                  reinterpret_cast<float4*>(dst)[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
              } else {
#pragma unroll
                for (int k = 0; k < 32; ++k)
                  if (rc + k < args.n_rows) dst[k] = v[k];
              }
            }
          } else if (MODE == 1) {
            // v >= theta exactly when v - theta' has a clear sign bit, theta' = theta with +0 taken as -0 (so that
            // v = -0 against theta = +0 gives +0, not -0): the sign bits are shifted in one instruction per row
            const float tq = th[hg] == 0.f ? -0.f : th[hg];
            uint32_t below = 0u;                         // bit 31 - k: row k is below theta
#pragma unroll
            for (int k = 0; k < 32; ++k) below = __funnelshift_l(__float_as_uint(v[k] - tq), below, 1);
            m = ~__brev(below);
            m &= range_mask(rc, args.arch_lo, min(args.arch_hi, args.n_rows));
            if (!valid) m = 0u;
          } else {
            const int64_t word = rc >> 5;
            const bool word_ok = valid && word < args.nw && rc < args.n_rows;
            // the page test is the producer's, per head: where it fails no row can fire (and a tile that every
            // head fails was skipped, its accumulator stale)
            const bool may = !page_skip || (rc < args.n_rows &&
                             page_may_fire(args.lam, p3[hg], p2[hg], th[hg],
                                           args.page_knorm[(int64_t)b * args.n_pages + rc / PAGE],
                                           args.page_eta[(int64_t)b * args.n_pages + rc / PAGE]));
            if (may) {
              const uint32_t sel = word_ok ? args.selbm[bh * args.nw + word] : 0xffffffffu;
              const float pr = rc < args.n_rows ? args.page_res[(int64_t)b * args.n_pages + rc / PAGE] : 0.f;
              const float add = p1[hg] * pr;
              if (eta_tile) {                          // staged in shared memory by the producer
                const float* etl = eta_tile + (rc - row0);
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                  const float T = args.lam * (v[k] + add + p2[hg] * etl[k]);
                  v[k] = T;
                  m |= (T > th[hg] ? 1u : 0u) << k;
                }
              } else {
                const float* eta = args.eta + (int64_t)b * args.N + rc;
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                  const float e = rc + k < args.n_rows ? eta[k] : 0.f;
                  const float T = args.lam * (v[k] + add + p2[hg] * e);
                  v[k] = T;
                  m |= (T > th[hg] ? 1u : 0u) << k;
                }
              }
              m &= range_mask(rc, args.arch_lo, min(args.arch_hi, args.n_rows)) & ~sel;
            }
            if (!word_ok) m = 0u;
            if (!emit && word_ok) args.firebm[bh * args.nw + word] = m;
          }
          msk[j] = m;
          cnt += __popc(m);
          if constexpr (NCT == 1) {
#pragma unroll
            for (int k = 0; k < 32; ++k) keep[k] = v[k];
          }
        }
        if (emit) {
          // reserve the head's room for this tile, then stage each chunk that has hits and visit only its set bits
          int pos = cnt ? atomicAdd(&args.cand_cnt[bh], cnt) : 0;
#pragma unroll
          for (int j = 0; j < NCT; ++j) {
            const int c = sub + L::WPQ * j;
            if (!__any_sync(0xffffffffu, msk[j] != 0u)) continue;
            float v[32];
            const int rc = row0 + (MH == 128 ? 32 * c : 64 * c + 32 * (lane >> 4));
            if constexpr (NCT == 1) {
#pragma unroll
              for (int k = 0; k < 32; ++k) v[k] = keep[k];
            } else {
              tmem_ld_chunk<MH>(taddr + (MH == 128 ? 32 * c : 64 * c), v);
              tmem_wait_ld();
            }
            if (MODE == 2 && NCT > 1) {
              const float pr = args.page_res[(int64_t)b * args.n_pages + rc / PAGE];
              const float add = p1[hg] * pr;
              const float* eta = args.eta + (int64_t)b * args.N + rc;
              if (eta_tile) {
#pragma unroll
                for (int k = 0; k < 32; ++k) v[k] = args.lam * (v[k] + add + p2[hg] * eta_tile[rc - row0 + k]);
              } else {
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                  const float e = rc + k < args.n_rows ? eta[k] : 0.f;
                  v[k] = args.lam * (v[k] + add + p2[hg] * e);
                }
              }
            }
            uint32_t m = msk[j];
            if (m) {
#pragma unroll
              for (int k = 0; k < 8; ++k)
                reinterpret_cast<float4*>(my_stg)[k ^ (lane & 7)] =
                    make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
              while (m) {
                const int k = __ffs(m) - 1;
                m &= m - 1;
                const float val = my_stg[(((k >> 2) ^ (lane & 7)) << 2) | (k & 3)];
                if (pos < args.capc) args.cand[bh * args.capc + pos] = make_int2(rc + k, __float_as_int(val));
                ++pos;
              }
            }
          }
        }
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&d_empty[ds]);
        if (MODE == 2) mbar_arrive(&e_empty[i % L::E]);
      }
    }
  }

  // wind down: every warp is done with tensor memory once all epilogue arrivals happened
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, 512);
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
  return v.dtype == VK_BF16 && (r == 8 || r == 16 || r == 32 || r == D_ROPE) && v.H % 16 == 0 && v.H >= 16 &&
         v.H <= 256 && (v.rope_ld * 2) % 16 == 0 && (v.rope_bstride * 2) % 16 == 0 && encode_fn() != nullptr;
}

// Configurations (MH, NHG, TM, G, WPQ): 128-row tiles and 4 / NHG epilogue groups of one warp per lane quarter.
// Measured slower for the candidate pass (sample, theta and candidates at B = 64, N = 65536, H = 64: 0.21 ms):
// 64-row tiles with six groups over eight accumulators (0.29 ms), and three groups of two warps per lane quarter,
// each thread one 32-row chunk kept in registers from the compare to the emission (0.23 ms).
static CUtensorMapSwizzle swizzle_for(int row_bytes) {
  return row_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
         : row_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
         : row_bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                           : CU_TENSOR_MAP_SWIZZLE_NONE;
}

template <int MH, int NHG, int MODE, int TM, int G, int WPQ, int RW, int SK = 0>
static cudaError_t launch_cfg(const vk_view& v, const void* keys, int64_t key_ld, int64_t key_bstride,
                              const void* qsrc, int row_stride, int n_rows, ScoreTcArgs args, cudaStream_t st) {
  using L = TcCfg<MH, NHG, TM, G, WPQ, RW, SK, MODE>;
  auto encode = encode_fn();
  CUtensorMap kmap, qmap, smap, sqmap, emap;
  cuuint64_t kdims[3] = {(cuuint64_t)RW, (cuuint64_t)n_rows, (cuuint64_t)v.B};
  cuuint64_t kstr[2] = {(cuuint64_t)(key_ld * row_stride * 2), (cuuint64_t)(key_bstride * 2)};
  cuuint32_t kbox[3] = {(cuuint32_t)RW, (cuuint32_t)TM, 1};
  cuuint32_t es3[3] = {1, 1, 1};
  // RoPE rows: one 128-byte segment per 1152-byte row, no L2 promotion, so DRAM reads only those bytes
  if (encode(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(keys), kdims, kstr, kbox, es3,
             CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(RW * 2),
             RW == 64 ? CU_TENSOR_MAP_L2_PROMOTION_NONE : CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  cuuint64_t qdims[2] = {(cuuint64_t)L::KP, (cuuint64_t)v.B * v.H * L::QPARTS};
  cuuint64_t qstr[1] = {(cuuint64_t)L::QROW};
  cuuint32_t qbox[2] = {(cuuint32_t)L::KP, (cuuint32_t)v.H};
  cuuint32_t es2[2] = {1, 1};
  if (encode(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(qsrc), qdims, qstr, qbox, es2,
             CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(L::QROW), CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  smap = kmap;
  sqmap = qmap;
  emap = kmap;
  args.eta_tma = 0;
  if constexpr (MODE == 2) {
    // eta [B][N] fp32 as a 2D map, TM-row boxes (zero past N); its row stride must be a multiple of 16 bytes
    if (row_stride == 1 && v.N % 4 == 0 && (reinterpret_cast<uintptr_t>(args.eta) & 15u) == 0) {
      cuuint64_t edims[2] = {(cuuint64_t)v.N, (cuuint64_t)v.B};
      cuuint64_t estr[1] = {(cuuint64_t)v.N * 4};
      cuuint32_t ebox[2] = {(cuuint32_t)TM, 1};
      cuuint32_t ees[2] = {1, 1};
      if (encode(&emap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(args.eta), edims, estr, ebox, ees,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
      args.eta_tma = 1;
    }
  }
  if constexpr (SK > 0) {
    // sketch rows [B][N][SK] (all N rows: the trigger scans with row stride 1) and the query parts [B][2][H][SK]
    if (row_stride != 1 || !args.sketch || !args.sketch_q) return cudaErrorInvalidValue;
    cuuint64_t sdims[3] = {(cuuint64_t)SK, (cuuint64_t)n_rows, (cuuint64_t)v.B};
    cuuint64_t sstr[2] = {(cuuint64_t)SK * 2, (cuuint64_t)v.N * SK * 2};
    cuuint32_t sbox[3] = {(cuuint32_t)SK, (cuuint32_t)TM, 1};
    if (encode(&smap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(args.sketch), sdims, sstr, sbox, es3,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(SK * 2), CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    cuuint64_t pdims[2] = {(cuuint64_t)SK, (cuuint64_t)v.B * 2 * v.H};
    cuuint64_t pstr[1] = {(cuuint64_t)SK * 2};
    cuuint32_t pbox[2] = {(cuuint32_t)SK, (cuuint32_t)v.H};
    if (encode(&sqmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(args.sketch_q), pdims, pstr, pbox, es2,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(SK * 2), CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  args.B = v.B;
  args.H = v.H;
  args.N = v.N;
  args.n_rows = n_rows;
  args.tiles_per_seq = (n_rows + TM - 1) / TM;
  args.total_tiles = (int64_t)args.tiles_per_seq * v.B;
  args.n_pages = (v.N + PAGE - 1) / PAGE;
  args.tmem_cols = 512;
  const int grid = (int)std::min<int64_t>(args.total_tiles, sm_count());   // persistent: one CTA per SM
  auto kernel = k_score_tc<MH, NHG, MODE, TM, G, WPQ, RW, SK>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L::total);
  if (e != cudaSuccess) return e;
  if (grid > 0) {
    kernel<<<grid, L::THREADS, L::total, st>>>(kmap, qmap, smap, sqmap, emap, args);
    count_launches(1);
  }
  return cudaGetLastError();
}

template <int MH, int NHG, int RW>
static cudaError_t launch_heads(const vk_view& v, const void* keys, int64_t key_ld, int64_t key_bstride,
                                const void* qsrc, int row_stride, int n_rows, const ScoreTcArgs& args,
                                cudaStream_t st) {
  constexpr int G4 = 4 / NHG;
  if (args.mode == 2 && args.r_sk > 0) {
    // with the sketch: two epilogue groups and one query buffer leave room for four or more stages of key + sketch
    if constexpr (NHG == 1 && RW == 64) {
      if (args.r_sk == 64)
        return launch_cfg<MH, 1, 2, 128, 2, 1, 64, 64>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
      if (args.r_sk == 32)
        return launch_cfg<MH, 1, 2, 128, 2, 1, 64, 32>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
      if (args.r_sk == 16)
        return launch_cfg<MH, 1, 2, 128, 2, 1, 64, 16>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
    }
    return cudaErrorInvalidValue;
  }
  if (args.mode == 0)
    return launch_cfg<MH, NHG, 0, 128, G4, 1, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
  if (args.mode == 2)
    return launch_cfg<MH, NHG, 2, 128, G4, 1, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
  return launch_cfg<MH, NHG, 1, 128, G4, 1, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
}

template <int RW>
static cudaError_t launch_width(const vk_view& v, const void* keys, int64_t key_ld, int64_t key_bstride,
                                const void* qsrc, int row_stride, int n_rows, const ScoreTcArgs& args,
                                cudaStream_t st) {
  if (v.H <= 64) return launch_heads<64, 1, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
  if (v.H <= 128) return launch_heads<128, 1, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
  return launch_heads<128, 2, RW>(v, keys, key_ld, key_bstride, qsrc, row_stride, n_rows, args, st);
}

cudaError_t launch_score_tc(const vk_view& v, int r, const void* digest, const void* qhl, int row_offset,
                            int row_stride, int n_rows, ScoreTcArgs args, cudaStream_t st) {
  if (!encode_fn()) return cudaErrorNotSupported;
  if (r == D_ROPE) {
    const auto* rope = static_cast<const __nv_bfloat16*>(v.rope) + (int64_t)row_offset * v.rope_ld;
    return launch_width<64>(v, rope, v.rope_ld, v.rope_bstride, v.q_rope, row_stride, n_rows, args, st);
  }
  const auto* dig = static_cast<const __nv_bfloat16*>(digest) + (int64_t)row_offset * r;
  const int64_t bs = (int64_t)v.N * r;
  if (r == 32) return launch_width<32>(v, dig, r, bs, qhl, row_stride, n_rows, args, st);
  if (r == 16) return launch_width<16>(v, dig, r, bs, qhl, row_stride, n_rows, args, st);
  if (r == 8) return launch_width<8>(v, dig, r, bs, qhl, row_stride, n_rows, args, st);
  return cudaErrorInvalidValue;
}

}  // namespace vk
