// k_attn_tc.cu -- gather + absorbed-MLA attention for bf16 caches, both contractions on the tensor cores.
//
// Persistent: one CTA per SM. The work is B * n_hg segments (sequence b, group of <= 64 heads), each walked in tiles
// of 64 rows. The B * T (sequence, row tile) positions are cut into equal contiguous ranges, and each range goes to
// n_hg neighbouring CTAs, one per head group, so a CTA covers the end of one sequence, whole sequences and the
// start of another for its group. The CTAs of a range read the same tiles at the same pace, so with two or more
// head groups a tile comes from HBM about once and from L2 for the other groups. A tile that no head of the CTA's
// group selects is neither loaded nor computed. Per tile:
//   warp 0 (producer)  stages the heads' two 32-bit selection words of the tile, then TMA-loads its 64 rows x 576
//                      columns (128-byte swizzle, one 8 KB block per 64 columns) as five groups -- the RoPE block
//                      first, then four pairs of latent blocks, each as soon as the tile before it in that slot has
//                      released it -- into one of two tile slots; at a segment's first tile it loads the segment's
//                      queries once the previous segment's S products are done with the query buffer;
//   warps 1, 7 (S)     S = Q . X^T on tcgen05 (M = 64 heads, N = 64 rows, K = 576: 36 instructions) in two parts
//                      (24 + 12 instructions), each issued by its own thread, one burst per load group as the group
//                      lands, into their own accumulators (double-buffered); with M = 64 the logit of head 16 g + i
//                      and row j sits in TMEM lane 32 g + i, column j, and the softmax adds the two parts;
//   warp 6 (O^T)       once the softmax warps have written P^T, O^T += X_lat^T . P^T (M = 128 latent dims x 4
//                      blocks, N = 64 heads, K = 64 rows: 16 instructions) into the O^T accumulator, which stays in
//                      tensor memory for the whole segment. X_lat^T is read straight from the tile slot as an MN-major
//                      operand (the next 64 dims one 8 KB block away), so each latent row is staged in shared memory
//                      once and feeds both contractions. Two issuing threads, so neither contraction waits behind
//                      the other's issue;
//   warps 2..5, 8..11  softmax, two warps per TMEM lane quarter g (warp % 4); lanes i and 16 + i own head 16 g + i,
//                      and lane half t = 0, 1 reads rows 32 t .. 32 t + 31. Both warps of a quarter read all 64 of
//                      the head's logits, so each finds the same tile max without an exchange; warps 2..5 then
//                      write rows 32 t .. + 15, warps 8..11 rows 32 t + 16 .. + 31. They mask the logits with the
//                      head's selection words,
//                      and write P^T[h][row] = 2^(s lambda log2(e) - m_h)
//                      (0 where the head did not select the row) in bf16 into shared memory (K-major, 128-byte
//                      swizzle). m_h is a running max that only moves when a tile's max exceeds it by more than 32
//                      (log2 units), so P stays <= 2^32 and a rescale is rare: the O^T issuer sees it in the tile's
//                      published flags and has softmax warps 2..5 scale the head's O^T column in tensor memory
//                      (each its quarter of the dims) before the tile's product; there is no per-tile sync of the
//                      softmax warps otherwise. The exact max is tracked beside it, and at the end the head's sum
//                      and output are re-based on it, so the partial carries the true max logit. At a segment's end
//                      they write its partial and hand the O^T accumulator back to the O^T issuer.
// The partials (max, sum, out) of a segment, one per CTA it spans, are merged by the LSE combine (Lemma 1): with
// every CTA resident for the whole launch there is no tail of partly filled waves, and a long segment yields a
// few partials instead of one per fixed-length split. Rows inside a loaded tile that
// no head selected still enter the O^T product with weight 0, so every row in [0, N) must hold finite values.
// All waits are bounded: a wait that gives up raises VK_ERR_TIMEOUT and every role drains and leaves.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"

namespace vk {

constexpr int AT_T = 64;                               // rows per tile
constexpr int AT_SMX = 8;                              // softmax warps: two per TMEM lane quarter (rows 0..31, 32..63)
constexpr int AT_THREADS = (4 + AT_SMX) * 32;   // producer, S issuer, softmax x4, O^T issuer, S issuer, softmax x4
constexpr int AT_W_OT = 6, AT_W_SB = 7;               // the O^T issuer and the second S issuer
constexpr uint32_t AT_KBLK = 64 * 128;                 // one 64-column block of 64 rows (or 64 heads): 8 KB
constexpr uint32_t AT_TILE = 9 * AT_KBLK;              // 73,728: one tile slot, and the queries
constexpr int AT_NG = 5;                               // load groups per tile: latent pairs 0..3, RoPE block 4
constexpr float AT_TAU = 32.f;                         // log2 slack before a running max moves (P <= 2^32)
constexpr uint32_t AT_TMEM_COLS = 512;
constexpr uint32_t AT_S_COL = 0;                       // S (latent 0..383) buffers: columns 0..63, 64..127
constexpr uint32_t AT_SB_COL = 384;                    // S (latent 384..511 + RoPE) buffers: columns 384..447, 448..511
constexpr uint32_t AT_O_COL = 128;                     // O^T block j: columns 128 + 64 j .. + 63

// Shared memory, from a 1024-byte aligned base. Barriers: xfull/xrel [2 slots][5 groups], sfull/sfree [2],
// wfull/wfree [2], pfull [2], pfree [2], qfull, qfree, rdone, odec [2], ebar, odone, ofree, sdone [2]. P^T has no region of its
// own: a tile's P^T (64 heads x 64 rows, bf16, 8 KB) is written over its slot's RoPE block once S has read it.
struct AtSmem {
  static constexpr uint32_t q = 0;
  static constexpr uint32_t x = q + AT_TILE;
  static constexpr uint32_t p = x + 2 * AT_TILE;
  static constexpr uint32_t words = p;                 // [2][64 heads][2] u32
  static constexpr uint32_t uni = words + 2 * 64 * 2 * 4;
  static constexpr uint32_t fac = uni + 2 * 4;         // [2][64] f32
  static constexpr uint32_t anyw = fac + 2 * 64 * 4;   // [2][4] u32
  static constexpr uint32_t lpart = anyw + 2 * 4 * 4;  // [64] f32: the second row half's sum, at the end
  static constexpr uint32_t misc = lpart + 64 * 4;     // TMEM base, abort flag, rescale request (tile, count)
  static constexpr uint32_t bars = (misc + 16 + 7) & ~7u;
  static constexpr uint32_t nbars = 2 * AT_NG * 2 + 2 * 4 + 6 + 4 + 4;
  static constexpr uint32_t total = bars + nbars * 8;
};
static_assert(AtSmem::total + 1024 <= 232448, "attention shared memory exceeds the 227 KB opt-in limit");

struct AttnTcArgs {
  int H, N;
  AttnGeom g;            // persistent layout: G = gridDim.x ranges over total = B * n_hg * T tiles
  int slot0, nslot;
  int64_t nw;
  float lam_log2e;
  const uint32_t* bitmap;
  float* part_o;
  float* part_ml;
  int hold_first;        // VK_FLAG_TEST_TIMEOUT: CTA 0 withholds its first tile's loads
  int* status;
  int* part_arg;         // ARG instantiation: the row of each partial's max logit, [B][nslot][H]
  const int* skip;       // when non-NULL and *skip != 0 the launch does nothing (another kernel took this pass)
};

__device__ __forceinline__ void tma_load_3d_(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}
// Shared-memory matrix descriptor, 128-byte swizzle, 8-row groups 1024 B apart. `lbo` is the byte distance between
// 64-element atoms along M/N for an MN-major operand (unused by K-major ones).
__device__ __forceinline__ uint64_t sdesc_(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024u >> 4) << 32) | ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
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
__device__ __forceinline__ float tmem_ld1_(uint32_t taddr) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];\n" : "=r"(r) : "r"(taddr) : "memory");
  return __uint_as_float(r);
}
__device__ __forceinline__ void tmem_st1_(uint32_t taddr, float v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};\n" ::"r"(taddr), "r"(__float_as_uint(v)) : "memory");
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
// Generic-proxy shared-memory writes become visible to the tensor core (async proxy).
__device__ __forceinline__ void fence_async_smem_() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }
// Warp-uniform bounded wait: lane 0 polls, the warp takes its verdict.
__device__ __forceinline__ bool warp_wait_(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int lane) {
  bool w = true;
  if (lane == 0) w = mbar_wait(bar, parity, abort_flag);
  return __shfl_sync(0xffffffffu, w, 0);
}

// 32 columns of the M = 64 accumulator's 16 TMEM lanes: lanes 0..15 of the warp get columns col .. col + 31, lanes
// 16..31 columns col + 32 .. col + 63 of the same TMEM lanes (asynchronous until tmem_wait_ld).
__device__ __forceinline__ void tmem_ld32x2_(uint32_t taddr, float* v) {
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
// A rescale request of the O^T issuer (tile r: some head's running max moved there), served by one softmax warp
// (warp-collective): once O^T(r - 1) is complete, scale the warp's quarter of the dims (TMEM lanes lrow..) of every
// such head's O^T column by its factor in fac[r & 1], then report on rdone. Out of line: it is rare.
static __device__ __noinline__ bool attn_handle_request(volatile int* rq_tile, uint64_t* pfree, uint64_t* rdone,
                                                        const float* fac, uint32_t lrow, volatile int* abort_flag,
                                                        int lane) {
  int r = 0;
  if (lane == 0) {
    __threadfence_block();                             // the count was read first; the tile was written first
    r = *rq_tile;
  }
  r = __shfl_sync(0xffffffffu, r, 0);
  __syncwarp();
  __threadfence_block();                               // the factors were published before the request
  if (!warp_wait_(&pfree[(r - 1) & 1], ((r - 1) >> 1) & 1, abort_flag, lane)) return false;
  tmem_fence_after();
  const float* fr = fac + (r & 1) * 64;
  for (int h = 0; h < 64; ++h) {
    const float fh = fr[h];
    if (fh != 1.f) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t a = lrow + AT_O_COL + 64 * j + h;
        const float v = tmem_ld1_(a);
        tmem_wait_ld();
        tmem_st1_(a, v * fh);
      }
    }
  }
  tmem_wait_st();
  tmem_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(rdone);
  return true;
}

// Position of a CTA's tile: the row tile kt of sequence b; the head group hg is the CTA's own. Stepped without
// divisions (the per-tile bookkeeping sits on the issuing threads' critical path).
struct TilePos {
  int kt, hg, b;
  __device__ __forceinline__ void init(long long pos, int T, int group) {
    b = (int)(pos / T);
    kt = (int)(pos - (long long)b * T);
    hg = group;
  }
  __device__ __forceinline__ void next(int T) {
    if (++kt == T) {
      kt = 0;
      ++b;
    }
  }
};

// ARG (the calibration's instantiation) also tracks, per head, the row of the exact max logit (ties: the smaller
// row) and writes it beside each partial; the decode step's instantiation does not.
template <bool ARG>
__global__ void __launch_bounds__(AT_THREADS, 1) k_attn_tc(const __grid_constant__ CUtensorMap lmap,
                                                         const __grid_constant__ CUtensorMap rmap,
                                                         const __grid_constant__ CUtensorMap qlmap,
                                                         const __grid_constant__ CUtensorMap qrmap,
                                                         const AttnTcArgs args) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  if (args.skip && *args.skip) return;               // every thread reads the same word: the whole CTA leaves
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sq = smem + AtSmem::q;
  unsigned char* sx = smem + AtSmem::x;
  uint32_t* words = reinterpret_cast<uint32_t*>(smem + AtSmem::words);
  uint32_t* unis = reinterpret_cast<uint32_t*>(smem + AtSmem::uni);
  float* fac = reinterpret_cast<float*>(smem + AtSmem::fac);
  float* lparts = reinterpret_cast<float*>(smem + AtSmem::lpart);
  uint32_t* anyw = reinterpret_cast<uint32_t*>(smem + AtSmem::anyw);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + AtSmem::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + AtSmem::misc + 4);
  volatile int* rq_tile = reinterpret_cast<volatile int*>(smem + AtSmem::misc + 8);    // tile of the last request
  volatile int* rq_count = reinterpret_cast<volatile int*>(smem + AtSmem::misc + 12);  // requests made so far
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + AtSmem::bars);
  uint64_t* xfull = bars;                     // [2][5]
  uint64_t* xrel = bars + 2 * AT_NG;          // [2][5]
  uint64_t* sfull = bars + 4 * AT_NG;         // [2]
  uint64_t* sfree = sfull + 2;                // [2]
  uint64_t* wfull = sfree + 2;                // [2]
  uint64_t* wfree = wfull + 2;                // [2]
  // [2] a tile's P^T is written, by slot. One barrier per slot: the softmax warps do not wait for the O^T product
  // between tiles, so a single barrier could complete twice before the O^T issuer looked at it.
  uint64_t* pfull = wfree + 2;
  uint64_t* pfree = pfull + 2;                // [2] a tile's O^T product is complete, by tile parity
  uint64_t* qfull = pfree + 2;                // a segment's queries landed (one phase per segment)
  uint64_t* qfree = qfull + 1;                // both S issuers are done with the previous segment's queries
  uint64_t* rdone = qfree + 1;                // the softmax warps have applied a requested O^T rescale
  uint64_t* odec = rdone + 1;                 // [2] the O^T issuer has seen a tile's P^T (and asked for any rescale)
  uint64_t* ebar = odec + 2;                  // softmax-group syncs of a segment's epilogue (two per segment)
  uint64_t* odone = ebar + 1;                 // the segment's O^T products are complete (O^T issuer's commit)
  uint64_t* ofree = odone + 1;                // the softmax warps have read the segment's O^T out of tensor memory
  uint64_t* sdone = ofree + 1;                // [2] each S issuer's final commit

  const AttnGeom& geo = args.g;
  const int H = args.H, T = geo.T;
  // this CTA: head group `grp` of position range `rng` (the groups of one range are neighbouring CTAs)
  const int nranges = gridDim.x / geo.n_hg;
  const int rng = blockIdx.x / geo.n_hg, grp = blockIdx.x - rng * geo.n_hg;
  const long long npos = geo.total / geo.n_hg;
  const long long t0 = npos * rng / nranges, t1 = npos * (rng + 1) / nranges;
  const int ntile = (int)(t1 - t0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // a segment's first tile, or the first of this CTA's range, starts a new segment for every role
  TilePos tp;
  tp.init(t0, T, grp);

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    *rq_tile = -1;
    *rq_count = 0;
    for (int i = 0; i < 2 * AT_NG; ++i) { mbar_init(&xfull[i], 1); mbar_init(&xrel[i], 1); }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sfull[i], 2);                    // one commit from each S issuer
      mbar_init(&sfree[i], AT_SMX);
      mbar_init(&wfull[i], 1);
      mbar_init(&wfree[i], AT_SMX + 3);
      mbar_init(&sdone[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&pfull[i], AT_SMX);
      mbar_init(&pfree[i], 1);
    }
    mbar_init(qfull, 1);
    mbar_init(qfree, 2);
    mbar_init(rdone, 4);
    mbar_init(&odec[0], 1);
    mbar_init(&odec[1], 1);
    mbar_init(ebar, AT_SMX);
    mbar_init(odone, 1);
    mbar_init(ofree, AT_SMX);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, AT_TMEM_COLS);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    int last_use[2 * AT_NG];                           // last load issued per (slot, group), for the drain
#pragma unroll
    for (int i = 0; i < 2 * AT_NG; ++i) last_use[i] = -1;
    int nq = 0;                                        // query loads issued
    // selection words of tile i (at position fp): the lane holds heads lane and lane + 32, rows 0..31 and 32..63
    TilePos fp = tp;
    auto fetch = [&](int i, uint4& w) {
      w = make_uint4(0u, 0u, 0u, 0u);
      if (i >= ntile) return;
      const int b = fp.b, h0 = fp.hg * 64, nh = min(64, H - h0);
      const int pos0 = fp.kt * AT_T;
      const int64_t wi = pos0 >> 5;
      const int left = args.N - pos0;                  // >= 1
      const uint32_t m0 = left >= 32 ? 0xffffffffu : ((1u << left) - 1u);
      const uint32_t m1 = left >= 64 ? 0xffffffffu : (left <= 32 ? 0u : ((1u << (left - 32)) - 1u));
      const uint32_t* bm = args.bitmap + ((int64_t)b * H + h0) * args.nw;
      if (lane < nh) {
        const uint32_t* r = bm + (int64_t)lane * args.nw + wi;
        w.x = r[0] & m0;
        if (m1) w.y = r[1] & m1;
      }
      if (lane + 32 < nh) {
        const uint32_t* r = bm + (int64_t)(lane + 32) * args.nw + wi;
        w.z = r[0] & m0;
        if (m1) w.w = r[1] & m1;
      }
    };
    uint4 cur, nxt;
    fetch(0, cur);
    fp.next(T);
    int u = 0;                                         // tiles loaded so far
    bool ok = true;
    for (int i = 0; i < ntile; ++i, tp.next(T)) {
      fetch(i + 1, nxt);
      fp.next(T);
      const int ws = i & 1;
      if (i >= 2 && !warp_wait_(&wfree[ws], ((i >> 1) - 1) & 1, abort_flag, lane)) { ok = false; break; }
      uint32_t* wd = words + ws * 128;
      wd[lane * 2] = cur.x;
      wd[lane * 2 + 1] = cur.y;
      wd[(lane + 32) * 2] = cur.z;
      wd[(lane + 32) * 2 + 1] = cur.w;
      const uint32_t uni = __reduce_or_sync(0xffffffffu, cur.x | cur.y | cur.z | cur.w);
      if (lane == 0) unis[ws] = uni;
      __syncwarp();
      if (lane == 0) mbar_arrive(&wfull[ws]);
      const int b = tp.b, h0 = tp.hg * 64;
      bool lok = true;
      if (uni && args.hold_first && i == 0 && blockIdx.x == 0) {
        ++u;                                           // test hook: these loads are never issued
      } else if (uni) {
        const int s = u & 1, use = u >> 1;
        const int pos0 = tp.kt * AT_T;
        unsigned char* xs = sx + s * AT_TILE;
        if (lane == 0) {
          for (int g = 0; g < AT_NG; ++g) {
            const int grp = g;                         // latent pairs 0..3 in release order, then the RoPE block
            uint64_t* fb = &xfull[s * AT_NG + grp];
            if (use > 0 && !mbar_wait(&xrel[s * AT_NG + grp], (use - 1) & 1, abort_flag)) { lok = false; break; }
            if (grp == 4) {
              mbar_arrive_expect_tx(fb, AT_KBLK);
              tma_load_3d_(xs + 8 * AT_KBLK, &rmap, 0, pos0, b, fb);
            } else {
              mbar_arrive_expect_tx(fb, 2 * AT_KBLK);
              tma_load_3d_(xs + (2 * grp) * AT_KBLK, &lmap, 128 * grp, pos0, b, fb);
              tma_load_3d_(xs + (2 * grp + 1) * AT_KBLK, &lmap, 128 * grp + 64, pos0, b, fb);
            }
            last_use[s * AT_NG + grp] = use;
          }
        }
        ++u;
      }
      if ((i == 0 || tp.kt == 0) && lane == 0 && lok) {
        // the segment's queries, once both S issuers are done with the previous segment's
        if (nq > 0 && !mbar_wait(qfree, (nq - 1) & 1, abort_flag)) {
          lok = false;
        } else {
          const int qrow = b * H + h0;   // rows past the group's heads belong to other heads (or are zero-filled)
          mbar_arrive_expect_tx(qfull, AT_TILE);
          for (int k = 0; k < 8; ++k) tma_load_3d_(sq + k * AT_KBLK, &qlmap, 64 * k, qrow, 0, qfull);
          tma_load_3d_(sq + 8 * AT_KBLK, &qrmap, 0, qrow, 0, qfull);
          ++nq;
        }
      }
      if (!__shfl_sync(0xffffffffu, lok, 0)) { ok = false; break; }
      cur = nxt;
    }
    if (!ok && lane == 0) { raise_status(args.status, VK_ERR_TIMEOUT); *abort_flag = 1; }
    // drain: every load issued must have landed before the CTA leaves (only matters after an abort; a query load
    // is issued only after the previous one was consumed, so the last is the only one that can be in flight)
    if (lane == 0) {
      if (nq > 0) mbar_wait(qfull, (nq - 1) & 1, nullptr);
      for (int i = 0; i < 2 * AT_NG; ++i)
        if (last_use[i] >= 0) mbar_wait(&xfull[i], last_use[i] & 1, nullptr);
    }
  } else if (warp == 1 || warp == AT_W_SB) {
    // ------------------------------------------------------------------ S issuers
    // Two threads issue the two parts of the K = 576 contraction into their own accumulators (the softmax adds
    // them): warp 1 latent dims 0..383 (24 instructions), warp 7 latent dims 384..511 and the RoPE block (12). The
    // groups land in the order the previous tile's O^T product releases them: latent pairs 0..3, then the RoPE
    // block, which holds that tile's P^T until its O^T is done. Each thread issues a group's instructions as soon
    // as that group has landed, so after the last group lands only its four instructions remain.
    const int half = warp == 1 ? 0 : 1;
    if (lane == 0 && ntile > 0) {
      // S: M = 64 heads, N = 64 rows, A = Q and B = X, both K-major
      const uint32_t idesc_s =
          (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(AT_T >> 3) << 17) | ((uint32_t)(64 >> 4) << 24);
      const uint64_t qd = sdesc_(smem_addr(sq), 16);
      uint64_t* done_bar = &sdone[half];
      bool ok = true;
      int u = 0, nq = 0;
      for (int i = 0; i < ntile; ++i, tp.next(T)) {
        if (!mbar_wait(&wfull[i & 1], (i >> 1) & 1, abort_flag)) { ok = false; break; }
        const uint32_t uni = unis[i & 1];
        mbar_arrive(&wfree[i & 1]);
        if (i == 0 || tp.kt == 0) {
          if (nq > 0) mma_commit_(qfree);            // every S of the previous segment issued: its queries may go
          if (!mbar_wait(qfull, nq & 1, abort_flag)) { ok = false; break; }
          ++nq;
        }
        if (!uni) continue;
        const int s = u & 1, use = u >> 1;
        if (use > 0 && !mbar_wait(&sfree[s], (use - 1) & 1, abort_flag)) { ok = false; break; }
        const uint64_t xd = sdesc_(smem_addr(sx + s * AT_TILE), 16);
        // one branch-free burst per load group: control flow between tcgen05.mma issues costs the issuing thread far
        // more than the instructions themselves, so the only test between bursts is the next group's wait
        if (half == 0) {
          const uint32_t d = tmem + AT_S_COL + 64 * s;
#pragma unroll
          for (int g = 0; g < 3; ++g) {
            if (!mbar_wait(&xfull[s * AT_NG + g], use & 1, abort_flag)) { ok = false; break; }
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
              const int j = 8 * g + jj;
              const uint64_t off = (uint64_t)(((j >> 2) * AT_KBLK + 32 * (j & 3)) >> 4);
              mma_bf16_(d, qd + off, xd + off, idesc_s, j > 0 ? 1u : 0u);
            }
          }
          if (!ok) break;
          mma_commit_(&sfull[s]);
        } else {
          const uint32_t d = tmem + AT_SB_COL + 64 * s;
#pragma unroll
          for (int g = 3; g < 5; ++g) {
            if (!mbar_wait(&xfull[s * AT_NG + g], use & 1, abort_flag)) { ok = false; break; }
            if (g < 4) {
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) {
                const int j = 8 * (g - 3) + jj;
                const uint64_t off = (uint64_t)(((6 + (j >> 2)) * AT_KBLK + 32 * (j & 3)) >> 4);
                mma_bf16_(d, qd + off, xd + off, idesc_s, j > 0 ? 1u : 0u);
              }
            } else {
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const uint64_t off = (uint64_t)((8 * AT_KBLK + 32 * j) >> 4);
                mma_bf16_(d, qd + off, xd + off, idesc_s, 1u);
              }
            }
          }
          if (!ok) break;
          mma_commit_(&sfull[s]);
        }
        ++u;
      }
      mma_commit_(done_bar);
      if (!ok) { raise_status(args.status, VK_ERR_TIMEOUT); *abort_flag = 1; }
      mbar_wait(done_bar, 0, nullptr);                 // nothing this thread issued may outlive the CTA
    }
  } else if (warp == AT_W_OT) {
    // ------------------------------------------------------------------ O^T issuer
    // Issues each loaded tile's O^T += X_lat^T . P^T as soon as its P^T is written; its commits release the tile's
    // latent blocks for the next load into the slot. (A commit tracks this thread's own MMAs; the tile's S, issued
    // by the other thread, completed before its softmax could start.) At a segment boundary it commits odone (the
    // epilogue may read O^T) and waits for ofree before the next segment's first product overwrites it.
    if (lane == 0 && ntile > 0) {
      // O^T: M = 128 dims, N = 64 heads, A = X_lat^T MN-major (bit 15), B = P^T K-major
      const uint32_t idesc_o =
          (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | ((uint32_t)(64 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
      bool ok = true;
      int u = 0, useg = 0, nseg = 0, ncommit = 0, nreq = 0;
      for (int i = 0; i < ntile; ++i, tp.next(T)) {
        if (!mbar_wait(&wfull[i & 1], (i >> 1) & 1, abort_flag)) { ok = false; break; }
        const uint32_t uni = unis[i & 1];
        mbar_arrive(&wfree[i & 1]);
        if (i == 0 || tp.kt == 0) {
          if (nseg > 0) {
            mma_commit_(odone);
            ++ncommit;
            if (!mbar_wait(ofree, (nseg - 1) & 1, abort_flag)) { ok = false; break; }
            tmem_fence_after();                        // the epilogue's reads of O^T came first
          }
          ++nseg;
          useg = 0;
        }
        if (!uni) continue;
        const int s = u & 1;
        if (!mbar_wait(&pfull[s], (u >> 1) & 1, abort_flag)) { ok = false; break; }
        if (anyw[s * 4] | anyw[s * 4 + 1] | anyw[s * 4 + 2] | anyw[s * 4 + 3]) {
          // a head's running max moved on this tile: the softmax warps rescale its O^T column (each its quarter of
          // the dims) before this tile's product is added; they look for the request when they see odec
          *rq_tile = u;
          __threadfence_block();
          *rq_count = ++nreq;
          mbar_arrive(&odec[s]);
          if (!mbar_wait(rdone, (nreq - 1) & 1, abort_flag)) { ok = false; break; }
        } else {
          mbar_arrive(&odec[s]);
        }
        tmem_fence_after();                            // P^T and any O^T rescale come from the softmax warps
        const uint64_t xd = sdesc_(smem_addr(sx + s * AT_TILE), AT_KBLK);
        const uint64_t pd = sdesc_(smem_addr(sx + s * AT_TILE + 8 * AT_KBLK), 16);   // this tile's P^T
#pragma unroll
        for (int j = 0; j < 4; ++j) {
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            mma_bf16_(tmem + AT_O_COL + 64 * j, xd + (uint64_t)((2 * j * AT_KBLK + ks * 2048) >> 4),
                      pd + (uint64_t)(ks * 2), idesc_o, (useg > 0 || ks > 0) ? 1u : 0u);
          mma_commit_(&xrel[s * AT_NG + j]);           // latent blocks 2j, 2j+1 of this slot are free again
        }
        mma_commit_(&xrel[s * AT_NG + 4]);             // P^T read: the RoPE block may be reloaded
        mma_commit_(&pfree[u & 1]);                    // O^T up to date through this tile
        ++u;
        ++useg;
      }
      if (nseg > 0) {
        mma_commit_(odone);                            // the last segment's O^T is complete
        ++ncommit;
      }
      if (!ok) { raise_status(args.status, VK_ERR_TIMEOUT); *abort_flag = 1; }
      if (ncommit > 0) mbar_wait(odone, (ncommit - 1) & 1, nullptr);
    }
  } else {
    // ------------------------------------------------------------------ softmax
    // Two warps per TMEM lane quarter. Head hl = 16 q + (lane % 16); one tcgen05.ld 16x32bx2 per S part gives lanes
    // 0..15 the head's rows 0..31 and lanes 16..31 its rows 32..63, so both warps of a quarter see the whole tile and
    // take its max alone. Of its 32 rows a lane writes P for 16: rows 32 hh + 16 rh .. + 15 (rh = 0 for warps 2..5,
    // 1 for warps 8..11). The rh = 0 warps publish the rescale factors and serve rescales.
    const int q = warp & 3;                            // TMEM lane quarter of this warp
    const int rh = warp >= 8 ? 1 : 0;                  // which 16 of the lane's 32 rows this warp writes
    const int hh = lane >> 4;                          // which 32 rows of the tile the lane reads
    const int hl = 16 * q + (lane & 15);               // this lane's head
    const bool own = hh == 0;                          // the lane that publishes per-head values
    const float L = args.lam_log2e;
    const uint32_t lrow = tmem + ((uint32_t)(32 * q) << 16);
    float m = -INFINITY, mex = -INFINITY, lsum = 0.f;  // lsum: this warp's share of the head's sum
    int mpos = 0;                                      // ARG: the row of mex
    int u = 0, useg = 0, nseg = 0;
    int sb = 0, shg = 0;                               // the current segment's sequence and head group
    int handled = 0;                                   // rescale requests applied by this warp
    bool ok = true;
    // Before a wait that may depend on O^T(t) -- S(t + 2) reuses its slot, the epilogue needs it done -- take the
    // O^T issuer's decision on tile t (odec) and serve its rescale request if it made one. Cheap when there is none
    // (the usual case: a head's running max moves only by more than AT_TAU).
    auto check = [&](int t) -> bool {
      if (rh) return true;                             // the rh = 0 warps serve requests
      if (!warp_wait_(&odec[t & 1], (t >> 1) & 1, abort_flag, lane)) return false;
      int pend = 0;
      if (lane == 0) pend = *rq_count != handled;
      if (__shfl_sync(0xffffffffu, pend, 0)) {
        if (!attn_handle_request(rq_tile, pfree, rdone, fac, lrow, abort_flag, lane)) return false;
        ++handled;
      }
      return true;
    };
    // A segment's partial: re-base each head on its exact max, write (max, sum) and the output (unnormalised),
    // then release the O^T accumulator. The re-basing factors go through the parity buffer the last tile did not
    // use; a second group sync keeps the next tile from overwriting them while a warp still reads.
    auto epilogue = [&]() -> bool {
      if ((u >= 2 && !check(u - 2)) || (u >= 1 && !check(u - 1))) return false;
      if (!warp_wait_(odone, (nseg - 1) & 1, abort_flag, lane)) return false;   // the segment's O^T is complete
      float lt = lsum + __shfl_xor_sync(0xffffffffu, lsum, 16);                // this warp's 32 rows
      float ff = 1.f;
      if (mex != -INFINITY && m != mex) ff = ex2(m - mex);
      float* facf = fac + (u & 1) * 64;
      if (own && rh == 0) facf[hl] = ff;
      if (own && rh == 1) lparts[hl] = lt;
      __syncwarp();
      if (lane == 0) mbar_arrive(ebar);
      if (!warp_wait_(ebar, 0, abort_flag, lane)) return false;
      lt = (lt + lparts[hl]) * ff;                                               // both warps' rows (rh = 0 uses it)
      tmem_fence_after();
      const int h0 = shg * 64, nh = min(64, H - h0);
      const int slot = rng - attn_range_of(geo, ((long long)sb * geo.n_hg + shg) * T);
      const int64_t hbase = ((int64_t)sb * args.nslot + args.slot0 + slot) * H + h0;
      constexpr float LN2 = 0.6931471805599453f;
      if (own && rh == 0 && hl < nh) {
        args.part_ml[(hbase + hl) * 2] = mex * LN2;
        args.part_ml[(hbase + hl) * 2 + 1] = lt;
        if constexpr (ARG) args.part_arg[hbase + hl] = mpos;
      }
      // O^T block j on this warp's lanes: dims 128 j + 32 q + lane; columns: heads (blocks 2 rh, 2 rh + 1)
#pragma unroll 1
      for (int j = 2 * rh; j < 2 * rh + 2; ++j) {
        const int dim = 128 * j + 32 * q + lane;
#pragma unroll 1
        for (int c = 0; c < 64; c += 32) {
          float v[32];
          if (useg > 0) {
            tmem_ld32_(lrow + AT_O_COL + 64 * j + c, v);
            tmem_wait_ld();
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = 0.f;
          }
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (c + i < nh) args.part_o[(hbase + c + i) * D_LAT + dim] = v[i] * facf[c + i];
        }
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) { mbar_arrive(ofree); mbar_arrive(ebar); }
      return warp_wait_(ebar, 1, abort_flag, lane);
    };
    // one pass past the last tile closes the last segment: the epilogue has a single (inlined) call site, which
    // keeps the loop's code small (instruction fetch is shared with the issuing warps' loops)
    for (int i = 0; i <= ntile; ++i, tp.next(T)) {
      const int ws = i & 1;
      uint32_t uni = 0u, w = 0u;
      const bool fresh = i == ntile || i == 0 || tp.kt == 0;
      if (i < ntile) {
        if (!warp_wait_(&wfull[ws], (i >> 1) & 1, abort_flag, lane)) { ok = false; break; }
        uni = unis[ws];
        w = words[ws * 128 + hl * 2 + hh];            // rows 32 hh .. 32 hh + 31 of the head
        __syncwarp();
        if (lane == 0) mbar_arrive(&wfree[ws]);
      }
      if (fresh) {
        if (nseg > 0 && !epilogue()) { ok = false; break; }
        if (i == ntile) break;
        ++nseg;
        sb = tp.b;
        shg = tp.hg;
        useg = 0;
        m = mex = -INFINITY;
        mpos = 0;
        lsum = 0.f;
      }
      if (!uni) continue;
      const int s = u & 1, use = u >> 1, par = u & 1;
      if (u >= 2 && !check(u - 2)) { ok = false; break; }
      if (!warp_wait_(&sfull[s], use & 1, abort_flag, lane)) { ok = false; break; }
      tmem_fence_after();
      // this warp's 16 rows per lane (sv) and the other row half's (ov), both S parts added: each warp of a quarter
      // takes the whole tile's max itself, so both reach the same running max without an exchange
      float sv[32];
      {
        float sb[32];
        const uint32_t c0 = lrow + 64 * s;
        tmem_ld32x2_(c0 + AT_S_COL, sv);
        tmem_ld32x2_(c0 + AT_SB_COL, sb);
        tmem_wait_ld();
#pragma unroll
        for (int c = 0; c < 32; ++c) sv[c] += sb[c];
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfree[s]);
      float mr;
      int rpos = 0;                                    // ARG: the tile row of mr
      if constexpr (ARG) {
        float best = -INFINITY;
        int bp = 0;
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (((w >> c) & 1u) && sv[c] > best) { best = sv[c]; bp = 32 * hh + c; }
        const float ob = __shfl_xor_sync(0xffffffffu, best, 16);
        const int op = __shfl_xor_sync(0xffffffffu, bp, 16);
        // the lower row half wins ties: its rows come first
        const bool mine = hh == 0 ? best >= ob : best > ob;
        mr = mine ? best : ob;
        rpos = mine ? bp : op;
      } else {
        float mr0 = -INFINITY, mr1 = -INFINITY;
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
          if ((w >> c) & 1u) mr0 = fmaxf(mr0, sv[c]);
          if ((w >> (c + 1)) & 1u) mr1 = fmaxf(mr1, sv[c + 1]);
        }
        mr = fmaxf(mr0, mr1);
        mr = fmaxf(mr, __shfl_xor_sync(0xffffffffu, mr, 16));
      }
      // this warp's P rows: 32 hh + 16 rh .. + 15
      const uint32_t w16 = (w >> (16 * rh)) & 0xffffu;
      float pv[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) pv[c] = rh ? sv[16 + c] : sv[c];
      const float mt = mr * L;
      if constexpr (ARG) {
        if (mt > mex) { mex = mt; mpos = tp.kt * AT_T + rpos; }   // an earlier tile keeps a tie
      } else {
        mex = fmaxf(mex, mt);
      }
      float f = 1.f;
      if (mt > m + AT_TAU) {                           // includes the head's first selected row (m = -inf)
        if (m != -INFINITY) f = ex2(m - mt);
        m = mt;
        lsum *= f;
      }
      uint32_t pk[8];
      float ls0 = 0.f, ls1 = 0.f;
#pragma unroll
      for (int c = 0; c < 16; c += 2) {
        const float e0 = ((w16 >> c) & 1u) ? ex2(fmaf(pv[c], L, -m)) : 0.f;
        const float e1 = ((w16 >> (c + 1)) & 1u) ? ex2(fmaf(pv[c + 1], L, -m)) : 0.f;
        const __nv_bfloat162 pb = __floats2bfloat162_rn(e0, e1);
        ls0 += e0;
        ls1 += e1;
        pk[c >> 1] = *reinterpret_cast<const uint32_t*>(&pb);
      }
      lsum += ls0 + ls1;
      // publish this group's rescale factors (by tile parity; both warps of the quarter hold the same ones, rh = 0 publishes);
      // the O^T issuer reads them after pfull and, when a head needs one, has the rh = 0 softmax warps apply them
      // (handle_request) before this tile's product
      if (rh == 0) {
        const uint32_t need = __ballot_sync(0xffffffffu, own && f != 1.f);
        if (own) fac[par * 64 + hl] = f;
        if (lane == 0) anyw[par * 4 + q] = need;
      }
      {
        // P^T row hl, rows 32 hh + 16 rh .. + 15 of the tile: two 16-byte chunks, 128-byte swizzle, over the slot's
        // RoPE block (S has read it: sfull)
        unsigned char* row = sx + s * AT_TILE + 8 * AT_KBLK + hl * 128;
#pragma unroll
        for (int i = 0; i < 2; ++i)
          *reinterpret_cast<uint4*>(row + (((4 * hh + 2 * rh + i) ^ (hl & 7)) * 16)) =
              make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
      }
      fence_async_smem_();
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[s]);
      ++u;
      ++useg;
    }
    if (!ok && lane == 0) {
      raise_status(args.status, VK_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  }
  // every role has finished its waits and its tensor-memory accesses: release tensor memory
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    tmem_dealloc(tmem, AT_TMEM_COLS);
  }
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

cudaError_t launch_attn_tc(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, const AttnGeom& g,
                           int slot0, int nslot, float* part_o, float* part_ml, uint32_t flags, int* status,
                           cudaStream_t st, int* part_arg, const int* skip) {
  if (!encode2()) return cudaErrorNotSupported;
  if (g.G < 1 || g.G > g.total || g.G % g.n_hg != 0 || g.T != (v.N + AT_T - 1) / AT_T ||
      g.n_hg != (v.H + 63) / 64 || g.total != (long long)v.B * g.n_hg * g.T)
    return cudaErrorInvalidValue;
  CUtensorMap lmap, rmap, qlmap, qrmap;
  // cache rows: latent [B][N][512] and RoPE [B][N][64]; queries: [B*H][512] and [B*H][64]; 64-row boxes
  if (!make_map3(&lmap, v.latent, D_LAT, v.N, v.B, v.latent_ld, v.latent_bstride, AT_T) ||
      !make_map3(&rmap, v.rope, D_ROPE, v.N, v.B, v.rope_ld, v.rope_bstride, AT_T) ||
      !make_map3(&qlmap, v.q_latent, D_LAT, (uint64_t)v.B * v.H, 1, D_LAT, (int64_t)v.B * v.H * D_LAT, 64) ||
      !make_map3(&qrmap, v.q_rope, D_ROPE, (uint64_t)v.B * v.H, 1, D_ROPE, (int64_t)v.B * v.H * D_ROPE, 64))
    return cudaErrorInvalidValue;
  AttnTcArgs a{};
  a.H = v.H;
  a.N = v.N;
  a.g = g;
  a.slot0 = slot0;
  a.nslot = nslot;
  a.nw = nw;
  a.lam_log2e = lam * 1.4426950408889634f;
  a.bitmap = bitmap;
  a.part_o = part_o;
  a.part_ml = part_ml;
  a.hold_first = (flags & VK_FLAG_TEST_TIMEOUT) ? 1 : 0;
  a.status = status;
  a.part_arg = part_arg;
  a.skip = skip;
  const size_t smem = AtSmem::total + 1024;
  auto kernel = part_arg ? k_attn_tc<true> : k_attn_tc<false>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kernel<<<g.G, AT_THREADS, smem, st>>>(lmap, rmap, qlmap, qrmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
