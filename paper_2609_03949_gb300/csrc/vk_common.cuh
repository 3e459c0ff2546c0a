// vk_common.cuh -- device helpers and launch declarations shared by the libvk.so translation units.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/vk.h"

namespace vk {

constexpr int D_LAT = 512;
constexpr int D_ROPE = 64;
constexpr int PAGE = 64;
constexpr int MAX_H = 256;           // heads per call supported by the kernels
constexpr int HG = 64;               // heads per attention CTA (one bit each in a 64-bit row mask)
constexpr int SPLIT_MAX = 4096;      // positions per attention split (bounds the CTA's union list)
constexpr int SMEM_OPTIN = 227 * 1024;  // opt-in shared memory per CTA on sm_103a (static + dynamic)
constexpr int SMEM_BUDGET = 220 * 1024; // what the host plans dynamic shared memory against

// ------------------------------------------------------------------------------------------ scalar helpers
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Order-preserving map float -> uint32 (a < b  <=>  key(a) < key(b)); -0 is folded onto +0 first.
__device__ __forceinline__ uint32_t fkey(float f) {
  if (f == 0.0f) f = 0.0f;
  uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float funkey(uint32_t k) {
  uint32_t b = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
  return __uint_as_float(b);
}

// First error wins; later ones are dropped until the host polls and clears the word.
__device__ __forceinline__ void raise_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// Block-wide exclusive scan of one int per thread (blockDim.x multiple of 32, <= 1024).
// `scratch` needs 33 ints. Returns the exclusive prefix; *total receives the block sum.
__device__ __forceinline__ int block_exclusive_scan(int v, int* scratch, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) scratch[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nwarps ? scratch[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nwarps) scratch[lane] = w;     // inclusive per-warp totals
    if (lane == 31) scratch[32] = w;
  }
  __syncthreads();
  int prefix = (warp ? scratch[warp - 1] : 0) + x - v;
  *total = scratch[32];
  __syncthreads();
  return prefix;
}

// ------------------------------------------------------------------------------------------ attention partials
// Where the attention writes its partial results (part_o [B][nslot][H][512], part_ml [B][nslot][H][2]). The work
// is made of B * n_hg segments (sequence, head group of 64), each of T = ceil(N / 64) row tiles.
//  * split layout (fp32 kernel, G = 0): every segment is cut into nsplit ranges of split_len positions, one CTA
//    each, and all nsplit slots of every segment are written;
//  * persistent layout (tensor-core kernel, G > 0): the B * T (sequence, row tile) positions, sequence-major, are
//    cut into P = G / n_hg equal contiguous ranges, and CTA p * n_hg + c takes head group c of range p. The n_hg
//    CTAs of a range walk the same rows in step, so the second head group's reads of a tile come from L2. A
//    segment (tiles t = s T .. s T + T - 1, s = b n_hg + hg) owns one slot per range its tiles fall in, numbered
//    from 0 by range, so segment s has attn_nvalid(s) written slots.
// nslot is the slot count of one tier (the largest attn_nvalid); the fired rows of the two-tier path use slots
// nslot .. 2 nslot - 1 the same way.
struct AttnGeom {
  int nslot;
  int nsplit, split_len;     // split layout
  int G, T, n_hg;            // persistent layout: G a multiple of n_hg
  long long total;           // B * n_hg * T
};
// The range of the persistent layout that holds tile t of segment t / T: ranges are [p npos / P, (p+1) npos / P)
// over the npos = B * T positions.
__host__ __device__ inline int attn_range_of(const AttnGeom& g, long long t) {
  const long long s = t / g.T, kt = t - s * g.T;
  const long long pos = (s / g.n_hg) * g.T + kt, npos = g.total / g.n_hg;
  return (int)(((pos + 1) * (long long)(g.G / g.n_hg) - 1) / npos);
}
// Written slots of segment s (per tier).
__host__ __device__ inline int attn_nvalid(const AttnGeom& g, long long s) {
  if (g.G == 0) return g.nslot;
  return attn_range_of(g, (s + 1) * g.T - 1) - attn_range_of(g, s * g.T) + 1;
}

}  // namespace vk

// ------------------------------------------------------------------------------------------ workspace
// Byte offsets of every scratch region inside the caller's workspace, for one set of shapes.
struct VkLayout {
  int64_t B, H, N, nw;          // nw = 32-bit words per head bitmap
  vk::AttnGeom ag;              // where the attention writes its partials
  int64_t n_hg;                 // head groups of 64
  bool dense_scores;            // materialised [B,H,N] scores are part of the layout
  bool two_tier;
  bool tc;                      // bf16, r = 64, H % 16 == 0: scoring on tcgen05
  bool fused;                   // threshold-candidate selection (no materialised scores)
  int64_t ss, soff, ns, sld, j; // fused: sample stride, offset, rows per sequence, row stride (ns rounded up to 8),
                                //        order statistic for theta
  int64_t capc;                 // fused: candidate capacity per head
  int64_t fcap;                 // two-tier top_j (fused path or page trigger): fired-candidate capacity per head
  size_t off_status, off_qt, off_qhl, off_qcn, off_qrn, off_qrf, off_smax1, off_nfired, off_scores, off_selbm, off_firebm,
      off_part_o, off_part_ml, off_sample, off_theta, off_ccnt, off_cand, off_fcnt, off_fcand, off_skp, off_skhl,
      off_rho, off_fmode, total;
  bool sketch;                  // row-level trigger with a content sketch (r_sk > 0)
};

// ------------------------------------------------------------------------------------------ launchers
// Every launcher enqueues on `st`, counts its kernel launches and returns cudaGetLastError().
namespace vk {
void count_launches(int n);
// qhl (may be NULL; r < 64): the rotated query's first r values as bf16 high and low parts, [B][2][H][max(r, 16)]
// with zeros past r, the query operand of the tensor-core digest scoring.
cudaError_t launch_qprep(const vk_view& v, int r, const float* rot, float* qt, float* qcn, float* qrn, float* qrf,
                         __nv_bfloat16* qhl, cudaStream_t st);
cudaError_t launch_score_simt(const vk_view& v, int r, const float* qt, const __nv_bfloat16* digest,
                              float* scores, cudaStream_t st);
cudaError_t launch_select_dense(int B, int H, int N, const float* scores, const int64_t* k_per_head,
                                int64_t k, int W, int n_sink, int32_t* idx, int32_t* count, int cap,
                                int append_from_count, float* kth, uint32_t* bitmap, int64_t nw, int* status,
                                cudaStream_t st);
cudaError_t launch_build_digest(const vk_view& v, int r, const float* rot, __nv_bfloat16* digest, float* eta,
                                float* page_res, float* page_knorm, float* page_eta, cudaStream_t st);
cudaError_t launch_trigger_page(int B, int H, int N, int W, int n_sink, float lam, float z_eff, const float* qcn,
                                const float* qrf, const float* page_knorm, const float* page_eta, const float* smax1,
                                const uint32_t* selbm, uint32_t* firebm, int64_t nw, int top_j, int* fcnt,
                                int2* fcand, int fcap, cudaStream_t st);
cudaError_t launch_list_to_bitmap(int B, int H, int N, const int32_t* idx, const int32_t* count, int cap,
                                  uint32_t* bitmap, int64_t nw, int* status, cudaStream_t st);
size_t attn_smem_bytes(int dtype, int H, int split_len);
bool attn_tc_supported(const vk_view& v);
// SMs of the current device (152 on GB300; also the value used when it cannot be read): the persistent kernels'
// CTA count, one per SM.
int sm_count();
AttnGeom attn_geom(const vk_view& v);
// part_arg (bf16 caches, may be NULL): also the row of every partial's max logit, [B][nslot][H] (the calibration's
// argmax over the attended rows).
cudaError_t launch_attn_tc(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, const AttnGeom& g,
                           int slot0, int nslot, float* part_o, float* part_ml, uint32_t flags, int* status,
                           cudaStream_t st, int* part_arg = nullptr, const int* skip = nullptr);
// skip (device, may be NULL): when *skip != 0 the launch does nothing (the fired rows' pass taken by k_attn_list)
cudaError_t launch_attn(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, const AttnGeom& g, int slot0,
                        int nslot, float* part_o, float* part_ml, uint32_t flags, int* status, cudaStream_t st,
                        const int* skip = nullptr);
cudaError_t launch_smax_reduce(int B, int H, const AttnGeom& g, int nslot, const float* part_ml, float* smax,
                               cudaStream_t st);
cudaError_t launch_combine(int B, int H, const AttnGeom& g, int nslot, const float* part_o, const float* part_ml,
                           float* out, float* lse, float* smax, cudaStream_t st, int nf = -1,
                           const int* mode = nullptr);
// The fired rows' attention (k_attn_list.cu): one partial per (b, h) over the rows its fired bitmap [B][H][nw] marks,
// into slot `slot` of the [B][nslot][H] partial layout; nothing when *mode == 0. launch_fired_mode sets mode[0] = 1 when
// every head fired at most `limit` rows (count[i] - n0), else 0.
cudaError_t launch_fired_mode(int64_t BH, const int32_t* count, int n0, int limit, int* mode, cudaStream_t st);
cudaError_t launch_attn_list(const vk_view& v, float lam, const uint32_t* bitmap, int64_t nw, int nslot, int slot,
                             float* part_o, float* part_ml, int* status, const int* mode, cudaStream_t st);
cudaError_t launch_trigger_dense(int B, int H, int N, int W, int n_sink, float lam, float z_eff, int top_j,
                                 float* scores, const float* qcn, const float* qrn, const float* eta,
                                 const float* page_res, const float* smax1, const uint32_t* selbm,
                                 uint32_t* firebm, int64_t nw, int64_t* nfired, cudaStream_t st, int r_sk = 0,
                                 const void* sketch = nullptr, const float* skp = nullptr);
// Content sketch (k_sketch.cu): the index entry of every row (sketch bf16 [B][N][r_sk], eta [B][N]), the query side
// (p fp32 [B][H][r_sk], its bf16 high/low parts [B][2][H][r_sk], rho [B][H]), and the basis from n queries.
cudaError_t launch_build_sketch(const vk_view& v, int r_sk, const float* basis, void* sketch, float* eta,
                                cudaStream_t st);
cudaError_t launch_sketch_query(const vk_view& v, int r_sk, const float* basis, float* p, void* phl, float* rho,
                                cudaStream_t st);
size_t sketch_basis_ws_bytes();
cudaError_t launch_sketch_basis(const void* queries, int dtype, int64_t n, int r_sk, float* basis, float* eig,
                                void* ws, cudaStream_t st);
// The 64 x 64 fp64 symmetric eigensolver of the PCA basis (k_pca.cu): eigenvectors as rows of vec (fp32), by
// decreasing eigenvalue.
cudaError_t launch_sym_eig64(const double* A, float* vec, float* eig, cudaStream_t st);
cudaError_t launch_theta(int B, int H, int ns, int ld, int off, int stride, int lo, int hi, int j, const void* sample,
                         float* theta, cudaStream_t st,
                         int* zero_cnt = nullptr);
cudaError_t launch_select_cand(int B, int H, int N, int lo, int hi, int64_t k, const int64_t* k_per_head,
                               const int* cand_cnt, const int2* cand, int capc, int force_fallback, const vk_view& v,
                               int r, const void* digest, const float* qt, int32_t* idx, int32_t* count, int cap,
                               int append, float* kth, uint32_t* bitmap, int64_t nw, int* status, cudaStream_t st);
struct ScoreTcArgs;
bool score_tc_supported(const vk_view& v, int r);
// r = 64 reads the RoPE columns and the RoPE query; r in {8, 16, 32} the [B, N, r] digest and the query prep's
// bf16 high and low parts qhl [B][2][H][max(r, 16)]. Rows row_offset + row_stride i, i < n_rows, of every sequence.
cudaError_t launch_score_tc(const vk_view& v, int r, const void* digest, const void* qhl, int row_offset,
                            int row_stride, int n_rows, ScoreTcArgs args, cudaStream_t st);
cudaError_t launch_bitmap_to_list(int B, int H, int N, const uint32_t* bitmap, int64_t nw, int32_t* idx,
                                  int32_t* count, int cap, int* status, cudaStream_t st);
// conformal calibration (k_calib.cu): per-query required inflations zq [B,H] from the all-rows argmax partials
// (slots slot0 ..), then z_out = {z, z_eff, n_hard}
size_t conformal_smem_bytes(int64_t BH);
cudaError_t launch_calib(const vk_view& v, int r, const AttnGeom& g, int slot0, int nslot, const float* part_ml,
                         const int* part_arg, const float* smax1, const uint32_t* selbm, int64_t nw, const float* qt,
                         const float* qcn, const float* qrn, const void* digest, const float* eta,
                         const float* page_res, float lam, double tau_s, int min_hard, float z_max, float* zq,
                         float* z_out, cudaStream_t st, int r_sk = 0, const float* skp = nullptr,
                         const void* sketch = nullptr, const float* rho = nullptr);
// PCA digest basis (k_pca.cu): workspace = status word + the fp64 second moment
size_t pca_workspace_bytes();
cudaError_t launch_pca_basis(const vk_view& v, float* rot, float* eig, void* ws, cudaStream_t st);
// sigma selector (k_sigma.cu): workspace = status word + the two bf16 copies of the low-pass basis
int sigma_basis_cols(int kappa);
size_t sigma_workspace_bytes(int T, int kappa);
cudaError_t launch_sigma(const vk_view& v, int T, int kappa, float* sigma, void* ws, cudaStream_t st);
}  // namespace vk
