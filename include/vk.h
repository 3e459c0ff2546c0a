/*
 * vk.h -- C ABI of libvk.so: the decode hot path of VestigeKV (arXiv 2609.03949) on one GB300 (sm_103a).
 *
 * One decode step of one attention layer over B independent sequences, each with an MLA cache of N rows.
 * Row u of sequence b is C_u = [L_u ; K_u]: the 512-wide compressed latent and the 64-wide decoupled RoPE key,
 * stored already rotated at position u (Sec. 3, Eq. 1). The query of head h is absorbed: Qc_h (512 wide, the
 * latent-side query W_UK^T q^c) and Qr_h (64 wide, rotated at position N). The step is
 *
 *   score   a[h,u] = Qr_h . K_u, or (O Qr_h)[0:r] . D_u on a width-r rotated digest D_u
 *           (Eq. 4's exact summand; the width-r digest follows the branch-width ablation of the appendix)
 *   select  S_h = top-k of a[h, .] over the archive A = [n_sink, N-W) (ties -> smaller position),
 *           k = min(ceil(rho*N), |A|), joined with the recent window [N-W, N) and the sinks [0, n_sink)
 *           (Sec. 4.1: keep top-m plus sinks plus the recent window)
 *   attend  s[h,u] = lambda (Qc_h . L_u + Qr_h . K_u) over u in S_h; out_h = sum softmax(s) L_u (512 wide),
 *           lse_h, and s*_h = max s (Eq. 1, Lemma 1)
 *   trigger (two-tier) F_h = { u in A \ S_h : lambda (a[h,u] + |(O Qr_h)[r:]| P_res[u/64]
 *           + z_eff |Qc_h| eta_u) > s*_h }, optionally the top_j of them (Eq. 4 with sketch rank 0,
 *           Lemma 2; the fetch of rows that beat the tier-1 max), attended too and merged by LSE.
 *           Reading B admits whole 64-row pages instead: every archived row outside S_h of a page P with
 *           lambda (|Qr_h| max_P |K_u| + z_eff |Qc_h| max_P eta_u) > s*_h (Lemma 2 on the page's extreme norms).
 *
 * Conventions
 *   - Every pointer in vk_view / vk_index and every output is DEVICE memory owned by the caller.
 *     The library never allocates device memory; scratch comes from the caller's workspace.
 *   - Every call is asynchronous on `stream` (a cudaStream_t, NULL = the legacy default stream) and
 *     does not synchronise with the host, except vk_poll_status.
 *   - Arguments are checked on the host before any launch; a bad argument returns VK_ERR_INVALID_ARG or
 *     VK_ERR_UNSUPPORTED and launches nothing (it is never clamped). vk_last_error() describes it.
 *   - Element strides (ld, bstride) are in elements of `dtype`. Device pointers must be 16-byte aligned
 *     and ld * element size a multiple of 16 bytes.
 *   - Errors found on the device (an id out of range, a full list, a bounded wait that gave up) are written
 *     to a status word at the start of the workspace; vk_poll_status reads and clears it. The first error
 *     since the last poll is kept. A new workspace is zeroed once with vk_workspace_init.
 *   - Calls that share a workspace must be ordered (same stream, or synchronised): they reuse its scratch.
 */
#ifndef VK_H
#define VK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  VK_OK = 0,
  VK_ERR_INVALID_ARG = -1,  /* a size, pointer, stride or parameter is out of its documented range */
  VK_ERR_UNSUPPORTED = -2,  /* valid but not built (e.g. a dtype/shape combination without a kernel) */
  VK_ERR_WORKSPACE = -3,    /* ws is NULL or smaller than vk_workspace_bytes() */
  VK_ERR_CAPACITY = -4,     /* an output list was longer than cap (device status) */
  VK_ERR_CUDA = -5,         /* a CUDA launch or runtime call failed */
  VK_ERR_TIMEOUT = -6       /* a bounded device-side wait gave up (device status) */
} vk_status;

typedef enum { VK_BF16 = 0, VK_F32 = 1 } vk_dtype;

typedef enum {
  VK_TRIG_OFF = 0,     /* tier 1 only: the top-k plus window (plus sinks) */
  VK_TRIG_CS = 1,      /* two-tier, row level (reading A): fetch the archived rows whose Cauchy-Schwarz trigger
                          score (Eq. 4, with sketch rank 0 or params->r_sk) beats s* */
  VK_TRIG_CS_PAGE = 2  /* two-tier, page level (reading B): fetch every archived row of each 64-row page whose
                          page-level bound lambda (|Qr| max|K| + z_eff |Qc| max eta) beats s*; needs
                          index->page_knorm and index->page_eta. With top_j, the top_j fired rows by (page bound
                          desc, position asc) */
} vk_trigger;

/* The cache and the query of one decode step. */
typedef struct {
  int32_t B, H, N;          /* sequences, heads, cached rows per sequence (1 <= N <= 2^24 - 1) */
  int32_t dtype;            /* vk_dtype of latent, rope, q_latent and q_rope */
  const void* latent;       /* [B, N, 512]: row u of sequence b at latent + b*latent_bstride + u*latent_ld */
  int64_t latent_ld, latent_bstride;
  const void* rope;         /* [B, N, 64]; may alias latent + 512 with rope_ld = latent_ld = 576 */
  int64_t rope_ld, rope_bstride;
  const void* q_latent;     /* [B, H, 512] contiguous: the absorbed latent-side query */
  const void* q_rope;       /* [B, H, 64] contiguous: the RoPE query, rotated at position N */
} vk_view;

/* Selection and trigger parameters. */
typedef struct {
  double rho;               /* keep ratio, 0 < rho <= 1 */
  int32_t r;                /* score width: 64 (the RoPE columns) or a digest width in {4, 8, 16, 32} */
  int32_t window;           /* recent window W, 0 <= W <= N */
  int32_t n_sink;           /* leading sink rows, 0 <= n_sink <= N - W */
  float sm_scale;           /* attention scale lambda > 0 (1/sqrt(192) for 128 + 64 qk head dims) */
  int32_t trigger;          /* vk_trigger */
  float z_eff;              /* trigger certificate multiplier z / sqrt(d_c - r_sk); 1 = the sound bound */
  int32_t top_j;            /* keep only the top_j fired rows per head; 0 = uncapped */
  uint32_t flags;           /* VK_FLAG_* below; 0 for normal use */
  int32_t r_sk;             /* content sketch rank of the row-level trigger (Sec. 4.2, Eq. 4): 0 (the content
                               summand bounded whole, eta_u = |L_u|), or 16, 32, 64 with index->sketch and
                               index->sketch_basis; VK_TRIG_CS only */
} vk_params;

/* Force the exact fallback of the fused selection on every head (for tests; results are unchanged). */
#define VK_FLAG_FORCE_FALLBACK 0x1u
/* Use the materialised-score selection path even where the fused path would run (for tests). */
#define VK_FLAG_FORCE_DENSE 0x2u
/* Test hook for failure detection (bf16 caches): one attention CTA withholds its first tile's loads, so its
 * bounded waits expire after about a second, it reports VK_ERR_TIMEOUT in the device status word and every
 * role of that CTA winds down; vk_poll_status then returns VK_ERR_TIMEOUT. No other call uses it. */
#define VK_FLAG_TEST_TIMEOUT 0x4u
/* Turn off the page skip of the row-level trigger scan (for tests; the fired sets are the same either way).
 * With index->page_knorm and index->page_eta given, the r = 64 scan of VK_TRIG_CS skips every 128-row tile in which
 * no head's page bound lambda (|Qr_h| max|K| + z_eff |Qc_h| max eta) reaches s*_h: no row there can fire. */
#define VK_FLAG_NO_PAGE_SKIP 0x8u
/* Attend the fired rows with the tile pass even when every head fired few rows (for tests; the outputs are the same
 * up to fp32 rounding). By default the step attends a head's fired rows with a per-head pass over its fired bitmap
 * when no head fired more than 512 rows, and with the tile pass otherwise. */
#define VK_FLAG_FIRED_TILES 0x10u

/* The per-cache index built once by vk_build_digest (Sec. 4.2 index entry with sketch rank 0). */
typedef struct {
  const void* digest;       /* [B, N, r] bf16 contiguous, (O K_u)[0:r] rounded to nearest even; NULL iff r = 64 */
  const float* eta;         /* [B, N] |L_u|_2; needed only by the trigger */
  const float* page_res;    /* [B, ceil(N/64)] max over the page of |(O K_u)[r:64]| (0 when r = 64); trigger only */
  const float* rot;         /* [64, 64] row-major orthogonal O; NULL iff r = 64 */
  const float* page_knorm;  /* [B, ceil(N/64)] max over the page of |K_u| (all 64 RoPE dims); VK_TRIG_CS_PAGE needs
                               it, VK_TRIG_CS uses it for the page skip; may be NULL otherwise */
  const float* page_eta;    /* [B, ceil(N/64)] max over the page of eta_u; with page_knorm */
  const void* sketch;       /* [B, N, r_sk] bf16 contiguous, s_u = V_r^T L_u rounded to nearest even (vk_build_sketch);
                               with r_sk > 0, when eta must be the sketch residual |L_u - V_r s_u| */
  const float* sketch_basis;/* [r_sk, 512] fp32: the rows are V_r's orthonormal directions (vk_sketch_basis) */
} vk_index;

/* k = min(ceil(rho*N), N - W - n_sink): archived rows kept per head (-1 on bad arguments). */
int64_t vk_keep_count(int32_t N, double rho, int32_t window, int32_t n_sink);

/* Smallest cap that vk_select / vk_decode_step accept: k + W + n_sink (tier 1 only). */
int32_t vk_min_cap(const vk_view* view, const vk_params* params);

/* Workspace bytes that every call below needs for these shapes with this cap (the worst case; the same
 * buffer may be reused by consecutive calls on one stream). 0 on bad arguments. */
size_t vk_workspace_bytes(const vk_view* view, const vk_params* params, int32_t cap);

/* Index build (the compression-time work of Sec. 4.2): for every row, digest = bf16((O K_u)[0:r]) when
 * r < 64, eta_u = |L_u|_2, and per 64-row page the max of |(O K_u)[r:64]|, of |K_u| and of eta_u. Any output
 * may be NULL to skip it. rot64: [64,64] row-major fp32 orthogonal matrix (device); may be NULL when r = 64. */
int vk_build_digest(const vk_view* view, const vk_params* params, const float* rot64, void* digest, float* eta,
                    float* page_res, float* page_knorm, float* page_eta, void* stream);

/* Content sketch of the index (Sec. 4.2, Eq. 4, Lemma 1): for every row s_u = V_r^T L_u (r_sk values, stored in bf16
 * by round-to-nearest-even into sketch [B, N, r_sk]) and eta_u = |L_u - V_r s_u| (fp32 [B, N], with the unrounded s_u).
 * basis: [r_sk, 512] fp32 (device), orthonormal rows. r_sk in {16, 32, 64}. Either output may be NULL. By Lemma 1,
 * qc . L_u differs from (V_r^T qc) . s_u by at most |(I - V_r V_r^T) qc| eta_u. The paper's index keeps this entry
 * for every archived row; the trigger of vk_decode_step reads it when params->r_sk > 0. */
int vk_build_sketch(const vk_view* view, int32_t r_sk, const float* basis, void* sketch, float* eta, void* stream);

/* Workspace bytes of vk_sketch_basis; 0 on bad arguments. */
size_t vk_sketch_basis_workspace_bytes(int64_t n, int32_t r_sk);

/* The sketch basis from n queries of the context (Sec. 4.2: V_r from the context's own prefix queries): the r_sk
 * leading eigenvectors of their uncentred second moment sum_i q_i q_i^T, by decreasing eigenvalue, each signed so that
 * its entry of largest magnitude is positive, as the rows of basis [r_sk, 512] fp32, and their eigenvalues in eig
 * [r_sk] fp32 (device; eig may be NULL). queries: [n, 512] contiguous, dtype a vk_dtype (device). r_sk in {16, 32,
 * 64}, n >= r_sk. The moment is accumulated in fp32 and its leading subspace found by orthogonal iteration with a
 * Rayleigh-Ritz step in fp64: directions whose eigenvalues are close are accurate as a subspace, not one by one.
 * Queries whose second moment has rank below r_sk (fewer than r_sk independent directions) leave the iteration's
 * Cholesky factorisation with a pivot at the rounding level: the directions beyond the rank then come out as some
 * orthonormal completion, or, where a pivot is not positive, the device status word of ws is set to
 * VK_ERR_INVALID_ARG (read it with vk_poll_status) and basis is not valid. */
int vk_sketch_basis(const void* queries, int32_t dtype, int64_t n, int32_t r_sk, float* basis, float* eig, void* ws,
                    size_t ws_bytes, void* stream);

/* Score every cached row: scores[b,h,u] = a[h,u] (unscaled) as fp32, [B, H, N] contiguous. The RoPE columns
 * are read when r = 64, the index's digest otherwise. ws holds the rotated queries. */
int vk_score(const vk_view* view, const vk_params* params, const vk_index* index, float* scores, void* ws,
             size_t ws_bytes, void* stream);

/* Per-head selection from materialised scores ([B,H,N] fp32, e.g. from vk_score): idx[b,h,0:count) lists
 * S_h in ascending position, count[b,h] = k + W + n_sink, kth[b,h] = the k-th largest archive score
 * (+inf when k = 0; kth may be NULL). cap >= vk_min_cap. */
int vk_select(const vk_view* view, const vk_params* params, const float* scores, int32_t* idx, int32_t* count,
              float* kth, int32_t cap, void* ws, size_t ws_bytes, void* stream);

/* Absorbed-MLA attention over caller-given sets idx[b,h,0:count[b,h]) (distinct positions in [0,N); an
 * id out of range is skipped and flags VK_ERR_INVALID_ARG in the device status). out [B,H,512] fp32,
 * lse [B,H] and smax [B,H] (s*, the max logit) fp32; lse and smax may be NULL. An empty set gives
 * out = 0 and lse = smax = -inf. For bf16 caches the rows are read in 64-row tiles and rows no head
 * selected enter the product with weight 0, so every one of the N cached rows must hold finite values. */
int vk_sparse_attn(const vk_view* view, const vk_params* params, const int32_t* idx, const int32_t* count,
                   int32_t cap, float* out, float* lse, float* smax, void* ws, size_t ws_bytes, void* stream);

/* The whole step: score, select, attend, and with params->trigger = VK_TRIG_CS (or VK_TRIG_CS_PAGE) also the
 * trigger scan (or the page-bound test), the attention over the fired rows and the LSE merge. out [B,H,512], lse [B,H]; smax [B,H] (s* of the tier-1
 * set; may be NULL). idx[b,h,:] lists S_h (ascending) followed by F_h (ascending) and count[b,h] is
 * |S_h| + |F_h|; fired rows that do not fit in cap are still attended (out/lse stay exact) but are left
 * out of the list, and VK_ERR_CAPACITY is raised in the device status. index may be NULL when r = 64
 * and the trigger is off. Nothing synchronises with the host; the call can be captured in a CUDA graph. */
int vk_decode_step(const vk_view* view, const vk_params* params, const vk_index* index, float* out, float* lse,
                   float* smax, int32_t* idx, int32_t* count, int32_t cap, void* ws, size_t ws_bytes,
                   void* stream);

/* Zero the device status word of a new workspace (asynchronous on `stream`). Call once after allocating it. */
int vk_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* Scratch size of vk_decode_step_noalloc: 16 MiB of device memory in a static array of this library. */
#define VK_NOALLOC_SCRATCH_BYTES (16u << 20)

/* The decode step of vk_decode_step for callers that cannot allocate device memory, so cannot pass a
 * workspace: a plugin that may use only memory its host program gave it and has no allocator behind a C
 * interface, or a serving loop that fixed its device-memory budget at start-up and forbids later cudaMalloc
 * calls. The paper has no counterpart; this is a deployment convenience.
 *   - Scratch comes from one static device array of VK_NOALLOC_SCRATCH_BYTES, which the CUDA runtime sets
 *     aside on every GPU where this library's code is loaded and keeps until the process exits. The call
 *     allocates nothing itself (no cudaMalloc, no allocating library routine).
 *   - Problems whose vk_workspace_bytes() exceeds VK_NOALLOC_SCRATCH_BYTES are rejected with
 *     VK_ERR_WORKSPACE; bad arguments are refused exactly as vk_decode_step refuses them.
 *   - Every call looks up the array's device address on the current device (cudaGetSymbolAddress); the
 *     first call on a device may also load the library's device code there, so make that first call before
 *     any stream capture on that device.
 *   - Every call on a device shares the one array and it keeps the last call's contents; the call clears
 *     the status word it needs at zero. Calls that overlap on the GPU (other streams, other host threads,
 *     without ordering between them) race on the array and corrupt each other's results.
 *   - Device-side status (VK_ERR_CAPACITY, VK_ERR_TIMEOUT) is not reported: the status word is reset at
 *     the start of every call. Outputs are the same as vk_decode_step's. */
int vk_decode_step_noalloc(const vk_view* view, const vk_params* params, const vk_index* index, float* out,
                           float* lse, float* smax, int32_t* idx, int32_t* count, int32_t cap, void* stream);

/* ---------------------------------------------------------------------------------------------------------------
 * Conformal calibration of the trigger's z (Sec. 4.2, Sec. 5 "Recommended configuration"). Every (b, h) of the
 * view is one calibration query, with its attended set S_h given as vk_decode_step lists it (idx, count, cap; the
 * tier-1 part of a step with the same params). A query is hard when its exact argmax row over all cached rows (ties:
 * the smaller position) lies outside S_h; its required inflation is zq = (s* - idx_t) / cert_t, s* the max logit
 * over S_h, idx_t = lambda (a[h,u*] + |(O Qr_h)[r:]| page_res[page(u*)]), cert_t = lambda |Qc_h| eta_u* / sqrt(512)
 * (the sketch-rank-0 index part and certificate of Eq. 4). With alpha = (1 - tau)/2, tau_s = tau / (1 - alpha) and
 * min_hard = ceil(tau_s / (1 - tau_s)), z is the ceil((n+1) tau_s)-th smallest zq over the n hard queries, z_max
 * when n < min_hard or that index passes n, clamped to [0, z_max]. Outputs (device): zq [B, H] fp32, NaN where the
 * query is not hard; z_out[3] = {z, z_eff = z / sqrt(512) (the decode step's z_eff), n_hard}. index needs eta and
 * page_res (and the digest and rotation when r < 64); bf16 caches only (the argmax runs on the tensor-core
 * attention over every row); B * H <= 16384 (one block sorts the zq). With params->r_sk > 0 (and the index's sketch
 * and basis, eta the sketch residual) the index part gains p_h . s_u* and cert_t = lambda rho_h eta_u* /
 * sqrt(512 - r_sk), the sketch certificate of Eq. 4; z_out[1] is then z / sqrt(512 - r_sk). */
size_t vk_conformal_workspace_bytes(const vk_view* view, const vk_params* params);
int vk_conformal_z(const vk_view* view, const vk_params* params, const vk_index* index, const int32_t* idx,
                   const int32_t* count, int32_t cap, float tau, float z_max, float* zq, float* z_out, void* ws,
                   size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------------------------------
 * The PCA digest basis (the appendix's branch-width ablation: principal directions of the branch instead of a
 * random rotation). rot [64, 64] row-major fp32 (device): the eigenvectors of M = sum over every row of every
 * sequence of the view of K_u K_u^T, by decreasing eigenvalue, each signed so that its largest entry is positive;
 * usable as index->rot and as vk_build_digest's rot64, so that the width-r digest keeps the most branch energy.
 * eig [64] fp32 (device, may be NULL): the eigenvalues. M is accumulated on the tensor cores (bf16 rows, fp32 per
 * CTA, fp64 across CTAs); the 64 x 64 eigenproblem is solved by cyclic Jacobi, sweeps in fp32 finished by sweeps in
 * fp64 on the fp64 projection of M onto the re-orthonormalised fp32 eigenvectors. bf16 caches only. */
size_t vk_pca_workspace_bytes(void);
int vk_pca_basis(const vk_view* view, float* rot, float* eig, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------------------------------
 * The sigma selector of tier 1 (Sec. 4.1, Eq. 3; Corollary 1): a query-independent ranking of cached rows by how
 * far their 64-wide RoPE branch lies from its low-pass reconstruction. Rows are cut into fixed blocks of T rows
 * (4096 in the paper); within each closed block, per RoPE dim, the sequence-axis DFT is kept on bins
 * 0 .. kappa-1 (the one-sided spectrum of a real signal) and inverted, and sigma_u = |r_u - low_u|_2 over the 64
 * dims. A block's sigma depends on that block alone, so a stream of closes gives the same values as one pass. */

/* Workspace bytes of vk_sigma for a block length T and bandwidth kappa; 0 on bad arguments (T a positive multiple
 * of 128, 1 <= kappa <= 64). The workspace starts with the device status word read by vk_poll_status. */
size_t vk_sigma_workspace_bytes(int32_t T, int32_t kappa);

/* sigma [B, N] fp32 (device) for every row of every sequence of the view (only its RoPE columns are read; bf16
 * caches, VK_ERR_UNSUPPORTED otherwise). Rows past the last whole block of T rows (the open tail) get -1. The two
 * contractions per block run on the tensor cores with the low-pass basis and its coefficients rounded to bf16
 * (fp32 accumulation): sigma is exact to about 1e-4 relative. */
int vk_sigma(const vk_view* view, int32_t T, int32_t kappa, float* sigma, void* ws, size_t ws_bytes, void* stream);

/* The sigma selector's attended set of every sequence (Sec. 4.1: sinks, the open tail, and the top m closed rows):
 * the sinks [0, min(n_sink, closed)), the rows past the last whole block of T rows, and the m closed rows outside
 * the sinks with the largest sigma (ties: the smaller position; m is clamped to the rows available), listed in
 * ascending position in idx[b, 0:count[b]) (idx [B, cap] int32, count [B] int32; device). sigma [B, N] as written
 * by vk_sigma. cap must hold the whole set. ws: at least 256 bytes (the device status word). */
int vk_sigma_select(int32_t B, int32_t N, int32_t T, const float* sigma, int32_t n_sink, int64_t m, int32_t* idx,
                    int32_t* count, int32_t cap, void* ws, size_t ws_bytes, void* stream);

/* Wait for `stream`, read the device status word at the start of ws (VK_OK or a device-side error of the
 * calls since the last poll) and clear it. */
int vk_poll_status(void* ws, void* stream);

/* Profiling: record events[i] (cudaEvent_t handles) on the step's stream at the stage boundaries of every
 * later vk_decode_step on this host thread: [0] start, then after [1] query prep, [2] scoring, [3] selection,
 * [4] tier-1 attention, [5] trigger and fired attention (recorded right after [4] when the trigger is off),
 * [6] the merge. n must be 0 (recording off) or 7. The events must outlive the calls that record them. */
int vk_profile_set_events(void* const* events, int32_t n);

/* Kernels launched through the library by this host thread since it started. */
int64_t vk_profile_launches(void);

/* Description of the last error returned on this host thread ("" if none). */
const char* vk_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* VK_H */
