// vk_api.cu -- the extern "C" entry points of libvk.so: argument checks, workspace layout, launch order.
//
// Every entry point checks its arguments on the host before touching the GPU and refuses (never clamps) a
// bad one. The launch sequence of a decode step has no host synchronisation and no allocation, so a CUDA
// graph can capture it.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_score_tc.h"

namespace vk {
thread_local int64_t g_launches = 0;
void count_launches(int n) { g_launches += n; }
int record_error(int code, const char* msg);
}  // namespace vk

namespace {

thread_local char g_err[512] = "";
thread_local cudaEvent_t g_prof_events[7];
thread_local int g_prof_n = 0;

void prof(int i, cudaStream_t st) {
  if (g_prof_n) cudaEventRecord(g_prof_events[i], st);
}

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(VK_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int64_t MAX_N = (1 << 24) - 1;

int check_view(const vk_view* v) {
  if (!v) return fail(VK_ERR_INVALID_ARG, "view is NULL");
  if (v->B < 1 || v->H < 1 || v->N < 1) return fail(VK_ERR_INVALID_ARG, "B, H, N must be >= 1 (got %d, %d, %d)", v->B, v->H, v->N);
  if (v->N > MAX_N) return fail(VK_ERR_INVALID_ARG, "N = %d exceeds %lld", v->N, (long long)MAX_N);
  if (v->H > vk::MAX_H) return fail(VK_ERR_UNSUPPORTED, "H = %d exceeds %d", v->H, vk::MAX_H);
  if (v->dtype != VK_BF16 && v->dtype != VK_F32) return fail(VK_ERR_INVALID_ARG, "dtype %d is not VK_BF16/VK_F32", v->dtype);
  if (!v->latent || !v->rope || !v->q_latent || !v->q_rope) return fail(VK_ERR_INVALID_ARG, "a view pointer is NULL");
  if (!aligned16(v->latent) || !aligned16(v->rope) || !aligned16(v->q_latent) || !aligned16(v->q_rope))
    return fail(VK_ERR_INVALID_ARG, "view pointers must be 16-byte aligned");
  const int64_t esz = v->dtype == VK_BF16 ? 2 : 4;
  if (v->latent_ld < vk::D_LAT || v->rope_ld < vk::D_ROPE)
    return fail(VK_ERR_INVALID_ARG, "latent_ld >= 512 and rope_ld >= 64 required (got %lld, %lld)",
                (long long)v->latent_ld, (long long)v->rope_ld);
  if ((v->latent_ld * esz) % 16 || (v->rope_ld * esz) % 16 || (v->latent_bstride * esz) % 16 ||
      (v->rope_bstride * esz) % 16)
    return fail(VK_ERR_INVALID_ARG, "row and batch strides must be multiples of 16 bytes");
  if (v->B > 1 && (v->latent_bstride < (int64_t)(v->N - 1) * v->latent_ld + vk::D_LAT ||
                   v->rope_bstride < (int64_t)(v->N - 1) * v->rope_ld + vk::D_ROPE))
    return fail(VK_ERR_INVALID_ARG, "batch strides overlap the previous sequence");
  return VK_OK;
}

int64_t keep_count(int64_t N, double rho, int64_t W, int64_t s) {
  int64_t A = N - W - s;
  if (A < 0) A = 0;
  int64_t k = (int64_t)std::ceil(rho * (double)N);
  return k < A ? k : A;
}

int check_params(const vk_view* v, const vk_params* p) {
  if (!p) return fail(VK_ERR_INVALID_ARG, "params is NULL");
  if (!(p->rho > 0.0 && p->rho <= 1.0)) return fail(VK_ERR_INVALID_ARG, "rho = %g is outside (0, 1]", p->rho);
  if (p->r != 4 && p->r != 8 && p->r != 16 && p->r != 32 && p->r != 64)
    return fail(VK_ERR_INVALID_ARG, "r = %d is not in {4, 8, 16, 32, 64}", p->r);
  if (p->window < 0 || p->window > v->N) return fail(VK_ERR_INVALID_ARG, "window = %d is outside [0, N]", p->window);
  if (p->n_sink < 0 || p->n_sink > v->N - p->window)
    return fail(VK_ERR_INVALID_ARG, "n_sink = %d is outside [0, N - window]", p->n_sink);
  if (!(p->sm_scale > 0.f) || !std::isfinite(p->sm_scale)) return fail(VK_ERR_INVALID_ARG, "sm_scale must be finite and > 0");
  if (p->trigger != VK_TRIG_OFF && p->trigger != VK_TRIG_CS && p->trigger != VK_TRIG_CS_PAGE)
    return fail(VK_ERR_INVALID_ARG, "trigger = %d is unknown", p->trigger);
  if (!(p->z_eff >= 0.f) || !std::isfinite(p->z_eff)) return fail(VK_ERR_INVALID_ARG, "z_eff must be finite and >= 0");
  if (p->top_j < 0) return fail(VK_ERR_INVALID_ARG, "top_j must be >= 0");
  if (p->flags & ~(VK_FLAG_FORCE_FALLBACK | VK_FLAG_FORCE_DENSE | VK_FLAG_TEST_TIMEOUT | VK_FLAG_NO_PAGE_SKIP |
                   VK_FLAG_FIRED_TILES))
    return fail(VK_ERR_INVALID_ARG, "unknown flags 0x%x", p->flags);
  if (p->r_sk != 0 && p->r_sk != 16 && p->r_sk != 32 && p->r_sk != 64)
    return fail(VK_ERR_INVALID_ARG, "r_sk = %d is not in {0, 16, 32, 64}", p->r_sk);
  if (p->r_sk > 0 && p->trigger != VK_TRIG_CS)
    return fail(VK_ERR_INVALID_ARG, "the content sketch (r_sk = %d) belongs to the row-level trigger VK_TRIG_CS", p->r_sk);
  return VK_OK;
}

int check_index(const vk_view* v, const vk_params* p, const vk_index* ix, bool need_trigger) {
  if (p->r < vk::D_ROPE) {
    if (!ix || !ix->digest || !ix->rot) return fail(VK_ERR_INVALID_ARG, "r < 64 needs index->digest and index->rot");
    if (!aligned16(ix->digest) || !aligned16(ix->rot)) return fail(VK_ERR_INVALID_ARG, "index pointers must be 16-byte aligned");
  }
  if (need_trigger && p->trigger == VK_TRIG_CS) {
    if (!ix || !ix->eta || !ix->page_res) return fail(VK_ERR_INVALID_ARG, "the trigger needs index->eta and index->page_res");
    if ((ix->page_knorm == nullptr) != (ix->page_eta == nullptr))
      return fail(VK_ERR_INVALID_ARG, "index->page_knorm and index->page_eta go together");
  }
  if (need_trigger && p->trigger == VK_TRIG_CS && p->r_sk > 0) {
    if (!ix->sketch || !ix->sketch_basis)
      return fail(VK_ERR_INVALID_ARG, "r_sk > 0 needs index->sketch and index->sketch_basis");
    if (!aligned16(ix->sketch) || !aligned16(ix->sketch_basis))
      return fail(VK_ERR_INVALID_ARG, "index->sketch and index->sketch_basis must be 16-byte aligned");
  }
  if (need_trigger && p->trigger == VK_TRIG_CS_PAGE) {
    if (!ix || !ix->page_knorm || !ix->page_eta)
      return fail(VK_ERR_INVALID_ARG, "the page trigger needs index->page_knorm and index->page_eta");
  }
  (void)v;
  return VK_OK;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Positions per attention split, a multiple of 64 (the attention tile). One attention CTA is resident per SM,
// so the split count is chosen to fill the SMs in whole waves: maximise (work) / (waves x SMs x positions per
// CTA), preferring longer splits (fewer partials to merge) when two counts are equally good.
void choose_splits(const vk_view& v, int64_t* nsplit, int64_t* split_len) {
  const int64_t per_pos = (int64_t)v.B * ((v.H + vk::HG - 1) / vk::HG);
  const int64_t N = v.N;
  const int64_t lo = std::max<int64_t>(1, (N + 16383) / 16384);
  const int64_t hi = std::max<int64_t>(lo, std::min<int64_t>((N + 255) / 256, 2048));
  const int64_t sms = vk::sm_count();
  double best = -1.0;
  int64_t best_len = ((N + 63) / 64) * 64;
  for (int64_t ns = lo; ns <= hi; ++ns) {
    const int64_t len = ((N + ns - 1) / ns + 63) / 64 * 64;
    const int64_t ns_eff = (N + len - 1) / len;
    const int64_t ctas = per_pos * ns_eff;
    const int64_t waves = (ctas + sms - 1) / sms;
    const double eff = (double)(per_pos * N) / ((double)waves * sms * len);
    if (eff > best + 1e-9) { best = eff; best_len = len; }
  }
  *split_len = best_len;
  *nsplit = (N + best_len - 1) / best_len;
}

}  // namespace

namespace vk {
// Partial-result layout of the attention kernel that runs for this view: the persistent layout for the
// tensor-core kernel, the split layout for the fp32 kernel. Persistent: one CTA per SM, but at least 4 tiles per
// CTA -- a partial (64 heads x 512 fp32 = 128 KB) costs more traffic than a tile (72 KB), so small problems take
// fewer, longer ranges.
int sm_count() {
  static int cached[64] = {0};
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return 152;
  }
  if (cached[dev] > 0) return cached[dev];
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = 152;
  }
  cached[dev] = n;
  return n;
}

AttnGeom attn_geom(const vk_view& v) {
  AttnGeom g{};
  g.n_hg = (v.H + HG - 1) / HG;
  g.T = (v.N + 63) / 64;
  g.total = (long long)v.B * g.n_hg * g.T;
  if (attn_tc_supported(v)) {
    // P ranges of at least 4 positions, n_hg CTAs each, at most one CTA per SM where the groups allow
    const long long P = std::min<long long>(std::max<long long>(1, (long long)v.B * g.T / 4),
                                            std::max(1, sm_count() / g.n_hg));
    g.G = (int)(P * g.n_hg);
    g.nslot = 1;
    for (long long s = 0; s < (long long)v.B * g.n_hg; ++s) g.nslot = std::max(g.nslot, attn_nvalid(g, s));
  } else {
    int64_t ns = 0, len = 0;
    choose_splits(v, &ns, &len);
    g.nsplit = (int)ns;
    g.split_len = (int)len;
    g.nslot = (int)ns;
  }
  return g;
}
}  // namespace vk

namespace {

// Fused selection parameters: a strided sample of about 2048+ archive rows per head gives theta = its j-th
// largest score, with j chosen so that ~1.5 k + 8 samples' worth of archive rows pass; the candidate list has
// room for twice that (+2048) before the exact fallback takes over.
void fused_params(int64_t N, int64_t lo, int64_t hi, int64_t k, VkLayout* L) {
  const int64_t A = std::max<int64_t>(0, hi - lo);
  L->ss = A >= 49152 ? 32 : A >= 32768 ? 16 : std::max<int64_t>(1, A / 2048);
  L->soff = L->ss / 2;
  L->ns = N > L->soff ? (N - L->soff + L->ss - 1) / L->ss : 0;
  L->sld = (L->ns + 7) / 8 * 8;            // sample rows start on 16-byte boundaries
  int64_t n_arch = 0;                      // sampled rows inside the archive
  for (int64_t i = 0; i < L->ns; ++i) {
    const int64_t u = L->soff + L->ss * i;
    n_arch += (u >= lo && u < hi);
  }
  L->j = n_arch ? (int64_t)std::ceil(1.5 * (double)k * (double)n_arch / (double)A) + 8 : 0;
  const int64_t expect = n_arch ? (int64_t)std::ceil((double)std::min(L->j, n_arch) * (double)A / (double)n_arch) : 0;
  L->capc = std::max<int64_t>(std::min<int64_t>(A, 2 * expect + 2048), std::max<int64_t>(k, 1));
}

VkLayout make_layout(const vk_view& v, const vk_params& p) {
  VkLayout L{};
  L.B = v.B; L.H = v.H; L.N = v.N;
  L.nw = (v.N + 31) / 32;
  L.n_hg = (v.H + vk::HG - 1) / vk::HG;
  L.ag = vk::attn_geom(v);
  L.two_tier = p.trigger != VK_TRIG_OFF;
  L.tc = vk::score_tc_supported(v, p.r);
  L.sketch = p.trigger == VK_TRIG_CS && p.r_sk > 0;
  // the tensor-core trigger carries the sketch at r = 64 for up to 128 heads; otherwise the scores are materialised
  // and the dense trigger adds the sketch term
  L.fused = L.tc && !(p.flags & VK_FLAG_FORCE_DENSE) && !(L.sketch && (p.r != vk::D_ROPE || v.H > 128));
  L.dense_scores = !L.fused;
  const int64_t lo = p.n_sink, hi = (int64_t)v.N - p.window;
  const int64_t k = keep_count(v.N, p.rho, p.window, p.n_sink);
  if (L.fused) fused_params(v.N, lo, hi, k, &L);
  const bool page_trig = p.trigger == VK_TRIG_CS_PAGE;
  L.fcap = ((L.fused || page_trig) && L.two_tier && p.top_j > 0) ? std::max<int64_t>(1, hi - lo) : 0;
  const int64_t BH = (int64_t)v.B * v.H;
  const int64_t nslot = (int64_t)L.ag.nslot * (L.two_tier ? 2 : 1);
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
  L.off_status = take(256);
  L.off_qt = take(sizeof(float) * BH * vk::D_ROPE);
  L.off_qhl = take(sizeof(uint16_t) * BH * 2 * 32);                   // bf16 query parts of a digest (r <= 32)
  L.off_qcn = take(sizeof(float) * BH);
  L.off_qrn = take(sizeof(float) * BH);
  L.off_qrf = take(sizeof(float) * BH);
  L.off_smax1 = take(sizeof(float) * BH);
  L.off_nfired = take(sizeof(int64_t) * BH);
  L.off_scores = take(L.dense_scores ? sizeof(float) * BH * v.N : 0);
  L.off_selbm = take(sizeof(uint32_t) * BH * L.nw);
  L.off_firebm = take(L.two_tier ? sizeof(uint32_t) * BH * L.nw : 0);
  L.off_part_o = take(sizeof(float) * v.B * nslot * v.H * vk::D_LAT);
  L.off_part_ml = take(sizeof(float) * v.B * nslot * v.H * 2);
  L.off_sample = take(L.fused ? sizeof(uint16_t) * BH * L.sld : 0);    // bf16 sample scores
  L.off_theta = take(L.fused ? sizeof(float) * BH : 0);
  L.off_ccnt = take(L.fused ? sizeof(int) * BH : 0);
  L.off_cand = take(L.fused ? sizeof(int2) * BH * L.capc : 0);
  L.off_fcnt = take(L.fcap ? sizeof(int) * BH : 0);
  L.off_fcand = take(L.fcap ? sizeof(int2) * BH * L.fcap : 0);
  L.off_skp = take(L.sketch ? sizeof(float) * BH * p.r_sk : 0);
  L.off_skhl = take(L.sketch ? sizeof(uint16_t) * BH * 2 * p.r_sk : 0);
  L.off_rho = take(L.sketch ? sizeof(float) * BH : 0);
  L.off_fmode = take(L.two_tier ? sizeof(int) : 0);
  L.total = off;
  return L;
}

template <typename T>
T* at(void* ws, size_t off) { return reinterpret_cast<T*>(static_cast<char*>(ws) + off); }

int check_ws(const VkLayout& L, void* ws, size_t ws_bytes) {
  if (!ws) return fail(VK_ERR_WORKSPACE, "workspace is NULL (%zu bytes needed)", L.total);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(VK_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (ws_bytes < L.total) return fail(VK_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", ws_bytes, L.total);
  return VK_OK;
}

#define VK_CUDA(call, where)                         \
  do {                                               \
    cudaError_t e_ = (call);                         \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

}  // namespace

// Error reporting for entry points defined in other translation units.
int vk::record_error(int code, const char* msg) { return fail(code, "%s", msg); }

extern "C" {

const char* vk_last_error(void) { return g_err; }

int vk_profile_set_events(void* const* events, int32_t n) {
  g_err[0] = 0;
  if (n != 0 && n != 7) return fail(VK_ERR_INVALID_ARG, "n must be 0 or 7 (got %d)", n);
  if (n && !events) return fail(VK_ERR_INVALID_ARG, "events is NULL");
  for (int i = 0; i < n; ++i) {
    if (!events[i]) return fail(VK_ERR_INVALID_ARG, "events[%d] is NULL", i);
    g_prof_events[i] = static_cast<cudaEvent_t>(events[i]);
  }
  g_prof_n = n;
  return VK_OK;
}

int64_t vk_profile_launches(void) { return vk::g_launches; }

int64_t vk_keep_count(int32_t N, double rho, int32_t window, int32_t n_sink) {
  if (N < 1 || !(rho > 0.0 && rho <= 1.0) || window < 0 || window > N || n_sink < 0 || n_sink > N - window) return -1;
  return keep_count(N, rho, window, n_sink);
}

int32_t vk_min_cap(const vk_view* view, const vk_params* params) {
  if (check_view(view) != VK_OK || check_params(view, params) != VK_OK) return -1;
  return (int32_t)(keep_count(view->N, params->rho, params->window, params->n_sink) + params->window + params->n_sink);
}

size_t vk_workspace_bytes(const vk_view* view, const vk_params* params, int32_t cap) {
  if (check_view(view) != VK_OK || check_params(view, params) != VK_OK) return 0;
  (void)cap;
  return make_layout(*view, *params).total;
}

int vk_build_digest(const vk_view* view, const vk_params* params, const float* rot64, void* digest, float* eta,
                    float* page_res, float* page_knorm, float* page_eta, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK) return rc;
  if (params->r < vk::D_ROPE && (digest || page_res) && !rot64)
    return fail(VK_ERR_INVALID_ARG, "r < 64 needs rot64 for the digest and page_res");
  if ((digest && !aligned16(digest)) || (eta && !aligned16(eta)) || (page_res && !aligned16(page_res)) ||
      (page_knorm && !aligned16(page_knorm)) || (page_eta && !aligned16(page_eta)))
    return fail(VK_ERR_INVALID_ARG, "outputs must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  VK_CUDA(vk::launch_build_digest(*view, params->r, rot64, static_cast<__nv_bfloat16*>(digest), eta, page_res,
                                  page_knorm, page_eta, st),
          "build_digest");
  return VK_OK;
}

int vk_workspace_init(void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  if (!ws || ws_bytes < 256) return fail(VK_ERR_WORKSPACE, "workspace is NULL or smaller than 256 bytes");
  VK_CUDA(cudaMemsetAsync(ws, 0, 256, static_cast<cudaStream_t>(stream)), "workspace init");
  return VK_OK;
}

int vk_score(const vk_view* view, const vk_params* params, const vk_index* index, float* scores, void* ws,
             size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK ||
      (rc = check_index(view, params, index, false)) != VK_OK)
    return rc;
  if (!scores || !aligned16(scores)) return fail(VK_ERR_INVALID_ARG, "scores must be a 16-byte aligned pointer");
  const VkLayout L = make_layout(*view, *params);
  if ((rc = check_ws(L, ws, ws_bytes)) != VK_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* qt = at<float>(ws, L.off_qt);
  __nv_bfloat16* qhl = at<__nv_bfloat16>(ws, L.off_qhl);
  if (!L.tc || params->r < vk::D_ROPE)
    VK_CUDA(vk::launch_qprep(*view, params->r, index ? index->rot : nullptr, qt, at<float>(ws, L.off_qcn),
                             at<float>(ws, L.off_qrn), at<float>(ws, L.off_qrf), L.tc ? qhl : nullptr, st), "qprep");
  if (L.tc) {
    vk::ScoreTcArgs a{};
    a.mode = 0;
    a.scores = scores;
    a.scores_ld = view->N;
    a.status = at<int>(ws, L.off_status);
    VK_CUDA(vk::launch_score_tc(*view, params->r, index ? index->digest : nullptr, qhl, 0, 1, view->N, a, st),
            "score (tcgen05)");
    return VK_OK;
  }
  VK_CUDA(vk::launch_score_simt(*view, params->r, qt,
                                static_cast<const __nv_bfloat16*>(index ? index->digest : nullptr), scores, st),
          "score");
  return VK_OK;
}

int vk_select(const vk_view* view, const vk_params* params, const float* scores, int32_t* idx, int32_t* count,
              float* kth, int32_t cap, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK) return rc;
  if (!scores || !idx || !count) return fail(VK_ERR_INVALID_ARG, "scores, idx and count must be non-NULL");
  const int64_t k = keep_count(view->N, params->rho, params->window, params->n_sink);
  if ((int64_t)cap < k + params->window + params->n_sink)
    return fail(VK_ERR_INVALID_ARG, "cap = %d < k + W + n_sink = %lld", cap, (long long)(k + params->window + params->n_sink));
  int* status = nullptr;
  if (ws) {
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < 256) return fail(VK_ERR_WORKSPACE, "workspace too small or misaligned");
    status = at<int>(ws, 0);
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  VK_CUDA(vk::launch_select_dense(view->B, view->H, view->N, scores, nullptr, k, params->window, params->n_sink, idx,
                                  count, cap, 0, kth, nullptr, 0, status, st), "select");
  return VK_OK;
}

int vk_sparse_attn(const vk_view* view, const vk_params* params, const int32_t* idx, const int32_t* count,
                   int32_t cap, float* out, float* lse, float* smax, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK) return rc;
  if (!idx || !count || !out || cap < 0) return fail(VK_ERR_INVALID_ARG, "idx, count and out must be non-NULL, cap >= 0");
  if (!aligned16(out)) return fail(VK_ERR_INVALID_ARG, "out must be 16-byte aligned");
  const VkLayout L = make_layout(*view, *params);
  if ((rc = check_ws(L, ws, ws_bytes)) != VK_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* status = at<int>(ws, L.off_status);
  uint32_t* bm = at<uint32_t>(ws, L.off_selbm);
  float* po = at<float>(ws, L.off_part_o);
  float* pml = at<float>(ws, L.off_part_ml);
  VK_CUDA(vk::launch_list_to_bitmap(view->B, view->H, view->N, idx, count, cap, bm, L.nw, status, st), "list_to_bitmap");
  VK_CUDA(vk::launch_attn(*view, params->sm_scale, bm, L.nw, L.ag, 0, L.ag.nslot, po, pml, params->flags, status, st),
          "attention");
  VK_CUDA(vk::launch_combine(view->B, view->H, L.ag, L.ag.nslot, po, pml, out, lse, smax, st), "combine");
  return VK_OK;
}

// Largest fired set per head for which the per-head pass over the fired rows beats the tile pass.
constexpr int kFiredListMax = 512;

int vk_decode_step(const vk_view* view, const vk_params* params, const vk_index* index, float* out, float* lse,
                   float* smax, int32_t* idx, int32_t* count, int32_t cap, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK) return rc;
  const bool two_tier = params->trigger != VK_TRIG_OFF;
  if ((rc = check_index(view, params, index, two_tier)) != VK_OK) return rc;
  if (!out || !lse || !idx || !count) return fail(VK_ERR_INVALID_ARG, "out, lse, idx and count must be non-NULL");
  if (!aligned16(out)) return fail(VK_ERR_INVALID_ARG, "out must be 16-byte aligned");
  const int64_t k = keep_count(view->N, params->rho, params->window, params->n_sink);
  if ((int64_t)cap < k + params->window + params->n_sink)
    return fail(VK_ERR_INVALID_ARG, "cap = %d < k + W + n_sink = %lld", cap, (long long)(k + params->window + params->n_sink));
  const VkLayout L = make_layout(*view, *params);
  if ((rc = check_ws(L, ws, ws_bytes)) != VK_OK) return rc;

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const vk_view& v = *view;
  const int B = v.B, H = v.H, N = v.N, W = params->window, S = params->n_sink;
  int* status = at<int>(ws, L.off_status);
  float* qt = at<float>(ws, L.off_qt);
  float* qcn = at<float>(ws, L.off_qcn);
  float* qrn = at<float>(ws, L.off_qrn);
  float* qrf = at<float>(ws, L.off_qrf);
  __nv_bfloat16* qhl = at<__nv_bfloat16>(ws, L.off_qhl);
  const void* digest = index ? index->digest : nullptr;
  const int r = params->r;
  float* scores = at<float>(ws, L.off_scores);
  uint32_t* selbm = at<uint32_t>(ws, L.off_selbm);
  float* po = at<float>(ws, L.off_part_o);
  float* pml = at<float>(ws, L.off_part_ml);
  const int ns = L.ag.nslot, nslot = two_tier ? 2 * ns : ns;

  const int lo = S, hi = N - W;
  prof(0, st);
  // the query prep feeds the materialised-score path, the trigger and digest scoring on the tensor cores (the bf16
  // query parts); the fused path at r = 64 scores with the RoPE query as it is (its exact fallback reads it directly)
  const bool qprep = !L.fused || two_tier || r < vk::D_ROPE;
  if (qprep)
    VK_CUDA(vk::launch_qprep(v, r, index ? index->rot : nullptr, qt, qcn, qrn, qrf, L.tc ? qhl : nullptr, st), "qprep");
  prof(1, st);
  if (L.fused) {
    // threshold from a strided sample, then one scoring pass that keeps only the rows above it
    float* sample = at<float>(ws, L.off_sample);
    float* theta = at<float>(ws, L.off_theta);
    int* ccnt = at<int>(ws, L.off_ccnt);
    int2* cand = at<int2>(ws, L.off_cand);
    if (k == 0) VK_CUDA(cudaMemsetAsync(ccnt, 0, sizeof(int) * B * H, st), "candidate counts");
    if (k > 0) {
      vk::ScoreTcArgs a{};
      a.mode = 0;
      a.scores = sample;
      a.scores_ld = L.sld;
      a.scores_bf16 = 1;
      a.status = status;
      VK_CUDA(vk::launch_score_tc(v, r, digest, qhl, (int)L.soff, (int)L.ss, (int)L.ns, a, st), "sample scores");
      VK_CUDA(vk::launch_theta(B, H, (int)L.ns, (int)L.sld, (int)L.soff, (int)L.ss, lo, hi, (int)L.j, sample, theta, st,
                               ccnt),   // also zeroes the candidate counts
              "theta");
      vk::ScoreTcArgs c{};
      c.mode = 1;
      c.theta = theta;
      c.arch_lo = lo;
      c.arch_hi = hi;
      c.cand_cnt = ccnt;
      c.cand = cand;
      c.capc = (int)L.capc;
      c.status = status;
      VK_CUDA(vk::launch_score_tc(v, r, digest, qhl, 0, 1, N, c, st), "score (candidates)");
    }
    prof(2, st);
    VK_CUDA(vk::launch_select_cand(B, H, N, lo, hi, k, nullptr, ccnt, cand, (int)L.capc,
                                   (params->flags & VK_FLAG_FORCE_FALLBACK) ? 1 : 0, v, r, digest, qprep ? qt : nullptr,
                                   idx, count, cap, 0, nullptr, selbm, L.nw, status, st),
            "select (candidates)");
  } else {
    if (L.tc) {
      vk::ScoreTcArgs a{};
      a.mode = 0;
      a.scores = scores;
      a.scores_ld = N;
      a.status = status;
      VK_CUDA(vk::launch_score_tc(v, r, digest, qhl, 0, 1, N, a, st), "score (tcgen05)");
    } else {
      VK_CUDA(vk::launch_score_simt(v, params->r, qt, static_cast<const __nv_bfloat16*>(index ? index->digest : nullptr),
                                    scores, st), "score");
    }
    prof(2, st);
    VK_CUDA(vk::launch_select_dense(B, H, N, scores, nullptr, k, W, S, idx, count, cap, 0, nullptr, selbm, L.nw, status, st),
            "select");
  }
  prof(3, st);
  VK_CUDA(vk::launch_attn(v, params->sm_scale, selbm, L.nw, L.ag, 0, nslot, po, pml, params->flags, status, st),
          "attention");
  prof(4, st);
  if (two_tier) {
    float* smax1 = at<float>(ws, L.off_smax1);
    int64_t* nfired = at<int64_t>(ws, L.off_nfired);
    uint32_t* firebm = at<uint32_t>(ws, L.off_firebm);
    VK_CUDA(vk::launch_smax_reduce(B, H, L.ag, nslot, pml, smax1, st), "smax");
    // with a content sketch the certificate's query norm is the sketch residual rho_h (Lemma 1), passed as |Qc|
    const float* cq = qcn;
    float* skp = nullptr;
    void* skhl = nullptr;
    if (L.sketch) {
      float* rho = at<float>(ws, L.off_rho);
      skp = at<float>(ws, L.off_skp);
      skhl = at<uint16_t>(ws, L.off_skhl);
      VK_CUDA(vk::launch_sketch_query(v, params->r_sk, index->sketch_basis, skp, skhl, rho, st), "sketch query");
      cq = rho;
    }
    if (params->trigger == VK_TRIG_CS_PAGE) {
      // reading B: whole pages by their page-level bound (no scan of the scores)
      int* fcnt = params->top_j > 0 ? at<int>(ws, L.off_fcnt) : nullptr;
      int2* fcand = params->top_j > 0 ? at<int2>(ws, L.off_fcand) : nullptr;
      VK_CUDA(vk::launch_trigger_page(B, H, N, W, S, params->sm_scale, params->z_eff, qcn, qrf, index->page_knorm,
                                      index->page_eta, smax1, selbm, firebm, L.nw, params->top_j, fcnt, fcand,
                                      (int)L.fcap, st), "page trigger");
      if (params->top_j > 0) {
        VK_CUDA(vk::launch_select_cand(B, H, N, lo, hi, params->top_j, nullptr, fcnt, fcand, (int)L.fcap, 0, v, r, digest,
                                       qt, idx, count, cap, 1, nullptr, firebm, L.nw, status, st), "top_j");
      } else {
        VK_CUDA(vk::launch_bitmap_to_list(B, H, N, firebm, L.nw, idx, count, cap, status, st), "fired list");
      }
    } else if (L.fused) {
      vk::ScoreTcArgs t{};
      t.mode = 2;
      t.arch_lo = lo;
      t.arch_hi = hi;
      t.qcn = cq;
      t.qrn = qrn;
      t.eta = index->eta;
      t.page_res = index->page_res;
      t.smax1 = smax1;
      t.lam = params->sm_scale;
      t.z = params->z_eff;
      t.selbm = selbm;
      t.firebm = firebm;
      t.nw = L.nw;
      t.top_j = params->top_j;
      t.status = status;
      if (L.sketch) {
        t.r_sk = params->r_sk;
        t.sketch = index->sketch;
        t.sketch_q = skhl;
      } else if (index->page_knorm && !(params->flags & VK_FLAG_NO_PAGE_SKIP)) {
        t.qrf = qrf;
        t.page_knorm = index->page_knorm;
        t.page_eta = index->page_eta;
      }
      if (params->top_j > 0) {
        int* fcnt = at<int>(ws, L.off_fcnt);
        int2* fcand = at<int2>(ws, L.off_fcand);
        VK_CUDA(cudaMemsetAsync(fcnt, 0, sizeof(int) * B * H, st), "fired counts");
        t.cand_cnt = fcnt;
        t.cand = fcand;
        t.capc = (int)L.fcap;
        VK_CUDA(vk::launch_score_tc(v, r, digest, qhl, 0, 1, N, t, st), "trigger (candidates)");
        VK_CUDA(vk::launch_select_cand(B, H, N, lo, hi, params->top_j, nullptr, fcnt, fcand, (int)L.fcap, 0, v, r, digest,
                                       qt, idx, count, cap, 1, nullptr, firebm, L.nw, status, st), "top_j");
      } else {
        VK_CUDA(vk::launch_score_tc(v, r, digest, qhl, 0, 1, N, t, st), "trigger");
        VK_CUDA(vk::launch_bitmap_to_list(B, H, N, firebm, L.nw, idx, count, cap, status, st), "fired list");
      }
    } else {
      VK_CUDA(vk::launch_trigger_dense(B, H, N, W, S, params->sm_scale, params->z_eff, params->top_j, scores, cq, qrn,
                                       index->eta, index->page_res, smax1, selbm, firebm, L.nw, nfired, st,
                                       L.sketch ? params->r_sk : 0, L.sketch ? index->sketch : nullptr, skp),
              "trigger");
      if (params->top_j > 0) {
        VK_CUDA(vk::launch_select_dense(B, H, N, scores, nfired, params->top_j, 0, 0, idx, count, cap, 1, nullptr, firebm,
                                        L.nw, status, st), "top_j");
      } else {
        VK_CUDA(vk::launch_bitmap_to_list(B, H, N, firebm, L.nw, idx, count, cap, status, st), "fired list");
      }
    }
    // The fired rows: when every head fired at most kFiredListMax rows (the usual case: the tier fetches only rows
    // that could still compete), one partial per (b, h) over its own fired bitmap, in the first fired slot; otherwise
    // the tile pass, which shares each loaded tile among a group's heads. The choice is made on the device from the
    // fired counts; the pass not chosen, and the merge, read the same flag.
    int* fmode = at<int>(ws, L.off_fmode);
    const int list_max = (params->flags & VK_FLAG_FIRED_TILES) ? -1 : kFiredListMax;
    VK_CUDA(vk::launch_fired_mode((int64_t)B * H, count, (int)(k + W + S), list_max, fmode, st), "fired mode");
    VK_CUDA(vk::launch_attn_list(v, params->sm_scale, firebm, L.nw, nslot, ns, po, pml, status, fmode, st),
            "fired attention (per head)");
    VK_CUDA(vk::launch_attn(v, params->sm_scale, firebm, L.nw, L.ag, ns, nslot, po, pml, 0u, status, st, fmode),
            "fired attention (tiles)");
  }
  prof(5, st);
  VK_CUDA(vk::launch_combine(B, H, L.ag, nslot, po, pml, out, lse, smax, st, -1,
                             two_tier ? at<int>(ws, L.off_fmode) : nullptr), "combine");
  prof(6, st);
  return VK_OK;
}

namespace {
// The calibration reuses a two-tier step's layout (tier-1 partials in slots 0 .., the all-rows pass in the second
// half, the all-rows bitmap in the fired bitmap's place) plus the argmax rows of the all-rows partials.
vk_params calib_params(const vk_params& p) {
  vk_params q = p;
  q.trigger = VK_TRIG_CS;
  q.top_j = 0;
  q.flags = 0;
  return q;
}
size_t calib_arg_offset(const VkLayout& L) { return align_up(L.total, 256); }
size_t calib_bytes(const VkLayout& L, const vk_view& v) {
  return calib_arg_offset(L) + sizeof(int) * (size_t)v.B * 2 * L.ag.nslot * v.H;
}
}  // namespace

size_t vk_conformal_workspace_bytes(const vk_view* view, const vk_params* params) {
  if (check_view(view) != VK_OK || check_params(view, params) != VK_OK) return 0;
  const vk_params q = calib_params(*params);
  return calib_bytes(make_layout(*view, q), *view);
}

int vk_conformal_z(const vk_view* view, const vk_params* params, const vk_index* index, const int32_t* idx,
                   const int32_t* count, int32_t cap, float tau, float z_max, float* zq, float* z_out, void* ws,
                   size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK || (rc = check_params(view, params)) != VK_OK) return rc;
  const vk_params q = calib_params(*params);
  if ((rc = check_index(view, &q, index, true)) != VK_OK) return rc;
  if (!vk::attn_tc_supported(*view)) return fail(VK_ERR_UNSUPPORTED, "the calibration's argmax pass reads bf16 caches");
  if (!(tau > 0.f && tau < 1.f)) return fail(VK_ERR_INVALID_ARG, "tau = %g is outside (0, 1)", tau);
  if (!(z_max >= 0.f) || !std::isfinite(z_max)) return fail(VK_ERR_INVALID_ARG, "z_max must be finite and >= 0");
  if (!idx || !count || cap < 1 || !zq || !z_out) return fail(VK_ERR_INVALID_ARG, "idx, count, zq, z_out needed, cap >= 1");
  const int64_t BH = (int64_t)view->B * view->H;
  if (vk::conformal_smem_bytes(BH) > (size_t)vk::SMEM_BUDGET)
    return fail(VK_ERR_UNSUPPORTED, "B * H = %lld calibration queries exceed one block's sort", (long long)BH);
  const VkLayout L = make_layout(*view, q);
  const size_t need = calib_bytes(L, *view);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < need)
    return fail(VK_ERR_WORKSPACE, "the calibration workspace needs %zu bytes, 256-byte aligned", need);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const vk_view& v = *view;
  int* status = at<int>(ws, L.off_status);
  float* qt = at<float>(ws, L.off_qt);
  float* qcn = at<float>(ws, L.off_qcn);
  float* qrn = at<float>(ws, L.off_qrn);
  float* smax1 = at<float>(ws, L.off_smax1);
  uint32_t* selbm = at<uint32_t>(ws, L.off_selbm);
  uint32_t* allbm = at<uint32_t>(ws, L.off_firebm);
  float* po = at<float>(ws, L.off_part_o);
  float* pml = at<float>(ws, L.off_part_ml);
  int* parg = at<int>(ws, calib_arg_offset(L));
  const int ns = L.ag.nslot, nslot = 2 * ns;
  const double alpha = (1.0 - (double)tau) / 2.0, tau_s = (double)tau / (1.0 - alpha);
  const int min_hard = (int)std::ceil(tau_s / (1.0 - tau_s) - 1e-9);
  VK_CUDA(vk::launch_qprep(v, q.r, index->rot, qt, qcn, qrn, at<float>(ws, L.off_qrf), nullptr, st), "qprep");
  // s*: the max logit over each query's attended set
  VK_CUDA(vk::launch_list_to_bitmap(v.B, v.H, v.N, idx, count, cap, selbm, L.nw, status, st), "list_to_bitmap");
  VK_CUDA(vk::launch_attn(v, q.sm_scale, selbm, L.nw, L.ag, 0, nslot, po, pml, 0u, status, st), "attention (S)");
  VK_CUDA(vk::launch_smax_reduce(v.B, v.H, L.ag, nslot, pml, smax1, st), "smax");
  // the exact max logit over every row and its row
  VK_CUDA(cudaMemsetAsync(allbm, 0xff, sizeof(uint32_t) * BH * L.nw, st), "all rows");
  VK_CUDA(vk::launch_attn_tc(v, q.sm_scale, allbm, L.nw, L.ag, ns, nslot, po, pml, 0u, status, st, parg),
          "attention (all rows)");
  // with a content sketch: the queries' sketch coordinates and residual norms for the index part and certificate
  float* skp = nullptr;
  float* rho = nullptr;
  if (L.sketch) {
    skp = at<float>(ws, L.off_skp);
    rho = at<float>(ws, L.off_rho);
    VK_CUDA(vk::launch_sketch_query(v, q.r_sk, index->sketch_basis, skp, nullptr, rho, st), "sketch query");
  }
  VK_CUDA(vk::launch_calib(v, q.r, L.ag, ns, nslot, pml, parg, smax1, selbm, L.nw, qt, qcn, qrn, index->digest,
                           index->eta, index->page_res, q.sm_scale, tau_s, min_hard, z_max, zq, z_out, st,
                           L.sketch ? q.r_sk : 0, skp, L.sketch ? index->sketch : nullptr, rho),
          "conformal z");
  return VK_OK;
}

size_t vk_pca_workspace_bytes(void) { return vk::pca_workspace_bytes(); }

int vk_pca_basis(const vk_view* view, float* rot, float* eig, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK) return rc;
  if (view->dtype != VK_BF16) return fail(VK_ERR_UNSUPPORTED, "the PCA basis kernel reads bf16 caches");
  if (!rot || !aligned16(rot)) return fail(VK_ERR_INVALID_ARG, "rot must be a 16-byte aligned pointer");
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < vk::pca_workspace_bytes())
    return fail(VK_ERR_WORKSPACE, "the PCA workspace needs %zu bytes, 256-byte aligned", vk::pca_workspace_bytes());
  VK_CUDA(vk::launch_pca_basis(*view, rot, eig, ws, static_cast<cudaStream_t>(stream)), "pca basis");
  return VK_OK;
}

int vk_build_sketch(const vk_view* view, int32_t r_sk, const float* basis, void* sketch, float* eta, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK) return rc;
  if (r_sk != 16 && r_sk != 32 && r_sk != 64) return fail(VK_ERR_INVALID_ARG, "r_sk = %d is not in {16, 32, 64}", r_sk);
  if (!basis || !aligned16(basis)) return fail(VK_ERR_INVALID_ARG, "basis must be a 16-byte aligned pointer");
  if ((sketch && !aligned16(sketch)) || (eta && !aligned16(eta)))
    return fail(VK_ERR_INVALID_ARG, "sketch and eta must be 16-byte aligned");
  if (!sketch && !eta) return VK_OK;
  VK_CUDA(vk::launch_build_sketch(*view, r_sk, basis, sketch, eta, static_cast<cudaStream_t>(stream)), "build sketch");
  return VK_OK;
}

size_t vk_sketch_basis_workspace_bytes(int64_t n, int32_t r_sk) {
  if (n < 1 || (r_sk != 16 && r_sk != 32 && r_sk != 64) || n < r_sk) return 0;
  return vk::sketch_basis_ws_bytes();
}

int vk_sketch_basis(const void* queries, int32_t dtype, int64_t n, int32_t r_sk, float* basis, float* eig, void* ws,
                    size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  if (r_sk != 16 && r_sk != 32 && r_sk != 64) return fail(VK_ERR_INVALID_ARG, "r_sk = %d is not in {16, 32, 64}", r_sk);
  if (n < r_sk) return fail(VK_ERR_INVALID_ARG, "n = %lld queries cannot span r_sk = %d directions", (long long)n, r_sk);
  if (dtype != VK_BF16 && dtype != VK_F32) return fail(VK_ERR_INVALID_ARG, "dtype = %d is unknown", dtype);
  if (!queries || !aligned16(queries) || !basis || !aligned16(basis))
    return fail(VK_ERR_INVALID_ARG, "queries and basis must be 16-byte aligned pointers");
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < vk::sketch_basis_ws_bytes())
    return fail(VK_ERR_WORKSPACE, "the sketch-basis workspace needs %zu bytes, 256-byte aligned",
                vk::sketch_basis_ws_bytes());
  VK_CUDA(vk::launch_sketch_basis(queries, dtype, n, r_sk, basis, eig, ws, static_cast<cudaStream_t>(stream)),
          "sketch basis");
  return VK_OK;
}

size_t vk_sigma_workspace_bytes(int32_t T, int32_t kappa) {
  if (T < 128 || T % 128 != 0 || kappa < 1 || kappa > 64) return 0;
  return vk::sigma_workspace_bytes(T, kappa);
}

int vk_sigma(const vk_view* view, int32_t T, int32_t kappa, float* sigma, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  int rc;
  if ((rc = check_view(view)) != VK_OK) return rc;
  if (T < 128 || T % 128 != 0) return fail(VK_ERR_INVALID_ARG, "T = %d must be a positive multiple of 128", T);
  if (kappa < 1 || kappa > 64) return fail(VK_ERR_INVALID_ARG, "kappa = %d is outside [1, 64]", kappa);
  if (view->dtype != VK_BF16) return fail(VK_ERR_UNSUPPORTED, "the sigma kernel reads bf16 caches");
  if (!sigma) return fail(VK_ERR_INVALID_ARG, "sigma is NULL");
  const size_t need = vk::sigma_workspace_bytes(T, kappa);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < need)
    return fail(VK_ERR_WORKSPACE, "the sigma workspace needs %zu bytes, 256-byte aligned", need);
  VK_CUDA(vk::launch_sigma(*view, T, kappa, sigma, ws, static_cast<cudaStream_t>(stream)), "sigma");
  return VK_OK;
}

int vk_sigma_select(int32_t B, int32_t N, int32_t T, const float* sigma, int32_t n_sink, int64_t m, int32_t* idx,
                    int32_t* count, int32_t cap, void* ws, size_t ws_bytes, void* stream) {
  g_err[0] = 0;
  if (B < 1 || N < 1 || N > MAX_N) return fail(VK_ERR_INVALID_ARG, "B >= 1 and 1 <= N <= %lld required", (long long)MAX_N);
  if (T < 1) return fail(VK_ERR_INVALID_ARG, "T must be >= 1");
  if (n_sink < 0 || m < 0) return fail(VK_ERR_INVALID_ARG, "n_sink and m must be >= 0");
  if (!sigma || !idx || !count) return fail(VK_ERR_INVALID_ARG, "sigma, idx and count must be non-NULL");
  const int64_t closed = (int64_t)(N / T) * T;
  const int64_t sinks = std::min<int64_t>(n_sink, closed);
  const int64_t k = std::min<int64_t>(m, closed - sinks);
  if ((int64_t)cap < sinks + k + (N - closed))
    return fail(VK_ERR_INVALID_ARG, "cap = %d < sinks + m + open tail = %lld", cap, (long long)(sinks + k + N - closed));
  if (!ws || ws_bytes < 256 || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(VK_ERR_WORKSPACE, "a 256-byte aligned workspace of at least 256 bytes is needed (status word)");
  // the selection of the per-head path with one "head" per sequence: the open tail is always kept like the recent
  // window, the sinks like the sinks, and the top m of the closed rows by (sigma desc, position asc)
  VK_CUDA(vk::launch_select_dense(B, 1, N, sigma, nullptr, k, (int)(N - closed), (int)sinks, idx, count, cap, 0,
                                  nullptr, nullptr, 0, static_cast<int*>(ws), static_cast<cudaStream_t>(stream)),
          "sigma select");
  return VK_OK;
}

int vk_poll_status(void* ws, void* stream) {
  g_err[0] = 0;
  if (!ws) return fail(VK_ERR_WORKSPACE, "workspace is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int code = 0;
  VK_CUDA(cudaStreamSynchronize(st), "poll: synchronize");
  VK_CUDA(cudaMemcpy(&code, ws, sizeof(int), cudaMemcpyDeviceToHost), "poll: read");
  VK_CUDA(cudaMemset(ws, 0, sizeof(int)), "poll: clear");
  if (code != 0) return fail(code, "device status %d", code);
  return VK_OK;
}

}  // extern "C"
