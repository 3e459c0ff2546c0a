// k_index.cu -- query preparation, the per-cache index build, SIMT scoring and the dense trigger scan.
//
// Query prep (Eq. 4 inputs): qt_h = O Qr_h (or Qr_h when r = 64), |Qc_h|, |(O Qr_h)[r:]|, |Qr_h|.
// Index build (Sec. 4.2 index entry with sketch rank 0): digest = bf16((O K_u)[0:r]), eta_u = |L_u|,
// page_res[page] = max_u |(O K_u)[r:64]|, and the page maxima of |K_u| and eta_u (the page-level bound).
// Page trigger (reading B): every archived row outside S_h of a page whose bound beats s*_h fires.
// SIMT scoring: a[h,u] = qt_h[0:r] . key_u[0:r] (fp32) for fp32 caches, digests and small problems.
// Dense trigger (Eq. 4, Lemma 2): T = lambda (a + |(O Qr)[r:]| page_res + z_eff |Qc| eta) > s*_h; with a content
// sketch, T = lambda (a + |(O Qr)[r:]| page_res + p_h . s_u + z_eff rho_h eta_u) (rho_h passed as |Qc|).
#include "vk_common.cuh"

namespace vk {

template <typename T>
__host__ __device__ __forceinline__ const T* tptr(const void* p) { return reinterpret_cast<const T*>(p); }

// ---------------------------------------------------------------------------------------------- query prep
// One warp per (b, h); lane l owns RoPE coordinates l and l + 32. With a digest the block first stages the 64 x 64
// rotation in shared memory (transposed and padded, so that the lanes' reads of one column hit distinct banks).
template <typename T>
__global__ void k_qprep(const T* __restrict__ q_latent, const T* __restrict__ q_rope, int BH, int H, int r,
                        const float* __restrict__ rot, float* __restrict__ qt, float* __restrict__ qcn,
                        float* __restrict__ qrn, float* __restrict__ qrf, __nv_bfloat16* __restrict__ qhl) {
  __shared__ float rot_t[D_ROPE][D_ROPE + 1];        // rot_t[i][j] = O[j][i]
  if (r < D_ROPE) {
    for (int e = threadIdx.x; e < D_ROPE * D_ROPE; e += blockDim.x) rot_t[e % D_ROPE][e / D_ROPE] = rot[e];
    __syncthreads();
  }
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= BH) return;
  const T* qc = q_latent + (int64_t)warp * D_LAT;
  const T* qr = q_rope + (int64_t)warp * D_ROPE;
  float ss = 0.f;
  for (int j = lane; j < D_LAT; j += 32) { float x = to_f(qc[j]); ss = fmaf(x, x, ss); }
  for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  float q0 = to_f(qr[lane]), q1 = to_f(qr[lane + 32]);
  float qq = fmaf(q1, q1, q0 * q0);
  for (int o = 16; o; o >>= 1) qq += __shfl_xor_sync(0xffffffffu, qq, o);
  float y0 = q0, y1 = q1;
  if (r < D_ROPE) {
    // y_j = sum_i O[j][i] q_i ; lane owns outputs j = lane and lane + 32.
    y0 = 0.f; y1 = 0.f;
    for (int i = 0; i < D_ROPE; ++i) {
      float qi = __shfl_sync(0xffffffffu, i < 32 ? q0 : q1, i & 31);
      y0 = fmaf(rot_t[i][lane], qi, y0);
      y1 = fmaf(rot_t[i][lane + 32], qi, y1);
    }
  }
  float res = 0.f;
  if (r < D_ROPE) {
    if (lane >= r) res = fmaf(y0, y0, res);
    if (lane + 32 >= r) res = fmaf(y1, y1, res);
  }
  for (int o = 16; o; o >>= 1) res += __shfl_xor_sync(0xffffffffu, res, o);
  qt[(int64_t)warp * D_ROPE + lane] = y0;
  qt[(int64_t)warp * D_ROPE + lane + 32] = y1;
  if (qhl && r < D_ROPE) {
    // the tensor-core query operand: high part bf16(y), low part bf16(y - high), zero past r (up to 16)
    const int kp = r < 16 ? 16 : r, b = warp / H, h = warp - b * H;
    __nv_bfloat16* hi = qhl + ((int64_t)(2 * b) * H + h) * kp;
    __nv_bfloat16* lo = qhl + ((int64_t)(2 * b + 1) * H + h) * kp;
    for (int j = lane; j < kp; j += 32) {
      const float y = j < r ? (j < 32 ? y0 : y1) : 0.f;
      const __nv_bfloat16 yh = __float2bfloat16_rn(y);
      hi[j] = yh;
      lo[j] = __float2bfloat16_rn(y - __bfloat162float(yh));
    }
  }
  if (lane == 0) {
    qcn[warp] = sqrtf(ss);
    qrn[warp] = sqrtf(res);
    if (qrf) qrf[warp] = sqrtf(qq);
  }
}

cudaError_t launch_qprep(const vk_view& v, int r, const float* rot, float* qt, float* qcn, float* qrn, float* qrf,
                         __nv_bfloat16* qhl, cudaStream_t st) {
  const int BH = v.B * v.H, threads = 256, blocks = (BH * 32 + threads - 1) / threads;
  if (v.dtype == VK_BF16)
    k_qprep<__nv_bfloat16><<<blocks, threads, 0, st>>>(tptr<__nv_bfloat16>(v.q_latent), tptr<__nv_bfloat16>(v.q_rope),
                                                       BH, v.H, r, rot, qt, qcn, qrn, qrf, qhl);
  else
    k_qprep<float><<<blocks, threads, 0, st>>>(tptr<float>(v.q_latent), tptr<float>(v.q_rope), BH, v.H, r, rot, qt,
                                               qcn, qrn, qrf, qhl);
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- index build
// One warp per row: lane owns latent coords [16 lane, 16 lane + 16) and RoPE coords lane, lane + 32.
template <typename T>
__global__ void k_build_digest(const T* __restrict__ latent, int64_t lld, int64_t lbs, const T* __restrict__ rope,
                               int64_t rld, int64_t rbs, int N, int64_t total_rows, int r,
                               const float* __restrict__ rot, __nv_bfloat16* __restrict__ digest,
                               float* __restrict__ eta, float* __restrict__ page_res, float* __restrict__ page_knorm,
                               float* __restrict__ page_eta) {
  __shared__ float rot_t[D_ROPE][D_ROPE + 1];        // rot_t[i][j] = O[j][i] (staged once per block)
  if (r < D_ROPE) {
    for (int e = threadIdx.x; e < D_ROPE * D_ROPE; e += blockDim.x) rot_t[e % D_ROPE][e / D_ROPE] = rot[e];
    __syncthreads();
  }
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= total_rows) return;
  const int64_t b = row / N, u = row % N;
  const T* L = latent + b * lbs + u * lld;
  const T* K = rope + b * rbs + u * rld;
  const int64_t page = b * ((N + PAGE - 1) / PAGE) + u / PAGE;
  // norms are >= 0, so their float bit patterns order like unsigned integers (atomicMax on the bits)
  if (eta || page_eta) {
    float ss = 0.f;
    for (int j = lane; j < D_LAT; j += 32) { float x = to_f(L[j]); ss = fmaf(x, x, ss); }
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0 && eta) eta[row] = sqrtf(ss);
    if (lane == 0 && page_eta) atomicMax(reinterpret_cast<unsigned int*>(page_eta) + page, __float_as_uint(sqrtf(ss)));
  }
  if (page_knorm) {
    const float k0 = to_f(K[lane]), k1 = to_f(K[lane + 32]);
    float kk = fmaf(k1, k1, k0 * k0);
    for (int o = 16; o; o >>= 1) kk += __shfl_xor_sync(0xffffffffu, kk, o);
    if (lane == 0) atomicMax(reinterpret_cast<unsigned int*>(page_knorm) + page, __float_as_uint(sqrtf(kk)));
  }
  if (r < D_ROPE) {
    float k0 = to_f(K[lane]), k1 = to_f(K[lane + 32]);
    float y0 = 0.f, y1 = 0.f;
    for (int i = 0; i < D_ROPE; ++i) {
      float ki = __shfl_sync(0xffffffffu, i < 32 ? k0 : k1, i & 31);
      y0 = fmaf(rot_t[i][lane], ki, y0);
      y1 = fmaf(rot_t[i][lane + 32], ki, y1);
    }
    if (digest) {
      if (lane < r) digest[row * r + lane] = __float2bfloat16_rn(y0);
      if (lane + 32 < r) digest[row * r + lane + 32] = __float2bfloat16_rn(y1);
    }
    float res = 0.f;
    if (lane >= r) res = fmaf(y0, y0, res);
    if (lane + 32 >= r) res = fmaf(y1, y1, res);
    for (int o = 16; o; o >>= 1) res += __shfl_xor_sync(0xffffffffu, res, o);
    if (page_res && lane == 0) atomicMax(reinterpret_cast<unsigned int*>(page_res) + page, __float_as_uint(sqrtf(res)));
  }
}

cudaError_t launch_build_digest(const vk_view& v, int r, const float* rot, __nv_bfloat16* digest, float* eta,
                                float* page_res, float* page_knorm, float* page_eta, cudaStream_t st) {
  const int64_t rows = (int64_t)v.B * v.N;
  const int wpb = 8;
  const int64_t blocks = (rows + wpb - 1) / wpb;
  const size_t page_bytes = sizeof(float) * v.B * ((v.N + PAGE - 1) / PAGE);
  for (float* pg : {page_res, page_knorm, page_eta}) {
    if (!pg) continue;
    cudaError_t e = cudaMemsetAsync(pg, 0, page_bytes, st);
    if (e != cudaSuccess) return e;
  }
  if (!digest && !page_res) r = D_ROPE;   // no digest output: the rotation is not needed
  if (!eta && !page_knorm && !page_eta && r == D_ROPE) return cudaSuccess;
  if (v.dtype == VK_BF16)
    k_build_digest<__nv_bfloat16><<<(unsigned)blocks, wpb * 32, 0, st>>>(
        tptr<__nv_bfloat16>(v.latent), v.latent_ld, v.latent_bstride, tptr<__nv_bfloat16>(v.rope), v.rope_ld,
        v.rope_bstride, v.N, rows, r, rot, digest, eta, page_res, page_knorm, page_eta);
  else
    k_build_digest<float><<<(unsigned)blocks, wpb * 32, 0, st>>>(
        tptr<float>(v.latent), v.latent_ld, v.latent_bstride, tptr<float>(v.rope), v.rope_ld, v.rope_bstride, v.N,
        rows, r, rot, digest, eta, page_res, page_knorm, page_eta);
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- SIMT score
// CTA = (tile of 128 rows, sequence b). Keys staged as fp32 [128][r+1] (padded against bank conflicts),
// the H query rows as fp32 [H][r]. Thread t computes (h, u) pairs with u fastest, so writes are coalesced.
constexpr int SC_TILE = 128;

template <typename T>
__global__ void k_score_simt(const T* __restrict__ rope, int64_t rld, int64_t rbs,
                             const __nv_bfloat16* __restrict__ digest, int r, int N, int H,
                             const float* __restrict__ qt, float* __restrict__ scores) {
  extern __shared__ float sm[];
  const int b = blockIdx.y, u0 = blockIdx.x * SC_TILE;
  const int rp = r + 1;
  float* keys = sm;                       // [SC_TILE][rp]
  float* q = sm + SC_TILE * rp;           // [H][r]
  for (int i = threadIdx.x; i < SC_TILE * r; i += blockDim.x) {
    const int j = i / r, d = i % r, u = u0 + j;
    float x = 0.f;
    if (u < N) x = (r == D_ROPE) ? to_f(rope[(int64_t)b * rbs + (int64_t)u * rld + d])
                                 : __bfloat162float(digest[((int64_t)b * N + u) * r + d]);
    keys[j * rp + d] = x;
  }
  for (int i = threadIdx.x; i < H * r; i += blockDim.x) {
    const int h = i / r, d = i % r;
    q[i] = qt[((int64_t)b * H + h) * D_ROPE + d];
  }
  __syncthreads();
  for (int p = threadIdx.x; p < H * SC_TILE; p += blockDim.x) {
    const int h = p / SC_TILE, j = p % SC_TILE, u = u0 + j;
    if (u >= N) continue;
    const float* kr = keys + j * rp;
    const float* qh = q + h * r;
    float acc = 0.f;
    for (int d = 0; d < r; ++d) acc = fmaf(qh[d], kr[d], acc);
    scores[((int64_t)b * H + h) * N + u] = acc;
  }
}

cudaError_t launch_score_simt(const vk_view& v, int r, const float* qt, const __nv_bfloat16* digest,
                              float* scores, cudaStream_t st) {
  dim3 grid((v.N + SC_TILE - 1) / SC_TILE, v.B);
  const size_t smem = sizeof(float) * (SC_TILE * (r + 1) + (size_t)v.H * r);
  static bool attr_set[2] = {false, false};
  if (v.dtype == VK_BF16) {
    if (!attr_set[0]) {
      cudaError_t e = cudaFuncSetAttribute(k_score_simt<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           200 * 1024);
      if (e != cudaSuccess) return e;
      attr_set[0] = true;
    }
    k_score_simt<__nv_bfloat16><<<grid, 256, smem, st>>>(tptr<__nv_bfloat16>(v.rope), v.rope_ld, v.rope_bstride,
                                                         digest, r, v.N, v.H, qt, scores);
  } else {
    if (!attr_set[1]) {
      cudaError_t e = cudaFuncSetAttribute(k_score_simt<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
      if (e != cudaSuccess) return e;
      attr_set[1] = true;
    }
    k_score_simt<float><<<grid, 256, smem, st>>>(tptr<float>(v.rope), v.rope_ld, v.rope_bstride, digest, r, v.N,
                                                 v.H, qt, scores);
  }
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- dense trigger
// CTA = (word block, (b,h)). Thread t evaluates 32 consecutive positions (one bitmap word) of one head:
// archived rows not already selected whose trigger score beats s*_h set a bit in the fired bitmap. With
// top_j > 0 the trigger score replaces the row's score (non-fired rows get -inf) for the later top_j select.
__global__ void k_trigger_dense(int H, int N, int W, int n_sink, float lam, float z_eff, int top_j,
                                float* __restrict__ scores, const float* __restrict__ qcn,
                                const float* __restrict__ qrn, const float* __restrict__ eta,
                                const float* __restrict__ page_res, const float* __restrict__ smax1,
                                const uint32_t* __restrict__ selbm, uint32_t* __restrict__ firebm, int64_t nw,
                                long long* __restrict__ nfired, int r_sk, const __nv_bfloat16* __restrict__ sketch,
                                const float* __restrict__ skp) {
  const int64_t bh = blockIdx.y;
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= nw) return;
  const int64_t b = bh / H;
  const int64_t P = (N + PAGE - 1) / PAGE;
  const float sstar = smax1[bh], cq = qrn[bh], cz = z_eff * qcn[bh];
  const uint32_t sel = selbm[bh * nw + w];
  float* a = scores + bh * N;
  uint32_t bits = 0;
  for (int i = 0; i < 32; ++i) {
    const int64_t u = w * 32 + i;
    if (u >= N) break;
    const bool arch = (u >= n_sink) && (u < (int64_t)N - W);
    bool fire = false;
    float t = -INFINITY;
    if (arch && !((sel >> i) & 1u)) {
      float skt = 0.f;                               // the content sketch term p_h . s_u (Eq. 4), r_sk > 0
      for (int j = 0; j < r_sk; ++j) skt = fmaf(skp[bh * r_sk + j], __bfloat162float(sketch[(b * N + u) * r_sk + j]), skt);
      t = lam * (a[u] + cq * page_res[b * P + u / PAGE] + skt + cz * eta[b * N + u]);
      fire = t > sstar;
    }
    if (fire) bits |= 1u << i;
    if (top_j > 0) a[u] = fire ? t : -INFINITY;
  }
  firebm[bh * nw + w] = bits;
  if (bits) atomicAdd(reinterpret_cast<unsigned long long*>(nfired) + bh, (unsigned long long)__popc(bits));
}

cudaError_t launch_trigger_dense(int B, int H, int N, int W, int n_sink, float lam, float z_eff, int top_j,
                                 float* scores, const float* qcn, const float* qrn, const float* eta,
                                 const float* page_res, const float* smax1, const uint32_t* selbm,
                                 uint32_t* firebm, int64_t nw, int64_t* nfired, cudaStream_t st, int r_sk,
                                 const void* sketch, const float* skp) {
  cudaError_t e = cudaMemsetAsync(nfired, 0, sizeof(int64_t) * B * H, st);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((nw + 127) / 128), B * H);
  k_trigger_dense<<<grid, 128, 0, st>>>(H, N, W, n_sink, lam, z_eff, top_j, scores, qcn, qrn, eta, page_res, smax1,
                                        selbm, firebm, nw, reinterpret_cast<long long*>(nfired), r_sk,
                                        static_cast<const __nv_bfloat16*>(sketch), skp);
  count_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------- page trigger
// Reading B of the trigger: one block per (b, h). A 64-row page P fires for head h when
// lambda (|Qr_h| page_knorm[P] + z_eff |Qc_h| page_eta[P]) > s*_h; its archived rows outside S_h join F_h. Each
// thread takes whole bitmap words (two per page). Without top_j the fired words go straight into the fired bitmap;
// with top_j every fired row is also listed as a candidate (position, page bound) for the top_j selection, the
// list's order fixed by a block-wide scan of the threads' counts.
constexpr int PT_THREADS = 256;
__global__ void __launch_bounds__(PT_THREADS) k_trigger_page(int H, int N, int W, int n_sink, float lam, float z_eff,
                                                             const float* __restrict__ qcn, const float* __restrict__ qrf,
                                                             const float* __restrict__ page_knorm,
                                                             const float* __restrict__ page_eta,
                                                             const float* __restrict__ smax1,
                                                             const uint32_t* __restrict__ selbm,
                                                             uint32_t* __restrict__ firebm, int64_t nw, int top_j,
                                                             int* __restrict__ fcnt, int2* __restrict__ fcand,
                                                             int fcap) {
  __shared__ int scan_scratch[33];
  const int64_t bh = blockIdx.x;
  const int64_t b = bh / H;
  const int64_t P = (N + PAGE - 1) / PAGE;
  const float sstar = smax1[bh], cq = qrf[bh], cz = z_eff * qcn[bh];
  const int lo = n_sink, hi = N - W;
  const uint32_t* sel = selbm + bh * nw;
  uint32_t* fire = firebm + bh * nw;
  int base = 0;
  for (int64_t w0 = 0; w0 < nw; w0 += PT_THREADS) {
    const int64_t w = w0 + threadIdx.x;
    uint32_t bits = 0u;
    float bound = 0.f;
    if (w < nw) {
      const int64_t pg = b * P + (w * 32) / PAGE;
      bound = lam * (cq * page_knorm[pg] + cz * page_eta[pg]);
      if (bound > sstar) {
        const int r0 = (int)(w * 32);
        const int a = max(lo - r0, 0), e = min(min(hi, N) - r0, 32);
        if (e > a) {
          const uint32_t upto = e >= 32 ? 0xffffffffu : ((1u << e) - 1u);
          bits = (upto & ~((1u << a) - 1u)) & ~sel[w];
        }
      }
      if (top_j == 0) fire[w] = bits;
    }
    if (top_j > 0) {
      int tot;
      const int pos = base + block_exclusive_scan(__popc(bits), scan_scratch, &tot);
      int p = pos;
      for (uint32_t m = bits; m; m &= m - 1, ++p)
        if (p < fcap) fcand[bh * (int64_t)fcap + p] = make_int2((int)(w * 32) + __ffs(m) - 1, __float_as_int(bound));
      base += tot;
    }
  }
  if (top_j > 0 && threadIdx.x == 0) fcnt[bh] = base;
}

cudaError_t launch_trigger_page(int B, int H, int N, int W, int n_sink, float lam, float z_eff, const float* qcn,
                                const float* qrf, const float* page_knorm, const float* page_eta, const float* smax1,
                                const uint32_t* selbm, uint32_t* firebm, int64_t nw, int top_j, int* fcnt,
                                int2* fcand, int fcap, cudaStream_t st) {
  k_trigger_page<<<B * H, PT_THREADS, 0, st>>>(H, N, W, n_sink, lam, z_eff, qcn, qrf, page_knorm, page_eta, smax1,
                                               selbm, firebm, nw, top_j, fcnt, fcand, fcap);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
