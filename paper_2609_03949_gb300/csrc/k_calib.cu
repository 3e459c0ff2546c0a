// k_calib.cu -- conformal calibration of the trigger's certificate multiplier z (Sec. 4.2; Sec. 5).
//
// Every (b, h) of a batch is one calibration query. Its exact max logit over all cached rows and that row u* come
// from the tensor-core attention run over every row (its ARG instantiation, one partial per CTA); the query is hard
// when u* lies outside its attended set S_h. For a hard query the required inflation is
//   zq = (s* - idx_t) / cert_t,  idx_t = lambda (a[h,u*] + |(O Qr_h)[r:]| page_res[page(u*)]),
//                                cert_t = lambda |Qc_h| eta_u* / sqrt(d_c),  d_c = 512 (sketch rank 0),
// with s* the max logit over S_h. With a rank-r_sk content sketch the index part gains p_h . s_u* and the certificate
// is lambda rho_h eta_u* / sqrt(d_c - r_sk) (eta the sketch residual). z is then the ceil((n+1) tau_s)-th smallest zq
// over the n hard queries (tau_s = tau / (1 - alpha), alpha = (1 - tau)/2), Z_max when n < min_hard =
// ceil(tau_s / (1 - tau_s)) or the index passes n, clamped to [0, Z_max]; z_eff = z / sqrt(d_c - r_sk) is the decode
// step's parameter.
#include <cmath>

#include "vk_common.cuh"

namespace vk {

namespace {

__global__ void k_calib_zq(int B, int H, int N, AttnGeom g, int slot0, int nslot, const float* __restrict__ part_ml,
                           const int* __restrict__ part_arg, const float* __restrict__ smax1,
                           const uint32_t* __restrict__ selbm, int64_t nw, int r, const float* __restrict__ qt,
                           const float* __restrict__ qcn, const float* __restrict__ qrn,
                           const __nv_bfloat16* __restrict__ rope, int64_t rld, int64_t rbs,
                           const __nv_bfloat16* __restrict__ digest, const float* __restrict__ eta,
                           const float* __restrict__ page_res, float lam, int r_sk, const float* __restrict__ skp,
                           const __nv_bfloat16* __restrict__ sketch, const float* __restrict__ rho,
                           float* __restrict__ zq) {
  const int64_t bh = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (bh >= (int64_t)B * H) return;
  const int b = (int)(bh / H), h = (int)(bh - (int64_t)b * H);
  const long long seg = (long long)b * g.n_hg + h / HG;
  const int nv = attn_nvalid(g, seg);
  float best = -INFINITY;
  int pos = 0;
  for (int i = 0; i < nv; ++i) {                     // the partials cover increasing rows: an earlier one keeps a tie
    const int64_t pi = ((int64_t)b * nslot + slot0 + i) * H + h;
    const float v = part_ml[pi * 2];
    if (v > best) { best = v; pos = part_arg[pi]; }
  }
  const bool in_set = (selbm[bh * nw + (pos >> 5)] >> (pos & 31)) & 1u;
  if (in_set || best == -INFINITY) {
    zq[bh] = NAN;
    return;
  }
  float a = 0.f;
  const float* q = qt + bh * D_ROPE;
  if (r == D_ROPE) {
    const __nv_bfloat16* k = rope + (int64_t)b * rbs + (int64_t)pos * rld;
    for (int j = 0; j < D_ROPE; ++j) a = fmaf(q[j], __bfloat162float(k[j]), a);
  } else {
    const __nv_bfloat16* d = digest + ((int64_t)b * N + pos) * r;
    for (int j = 0; j < r; ++j) a = fmaf(q[j], __bfloat162float(d[j]), a);
  }
  for (int j = 0; j < r_sk; ++j)
    a = fmaf(skp[bh * r_sk + j], __bfloat162float(sketch[((int64_t)b * N + pos) * r_sk + j]), a);
  const int64_t P = (N + PAGE - 1) / PAGE;
  const float idx_t = lam * (a + qrn[bh] * page_res[(int64_t)b * P + pos / PAGE]);
  const float cq = r_sk > 0 ? rho[bh] : qcn[bh];
  const float cert_t = lam * cq * eta[(int64_t)b * N + pos] * (1.0f / sqrtf((float)(D_LAT - r_sk)));
  zq[bh] = (smax1[bh] - idx_t) / cert_t;
}

// One block: the hard queries' zq (NaN marks the others) gathered into shared memory, sorted (bitonic, padded with
// +inf to a power of two), and the order statistic taken. out = {z, z / sqrt(d_c), n_hard}.
constexpr int CQ_THREADS = 1024;
__global__ void __launch_bounds__(CQ_THREADS) k_conformal_quantile(int64_t BH, const float* __restrict__ zq,
                                                                 double tau_s, int min_hard, float z_max,
                                                                 int r_sk, float* __restrict__ out) {
  extern __shared__ float vals[];
  __shared__ int cnt;
  if (threadIdx.x == 0) cnt = 0;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < BH; i += CQ_THREADS) {
    const float v = zq[i];
    if (!isnan(v)) vals[atomicAdd(&cnt, 1)] = v;
  }
  __syncthreads();
  const int n = cnt;
  int np2 = 1;
  while (np2 < n) np2 <<= 1;
  for (int i = n + threadIdx.x; i < np2; i += CQ_THREADS) vals[i] = INFINITY;
  __syncthreads();
  for (int size = 2; size <= np2; size <<= 1)
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < np2; i += CQ_THREADS) {
        const int j = i ^ stride;
        if (j > i) {
          const bool up = (i & size) == 0;
          const float x = vals[i], y = vals[j];
          if ((x > y) == up) { vals[i] = y; vals[j] = x; }
        }
      }
      __syncthreads();
    }
  if (threadIdx.x == 0) {
    float z = z_max;
    if (n >= min_hard) {
      const long long k = (long long)ceil((double)(n + 1) * tau_s - 1e-9);
      if (k >= 1 && k <= n) z = fminf(fmaxf(vals[k - 1], 0.f), z_max);
    }
    out[0] = z;
    out[1] = z * (1.0f / sqrtf((float)(D_LAT - r_sk)));
    out[2] = (float)n;
  }
}

}  // namespace

size_t conformal_smem_bytes(int64_t BH) {
  int64_t np2 = 1;
  while (np2 < BH) np2 <<= 1;
  return (size_t)np2 * sizeof(float);
}

cudaError_t launch_calib(const vk_view& v, int r, const AttnGeom& g, int slot0, int nslot, const float* part_ml,
                         const int* part_arg, const float* smax1, const uint32_t* selbm, int64_t nw, const float* qt,
                         const float* qcn, const float* qrn, const void* digest, const float* eta,
                         const float* page_res, float lam, double tau_s, int min_hard, float z_max, float* zq,
                         float* z_out, cudaStream_t st, int r_sk, const float* skp, const void* sketch,
                         const float* rho) {
  const int64_t BH = (int64_t)v.B * v.H;
  k_calib_zq<<<(unsigned)((BH + 127) / 128), 128, 0, st>>>(
      v.B, v.H, v.N, g, slot0, nslot, part_ml, part_arg, smax1, selbm, nw, r, qt, qcn, qrn,
      static_cast<const __nv_bfloat16*>(v.rope), v.rope_ld, v.rope_bstride, static_cast<const __nv_bfloat16*>(digest),
      eta, page_res, lam, r_sk, skp, static_cast<const __nv_bfloat16*>(sketch), rho, zq);
  const size_t smem = conformal_smem_bytes(BH);
  cudaError_t e = cudaFuncSetAttribute(k_conformal_quantile, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_conformal_quantile<<<1, CQ_THREADS, smem, st>>>(BH, zq, tau_s, min_hard, z_max, r_sk, z_out);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace vk
