// k_sketch.cu -- the rank-r_sk content sketch of the recall trigger (Sec. 4.2, Eq. 4, Lemma 1).
//
// V (r_sk orthonormal directions of the 512-wide content space, the rows of basis [r_sk][512] fp32) splits the content
// logit: qc . L = (V qc) . (V L) + delta with |delta| <= |(I - V^T V) qc| |(I - V^T V) L|.
//   k_sketch_rows   index entry of every cached row: s_u = V L_u (bf16, round to nearest even) and eta_u =
//                   |L_u - V^T s_u| (with the fp32 s_u). Four rows per warp, lane l holding dims l + 32 i of each;
//                   the basis sits in shared memory, and each of its rows is read once for the four.
//   k_sketch_query  per (b, h): p = V qc (fp32, and its bf16 high and low parts in the [B][2][H][r_sk] layout the
//                   tensor-core trigger loads) and rho = |qc - V^T p|, the certificate's query norm.
//   basis from the context's queries (V from the prefix queries): the second moment M = sum_i q_i q_i^T in fp32
//   (k_sk_moment), orthogonal iteration X <- orth(M X) on one CTA with two Cholesky-QR passes per step
//   (k_sk_iterate), the Rayleigh-Ritz matrix X^T M X solved by the 64 x 64 fp64 Jacobi kernel of the PCA basis,
//   and the rotation of X into the Ritz vectors with the sign rule (entry of largest magnitude positive, ties the
//   smaller index) in k_sk_finish.
#include <algorithm>

#include "vk_common.cuh"

namespace vk {

namespace {

constexpr int SKR_RW = 4, SKR_NT = 256;             // rows per warp and threads per block of the index build

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// One 512-wide vector x (lane l holds x[l + 32 i]) against the basis rows in shared memory: s[j] = V_j . x for every j
// (lane j % 32 keeps s[j] in sv[j / 32]) and the residual norm |x - V^T s|.
__device__ __forceinline__ float project(const float* __restrict__ vb, int r_sk, const float (&x)[16], float (&sv)[2],
                                         int lane) {
  float res[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) res[i] = x[i];
  sv[0] = sv[1] = 0.f;
  for (int j = 0; j < r_sk; ++j) {
    const float* v = vb + j * D_LAT + lane;
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) acc = fmaf(v[32 * i], x[i], acc);
    acc = warp_sum(acc);
    if ((j & 31) == lane) sv[j >> 5] = acc;
#pragma unroll
    for (int i = 0; i < 16; ++i) res[i] = fmaf(-acc, v[32 * i], res[i]);
  }
  float e = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) e = fmaf(res[i], res[i], e);
  return sqrtf(warp_sum(e));
}

// RW rows per warp: each basis row is loaded from shared memory once for all of them, and their warp sums run side by
// side; every row takes the same operations in the same order as project() (the results do not depend on RW).
template <typename T, int RW, int NT>
__global__ void __launch_bounds__(NT) k_sketch_rows(int64_t rows, int N, int r_sk, const T* __restrict__ latent,
                                                    int64_t lld, int64_t lbs, const float* __restrict__ basis,
                                                    __nv_bfloat16* __restrict__ sketch, float* __restrict__ eta) {
  extern __shared__ float vb[];                       // [r_sk][512]
  for (int e = threadIdx.x; e < r_sk * D_LAT; e += blockDim.x) vb[e] = basis[e];
  __syncthreads();
  const int lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  const int64_t groups = (rows + RW - 1) / RW;
  for (int64_t g = (int64_t)blockIdx.x * warps + (threadIdx.x >> 5); g < groups; g += (int64_t)gridDim.x * warps) {
    float x[RW][16], res[RW][16], sv[RW][2];
#pragma unroll
    for (int q = 0; q < RW; ++q) {
      const int64_t row = g * RW + q;
      const int64_t rr = row < rows ? row : rows - 1;  // a short last group repeats a row and stores nothing for it
      const int64_t b = rr / N, u = rr - b * N;
      const T* L = latent + b * lbs + u * lld;
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        x[q][i] = to_f(L[lane + 32 * i]);
        res[q][i] = x[q][i];
      }
      sv[q][0] = sv[q][1] = 0.f;
    }
    for (int j = 0; j < r_sk; ++j) {
      const float* v = vb + j * D_LAT + lane;
      float vv[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) vv[i] = v[32 * i];
      float acc[RW];
#pragma unroll
      for (int q = 0; q < RW; ++q) {
        acc[q] = 0.f;
#pragma unroll
        for (int i = 0; i < 16; ++i) acc[q] = fmaf(vv[i], x[q][i], acc[q]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) {
#pragma unroll
        for (int q = 0; q < RW; ++q) acc[q] += __shfl_xor_sync(0xffffffffu, acc[q], o);
      }
#pragma unroll
      for (int q = 0; q < RW; ++q) {
        if ((j & 31) == lane) sv[q][j >> 5] = acc[q];
#pragma unroll
        for (int i = 0; i < 16; ++i) res[q][i] = fmaf(-acc[q], vv[i], res[q][i]);
      }
    }
#pragma unroll
    for (int q = 0; q < RW; ++q) {
      const int64_t row = g * RW + q;
      float e = 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) e = fmaf(res[q][i], res[q][i], e);
      e = sqrtf(warp_sum(e));
      if (row >= rows) continue;
      if (eta && lane == 0) eta[row] = e;
      if (sketch) {
        __nv_bfloat16* dst = sketch + row * r_sk;
        if (lane < r_sk) dst[lane] = __float2bfloat16_rn(sv[q][0]);
        if (lane + 32 < r_sk) dst[lane + 32] = __float2bfloat16_rn(sv[q][1]);
      }
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(512) k_sketch_query(int B, int H, int r_sk, const T* __restrict__ q_latent,
                                                      const float* __restrict__ basis, float* __restrict__ p,
                                                      __nv_bfloat16* __restrict__ phl, float* __restrict__ rho) {
  extern __shared__ float vb[];
  for (int e = threadIdx.x; e < r_sk * D_LAT; e += blockDim.x) vb[e] = basis[e];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t bh = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (bh >= (int64_t)B * H) return;
  const int64_t b = bh / H, h = bh - b * H;
  const T* q = q_latent + bh * D_LAT;
  float x[16], sv[2];
#pragma unroll
  for (int i = 0; i < 16; ++i) x[i] = to_f(q[lane + 32 * i]);
  const float e = project(vb, r_sk, x, sv, lane);
  if (lane == 0) rho[bh] = e;
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int j = lane + 32 * k;
    if (j >= r_sk) continue;
    const float v = sv[k];
    if (p) p[bh * r_sk + j] = v;
    if (phl) {
      const __nv_bfloat16 hi = __float2bfloat16_rn(v);
      const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
      phl[((b * 2 + 0) * H + h) * r_sk + j] = hi;
      phl[((b * 2 + 1) * H + h) * r_sk + j] = lo;
    }
  }
}

// ---------------------------------------------------------------------------------------------- basis
// M [512][512] fp32: block (bi, bj) computes the 32 x 32 tile M[32 bi .., 32 bj ..] over all queries, staging 64
// queries' two 32-dim slices at a time.
template <typename T>
__global__ void __launch_bounds__(256) k_sk_moment(int64_t n, const T* __restrict__ q, float* __restrict__ M) {
  __shared__ float qa[64][33], qb[64][33];
  const int bi = blockIdx.y, bj = blockIdx.x, t = threadIdx.x;
  const int ti = t >> 3, tj = (t & 7) * 4;            // this thread: row ti, columns tj .. tj + 3 of the tile
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int64_t q0 = 0; q0 < n; q0 += 64) {
    for (int e = t; e < 64 * 32; e += 256) {
      const int r = e >> 5, c = e & 31;
      const int64_t row = q0 + r;
      qa[r][c] = row < n ? to_f(q[row * D_LAT + 32 * bi + c]) : 0.f;
      qb[r][c] = row < n ? to_f(q[row * D_LAT + 32 * bj + c]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int r = 0; r < 64; ++r) {
      const float a = qa[r][ti];
#pragma unroll
      for (int k = 0; k < 4; ++k) acc[k] = fmaf(a, qb[r][tj + k], acc[k]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) M[(32 * bi + ti) * D_LAT + 32 * bj + tj + k] = acc[k];
}

constexpr int SKI_THREADS = 512;                   // one row of X per thread
constexpr int SK_LD = 64;                             // row stride of X and Y (r_sk <= 64)

// Y[i][c] = sum_k M[i][k] X[k][c] for c < r (thread t: row t; the warp reads one X row at a time, a broadcast);
// Y global.
__device__ void sk_mx(const float* __restrict__ M, const float* X, float* Y, int r) {
  const int i = threadIdx.x;
  float acc[SK_LD];
#pragma unroll
  for (int c = 0; c < SK_LD; ++c) acc[c] = 0.f;
  const float* mi = M + (int64_t)i * D_LAT;
  for (int k = 0; k < D_LAT; ++k) {
    const float m = mi[k];
    const float* xk = X + k * SK_LD;
#pragma unroll
    for (int c = 0; c < SK_LD; ++c) acc[c] = fmaf(m, xk[c], acc[c]);
  }
#pragma unroll
  for (int c = 0; c < SK_LD; ++c)
    if (c < r) Y[i * SK_LD + c] = acc[c];
  __syncthreads();
}

// The same product into X itself: each thread keeps its row of M X in registers until every thread is done reading X.
__device__ void sk_mx_inplace(const float* __restrict__ M, float* X, int r) {
  const int i = threadIdx.x;
  float acc[SK_LD];
#pragma unroll
  for (int c = 0; c < SK_LD; ++c) acc[c] = 0.f;
  const float* mi = M + (int64_t)i * D_LAT;
  for (int k = 0; k < D_LAT; ++k) {
    const float m = mi[k];
    const float* xk = X + k * SK_LD;
#pragma unroll
    for (int c = 0; c < SK_LD; ++c) acc[c] = fmaf(m, xk[c], acc[c]);
  }
  __syncthreads();
#pragma unroll
  for (int c = 0; c < SK_LD; ++c)
    if (c < r) X[i * SK_LD + c] = acc[c];
  __syncthreads();
}

// One Cholesky-QR pass: C = S^T S, C = L L^T, X = S L^-T (S and X [512][64], only r columns; X may be S). Returns false
// when a pivot is not positive (the columns are dependent).
__device__ bool sk_cholqr(const float* S, float* X, float* C /* [64][65] */, int r, int* bad) {
  const int t = threadIdx.x;
  for (int e = t; e < r * r; e += SKI_THREADS) {
    const int a = e / r, b = e - a * r;
    if (b > a) continue;
    float acc = 0.f;
    for (int i = 0; i < D_LAT; ++i) acc = fmaf(S[i * SK_LD + a], S[i * SK_LD + b], acc);
    C[a * 65 + b] = acc;
  }
  if (t == 0) *bad = 0;
  __syncthreads();
  for (int k = 0; k < r; ++k) {
    if (t == 0) {
      const float d = C[k * 65 + k];
      if (!(d > 0.f)) *bad = 1;
      C[k * 65 + k] = d > 0.f ? sqrtf(d) : 1.f;
    }
    __syncthreads();
    const float dk = C[k * 65 + k];
    for (int i = k + 1 + t; i < r; i += SKI_THREADS) C[i * 65 + k] /= dk;
    __syncthreads();
    const int m = r - k - 1;
    for (int e = t; e < m * m; e += SKI_THREADS) {
      const int i = k + 1 + e / m, j = k + 1 + e % m;
      if (j <= i) C[i * 65 + j] = fmaf(-C[i * 65 + k], C[j * 65 + k], C[i * 65 + j]);
    }
    __syncthreads();
  }
  {
    // row t: x L^T = s, forward substitution over the columns
    float x[SK_LD];
#pragma unroll
    for (int j = 0; j < SK_LD; ++j) {
      if (j < r) {
        float acc = S[t * SK_LD + j];
        for (int k = 0; k < j; ++k) acc = fmaf(-x[k], C[j * 65 + k], acc);
        x[j] = acc / C[j * 65 + j];
      }
    }
#pragma unroll
    for (int j = 0; j < SK_LD; ++j)
      if (j < r) X[t * SK_LD + j] = x[j];
  }
  __syncthreads();
  return *bad == 0;
}

// Orthogonal iteration on one CTA: X0 = orth(M G) with G a fixed +-1 pattern, then iters steps X <- orth(M X)
// (two Cholesky-QR passes each), then the Rayleigh-Ritz matrix R = X^T M X into Bout [64][64] fp64 (zero past r) and
// X into Xout [512][64].
__global__ void __launch_bounds__(SKI_THREADS, 1) k_sk_iterate(const float* __restrict__ M, int r, int iters,
                                                             float* __restrict__ Y, float* __restrict__ Xout,
                                                             double* __restrict__ Bout, int* __restrict__ status) {
  extern __shared__ float smf[];
  float* X = smf;                                     // [512][64]
  float* C = X + D_LAT * SK_LD;                       // [64][65]
  __shared__ int bad;
  const int t = threadIdx.x;
  for (int e = t; e < D_LAT * SK_LD; e += SKI_THREADS) {
    uint32_t h = (uint32_t)e * 2654435761u;           // Knuth's multiplicative hash, then a xorshift round
    h ^= h >> 15;
    h *= 2246822519u;
    h ^= h >> 13;
    X[e] = (h & 1u) ? 1.f : -1.f;
  }
  __syncthreads();
  bool ok = true;
  for (int it = 0; it <= iters && ok; ++it) {
    // the product stays in shared memory: both Cholesky-QR passes read their operand from there
    sk_mx_inplace(M, X, r);
    ok = sk_cholqr(X, X, C, r, &bad) && sk_cholqr(X, X, C, r, &bad);
  }
  if (!ok) {
    if (t == 0) raise_status(status, VK_ERR_INVALID_ARG);
    return;
  }
  sk_mx(M, X, Y, r);
  for (int e = t; e < 64 * 64; e += SKI_THREADS) {
    const int a = e >> 6, b = e & 63;
    double v = 0.0;
    if (a < r && b < r) {
      float acc = 0.f;
      for (int i = 0; i < D_LAT; ++i) acc = fmaf(X[i * SK_LD + a], Y[i * SK_LD + b], acc);
      v = acc;
    }
    Bout[e] = v;
  }
  for (int e = t; e < D_LAT * SK_LD; e += SKI_THREADS) Xout[e] = X[e];
}

// basis row i = sum_j W[i][j] X[:, j] (W: the Ritz rotation's rows, by decreasing eigenvalue), signed so that its
// entry of largest magnitude (ties: the smaller index) is positive. One block of 512 threads per row.
__global__ void __launch_bounds__(512) k_sk_finish(int r, const float* __restrict__ W, const float* __restrict__ X,
                                                  const float* __restrict__ eig64, float* __restrict__ basis,
                                                  float* __restrict__ eig) {
  __shared__ float bv[16];
  __shared__ int bi[16];
  const int i = blockIdx.x, d = threadIdx.x, lane = d & 31, w = d >> 5;
  float v = 0.f;
  for (int j = 0; j < r; ++j) v = fmaf(W[i * 64 + j], X[d * SK_LD + j], v);
  float a = fabsf(v);
  int at = d;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float oa = __shfl_xor_sync(0xffffffffu, a, o);
    const int ot = __shfl_xor_sync(0xffffffffu, at, o);
    if (oa > a || (oa == a && ot < at)) { a = oa; at = ot; }
  }
  if (lane == 0) { bv[w] = a; bi[w] = at; }
  __syncthreads();
  if (w == 0) {
    a = lane < 16 ? bv[lane] : -1.f;
    at = lane < 16 ? bi[lane] : D_LAT;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float oa = __shfl_xor_sync(0xffffffffu, a, o);
      const int ot = __shfl_xor_sync(0xffffffffu, at, o);
      if (oa > a || (oa == a && ot < at)) { a = oa; at = ot; }
    }
    if (lane == 0) bi[0] = at;
  }
  __syncthreads();
  const int big = bi[0];
  __shared__ float vbig;
  if (d == big) vbig = v;
  __syncthreads();
  basis[(int64_t)i * D_LAT + d] = vbig < 0.f ? -v : v;
  if (d == 0 && eig) eig[i] = eig64[i];
}

size_t vb_smem(int r_sk) { return sizeof(float) * (size_t)r_sk * D_LAT; }

template <typename F>
cudaError_t allow_smem(F kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace

cudaError_t launch_build_sketch(const vk_view& v, int r_sk, const float* basis, void* sketch, float* eta,
                                cudaStream_t st) {
  const int64_t rows = (int64_t)v.B * v.N;
  const size_t smem = vb_smem(r_sk);
  constexpr int RW = SKR_RW, NT = SKR_NT;
  const int64_t groups = (rows + RW - 1) / RW;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((groups + NT / 32 - 1) / (NT / 32), sm_count()));
  auto* sk = static_cast<__nv_bfloat16*>(sketch);
  cudaError_t e;
  if (v.dtype == VK_BF16) {
    auto kern = k_sketch_rows<__nv_bfloat16, RW, NT>;
    if ((e = allow_smem(kern, smem)) != cudaSuccess) return e;
    kern<<<grid, NT, smem, st>>>(rows, v.N, r_sk, static_cast<const __nv_bfloat16*>(v.latent), v.latent_ld,
                                 v.latent_bstride, basis, sk, eta);
  } else {
    auto kern = k_sketch_rows<float, RW, NT>;
    if ((e = allow_smem(kern, smem)) != cudaSuccess) return e;
    kern<<<grid, NT, smem, st>>>(rows, v.N, r_sk, static_cast<const float*>(v.latent), v.latent_ld, v.latent_bstride,
                                 basis, sk, eta);
  }
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_sketch_query(const vk_view& v, int r_sk, const float* basis, float* p, void* phl, float* rho,
                                cudaStream_t st) {
  const int64_t BH = (int64_t)v.B * v.H;
  const size_t smem = vb_smem(r_sk);
  // 16 queries per block: each block stages the basis (up to 128 KB) once for 16 warps
  const int grid = (int)((BH + 15) / 16);
  auto* hl = static_cast<__nv_bfloat16*>(phl);
  cudaError_t e;
  if (v.dtype == VK_BF16) {
    if ((e = allow_smem(k_sketch_query<__nv_bfloat16>, smem)) != cudaSuccess) return e;
    k_sketch_query<__nv_bfloat16><<<grid, 512, smem, st>>>(v.B, v.H, r_sk,
                                                          static_cast<const __nv_bfloat16*>(v.q_latent), basis, p, hl,
                                                          rho);
  } else {
    if ((e = allow_smem(k_sketch_query<float>, smem)) != cudaSuccess) return e;
    k_sketch_query<float><<<grid, 512, smem, st>>>(v.B, v.H, r_sk, static_cast<const float*>(v.q_latent), basis, p,
                                                  hl, rho);
  }
  count_launches(1);
  return cudaGetLastError();
}

// Workspace: status word, M [512][512] fp32, Y and X [512][64] fp32, the Ritz matrix [64][64] fp64, W [64][64] and
// the 64 Ritz values (fp32).
namespace {
struct SkLayout {
  static constexpr size_t m = 256;
  static constexpr size_t y = m + sizeof(float) * D_LAT * D_LAT;
  static constexpr size_t x = y + sizeof(float) * D_LAT * 64;
  static constexpr size_t bm = x + sizeof(float) * D_LAT * 64;
  static constexpr size_t w = bm + sizeof(double) * 64 * 64;
  static constexpr size_t e = w + sizeof(float) * 64 * 64;
  static constexpr size_t total = e + sizeof(float) * 64;
};
}  // namespace

size_t sketch_basis_ws_bytes() { return SkLayout::total; }

constexpr int SK_ITERS = 40;

cudaError_t launch_sketch_basis(const void* queries, int dtype, int64_t n, int r_sk, float* basis, float* eig,
                                void* ws, cudaStream_t st) {
  char* w = static_cast<char*>(ws);
  int* status = reinterpret_cast<int*>(w);
  float* M = reinterpret_cast<float*>(w + SkLayout::m);
  float* Y = reinterpret_cast<float*>(w + SkLayout::y);
  float* X = reinterpret_cast<float*>(w + SkLayout::x);
  double* Bm = reinterpret_cast<double*>(w + SkLayout::bm);
  float* W = reinterpret_cast<float*>(w + SkLayout::w);
  float* E = reinterpret_cast<float*>(w + SkLayout::e);
  cudaError_t e;
  dim3 mg(D_LAT / 32, D_LAT / 32);
  if (dtype == VK_BF16)
    k_sk_moment<__nv_bfloat16><<<mg, 256, 0, st>>>(n, static_cast<const __nv_bfloat16*>(queries), M);
  else
    k_sk_moment<float><<<mg, 256, 0, st>>>(n, static_cast<const float*>(queries), M);
  const size_t ismem = sizeof(float) * (D_LAT * SK_LD + 64 * 65);
  if ((e = allow_smem(k_sk_iterate, ismem)) != cudaSuccess) return e;
  k_sk_iterate<<<1, SKI_THREADS, ismem, st>>>(M, r_sk, SK_ITERS, Y, X, Bm, status);
  if ((e = launch_sym_eig64(Bm, W, E, st)) != cudaSuccess) return e;
  k_sk_finish<<<r_sk, 512, 0, st>>>(r_sk, W, X, E, basis, eig);
  count_launches(3);
  return cudaGetLastError();
}

}  // namespace vk
