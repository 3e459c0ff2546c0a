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
//   (k_sk_iterate), the Rayleigh-Ritz matrix X^T M X solved by the 64 x 64 Jacobi kernel of the PCA basis (fp64 result),
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
constexpr int SK_LD = 64;                             // row length of X and Y (r_sk <= 64)
constexpr int SK_XLD = 68;                            // row stride of X and of L's rows in shared memory

// X [512][64] sits in shared memory with rows 68 floats apart: chunk q (16 bytes) of row i is 16-byte unit 17 i + q,
// so threads of a quarter-warp that read or write their own rows chunk by chunk meet distinct banks, and a warp
// reading one row (a broadcast) reads 16 contiguous chunks. The rows of the Cholesky factor L use the same stride.
__device__ __forceinline__ int sx_chunk(int i, int q) { return i * (SK_XLD / 4) + q; }
__device__ __forceinline__ int sx(int i, int c) { return i * SK_XLD + c; }

// acc[c] = sum_k M[i][k] X[k][c] for thread i's row, k ascending. M is symmetric (its tiles (a, b) and (b, a) sum the
// same products in the same order), so column i is read: one coalesced load per k for the warp. The warp reads one
// X row at a time, a broadcast.
__device__ __forceinline__ void sk_mx_row(const float* __restrict__ M, const float* X, float (&acc)[SK_LD]) {
  const int i = threadIdx.x;
#pragma unroll
  for (int c = 0; c < SK_LD; ++c) acc[c] = 0.f;
  const float4* X4 = reinterpret_cast<const float4*>(X);
  // M's entries are loaded four k ahead of their use (each k is a new line for the warp)
  float m0 = M[i], m1 = M[D_LAT + i], m2 = M[2 * D_LAT + i], m3 = M[3 * D_LAT + i];
#pragma unroll 1
  for (int k = 0; k < D_LAT; ++k) {
    const float m = m0;
    m0 = m1;
    m1 = m2;
    m2 = m3;
    m3 = k + 4 < D_LAT ? M[(int64_t)(k + 4) * D_LAT + i] : 0.f;
    const float4* xk = X4 + sx_chunk(k, 0);
#pragma unroll
    for (int q = 0; q < SK_LD / 4; ++q) {
      const float4 x = xk[q];
      acc[4 * q + 0] = fmaf(m, x.x, acc[4 * q + 0]);
      acc[4 * q + 1] = fmaf(m, x.y, acc[4 * q + 1]);
      acc[4 * q + 2] = fmaf(m, x.z, acc[4 * q + 2]);
      acc[4 * q + 3] = fmaf(m, x.w, acc[4 * q + 3]);
    }
  }
}

// Y = M X (columns c < r) into global memory, row-major [512][64].
__device__ void sk_mx(const float* __restrict__ M, const float* X, float* Y, int r) {
  const int i = threadIdx.x;
  float acc[SK_LD];
  sk_mx_row(M, X, acc);
#pragma unroll
  for (int c = 0; c < SK_LD; ++c)
    if (c < r) Y[i * SK_LD + c] = acc[c];
  __syncthreads();
}

// The same product into X itself: each thread keeps its row of M X in registers until every thread is done reading X
// (r is a multiple of 16, so whole chunks are written).
__device__ void sk_mx_inplace(const float* __restrict__ M, float* X, int r) {
  const int i = threadIdx.x;
  float acc[SK_LD];
  sk_mx_row(M, X, acc);
  __syncthreads();
  float4* X4 = reinterpret_cast<float4*>(X);
#pragma unroll
  for (int q = 0; q < SK_LD / 4; ++q)
    if (4 * q < r) X4[sx_chunk(i, q)] = make_float4(acc[4 * q], acc[4 * q + 1], acc[4 * q + 2], acc[4 * q + 3]);
  __syncthreads();
}

// Shared scratch of a Cholesky-QR pass: the Gram matrix C [64][65] (lower triangle), the factor L twice (rows at the
// stride of X for the substitution, columns contiguous for the trailing update) and its diagonal.
struct SkChol {
  float* C;
  float* Lr;
  float* Lc;
  float* Dg;
};

// One Cholesky-QR pass on X in place, first r columns: C = X^T X, C = L L^T, X <- X L^-T. Returns false when a pivot
// is not positive (the columns are dependent). Each entry of C sums over the rows in ascending order; column k of L
// is C's column k over the square root of the pivot, and the trailing update subtracts l_ik l_jk; each row of
// X L^-T is solved by forward substitution, k ascending.
__device__ bool sk_cholqr(float* X, const SkChol& w, int r, int* bad) {
  const int t = threadIdx.x;
  float* C = w.C;
  // Gram matrix: thread t takes rows a0, a0 + 1 and columns b0 .. b0 + 3 of C, tiles wholly above the diagonal idle
  {
    const int a0 = (t >> 4) * 2, b0 = (t & 15) * 4;
    if (b0 <= a0 + 1 && a0 < r && b0 < r) {
      float acc[2][4];
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = 0.f;
      const float4* X4 = reinterpret_cast<const float4*>(X);
#pragma unroll 4
      for (int i = 0; i < D_LAT; ++i) {
        const float4 xb = X4[sx_chunk(i, b0 >> 2)];
        const float2 xa = *reinterpret_cast<const float2*>(X + sx(i, a0));
        const float xav[2] = {xa.x, xa.y}, xbv[4] = {xb.x, xb.y, xb.z, xb.w};
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(xav[u], xbv[v], acc[u][v]);
      }
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v)
          if (b0 + v <= a0 + u) C[(a0 + u) * 65 + b0 + v] = acc[u][v];
    }
  }
  if (t == 0) *bad = 0;
  __syncthreads();
  // right-looking Cholesky, two barriers per column: thread t updates row t & 63, columns (t >> 6) + 8 m
  const int ci = t & 63, cj0 = t >> 6;
  for (int k = 0; k < r; ++k) {
    const float d = C[k * 65 + k];
    const float dk = d > 0.f ? sqrtf(d) : 1.f;
    if (t == 0) {
      if (!(d > 0.f)) *bad = 1;
      w.Dg[k] = dk;
    }
    if (t > k && t < r) {
      const float l = C[t * 65 + k] / dk;
      w.Lc[k * 64 + t] = l;
      w.Lr[sx(t, k)] = l;
    }
    __syncthreads();
    if (ci > k && ci < r) {
      const float lik = w.Lc[k * 64 + ci];
#pragma unroll
      for (int m = 0; m < 8; ++m) {
        const int j = cj0 + 8 * m;
        if (j > k && j <= ci) C[ci * 65 + j] = fmaf(-lik, w.Lc[k * 64 + j], C[ci * 65 + j]);
      }
    }
    __syncthreads();
  }
  // row t: x L^T = s by forward substitution over the columns (x in registers: every index below is a constant)
  {
    float4* X4 = reinterpret_cast<float4*>(X);
    const float4* L4 = reinterpret_cast<const float4*>(w.Lr);
    float x[SK_LD];
#pragma unroll
    for (int q = 0; q < SK_LD / 4; ++q) {
      const float4 v = 4 * q < r ? X4[sx_chunk(t, q)] : make_float4(0.f, 0.f, 0.f, 0.f);
      x[4 * q] = v.x;
      x[4 * q + 1] = v.y;
      x[4 * q + 2] = v.z;
      x[4 * q + 3] = v.w;
    }
#pragma unroll
    for (int j = 0; j < SK_LD; ++j) {
      if (j < r) {
        float acc = x[j];
#pragma unroll
        for (int q = 0; q < (j + 3) / 4; ++q) {
          const float4 l = L4[sx_chunk(j, q)];
          const float lv[4] = {l.x, l.y, l.z, l.w};
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (4 * q + u < j) acc = fmaf(-x[4 * q + u], lv[u], acc);
        }
        x[j] = acc / w.Dg[j];
      }
    }
#pragma unroll
    for (int q = 0; q < SK_LD / 4; ++q)
      if (4 * q < r) X4[sx_chunk(t, q)] = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
  }
  __syncthreads();
  return *bad == 0;
}

// Orthogonal iteration on one CTA: X0 = orth(M G) with G a fixed +-1 pattern, then iters steps X <- orth(M X)
// (two Cholesky-QR passes each), then the Rayleigh-Ritz matrix R = X^T M X into Bout [64][64] fp64 (zero past r) and
// X into Xout [512][64] (row-major).
__global__ void __launch_bounds__(SKI_THREADS, 1) k_sk_iterate(const float* __restrict__ M, int r, int iters,
                                                             float* __restrict__ Y, float* __restrict__ Xout,
                                                             double* __restrict__ Bout, int* __restrict__ status) {
  extern __shared__ __align__(16) float smf[];
  float* X = smf;                                     // [512][64], rows SK_XLD apart
  SkChol w;
  w.C = X + D_LAT * SK_XLD;                           // [64][65]
  w.Lr = w.C + 64 * 65;                               // [64][64], rows SK_XLD apart
  w.Lc = w.Lr + 64 * SK_XLD;                          // [64][64], L^T row-major
  w.Dg = w.Lc + 64 * 64;                              // [64]
  __shared__ int bad;
  const int t = threadIdx.x;
  for (int e = t; e < D_LAT * SK_LD; e += SKI_THREADS) {
    uint32_t h = (uint32_t)e * 2654435761u;           // Knuth's multiplicative hash, then a xorshift round
    h ^= h >> 15;
    h *= 2246822519u;
    h ^= h >> 13;
    X[sx(e >> 6, e & 63)] = (h & 1u) ? 1.f : -1.f;
  }
  __syncthreads();
  bool ok = true;
  for (int it = 0; it <= iters && ok; ++it) {
    // the product stays in shared memory: both Cholesky-QR passes read their operand from there
    sk_mx_inplace(M, X, r);
    ok = sk_cholqr(X, w, r, &bad) && sk_cholqr(X, w, r, &bad);
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
      for (int i = 0; i < D_LAT; ++i) acc = fmaf(X[sx(i, a)], Y[i * SK_LD + b], acc);
      v = acc;
    }
    Bout[e] = v;
  }
  for (int e = t; e < D_LAT * SK_LD; e += SKI_THREADS) Xout[e] = X[sx(e >> 6, e & 63)];
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
  const size_t ismem = sizeof(float) * (D_LAT * SK_XLD + 64 * 65 + 64 * SK_XLD + 64 * 64 + 64);
  if ((e = allow_smem(k_sk_iterate, ismem)) != cudaSuccess) return e;
  k_sk_iterate<<<1, SKI_THREADS, ismem, st>>>(M, r_sk, SK_ITERS, Y, X, Bm, status);
  if ((e = launch_sym_eig64(Bm, W, E, st)) != cudaSuccess) return e;
  k_sk_finish<<<r_sk, 512, 0, st>>>(r_sk, W, X, E, basis, eig);
  count_launches(3);
  return cudaGetLastError();
}

}  // namespace vk
