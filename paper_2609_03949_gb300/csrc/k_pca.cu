// k_pca.cu -- the PCA digest basis (the appendix's branch-width ablation): principal directions of the RoPE branch.
//
// M = sum over every cached row of every sequence of K_u K_u^T (64 x 64), then its eigenvectors by decreasing
// eigenvalue, as the rows of the digest rotation (index->rot): the width-r digest (O K_u)[0:r] then keeps the most
// branch energy a width-r truncation can keep.
//   k_pca_moment  one CTA per SM over a range of 128-row chunks: each chunk's 64 RoPE columns are TMA-loaded once
//                 and serve as both operands of D += R^T R on tcgen05 (M = N = 64, K = 128 rows, both read
//                 MN-major from the same tile); the CTA's fp32 sum is added into the fp64 moment at the end.
//   k_pca_jacobi  one CTA: cyclic Jacobi with the round-robin ordering (32 disjoint rotations at a time, 63 steps per
//                 sweep), first in fp32, then re-orthonormalised and finished in fp64; then the eigenpairs sorted by
//                 decreasing eigenvalue, each eigenvector signed so that its largest entry is positive.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "vk_common.cuh"
#include "vk_ptx.cuh"

namespace vk {

namespace {

constexpr int PC_STAGES = 6;
constexpr uint32_t PC_TILE = 128 * 128;      // 128 rows x 64 bf16
constexpr int PC_THREADS = 6 * 32;           // producer, MMA issuer, four readout warps

__device__ __forceinline__ void pc_tma_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}
// 128-byte swizzle descriptor, 8-row groups 1024 B apart (the MN-major reading of a [rows x 64] tile: one 64-element
// atom along M/N, K = rows).
__device__ __forceinline__ uint64_t pc_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}
__device__ __forceinline__ void pc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void pc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_addr(bar))
               : "memory");
}

struct PcaArgs {
  int B, N, cps;             // chunks per sequence
  long long chunks;          // B * cps
  double* moment;            // [64 * 64], zeroed
  int* status;
};

__global__ void __launch_bounds__(PC_THREADS, 1) k_pca_moment(const __grid_constant__ CUtensorMap rmap,
                                                            const PcaArgs args) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + PC_STAGES * PC_TILE);
  uint64_t* full = bars;
  uint64_t* empty = bars + PC_STAGES;
  uint64_t* done = empty + PC_STAGES;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long c0 = args.chunks * blockIdx.x / gridDim.x, c1 = args.chunks * (blockIdx.x + 1) / gridDim.x;
  const int n = (int)(c1 - c0);
  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < PC_STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(done, 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, 64);
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      int b = (int)(c0 / args.cps), c = (int)(c0 - (long long)b * args.cps);
      bool ok = true;
      for (int i = 0; i < n; ++i) {
        const int s = i % PC_STAGES, use = i / PC_STAGES;
        if (use > 0 && !mbar_wait(&empty[s], (use - 1) & 1, &abort_flag)) { ok = false; break; }
        mbar_arrive_expect_tx(&full[s], PC_TILE);
        pc_tma_3d(smem + s * PC_TILE, &rmap, 0, c * 128, b, &full[s]);   // rows past N read as zeros
        if (++c == args.cps) { c = 0; ++b; }
      }
      if (!ok) abort_flag = 1;
      for (int k = std::max(0, n - PC_STAGES); k < n; ++k) mbar_wait(&full[k % PC_STAGES], (k / PC_STAGES) & 1, nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // D = R^T R: M = N = 64 dims, A and B both MN-major (bits 15, 16) from the same tile, K = 16 rows per instruction
      constexpr uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) |
                                 ((uint32_t)(64 >> 3) << 17) | ((uint32_t)(64 >> 4) << 24);
      bool ok = true;
      for (int i = 0; i < n; ++i) {
        const int s = i % PC_STAGES, use = i / PC_STAGES;
        if (!mbar_wait(&full[s], use & 1, &abort_flag)) { ok = false; break; }
        tmem_fence_after();
        const uint32_t st = smem_addr(smem + s * PC_TILE);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint64_t d = pc_desc(st + j * 2048);
          pc_mma(tmem, d, d, idesc, (i > 0 || j > 0) ? 1u : 0u);
        }
        pc_commit(&empty[s]);
      }
      if (!ok) {
        abort_flag = 1;
        raise_status(args.status, VK_ERR_TIMEOUT);
      }
      pc_commit(done);
    }
  } else {
    // readout: the M = 64 accumulator holds row 16 q + i in lane 32 q + i; lanes 0..15 of the warp get columns 0..31,
    // lanes 16..31 columns 32..63 of the same rows
    const int q = warp & 3;
    if (n > 0) {
      bool w = true;
      if (lane == 0) w = mbar_wait(done, 0, &abort_flag);
      w = __shfl_sync(0xffffffffu, w, 0);
      tmem_fence_after();
      if (w) {
        float v[32];
        uint32_t* r = reinterpret_cast<uint32_t*>(v);
        const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16);
        asm volatile(
            "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
            "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], 32;\n"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
              "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
              "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]),
              "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
              "=r"(r[30]), "=r"(r[31])
            : "r"(taddr)
            : "memory");
        tmem_wait_ld();
        const int row = 16 * q + (lane & 15), col0 = 32 * (lane >> 4);
#pragma unroll
        for (int k = 0; k < 32; ++k) atomicAdd(&args.moment[row * 64 + col0 + k], (double)v[k]);
      } else if (lane == 0) {
        raise_status(args.status, VK_ERR_TIMEOUT);
      }
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    tmem_dealloc(tmem, 64);
  }
}

// One CTA of 256 threads: the symmetric 64 x 64 eigenproblem by cyclic Jacobi, 32 disjoint rotations per step.
constexpr int JC_THREADS = 256;
constexpr size_t JC_SMEM = 3 * 64 * 65 * sizeof(double) + 2 * 64 * 65 * sizeof(float);

// Sum of x over the block (every thread gets it).
__device__ __forceinline__ double jc_block_sum(double x, double* red) {
  const int t = threadIdx.x;
  red[t] = x;
  __syncthreads();
  for (int o = JC_THREADS / 2; o; o >>= 1) {
    if (t < o) red[t] += red[t + o];
    __syncthreads();
  }
  const double v = red[0];
  __syncthreads();
  return v;
}

// Largest x over the block (every thread gets it).
__device__ __forceinline__ double jc_block_max(double x, double* red) {
  const int t = threadIdx.x;
  red[t] = x;
  __syncthreads();
  for (int o = JC_THREADS / 2; o; o >>= 1) {
    if (t < o) red[t] = fmax(red[t], red[t + o]);
    __syncthreads();
  }
  const double v = red[0];
  __syncthreads();
  return v;
}

// Cyclic Jacobi sweeps on A (V accumulates the rotations) in precision T, until the off-diagonal squared norm is at
// most tol times the total squared norm, or it falls by less than 4x in a sweep once below stall times the total (the
// rounding floor of precision T), or max_sweeps. Each rotation sets its a_pq, a_qp to zero and its a_pp, a_qq to
// a_pp - t a_pq, a_qq + t a_pq (t = tan of the angle) instead of taking them from the update products, so that the
// off-diagonal norm is not held up by their rounding.
template <typename T>
__device__ void jc_sweeps(T (*A)[65], T (*V)[65], double* red, double tol, double stall, int max_sweeps) {
  __shared__ T cs[32][2];
  __shared__ T dg[32][2];
  __shared__ int pr[32][2];
  const int t = threadIdx.x;
  double total = 0.0;
  for (int i = t; i < 64 * 64; i += JC_THREADS) total += (double)A[i / 64][i % 64] * (double)A[i / 64][i % 64];
  total = jc_block_sum(total, red);
  double prev = 0.0;
  for (int sweep = 0; sweep < max_sweeps; ++sweep) {
    double off = 0.0;
    for (int i = t; i < 64 * 64; i += JC_THREADS)
      if (i / 64 != i % 64) off += (double)A[i / 64][i % 64] * (double)A[i / 64][i % 64];
    off = jc_block_sum(off, red);
    if (off <= tol * total || (sweep > 0 && off <= stall * total && off > 0.25 * prev)) break;
    prev = off;
    for (int step = 0; step < 63; ++step) {
      if (t < 32) {
        // round-robin: index 63 meets step; the others pair up symmetrically around it
        int p = t == 0 ? 63 : (step + t) % 63, q = t == 0 ? step : (step - t + 63) % 63;
        if (p > q) { const int x = p; p = q; q = x; }
        pr[t][0] = p;
        pr[t][1] = q;
        const T apq = A[p][q], app = A[p][p], aqq = A[q][q];
        T c = T(1), sn = T(0), tt = T(0);
        if (apq != T(0)) {
          const T theta = (aqq - app) / (T(2) * apq);
          tt = (theta >= T(0) ? T(1) : T(-1)) / (fabs(theta) + sqrt(theta * theta + T(1)));
          c = T(1) / sqrt(tt * tt + T(1));
          sn = tt * c;
        }
        cs[t][0] = c;
        cs[t][1] = sn;
        dg[t][0] = app - tt * apq;
        dg[t][1] = aqq + tt * apq;
      }
      __syncthreads();
      // rows p, q of every pair: A <- J^T A
      for (int e = t; e < 32 * 64; e += JC_THREADS) {
        const int k = e & 63, w = e >> 6;
        const int p = pr[w][0], q = pr[w][1];
        const T c = cs[w][0], sn = cs[w][1];
        const T apk = A[p][k], aqk = A[q][k];
        A[p][k] = c * apk - sn * aqk;
        A[q][k] = sn * apk + c * aqk;
      }
      __syncthreads();
      // columns p, q: A <- A J, V <- V J
      for (int e = t; e < 32 * 64; e += JC_THREADS) {
        const int k = e & 63, w = e >> 6;
        const int p = pr[w][0], q = pr[w][1];
        const T c = cs[w][0], sn = cs[w][1];
        const T akp = A[k][p], akq = A[k][q];
        T np = c * akp - sn * akq, nq = sn * akp + c * akq;
        if (k == p) {
          np = dg[w][0];
          nq = T(0);
        } else if (k == q) {
          np = T(0);
          nq = dg[w][1];
        }
        A[k][p] = np;
        A[k][q] = nq;
        const T vkp = V[k][p], vkq = V[k][q];
        V[k][p] = c * vkp - sn * vkq;
        V[k][q] = sn * vkp + c * vkq;
      }
      __syncthreads();
    }
  }
}

// The sweeps run first in fp32, many times faster than fp64 on this part, down to an off-diagonal norm at fp32's
// level; the fp32 rotations are then re-orthonormalised in fp64 (classical Gram-Schmidt, twice), the moment is
// projected on them in fp64, and fp64 sweeps finish from there to the threshold of a pure fp64 solve.
__global__ void __launch_bounds__(JC_THREADS) k_pca_jacobi(const double* __restrict__ moment, float* __restrict__ rot,
                                                         float* __restrict__ eig_out) {
  extern __shared__ double jc_smem[];                 // padded 64 x 65 arrays against bank conflicts
  double(*A)[65] = reinterpret_cast<double(*)[65]>(jc_smem);                // the moment, then V^T M V
  double(*V)[65] = reinterpret_cast<double(*)[65]>(jc_smem + 64 * 65);      // the rotations
  double(*W)[65] = reinterpret_cast<double(*)[65]>(jc_smem + 2 * 64 * 65);  // M V
  float(*Af)[65] = reinterpret_cast<float(*)[65]>(jc_smem + 3 * 64 * 65);
  float(*Vf)[65] = Af + 64;
  __shared__ double red[JC_THREADS];
  __shared__ double coef[64];
  __shared__ int ord[64];
  const int t = threadIdx.x;
  // the fp32 copy is scaled by a power of two that brings the largest entry near 1, so that it neither overflows nor
  // underflows whatever the data's scale; the scaling is exact and the rotations do not depend on it
  double amax = 0.0;
  for (int i = t; i < 64 * 64; i += JC_THREADS) amax = fmax(amax, fabs(moment[i]));
  amax = jc_block_max(amax, red);
  const double sc = amax > 0.0 && isfinite(amax) ? ldexp(1.0, -ilogb(amax)) : 1.0;
  for (int i = t; i < 64 * 64; i += JC_THREADS) {
    const double m = moment[i];
    A[i / 64][i % 64] = m;
    Af[i / 64][i % 64] = (float)(m * sc);
    Vf[i / 64][i % 64] = (i / 64 == i % 64) ? 1.f : 0.f;
  }
  __syncthreads();
  jc_sweeps<float>(Af, Vf, red, 1e-12, 1e-7, 40);
  for (int i = t; i < 64 * 64; i += JC_THREADS) V[i / 64][i % 64] = (double)Vf[i / 64][i % 64];
  __syncthreads();
  for (int c = 0; c < 64; ++c) {
    for (int pass = 0; pass < 2; ++pass) {
      if (t < c) {
        double d = 0.0;
        for (int k = 0; k < 64; ++k) d = fma(V[k][t], V[k][c], d);
        coef[t] = d;
      }
      __syncthreads();
      if (t < 64) {
        double x = V[t][c];
        for (int d = 0; d < c; ++d) x = fma(-coef[d], V[t][d], x);
        V[t][c] = x;
      }
      __syncthreads();
    }
    const double nn = jc_block_sum(t < 64 ? V[t][c] * V[t][c] : 0.0, red);
    if (t < 64) V[t][c] /= sqrt(nn);
    __syncthreads();
  }
  for (int e = t; e < 64 * 64; e += JC_THREADS) {    // W = M V
    const int i = e / 64, j = e % 64;
    double x = 0.0;
    for (int k = 0; k < 64; ++k) x = fma(A[i][k], V[k][j], x);
    W[i][j] = x;
  }
  __syncthreads();
  for (int e = t; e < 64 * 64; e += JC_THREADS) {    // A = V^T W
    const int i = e / 64, j = e % 64;
    double x = 0.0;
    for (int k = 0; k < 64; ++k) x = fma(V[k][i], W[k][j], x);
    A[i][j] = x;
  }
  __syncthreads();
  jc_sweeps<double>(A, V, red, 1e-30, 1e-24, 40);
  if (t == 0) {
    for (int i = 0; i < 64; ++i) ord[i] = i;
    for (int i = 1; i < 64; ++i) {
      const int x = ord[i];
      int j = i - 1;
      while (j >= 0 && A[ord[j]][ord[j]] < A[x][x]) { ord[j + 1] = ord[j]; --j; }
      ord[j + 1] = x;
    }
  }
  __syncthreads();
  if (t < 64) {
    const int c = ord[t];
    int big = 0;
    for (int k = 1; k < 64; ++k)
      if (fabs(V[k][c]) > fabs(V[big][c])) big = k;
    const double sg = V[big][c] < 0.0 ? -1.0 : 1.0;
    for (int k = 0; k < 64; ++k) rot[t * 64 + k] = (float)(sg * V[k][c]);
    if (eig_out) eig_out[t] = (float)A[c][c];
  }
}

PFN_cuTensorMapEncodeTiled_v12000 pc_encode() {
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

}  // namespace

size_t pca_workspace_bytes() { return 256 + 64 * 64 * sizeof(double); }

cudaError_t launch_pca_basis(const vk_view& v, float* rot, float* eig, void* ws, cudaStream_t st) {
  auto encode = pc_encode();
  if (!encode) return cudaErrorNotSupported;
  int* status = static_cast<int*>(ws);
  double* moment = reinterpret_cast<double*>(static_cast<char*>(ws) + 256);
  cudaError_t e = cudaMemsetAsync(moment, 0, 64 * 64 * sizeof(double), st);
  if (e != cudaSuccess) return e;
  CUtensorMap rmap;
  cuuint64_t dims[3] = {(cuuint64_t)D_ROPE, (cuuint64_t)v.N, (cuuint64_t)v.B};
  cuuint64_t str[2] = {(cuuint64_t)(v.rope_ld * 2), (cuuint64_t)(v.rope_bstride * 2)};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t es[3] = {1, 1, 1};
  if (encode(&rmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(v.rope), dims, str, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  PcaArgs a{};
  a.B = v.B;
  a.N = v.N;
  a.cps = (v.N + 127) / 128;
  a.chunks = (long long)v.B * a.cps;
  a.moment = moment;
  a.status = status;
  const int grid = (int)std::min<long long>(a.chunks, sm_count());
  const size_t smem = PC_STAGES * PC_TILE + (2 * PC_STAGES + 1) * 8 + 1024;
  e = cudaFuncSetAttribute(k_pca_moment, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_pca_moment<<<grid, PC_THREADS, smem, st>>>(rmap, a);
  const size_t jsmem = JC_SMEM;
  e = cudaFuncSetAttribute(k_pca_jacobi, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)jsmem);
  if (e != cudaSuccess) return e;
  k_pca_jacobi<<<1, JC_THREADS, jsmem, st>>>(moment, rot, eig);
  count_launches(2);
  return cudaGetLastError();
}

cudaError_t launch_sym_eig64(const double* A, float* vec, float* eig, cudaStream_t st) {
  const size_t jsmem = JC_SMEM;
  cudaError_t e = cudaFuncSetAttribute(k_pca_jacobi, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)jsmem);
  if (e != cudaSuccess) return e;
  k_pca_jacobi<<<1, JC_THREADS, jsmem, st>>>(A, vec, eig);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace vk
