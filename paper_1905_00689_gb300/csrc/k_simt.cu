// Generic CUDA-core kernels of the approximate-LSTM recurrence.
//
// They cover every shape and both factor types and are the per-timestep
// path when neither the persistent cluster kernel nor the tensor-core
// kernels apply.  All arithmetic is fp32.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

__device__ __forceinline__ float load_f(const float* p, long long i) { return __ldg(p + i); }
__device__ __forceinline__ float load_f(const __nv_bfloat16* p, long long i) {
  return __bfloat162float(p[i]);
}

constexpr int BM = 64, BN = 64, BKT = 16;

// Tiled product over the packed factor rows (dot products prune(v)^T x~ of
// Eq. 1, for many inputs at once).  Each CTA computes 64 rows x 64 inputs;
// each thread a 4 x 4 block.
template <typename TF>
__global__ void __launch_bounds__(256) rows_gemm_kernel(const TF* __restrict__ A, int lda, int K, int Ks,
                                                        const float* __restrict__ Bm, int ldb, int N,
                                                        int Kdim, float* __restrict__ out, int ldo,
                                                        int mode, const float* __restrict__ sigma,
                                                        const float* __restrict__ P, int ldp) {
  __shared__ float As[BKT][BM + 4];
  __shared__ float Bs[BKT][BN + 4];
  const int tid = threadIdx.x;
  const int r0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
  const int nrows = 4 * K;
  const int tr = tid / 16, tc = tid % 16;
  float acc[4][4] = {};
  // loader mapping: 64 rows x 16 columns -> 4 elements per thread
  const int lrow = tid / 4, lk = (tid % 4) * 4;
  const int ar = r0 + lrow;
  const long long asrow = ar < nrows ? (long long)(ar / K) * Ks + ar % K : -1;
  const int bn = n0 + lrow;
  for (int k0 = 0; k0 < Kdim; k0 += BKT) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int kk = k0 + lk + e;
      As[lk + e][lrow] = (asrow >= 0 && kk < Kdim) ? load_f(A, asrow * lda + kk) : 0.f;
      Bs[lk + e][lrow] = (bn < N && kk < Kdim) ? __ldg(Bm + (long long)bn * ldb + kk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BKT; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][tr * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tc * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = r0 + tr * 4 + i;
    if (r >= nrows) continue;
    const long long srow = (long long)(r / K) * Ks + r % K;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tc * 4 + j;
      if (n >= N) continue;
      float v = acc[i][j];
      if (mode == 1) v = sigma[srow] * (v + P[(long long)n * ldp + srow]);
      out[(long long)n * ldo + srow] = v;
    }
  }
}

// One timestep for B streams: y_g = sum_k u_{g,k} * tau'_{g,k} (tau' already
// carries sigma), with the cell update applied to the k_j-prefix sums (the
// intermediate outputs) and to the full sum (the carried state).
template <typename TF>
__global__ void __launch_bounds__(128) cell_step_kernel(CellArgs a, const TF* __restrict__ U) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y;
  if (j >= a.H || b >= a.B) return;
  const float* tau = a.tau + (long long)b * a.ldt;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  float bias[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) bias[g] = a.bias[g * a.H + j];
  const float c_prev = a.c_state[(long long)b * a.H + j];
  int jj = 0;
  for (int k = 0; k < a.K; ++k) {
#pragma unroll
    for (int g = 0; g < 4; ++g)
      acc[g] = fmaf(load_f(U, g * a.gs + k * a.ks + j * a.js), tau[g * a.Ks + k], acc[g]);
    if (jj < a.ck.n && a.ck.k[jj] == k + 1) {
      float hh, cc;
      lstm_approx_dev::lstm_cell_f(acc[0] + bias[0], acc[1] + bias[1], acc[2] + bias[2], acc[3] + bias[3],
                                   c_prev, hh, cc);
      const long long o = jj * a.ck_stride + (long long)b * a.H + j;
      if (a.ckpt_h) a.ckpt_h[o] = hh;
      if (a.ckpt_c) a.ckpt_c[o] = cc;
      ++jj;
    }
  }
  float hh, cc;
  lstm_approx_dev::lstm_cell_f(acc[0] + bias[0], acc[1] + bias[1], acc[2] + bias[2], acc[3] + bias[3], c_prev,
                               hh, cc);
  a.c_state[(long long)b * a.H + j] = cc;
  a.h_state[(long long)b * a.H + j] = hh;
  if (a.out_h) a.out_h[(long long)b * a.H + j] = hh;
}

}  // namespace

cudaError_t launch_rows_gemm(const void* A, bool a_bf16, int lda, int K, int Ks, const float* Bm, int ldb,
                             int N, int Kdim, float* out, int ldo, int mode, const float* sigma,
                             const float* P, int ldp, cudaStream_t s) {
  dim3 grid((4 * K + BM - 1) / BM, (N + BN - 1) / BN);
  if (a_bf16)
    rows_gemm_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(A), lda, K, Ks, Bm,
                                                          ldb, N, Kdim, out, ldo, mode, sigma, P, ldp);
  else
    rows_gemm_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float*>(A), lda, K, Ks, Bm, ldb, N, Kdim,
                                                 out, ldo, mode, sigma, P, ldp);
  return cudaGetLastError();
}

cudaError_t launch_cell_step(const CellArgs& a, cudaStream_t s) {
  dim3 grid((a.H + 127) / 128, a.B);
  if (a.u_bf16)
    cell_step_kernel<__nv_bfloat16><<<grid, 128, 0, s>>>(a, static_cast<const __nv_bfloat16*>(a.U));
  else
    cell_step_kernel<float><<<grid, 128, 0, s>>>(a, static_cast<const float*>(a.U));
  return cudaGetLastError();
}

}  // namespace lstm_approx_impl
