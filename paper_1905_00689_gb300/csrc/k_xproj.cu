// Hoisted input projection for few columns (T*B <= 32): P[n][(g,k)] =
// prune(v_{g,k})[0:D]^T x_n for every timestep and stream at once (the x
// columns of x~ = [x_t; h_{t-1}], Sec. III, split off Eq. 1's dot products).
//
// With T*B this small the product is a skinny matrix times a thin one and
// the whole packed V_x is read once.  To spread it over the GPU the D axis is
// split over the 8 CTAs of a cluster: CTA (r, q) multiplies the 32 rows of
// block r by chunk q of the input, four k-groups of 64 threads each
// accumulate 4 x 4 register tiles, the k-groups are summed in shared memory,
// and the 8 chunk partials are summed through distributed shared memory in
// chunk order (deterministic), each CTA finishing 1/kSplit of the outputs.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kRows = 32;     // rows per CTA
constexpr int kCols = 32;     // max columns (T*B)
constexpr int kSplit = 8;     // CTAs per cluster along D
constexpr int kTileD = 128;   // D tile staged in shared memory
constexpr int kThreads = 256;

// 16 consecutive elements [d, d+16) of row `row` (ld = lda) as fp32, zero
// outside [0, d_hi) or for row < 0; vector loads when the run is aligned.
__device__ __forceinline__ void load16(const float* A, long long row, int lda, int d, int d_hi, float (&v)[16]) {
  if (row < 0) {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = 0.f;
    return;
  }
  const float* src = A + row * lda + d;
  if (d + 16 <= d_hi && ((reinterpret_cast<uintptr_t>(src) & 15u) == 0)) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldg(reinterpret_cast<const float4*>(src) + q);
      v[4 * q] = f.x; v[4 * q + 1] = f.y; v[4 * q + 2] = f.z; v[4 * q + 3] = f.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = d + e < d_hi ? __ldg(src + e) : 0.f;
  }
}
__device__ __forceinline__ void load16(const __nv_bfloat16* A, long long row, int lda, int d, int d_hi,
                                       float (&v)[16]) {
  if (row < 0) {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = 0.f;
    return;
  }
  const __nv_bfloat16* src = A + row * lda + d;
  if (d + 16 <= d_hi && ((reinterpret_cast<uintptr_t>(src) & 15u) == 0)) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const uint4 f = __ldg(reinterpret_cast<const uint4*>(src) + q);
      const uint32_t w[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[8 * q + 2 * i] = __uint_as_float(w[i] << 16);
        v[8 * q + 2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
      }
    }
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = d + e < d_hi ? __bfloat162float(src[e]) : 0.f;
  }
}

__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

template <typename TF>
__global__ void __launch_bounds__(kThreads) xproj_cluster_kernel(const TF* __restrict__ A, int lda, int K, int Ks,
                                                                 const float* __restrict__ X, int ldxin, int N,
                                                                 int D, float* __restrict__ out, int ldo) {
  __shared__ __align__(16) float Vs[kTileD][kRows + 4];
  __shared__ __align__(16) float Xs[kTileD][kCols];
  __shared__ float part[kRows * kCols];  // o = n * 32 + r

  const int tid = threadIdx.x;
  const int rb = blockIdx.x;
  const uint32_t q = cluster_ctarank();  // chunk of D (blockIdx.y within the cluster)
  const int nrows = 4 * K;
  const int dc = ((D + kSplit - 1) / kSplit + 3) & ~3;
  const int d_lo = min(D, (int)q * dc), d_hi = min(D, d_lo + dc);

  const int kg = tid >> 6, m = tid & 63;
  const int r0 = (m >> 3) << 2, n0 = (m & 7) << 2;
  float acc[4][4] = {};

  // loader mapping: 32 rows (or columns) x 8 slices of 16 d
  const int lrow = tid >> 3, lseg = (tid & 7) * 16;
  const int ar = rb * kRows + lrow;
  const long long asrow = ar < nrows ? (long long)(ar / K) * Ks + ar % K : -1;

  for (int d0 = d_lo; d0 < d_hi; d0 += kTileD) {
    const int dbase = d0 + lseg;
    float vv[16], xx[16];
    load16(A, asrow, lda, dbase, d_hi, vv);
    load16(X, lrow < N ? (long long)lrow : -1LL, ldxin, dbase, d_hi, xx);
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      Vs[lseg + e][lrow] = vv[e];
      Xs[lseg + e][lrow] = xx[e];
    }
    __syncthreads();
#pragma unroll 4
    for (int d = kg; d < kTileD; d += 4) {
      const float4 a = *reinterpret_cast<const float4*>(&Vs[d][r0]);
      const float4 x = *reinterpret_cast<const float4*>(&Xs[d][n0]);
      const float av[4] = {a.x, a.y, a.z, a.w}, xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], xv[j], acc[i][j]);
    }
    __syncthreads();
  }

  // sum the four k-groups (reusing the V tile as scratch: 4 x 1024 floats)
  float* red = &Vs[0][0];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) red[kg * 1024 + (n0 + j) * kRows + (r0 + i)] = acc[i][j];
  __syncthreads();
  for (int o = tid; o < kRows * kCols; o += kThreads)
    part[o] = red[o] + red[1024 + o] + red[2048 + o] + red[3072 + o];
  cluster_sync_all();

  // this CTA finishes outputs [q*OPC, (q+1)*OPC) from the kSplit chunk partials
  constexpr int kOPC = kRows * kCols / kSplit;
  for (int i = tid; i < kOPC; i += kThreads) {
    const int o = q * kOPC + i;
    const uint32_t la = smem_u32(&part[o]);
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < kSplit; ++c) s += ld_cluster_f32(mapa_shared(la, c));
    const int n = o / kRows, r = rb * kRows + o % kRows;
    if (n < N && r < nrows) out[(long long)n * ldo + (long long)(r / K) * Ks + r % K] = s;
  }
  cluster_sync_all();  // partials stay readable until every CTA has summed
}

}  // namespace

bool xproj_cluster_fits(int N) { return N >= 1 && N <= kCols; }

cudaError_t launch_xproj_cluster(const void* A, bool a_bf16, int lda, int K, int Ks, const float* X, int ldxin,
                                 int N, int D, float* out, int ldo, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((4 * K + kRows - 1) / kRows, kSplit, 1);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = kSplit;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (a_bf16)
    return cudaLaunchKernelEx(&cfg, xproj_cluster_kernel<__nv_bfloat16>, static_cast<const __nv_bfloat16*>(A), lda,
                              K, Ks, X, ldxin, N, D, out, ldo);
  return cudaLaunchKernelEx(&cfg, xproj_cluster_kernel<float>, static_cast<const float*>(A), lda, K, Ks, X, ldxin, N,
                            D, out, ldo);
}

}  // namespace lstm_approx_impl
