// Compressed alternative to the tau' GEMM of the tensor-core path (bf16
// factors): the recurrent part of the pruned v (Eq. 1, prune(v, NZ)) kept as
// its kept (column, value) entries per row instead of masked-dense rows,
// evaluated on the CUDA cores:
//
//   tau'[n][(g, k)] = sigma_{g,k} (P_t[n][(g, k)] + sum_{e in row (g, k)} val_e h_{t-1}[n][col_e])
//
// with h_{t-1} = hi + lo from the tensor path's bf16 pair, and tau' stored
// as its pair for the gate GEMM.  One CTA takes 32 streams and 256 rows: the
// streams' h (fp32, [H][32], column-major so that the 32 lanes of a warp read
// 32 consecutive words) is staged in shared memory once, then each warp runs
// 32 rows with lane = stream, each row's entries staged 32 at a time in a
// per-warp buffer that all lanes read at the same address.  Every
// multiply-add needs its own h value from shared memory (the rows' masks
// differ), so the kernel reads 4 bytes of shared memory per multiply-add and
// lane: bound by shared-memory bandwidth, not by the FMA pipes.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kStreams = 32;
constexpr int kWarpsPerCta = 8;
constexpr int kRowsPerWarp = 32;
constexpr int kRowsPerCta = kWarpsPerCta * kRowsPerWarp;

__global__ void __launch_bounds__(kWarpsPerCta * 32) tau_sparse_kernel(TauSparseArgs a) {
  extern __shared__ __align__(16) float hs[];                  // [H][32] h of this CTA's streams
  __shared__ float tile[kWarpsPerCta][kRowsPerWarp][kStreams + 1];  // tau' of a warp's rows, for the stores
  __shared__ int2 ent[kWarpsPerCta][32];                             // a row's next 32 (column, value) entries
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.y * kStreams;
  const int n = n0 + lane;
  griddep_wait();  // h_{t-1} is written by the gate kernel before this one
  for (int i = threadIdx.x; i < a.H * kStreams; i += blockDim.x) {
    const int c = i / kStreams, nn = n0 + i % kStreams;
    float v = 0.f;
    if (nn < a.B) {
      const long long o = (long long)nn * a.ldh + c;
      v = __bfloat162float(a.h[o]) + __bfloat162float(a.h[a.h_plane + o]);
    }
    hs[i] = v;
  }
  __syncthreads();
  griddep_launch_dependents();
  // rows r = g * Rp + k of the packed order (Rp = K rounded up to 64), at
  // storage row g * Ks + k; rows k >= K store zero (the gate GEMM reads
  // 64-term chunks)
  const int r0 = blockIdx.x * kRowsPerCta + warp * kRowsPerWarp;
  for (int i = 0; i < kRowsPerWarp; ++i) {
    const int r = r0 + i;
    float acc = 0.f;
    if (r < 4 * a.Rp) {
      const int g = r / a.Rp, k = r % a.Rp;
      if (k < a.K) {
        const int row = g * a.Ks + k;
        const int e0 = a.off[row], e1 = a.off[row + 1];
        for (int eb = e0; eb < e1; eb += 32) {
          const int e = eb + lane;
          __syncwarp();  // the previous chunk's entries have been read
          ent[warp][lane] = e < e1 ? make_int2(a.col[e], __float_as_int(a.val[e])) : make_int2(0, 0);
          __syncwarp();
          const int m = e1 - eb < 32 ? e1 - eb : 32;
#pragma unroll 4
          for (int j = 0; j < m; ++j) {
            const int2 cv = ent[warp][j];
            acc = fmaf(__int_as_float(cv.y), hs[cv.x * kStreams + lane], acc);
          }
        }
        if (n < a.B) acc = a.sigma[row] * (acc + a.P[(long long)n * a.ldp + row]);
      }
    }
    tile[warp][i][lane] = acc;
  }
  __syncwarp();
  // stores: lane = row, one stream at a time, so a warp writes 32 consecutive terms
  const int r = r0 + lane;
  if (r < 4 * a.Rp) {
    const int g = r / a.Rp, k = r % a.Rp;
    const long long row = (long long)g * a.Ks + k;
    for (int s = 0; s < kStreams; ++s) {
      const int nn = n0 + s;
      if (nn >= a.B) break;
      const float v = tile[warp][lane][s];
      const __nv_bfloat16 hi = __float2bfloat16_rn(v);
      const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
      a.tau[(long long)nn * a.ldt + row] = hi;
      a.tau[a.tau_plane + (long long)nn * a.ldt + row] = lo;
    }
  }
}

}  // namespace

size_t tau_sparse_smem(int H) { return (size_t)H * kStreams * sizeof(float); }
int tau_sparse_max_h() { return 1280; }  // 160 KB of h besides the 35 KB of static buffers

cudaError_t launch_tau_sparse(const TauSparseArgs& a, cudaStream_t s) {
  const size_t smem = tau_sparse_smem(a.H);
  static thread_local bool attr = false;
  if (!attr) {
    const cudaError_t e =
        cudaFuncSetAttribute(tau_sparse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)tau_sparse_smem(tau_sparse_max_h()));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((4 * a.Rp + kRowsPerCta - 1) / kRowsPerCta, (a.B + kStreams - 1) / kStreams);
  cfg.blockDim = dim3(kWarpsPerCta * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr1[1];
  attr1[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr1[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr1;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tau_sparse_kernel, a);
}

}  // namespace lstm_approx_impl
