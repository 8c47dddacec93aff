// Dense LSTM comparator: the recurrence of Sec. II with the full gate
// matrices W_g = [Wx_g Wh_g] (no approximation), as a persistent cluster
// kernel built the same way as the approximate ones, so that the speed-up of
// the approximation is measured against a dense kernel of the same design
// (the paper's own comparison is against dense baselines on each platform,
// Sec. VI-B, Table I).
//
// The input part Wx_g x_t is hoisted over all t by the input-projection
// kernels of the approximate path (the same product with the gate matrices'
// rows in place of the pruned v rows).  One cluster of CS CTAs serves one
// stream; CTA c owns UB hidden units, i.e. 4*UB rows of Wh (gate-major: row
// g*UB + u is gate g of unit c*UB + u), which stay in tensor memory for the
// whole launch.  Per timestep:
//
//   1. every warp forms the dot products of its rows with h_{t-1} (held in
//      shared memory), reading its rows' values with tcgen05.ld: lane l holds
//      the values at the h indices 4l + 128e + i (e < HQ, i < 4), so one
//      16-column load brings one h quad of four rows and the h reads are
//      conflict-free 16-byte loads;
//   2. the row sums are reduced over the lanes by a transposed butterfly,
//      offset by P_t and the bias, and written to shared memory;
//   3. one warp runs the cell update of its CTA's units (c stays in
//      registers) and pushes h_t to every CTA of the cluster with 16-byte
//      st.async stores that complete the receivers' mbarriers.
//
// So a timestep has one exchange (h), where the approximate kernels have
// the tau' exchange as well.  Every wait is bounded in wall time; a wait that
// runs out writes the status word, the CTA leaves the loop, and the cluster
// meets at a final barrier.
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>

#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
// workspace of lstm_approx_dense_run: status word, projection flags, P
constexpr size_t kDenseFlagsOffset = 256;
constexpr size_t kDensePOffset = kDenseFlagsOffset + kProjFlags * sizeof(unsigned);

struct DenseArgs {
  const float* Wh;    // [4H][H], row g*H + j = the recurrent part of row j of W_g
  const float* bias;  // [4][H] or null
  const float* P;     // [T][B][4H]: Wx_g x_t, row g*H + j
  const float* h0;    // [B][H] or null
  const float* c0;    // [B][H] or null
  float* out_h;       // [T][B][H]
  float* c_last;      // [B][H] or null
  int* err;
  int H, T, B, CS, UB;
  long long limit_ns;
  // non-null when the projection that writes P is launched after this kernel
  // (the approximate path's launch order, XprojSignal)
  const unsigned* proj_flags;
  int proj_nflags;
  unsigned proj_epoch;
};

// Sum of NV values over the 32 lanes, transposed (high lane bits first):
// afterwards lane l holds in v[0] the total of value l >> (5 - log2 NV).
template <int NV>
__device__ __forceinline__ void transpose_sum(float (&v)[NV], int lane) {
  constexpr int kSteps = NV == 8 ? 3 : 2;
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    const int half = NV >> (s + 1);
    const int mask = 16 >> s;
    const bool upper = (lane & mask) != 0;
#pragma unroll
    for (int i = 0; i < half; ++i) {
      const float keep = upper ? v[i + half] : v[i];
      const float send = upper ? v[i] : v[i + half];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
    }
  }
#pragma unroll
  for (int mask = 16 >> kSteps; mask > 0; mask >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], mask);
}

// HQ: h quads per lane (H <= 128 HQ); G: groups of four rows per warp (the
// CTA's 4*UB rows over 16 warps: UB = 16 * G).
template <int HQ, int G>
__global__ void __launch_bounds__(kThreads, 1) dense_kernel(DenseArgs a) {
  constexpr int NV = 4 * G;       // rows per warp
  constexpr int kCols = 16 * HQ;  // tensor-memory columns of one group of four rows
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);            // [0, 1]: h_t by parity
  uint32_t* taddr_s = reinterpret_cast<uint32_t*>(smem_raw + 64);
  float* ys = reinterpret_cast<float*>(smem_raw + 128);              // [4][UB] gate pre-activations
  const int UB = a.UB, H = a.H, CS = a.CS;
  const int h_len = (CS * UB > 128 * HQ) ? CS * UB : 128 * HQ;      // received values; lanes read 128 HQ
  float* h_s = ys + 4 * UB;                                          // [2][h_len]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  // a projection launched after this kernel may start now (it waits for nothing)
  if (a.proj_flags != nullptr) griddep_launch_dependents();
  const int b = blockIdx.x / CS;
  const uint64_t limit = static_cast<uint64_t>(a.limit_ns);
  const volatile int* err = a.err;
  const uint32_t bytes_h = static_cast<uint32_t>(CS * UB) * 4u;
  const uint32_t tcols = 4u * G * kCols;  // 64 G HQ: a power of two from 64 to 512

  if (tid == 0) {
    mbar_init(smem_u32(&bars[0]), kWarps);
    mbar_init(smem_u32(&bars[1]), kWarps);
    fence_mbarrier_init_cluster();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(taddr_s), tcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *taddr_s;
  if (lane == 0)  // first use of both h barriers: every warp arrives, warp 0 with the bytes
    for (int hb = 0; hb < 2; ++hb) {
      if (warp == 0) mbar_arrive_expect_tx(smem_u32(&bars[hb]), bytes_h);
      else mbar_arrive(smem_u32(&bars[hb]));
    }
  for (int i = tid; i < h_len; i += kThreads) {
    h_s[i] = (a.h0 != nullptr && i < H) ? a.h0[(long long)b * H + i] : 0.f;
    h_s[h_len + i] = 0.f;
  }

  // rows of this warp: v = 4 grp + r is CTA row warp * NV + v, gate
  // (row / UB), unit rank * UB + row % UB.  Group grp of the warp lives in
  // lane quarter (warp & 3), columns (warp >> 2) * G * kCols + grp * kCols
  // + 16 e + 4 r + i for the h index 4 lane + 128 e + i.
  const uint32_t t_lane = tmem_base + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
  const uint32_t t_col0 = static_cast<uint32_t>((warp >> 2) * G * kCols);
  const bool h_vec = (H & 3) == 0;
#pragma unroll
  for (int grp = 0; grp < G; ++grp) {
    const float* rowp[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int row = warp * NV + 4 * grp + r, g = row / UB, j = (int)rank * UB + row % UB;
      rowp[r] = j < H ? a.Wh + ((long long)g * H + j) * H : nullptr;
    }
#pragma unroll
    for (int e = 0; e < HQ; ++e) {
      const int hi = 4 * lane + 128 * e;
      float v[16];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (rowp[r] != nullptr && hi < H) {
          if (h_vec) {
            f = __ldg(reinterpret_cast<const float4*>(rowp[r] + hi));
          } else {
            f.x = __ldg(rowp[r] + hi);
            f.y = hi + 1 < H ? __ldg(rowp[r] + hi + 1) : 0.f;
            f.z = hi + 2 < H ? __ldg(rowp[r] + hi + 2) : 0.f;
            f.w = hi + 3 < H ? __ldg(rowp[r] + hi + 3) : 0.f;
          }
        }
        v[4 * r] = f.x; v[4 * r + 1] = f.y; v[4 * r + 2] = f.z; v[4 * r + 3] = f.w;
      }
      tmem_st16(t_lane + t_col0 + grp * kCols + 16 * e, v);
    }
  }
  tmem_wait_st();

  // the lane that ends up with row v's sum (transpose_sum: lane l holds
  // value l >> (5 - log2 NV)) adds P_t and the bias
  const int my_v = lane >> (NV == 8 ? 2 : 3);
  const int my_row = warp * NV + my_v, my_g = my_row / UB, my_u = my_row % UB;
  const int my_j = (int)rank * UB + my_u;
  const bool writer = (lane & ((32 / NV) - 1)) == 0;
  const long long p_off = (long long)my_g * H + my_j;
  const float my_bias = (a.bias != nullptr && my_j < H) ? a.bias[my_g * H + my_j] : 0.f;
  // cell state in warp 0: lane u < UB runs unit rank * UB + u
  const int cj = (int)rank * UB + lane;
  const bool cell_lane = warp == 0 && lane < UB && cj < H;
  float c_reg = (cell_lane && a.c0 != nullptr) ? a.c0[(long long)b * H + cj] : 0.f;

  // P is written by the projection launched just before this kernel, or just
  // after it (its CTAs then each raise a flag once their part is stored)
  bool setup_ok = true;
  if (a.proj_flags == nullptr) griddep_wait();
  else if (warp == 0) setup_ok = wait_flags_epoch(a.proj_flags, a.proj_nflags, a.proj_epoch, limit, err);
  if (!__syncthreads_and(setup_ok) && tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
  // P through L2 (it may have been written while this kernel ran)
  float p_cur = (writer && my_j < H) ? __ldcg(a.P + (long long)b * 4 * H + p_off) : 0.f;
  const uint32_t bar_h0 = smem_u32(&bars[0]);
  cluster_sync_all();  // every CTA's barriers are armed before any st.async
  const int t_end = *err == 0 ? a.T : 0;  // nothing to do after a failed set-up

  bool failed = false;
  for (int t = 0; t < t_end && !failed; ++t) {
    const int hb = t & 1;
    const float p_next = (writer && my_j < H && t + 1 < a.T)
                             ? __ldcg(a.P + ((long long)(t + 1) * a.B + b) * 4 * H + p_off)
                             : 0.f;
    bool fail = false;
    if (t > 0) {
      const bool ok = mbar_wait_bounded<true>(bar_h0 + 8u * hb, ((t - 1) >> 1) & 1, limit, err);
      fail = !__all_sync(0xffffffffu, ok);
      if (!fail && lane == 0) {  // re-arm this parity for step t + 2
        if (warp == 0) mbar_arrive_expect_tx(bar_h0 + 8u * hb, bytes_h);
        else mbar_arrive(bar_h0 + 8u * hb);
      }
    }
    if (!fail) {
      // ---- y = Wh h_{t-1} + P_t + b for this warp's rows ------------------
      const float* hsrc = h_s + hb * h_len + 4 * lane;
      float acc[NV];
#pragma unroll
      for (int v = 0; v < NV; ++v) acc[v] = 0.f;
#pragma unroll
      for (int e = 0; e < HQ; ++e) {
        const float4 hq = *reinterpret_cast<const float4*>(hsrc + 128 * e);
        float w[G][16];
        if constexpr (G == 2) {
          tmem_ld16x2_sync(t_lane + t_col0 + 16 * e, t_lane + t_col0 + kCols + 16 * e, w[0], w[1]);
        } else {
          tmem_ld16_sync(t_lane + t_col0 + 16 * e, w[0]);
        }
#pragma unroll
        for (int grp = 0; grp < G; ++grp)
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            float s = acc[4 * grp + r];
            s = fmaf(w[grp][4 * r + 0], hq.x, s);
            s = fmaf(w[grp][4 * r + 1], hq.y, s);
            s = fmaf(w[grp][4 * r + 2], hq.z, s);
            s = fmaf(w[grp][4 * r + 3], hq.w, s);
            acc[4 * grp + r] = s;
          }
      }
      transpose_sum<NV>(acc, lane);
      if (writer) ys[my_g * UB + my_u] = acc[0] + p_cur + my_bias;
    }
    if (fail && lane == 0) atomicCAS(a.err, 0, kErrWaitTimeoutB);
    if (__syncthreads_or(fail)) {
      failed = true;
      break;
    }
    // ---- cell update (Sec. II) and h_t to every CTA ------------------------
    if (warp == 0) {
      float h_new = 0.f;
      if (cell_lane) {
        float hh, cc;
        lstm_cell_f(ys[lane], ys[UB + lane], ys[2 * UB + lane], ys[3 * UB + lane], c_reg, hh, cc);
        c_reg = cc;
        h_new = hh;
      }
      if (t + 1 < a.T) {
        // message m = (piece m / CS, CTA m % CS): the 4 units of the piece
        const int nb = (t + 1) & 1;
        const int n_msg = (UB / 4) * CS;
        for (int m0 = 0; m0 < n_msg; m0 += 32) {
          const int m = m0 + lane;
          const int pc = m / CS, dst = m % CS;
          float hv[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) hv[e] = __shfl_sync(0xffffffffu, h_new, (4 * pc + e) & 31);
          if (m < n_msg) {
            const uint32_t off = 4u * (nb * h_len + rank * UB + 4 * pc);
            st_async_v4(mapa_shared(smem_u32(h_s), dst) + off, hv[0], hv[1], hv[2], hv[3],
                        mapa_shared(bar_h0 + 8u * nb, dst));
          }
        }
      }
      // the output store after the sends: it is not on the path to the next timestep
      if (cell_lane) a.out_h[((long long)t * a.B + b) * H + cj] = h_new;
    }
    p_cur = p_next;
  }

  if (cell_lane && a.c_last != nullptr) a.c_last[(long long)b * H + cj] = c_reg;
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, tcols);
  }
  cluster_sync_all();  // no CTA leaves while others may still address its shared memory
  if (__syncthreads_or(failed)) {
    // stores issued just before the peers stopped may still be in flight
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
  }
}

// Dynamic shared memory of at least this much keeps one CTA per SM, so that
// no two CTAs wait for each other's tensor memory.
constexpr size_t kMinSmemBytes = 116 * 1024;

template <int HQ, int G>
cudaError_t launch_dense_t(const DenseArgs& a, cudaStream_t s) {
  auto kern = dense_kernel<HQ, G>;
  const int h_len = (a.CS * a.UB > 128 * HQ) ? a.CS * a.UB : 128 * HQ;
  size_t smem = 128 + 16ull * a.UB + 8ull * h_len;
  if (smem < kMinSmemBytes) smem = kMinSmemBytes;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.CS * a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = a.CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // after the projection: its programmatic dependent; before it: an ordinary launch
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = a.proj_flags == nullptr ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

int report(char* msg, int msg_len, int code, const char* fmt, ...) {
  if (msg && msg_len > 0) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(msg, (size_t)msg_len, fmt, ap);
    va_end(ap);
  }
  return code;
}

}  // namespace

bool plan_dense(int H, int* CS, int* UB, int* HQ) {
  if (H < 1 || H > 512) return false;
  *HQ = H <= 128 ? 1 : (H <= 256 ? 2 : 4);
  *UB = H <= 256 ? 16 : 32;
  int cs = 4;
  while (cs * *UB < H) cs *= 2;
  *CS = cs;
  return cs <= 16;
}

cudaError_t launch_dense(const float* Wh, const float* bias, const float* P, const float* h0, const float* c0,
                         float* out_h, float* c_last, int* err, int H, int T, int B, long long limit_ns,
                         cudaStream_t s, const unsigned* proj_flags, int proj_nflags, unsigned proj_epoch) {
  DenseArgs a{};
  a.proj_flags = proj_flags;
  a.proj_nflags = proj_nflags;
  a.proj_epoch = proj_epoch;
  int HQ = 0;
  if (!plan_dense(H, &a.CS, &a.UB, &HQ)) return cudaErrorInvalidValue;
  a.Wh = Wh;
  a.bias = bias;
  a.P = P;
  a.h0 = h0;
  a.c0 = c0;
  a.out_h = out_h;
  a.c_last = c_last;
  a.err = err;
  a.H = H;
  a.T = T;
  a.B = B;
  a.limit_ns = limit_ns;
  const int G = a.UB / 16;
  if (HQ == 1) return launch_dense_t<1, 1>(a, s);
  if (HQ == 2) return launch_dense_t<2, 1>(a, s);
  return G == 2 ? launch_dense_t<4, 2>(a, s) : launch_dense_t<4, 1>(a, s);
}

}  // namespace lstm_approx_impl

using namespace lstm_approx_impl;

namespace {
std::atomic<int> g_dense_launch_order{0};
}  // namespace

extern "C" int lstm_approx_dense_set_launch_order(int order) {
  if (order < 0 || order > 1) return LSTM_APPROX_EINVAL;
  g_dense_launch_order.store(order);
  return LSTM_APPROX_OK;
}

extern "C" int lstm_approx_dense_run(const float* Wx, const float* Wh, const float* bias, int D, int H,
                                     const float* x, int T, int B, const float* h0, const float* c0, float* out_h,
                                     float* out_c, void* workspace, size_t workspace_bytes, void* cuda_stream,
                                     char* msg, int msg_len) {
  if (msg && msg_len > 0) msg[0] = '\0';
  if (!Wx || !Wh || !x || !out_h || !workspace)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "Wx, Wh, x, out_h and workspace must not be NULL");
  if (D < 1 || H < 1 || H > 512 || T < 1 || B < 1)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "need D, T, B >= 1 and 1 <= H <= 512");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "workspace must be 256-byte aligned");
  const size_t need = lstm_approx_dense_workspace_bytes(H, T, B);
  if (workspace_bytes < need)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "workspace of %zu bytes, %zu needed", workspace_bytes, need);
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "no CUDA device");
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return report(msg, msg_len, LSTM_APPROX_ECUDA, "needs an sm_103 device");
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  // workspace: the status word, the projection's completion flags, then P
  int* status = static_cast<int*>(workspace);
  unsigned* flags = reinterpret_cast<unsigned*>(static_cast<char*>(workspace) + kDenseFlagsOffset);
  float* P = reinterpret_cast<float*>(static_cast<char*>(workspace) + kDensePOffset);
  // Wx x_t for all t: the approximate path's projection with the 4H gate rows
  // of Wx in place of the pruned v rows (K = Ks = H).  For one stream it is
  // launched after the recurrence, as the approximate path does (the flags
  // are cleared first, every call, so that epoch 1 always marks this call).
  const bool cluster_x = xproj_cluster_fits(T * B, D, Wx, D, x, D, false);
  const int proj_ctas = cluster_x ? xproj_cluster_ctas(H, T * B, D, 8) : 0;
  const char* blocking = std::getenv("CUDA_LAUNCH_BLOCKING");  // every launch blocking: never side by side
  cudaStreamCaptureStatus capture = cudaStreamCaptureStatusNone;  // (the call synchronises: never captured,
  if (cudaStreamIsCapturing(s, &capture) != cudaSuccess) capture = cudaStreamCaptureStatusActive;  // but checked)
  const bool rec_first = B == 1 && cluster_x && proj_ctas <= kProjFlags && g_dense_launch_order.load() == 0 &&
                         !(blocking != nullptr && blocking[0] == '1') && capture == cudaStreamCaptureStatusNone &&
                         xproj_cluster_prepare(false, T * B) == cudaSuccess;
  cudaError_t e = cudaMemsetAsync(workspace, 0, kDensePOffset, s);
  XprojSignal sig;
  sig.flags = flags;
  sig.epoch = 1u;
  auto projection = [&]() {
    return cluster_x ? launch_xproj_cluster(Wx, false, D, H, H, x, D, T * B, D, P, 4 * H, status, 2000000000LL, s,
                                            8, rec_first ? &sig : nullptr)
                     : launch_rows_gemm(Wx, false, D, H, H, x, D, T * B, D, P, 4 * H, 0, nullptr, nullptr, 0, s);
  };
  if (e == cudaSuccess && !rec_first) e = projection();
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "projection launch: %s", cudaGetErrorString(e));
  e = launch_dense(Wh, bias, P, h0, c0, out_h, out_c, status, H, T, B, 2000000000LL, s, rec_first ? flags : nullptr,
                   proj_ctas, 1u);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "recurrence launch: %s", cudaGetErrorString(e));
  if (rec_first) {
    e = projection();
    if (e != cudaSuccess)
      return report(msg, msg_len, LSTM_APPROX_ECUDA, "projection launch: %s", cudaGetErrorString(e));
  }
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "synchronise: %s", cudaGetErrorString(e));
  int code = 0;
  e = cudaMemcpy(&code, status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "status read: %s", cudaGetErrorString(e));
  if (code != 0) return report(msg, msg_len, LSTM_APPROX_ETIMEOUT, "a bounded in-kernel wait ran out (code %d)", code);
  return LSTM_APPROX_OK;
}

extern "C" size_t lstm_approx_dense_workspace_bytes(int H, int T, int B) {
  if (H < 1 || T < 1 || B < 1) return 0;
  return kDensePOffset + (size_t)T * B * 4 * H * sizeof(float);
}
