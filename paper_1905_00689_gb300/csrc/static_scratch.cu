// Allocation-free entry point: the single-layer fp32 recurrence with its
// scratch in a fixed device array instead of handle-owned allocations.
//
// Who needs this: callers that must not allocate device memory once they
// are running.  A hard real-time control loop (the paper's own setting, a
// vehicle that must act within a latency budget) cannot afford cudaMalloc:
// its latency is unbounded, it can synchronise the device, and safety rules
// for such systems often forbid dynamic allocation after start-up.  A
// plug-in that runs inside a host framework which owns all device memory
// through its own allocator cannot call cudaMalloc either.  Such callers
// allocate the factors, inputs and outputs once, at start-up, and then call
// lstm_approx_run_static, which allocates nothing.
//
// The scratch (the hoisted input projection, the kernel status word and a
// zero bias) lives in g_static_scratch, a file-scope __device__ array of
// kStaticScratchFloats floats (4 MiB) that every GPU which loads this
// library holds until the process exits.  Host code cannot use the array's
// name as a device address, so the first call on each device looks the
// address up with cudaGetSymbolAddress (with that device current) and keeps
// it; that first call should therefore come before any stream capture.
// All calls share the array and it keeps the last call's contents: the
// status word and the zero bias are cleared on every call, and calls whose
// work overlaps on the GPU (other streams, other threads) race on it.
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <mutex>

#include "internal.h"

using namespace lstm_approx_impl;

namespace {

constexpr size_t kStaticScratchFloats = size_t(1) << 20;  // 4 MiB
constexpr size_t kHeaderFloats = 64;                      // status word, padding to 256 B

static __device__ __align__(256) float g_static_scratch[kStaticScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
float* g_scratch_addr[kMaxDevices] = {};

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

extern "C" int lstm_approx_run_static(const float* Vx, const float* Vh, const float* U, const float* sigma,
                                      const float* bias, int D, int H, int K, const float* x, int T, int B,
                                      const float* h0, const float* c0, float* out_h, float* out_c,
                                      const int* checkpoints, int J, float* ckpt_h, float* ckpt_c,
                                      void* cuda_stream, char* msg, int msg_len) {
  if (msg && msg_len > 0) msg[0] = '\0';
  if (!Vx || !Vh || !U || !sigma || !x || !out_h)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "Vx, Vh, U, sigma, x and out_h must not be NULL");
  if (D < 1 || H < 4 || H % 4 != 0 || K < 1 || T < 1 || B < 1)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "need D >= 1, H >= 4 with H %% 4 == 0, K, T, B >= 1");
  if ((reinterpret_cast<uintptr_t>(Vh) | reinterpret_cast<uintptr_t>(U)) & 15u)
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "Vh and U must be 16-byte aligned");
  if (J < 0 || J > kMaxCheckpoints || (J > 0 && !checkpoints))
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "J must be in [0, %d] with a checkpoint array", kMaxCheckpoints);
  Checkpoints ck;
  ck.n = J;
  for (int j = 0; j < kMaxCheckpoints; ++j) ck.k[j] = 0;
  for (int j = 0; j < J; ++j) {
    if (checkpoints[j] < 1 || checkpoints[j] > K || (j > 0 && checkpoints[j] <= checkpoints[j - 1]))
      return report(msg, msg_len, LSTM_APPROX_EINVAL, "checkpoints must increase strictly within [1, K]");
    ck.k[j] = checkpoints[j];
  }
  // scratch: header | zero bias (4H) | P (T*B*4K), each piece 256-byte aligned
  const size_t bias_floats = ((4ull * H + 63) / 64) * 64;
  const size_t p_floats = (size_t)T * B * 4ull * K;
  const size_t need = kHeaderFloats + bias_floats + p_floats;
  if (need > kStaticScratchFloats)
    return report(msg, msg_len, LSTM_APPROX_EINVAL,
                  "T*B*4K + 4H = %zu floats of scratch needed; the static scratch holds %zu floats "
                  "(T*B*K up to about %zu)",
                  need - kHeaderFloats, kStaticScratchFloats - kHeaderFloats,
                  (kStaticScratchFloats - kHeaderFloats - bias_floats) / 4);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  int major = 0, minor = 0, sms = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (major != 10 || minor != 3) return report(msg, msg_len, LSTM_APPROX_ECUDA, "needs an sm_103 device");
  if (dev < 0 || dev >= kMaxDevices) return report(msg, msg_len, LSTM_APPROX_ECUDA, "device index %d too large", dev);

  PersistentChoice plan;
  std::string why;
  if (!choose_persistent(H, K, T, ck, 0, sms, 0, &plan, &why))
    return report(msg, msg_len, LSTM_APPROX_EINVAL, "shape does not fit: %s", why.c_str());

  float* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_addr[dev]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_static_scratch);
      if (e != cudaSuccess)
        return report(msg, msg_len, LSTM_APPROX_ECUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
      g_scratch_addr[dev] = static_cast<float*>(p);
    }
    base = g_scratch_addr[dev];
  }
  int* status = reinterpret_cast<int*>(base);
  float* zero_bias = base + kHeaderFloats;
  float* P = zero_bias + bias_floats;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);

  e = cudaMemsetAsync(base, 0, (kHeaderFloats + (bias ? 0 : bias_floats)) * sizeof(float), s);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "clearing scratch: %s", cudaGetErrorString(e));
  // (a1) hoisted input projection into the static scratch
  e = xproj_cluster_fits(T * B, D, Vx, D, x, D, false)
          ? launch_xproj_cluster(Vx, false, D, K, K, x, D, T * B, D, P, 4 * K, status, 2000000000LL, s, 8)
          : launch_rows_gemm(Vx, false, D, K, K, x, D, T * B, D, P, 4 * K, 0, nullptr, nullptr, 0, s);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "projection launch: %s", cudaGetErrorString(e));
  PersistentArgs a{};
  a.Vh = Vh;
  a.U = U;
  a.sigma = sigma;
  a.bias = bias ? bias : zero_bias;
  a.P = P;
  a.h0 = h0;
  a.c0 = c0;
  a.out_h = out_h;
  a.c_last = out_c;
  a.ckpt_h = ckpt_h;
  a.ckpt_c = ckpt_c;
  a.err = status;
  a.H = H;
  a.K = K;
  a.Ks = K;
  a.ldh = H;
  a.T = T;
  a.B = B;
  a.ck = ck;
  a.wait_limit_ns = 2000000000LL;
  a.test_stall = 0;
  e = launch_persistent_choice(plan, a, s);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "recurrence launch: %s", cudaGetErrorString(e));
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "synchronise: %s", cudaGetErrorString(e));
  int code = 0;
  e = cudaMemcpy(&code, status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return report(msg, msg_len, LSTM_APPROX_ECUDA, "status read: %s", cudaGetErrorString(e));
  if (code != 0)
    return report(msg, msg_len, LSTM_APPROX_ETIMEOUT, "a bounded in-kernel wait ran out (code %d)", code);
  return LSTM_APPROX_OK;
}
