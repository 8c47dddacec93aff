// Inline-PTX helpers for sm_103a: shared-memory addressing, cluster ranks,
// distributed shared memory, mbarriers with bounded waits, TMA and tcgen05.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace lstm_approx_dev {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Address of the same shared-memory variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void fence_mbarrier_init_cluster() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_init(uint32_t mb, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(mb), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t mb, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t mb) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(mb) : "memory");
}

// One poll of an mbarrier phase (acquire at cluster scope, so data written
// by st.async from other CTAs of the cluster is visible once it returns 1).
// The suspend-time hint (ns) lets a waiting warp sleep in hardware instead
// of spinning, so it does not take issue slots from warps still working.
__device__ __forceinline__ uint32_t mbar_try_wait_cluster(uint32_t mb, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(mb), "r"(parity), "r"(20000u)
      : "memory");
  return ok;
}

__device__ __forceinline__ uint32_t mbar_try_wait_cta(uint32_t mb, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(mb), "r"(parity)
      : "memory");
  return ok;
}

// Bounded wait on an mbarrier phase.  Gives up after `limit_ns` of wall
// time, or early when *err is already non-zero (another CTA gave up).
// Returns true when the phase completed.
template <bool kCluster>
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t mb, uint32_t parity, uint64_t limit_ns,
                                                  const volatile int* err) {
  if (kCluster ? mbar_try_wait_cluster(mb, parity) : mbar_try_wait_cta(mb, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (kCluster ? mbar_try_wait_cluster(mb, parity) : mbar_try_wait_cta(mb, parity)) return true;
    if ((i & 15u) == 0u) {
      if (*err != 0) return false;
      if (global_timer_ns() - t0 > limit_ns) return false;
    }
  }
}

// 16-byte store into (possibly remote) shared memory of the cluster, which
// completes `bytes` of the transaction count of the mbarrier at `remote_mb`
// in the destination CTA.
__device__ __forceinline__ void st_async_v4(uint32_t remote_addr, float a, float b, float c, float d,
                                            uint32_t remote_mb) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
          remote_addr),
      "f"(a), "f"(b), "f"(c), "f"(d), "r"(remote_mb)
      : "memory");
}

// Bulk copy (TMA engine, no tensor map) of `bytes` from global to this CTA's
// shared memory, completing `bytes` on the mbarrier at `mb`.  Addresses and
// size must be multiples of 16 bytes.
__device__ __forceinline__ void bulk_copy_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t mb) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(mb)
               : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Logistic function from the hardware exponential and a correctly rounded
// reciprocal: relative error a few units in the last place of fp32.
__device__ __forceinline__ float sigmoid_f(float z) { return __frcp_rn(1.0f + __expf(-z)); }

// Gate nonlinearities and cell update (Sec. II): i, f, o sigmoid, g tanh;
// c = f c_prev + i g; h = o tanh(c).  Pre-activations already include bias.
__device__ __forceinline__ void lstm_cell_f(float yi, float yf, float yg, float yo, float c_prev,
                                            float& h_out, float& c_out) {
  const float i = sigmoid_f(yi), f = sigmoid_f(yf), g = tanhf(yg), o = sigmoid_f(yo);
  c_out = fmaf(f, c_prev, i * g);
  h_out = o * tanhf(c_out);
}

}  // namespace lstm_approx_dev
