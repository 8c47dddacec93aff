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

// Bulk copy (TMA engine) of `bytes` from this CTA's shared memory to shared
// memory of a CTA of the cluster (dst and the mbarrier are cluster addresses
// of that CTA, from mapa), completing `bytes` on that mbarrier.  Addresses
// and size are multiples of 16 bytes.
__device__ __forceinline__ void bulk_copy_s2cluster(uint32_t dst_cluster, uint32_t src_cta, uint32_t bytes,
                                                    uint32_t mb_cluster) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst_cluster),
      "r"(src_cta), "r"(bytes), "r"(mb_cluster)
      : "memory");
}

// 4-byte load from shared memory of a CTA of the cluster (address from mapa).
__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

// Orders this thread's generic-proxy shared-memory writes before later
// async-proxy (bulk copy) reads of them.
__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bulk copy (TMA engine, no tensor map) of `bytes` from global to this CTA's
// shared memory, completing `bytes` on the mbarrier at `mb`.  Addresses and
// size must be multiples of 16 bytes.
__device__ __forceinline__ void bulk_copy_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t mb) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(mb)
               : "memory");
}

// Programmatic dependent launch: the kernel that follows in the stream may
// start (and run its set-up) once every CTA of this grid has signalled;
// griddep_wait() in that kernel blocks until this grid has completed and
// its memory operations are visible.
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Completion flag of a CTA of another grid: its stores before the call are
// visible to a thread that reads `epoch` from the flag with acquire
// semantics.  The caller orders the CTA's stores before it (a CTA barrier).
__device__ __forceinline__ void flag_release(unsigned* flag, unsigned epoch) {
  __threadfence();
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(flag), "r"(epoch) : "memory");
}

// Bounded wait of the calling warp until flags[0, n) all hold `epoch`;
// gives up after limit_ns of wall time or once *err is set.  Each pass
// reads every flag with relaxed loads (they overlap, where acquire loads
// would each wait for the one before), and one acquire fence after the
// pass that saw them all orders the caller's later reads after the writes
// the flags release.  Warp-uniform result.
__device__ __forceinline__ bool wait_flags_epoch(const unsigned* flags, int n, unsigned epoch, uint64_t limit_ns,
                                                 const volatile int* err) {
  const int lane = threadIdx.x & 31;
  uint64_t t0 = 0;
  for (;;) {
    bool mine = true;
    for (int i = lane; i < n; i += 32) {
      unsigned v;
      asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(flags + i) : "memory");
      mine = mine && v == epoch;
    }
    if (__all_sync(0xffffffffu, mine)) {
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
      return true;
    }
    if (__any_sync(0xffffffffu, *err != 0)) return false;
    const uint64_t now = global_timer_ns();
    if (t0 == 0) t0 = now;
    else if (now - t0 > limit_ns) return false;
    __nanosleep(32);
  }
}

// Makes a value opaque to the compiler, so that it stays in its register for
// the rest of a persistent kernel instead of being loaded again from memory
// where it is used.
__device__ __forceinline__ void keep_in_register(float& v) { asm volatile("" : "+f"(v)); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// 1/x from the hardware approximation (rcp.approx: about 1 ulp; 1/inf = 0).
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// Logistic function 1 / (1 + e^-z) from the hardware exponential and
// reciprocal: absolute error of a few 1e-7 over the whole range.
__device__ __forceinline__ float sigmoid_f(float z) { return rcp_approx(1.0f + __expf(-z)); }

// tanh z with a relative error of a few 1e-7: (1 - e) / (1 + e), e = exp(-2|z|),
// for |z| >= 1/4, and the Taylor series of tanh to z^9 below (its first
// omitted term, 1382 z^11 / 155925, is under 3e-9 there), which avoids the
// cancellation of 1 - e at small |z|.
__device__ __forceinline__ float tanh_f(float z) {
  const float a = fabsf(z);
  const float e = __expf(-2.0f * a);
  const float big = copysignf((1.0f - e) * rcp_approx(1.0f + e), z);
  const float z2 = z * z;
  const float poly = z2 * fmaf(z2, fmaf(z2, fmaf(z2, 62.0f / 2835.0f, -17.0f / 315.0f), 2.0f / 15.0f), -1.0f / 3.0f);
  const float small = fmaf(z, poly, z);
  return a < 0.25f ? small : big;
}

// tanh z = 2 sigmoid(2z) - 1: branch-free, absolute error about 2e-7 (the
// cancellation near 0 costs relative accuracy there, not absolute).  For
// the bf16 tensor-core epilogues, whose bound is 2e-2 elementwise; the fp32
// paths use tanh_f.
__device__ __forceinline__ float tanh_s(float z) { return fmaf(2.0f, sigmoid_f(2.0f * z), -1.0f); }

// The cell update below for the bf16 tensor-core epilogues, with seven
// special-function operations per cell instead of ten: the four gates are
// sigmoids (the cell gate as tanh z = 2 sigmoid(2z) - 1) of denominators
// d = 1 + e^-z, and their four reciprocals come from one reciprocal of the
// product d0 d1 d2 d3 (1/d0 = d1 (d2 d3) / (d0 d1 d2 d3), and so on: about
// 4 ulp).  The arguments are clamped at -20 so that the product stays
// finite; that moves a sigmoid by at most 2.1e-9.
__device__ __forceinline__ void lstm_cell_s(float yi, float yf, float yg, float yo, float c_prev, float& h_out,
                                            float& c_out) {
  const float d0 = 1.0f + __expf(-fmaxf(yi, -20.0f)), d1 = 1.0f + __expf(-fmaxf(yf, -20.0f));
  const float d2 = 1.0f + __expf(-fmaxf(2.0f * yg, -20.0f)), d3 = 1.0f + __expf(-fmaxf(yo, -20.0f));
  const float p01 = d0 * d1, p23 = d2 * d3;
  const float r = rcp_approx(p01 * p23);
  const float r01 = r * p23, r23 = r * p01;  // 1 / (d0 d1), 1 / (d2 d3)
  const float i = r01 * d1, f = r01 * d0, g = fmaf(2.0f, r23 * d3, -1.0f), o = r23 * d2;
  c_out = fmaf(f, c_prev, i * g);
  h_out = o * tanh_s(c_out);
}

// Gate nonlinearities and cell update (Sec. II): i, f, o sigmoid, g tanh;
// c = f c_prev + i g; h = o tanh(c).  Pre-activations already include bias.
__device__ __forceinline__ void lstm_cell_f(float yi, float yf, float yg, float yo, float c_prev,
                                            float& h_out, float& c_out) {
  const float i = sigmoid_f(yi), f = sigmoid_f(yf), g = tanh_f(yg), o = sigmoid_f(yo);
  c_out = fmaf(f, c_prev, i * g);
  h_out = o * tanh_f(c_out);
}


// ---- TMA (tensor maps) ---------------------------------------------------

// 2-D tiled load of the box at (c0 = innermost element, c1 = row) into
// shared memory at `dst`, completing its bytes on the mbarrier `mb`.  c0 must
// be a multiple of 16 bytes' worth of elements.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, uint32_t mb, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(mb), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ void tma_prefetch_map(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

// ---- tcgen05: tensor memory and the 5th-generation MMA --------------------

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 operands, fp32 accumulate; issued by
// one thread.  `accumulate` = 0 overwrites D.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier when every tcgen05 operation issued so far by
// this thread has completed.
__device__ __forceinline__ void umma_commit(uint32_t mb) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mb) : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns of tensor memory: thread i of the
// warp gets row (lane base + i), columns [col, col + 16).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 lanes x 8 consecutive 32-bit columns and the wait for them in one
// statement.
__device__ __forceinline__ void tmem_ld8_sync(uint32_t taddr, float (&v)[8]) {
  uint32_t r[8];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// Four loads of 32 lanes x 8 consecutive 32-bit columns (at t0 .. t3) and
// the wait for them in one statement, so that no use of the values can be
// scheduled before they have arrived: v[i][c] = column t_i + c of this
// thread's row.
__device__ __forceinline__ void tmem_ld8x4_sync(uint32_t t0, uint32_t t1, uint32_t t2, uint32_t t3,
                                                float (&v)[4][8]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%8, %9, %10, %11, %12, %13, %14, %15}, [%33];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%16, %17, %18, %19, %20, %21, %22, %23}, [%34];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%24, %25, %26, %27, %28, %29, %30, %31}, [%35];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(t0), "r"(t1), "r"(t2), "r"(t3)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i >> 3][i & 7] = __uint_as_float(r[i]);
}

// Five loads of 32 lanes x 8 consecutive 32-bit columns (at t0 .. t4) and
// the wait for them in one statement: v[i][c] = column t_i + c of this
// thread's row (i < 4), w[c] = column t4 + c.
__device__ __forceinline__ void tmem_ld8x5_sync(uint32_t t0, uint32_t t1, uint32_t t2, uint32_t t3, uint32_t t4,
                                                float (&v)[4][8], float (&w)[8]) {
  uint32_t r[40];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%40];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%8, %9, %10, %11, %12, %13, %14, %15}, [%41];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%16, %17, %18, %19, %20, %21, %22, %23}, [%42];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%24, %25, %26, %27, %28, %29, %30, %31}, [%43];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%32, %33, %34, %35, %36, %37, %38, %39}, [%44];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39])
      : "r"(t0), "r"(t1), "r"(t2), "r"(t3), "r"(t4)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i >> 3][i & 7] = __uint_as_float(r[i]);
#pragma unroll
  for (int i = 0; i < 8; ++i) w[i] = __uint_as_float(r[32 + i]);
}

// Two tmem_ld16 and one wait for both in one statement, so that no use of
// the values can be scheduled before they have arrived.
__device__ __forceinline__ void tmem_ld16x2_sync(uint32_t ta, uint32_t tb, float (&va)[16], float (&vb)[16]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, "
      "%29, %30, %31}, [%33];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(ta), "r"(tb)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    va[i] = __uint_as_float(r[i]);
    vb[i] = __uint_as_float(r[16 + i]);
  }
}

// Two 16-column tensor-memory loads issued without waiting for them: the
// values may be used only after tmem_wait_ld_tie32 on the same array, which
// waits for every tensor-memory load of the thread and then marks the
// registers as redefined, so that the compiler schedules no use before it.
__device__ __forceinline__ void tmem_ld16x2_issue(uint32_t ta, uint32_t tb, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, "
      "%29, %30, %31}, [%33];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(ta), "r"(tb)
      : "memory");
}
__device__ __forceinline__ void tmem_wait_ld_tie32(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
  asm volatile("" : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]));
  asm volatile("" : "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31]));
}

// tmem_ld16 and the wait for it in one statement, so that no use of the
// values can be scheduled before they have arrived.
__device__ __forceinline__ void tmem_ld16_sync(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Store 16 consecutive 32-bit columns per lane (rows lane base + i) into
// tensor memory; complete with tmem_wait_st().
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])),
      "r"(__float_as_uint(v[11])), "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])),
      "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15]))
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with
// 128-byte swizzling: rows of 64 elements (128 B), 8-row groups 1024 B apart.
// The tile must start on a 1024-byte boundary; advancing along K inside the
// 128-byte row adds the byte offset to the start-address field.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);  // start address (16-byte units)
  d |= static_cast<uint64_t>(1) << 16;                   // leading-dimension offset (unused when swizzled)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;           // stride-dimension offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1) << 46;                   // descriptor version of tcgen05
  d |= static_cast<uint64_t>(2) << 61;                   // 128-byte swizzle
  return d;
}

// The same with 8-row groups `sbo` bytes apart (a multiple of 1024), for a
// tile whose row groups are interleaved with other tiles' groups.
__device__ __forceinline__ uint64_t umma_desc_sw128_sbo(uint32_t saddr, uint32_t sbo) {
  return (umma_desc_sw128(saddr) & ~(static_cast<uint64_t>(0x3FFF) << 32)) |
         (static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32);
}

// Byte offset of bf16 element k (< 64) of row r in a K-major tile of
// 128-byte rows with 128-byte swizzling (the layout TMA writes and the MMA
// descriptors above read), relative to the 1024-byte aligned group of 8 rows
// that holds row r: the 16-byte chunk index is XORed with r mod 8.
__host__ __device__ __forceinline__ uint32_t sw128_offset(int r, int k) {
  return static_cast<uint32_t>((r & 7) * 128 + ((((k >> 3) ^ r) & 7) << 4) + (k & 7) * 2);
}

// Shared-memory matrix descriptor of a K-major bf16 tile with 64-byte
// swizzling: rows of 32 elements (64 B), 8-row groups `sbo` bytes apart
// (512 when dense).  The tile starts on a 512-byte boundary; advancing by 16
// elements inside the row adds 32 B to the start address.
__device__ __forceinline__ uint64_t umma_desc_sw64(uint32_t saddr, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(4) << 61;  // 64-byte swizzle
  return d;
}

// Byte offset of bf16 element k (< 32) of row r in a K-major tile of 64-byte
// rows with 64-byte swizzling, relative to the 512-byte aligned group of 8
// rows: the 16-byte chunk index (2 bits) is XORed with address bits 7-8,
// which within the group are (r mod 8) / 2.
__host__ __device__ __forceinline__ uint32_t sw64_offset(int r, int k) {
  return static_cast<uint32_t>((r & 7) * 64 + ((((k >> 3) ^ ((r & 7) >> 1)) & 3) << 4) + (k & 7) * 2);
}

// Instruction descriptor of kind::f16 with bf16 A and B, fp32 D, both
// operands K-major, M x N.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

}  // namespace lstm_approx_dev
