// Hoisted input projection for few columns (T*B <= 256, 32 columns per
// launch chunk along grid z): P[n][(g,k)] =
// prune(v_{g,k})[0:D]^T x_n for every timestep and stream at once (the x
// columns of x~ = [x_t; h_{t-1}], Sec. III, split off Eq. 1's dot products).
//
// With T*B this small the product is a skinny matrix times a thin one and
// the whole packed V_x is read once, so the kernel is about latency: every
// CTA owns 32 rows and one of S chunks of D (S CTAs of a cluster along D).
// It stages its chunk of D, 128 values of its 32 rows of V_x and of the x
// columns at a time, with 16-byte asynchronous copies spread over all its
// threads, through a ring of as many such groups as about 200 KB of shared
// memory holds (one commit group each): all of them are in flight from the
// start, the 8 warps consume them in order, and a freed slot is refilled
// with the next group.  Each lane accumulates a 4-row x NC-column register
// tile.  The 8 warp partials are summed in shared memory in warp
// order; each CTA then pushes its chunk sums of the outputs another CTA
// finishes to that CTA (16-byte st.async completing the owner's mbarrier),
// and the owner adds the S chunk sums in chunk order, so the result does not
// depend on timing.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kRows = 32;     // rows per CTA
constexpr int kCols = 32;     // columns per launch chunk (grid z covers T*B <= 256)
constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kGrp = 128;     // values of D per staged group (one commit group)
constexpr int kPadF = 4;      // floats of padding after each staged row
constexpr int kMaxSplit = 8;  // CTAs per cluster along D (16-CTA clusters start too far apart)
constexpr int kHdr = 32;      // mbarrier of the incoming chunk sums
constexpr size_t kRingBudget = 200 * 1024;  // shared memory of the staging ring
static_assert(kRows * kCols == 4 * kThreads, "each thread pushes one float4 of chunk sums");

template <typename TF>
constexpr int v_stride() {  // staged V_x row stride in elements (16-byte multiple)
  return kGrp + kPadF * 4 / (int)sizeof(TF);
}
constexpr int kXStride = kGrp + kPadF;

// one ring slot: 32 rows of V_x and the 4 NC x columns of one group
template <typename TF, int NC>
constexpr size_t slot_bytes() {
  return (size_t)kRows * v_stride<TF>() * sizeof(TF) + (size_t)4 * NC * kXStride * 4;
}
template <typename TF, int NC>
constexpr int ring_slots() {
  return kRingBudget / slot_bytes<TF, NC>() > 8 ? 8 : (int)(kRingBudget / slot_bytes<TF, NC>());
}

// header | staging ring (later the warp partials) | red [32*32] | slot [32*32]
template <typename TF, int NC>
constexpr size_t smem_bytes() {
  const size_t ring = (size_t)ring_slots<TF, NC>() * slot_bytes<TF, NC>();
  const size_t parts = (size_t)kWarps * kRows * kCols * 4;
  return kHdr + (ring > parts ? ring : parts) + 2 * (size_t)kRows * kCols * 4;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Issues the 16-byte copies of values [d0, d0 + len) of the CTA's rows of
// V_x and of the N x columns into one ring slot, as one commit group.
template <typename TF>
__device__ __forceinline__ void stage_group(const TF* A, int lda, int K, int Ks, int row0, int vrows,
                                            const float* X, int ldxin, int N, int d0, int len, TF* vs,
                                            float* xs, int tid) {
  constexpr int VS = v_stride<TF>();
  constexpr int kPer = 16 / (int)sizeof(TF);  // values per copy
  const int vq = len / kPer;
  for (int i = tid; i < vrows * vq; i += kThreads) {
    const int rr = i / vq, c = i - rr * vq;
    const int r = row0 + rr;
    const TF* src = A + (long long)((r / K) * Ks + r % K) * lda + d0 + c * kPer;
    cp_async16(smem_u32(vs + rr * VS + c * kPer), src);
  }
  const int xq = len / 4;
  for (int i = tid; i < N * xq; i += kThreads) {
    const int n = i / xq, c = i - n * xq;
    cp_async16(smem_u32(xs + n * kXStride + 4 * c), X + (long long)n * ldxin + d0 + 4 * c);
  }
  cp_async_commit();
}

// The same for a full group of kGrp values, from per-thread source pointers
// computed once per kernel: thread tid copies piece tid % VQ of V_x rows
// tid / VQ + RP j and of x columns tid / 32 + 8 j.
template <typename TF>
struct FullGroupCopies {
  static constexpr int kPer = 16 / (int)sizeof(TF);  // values per copy
  static constexpr int VQ = kGrp / kPer;              // copies per row
  static constexpr int RP = kThreads / VQ;            // rows per pass
  static constexpr int NP = kRows / RP;               // passes over the 32 rows
  const TF* v[NP];     // source of this thread's piece of row tid / VQ + RP j at d = 0 (null: no row)
  const float* x[4];   // source of its piece of x column tid / 32 + 8 j (null: no column)
  __device__ FullGroupCopies(const TF* A, int lda, int K, int Ks, int row0, int vrows, const float* X, int ldxin,
                             int N, int tid) {
#pragma unroll
    for (int j = 0; j < NP; ++j) {
      const int rr = tid / VQ + RP * j, r = row0 + rr;
      v[j] = rr < vrows ? A + (long long)((r / K) * Ks + r % K) * lda + (tid % VQ) * kPer : nullptr;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = tid / 32 + 8 * j;
      x[j] = n < N ? X + (long long)n * ldxin + 4 * (tid % 32) : nullptr;
    }
  }
  __device__ void issue(int d0, TF* vs, float* xs, int tid) const {
    constexpr int VS = v_stride<TF>();
#pragma unroll
    for (int j = 0; j < NP; ++j)
      if (v[j] != nullptr) cp_async16(smem_u32(vs + (tid / VQ + RP * j) * VS + (tid % VQ) * kPer), v[j] + d0);
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (x[j] != nullptr) cp_async16(smem_u32(xs + (tid / 32 + 8 * j) * kXStride + 4 * (tid % 32)), x[j] + d0);
    cp_async_commit();
  }
};

__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ float4 lds4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ float4 lds4(const __nv_bfloat16* p) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u), __uint_as_float(u.y << 16),
                     __uint_as_float(u.y & 0xFFFF0000u));
}

// Lane (rg = lane >> 2, cg = lane & 3) of every warp owns rows 4*rg .. 4*rg+3
// of the CTA's 32 and columns cg*NC .. cg*NC + NC - 1.
template <typename TF, int NC>
__global__ void __launch_bounds__(kThreads) xproj_kernel(const TF* __restrict__ A, int lda, int K, int Ks,
                                                         const float* __restrict__ X, int ldxin, int N, int D,
                                                         int dchunk, float* __restrict__ out, int ldo, int S,
                                                         int* err, long long limit_ns, unsigned* done_flags,
                                                         unsigned epoch) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);  // [0]: incoming chunk sums
  // ring slot s: V_x rows [32][v_stride] then x columns [4 NC][kXStride]
  unsigned char* ring = smem_raw + kHdr;
  constexpr size_t kSlot = slot_bytes<TF, NC>();
  constexpr int NG = ring_slots<TF, NC>();
  float* part = reinterpret_cast<float*>(smem_raw + kHdr);  // [warp][n * 32 + r], after the last group
  float* red = reinterpret_cast<float*>(smem_raw + smem_bytes<TF, NC>() - 2 * (size_t)kRows * kCols * 4);
  float* slot = red + kRows * kCols;  // [S][opc]: chunk c's sums of the outputs this CTA finishes
  constexpr int VS = v_stride<TF>();

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rg = lane >> 2, cg = lane & 3;
  const int rb = blockIdx.x;
  // column chunk blockIdx.z of 32 (launches with more than 32 columns)
  X += (long long)blockIdx.z * kCols * ldxin;
  out += (long long)blockIdx.z * kCols * ldo;
  N = min(kCols, N - (int)blockIdx.z * kCols);
  const uint32_t q = S > 1 ? cluster_ctarank() : 0u;  // chunk of D
  const int nrows = 4 * K;
  const int vrows = min(kRows, nrows - rb * kRows);
  const int c_lo = min(D, (int)q * dchunk), c_hi = min(D, c_lo + dchunk);
  const int opc = kRows * kCols / S;  // outputs finished per CTA
  const uint32_t bar_red = smem_u32(&bars[0]);
  const uint64_t limit = static_cast<uint64_t>(limit_ns);

  griddep_launch_dependents();  // the recurrence kernel may start its set-up
  if (tid == 0) {
    mbar_init(bar_red, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (S > 1) mbar_arrive_expect_tx(bar_red, (uint32_t)((S - 1) * opc * 4));
  }
  __syncthreads();
  // the peers push their chunk sums only after this CTA's barrier is armed
  // (their cluster wait below); arriving now hides the barrier's latency
  if (S > 1) cluster_arrive_release();

  float acc[4][NC];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < NC; ++j) acc[i][j] = 0.f;

  bool ok = true;
  auto slot_v = [&](int sl) { return reinterpret_cast<TF*>(ring + sl * kSlot); };
  auto slot_x = [&](int sl) {
    return reinterpret_cast<float*>(ring + sl * kSlot + (size_t)kRows * VS * sizeof(TF));
  };
  const int ngrp = (c_hi - c_lo + kGrp - 1) / kGrp;
  const FullGroupCopies<TF> full(A, lda, K, Ks, rb * kRows, vrows, X, ldxin, N, tid);
  auto stage = [&](int gi, int sl) {  // group gi of the chunk into ring slot sl
    const int d0 = c_lo + gi * kGrp, len = min(kGrp, c_hi - d0);
    if (len == kGrp) full.issue(d0, slot_v(sl), slot_x(sl), tid);
    else stage_group(A, lda, K, Ks, rb * kRows, vrows, X, ldxin, N, d0, len, slot_v(sl), slot_x(sl), tid);
  };
  // the first NG groups all in flight (an empty commit group past the end
  // keeps the count of groups behind the one consumed constant)
#pragma unroll 1
  for (int i = 0; i < NG; ++i) {
    if (i < ngrp) stage(i, i);
    else cp_async_commit();
  }
  // rows and columns that are never loaded read as zero (filled while the
  // copies are in flight; disjoint from what they write)
  if (vrows < kRows || N < 4 * NC) {
    for (int sl = 0; sl < NG && sl < ngrp; ++sl) {
      TF* vs = slot_v(sl);
      float* xs = slot_x(sl);
      for (int i = vrows * VS + tid; i < kRows * VS; i += kThreads) vs[i] = TF(0.f);
      for (int i = N * kXStride + tid; i < 4 * NC * kXStride; i += kThreads) xs[i] = 0.f;
    }
  }
#pragma unroll 1
  for (int i = 0; i < ngrp; ++i) {
    const int sl = i % NG, len = min(kGrp, c_hi - (c_lo + i * kGrp));  // a multiple of 8 (D % 8 == 0)
    cp_async_wait<NG - 1>();  // group i has landed (NG - 1 later groups may still be in flight)
    __syncthreads();          // every thread's copies of it (and the zero fill) are visible
    const TF* vs = slot_v(sl);
    const float* xs = slot_x(sl);
    // this warp's share of the group, in multiples of 4
    const int wlen = ((len + kWarps - 1) / kWarps + 3) & ~3;
    const int e_lo = min(len, warp * wlen), e_hi = min(len, warp * wlen + wlen);
    for (int e = e_lo; e < e_hi; e += 4) {
      float4 va[4], xb[NC];
#pragma unroll
      for (int r = 0; r < 4; ++r) va[r] = lds4(vs + (4 * rg + r) * VS + e);
#pragma unroll
      for (int j = 0; j < NC; ++j) xb[j] = lds4(xs + (cg * NC + j) * kXStride + e);
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int j = 0; j < NC; ++j) {
          float s = acc[r][j];
          s = fmaf(va[r].x, xb[j].x, s);
          s = fmaf(va[r].y, xb[j].y, s);
          s = fmaf(va[r].z, xb[j].z, s);
          s = fmaf(va[r].w, xb[j].w, s);
          acc[r][j] = s;
        }
    }
    __syncthreads();  // the slot is free: refill it with group i + NG
    if (i + NG < ngrp) stage(i + NG, sl);
    else cp_async_commit();
  }

  // warp partials, then their sum in warp order
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < NC; ++j) {
      const int n = cg * NC + j;
      if (n < kCols) part[(warp * kCols + n) * kRows + 4 * rg + i] = acc[i][j];
    }
  __syncthreads();
  for (int o = tid; o < kRows * kCols; o += kThreads) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += part[w * kRows * kCols + o];
    red[o] = s;
  }
  __syncthreads();
  if (S > 1) {
    cluster_wait_acquire();  // every CTA of the cluster has armed its barrier
    // thread tid hands outputs 4 tid .. 4 tid + 3 to the CTA that finishes them
    const int o = 4 * tid, owner = o / opc;
    const float4 v = *reinterpret_cast<const float4*>(red + o);
    float* dst = slot + q * opc + (o - owner * opc);
    if (owner == (int)q) {
      *reinterpret_cast<float4*>(dst) = v;
    } else {
      st_async_v4(mapa_shared(smem_u32(dst), (uint32_t)owner), v.x, v.y, v.z, v.w,
                  mapa_shared(bar_red, (uint32_t)owner));
    }
    const bool got = mbar_wait_bounded<true>(bar_red, 0, limit, err);
    if (!got) atomicCAS(err, 0, kErrTcTimeout);
    ok = __syncthreads_and(ok && got);  // also publishes the local slot writes
    if (ok) {
      for (int i = tid; i < opc; i += kThreads) {
        float s = 0.f;
        for (int c = 0; c < S; ++c) s += slot[c * opc + i];
        const int oo = (int)q * opc + i;
        const int n = oo / kRows, r = rb * kRows + oo % kRows;
        if (n < N && r < nrows) out[(long long)n * ldo + (long long)(r / K) * Ks + r % K] = s;
      }
    }
  } else if (ok) {
    for (int o = tid; o < kRows * kCols; o += kThreads) {
      const int n = o / kRows, r = rb * kRows + o % kRows;
      if (n < N && r < nrows) out[(long long)n * ldo + (long long)(r / K) * Ks + r % K] = red[o];
    }
  }
  if (done_flags != nullptr) {
    // the recurrence kernel launched before this one waits for every CTA's flag
    __syncthreads();  // this CTA's outputs are stored
    if (tid == 0 && ok)
      flag_release(done_flags + ((long long)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x, epoch);
    // CTA 0 then stays until that recurrence has finished, so that this grid
    // completes after it: work later in the stream that starts as this grid's
    // programmatic dependent and waits for it sees the recurrence's outputs
    if (blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0) griddep_wait();
  }
  if (!ok) {
    // a wait ran out: copies or pushes issued before it may still be in
    // flight towards this CTA; let them land before it exits
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
  }
}

// Chunks of D per cluster: about half a CTA per SM in total, at least 128
// values of D each, and at most max_split.  (Beside a resident recurrence,
// twice as many CTAs made the whole call slower: D = 1024, 4K = 1024,
// T*B = 20: 68.7 against 60.0 us.)
int xproj_split(int row_tiles, int col_chunks, int D, int max_split) {
  int S = 1;
  while (S < kMaxSplit && S < max_split && row_tiles * col_chunks * S * 2 <= 148 && D >= 2 * S * 128) S *= 2;
  return S;
}

// Sets the kernel's shared-memory limit once per thread and device; this
// also loads the kernel's code on that device if the module is loaded
// lazily, which a launch that must start while another kernel runs
// (XprojSignal) cannot wait for.
template <typename TF, int NC>
cudaError_t prepare_nc() {
  static thread_local unsigned long long done = 0;  // bit d: device d prepared
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = dev < 64 ? 1ull << dev : 0ull;
  if (bit == 0 || (done & bit) == 0) {
    e = cudaFuncSetAttribute(xproj_kernel<TF, NC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem_bytes<TF, NC>());
    if (e != cudaSuccess) return e;
    done |= bit;
  }
  return cudaSuccess;
}

template <typename TF>
cudaError_t prepare_typed(int N) {
  switch ((min(N, kCols) + 3) / 4) {
    case 1: return prepare_nc<TF, 1>();
    case 2: return prepare_nc<TF, 2>();
    case 3: return prepare_nc<TF, 3>();
    case 4: return prepare_nc<TF, 4>();
    case 5: return prepare_nc<TF, 5>();
    case 6: return prepare_nc<TF, 6>();
    case 7: return prepare_nc<TF, 7>();
    case 8: return prepare_nc<TF, 8>();
    default: return cudaErrorInvalidValue;
  }
}

template <typename TF, int NC>
cudaError_t launch_nc(const TF* A, int lda, int K, int Ks, const float* X, int ldxin, int N, int D, float* out,
                      int ldo, int* err, long long limit_ns, cudaStream_t s, int max_split, const XprojSignal* sig) {
  auto kern = xproj_kernel<TF, NC>;
  constexpr size_t smem = smem_bytes<TF, NC>();
  const cudaError_t pe = prepare_nc<TF, NC>();
  if (pe != cudaSuccess) return pe;
  const int row_tiles = (4 * K + kRows - 1) / kRows;
  const int col_chunks = (N + kCols - 1) / kCols;
  const bool signals = sig != nullptr && sig->flags != nullptr;
  const int S = xproj_split(row_tiles, col_chunks, D, max_split);
  const int dchunk = (((D + S - 1) / S) + 7) & ~7;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(row_tiles, S, col_chunks);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = S;
  attr[0].val.clusterDim.z = 1;
  // after a recurrence kernel that waits for this one's flags: start as its
  // programmatic dependent (it signals at its start), never wait for it
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = signals ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, A, lda, K, Ks, X, ldxin, N, D, dchunk, out, ldo, S, err, limit_ns,
                            signals ? sig->flags : nullptr, signals ? sig->epoch : 0u);
}

template <typename TF>
cudaError_t launch_typed(const TF* A, int lda, int K, int Ks, const float* X, int ldxin, int N, int D, float* out,
                         int ldo, int* err, long long limit_ns, cudaStream_t s, int max_split,
                         const XprojSignal* sig) {
  switch ((min(N, kCols) + 3) / 4) {  // columns per lane (more than 32: chunks of 32)
    case 1: return launch_nc<TF, 1>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 2: return launch_nc<TF, 2>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 3: return launch_nc<TF, 3>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 4: return launch_nc<TF, 4>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 5: return launch_nc<TF, 5>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 6: return launch_nc<TF, 6>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 7: return launch_nc<TF, 7>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    case 8: return launch_nc<TF, 8>(A, lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split, sig);
    default: return cudaErrorInvalidValue;
  }
}

// ---------------------------------------------------------------------------
// compressed variant for very sparse v (few kept x columns per row): one warp
// per packed row walks its kept entries (value, column) and gathers the x
// values; lane partials are summed by a transposed butterfly, so lane l ends
// with column l >> (5 - log2 NC) of the row
// ---------------------------------------------------------------------------
template <int NV>
__device__ __forceinline__ void lanes_transpose_sum(float (&v)[NV], int lane) {
  constexpr int kSteps = NV == 32 ? 5 : NV == 16 ? 4 : NV == 8 ? 3 : NV == 4 ? 2 : NV == 2 ? 1 : 0;
#pragma unroll
  for (int st = 0; st < kSteps; ++st) {
    const int half = NV >> (st + 1);
    const int mask = 16 >> st;
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

template <int NC>
__global__ void __launch_bounds__(256) xproj_sparse_kernel(SparseXRows sr, int K, int Ks, const float* __restrict__ X,
                                                           int ldxin, int N, float* __restrict__ out, int ldo) {
  griddep_launch_dependents();  // the recurrence kernel may start its set-up
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);  // packed row (g, k)
  if (r >= 4 * K) return;
  const int g = r / K, k = r - g * K;
  const int beg = __ldg(sr.off[g] + k), end = __ldg(sr.off[g] + k + 1);
  float acc[NC];
#pragma unroll
  for (int n = 0; n < NC; ++n) acc[n] = 0.f;
  for (int e = beg + lane; e < end; e += 32) {
    const float v = __ldg(sr.val[g] + e);
    const int c = __ldg(sr.idx[g] + e);
#pragma unroll
    for (int n = 0; n < NC; ++n)
      if (n < N) acc[n] = fmaf(v, __ldg(X + (long long)n * ldxin + c), acc[n]);
  }
  lanes_transpose_sum<NC>(acc, lane);
  constexpr int kShift = NC == 32 ? 0 : NC == 16 ? 1 : NC == 8 ? 2 : NC == 4 ? 3 : NC == 2 ? 4 : 5;
  const int n = lane >> kShift;
  if ((lane & ((1 << kShift) - 1)) == 0 && n < N) out[(long long)n * ldo + (long long)g * Ks + k] = acc[0];
}

template <int NC>
cudaError_t launch_sparse_nc(const SparseXRows& sr, int K, int Ks, const float* X, int ldxin, int N, float* out,
                             int ldo, cudaStream_t s) {
  xproj_sparse_kernel<NC><<<(4 * K + 7) / 8, 256, 0, s>>>(sr, K, Ks, X, ldxin, N, out, ldo);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_xproj_sparse(const SparseXRows& sr, int K, int Ks, const float* X, int ldxin, int N, float* out,
                                int ldo, cudaStream_t s) {
  if (N <= 1) return launch_sparse_nc<1>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  if (N <= 2) return launch_sparse_nc<2>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  if (N <= 4) return launch_sparse_nc<4>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  if (N <= 8) return launch_sparse_nc<8>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  if (N <= 16) return launch_sparse_nc<16>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  if (N <= 32) return launch_sparse_nc<32>(sr, K, Ks, X, ldxin, N, out, ldo, s);
  return cudaErrorInvalidValue;
}

bool xproj_cluster_fits(int N, int D, const void* A, int lda, const float* X, int ldxin, bool a_bf16) {
  // 16-byte asynchronous copies need 16-byte aligned base pointers, rows and lengths
  const int a_align = a_bf16 ? 8 : 4;
  const bool bases_aligned = ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(X)) & 15u) == 0;
  // up to 8 chunks of 32 columns: beyond that every chunk re-reading the
  // CTA's rows costs more than a tiled GEMM
  return N >= 1 && N <= 8 * kCols && D % 8 == 0 && lda % a_align == 0 && ldxin % 4 == 0 && bases_aligned;
}

cudaError_t launch_xproj_cluster(const void* A, bool a_bf16, int lda, int K, int Ks, const float* X, int ldxin,
                                 int N, int D, float* out, int ldo, int* err, long long limit_ns, cudaStream_t s,
                                 int max_split, const XprojSignal* sig) {
  if (a_bf16)
    return launch_typed(static_cast<const __nv_bfloat16*>(A), lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns,
                        s, max_split, sig);
  return launch_typed(static_cast<const float*>(A), lda, K, Ks, X, ldxin, N, D, out, ldo, err, limit_ns, s, max_split,
                      sig);
}

cudaError_t xproj_cluster_prepare(bool a_bf16, int N) {
  return a_bf16 ? prepare_typed<__nv_bfloat16>(N) : prepare_typed<float>(N);
}

int xproj_cluster_ctas(int K, int N, int D, int max_split) {
  const int row_tiles = (4 * K + kRows - 1) / kRows;
  const int col_chunks = (N + kCols - 1) / kCols;
  return row_tiles * col_chunks * xproj_split(row_tiles, col_chunks, D, max_split);
}

}  // namespace lstm_approx_impl
