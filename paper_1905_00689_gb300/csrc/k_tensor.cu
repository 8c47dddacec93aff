// Large-batch tensor-core path (bf16 factors, fp32 accumulate).
//
// The factors u, v are stored in bf16.  The activations x, h and tau' are
// fp32 values; each enters the MMAs as a pair of bf16 planes, hi = bf16(a)
// and lo = bf16(a - hi), so that hi + lo equals a to about 2^-17 relative
// and every product is issued twice (factor tile x hi, factor tile x lo)
// into the same fp32 accumulator.  Rounding the activations to one bf16
// (unit roundoff 2^-9) instead gives elementwise errors of 0.03-0.2 on h
// and c; with the pair the kernels differ from fp64 arithmetic on the same
// bf16 factors by a few 1e-4.
//
// The two products of one timestep are dense contractions over B streams:
//   (a2) tau'[n][(g,k)] = sigma_{g,k} (P_t[n][(g,k)] + sum_j Vh[(g,k)][j] h_{t-1}[n][j])
//   (a3) y_g[n][j]      = sum_k U_g[j][k] tau'[n][(g,k)]
// and the hoisted input projection (a1) is the first one with x in place of
// h over all T*B columns (Eq. 1 with the augmentation of Sec. III).
//
// tc_rows_kernel computes one 128-row x BN-column tile of the first kind:
// warp 0 streams K-major tiles of the factor and of both planes of the
// activation with TMA (128-byte swizzle) through an S-stage mbarrier ring,
// one thread of warp 1 issues tcgen05.mma (M = 128, N = BN, K = 16 per
// instruction, once per plane) into a tensor-memory accumulator, and warps
// 4..11 (two per 32-lane quarter of tensor memory) read it back with
// tcgen05.ld for the epilogue: store P, or form tau' and store it as its
// bf16 pair.  For tau' the epilogue warps load their P_t values into
// registers while the mainloop streams.
//
// tc_gates_kernel computes, for 128 hidden units x NT streams, the four gate
// sums at once in four tensor-memory accumulators and runs the cell update
// of Sec. II in the epilogue (fp32 sigmoid, tanh as 2 sigmoid(2z) - 1:
// absolute error about 2e-7), storing h_t as its bf16 pair for the next step.  Intermediate depths k_j (multiples of 16) are
// read from the same accumulators when the MMA stream reaches them: the MMA
// thread commits, the epilogue warps compute the cell from the partial sums
// and hand the accumulators back -- no prefix is recomputed.
//
// When the stream tiles are too few to fill the GPU (small B), the gate
// GEMM's term axis is split over up to 8 CTAs per tile (grid z, 64-term
// chunks [kb0, kb1) each).  Such a CTA stores its raw gate sums, and at a
// depth that ends inside its range the sums up to that depth, to a scratch
// array; tc_gates_reduce_kernel then adds the splits in split order and runs
// the cell update at full depth and at every intermediate depth.  The same
// raw-sum mode (with one split if the grid is large enough) serves runs with
// an intermediate depth that is not a multiple of the MMA's 16 terms: the
// MMA stream stops at the depth's last slice boundary and the reduce kernel
// adds the remaining terms from U and the stored tau' pair.
//
// Every mbarrier wait is bounded in wall time; a wait that runs out writes
// the device status word, the CTA stops issuing work, waits (bounded) for
// its copies and MMAs in flight, frees its tensor memory and returns.
#include <cuda.h>

#include <cstring>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kTcThreads = 384;  // warps 0..3: TMA, MMA, TMEM, spare; warps 4..11: epilogue
constexpr int kTileM = 128;
constexpr int kTileK = 64;  // bf16 elements in one 128-byte swizzled row
constexpr uint32_t kABytes = kTileM * kTileK * 2;
constexpr int kConvGroups = 2;  // groups of epilogue warps converting alternate stages of fp32 activations

// Named barrier `id` of `count` threads; returns whether any of them passed `pred`.
__device__ __forceinline__ bool block_or(int id, int count, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
      "barrier.cta.red.or.pred q, %2, %3, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(pred ? 1u : 0u), "r"(id), "r"(count)
      : "memory");
  return r != 0u;
}
__device__ __forceinline__ void named_barrier(int id, int count) {
  asm volatile("barrier.cta.sync.aligned %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ bool wait_cta(uint32_t mb, uint32_t parity, uint64_t limit, const volatile int* err) {
  return mbar_wait_bounded<false>(mb, parity, limit, err);
}

// The bf16 pair of an fp32 value: hi = bf16(v), lo = bf16(v - hi), both
// round-to-nearest-even (v - hi is exact in fp32).
__device__ __forceinline__ void bf16_pair(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& w, float* f) {
  const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    f[2 * e] = __uint_as_float(v[e] << 16);
    f[2 * e + 1] = __uint_as_float(v[e] & 0xFFFF0000u);
  }
}

// Terms [k0, k0 + r) of gate g for stream n and unit j (0 < r < 16, k0 a
// multiple of 16): sum of u_{g,k}[j] (tau'_hi + tau'_lo)[n][(g, k)], from the
// factor U and the stored tau' pair.  These are the terms of an intermediate
// depth k_j = k0 + r that is not a multiple of the MMA's 16-term slices: the
// MMA stream stops at k0 and the reduce kernel adds them on the CUDA cores.
__device__ __forceinline__ float remainder_terms(const TcGatesArgs& a, int g, int n, int j, int k0, int r) {
  const uint4* up = reinterpret_cast<const uint4*>(a.U + ((long long)g * a.H + j) * a.Ks + k0);
  const long long o = (long long)n * a.ldt + (long long)g * a.Ks + k0;
  const uint4* th = reinterpret_cast<const uint4*>(a.tau + o);
  const uint4* tl = reinterpret_cast<const uint4*>(a.tau + a.tau_plane + o);
  float acc = 0.f;
#pragma unroll
  for (int h8 = 0; h8 < 2; ++h8) {
    float u[8], hi[8], lo[8];
    bf16x8_to_f32(__ldg(up + h8), u);
    bf16x8_to_f32(th[h8], hi);
    bf16x8_to_f32(tl[h8], lo);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (8 * h8 + k < r) acc = fmaf(u[k], hi[k] + lo[k], acc);
  }
  return acc;
}

// ---------------------------------------------------------------------------
// tile of tau' / P: rows of the packed factor matrix x columns (streams)
// ---------------------------------------------------------------------------
// XF (the projection with packed gates): the activation comes as fp32
// tiles (tmb is an fp32 map with boxes of 32 columns), and the epilogue
// warps, idle until the accumulator is complete, convert each stage's tile
// into its bf16 pair before the MMAs read it: x is read once from memory as
// fp32 instead of being converted by a separate pass (which reads it and
// writes its pair, the same bytes again).  The fp32 tile (BN rows x 64
// columns) lands where the pair goes (both planes: the same bytes); the
// converting threads read all of it into registers, meet at a named
// barrier, and write the pair over it.
template <int BN, int S, bool XF>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_rows_kernel(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmb, TcRowsArgs a) {
  extern __shared__ uint8_t smem_raw[];
  static_assert(BN <= 128, "the epilogue holds P_t of its columns in registers");
  constexpr uint32_t kBBytes = BN * kTileK * 2;        // one plane of the activation tile
  constexpr uint32_t kStage = kABytes + 2 * kBBytes;   // factor tile, hi plane, lo plane (XF: first the fp32 tile)
  constexpr uint32_t kCols = BN < 32 ? 32 : BN;
  constexpr int kNb = XF ? 3 * S : 2 * S;  // full[S] | empty[S] (| converted[S])
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t bar0 = base + S * kStage;  // the stage barriers, accum | drain | split | tmem slot
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem_raw + (bar0 - raw) + 8 * (kNb + 3));
  const uint32_t accum_bar = bar0 + 8u * kNb, drain_bar = accum_bar + 8u, split_bar = accum_bar + 16u;
  const uint32_t conv0 = bar0 + 8u * (2 * S);  // converted[s] (XF)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x / a.kt_per_gate, kt = blockIdx.x % a.kt_per_gate;
  const int row0 = g * a.Ks + kt * kTileM;
  // packed gates (a.rpg > 0, K <= rpg <= 32): the tile's rows are the first
  // rpg terms of each gate, gate g at tile rows [g rpg, (g + 1) rpg), loaded
  // by four copies of rpg rows; tile rows from 4 rpg on stay zero
  const int rpg = a.rpg;
  const uint32_t a_bytes = rpg > 0 ? 4u * rpg * kTileK * 2 : kABytes;
  const int col0 = blockIdx.y * BN;
  const int nkb = (a.Kdim + kTileK - 1) / kTileK;
  // reduction axis split over the sk CTAs of a cluster (grid z, mode 1):
  // this CTA's 64-element chunks [kb0, kb0 + nloc)
  const int sk = (!XF && BN <= 64 && a.sk > 1) ? a.sk : 1;
  const int kb0 = sk > 1 ? (int)blockIdx.z * a.nkb_per : 0;
  const int nloc = sk > 1 ? max(0, min(nkb, kb0 + a.nkb_per) - kb0) : nkb;
  const volatile int* err = a.err;
  const uint64_t limit = static_cast<uint64_t>(a.limit_ns);
  const bool add_p = a.mode == 1;  // tau' = sigma * (accumulator + P_t)
  // split (sk > 1, tiles of at most 64 columns): an epilogue thread's row and
  // columns of this CTA's partial sums, and that row's sigma and P_t
  constexpr int kSplitCols = BN <= 64 ? BN / 2 : 1;
  float sp_val[kSplitCols], sp_p[kSplitCols];
  float sp_sig = 0.f;

  griddep_launch_dependents();  // the next kernel may start its own set-up
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(bar0 + 8u * i, 1);
      mbar_init(bar0 + 8u * (S + i), 1);
      if (XF) mbar_init(conv0 + 8u * i, 8 / kConvGroups);  // one arrival per warp of the stage's converting group
    }
    mbar_init(accum_bar, 1);
    mbar_init(drain_bar, 1);
    // split: the partial sums of this CTA's rows pushed by the sk - 1 peers
    if (sk > 1) mbar_init(split_bar, 1);
    fence_mbarrier_init_cluster();
    if (sk > 1) mbar_arrive_expect_tx(split_bar, (uint32_t)((sk - 1) * (kTileM / sk) * BN * 4));
  }
  if (rpg > 0) {  // the factor tile's rows no copy writes: zero in every stage, before the MMAs read them
    const uint32_t zbytes = kABytes - a_bytes;
    for (uint32_t i = threadIdx.x; i < S * (zbytes / 16); i += blockDim.x) {
      const uint32_t st = i / (zbytes / 16), o = i % (zbytes / 16);
      *reinterpret_cast<uint4*>(smem_raw + (base - raw) + st * kStage + a_bytes + 16 * o) = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_shared();
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the factor copies of one stage into the tile at st
  auto load_a = [&](uint32_t st, uint32_t bar, int kb) {
    if (rpg == 0) {
      tma_load_2d(st, &tma, bar, kb * kTileK, row0);
    } else {
#pragma unroll
      for (int gg = 0; gg < 4; ++gg) tma_load_2d(st + gg * rpg * kTileK * 2, &tma, bar, kb * kTileK, gg * a.Ks);
    }
  };

  if (warp == 0 && lane == 0) {  // ---- TMA producer ----
    tma_prefetch_map(&tma);
    tma_prefetch_map(&tmb);
    int issued = 0;
    bool ok = true;
    // the factor tiles of the first S stages do not depend on the kernel
    // before this one: issue them before waiting for it
    const int npre = nloc < S ? nloc : S;
    constexpr uint32_t b_bytes = 2 * kBBytes;  // the pair, or (XF) the fp32 tile: the same bytes
    for (int i = 0; i < npre; ++i) {
      mbar_arrive_expect_tx(bar0 + 8u * i, a_bytes + b_bytes);
      load_a(base + i * kStage, bar0 + 8u * i, kb0 + i);
    }
    griddep_wait();
    for (int i = 0; i < nloc; ++i) {
      const int s = i % S, kb = kb0 + i;
      if (i >= S && !(ok = wait_cta(bar0 + 8u * (S + s), ((i / S) - 1) & 1, limit, err))) break;
      const uint32_t st = base + s * kStage;
      if (i >= npre) {
        mbar_arrive_expect_tx(bar0 + 8u * s, a_bytes + b_bytes);
        load_a(st, bar0 + 8u * s, kb);
      }
      if constexpr (XF) {  // the fp32 tile, columns [64 kb, 64 kb + 32) and [64 kb + 32, 64 kb + 64)
        tma_load_2d(st + kABytes, &tmb, bar0 + 8u * s, kb * kTileK, col0);
        tma_load_2d(st + kABytes + BN * 128u, &tmb, bar0 + 8u * s, kb * kTileK + 32, col0);
      } else {
        tma_load_2d(st + kABytes, &tmb, bar0 + 8u * s, kb * kTileK, col0);                      // hi plane
        tma_load_2d(st + kABytes + kBBytes, &tmb, bar0 + 8u * s, kb * kTileK, a.b_plane + col0);  // lo plane
      }
      ++issued;
    }
    if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
    // every issued copy has landed before the CTA may leave
    for (int s = 0; s < S && s < issued; ++s) {
      const int last = s + ((issued - 1 - s) / S) * S;
      wait_cta(bar0 + 8u * s, (last / S) & 1, limit, err);
    }
  } else if (warp == 1 && lane == 0) {  // ---- MMA issuer ----
    constexpr uint32_t idesc = umma_idesc_bf16(kTileM, BN);
    bool ok = true;
    for (int i = 0; i < nloc && ok; ++i) {
      const int s = i % S;
      // the stage's copies have landed (XF: and its activation has been converted)
      if (!(ok = wait_cta((XF ? conv0 : bar0) + 8u * s, (i / S) & 1, limit, err))) break;
      tc_fence_after();
      const uint32_t st = base + s * kStage;
      const uint64_t da = umma_desc_sw128(st);
      const uint64_t dhi = umma_desc_sw128(st + kABytes), dlo = umma_desc_sw128(st + kABytes + kBBytes);
#pragma unroll
      for (int kk = 0; kk < kTileK / 16; ++kk) {
        umma_bf16(tmem, da + 2ull * kk, dhi + 2ull * kk, idesc, (i | kk) != 0 ? 1u : 0u);
        umma_bf16(tmem, da + 2ull * kk, dlo + 2ull * kk, idesc, 1u);
      }
      umma_commit(bar0 + 8u * (S + s));  // frees the stage once these MMAs are done
    }
    if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
    umma_commit(accum_bar);
    umma_commit(drain_bar);
    wait_cta(drain_bar, 0, limit, err);
  } else if (warp >= 4) {  // ---- epilogue: warps 4..11, two per lane quarter ----
    const int ep = warp - 4, q = ep & 3;
    constexpr int kHalf = BN / 2;
    if constexpr (XF) {  // each stage's fp32 activation tile -> its bf16 pair, in place
      // kConvGroups groups of warps take the stages in turn (group g: stages kb = g mod kConvGroups),
      // so that several stages are converted at once
      constexpr int kGt = 256 / kConvGroups;  // threads per group
      static_assert(BN * 16 % kGt == 0, "whole chunks per thread");
      constexpr int kChunks = BN * 16 / kGt;  // 16-byte chunks of four columns per thread
      const int grp = ep / (8 / kConvGroups), ce = (threadIdx.x - 128) % kGt;
      uint8_t* gbase = smem_raw + (base - raw);
      bool cok = true;
      for (int kb = grp; kb < nkb; kb += kConvGroups) {
        const int s = kb % S;
        // every thread of the group takes the same decision (reduction barrier), so that
        // none of them waits at the group's second barrier for one that left
        const bool failed = !wait_cta(bar0 + 8u * s, (kb / S) & 1, limit, err);
        if (block_or(1 + 2 * grp, kGt, failed)) {
          cok = false;
          break;
        }
        uint8_t* st = gbase + s * kStage + kABytes;
        // chunk c = row n, columns [4 (c mod 16), +4): box (k4 / 32) of the fp32 tile
        float4 v[kChunks];
#pragma unroll
        for (int i = 0; i < kChunks; ++i) {
          const int c = ce + kGt * i, n = c >> 4, k4 = (c & 15) * 4;
          v[i] = *reinterpret_cast<const float4*>(st + (k4 >> 5) * (BN * 128) + n * 128 + (k4 & 31) * 4);
        }
        named_barrier(2 + 2 * grp, kGt);  // the whole fp32 tile is read before the pair overwrites it
#pragma unroll
        for (int i = 0; i < kChunks; ++i) {
          const int c = ce + kGt * i, n = c >> 4, k4 = (c & 15) * 4;
          __nv_bfloat16 h[4], l[4];
          bf16_pair(v[i].x, h[0], l[0]);
          bf16_pair(v[i].y, h[1], l[1]);
          bf16_pair(v[i].z, h[2], l[2]);
          bf16_pair(v[i].w, h[3], l[3]);
          const uint32_t o = sw128_offset(n, k4) + (uint32_t)(n >> 3) * 1024u;
          *reinterpret_cast<uint2*>(st + o) =
              make_uint2((uint32_t)__bfloat16_as_ushort(h[0]) | ((uint32_t)__bfloat16_as_ushort(h[1]) << 16),
                         (uint32_t)__bfloat16_as_ushort(h[2]) | ((uint32_t)__bfloat16_as_ushort(h[3]) << 16));
          *reinterpret_cast<uint2*>(st + kBBytes + o) =
              make_uint2((uint32_t)__bfloat16_as_ushort(l[0]) | ((uint32_t)__bfloat16_as_ushort(l[1]) << 16),
                         (uint32_t)__bfloat16_as_ushort(l[2]) | ((uint32_t)__bfloat16_as_ushort(l[3]) << 16));
        }
        fence_proxy_async_shared();
        __syncwarp();
        if (lane == 0) mbar_arrive(conv0 + 8u * s);
      }
      if (!cok) atomicCAS(a.err, 0, kErrTcTimeout);
    }
    const int cbeg = (ep >> 2) * kHalf;
    const int lrow = 32 * q + lane;
    const int k = rpg > 0 ? lrow % rpg : kt * kTileM + lrow;
    const int row = rpg > 0 ? (lrow / rpg) * a.Ks + k : row0 + lrow;
    const bool row_ok = k < a.K && (rpg == 0 || lrow < 4 * rpg);
    const uint32_t trow = tmem + ((32u * q) << 16);
    if (sk > 1) {
      // split: this thread's row and columns of the CTA's partial sums, and
      // (for the row's owner, below) its sigma and P_t, loaded while the
      // mainloop runs
      if constexpr (BN <= 64) {
#pragma unroll
        for (int c = 0; c < kHalf; ++c) {
          const int n = col0 + cbeg + c;
          sp_p[c] = (row_ok && n < a.N) ? __ldg(a.P + (long long)n * a.ldp + row) : 0.f;
        }
        sp_sig = row_ok ? a.sigma[row] : 0.f;
        const bool ok = wait_cta(accum_bar, 0, limit, err);
        tc_fence_after();
#pragma unroll
        for (int cc = 0; cc < kHalf; cc += 16) {
          float v[16];
          tmem_ld16(trow + cbeg + cc, v);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 16; ++j) sp_val[cc + j] = (ok && nloc > 0) ? v[j] : 0.f;
        }
      }
    } else {
    float preg[kHalf];  // P_t of this thread's row and columns, loaded while the mainloop runs
    if (add_p) {
#pragma unroll
      for (int c = 0; c < kHalf; ++c) {
        const int n = col0 + cbeg + c;
        preg[c] = (row_ok && n < a.N) ? __ldg(a.P + (long long)n * a.ldp + row) : 0.f;
      }
    }
    griddep_wait();  // the outputs below may still be read by the kernel before this one
    const bool ok = wait_cta(accum_bar, 0, limit, err);
    tc_fence_after();
    const float sig = (add_p && row_ok) ? a.sigma[row] : 0.f;
    const bool write = ok && *err == 0;
#pragma unroll
    for (int cc = 0; cc < kHalf; cc += 16) {
      const int c0 = cbeg + cc;
      float v[16];
      tmem_ld16(trow + c0, v);
      tmem_wait_ld();
      if (!write) continue;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int n = col0 + c0 + j;
        if (n >= a.N) break;
        if (!add_p) {
          if (row_ok) a.P[(long long)n * a.ldp + row] = v[j];
        } else if (rpg == 0 || lrow < 4 * rpg) {
          __nv_bfloat16 hi, lo;
          bf16_pair(row_ok ? sig * (v[j] + preg[cc + j]) : 0.f, hi, lo);
          a.tau[(long long)n * a.ldt + row] = hi;
          a.tau[a.tau_plane + (long long)n * a.ldt + row] = lo;
        }
      }
    }
    }
  }
  if constexpr (BN <= 64) {
    if (sk > 1) {
      // Every CTA of the cluster holds its partial sums of the whole tile (in
      // its epilogue threads' registers); CTA z finishes rows
      // [z RS, (z + 1) RS).  The threads of other rows push their values
      // into the owner's receive buffer (over its stage ring, free once the
      // cluster barrier shows every accumulator complete) with st.async,
      // which completes the owner's split barrier; each owning thread adds
      // the sk partials of its row in rank order (the result does not depend
      // on timing), forms tau' = sigma (sum + P_t) and stores its pair.
      __syncwarp();  // warps 0 and 1 reconverge after their single-lane roles
      cluster_sync_all();
      bool split_failed = false;  // an owning thread's wait for the pushes ran out
      if (warp >= 4) {
        const int ep = warp - 4, q = ep & 3, lrow = 32 * q + lane, cbeg = (ep >> 2) * (BN / 2);
        const int z = (int)blockIdx.z, RS = kTileM / sk, owner = lrow / RS;
        constexpr int RSTR = BN + 4;  // receive-row stride in floats (16-byte rows, banks skewed)
        // receive buffer [sender][row of the owner's block][RSTR] at the start of the stage ring
        const uint32_t recv = base;
        if (owner != z) {
          const uint32_t dst = mapa_shared(recv, (uint32_t)owner) +
                               4u * (uint32_t)((z * RS + (lrow - owner * RS)) * RSTR + cbeg);
          const uint32_t bar = mapa_shared(split_bar, (uint32_t)owner);
#pragma unroll
          for (int c = 0; c < BN / 2; c += 4)
            st_async_v4(dst + 4u * c, sp_val[c], sp_val[c + 1], sp_val[c + 2], sp_val[c + 3], bar);
        } else {
          const bool got = mbar_wait_bounded<true>(split_bar, 0, limit, err);  // pushes from other CTAs
          split_failed = !got;
          const float* rb = reinterpret_cast<const float*>(smem_raw + (recv - raw));
          griddep_wait();  // tau' may still be read by the kernel before this one
          const bool write = got && *err == 0;
          const int kr = kt * kTileM + lrow;
#pragma unroll
          for (int c = 0; c < BN / 2; ++c) {
            float sum = 0.f;
#pragma unroll
            for (int zz = 0; zz < 4; ++zz)
              if (zz < sk) sum += zz == z ? sp_val[c] : rb[(zz * RS + (lrow - z * RS)) * RSTR + cbeg + c];
            const int n = col0 + cbeg + c;
            if (write && n < a.N) {
              __nv_bfloat16 hi, lo;
              bf16_pair(kr < a.K ? sp_sig * (sum + sp_p[c]) : 0.f, hi, lo);
              a.tau[(long long)n * a.ldt + row0 + lrow] = hi;
              a.tau[a.tau_plane + (long long)n * a.ldt + row0 + lrow] = lo;
            }
          }
        }
      }
      // A CTA may leave once the pushes towards it have landed, which its
      // owning threads waited for (a CTA that only pushes leaves at once, so
      // the next kernel's CTAs can take its SM); if such a wait ran out,
      // pushes may still be in flight: let them land first.
      if (__syncthreads_or(split_failed)) {
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
}

// ---------------------------------------------------------------------------
// four gate sums for 128 units x NT streams, cell update in the epilogue
// ---------------------------------------------------------------------------
template <int NT, int S, bool SPLIT>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_gates_kernel(const __grid_constant__ CUtensorMap tmu, const __grid_constant__ CUtensorMap tmt, TcGatesArgs a) {
  extern __shared__ uint8_t smem_raw[];
  constexpr uint32_t kBBytes = NT * kTileK * 2;       // one plane of the tau' tile
  constexpr uint32_t kStage = kABytes + 2 * kBBytes;  // U tile, hi plane, lo plane
  constexpr uint32_t kAcc = 4 * NT < 32 ? 32 : 4 * NT;  // the four gate accumulators
  // up to 64 streams per tile, c_{t-1} of the tile is staged in tensor memory
  // too (columns kAcc .. kAcc + NT), so the cell loop reads it with the sums
  constexpr bool kCTmem = !SPLIT && NT <= 64;
  constexpr uint32_t kCols = kCTmem ? 2 * kAcc : kAcc;
  static_assert(S >= 4, "a chunk of all four gates must be resident");
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t bar0 = base + S * kStage;  // full[S] | empty[S] | accum | drain | ckpt | ckpt_done | slot
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem_raw + (bar0 - raw) + 8 * (2 * S + 4));
  const uint32_t accum_bar = bar0 + 8u * (2 * S), drain_bar = accum_bar + 8u;
  const uint32_t ckpt_bar = accum_bar + 16u, ckpt_done = accum_bar + 24u;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j0 = blockIdx.x * kTileM;
  const int n0 = blockIdx.y * NT;
  // this CTA's 64-term chunks [kb0, kb1) (all of them without a split), and
  // the intermediate depths that end inside them, [jj_lo, jj_hi)
  constexpr bool split = SPLIT;
  const int kb0 = split ? (int)blockIdx.z * a.nkb_per : 0;
  const int kb1 = split ? min(a.nkb, kb0 + a.nkb_per) : a.nkb;
  const int nkb = kb1 - kb0;
  const int J = a.ck.n;
  int jj_lo = 0, jj_hi = J;
  if constexpr (SPLIT) {
    jj_hi = 0;
    for (int j = 0; j < J; ++j) {
      jj_lo += a.ck.k[j] <= kb0 * kTileK ? 1 : 0;
      jj_hi += a.ck.k[j] <= kb1 * kTileK ? 1 : 0;
    }
  }
  const volatile int* err = a.err;
  const uint64_t limit = static_cast<uint64_t>(a.limit_ns);

  griddep_launch_dependents();  // the next kernel may start its own set-up
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(bar0 + 8u * i, 1);
      mbar_init(bar0 + 8u * (S + i), 1);
    }
    mbar_init(accum_bar, 1);
    mbar_init(drain_bar, 1);
    mbar_init(ckpt_bar, 1);
    mbar_init(ckpt_done, 8 * 32);
    fence_mbarrier_init_cluster();
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {  // ---- TMA producer: stage i = (chunk i/4, gate i%4) ----
    tma_prefetch_map(&tmu);
    tma_prefetch_map(&tmt);
    const int nst = 4 * nkb;
    int issued = 0;
    bool ok = true;
    // U tiles of the first S stages first: they do not depend on the kernel before this one
    const int npre = nst < S ? nst : S;
    for (int i = 0; i < npre; ++i) {
      mbar_arrive_expect_tx(bar0 + 8u * i, kStage);
      tma_load_2d(base + i * kStage, &tmu, bar0 + 8u * i, (kb0 + (i >> 2)) * kTileK, (i & 3) * a.H + j0);
    }
    griddep_wait();
    for (int i = 0; i < nst; ++i) {
      const int s = i % S, kb = kb0 + (i >> 2), g = i & 3;
      if (i >= S && !(ok = wait_cta(bar0 + 8u * (S + s), ((i / S) - 1) & 1, limit, err))) break;
      const uint32_t st = base + s * kStage;
      if (i >= npre) {
        mbar_arrive_expect_tx(bar0 + 8u * s, kStage);
        tma_load_2d(st, &tmu, bar0 + 8u * s, kb * kTileK, g * a.H + j0);
      }
      tma_load_2d(st + kABytes, &tmt, bar0 + 8u * s, g * a.Ks + kb * kTileK, n0);                         // hi
      tma_load_2d(st + kABytes + kBBytes, &tmt, bar0 + 8u * s, g * a.Ks + kb * kTileK, a.tau_rows + n0);  // lo
      ++issued;
    }
    if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
    for (int s = 0; s < S && s < issued; ++s) {
      const int last = s + ((issued - 1 - s) / S) * S;
      wait_cta(bar0 + 8u * s, (last / S) & 1, limit, err);
    }
  } else if (warp == 1 && lane == 0) {  // ---- MMA issuer ----
    constexpr uint32_t idesc = umma_idesc_bf16(kTileM, NT);
    bool ok = true;
    int jj = jj_lo;
    for (int kl = 0; kl < nkb && ok; ++kl) {
      const int kb = kb0 + kl;
      uint64_t da[4], dhi[4], dlo[4];
      // 16-term slices of this chunk, cut at the last slice boundary at or
      // below an intermediate depth (the epilogue adds the terms between the
      // boundary and the depth); each gate's stage is used as soon as it
      // lands and freed as soon as its last slice is issued
      int kk0 = 0;
      while (kk0 < 4 && ok) {
        int kk1 = 4;
        const bool cut_here = jj < jj_hi && a.ck.k[jj] <= (kb + 1) * kTileK;
        if (cut_here) kk1 = (a.ck.k[jj] - kb * kTileK) / 16;
        for (int g = 0; g < 4 && ok; ++g) {
          const int i = 4 * kl + g, s = i % S;
          if (kk0 == 0) {
            if (!(ok = wait_cta(bar0 + 8u * s, (i / S) & 1, limit, err))) break;
            tc_fence_after();
            const uint32_t st = base + s * kStage;
            da[g] = umma_desc_sw128(st);
            dhi[g] = umma_desc_sw128(st + kABytes);
            dlo[g] = umma_desc_sw128(st + kABytes + kBBytes);
          }
          for (int kk = kk0; kk < kk1; ++kk) {
            umma_bf16(tmem + g * NT, da[g] + 2ull * kk, dhi[g] + 2ull * kk, idesc, (kl | kk) != 0 ? 1u : 0u);
            umma_bf16(tmem + g * NT, da[g] + 2ull * kk, dlo[g] + 2ull * kk, idesc, 1u);
          }
          if (kk1 == 4) umma_commit(bar0 + 8u * (S + s));  // frees this gate's stage
        }
        if (ok && cut_here) {  // partial sums up to depth k_jj are complete: hand them to the epilogue
          umma_commit(ckpt_bar);
          ok = wait_cta(ckpt_done, (jj - jj_lo) & 1, limit, err);
          tc_fence_after();
          ++jj;
        }
        kk0 = kk1;
      }
    }
    if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
    while (jj < jj_hi) {  // release epilogue warps still waiting for a depth (abort only)
      umma_commit(ckpt_bar);
      wait_cta(ckpt_done, (jj - jj_lo) & 1, limit, err);
      ++jj;
    }
    umma_commit(accum_bar);
    umma_commit(drain_bar);
    wait_cta(drain_bar, 0, limit, err);
  } else if (warp >= 4) {  // ---- epilogue: cell update of Sec. II (warps 4..11, two per lane quarter) ----
    const int ep = warp - 4, q = ep & 3;
    constexpr int kHalf = NT / 2;
    const int cbeg = (ep >> 2) * kHalf;
    const int j = j0 + 32 * q + lane;  // hidden unit of this thread
    const bool unit_ok = j < a.H;
    float bias[4] = {0.f, 0.f, 0.f, 0.f};
    if (unit_ok)
#pragma unroll
      for (int g = 0; g < 4; ++g) bias[g] = a.bias[g * a.H + j];
    const uint32_t trow = tmem + ((32u * q) << 16);
    griddep_wait();  // c_t-1 and the outputs are shared with the kernels before this one
    if constexpr (kCTmem) {  // c_{t-1} of this thread's unit and streams -> tensor memory, while the MMAs run
#pragma unroll
      for (int c0 = 0; c0 < kHalf; c0 += 16) {
        float cv[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const int n = n0 + cbeg + c0 + c;
          cv[c] = (unit_ok && n < a.B) ? a.c_state[(long long)n * a.H + j] : 0.f;
        }
        tmem_st16(trow + kAcc + cbeg + c0, cv);
      }
      tmem_wait_st();
    }
    for (int step = jj_lo; step <= jj_hi; ++step) {
      const bool final_sums = step == jj_hi;
      const bool ok = wait_cta(final_sums ? accum_bar : ckpt_bar, final_sums ? 0u : (uint32_t)((step - jj_lo) & 1),
                               limit, err);
      tc_fence_after();
      const bool write = ok && *err == 0 && unit_ok;
      // a depth whose last 16-term slice boundary is the start of this CTA's
      // range: no MMA was issued below it, the raw sums are zero (the reduce
      // kernel adds the terms past the boundary)
      const bool acc_valid = final_sums || ((a.ck.k[step] >> 4) << 4) > kb0 * kTileK;
      if constexpr (SPLIT) {
        // raw gate sums of this CTA's terms: slot z for its whole range, slot
        // ks + step at a depth that ends inside it
        const long long slot = final_sums ? (long long)blockIdx.z : (long long)(a.ks + step);
        for (int c0 = cbeg; c0 < cbeg + kHalf; c0 += 16) {
          float y[4][16];
#pragma unroll
          for (int g = 0; g < 4; ++g) tmem_ld16(trow + g * NT + c0, y[g]);
          tmem_wait_ld();
          if (!write) continue;
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const int n = n0 + c0 + c;
            if (n >= a.B) break;
#pragma unroll
            for (int g = 0; g < 4; ++g) a.part[((slot * 4 + g) * a.B + n) * a.H + j] = acc_valid ? y[g][c] : 0.f;
          }
        }
        if (!final_sums) {
          tc_fence_before();
          mbar_arrive(ckpt_done);
        }
        continue;
      }
      // eight streams per round: a compact loop that stays in the
      // instruction cache (fully unrolled cells of whole 16-stream chunks,
      // at about 50 instructions each, did not) with eight independent cells
      // per thread in flight; c_{t-1} comes from tensor memory, or for wider
      // tiles from global memory one round ahead
      auto load_c = [&](int cb, float (&dst)[8]) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int n = n0 + cb + e;
          dst[e] = (!kCTmem && write && cb < cbeg + kHalf && n < a.B) ? a.c_state[(long long)n * a.H + j] : 0.f;
        }
      };
      float cpn[8];
      load_c(cbeg, cpn);
#pragma unroll 1
      for (int c8 = cbeg; c8 < cbeg + kHalf; c8 += 8) {
        float cp[8], y[4][8];
#pragma unroll
        for (int e = 0; e < 8; ++e) cp[e] = cpn[e];  // loaded before any store of this round
        load_c(c8 + 8, cpn);
        __syncwarp();
        if constexpr (kCTmem) {
          tmem_ld8x5_sync(trow + c8, trow + NT + c8, trow + 2 * NT + c8, trow + 3 * NT + c8, trow + kAcc + c8, y, cp);
        } else {
          tmem_ld8x4_sync(trow + c8, trow + NT + c8, trow + 2 * NT + c8, trow + 3 * NT + c8, y);
        }
        if (write) {
          // the eight cells first (independent chains the scheduler can
          // interleave), then their stores
          float hv[8], cv[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            lstm_cell_s(y[0][e] + bias[0], y[1][e] + bias[1], y[2][e] + bias[2], y[3][e] + bias[3], cp[e], hv[e],
                        cv[e]);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int n = n0 + c8 + e;
            if (n >= a.B) break;
            const long long sj = (long long)n * a.H + j;
            const float hh = hv[e], cc = cv[e];
            if (!final_sums) {
              const long long o = (long long)step * a.ck_stride + sj;  // (no split: jj_lo = 0)
              if (a.ckpt_h) a.ckpt_h[o] = hh;
              if (a.ckpt_c) a.ckpt_c[o] = cc;
            } else {
              a.c_state[sj] = cc;
              if (a.out_h) a.out_h[sj] = hh;
              __nv_bfloat16 hi, lo;
              bf16_pair(hh, hi, lo);
              const long long hj = (long long)n * a.ldh + j;
              a.h_bf16[hj] = hi;
              a.h_bf16[a.h_plane + hj] = lo;
              if (a.seq_bf16) {
                a.seq_bf16[hj] = hi;
                a.seq_bf16[a.seq_plane + hj] = lo;
              }
            }
          }
        }
      }
      if (!final_sums) {
        tc_fence_before();
        mbar_arrive(ckpt_done);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
}

// After the gate GEMM in raw-sum mode (a term-axis split, or intermediate
// depths off the 16-term slices): one thread per (stream n, unit j) adds the
// splits' raw gate sums in split order and runs the cell update of Sec. II,
// at full depth and at each intermediate depth k_j (the splits before the one
// k_j ends in, then that split's sums up to k_j's last slice boundary, then
// the terms from there to k_j).
__global__ void __launch_bounds__(256) tc_gates_reduce_kernel(TcGatesArgs a) {
  griddep_launch_dependents();  // the next step's tau' kernel may start its set-up
  const long long total = (long long)a.B * a.H;
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  griddep_wait();  // the partial sums of the gate GEMM before this kernel
  if (i >= total || *reinterpret_cast<volatile int*>(a.err) != 0) return;
  const int n = (int)(i / a.H), j = (int)(i - (long long)n * a.H);
  const long long gs = (long long)a.B * a.H;  // gate stride within a slot
  const float* part = a.part + (long long)n * a.H + j;
  float bias[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) bias[g] = a.bias[g * a.H + j];
  const float cp = a.c_state[i];
  for (int jj = 0; jj < a.ck.n; ++jj) {
    const int sj = ((a.ck.k[jj] + kTileK - 1) / kTileK - 1) / a.nkb_per;  // split the depth ends in
    const int r = a.ck.k[jj] & 15;  // terms past the depth's last 16-term slice boundary
    float y[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      float v = 0.f;
      for (int z = 0; z < sj; ++z) v += part[(z * 4 + g) * gs];
      y[g] = v + part[((a.ks + jj) * 4 + g) * gs] + bias[g];
      if (r != 0) y[g] += remainder_terms(a, g, n, j, a.ck.k[jj] - r, r);
    }
    float hh, cc;
    lstm_cell_s(y[0], y[1], y[2], y[3], cp, hh, cc);
    const long long o = (long long)jj * a.ck_stride + i;
    if (a.ckpt_h) a.ckpt_h[o] = hh;
    if (a.ckpt_c) a.ckpt_c[o] = cc;
  }
  float y[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    float v = 0.f;
    for (int z = 0; z < a.ks; ++z) v += part[(z * 4 + g) * gs];
    y[g] = v + bias[g];
  }
  float hh, cc;
  lstm_cell_s(y[0], y[1], y[2], y[3], cp, hh, cc);
  a.c_state[i] = cc;
  if (a.out_h) a.out_h[i] = hh;
  __nv_bfloat16 hi, lo;
  bf16_pair(hh, hi, lo);
  const long long hj = (long long)n * a.ldh + j;
  a.h_bf16[hj] = hi;
  a.h_bf16[a.h_plane + hj] = lo;
  if (a.seq_bf16) {
    a.seq_bf16[hj] = hi;
    a.seq_bf16[a.seq_plane + hj] = lo;
  }
}

// x (fp32 [N][D]) -> its bf16 pair, hi plane [N][ld] then lo plane [N][ld],
// with zero columns D..ld-1: one thread per 8 elements (one 16-byte store
// per plane), vector loads when x is 16-byte aligned and D is a multiple of 8
__global__ void to_bf16_kernel(const float* __restrict__ x, int N, int D, __nv_bfloat16* __restrict__ out, int ld,
                               bool vec) {
  const int c8 = ld >> 3;  // 8-element chunks per output row (ld is a multiple of 8)
  const long long total = (long long)N * c8;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const int n = (int)(i / c8), d0 = (int)(i % c8) * 8;
    float v[8];
    if (vec && d0 + 8 <= D) {
      const float4* src = reinterpret_cast<const float4*>(x + (long long)n * D + d0);
      const float4 a = __ldg(src), b = __ldg(src + 1);
      v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = d0 + e < D ? __ldg(x + (long long)n * D + d0 + e) : 0.f;
    }
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      __nv_bfloat16 h0, l0, h1, l1;
      bf16_pair(v[2 * e], h0, l0);
      bf16_pair(v[2 * e + 1], h1, l1);
      hw[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
      lw[e] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
    }
    reinterpret_cast<uint4*>(out)[i] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    reinterpret_cast<uint4*>(out)[total + i] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  }
}

// initial state of the tensor path: h0 -> the bf16 pair planes of the
// operand ([B][ldh] each), c0 -> fp32 state
__global__ void tc_init_state_kernel(const float* __restrict__ h0, const float* __restrict__ c0, int B, int H,
                                     __nv_bfloat16* __restrict__ h_bf16, int ldh, float* __restrict__ c_state) {
  const long long total = (long long)B * ldh;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const long long n = i / ldh;
    const int j = (int)(i % ldh);
    __nv_bfloat16 hi, lo;
    bf16_pair((h0 != nullptr && j < H) ? h0[n * H + j] : 0.f, hi, lo);
    h_bf16[i] = hi;
    h_bf16[total + i] = lo;
    if (j < H) c_state[n * H + j] = c0 != nullptr ? c0[n * H + j] : 0.f;
  }
}

// ---- host side -------------------------------------------------------------

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encoder() {
  static EncodeTiled fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiled>(p);
  });
  return fn;
}

// Launch with programmatic stream serialization: the kernel may start while
// the one before it in the stream finishes, and waits on it (griddep_wait)
// only where it reads that kernel's results or writes what it reads.
template <typename Kern, typename... Args>
cudaError_t launch_pdl_block(Kern kern, dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}
template <typename Kern, typename... Args>
cudaError_t launch_pdl(Kern kern, dim3 grid, size_t smem, cudaStream_t s, Args... args) {
  return launch_pdl_block(kern, grid, dim3(kTcThreads), smem, s, args...);
}

template <int BN, int S, bool XF>
size_t rows_smem() {
  return 1024 + S * (kABytes + 2 * BN * kTileK * 2) + 8 * ((XF ? 3 : 2) * S + 3) + 16;
}
template <int NT, int S>
size_t gates_smem() {
  return 1024 + S * (kABytes + 2 * NT * kTileK * 2) + 8 * (2 * S + 4) + 16;
}

template <int BN, int S, bool XF = false>
cudaError_t launch_rows_t(const TcMap& A, const TcMap& Bm, const TcRowsArgs& a, int n_cols, cudaStream_t s) {
  auto kern = tc_rows_kernel<BN, S, XF>;
  static thread_local bool attr = false;
  const size_t smem = rows_smem<BN, S, XF>();
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  static_assert((size_t)kTileM * (BN + 4) * 4 <= (size_t)S * (kABytes + 2 * BN * kTileK * 2),
                "a split's receive buffer fits over the stage ring");
  const int sk = (!XF && a.sk > 1) ? a.sk : 1;
  const dim3 grid(a.rpg > 0 ? 1 : 4 * a.kt_per_gate, (n_cols + BN - 1) / BN, sk);
  if (sk == 1)
    return launch_pdl(kern, grid, smem, s, *reinterpret_cast<const CUtensorMap*>(A.bytes),
                      *reinterpret_cast<const CUtensorMap*>(Bm.bytes), a);
  // the sk CTAs of a split tile form one cluster along z
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[0].val.programmaticStreamSerializationAllowed = 1;
  attrs[1].id = cudaLaunchAttributeClusterDimension;
  attrs[1].val.clusterDim.x = 1;
  attrs[1].val.clusterDim.y = 1;
  attrs[1].val.clusterDim.z = sk;
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, *reinterpret_cast<const CUtensorMap*>(A.bytes),
                            *reinterpret_cast<const CUtensorMap*>(Bm.bytes), a);
}

template <int NT, int S, bool SPLIT>
cudaError_t launch_gates_t(const TcMap& U, const TcMap& Tau, const TcGatesArgs& a, cudaStream_t s) {
  auto kern = tc_gates_kernel<NT, S, SPLIT>;
  static thread_local bool attr = false;
  const size_t smem = gates_smem<NT, S>();
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const cudaError_t e =
      launch_pdl(kern, dim3((a.H + kTileM - 1) / kTileM, (a.B + NT - 1) / NT, a.ks), smem, s,
                 *reinterpret_cast<const CUtensorMap*>(U.bytes), *reinterpret_cast<const CUtensorMap*>(Tau.bytes), a);
  if (e != cudaSuccess || !SPLIT) return e;
  const long long total = (long long)a.B * a.H;
  return launch_pdl_block(tc_gates_reduce_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), 0, s, a);
}

}  // namespace

bool tc_make_map(TcMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t pitch_bytes, uint32_t box_rows,
                 uint32_t swizzle_bytes) {
  static_assert(sizeof(CUtensorMap) <= sizeof(m->bytes), "tensor map storage");
  EncodeTiled enc = encoder();
  if (!enc) return false;
  std::memset(m->bytes, 0, sizeof(m->bytes));
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {pitch_bytes};
  const cuuint32_t box[2] = {swizzle_bytes / 2u, box_rows};  // one swizzled row of bf16 elements
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(reinterpret_cast<CUtensorMap*>(m->bytes), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                         const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int tc_rows_tile_n(int n_cols, int row_tiles) {
  // the narrowest of 32, 64, 128 columns that keeps one wave (few columns:
  // more CTAs, each streaming fewer activation bytes); many columns (the
  // projection over T*B): 128, where both planes of the activation make a
  // 128-column tile feed 256 columns of MMA work per factor tile
  for (int bn : {32, 64})
    if ((long long)row_tiles * ((n_cols + bn - 1) / bn) <= 148) return bn;
  return 128;
}
int tc_gates_splits(int tiles, int nkb, int* nkb_per) {
  // about one wave: as many splits as the GPU holds grids of `tiles` CTAs
  int ks = 148 / (tiles > 0 ? tiles : 1);
  if (ks > 8) ks = 8;
  if (ks > nkb) ks = nkb;
  if (ks < 2) {
    *nkb_per = nkb;
    return 1;
  }
  *nkb_per = (nkb + ks - 1) / ks;
  return (nkb + *nkb_per - 1) / *nkb_per;  // no empty split
}

int tc_gates_tile_n(int H, int B) {
  const int unit_tiles = (H + kTileM - 1) / kTileM;
  for (int nt : {32, 64, 128})
    if ((long long)unit_tiles * ((B + nt - 1) / nt) <= 148) return nt;
  return 128;
}

cudaError_t launch_tc_rows_xf32(const TcMap& A, const TcMap& Xf, const TcRowsArgs& a, int n_cols, cudaStream_t s) {
  return launch_rows_t<64, 6, true>(A, Xf, a, n_cols, s);
}

bool tc_make_map_f32(TcMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t pitch_bytes,
                     uint32_t box_rows) {
  EncodeTiled enc = encoder();
  if (!enc) return false;
  std::memset(m->bytes, 0, sizeof(m->bytes));
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {pitch_bytes};
  const cuuint32_t box[2] = {32u, box_rows};  // 128-byte rows, unswizzled
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(reinterpret_cast<CUtensorMap*>(m->bytes), CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
                         const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

cudaError_t launch_tc_rows(const TcMap& A, const TcMap& Bm, const TcRowsArgs& a, int n_cols, int bn, cudaStream_t s) {
  switch (bn) {
    case 128: return launch_rows_t<128, 4>(A, Bm, a, n_cols, s);
    case 32: return launch_rows_t<32, 8>(A, Bm, a, n_cols, s);
    default: return launch_rows_t<64, 6>(A, Bm, a, n_cols, s);
  }
}

cudaError_t launch_tc_gates(const TcMap& U, const TcMap& Tau, const TcGatesArgs& a, int nt, cudaStream_t s) {
  switch (nt) {
    case 128: return a.raw ? launch_gates_t<128, 4, true>(U, Tau, a, s) : launch_gates_t<128, 4, false>(U, Tau, a, s);
    case 64: return a.raw ? launch_gates_t<64, 6, true>(U, Tau, a, s) : launch_gates_t<64, 6, false>(U, Tau, a, s);
    default: return a.raw ? launch_gates_t<32, 8, true>(U, Tau, a, s) : launch_gates_t<32, 8, false>(U, Tau, a, s);
  }
}

cudaError_t launch_to_bf16(const float* x, int N, int D, __nv_bfloat16* out, int ld, cudaStream_t s) {
  const long long total = (long long)N * (ld >> 3);
  const int blocks = (int)std::min<long long>((total + 255) / 256, 152LL * 16);
  const bool vec = (D & 7) == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  to_bf16_kernel<<<blocks, 256, 0, s>>>(x, N, D, out, ld, vec);
  return cudaGetLastError();
}

cudaError_t launch_tc_init_state(const float* h0, const float* c0, int B, int H, __nv_bfloat16* h_bf16, int ldh,
                                 float* c_state, cudaStream_t s) {
  const long long total = (long long)B * ldh;
  const int blocks = (int)std::min<long long>((total + 255) / 256, 152LL * 16);
  tc_init_state_kernel<<<blocks, 256, 0, s>>>(h0, c0, B, H, h_bf16, ldh, c_state);
  return cudaGetLastError();
}

}  // namespace lstm_approx_impl
