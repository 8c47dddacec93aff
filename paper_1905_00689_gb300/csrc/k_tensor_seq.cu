// Tensor-core path for small K: one launch per tile of streams for all T
// timesteps of a layer (bf16 factors, fp32 accumulate, activations as bf16
// pairs as in k_tensor.cu).
//
// The per-timestep kernels of k_tensor.cu pay two dependent launches per
// step and stream their whole factor tiles through shared memory every step,
// which at small K costs about 14-18 us per step whatever K is.  Here a
// cluster of CS CTAs serves a tile of NS streams (32 or 64) for the whole
// sequence; CTA r owns UC = 128 MT hidden units [UC r, UC r + UC) (MT = 1 or
// 2, CS = H / UC) and keeps on chip:
//
//   - its columns of the packed V_h (the four gates' first rpg rows, rpg =
//     8, 16 or 32 >= K, the A operand of the tau' product), 32 KB per 128 units;
//   - its rows of U, the first 32 terms of each gate, 32 KB per 128 units;
//   - h_{t-1} of its units as the bf16 pair (the B operand of the tau'
//     product), c_{t-1} in registers of the epilogue threads;
//   - tau' of all terms and the tile's streams as the bf16 pair (the B
//     operand of the gate product).
//
// One timestep (Eq. 1 and Sec. II):
//   (a2) the CTA's partial tau' over its units, acc[(g,k)][n] =
//        sum_{j in CTA} Vh[(g,k)][j] h_{t-1}[n][j]  (M = 128, N = NS);
//   exchange 1: the epilogue warps read the partials from tensor memory and
//        send each CTA the columns of the streams it owns (SP = NS / CS
//        streams per CTA, 8 or 16) with st.async;
//   the owner adds the CS partials in rank order, forms
//        tau' = sigma (sum + P_t) (zero for k >= K) and its pair, writes them
//        into its tau' operand and, exchange 2, copies that block to every
//        other CTA with one bulk copy each;
//   (a3, a6) the four gate sums of the CTA's units, y_g = U_g tau'_g (one
//        tensor-memory accumulator per gate and 128 units), cut at each
//        intermediate depth (a multiple of 16) for the checkpoint cells, as
//        in k_tensor.cu;
//   (a4) the cells, with h_t written as the pair into the next step's tau'
//        operand, and as fp32 (and for a lower layer as the pair) to memory.
//
// Every mbarrier wait is bounded in wall time; a wait that runs out (or sees
// the status word set by another CTA) writes the status word and the CTA
// leaves its loop; all CTAs meet at the final cluster barrier, and a CTA
// that left early waits 50 us before freeing its shared memory so that
// copies already in flight towards it land first.
#include <cuda.h>

#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;


constexpr int kSeqMaxRed = 4;              // owner elements (tau' values) per epilogue thread at most
constexpr int kSeqMaxClusters4 = 36;       // clusters of 4 such CTAs resident at once on a GB300 (152 SMs)

// Threads: warp 0 issues the TMA copies and the MMAs, warp 1 owns tensor
// memory, and 4 EPW epilogue warps follow (EPW per 32-lane quarter of tensor
// memory, each taking 8 of the tile's streams per 128 units: 4 at NS >= 32,
// 2 at NS = 16).
__host__ __device__ constexpr int seq_epw(int ns) { return ns >= 32 ? 4 : 2; }
__host__ __device__ constexpr int seq_threads(int ns) { return 64 + 4 * seq_epw(ns) * 32; }

// Shared-memory layout, offsets from the 1024-byte aligned base (MT 128-unit
// tiles per CTA, NS streams, 4 rpg packed rows):
//   Atau  [2 MT unit blocks of 64][128 rows][128 B]        128-byte swizzle
//   Agate [4 gates][MT][128 units][64 B] (terms 0..31)     64-byte swizzle
//   Bh    [2 MT unit blocks of 64][NS/8 stream groups][2 planes][8 streams][128 B]
//   Btau  [NS/8 stream groups][2 planes][4 gates][8 streams][64 B]   64-byte swizzle
//   RS    [CS sources][4 rpg rows][SP streams] fp32 partial tau'
//   Cst   [MT 8 streams-per-warp blocks][epilogue threads] fp32 c_{t-1} of each thread's cells
//   barriers, tensor-memory slot
// The activation operands interleave the two planes of the pair by groups of
// 8 streams, so that one MMA of N = 2 NS rows (hi, lo, hi, lo, ... groups at
// a uniform stride) multiplies a factor tile by both planes: the factor tile
// is read once, and the accumulator holds the hi and lo products of stream
// group G in columns [16 G, 16 G + 8) and [16 G + 8, 16 G + 16).
struct SeqLayout {
  uint32_t agate, bh, btau, rs, cst, bar, total;
};
__host__ __device__ inline SeqLayout seq_layout(int ns, int mt, int r4) {
  SeqLayout l;
  l.agate = 32768u * mt;
  l.bh = l.agate + 32768u * mt;
  l.btau = l.bh + (uint32_t)ns * 512u * mt;
  l.rs = l.btau + (uint32_t)ns * 512u;
  l.cst = l.rs + (uint32_t)r4 * ns * 4u;
  // each epilogue thread's c: MT x (NS / EPW) values, EPW warps per quarter
  l.bar = l.cst + (uint32_t)mt * (uint32_t)(ns / seq_epw(ns)) * (uint32_t)(4 * seq_epw(ns) * 32) * 4u;
  l.total = l.bar + 128u + 1024u;  // barriers and slot, alignment slack
  return l;
}

__device__ __forceinline__ bool seq_wait(uint32_t mb, uint32_t parity, uint64_t limit, const volatile int* err) {
  return mbar_wait_bounded<false>(mb, parity, limit, err);
}
__device__ __forceinline__ bool seq_wait_cluster(uint32_t mb, uint32_t parity, uint64_t limit,
                                                 const volatile int* err) {
  return mbar_wait_bounded<true>(mb, parity, limit, err);
}

// The bf16 pair of an fp32 value: hi = bf16(v), lo = bf16(v - hi).
__device__ __forceinline__ void seq_pair(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

template <int NS, int MT>
__global__ void __launch_bounds__(seq_threads(NS), 1)
    tc_seq_kernel(const __grid_constant__ CUtensorMap tmv, const __grid_constant__ CUtensorMap tmu, TcSeqArgs a) {
  extern __shared__ uint8_t smem_raw[];
  constexpr int kSeqEpw = seq_epw(NS);
  constexpr int kSeqEpi = 4 * kSeqEpw * 32;  // epilogue threads
  constexpr int SPW = NS / kSeqEpw;  // streams per epilogue warp
  // owner elements per epilogue thread at most: 4 rpg rows x SP streams over the
  // epilogue threads; with 256 units per CTA the cluster has 4 CTAs and SP = NS / 4
  constexpr int kMaxRed = MT == 2 ? (128 * (NS / 4) + kSeqEpi - 1) / kSeqEpi : kSeqMaxRed;
  constexpr int UC = 128 * MT;       // hidden units per CTA
  constexpr int NU = UC / 64;        // 64-unit blocks (K-dim tiles of the tau' product)
  // tensor memory: the gate accumulators (gate g, unit tile m: 2 NS columns at (g MT + m) 2 NS);
  // the tau' accumulator shares the first 2 NS columns (it is read before the gate MMAs
  // start, and they are read before the next tau' MMAs start)
  constexpr uint32_t kUsed = 8u * MT * NS;
  constexpr uint32_t kCols = kUsed <= 256 ? 256 : 512;
  constexpr uint32_t tAcc = 0, tGate = 0;
  const int CS = a.cs, SP = NS / CS, rpg = a.rpg, R4 = 4 * rpg;
  const SeqLayout L = seq_layout(NS, MT, R4);
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gb = smem_raw + (base - raw);  // generic pointer to the base
  const uint32_t sAtau = base, sAgate = base + L.agate, sBh = base + L.bh, sBtau = base + L.btau,
                 sRS = base + L.rs, sBar = base + L.bar;
  const uint32_t fac_full = sBar, h_ready = sBar + 8, tacc_full = sBar + 16, rs_full = sBar + 24,
                 tau_full = sBar + 32, acc_full = sBar + 40, ckpt_bar = sBar + 48, ckpt_done = sBar + 56,
                 red_done = sBar + 64, drain_bar = sBar + 72;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gb + L.bar + 96);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_ctarank();
  const int j0 = rank * UC;             // first hidden unit of this CTA
  const int n0 = (int)blockIdx.y * NS;  // first stream of this cluster's tile
  const int T = a.T, B = a.B, H = a.H;
  const volatile int* err = a.err;
  const uint64_t limit = static_cast<uint64_t>(a.limit_ns);
  // MMA slices of 16 terms, and the slice count at each intermediate depth
  const int nsl = (a.K + 15) / 16;
  const int ncut = a.ck.n;
  int cut_sl[kMaxCheckpoints];
#pragma unroll
  for (int c = 0; c < kMaxCheckpoints; ++c) cut_sl[c] = c < ncut ? (a.ck.k[c] >= a.K ? nsl : a.ck.k[c] / 16) : 0;

  griddep_launch_dependents();
  if (threadIdx.x == 0) {
    mbar_init(fac_full, 1);
    mbar_init(h_ready, kSeqEpi / 32);  // one arrival per epilogue warp
    mbar_init(tacc_full, 1);
    mbar_init(rs_full, 1);
    mbar_init(tau_full, 1);
    mbar_init(acc_full, 1);
    mbar_init(ckpt_bar, 1);
    mbar_init(ckpt_done, kSeqEpi / 32);
    mbar_init(red_done, kSeqEpi / 32);
    mbar_init(drain_bar, 1);
    fence_mbarrier_init_cluster();
  }
  // zero what no copy writes: the V_h tiles' rows from 4 rpg on, and the
  // tau' operand (its terms from rpg on stay zero for the whole launch)
  {
    const uint32_t zrow = (uint32_t)R4 * 128u, zlen = 16384u - zrow;
    for (uint32_t i = threadIdx.x; i < NU * zlen / 16u; i += blockDim.x) {
      const uint32_t blk = i / (zlen / 16u), o = i % (zlen / 16u);
      *reinterpret_cast<uint4*>(gb + blk * 16384u + zrow + 16u * o) = make_uint4(0, 0, 0, 0);
    }
    for (uint32_t i = threadIdx.x; i < (uint32_t)NS * 512u / 16u; i += blockDim.x)
      *reinterpret_cast<uint4*>(gb + L.btau + 16u * i) = make_uint4(0, 0, 0, 0);
    fence_proxy_async_shared();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // every CTA's barriers are initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {  // ---- factor copies, then the MMA issue of every step ----
      tma_prefetch_map(&tmv);
      tma_prefetch_map(&tmu);
      mbar_arrive_expect_tx(fac_full, (uint32_t)NU * R4 * 128u + 4u * MT * 8192u);
      for (int g = 0; g < 4; ++g)
        for (int blk = 0; blk < NU; ++blk)
          tma_load_2d(sAtau + blk * 16384u + g * rpg * 128u, &tmv, fac_full, j0 + 64 * blk, g * a.Ks);
      for (int g = 0; g < 4; ++g)
        for (int m = 0; m < MT; ++m)
          tma_load_2d(sAgate + (g * MT + m) * 8192u, &tmu, fac_full, 0, g * H + j0 + 128 * m);
      bool ok = seq_wait(fac_full, 0, limit, err);
      constexpr uint32_t idesc = umma_idesc_bf16(128, 2 * NS);  // both planes of the activation
      for (int t = 0; t < T && ok; ++t) {
        // (a2) partial tau' of this CTA's units: UC / 16 slices, both planes of h_{t-1} at once
        if (!(ok = seq_wait(h_ready, t & 1, limit, err))) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < UC / 16; ++kk) {
          const uint32_t cb = kk >> 2, w = kk & 3;
          const uint64_t da = umma_desc_sw128(sAtau + cb * 16384u) + 2ull * w;
          const uint64_t db = umma_desc_sw128(sBh + cb * (2u * NS * 128u)) + 2ull * w;
          umma_bf16(tmem + tAcc, da, db, idesc, kk != 0 ? 1u : 0u);
        }
        umma_commit(tacc_full);
        // (a3) the four gate sums once every CTA's tau' block has landed
        if (!(ok = seq_wait_cluster(tau_full, t & 1, limit, err))) break;
        tc_fence_after();
        int s = 0;
        for (int c = 0; c <= ncut && ok; ++c) {
          const int s_end = c < ncut ? cut_sl[c] : nsl;
          for (; s < s_end; ++s)
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              const uint64_t db = umma_desc_sw64(sBtau + g * 512u, 2048u) + 2ull * s;
#pragma unroll
              for (int m = 0; m < MT; ++m) {
                const uint64_t da = umma_desc_sw64(sAgate + (g * MT + m) * 8192u, 512u) + 2ull * s;
                umma_bf16(tmem + tGate + (g * MT + m) * 2 * NS, da, db, idesc, s != 0 ? 1u : 0u);
              }
            }
          if (c < ncut) {  // partial sums at depth k_c: the epilogue runs the checkpoint cells
            umma_commit(ckpt_bar);
            ok = seq_wait(ckpt_done, (uint32_t)(t * ncut + c) & 1u, limit, err);
            tc_fence_after();
          }
        }
        if (ok) umma_commit(acc_full);
      }
      if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
      umma_commit(drain_bar);  // every MMA issued has completed before tensor memory is freed
      seq_wait(drain_bar, 0, limit, err);
    }
  } else if (warp >= 2) {  // ---- epilogue: exchanges, tau', cells ----
    // warp w reads tensor-memory lanes [32 (w mod 4), +32); four warps per quarter
    const int e = threadIdx.x - 64, q = warp & 3, part = (warp - 2) >> 2;
    const uint32_t trow = tmem + ((32u * q) << 16);
    // this thread's hidden units jl = 128 m + 32 q + lane (tensor-memory lane 32 q + lane of unit tile m)
    float bias[MT][4];
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
      for (int g = 0; g < 4; ++g) bias[m][g] = a.bias[g * H + j0 + 128 * m + 32 * q + lane];
    // owner elements: tau' of row (g, k) for stream rank*SP + sp, element
    // idx = row*SP + sp, taken by threads e, e + kSeqEpi, ... (recomputed
    // each step: SP and rpg are powers of two)
    const int E = R4 * SP;
    const int sp_sh = SP == 4 ? 2 : (SP == 8 ? 3 : 4), rpg_sh = rpg == 8 ? 3 : (rpg == 16 ? 4 : 5);
    struct Owned {
      int bt;   // byte offset in the tau' operand (hi plane)
      int pc;   // offset in P_t, or -1 (k >= K, or a stream past B)
    };
    auto owned = [&](int idx) {
      const int row = idx >> sp_sh, sp = idx & (SP - 1), g = row >> rpg_sh, k = row & (rpg - 1);
      const int nl = rank * SP + sp;
      Owned o;
      o.bt = (int)((nl >> 3) * 4096u + g * 512u + sw64_offset(nl, k));
      o.pc = (k < a.K && n0 + nl < B) ? (n0 + nl) * a.ldp + g * a.Ks + k : -1;
      return o;
    };
    // h pair of (local stream nl, local unit jl) in the tau' product's operand
    auto put_h = [&](int nl, int jl, float v) {
      __nv_bfloat16 hi, lo;
      seq_pair(v, hi, lo);
      const uint32_t o =
          (uint32_t)(jl >> 6) * (2u * NS * 128u) + (uint32_t)(nl >> 3) * 2048u + sw128_offset(nl, jl & 63);
      *reinterpret_cast<__nv_bfloat16*>(gb + L.bh + o) = hi;
      *reinterpret_cast<__nv_bfloat16*>(gb + L.bh + o + 1024u) = lo;
    };
    // one arrival per warp on an mbarrier counting epilogue warps, once every
    // lane of the warp has finished (its writes ordered by the warp barrier)
    auto warp_arrive = [&](uint32_t mb) {
      __syncwarp();
      if (lane == 0) mbar_arrive(mb);
    };
    // sigma of this thread's owner elements (0 for k >= K)
    float r_sig[kMaxRed];
#pragma unroll
    for (int i = 0; i < kMaxRed; ++i) {
      const int idx = e + i * kSeqEpi;
      r_sig[i] = 0.f;
      if (idx < E) {
        const int row = idx >> sp_sh, g = row >> rpg_sh, k = row & (rpg - 1);
        if (k < a.K) r_sig[i] = a.sigma[g * a.Ks + k];
      }
    }
    griddep_wait();  // P, h0 and c0 may come from the kernels before this one
    // c_{t-1} of this thread's cell (m, stream s of its SPW): word (m SPW + s) kSeqEpi + e
    float* cst = reinterpret_cast<float*>(gb + L.cst) + e;
#pragma unroll 1
    for (int m = 0; m < MT; ++m)
#pragma unroll 1
      for (int s = 0; s < SPW; ++s) {
        const int nl = part * SPW + s, n = n0 + nl, jl = 128 * m + 32 * q + lane;
        const long long o = (long long)n * H + j0 + jl;
        cst[(m * SPW + s) * kSeqEpi] = (a.c0 != nullptr && n < B) ? a.c0[o] : 0.f;
        put_h(nl, jl, (a.h0 != nullptr && n < B) ? a.h0[o] : 0.f);
      }
    fence_proxy_async_shared();
    tc_fence_before();
    warp_arrive(h_ready);
    const float* rsb = reinterpret_cast<const float*>(gb + L.rs);
    const int srcs = R4 * SP;  // floats per source in the RS buffer
    bool ok = true;
    for (int t = 0; t < T && ok; ++t) {
      float pv[kMaxRed];
#pragma unroll
      for (int i = 0; i < kMaxRed; ++i) {
        const int idx = e + i * kSeqEpi, pc = idx < E ? owned(idx).pc : -1;
        pv[i] = pc >= 0 ? __ldg(a.P + (long long)t * B * a.ldp + pc) : 0.f;
      }
      if (e == 0) mbar_arrive_expect_tx(rs_full, (uint32_t)(CS * srcs * 4));
      // exchange 1: this CTA's partial tau' of each stream -> the stream's owner
      ok = __all_sync(0xffffffffu, seq_wait(tacc_full, t & 1, limit, err));
      if (!ok) break;
      tc_fence_after();
      const bool stall = a.test_stall != 0 && rank == 0 && blockIdx.y == 0 && t == 0;
      if (32 * q < R4 && !stall) {
        const int row = 32 * q + lane;
#pragma unroll
        for (int i8 = 0; i8 < SPW / 8; ++i8) {
          const int c8 = part * SPW + 8 * i8;
          float hl[16], v[8];  // the group's hi products, then its lo products
          tmem_ld16_sync(trow + tAcc + 2 * c8, hl);
#pragma unroll
          for (int k8 = 0; k8 < 8; ++k8) v[k8] = hl[k8] + hl[8 + k8];
#pragma unroll
          for (int h4 = 0; h4 < 2; ++h4) {
            const int col = c8 + 4 * h4, d = col / SP, sp = col - d * SP;
            const uint32_t off = (uint32_t)((rank * R4 + row) * SP + sp) * 4u;
            st_async_v4(mapa_shared(sRS + off, d), v[4 * h4], v[4 * h4 + 1], v[4 * h4 + 2], v[4 * h4 + 3],
                        mapa_shared(rs_full, d));
          }
        }
      }
      // the owner's tau': partials added in rank order, sigma (sum + P_t), as its pair
      ok = __all_sync(0xffffffffu, seq_wait_cluster(rs_full, t & 1, limit, err));
      if (!ok) break;
#pragma unroll
      for (int i = 0; i < kMaxRed; ++i) {
        const int idx = e + i * kSeqEpi;
        if (idx >= E) break;
        const Owned o = owned(idx);
        float sum = 0.f;
        for (int src = 0; src < CS; ++src) sum += rsb[src * srcs + idx];
        __nv_bfloat16 hi, lo;
        seq_pair(r_sig[i] * (sum + pv[i]), hi, lo);
        *reinterpret_cast<__nv_bfloat16*>(gb + L.btau + o.bt) = hi;
        *reinterpret_cast<__nv_bfloat16*>(gb + L.btau + o.bt + 2048) = lo;
      }
      fence_proxy_async_shared();
      tc_fence_before();  // this thread's tensor-memory reads are done before the gate MMAs overwrite them
      warp_arrive(red_done);
      // exchange 2: this CTA's block of tau' (its SP streams, all terms) -> every other CTA:
      // one copy per peer of SP / 8 whole stream groups, or (SP = 4, half a group) eight
      // 256-byte pieces per peer, one per (plane, gate)
      const int ncopy = SP >= 8 ? CS - 1 : 8 * (CS - 1);
      if (e < ncopy) {
        if (!seq_wait(red_done, t & 1, limit, err)) {
          atomicCAS(a.err, 0, kErrTcTimeout);
        } else {
          if (e == 0) mbar_arrive_expect_tx(tau_full, (uint32_t)((CS - 1) * SP * 512));
          if (SP >= 8) {
            const int d = (rank + 1 + e) % CS;
            const uint32_t src = sBtau + (uint32_t)rank * SP * 512u;
            bulk_copy_s2cluster(mapa_shared(src, d), src, (uint32_t)SP * 512u, mapa_shared(tau_full, d));
          } else {
            const int d = (rank + 1 + (e >> 3)) % CS, piece = e & 7;  // piece = plane * 4 + gate
            const uint32_t src = sBtau + (uint32_t)(rank >> 1) * 4096u + (uint32_t)piece * 512u + (rank & 1) * 256u;
            bulk_copy_s2cluster(mapa_shared(src, d), src, 256u, mapa_shared(tau_full, d));
          }
        }
      }
      // (a4, a6) cells: at each intermediate depth from the partial sums, then at full depth
      for (int cj = 0; cj <= ncut; ++cj) {
        const bool fin = cj == ncut;
        ok = __all_sync(0xffffffffu, fin ? seq_wait(acc_full, t & 1, limit, err)
                                         : seq_wait(ckpt_bar, (uint32_t)(t * ncut + cj) & 1u, limit, err));
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          const int jl = 128 * m + 32 * q + lane, j = j0 + jl;
#pragma unroll
          for (int i8 = 0; i8 < SPW / 8; ++i8) {
            const int nl0 = part * SPW + 8 * i8;
            // gate g's sums of this group: hi products at tc0 + g 2 MT NS, lo products 8 columns on
            const uint32_t tc0 = trow + tGate + m * 2 * NS + 2 * nl0;
            float y[4][8];
            if constexpr (MT * NS >= 64) {  // one gate at a time: 16 registers in flight (the wide tiles need them)
#pragma unroll
              for (int g = 0; g < 4; ++g) {
                float a0[16];
                tmem_ld16_sync(tc0 + g * 2 * MT * NS, a0);
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8) y[g][k8] = a0[k8] + a0[8 + k8];
              }
            } else {  // two gates per wait
#pragma unroll
              for (int g = 0; g < 4; g += 2) {
                float a0[16], a1[16];
                tmem_ld16x2_sync(tc0 + g * 2 * MT * NS, tc0 + (g + 1) * 2 * MT * NS, a0, a1);
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8) {
                  y[g][k8] = a0[k8] + a0[8 + k8];
                  y[g + 1][k8] = a1[k8] + a1[8 + k8];
                }
              }
            }
            float hv[8], cv[8];
            float* cs8 = cst + (m * SPW + 8 * i8) * kSeqEpi;
#pragma unroll
            for (int k8 = 0; k8 < 8; ++k8)
              lstm_cell_s(y[0][k8] + bias[m][0], y[1][k8] + bias[m][1], y[2][k8] + bias[m][2],
                          y[3][k8] + bias[m][3], cs8[k8 * kSeqEpi], hv[k8], cv[k8]);
            // outputs of streams n0 + nl0 + k8 (k8 < nv) of unit j: element (t, n, j) at (t B + n) H + j
            const int nv = min(8, B - (n0 + nl0));
            const long long o0 = ((long long)t * B + n0 + nl0) * H + j;
            if (!fin) {
              if (a.ckpt_h) {
                float* p = a.ckpt_h + (long long)cj * a.ck_stride + o0;
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8)
                  if (k8 < nv) p[(long long)k8 * H] = hv[k8];
              }
              if (a.ckpt_c) {
                float* p = a.ckpt_c + (long long)cj * a.ck_stride + o0;
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8)
                  if (k8 < nv) p[(long long)k8 * H] = cv[k8];
              }
              continue;
            }
            {  // h_t as the pair into the next step's operand (streams nl0 .. nl0 + 7 of unit jl)
              const uint32_t hb = L.bh + (uint32_t)(jl >> 6) * (2u * NS * 128u) + (uint32_t)(nl0 >> 3) * 2048u +
                                  (uint32_t)(jl & 7) * 2u;
              const uint32_t cjl = (uint32_t)(jl & 63) >> 3;
#pragma unroll
              for (int k8 = 0; k8 < 8; ++k8) {
                cs8[k8 * kSeqEpi] = cv[k8];
                __nv_bfloat16 hi, lo;
                seq_pair(hv[k8], hi, lo);
                const uint32_t off = hb + k8 * 128u + ((cjl ^ (uint32_t)k8) << 4);
                *reinterpret_cast<__nv_bfloat16*>(gb + off) = hi;
                *reinterpret_cast<__nv_bfloat16*>(gb + off + 1024u) = lo;
              }
            }
            if (a.out_h) {
              float* p = a.out_h + o0;
#pragma unroll
              for (int k8 = 0; k8 < 8; ++k8)
                if (k8 < nv) p[(long long)k8 * H] = hv[k8];
            }
            if (a.seq_bf16) {
              __nv_bfloat16* p = a.seq_bf16 + ((long long)t * B + n0 + nl0) * a.ldh + j;
#pragma unroll
              for (int k8 = 0; k8 < 8; ++k8)
                if (k8 < nv) {
                  __nv_bfloat16 hi, lo;
                  seq_pair(hv[k8], hi, lo);
                  p[(long long)k8 * a.ldh] = hi;
                  p[a.seq_plane + (long long)k8 * a.ldh] = lo;
                }
            }
            if (a.c_last && t == T - 1) {
              float* p = a.c_last + (long long)(n0 + nl0) * H + j;
#pragma unroll
              for (int k8 = 0; k8 < 8; ++k8)
                if (k8 < nv) p[(long long)k8 * H] = cv[k8];
            }
          }
        }
        if (!fin) {
          tc_fence_before();
          warp_arrive(ckpt_done);
        }
      }
      if (!ok) break;
      fence_proxy_async_shared();  // h_t in the operand, before the next step's MMAs read it
      tc_fence_before();
      warp_arrive(h_ready);
    }
    if (!ok) atomicCAS(a.err, 0, kErrTcTimeout);
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA frees its shared memory while a peer may still write into it
  if (*err != 0) {     // after an abort: let copies already in flight towards this CTA land
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
}

template <int NS, int MT>
cudaError_t launch_seq_t(const TcMap& Vh_p, const TcMap& U64, const TcSeqArgs& a, cudaStream_t s) {
  auto kern = tc_seq_kernel<NS, MT>;
  const size_t smem = seq_layout(NS, MT, 128).total;  // the largest layout of this kernel
  static thread_local bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.cs, (a.B + NS - 1) / NS);
  cfg.blockDim = dim3(seq_threads(NS));
  cfg.dynamicSmemBytes = seq_layout(NS, MT, 4 * a.rpg).total;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeClusterDimension;
  attrs[0].val.clusterDim.x = a.cs;
  attrs[0].val.clusterDim.y = 1;
  attrs[0].val.clusterDim.z = 1;
  attrs[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, *reinterpret_cast<const CUtensorMap*>(Vh_p.bytes),
                            *reinterpret_cast<const CUtensorMap*>(U64.bytes), a);
}

}  // namespace

bool tc_seq_fits(int H, int B, int K, const Checkpoints& ck, int* ns, int* mt, std::string* why) {
  auto no = [&](const char* w) {
    if (why) *why = w;
    return false;
  };
  if (K > 32) return no("K above 32 (the factors of a CTA's units would not fit in shared memory)");
  for (int j = 0; j < ck.n; ++j)
    if (ck.k[j] % 16 != 0 && ck.k[j] < K) return no("an intermediate depth off the 16-term slices");
  // the narrowest tiles (16, 32 streams) whose clusters of 4 (or 2) CTAs fit
  // in one wave; each CTA owns 4, 8 or 16 streams of a tile, so its tau'
  // block (at most 128 rows x 16 streams) takes kSeqMaxRed elements per
  // epilogue thread at most
  const long long tiles16 = (B + 15) / 16, tiles32 = (B + 31) / 32;
  switch (H) {
    case 256: *ns = tiles16 <= 2 * kSeqMaxClusters4 ? 16 : 32; *mt = 1; return true;  // 2 CTAs x 128 units
    case 512:                                                                          // 4 x 128
      *ns = tiles16 <= kSeqMaxClusters4 ? 16 : (tiles32 <= kSeqMaxClusters4 ? 32 : 64);
      *mt = 1;
      return true;
    case 1024:  // 4 CTAs x 256 units (16 or 32 streams), else 8 x 128 (64 streams)
      if (tiles16 <= kSeqMaxClusters4) {
        *ns = 16;
        *mt = 2;
      } else if (tiles32 <= kSeqMaxClusters4) {
        *ns = 32;
        *mt = 2;
      } else {
        *ns = 64;
        *mt = 1;
      }
      return true;
    default: return no("H not 256, 512 or 1024");
  }
}

cudaError_t launch_tc_seq(const TcMap& Vh_p, const TcMap& U64, const TcSeqArgs& a, int ns, int mt, cudaStream_t s) {
  if (mt == 2) return ns == 16 ? launch_seq_t<16, 2>(Vh_p, U64, a, s) : launch_seq_t<32, 2>(Vh_p, U64, a, s);
  switch (ns) {
    case 16: return launch_seq_t<16, 1>(Vh_p, U64, a, s);
    case 32: return launch_seq_t<32, 1>(Vh_p, U64, a, s);
    default: return launch_seq_t<64, 1>(Vh_p, U64, a, s);
  }
}

}  // namespace lstm_approx_impl
