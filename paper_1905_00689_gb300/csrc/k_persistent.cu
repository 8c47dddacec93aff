// Persistent small-batch kernel: one cluster launch covers all T timesteps.
//
// The work of one timestep (Eq. 1 for the four gates, then the cell update
// of Sec. II) has two all-to-all dependencies: every refinement coefficient
// tau_{g,k} = prune(v_{g,k})^T [x_t; h_{t-1}] needs all of h_{t-1}, and every
// gate output y_g[j] = sum_k sigma_{g,k} u_{g,k}[j] tau_{g,k} needs all tau.
// One cluster of CS CTAs (CS <= 16) serves one stream:
//
//   phase A  CTA c owns RA coefficient rows (gate-major row g*Kp + k), in
//            groups of four per warp.  Its rows of the pruned V_h
//            (masked-dense, fp32) stay in shared memory for the whole launch;
//            the x part was hoisted into P = V_x X for all t by an earlier
//            launch and is prefetched one step ahead into registers.
//            tau' = sigma * (V_h h + P_t) for a group of rows is pushed into
//            every CTA's tau buffer with one 16-byte st.async per CTA, which
//            completes the transaction count of the receiver's mbarrier.
//   phase B  CTA c owns UB = 16 * UPW hidden units, warp w the UPW units
//            w*UPW + i.  The warp's slice of U (UPW units x 4 gates x K terms)
//            lives in registers for the whole launch, lane l holding terms
//            [l*KPL, (l+1)*KPL).  The 4*UPW gate sums are reduced across the
//            lanes with a transposed butterfly, the cell update runs on lane i
//            for unit i (which keeps c_t in a register), and h_t is pushed to
//            every CTA like tau.  Outputs at the intermediate depths k_j are
//            computed after h_t has left, off the critical path, from masked
//            sums over the same registers.
//
// No block-wide barrier sits in the time loop: every warp waits on the two
// mbarriers itself (arrival count = number of warps) and re-arms them after
// its own wait.  Both exchanges are double-buffered by timestep parity.
// Every wait is bounded in wall time; a warp whose wait runs out writes the
// device status word and leaves the loop, the others notice the word and
// leave too, and the cluster meets at one final barrier so that no CTA exits
// while a peer may still address its shared memory.
#include "internal.h"
#include "ptx.cuh"

#include <algorithm>

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTauSlack = 256;  // >= 32 * KPL: the widest read past the last row
constexpr int kMaxGroupsPerWarp = 8;

struct DevPlan {
  int CS, RA, UB, Kp;
};

struct SmemLayout {
  uint32_t vh, tau, h, total;  // float offsets after the barriers
};

__host__ __device__ inline SmemLayout smem_layout(const DevPlan& p, int H) {
  SmemLayout L;
  uint32_t o = 0;
  L.vh = o;  o += max(p.RA * H, 8 * p.UB);  // V_h slice; also the U staging area
  L.tau = o; o += 2 * (p.CS * p.RA + kTauSlack);
  L.h = o;   o += 2 * p.CS * p.UB;
  L.total = o;
  return L;
}
constexpr uint32_t kBarrierBytes = 64;

// Sum of NV values over the 32 lanes, transposed: after the call lane l
// holds in v[0] the total of value index l >> (5 - log2(NV)).
template <int NV>
__device__ __forceinline__ void butterfly_transpose(float (&v)[NV], int lane) {
  constexpr int kSteps = NV == 32 ? 5 : NV == 16 ? 4 : NV == 8 ? 3 : NV == 4 ? 2 : NV == 2 ? 1 : 0;
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

// Terms held by a lane: slot s of lane l is term k(l, s).  Lanes take
// interleaved 16-byte runs (4 l + 128 q + r for KPL >= 4) so that the
// 128-bit shared-memory reads of tau' are free of bank conflicts.
template <int KPL>
__device__ __forceinline__ int term_of(int lane, int s) {
  if constexpr (KPL >= 4) return 4 * lane + 128 * (s >> 2) + (s & 3);
  else return KPL * lane + s;
}

template <int KPL>
__device__ __forceinline__ void load_tau(const float* tau, int g, int Kp, int lane, float (&tv)[KPL]) {
  const float* src = tau + g * Kp;
  if constexpr (KPL >= 4) {
#pragma unroll
    for (int q = 0; q < KPL / 4; ++q) {
      const float4 f = *reinterpret_cast<const float4*>(src + 4 * lane + 128 * q);
      tv[4 * q] = f.x; tv[4 * q + 1] = f.y; tv[4 * q + 2] = f.z; tv[4 * q + 3] = f.w;
    }
  } else if constexpr (KPL == 2) {
    const float2 f = *reinterpret_cast<const float2*>(src + 2 * lane);
    tv[0] = f.x; tv[1] = f.y;
  } else {
    tv[0] = src[lane];
  }
}

// Partial gate sums of the warp's units over this lane's terms for NS depth
// cut-offs at once (set 0 = the full depth K; sets 1.. = intermediate depths):
// v[n][i*4 + g] = sum over the lane's terms k < cut[n] of u_{g,k}[unit i] tau'_{g,k}.
// The lane's terms come in runs of G = min(KPL, 4) consecutive terms; one
// accumulator per run is kept and the depth sets are formed from the runs
// with selects, so the FMA count does not grow with NS.  Exact when every
// cut-off is a multiple of G (the caller checks that).
template <int UPW, int KPL, int NS>
__device__ __forceinline__ void gate_partials(const float (&ureg)[UPW][4][KPL], const float* tau, int Kp, int lane,
                                              const int (&cut)[NS], float (&v)[NS][4 * UPW]) {
  constexpr int G = KPL < 4 ? KPL : 4;
  constexpr int NR = KPL / G;  // runs per lane
  float acc[NR][4 * UPW];
#pragma unroll
  for (int r = 0; r < NR; ++r)
#pragma unroll
    for (int i = 0; i < 4 * UPW; ++i) acc[r][i] = 0.f;
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    float tv[KPL];
    load_tau<KPL>(tau, g, Kp, lane, tv);
#pragma unroll
    for (int s = 0; s < KPL; ++s)
#pragma unroll
      for (int i = 0; i < UPW; ++i) acc[s / G][i * 4 + g] = fmaf(ureg[i][g][s], tv[s], acc[s / G][i * 4 + g]);
  }
#pragma unroll
  for (int n = 0; n < NS; ++n) {
#pragma unroll
    for (int i = 0; i < 4 * UPW; ++i) v[n][i] = 0.f;
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const bool in = term_of<KPL>(lane, r * G) < cut[n];  // the whole run is below the cut-off
#pragma unroll
      for (int i = 0; i < 4 * UPW; ++i) v[n][i] += in ? acc[r][i] : 0.f;
    }
  }
}

// Partial gate sums over this lane's terms k < kcut, term by term (any kcut).
template <int UPW, int KPL>
__device__ __forceinline__ void masked_partials(const float (&ureg)[UPW][4][KPL], const float* tau, int Kp, int lane,
                                                int kcut, float (&v)[4 * UPW]) {
#pragma unroll
  for (int i = 0; i < 4 * UPW; ++i) v[i] = 0.f;
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    float tv[KPL];
    load_tau<KPL>(tau, g, Kp, lane, tv);
#pragma unroll
    for (int s = 0; s < KPL; ++s) {
      const float t = term_of<KPL>(lane, s) < kcut ? tv[s] : 0.f;
#pragma unroll
      for (int i = 0; i < UPW; ++i) v[i * 4 + g] = fmaf(ureg[i][g][s], t, v[i * 4 + g]);
    }
  }
}

// Reduce one set of partials over the lanes and gather: lane i < UPW gets the
// four gate pre-activations of unit w*UPW + i in y[0..3].
template <int UPW>
__device__ __forceinline__ void reduce_gates(float (&v)[4 * UPW], int lane, float (&y)[4]) {
  constexpr int NV = 4 * UPW;
  constexpr int kShift = NV == 16 ? 1 : NV == 8 ? 2 : 3;  // 5 - log2(NV)
  butterfly_transpose<NV>(v, lane);
  const int src_unit = lane < UPW ? lane : 0;
#pragma unroll
  for (int g = 0; g < 4; ++g) y[g] = __shfl_sync(0xffffffffu, v[0], (src_unit * 4 + g) << kShift);
}

template <int UPW>
__device__ __forceinline__ void send_h(uint32_t dst, uint32_t bar, const float (&hv)[UPW]) {
  if constexpr (UPW == 4) {
    st_async_v4(dst, hv[0], hv[1], hv[2], hv[3], bar);
  } else if constexpr (UPW == 2) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(dst),
                 "f"(hv[0]), "f"(hv[1]), "r"(bar)
                 : "memory");
  } else {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(dst),
                 "r"(__float_as_uint(hv[0])), "r"(bar)
                 : "memory");
  }
}

template <int UPW, int KPL, int NCK>
__global__ void __launch_bounds__(kThreads, 1) persistent_kernel(PersistentArgs a, DevPlan p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);  // [0,1] tau, [2,3] h
  float* sm = reinterpret_cast<float*>(smem_raw + kBarrierBytes);
  const SmemLayout S = smem_layout(p, a.H);
  float* vh_s = sm + S.vh;
  float* tau_s = sm + S.tau;
  float* h_s = sm + S.h;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / p.CS;  // one cluster per stream
  const int H = a.H, K = a.K;
  const int tau_len = p.CS * p.RA + kTauSlack;
  const int h_len = p.CS * p.UB;
  const uint32_t bytes_tau = p.CS * p.RA * 4u;
  const uint32_t bytes_h = p.CS * p.UB * 4u;
  const uint64_t limit_ns = static_cast<uint64_t>(a.wait_limit_ns);
  const volatile int* err = a.err;

  // ---- set-up: barriers, resident factors, initial state -----------------
  if (tid == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&bars[i]), kWarps);
    mbar_init(smem_u32(&bars[4]), 1);
    int nvalid = 0;  // V_h rows of this CTA that exist (the rest is padding)
    for (int lr = 0; lr < p.RA; ++lr) {
      const int gr = rank * p.RA + lr;
      nvalid += (gr / p.Kp < 4 && gr % p.Kp < K) ? 1 : 0;
    }
    mbar_arrive_expect_tx(smem_u32(&bars[4]), 4u * H * nvalid);
    fence_mbarrier_init_cluster();
  }
  __syncthreads();
  if (lane == 0) {
    // first use of each barrier: every warp arrives once, warp 0 with the bytes
    for (int i = 0; i < 4; ++i) {
      const uint32_t bytes = (i < 2 ? bytes_tau : bytes_h) + ((i == 0 && a.test_stall) ? 16u : 0u);
      if (warp == 0) mbar_arrive_expect_tx(smem_u32(&bars[i]), bytes);
      else mbar_arrive(smem_u32(&bars[i]));
    }
  }
  for (int i = tid; i < 2 * tau_len; i += kThreads) tau_s[i] = 0.f;
  for (int i = tid; i < h_len; i += kThreads)
    h_s[i] = (a.h0 != nullptr && i < H) ? a.h0[(long long)b * H + i] : 0.f;

  // per-lane row data for phase A: lane 4q + r <-> row r of this warp's q-th group
  const int ngroups = p.RA >> 2;
  const int my_q = lane >> 2;
  const int my_group = warp + kWarps * my_q;
  const bool row_lane = my_q < kMaxGroupsPerWarp && my_group < ngroups;
  long long p_off = -1;  // offset of this lane's row inside one (t, b) slice of P
  float sig_r = 0.f;
  if (row_lane) {
    const int gr = rank * p.RA + my_group * 4 + (lane & 3);
    const int g = gr / p.Kp, k = gr % p.Kp;
    if (g < 4 && k < K) {
      p_off = (long long)g * a.Ks + k;
      sig_r = a.sigma[p_off];
    }
  }
  const long long p_stride = 4LL * a.Ks;

  // U slice in registers: unit w*UPW + i, gate g, slot s <-> term
  // term_of(lane, s).  U is K-major ([4][H][Ks]), so a lane's terms are
  // contiguous runs and the loads below are coalesced 128-bit reads, all
  // issued before any is used.
  float ureg[UPW][4][KPL];
  float bias_r[4] = {0.f, 0.f, 0.f, 0.f};
  float c_reg = 0.f;
  const int my_unit = warp * UPW + (lane < UPW ? lane : 0);
  const int my_j = rank * p.UB + my_unit;
  const bool cell_lane = lane < UPW && my_j < H;
  const bool u_vec = (a.Ks % 4 == 0) && ((reinterpret_cast<uintptr_t>(a.U) & 15u) == 0);
#pragma unroll
  for (int i = 0; i < UPW; ++i) {
    const int j = rank * p.UB + warp * UPW + i;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const float* row = a.U + ((long long)g * H + (j < H ? j : 0)) * a.Ks;
      if constexpr (KPL >= 4) {
#pragma unroll
        for (int q = 0; q < KPL / 4; ++q) {
          const int k0 = 4 * lane + 128 * q;
          float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
          if (j < H && k0 < K) {
            if (u_vec) {
              f = __ldg(reinterpret_cast<const float4*>(row + k0));
            } else {
              f.x = __ldg(row + k0);
              f.y = k0 + 1 < K ? __ldg(row + k0 + 1) : 0.f;
              f.z = k0 + 2 < K ? __ldg(row + k0 + 2) : 0.f;
              f.w = k0 + 3 < K ? __ldg(row + k0 + 3) : 0.f;
            }
          }
          ureg[i][g][4 * q + 0] = k0 + 0 < K ? f.x : 0.f;
          ureg[i][g][4 * q + 1] = k0 + 1 < K ? f.y : 0.f;
          ureg[i][g][4 * q + 2] = k0 + 2 < K ? f.z : 0.f;
          ureg[i][g][4 * q + 3] = k0 + 3 < K ? f.w : 0.f;
        }
      } else {
#pragma unroll
        for (int sl = 0; sl < KPL; ++sl) {
          const int k = term_of<KPL>(lane, sl);
          ureg[i][g][sl] = (j < H && k < K) ? __ldg(row + k) : 0.f;
        }
      }
    }
  }
  // V_h rows owned by this CTA (run row gr = rank*RA + lr = g*Kp + k): one
  // bulk copy per row into shared memory, completing on the set-up barrier;
  // padding rows are cleared with plain stores.
  const int H4 = H >> 2;
  const uint32_t bar_setup = smem_u32(&bars[4]);
  for (int lr = tid; lr < p.RA; lr += kThreads) {
    const int gr = rank * p.RA + lr;
    const int g = gr / p.Kp, k = gr % p.Kp;
    if (g < 4 && k < K) {
      bulk_copy_g2s(smem_u32(vh_s + lr * H), a.Vh + ((long long)g * a.Ks + k) * a.ldh, 4u * H, bar_setup);
    } else {
      float4* dst = reinterpret_cast<float4*>(vh_s + lr * H);
      for (int c4 = 0; c4 < H4; ++c4) dst[c4] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  // every lane holds the bias of unit lane % UPW (the combined reduction
  // below lets lane n*UPW + i run the cell of depth set n, unit i)
  {
    const int jb = rank * p.UB + warp * UPW + lane % UPW;
    if (jb < H) {
#pragma unroll
      for (int g = 0; g < 4; ++g) bias_r[g] = a.bias[g * H + jb];
    }
  }
  if (cell_lane) c_reg = a.c0 != nullptr ? a.c0[(long long)b * H + my_j] : 0.f;
  float p_cur = p_off >= 0 ? __ldg(a.P + (long long)b * p_stride + p_off) : 0.f;

  const bool setup_ok = __syncthreads_and(mbar_wait_bounded<false>(bar_setup, 0, limit_ns, err));
  if (!setup_ok && tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
  cluster_sync_all();  // every CTA's barriers are armed before any st.async

  const uint32_t bar_tau0 = smem_u32(&bars[0]);
  const uint32_t bar_h0 = smem_u32(&bars[2]);
  const uint32_t tau_base = smem_u32(tau_s);
  const uint32_t h_base = smem_u32(h_s);

  // intermediate depths handled in the fused pass: the leading ones (at most
  // NCK) that fall on a run boundary of the lanes' terms
  int nfused = 0;
  {
    constexpr int G = KPL < 4 ? KPL : 4;
    while (nfused < NCK && nfused < a.ck.n && a.ck.k[nfused] % G == 0) ++nfused;
  }
  for (int t = 0; t < (setup_ok ? a.T : 0); ++t) {
    const int hb = t & 1;
    // prefetch the next step's projection for this lane's row
    const float p_next = (p_off >= 0 && t + 1 < a.T)
                             ? __ldg(a.P + ((long long)(t + 1) * a.B + b) * p_stride + p_off)
                             : 0.f;
    // ---- wait for h_{t-1} (t = 0 uses h0, loaded locally) ----------------
    if (t > 0) {
      const bool ok = mbar_wait_bounded<true>(bar_h0 + 8u * hb, ((t - 1) >> 1) & 1, limit_ns, err);
      if (!__all_sync(0xffffffffu, ok)) {
        if (lane == 0) atomicCAS(a.err, 0, kErrWaitTimeoutB);
        break;
      }
      if (lane == 0) {
        if (warp == 0) mbar_arrive_expect_tx(bar_h0 + 8u * hb, bytes_h);
        else mbar_arrive(bar_h0 + 8u * hb);
      }
    }

    // ---- phase A: tau' = sigma * (V_h h_{t-1} + P_t) for the owned rows ---
    const float4* h4 = reinterpret_cast<const float4*>(h_s + hb * h_len);
    const float tpr_lane = sig_r;  // sigma of this lane's row (0 for padding rows)
    for (int q = 0; q < kMaxGroupsPerWarp; ++q) {
      const int grp = warp + kWarps * q;
      if (grp >= ngroups) break;
      const int lr0 = grp * 4;
      float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
      const float4* v0 = reinterpret_cast<const float4*>(vh_s + (lr0 + 0) * H);
      const float4* v1 = reinterpret_cast<const float4*>(vh_s + (lr0 + 1) * H);
      const float4* v2 = reinterpret_cast<const float4*>(vh_s + (lr0 + 2) * H);
      const float4* v3 = reinterpret_cast<const float4*>(vh_s + (lr0 + 3) * H);
#pragma unroll 1
      for (int c4 = lane; c4 < H4; c4 += 32) {
        const float4 hv = h4[c4];
        float4 w = v0[c4];
        acc0 = fmaf(w.x, hv.x, fmaf(w.y, hv.y, fmaf(w.z, hv.z, fmaf(w.w, hv.w, acc0))));
        w = v1[c4];
        acc1 = fmaf(w.x, hv.x, fmaf(w.y, hv.y, fmaf(w.z, hv.z, fmaf(w.w, hv.w, acc1))));
        w = v2[c4];
        acc2 = fmaf(w.x, hv.x, fmaf(w.y, hv.y, fmaf(w.z, hv.z, fmaf(w.w, hv.w, acc2))));
        w = v3[c4];
        acc3 = fmaf(w.x, hv.x, fmaf(w.y, hv.y, fmaf(w.z, hv.z, fmaf(w.w, hv.w, acc3))));
      }
      // transposed reduction of the four row sums: afterwards lane l holds the
      // full sum of row (l >> 3) of the group
      float rs[4] = {acc0, acc1, acc2, acc3};
      butterfly_transpose<4>(rs, lane);
      // lane 4q + r finishes row r of group q, then the senders gather the four
      const int r = lane & 3;
      const float mine = __shfl_sync(0xffffffffu, rs[0], r << 3);
      const float tpr = tpr_lane * (mine + p_cur);
      const float t0 = __shfl_sync(0xffffffffu, tpr, 4 * q + 0);
      const float t1 = __shfl_sync(0xffffffffu, tpr, 4 * q + 1);
      const float t2 = __shfl_sync(0xffffffffu, tpr, 4 * q + 2);
      const float t3 = __shfl_sync(0xffffffffu, tpr, 4 * q + 3);
      if (lane < p.CS) {
        const uint32_t off = 4u * (hb * tau_len + rank * p.RA + lr0);
        st_async_v4(mapa_shared(tau_base + off, lane), t0, t1, t2, t3, mapa_shared(bar_tau0 + 8u * hb, lane));
      }
    }

    // ---- wait for every CTA's tau' ----------------------------------------
    {
      const bool ok = mbar_wait_bounded<true>(bar_tau0 + 8u * hb, (t >> 1) & 1, limit_ns, err);
      if (!__all_sync(0xffffffffu, ok)) {
        if (lane == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
        break;
      }
      if (lane == 0) {
        if (warp == 0) mbar_arrive_expect_tx(bar_tau0 + 8u * hb, bytes_tau);
        else mbar_arrive(bar_tau0 + 8u * hb);
      }
    }

    // ---- phase B: gate sums (full depth + fused intermediate depths) ------
    const float* tau = tau_s + hb * tau_len;
    constexpr int NS = 1 + NCK;
    int cut[NS];
    cut[0] = K;
#pragma unroll
    for (int n = 1; n < NS; ++n) cut[n] = n - 1 < nfused ? a.ck.k[n - 1] : 0;
    float v[NS][4 * UPW];
    gate_partials<UPW, KPL, NS>(ureg, tau, p.Kp, lane, cut, v);
    const float c_prev = c_reg;
    float h_new = 0.f;
    constexpr int NT = NS * 4 * UPW;  // values to reduce over the lanes
    if constexpr (NS > 1 && NT <= 32) {
      // one transposed butterfly over every (depth set, unit, gate) value;
      // lane n*UPW + i then runs the cell of set n, unit i, all in parallel
      constexpr int P = NT <= 16 ? 16 : 32;
      constexpr int kShiftP = P == 32 ? 0 : 1;
      float w[P];
#pragma unroll
      for (int n = 0; n < NS; ++n)
#pragma unroll
        for (int e = 0; e < 4 * UPW; ++e) w[n * 4 * UPW + e] = v[n][e];
#pragma unroll
      for (int e = NT; e < P; ++e) w[e] = 0.f;
      butterfly_transpose<P>(w, lane);
      const int L = lane < NS * UPW ? lane : 0;
      const int n = L / UPW, iu = L % UPW;
      float yy[4];
#pragma unroll
      for (int g = 0; g < 4; ++g) yy[g] = __shfl_sync(0xffffffffu, w[0], (n * 4 * UPW + iu * 4 + g) << kShiftP);
      const float cp = __shfl_sync(0xffffffffu, c_reg, iu);
      const int jl = rank * p.UB + warp * UPW + iu;
      const long long tbl = ((long long)t * a.B + b) * H + jl;
      if (lane < NS * UPW && jl < H) {
        float hh, cc;
        lstm_cell_f(yy[0] + bias_r[0], yy[1] + bias_r[1], yy[2] + bias_r[2], yy[3] + bias_r[3], cp, hh, cc);
        if (n == 0) {
          c_reg = cc;
          h_new = hh;
          a.out_h[tbl] = hh;
        } else if (n - 1 < nfused) {
          const long long o = (long long)(n - 1) * a.T * a.B * H + tbl;
          if (a.ckpt_h) a.ckpt_h[o] = hh;
          if (a.ckpt_c) a.ckpt_c[o] = cc;
        }
      }
    } else {
      float y[4];
      reduce_gates<UPW>(v[0], lane, y);
      if (cell_lane) {
        float cn;
        lstm_cell_f(y[0] + bias_r[0], y[1] + bias_r[1], y[2] + bias_r[2], y[3] + bias_r[3], c_prev, h_new, cn);
        c_reg = cn;
        a.out_h[((long long)t * a.B + b) * H + my_j] = h_new;
      }
    }
    const long long tb = ((long long)t * a.B + b) * H + my_j;
    if (t + 1 < a.T) {
      float hv[UPW];
#pragma unroll
      for (int i = 0; i < UPW; ++i) hv[i] = __shfl_sync(0xffffffffu, h_new, i);
      if (lane < p.CS) {
        const int nb = (t + 1) & 1;
        const uint32_t off = 4u * (nb * h_len + rank * p.UB + warp * UPW);
        send_h<UPW>(mapa_shared(h_base + off, lane), mapa_shared(bar_h0 + 8u * nb, lane), hv);
      }
    }
    // ---- intermediate depths not covered above, after h_t has left --------
    const int first_seq = (NS > 1 && NT <= 32) ? nfused : 0;
    for (int jj = first_seq; jj < a.ck.n; ++jj) {
      float yk[4];
      if (jj < nfused) {
#pragma unroll
        for (int n = 1; n < NS; ++n)
          if (n - 1 == jj) reduce_gates<UPW>(v[n], lane, yk);
      } else {  // depths beyond the fused ones: one more pass each
        float v1[4 * UPW];
        masked_partials<UPW, KPL>(ureg, tau, p.Kp, lane, a.ck.k[jj], v1);
        reduce_gates<UPW>(v1, lane, yk);
      }
      if (cell_lane) {
        float hh, cc;
        lstm_cell_f(yk[0] + bias_r[0], yk[1] + bias_r[1], yk[2] + bias_r[2], yk[3] + bias_r[3], c_prev, hh, cc);
        const long long o = (long long)jj * a.T * a.B * H + tb;
        if (a.ckpt_h) a.ckpt_h[o] = hh;
        if (a.ckpt_c) a.ckpt_c[o] = cc;
      }
    }
    p_cur = p_next;
  }

  if (cell_lane && a.c_last != nullptr) a.c_last[(long long)b * H + my_j] = c_reg;
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while others may still address its shared memory
}

template <int UPW, int KPL, int NCK>
cudaError_t launch_t(const DevPlan& dp, size_t smem, const PersistentArgs& a, cudaStream_t s) {
  auto kern = persistent_kernel<UPW, KPL, NCK>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(dp.CS * a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = dp.CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // function attributes once per instantiation (the largest shared memory any
  // plan may ask for); the co-residency check once per (cluster size, smem)
  static thread_local bool attrs_set = false;
  static thread_local unsigned long long checked[16] = {};
  if (!attrs_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    attrs_set = true;
  }
  const unsigned long long key = (static_cast<unsigned long long>(smem) << 8) | static_cast<unsigned>(dp.CS);
  bool seen = false;
  for (unsigned long long k : checked) seen |= (k == key);
  if (!seen) {
    int nclusters = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg);
    if (e != cudaSuccess) return e;
    if (nclusters < 1) return cudaErrorNotPermitted;
    for (auto& k : checked)
      if (k == 0) {
        k = key;
        break;
      }
  }
  return cudaLaunchKernelEx(&cfg, kern, a, dp);
}

}  // namespace

bool plan_persistent(int H, int K, int T, const Checkpoints& ck, int want_cs, int sm_count, PersistentPlan* plan,
                     std::string* why) {
  (void)sm_count;
  (void)T;
  (void)ck;
  if (H % 4 != 0) {
    *why = "hidden size not a multiple of 4";
    return false;
  }
  if (K > 256) {
    *why = "K above 256";
    return false;
  }
  const int Kp = (K + 3) & ~3;
  const int rows = 4 * Kp;
  int kpl = 1;
  while (32 * kpl < K) kpl *= 2;
  const int cs_list[] = {1, 2, 4, 8, 16};
  PersistentPlan best;
  bool found = false;
  for (int cs : cs_list) {
    if (want_cs != 0 && cs != want_cs) continue;
    PersistentPlan p;
    p.CS = cs;
    p.RA = (((rows + cs - 1) / cs) + 3) & ~3;
    const int units = (H + cs - 1) / cs;
    p.upl = units <= 16 ? 1 : units <= 32 ? 2 : units <= 64 ? 4 : 0;  // units per warp
    if (p.upl == 0) continue;
    if (p.upl * 4 * kpl > 64) continue;
    if ((p.RA / 4 + kWarps - 1) / kWarps > kMaxGroupsPerWarp) continue;
    p.UB = 16 * p.upl;
    p.kpw = kpl;
    DevPlan dp{};
    dp.CS = p.CS; dp.RA = p.RA; dp.UB = p.UB; dp.Kp = Kp;
    const SmemLayout L = smem_layout(dp, H);
    p.smem = kBarrierBytes + 4ull * L.total;
    if (p.smem > 227u * 1024u) continue;
    best = p;
    found = true;
    if (want_cs != 0) break;
    // automatic choice: the first (smallest) cluster whose V_h slice is small
    if ((size_t)p.RA * H * 4 <= 32u * 1024u) break;
  }
  if (!found) {
    *why = "shape does not fit the persistent kernel (hidden size, K or shared memory)";
    return false;
  }
  *plan = best;
  return true;
}

cudaError_t launch_persistent(const PersistentPlan& plan, const PersistentArgs& a, cudaStream_t s) {
  DevPlan dp{};
  dp.CS = plan.CS; dp.RA = plan.RA; dp.UB = plan.UB; dp.Kp = (a.K + 3) & ~3;
  const int u = plan.upl, k = plan.kpw;
  const bool fused = a.ck.n > 0;
#define LA_CASE(U_, K_)                                            \
  if (u == U_ && k == K_)                                          \
    return fused ? launch_t<U_, K_, 2>(dp, plan.smem, a, s) : launch_t<U_, K_, 0>(dp, plan.smem, a, s);
  LA_CASE(1, 1) LA_CASE(1, 2) LA_CASE(1, 4) LA_CASE(1, 8)
  LA_CASE(2, 1) LA_CASE(2, 2) LA_CASE(2, 4) LA_CASE(2, 8)
  LA_CASE(4, 1) LA_CASE(4, 2) LA_CASE(4, 4)
#undef LA_CASE
  return cudaErrorInvalidValue;
}

}  // namespace lstm_approx_impl
