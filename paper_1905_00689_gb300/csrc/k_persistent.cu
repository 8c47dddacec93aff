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
//   phase B  CTA c owns UBv hidden units in four blocks of UW; warp w
//            serves gate w & 3 of unit block w >> 2, lane l the terms
//            [l*KT, (l+1)*KT).  The warp's slice of U (UW units x 32*KT terms
//            of one gate) lives in registers for the whole launch, so a lane
//            reads only its own KT values of tau' per step.  The UW partial
//            sums are reduced over the lanes by a transposed butterfly that
//            pairs neighbouring lanes first: after s steps lanes 0 .. 2^s - 1
//            hold the sums over the terms below KT * 2^s, so the gate sums at
//            the intermediate depths k_j of progressive inference fall out of
//            the same reduction (depths of another form take one masked pass
//            more).  After one block barrier thread (depth set n, unit u)
//            runs the cell update of Sec. II from the four gate sums: set 0
//            carries the state (c_t stays in a register), the other sets are
//            the outputs at the intermediate depths, computed from h_{t-1} and
//            c_{t-1} of the full-depth chain.  Warp 0 then pushes h_t to every
//            CTA like tau.
//
// Each warp waits on the exchange mbarriers itself (arrival count = number of
// warps) and re-arms them after its own wait; the partial sums, c_{t-1} and
// both exchanges are double-buffered by timestep parity, so the time loop
// holds one block barrier.  Every wait is bounded in wall time; a warp whose
// wait runs out writes the device status word, the whole CTA leaves the loop
// at that block barrier, and the cluster meets at one final barrier so that
// no CTA exits while a peer may still address its shared memory.
#include "internal.h"
#include "ptx.cuh"

#include <algorithm>

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTauSlack = 256;  // >= 32 * KT - Kp: lane reads past the last gate's rows
constexpr int kMaxGroupsPerWarp = 8;

struct DevPlan {
  int CS, RA, UBv, Kp, nset;
};

struct SmemLayout {
  uint32_t vh, tau, h, part, cs, hsend, total;  // float offsets after the barriers
};

// S4 = 4 * UW unit slots per CTA (the first UBv are real units).
__host__ __device__ inline SmemLayout smem_layout(const DevPlan& p, int H, int S4) {
  SmemLayout L;
  uint32_t o = 0;
  L.vh = o;    o += p.RA * H;
  L.tau = o;   o += 2 * (p.CS * p.RA + kTauSlack);
  L.h = o;     o += 2 * p.CS * p.UBv;
  L.part = o;  o += 2 * p.nset * 4 * S4;
  L.cs = o;    o += 2 * S4;
  L.hsend = o; o += S4;
  L.total = o;
  return L;
}
constexpr uint32_t kBarrierBytes = 128;  // 5 mbarriers, then the depths k_j

__host__ __device__ constexpr int ilog2(int v) { return v <= 1 ? 0 : 1 + ilog2(v >> 1); }

// Sum of NV values over the 32 lanes, transposed, pairing the high lane bits
// first: after the call lane l holds in v[0] the total of value l >> (5 - log2 NV).
template <int NV>
__device__ __forceinline__ void butterfly_transpose(float (&v)[NV], int lane) {
  constexpr int kSteps = ilog2(NV);
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

// Partial gate sums of the warp's UW units over this lane's terms s < lim
// (lim >= KT: all of them): v[i] = sum_s u[unit i][KT*lane + s] tau'[KT*lane + s].
template <int UW, int KT>
__device__ __forceinline__ void lane_partials(const float (&ureg)[UW][KT], const float* tau_lane, int lim,
                                              float (&v)[UW]) {
  float tv[KT];
  if constexpr (KT >= 4) {
#pragma unroll
    for (int q = 0; q < KT / 4; ++q) {
      const float4 f = *reinterpret_cast<const float4*>(tau_lane + 4 * q);
      tv[4 * q] = f.x; tv[4 * q + 1] = f.y; tv[4 * q + 2] = f.z; tv[4 * q + 3] = f.w;
    }
  } else if constexpr (KT == 2) {
    const float2 f = *reinterpret_cast<const float2*>(tau_lane);
    tv[0] = f.x; tv[1] = f.y;
  } else {
    tv[0] = tau_lane[0];
  }
#pragma unroll
  for (int s = 0; s < KT; ++s) tv[s] = s < lim ? tv[s] : 0.f;
#pragma unroll
  for (int i = 0; i < UW; ++i) {
    float acc = 0.f;
#pragma unroll
    for (int s = 0; s < KT; ++s) acc = fmaf(ureg[i][s], tv[s], acc);
    v[i] = acc;
  }
}

// Writes the values a lane holds after S steps of the neighbour-first
// butterfly: sums over the lanes 0 .. 2^S - 1, i.e. over the terms below
// KT * 2^S.  While S < log2 UW lane l < 2^S holds UW >> S values whose index
// has bit-reversed l as its top S bits; afterwards lane l < UW holds value
// bitrev(l).
template <int UW>
__device__ __forceinline__ void capture(const float (&v)[UW], int S, int lane, float* dst) {
  constexpr int L = ilog2(UW);
  if (S < L) {
    if (lane < (1 << S)) {
      const int base = S == 0 ? 0 : static_cast<int>(__brev(static_cast<unsigned>(lane)) >> (32 - S)) << (L - S);
#pragma unroll
      for (int i = 0; i < UW; ++i)
        if (i < (UW >> S)) dst[base + i] = v[i];
    }
  } else if (lane < UW) {
    dst[L == 0 ? 0 : static_cast<int>(__brev(static_cast<unsigned>(lane)) >> (32 - L))] = v[0];
  }
}

// Reduces the UW partials over the 32 lanes, neighbouring lanes first, and
// writes depth set n (bit n of cap[S]) to dst + n * set_stride after S steps.
template <int UW>
__device__ __forceinline__ void butterfly_depths(float (&v)[UW], int lane, const uint32_t (&cap)[6], float* dst,
                                                 int set_stride) {
  constexpr int L = ilog2(UW);
#pragma unroll
  for (int S = 0; S <= 5; ++S) {
    if (S > 0) {
      const int m = 1 << (S - 1);  // the step that makes S
      if (S - 1 < L) {
        const int half = UW >> S;
        const bool upper = (lane & m) != 0;
#pragma unroll
        for (int i = 0; i < UW / 2; ++i) {
          if (i < half) {
            const float keep = upper ? v[i + half] : v[i];
            const float send = upper ? v[i] : v[i + half];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, m);
          }
        }
      } else {
        v[0] += __shfl_xor_sync(0xffffffffu, v[0], m);
      }
    }
    for (uint32_t c = cap[S]; c != 0u; c &= c - 1u) capture<UW>(v, S, lane, dst + (__ffs(c) - 1) * set_stride);
  }
}

template <int UW, int KT>
__global__ void __launch_bounds__(kThreads, 1) persistent_kernel(PersistentArgs a, DevPlan p) {
  constexpr int S4 = 4 * UW;  // unit slots per CTA
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);  // [0,1] tau, [2,3] h, [4] set-up
  int* ck_s = reinterpret_cast<int*>(smem_raw + 48);        // the intermediate depths k_j
  float* sm = reinterpret_cast<float*>(smem_raw + kBarrierBytes);
  const SmemLayout SL = smem_layout(p, a.H, S4);
  float* vh_s = sm + SL.vh;
  float* tau_s = sm + SL.tau;
  float* h_s = sm + SL.h;
  float* part_s = sm + SL.part;    // [2][set][gate][S4] gate sums
  float* c_s = sm + SL.cs;         // [2][S4] c_{t-1} for the intermediate-depth cells
  float* hsend_s = sm + SL.hsend;  // [S4] h_t of this CTA's units
  const int part_buf = p.nset * 4 * S4;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / p.CS;  // one cluster per stream
  const int H = a.H, K = a.K, J = a.ck.n;
  const int tau_len = p.CS * p.RA + kTauSlack;
  const int h_len = p.CS * p.UBv;
  const uint32_t bytes_tau = p.CS * p.RA * 4u;
  const uint32_t bytes_h = p.CS * p.UBv * 4u;
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
    // first use of each exchange barrier: every warp arrives once, warp 0 with the bytes
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

  // U slice in registers: gate gw, unit slot ub*UW + i, term KT*lane + s.
  // U is K-major ([4][H][Ks]), so a lane's terms are one contiguous run and
  // the warp's reads are coalesced; all are issued before any is used.
  const int gw = warp & 3, ub = warp >> 2;
  const int k_lane = KT * lane;
  float ureg[UW][KT];
  const bool u_vec = (KT % 4 == 0) && (a.Ks % 4 == 0) && ((reinterpret_cast<uintptr_t>(a.U) & 15u) == 0);
#pragma unroll
  for (int i = 0; i < UW; ++i) {
    const int slot = ub * UW + i;
    const int j = rank * p.UBv + slot;
    const bool own = slot < p.UBv && j < H;
    const float* row = a.U + ((long long)gw * H + (own ? j : 0)) * a.Ks + k_lane;
    if constexpr (KT >= 4) {
#pragma unroll
      for (int q = 0; q < KT / 4; ++q) {
        const int kq = k_lane + 4 * q;
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (own && kq < K) {
          if (u_vec) {
            f = __ldg(reinterpret_cast<const float4*>(row + 4 * q));
          } else {
            f.x = __ldg(row + 4 * q);
            f.y = kq + 1 < K ? __ldg(row + 4 * q + 1) : 0.f;
            f.z = kq + 2 < K ? __ldg(row + 4 * q + 2) : 0.f;
            f.w = kq + 3 < K ? __ldg(row + 4 * q + 3) : 0.f;
          }
        }
        ureg[i][4 * q + 0] = kq + 0 < K ? f.x : 0.f;
        ureg[i][4 * q + 1] = kq + 1 < K ? f.y : 0.f;
        ureg[i][4 * q + 2] = kq + 2 < K ? f.z : 0.f;
        ureg[i][4 * q + 3] = kq + 3 < K ? f.w : 0.f;
      }
    } else {
#pragma unroll
      for (int s = 0; s < KT; ++s) ureg[i][s] = (own && k_lane + s < K) ? __ldg(row + s) : 0.f;
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
  // cell work: item n*S4 + u is depth set n of unit slot u; a thread takes
  // the items tid, tid + 512, ... which all have unit slot u = tid % S4
  const int cu = tid & (S4 - 1);
  const int cj = rank * p.UBv + cu;
  const bool unit_ok = cu < p.UBv && cj < H;
  float bias_r[4] = {0.f, 0.f, 0.f, 0.f};
  float c_reg = 0.f;  // the carried c of unit cu (threads tid < S4)
  if (unit_ok) {
#pragma unroll
    for (int g = 0; g < 4; ++g) bias_r[g] = a.bias[g * H + cj];
    if (tid < S4 && a.c0 != nullptr) c_reg = a.c0[(long long)b * H + cj];
  }
  if (tid < S4) c_s[tid] = c_reg;
  // where each depth set leaves the butterfly: set 0 (the full depth) and
  // every depth k_j >= K after all five steps, k_j = KT * 2^S after S steps;
  // other depths take a masked pass of their own
  uint32_t cap[6] = {0u, 0u, 0u, 0u, 0u, 1u};
  uint32_t masked = 0u;
#pragma unroll
  for (int n = 1; n <= kMaxCheckpoints; ++n) {
    if (n > J) break;
    const int c = a.ck.k[n - 1];
    if (tid == 0) ck_s[n - 1] = c;
    bool placed = c >= K;
    if (placed) cap[5] |= 1u << n;
#pragma unroll
    for (int S = 0; S < 5; ++S) {
      if (!placed && c == (KT << S)) {
        cap[S] |= 1u << n;
        placed = true;
      }
    }
    if (!placed) masked |= 1u << n;
  }
  float p_cur = p_off >= 0 ? __ldg(a.P + (long long)b * p_stride + p_off) : 0.f;

  const bool setup_ok = __syncthreads_and(mbar_wait_bounded<false>(bar_setup, 0, limit_ns, err));
  if (!setup_ok && tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
  cluster_sync_all();  // every CTA's barriers are armed before any st.async

  const uint32_t bar_tau0 = smem_u32(&bars[0]);
  const uint32_t bar_h0 = smem_u32(&bars[2]);
  const uint32_t tau_base = smem_u32(tau_s);
  const uint32_t h_base = smem_u32(h_s);

  for (int t = 0; t < (setup_ok ? a.T : 0); ++t) {
    const int hb = t & 1;
    int fail = 0;  // error code of a wait of this warp that ran out
    // prefetch the next step's projection for this lane's row
    const float p_next = (p_off >= 0 && t + 1 < a.T)
                             ? __ldg(a.P + ((long long)(t + 1) * a.B + b) * p_stride + p_off)
                             : 0.f;
    // ---- wait for h_{t-1} (t = 0 uses h0, loaded locally) ----------------
    if (t > 0) {
      const bool ok = mbar_wait_bounded<true>(bar_h0 + 8u * hb, ((t - 1) >> 1) & 1, limit_ns, err);
      if (!__all_sync(0xffffffffu, ok)) {
        fail = kErrWaitTimeoutB;
      } else if (lane == 0) {
        if (warp == 0) mbar_arrive_expect_tx(bar_h0 + 8u * hb, bytes_h);
        else mbar_arrive(bar_h0 + 8u * hb);
      }
    }

    // ---- phase A: tau' = sigma * (V_h h_{t-1} + P_t) for the owned rows ---
    const float4* h4 = reinterpret_cast<const float4*>(h_s + hb * h_len);
    for (int q = 0; fail == 0 && q < kMaxGroupsPerWarp; ++q) {
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
      const float tpr = sig_r * (mine + p_cur);
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
    if (fail == 0) {
      const bool ok = mbar_wait_bounded<true>(bar_tau0 + 8u * hb, (t >> 1) & 1, limit_ns, err);
      if (!__all_sync(0xffffffffu, ok)) {
        fail = kErrWaitTimeoutA;
      } else if (lane == 0) {
        if (warp == 0) mbar_arrive_expect_tx(bar_tau0 + 8u * hb, bytes_tau);
        else mbar_arrive(bar_tau0 + 8u * hb);
      }
    }

    // ---- phase B: gate sums of this warp's (gate, unit block) -------------
    float* pb = part_s + hb * part_buf;
    if (fail == 0) {
      const float* tau_lane = tau_s + hb * tau_len + gw * p.Kp + k_lane;
      float* dst = pb + gw * S4 + ub * UW;
      float v[UW];
      lane_partials<UW, KT>(ureg, tau_lane, KT, v);
      butterfly_depths<UW>(v, lane, cap, dst, 4 * S4);
      for (uint32_t m = masked; m != 0u; m &= m - 1u) {  // depths of another form
        const int n = __ffs(m) - 1;
        lane_partials<UW, KT>(ureg, tau_lane, ck_s[n - 1] - k_lane, v);
        butterfly_transpose<UW>(v, lane);
        // lane l holds the total of value l >> (5 - log2 UW)
        constexpr int kSh = 5 - ilog2(UW);
        if ((lane & ((1 << kSh) - 1)) == 0) dst[n * 4 * S4 + (lane >> kSh)] = v[0];
      }
    }
    // the one block barrier of the step: a wait that ran out in any warp ends
    // the time loop for the whole CTA here
    if (fail != 0 && lane == 0) atomicCAS(a.err, 0, fail);
    if (__syncthreads_or(fail)) break;

    // ---- the cell update (Sec. II) for every (depth set, unit) ------------
    const long long tbo = ((long long)t * a.B + b) * H;
    for (int item = tid; item < p.nset * S4; item += kThreads) {
      const int n = item / S4;
      const float* src = pb + n * 4 * S4 + cu;
      float hh = 0.f, cc = 0.f;
      if (unit_ok) {
        const float c_prev = n == 0 ? c_reg : c_s[hb * S4 + cu];
        lstm_cell_f(src[0] + bias_r[0], src[S4] + bias_r[1], src[2 * S4] + bias_r[2], src[3 * S4] + bias_r[3],
                    c_prev, hh, cc);
        if (n == 0) {
          c_reg = cc;
          a.out_h[tbo + cj] = hh;
        } else {
          const long long o = (long long)(n - 1) * a.T * a.B * H + tbo + cj;
          if (a.ckpt_h) a.ckpt_h[o] = hh;
          if (a.ckpt_c) a.ckpt_c[o] = cc;
        }
      }
      if (n == 0) {
        c_s[(hb ^ 1) * S4 + cu] = c_reg;
        hsend_s[cu] = hh;
      }
    }
    // ---- push h_t of this CTA's units to every CTA of the cluster ---------
    if (t + 1 < a.T) {
      bool send = false;
      if constexpr (S4 <= 32) {
        if (warp == 0) {
          __syncwarp();
          send = true;
        }
      } else {
        if (tid < S4) {
          asm volatile("bar.sync 1, %0;" ::"n"(S4) : "memory");  // the unit-slot threads of set 0
          send = warp == 0;
        }
      }
      if (send) {
        const int nb = (t + 1) & 1;
        const int nchunks = p.UBv >> 2;
        for (int m = lane; m < nchunks * p.CS; m += 32) {
          const int qd = m / p.CS, d = m - qd * p.CS;
          const float4 hv = *reinterpret_cast<const float4*>(hsend_s + 4 * qd);
          const uint32_t off = 4u * (nb * h_len + rank * p.UBv + 4 * qd);
          st_async_v4(mapa_shared(h_base + off, d), hv.x, hv.y, hv.z, hv.w, mapa_shared(bar_h0 + 8u * nb, d));
        }
      }
    }
    p_cur = p_next;
  }

  if (unit_ok && tid < S4 && a.c_last != nullptr) a.c_last[(long long)b * H + cj] = c_reg;
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while others may still address its shared memory
}

template <int UW, int KT>
cudaError_t launch_t(const DevPlan& dp, size_t smem, const PersistentArgs& a, cudaStream_t s) {
  auto kern = persistent_kernel<UW, KT>;
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
  int kt = 1;  // terms per lane: the smallest power of two that covers K with 32 lanes
  while (32 * kt < K) kt *= 2;
  const int cs_list[] = {1, 2, 4, 8, 16};
  PersistentPlan best;
  bool found = false;
  for (int cs : cs_list) {
    if (want_cs != 0 && cs != want_cs) continue;
    PersistentPlan p;
    p.CS = cs;
    p.RA = (((rows + cs - 1) / cs) + 3) & ~3;
    p.UB = (((H + cs - 1) / cs) + 3) & ~3;  // units owned by a CTA, a multiple of 4
    int uw = 1;                            // units per warp: four blocks cover UB
    while (4 * uw < p.UB) uw *= 2;
    if (uw > 16 || uw * kt > 64) continue;  // U registers per thread
    if ((p.RA / 4 + kWarps - 1) / kWarps > kMaxGroupsPerWarp) continue;
    p.upl = uw;
    p.kpw = kt;
    DevPlan dp{};
    dp.CS = p.CS; dp.RA = p.RA; dp.UBv = p.UB; dp.Kp = Kp; dp.nset = 1 + ck.n;
    p.smem = kBarrierBytes + 4ull * smem_layout(dp, H, 4 * uw).total;
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
  dp.CS = plan.CS; dp.RA = plan.RA; dp.UBv = plan.UB; dp.Kp = (a.K + 3) & ~3; dp.nset = 1 + a.ck.n;
  const int u = plan.upl, k = plan.kpw;
#define LA_CASE(U_, K_) \
  if (u == U_ && k == K_) return launch_t<U_, K_>(dp, plan.smem, a, s);
  LA_CASE(1, 1) LA_CASE(1, 2) LA_CASE(1, 4) LA_CASE(1, 8)
  LA_CASE(2, 1) LA_CASE(2, 2) LA_CASE(2, 4) LA_CASE(2, 8)
  LA_CASE(4, 1) LA_CASE(4, 2) LA_CASE(4, 4) LA_CASE(4, 8)
  LA_CASE(8, 1) LA_CASE(8, 2) LA_CASE(8, 4) LA_CASE(8, 8)
  LA_CASE(16, 1) LA_CASE(16, 2) LA_CASE(16, 4)
#undef LA_CASE
  return cudaErrorInvalidValue;
}

}  // namespace lstm_approx_impl
