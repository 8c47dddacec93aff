// Persistent small-batch kernel: one cluster launch covers all T timesteps.
//
// The work of one timestep (Eq. 1 for the four gates, then the cell update
// of Sec. II) has two all-to-all dependencies: every refinement coefficient
// tau_{g,k} = prune(v_{g,k})^T [x_t; h_{t-1}] needs all of h_{t-1}, and every
// gate output y_g[j] = sum_k sigma_{g,k} u_{g,k}[j] tau_{g,k} needs all tau.
// One cluster of CS CTAs (CS <= 16) serves one stream, and both halves of the
// factors stay on chip for the whole launch:
//
//   phase A  CTA c owns RA coefficient rows (gate-major row g*Kp + k) in
//            groups of four; warp w takes groups w, w + 16, ...  Its rows of
//            the pruned V_h (masked-dense, fp32) stay on chip: for hidden
//            sizes above 256 in tensor memory (HC = 1, 2), where lane l of the
//            warp holds the four rows' values at the h indices 4l + 128e + i
//            (e < 4*HC) and reads them with tcgen05.ld, so the
//            only shared-memory traffic is h itself; for smaller hidden sizes
//            (HC = 0) in shared memory, read with 128-bit loads.  The x part was hoisted
//            into P = V_x X for all t by an earlier launch and is prefetched
//            one step ahead.  tau' = sigma * (V_h h + P_t) of a group is
//            pushed into every CTA's tau buffer with one 16-byte st.async
//            per CTA, which completes the transaction count of the
//            receiver's mbarrier.
//   phase B  CTA c owns UBv hidden units in four blocks of UW; warp w serves
//            gate w & 3 of unit block w >> 2, lane l the terms
//            [l*KT, (l+1)*KT).  The warp's slice of U lives in registers, so
//            a lane reads only its own KT values of tau'.  The partial sums
//            are reduced over the lanes by a transposed butterfly that pairs
//            neighbouring lanes first: after s steps lanes 0 .. 2^s - 1 hold
//            the sums over the terms below KT * 2^s, so the gate sums at the
//            intermediate depths k_j of progressive inference fall out of the
//            same reduction (depths of another form take one masked pass
//            more).  The four warps of a unit block meet at a named barrier;
//            the block's leader warp then runs the cell update of Sec. II for
//            every (depth set, unit) of the block, keeping c_t of the full
//            depth in registers (the intermediate depths use h_{t-1} and
//            c_{t-1} of the full-depth chain), and pushes h_t of its units
//            to every CTA like tau.
//
// Each warp waits on the exchange mbarriers itself (arrival count = number of
// warps) and re-arms them after its own wait; the partial sums and both
// exchanges are double-buffered by timestep parity.  Every wait is bounded in
// wall time; a warp whose wait runs out writes the device status word and its
// unit block leaves the loop at the block barrier, the other blocks see the
// status word in their own waits, and the cluster meets at one final barrier
// so that no CTA exits while a peer may still address its shared memory.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTauSlack = 384;          // padding rows of the last CTA and lane reads past gate 3
constexpr int kMaxGroupsTmem = 2;       // groups of four V_h rows per warp, V_h in tensor memory
constexpr int kMaxGroupsSmem = 8;       // the same, V_h in shared memory
constexpr uint32_t kHeaderBytes = 192;  // 11 mbarriers, the TMEM address, the depths k_j
constexpr size_t kMinSmemBytes = 116 * 1024;

struct DevPlan {
  int CS, RA, UBv, Kp, nset, tcols;
};

struct SmemLayout {
  uint32_t vh, tau, h, part, total;  // float offsets after the header
};

__host__ __device__ constexpr int ilog2(int v) { return v <= 1 ? 0 : 1 + ilog2(v >> 1); }

// h buffer length: the CS * UBv received values, and at least the 32 * HL
// values the lanes of a tensor-memory phase A read (the tail stays zero).
__host__ __device__ inline int h_buffer_len(const DevPlan& p, int HC) {
  const int a = p.CS * p.UBv, b = 32 * 16 * HC;
  return a > b ? a : b;
}

// tau' layout: gate g's rows start at g * GP and term k sits at
// k + 4 * (k / 32), so that the 16-byte reads of neighbouring lanes in
// phase B fall into different banks; rows past the four gates (padding of
// the last CTA) follow at 4 * GP.
__host__ __device__ inline int tau_gate_len(int Kp) { return Kp + 4 * ((Kp + 31) / 32); }
__host__ __device__ inline int tau_pos(int row, int Kp) {
  const int g = row / Kp, k = row - g * Kp;
  return g < 4 ? g * tau_gate_len(Kp) + k + 4 * (k >> 5) : 4 * tau_gate_len(Kp) + (row - 4 * Kp);
}

// S4 = 4 * UW unit slots per CTA (the first UBv are real units).
__host__ __device__ inline SmemLayout smem_layout(const DevPlan& p, int H, int HC, int S4) {
  SmemLayout L;
  uint32_t o = 0;
  L.vh = o;   o += HC == 0 ? p.RA * H : 0;
  L.tau = o;  o += 2 * (4 * tau_gate_len(p.Kp) + kTauSlack);
  L.h = o;    o += 2 * h_buffer_len(p, HC);
  L.part = o; o += 2 * p.nset * 4 * S4;
  L.total = o;
  return L;
}

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

// The same from the warp's U values already loaded from tensor memory into
// registers (NP pairs of 16-column loads, value i*KT + s in pre[c/2][16 (c%2) + j]
// for column 16c + j).
template <int UW, int KT, int NP>
__device__ __forceinline__ void lane_partials_pre(const uint32_t (&pre)[2][32], const float* tau_lane,
                                                  float (&v)[UW]) {
  constexpr int NV = UW * KT;
  static_assert(NV <= 32 * NP, "prefetched columns cover the slice");
  float tv[KT];
#pragma unroll
  for (int q = 0; q < KT / 4; ++q) {
    const float4 f = *reinterpret_cast<const float4*>(tau_lane + 4 * q);
    tv[4 * q] = f.x; tv[4 * q + 1] = f.y; tv[4 * q + 2] = f.z; tv[4 * q + 3] = f.w;
  }
#pragma unroll
  for (int i = 0; i < UW; ++i) v[i] = 0.f;
#pragma unroll
  for (int idx = 0; idx < NV; ++idx)
    v[idx / KT] = fmaf(__uint_as_float(pre[idx / 32][idx % 32]), tv[idx % KT], v[idx / KT]);
}

// The same with the warp's slice of U in tensor memory at column u_col:
// value i*KT + s of the lane (unit i, term s) in column u_col + i*KT + s.
template <int UW, int KT>
__device__ __forceinline__ void lane_partials_tmem(uint32_t u_col, const float* tau_lane, int lim, float (&v)[UW]) {
  constexpr int NV = UW * KT;
  constexpr int NCH = (NV + 15) / 16;
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
  for (int i = 0; i < UW; ++i) v[i] = 0.f;
#pragma unroll
  for (int c = 0; c < NCH; c += 2) {
    float ua[16], ub[16];
    if (c + 1 < NCH) {
      tmem_ld16x2_sync(u_col + 16 * c, u_col + 16 * c + 16, ua, ub);
    } else {
      tmem_ld16_sync(u_col + 16 * c, ua);
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int idx = 16 * c + j;
      if (j < 16 || c + 1 < NCH) {
        if (idx < NV) {
          const float u = j < 16 ? ua[j] : ub[j - 16];
          v[idx / KT] = fmaf(u, tv[idx % KT], v[idx / KT]);
        }
      }
    }
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

// Named barrier of the `count` threads of one unit block; returns whether any
// of them passed `pred`.
__device__ __forceinline__ bool block_barrier_or(int id, int count, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
      "barrier.cta.red.or.pred q, %2, %3, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(pred ? 1u : 0u), "r"(id), "r"(count)
      : "memory");
  return r != 0u;
}

// One st.async of n = 1, 2 or 4 floats into (possibly remote) shared memory.
__device__ __forceinline__ void st_async_piece(uint32_t dst, const float (&v)[4], int n, uint32_t bar) {
  if (n == 4) {
    st_async_v4(dst, v[0], v[1], v[2], v[3], bar);
  } else if (n == 2) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(dst),
                 "f"(v[0]), "f"(v[1]), "r"(bar)
                 : "memory");
  } else {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(dst),
                 "r"(__float_as_uint(v[0])), "r"(bar)
                 : "memory");
  }
}

template <int UW, int KT, int HC>
__global__ void __launch_bounds__(kThreads, 1) persistent_kernel(PersistentArgs a, DevPlan p) {
  constexpr int S4 = 4 * UW;              // unit slots per CTA
  constexpr int HL = 16 * HC;             // h values per lane in a tensor-memory phase A
  constexpr bool kTmem = HC > 0;
  constexpr bool kUTmem = HC == 1;                     // U in tensor memory too
  // U (one or two column pairs) is loaded from tensor memory before the
  // tau' wait, so that the load latency hides behind the exchange (holding
  // V_h's columns across the h wait as well would spill registers)
  constexpr int kPreNP = (UW * KT + 31) / 32;
  constexpr bool kPreB = kUTmem && KT >= 4 && (UW * KT == 32 || UW * KT == 64);
  constexpr int UKC = kUTmem ? (UW * KT + 15) / 16 * 16 : 0;  // its columns per warp
  constexpr int kMaxGroups = kTmem ? kMaxGroupsTmem : kMaxGroupsSmem;
  constexpr int PIECE = UW < 4 ? UW : 4;  // units per h message
  extern __shared__ __align__(16) unsigned char smem_raw[];
  // mbarriers: [4 hb + g] tau' of gate g for parity hb, [8, 9] h, [10] set-up
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);
  uint32_t* taddr_s = reinterpret_cast<uint32_t*>(smem_raw + 96);  // TMEM base address
  int* ck_s = reinterpret_cast<int*>(smem_raw + 112);               // the intermediate depths k_j
  float* sm = reinterpret_cast<float*>(smem_raw + kHeaderBytes);
  const SmemLayout SL = smem_layout(p, a.H, HC, S4);
  float* vh_s = sm + SL.vh;  // V_h rows when they live in shared memory
  float* tau_s = sm + SL.tau;
  float* h_s = sm + SL.h;
  float* part_s = sm + SL.part;  // [2][set][gate][S4] gate sums
  const int part_buf = p.nset * 4 * S4;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / p.CS;  // one cluster per stream
  // a projection launched after this kernel may start now (it waits for nothing)
  if (a.proj_flags != nullptr) griddep_launch_dependents();
  const int H = a.H, K = a.K, J = a.ck.n;
  const int tau_len = 4 * tau_gate_len(p.Kp) + kTauSlack;
  const int h_len = h_buffer_len(p, HC);
  const uint32_t bytes_tau = p.Kp * 4u;  // one gate's rows (zero rows k >= K included)
  const uint32_t bytes_h = p.CS * p.UBv * 4u;
  const uint64_t limit_ns = static_cast<uint64_t>(a.wait_limit_ns);
  const volatile int* err = a.err;
  const int ngroups = p.RA >> 2;

  // ---- set-up: barriers, tensor memory, resident factors, initial state ---
  const uint32_t bar_setup = smem_u32(&bars[10]);
  if (tid == 0) {
    for (int i = 0; i < 8; ++i) mbar_init(smem_u32(&bars[i]), 4);  // the four warps of the gate
    for (int i = 8; i < 10; ++i) mbar_init(smem_u32(&bars[i]), kWarps);
    mbar_init(bar_setup, 1);
    if constexpr (!kTmem) {
      int nvalid = 0;  // V_h rows of this CTA that exist (the rest is padding)
      for (int lr = 0; lr < p.RA; ++lr) {
        const int gr = rank * p.RA + lr;
        nvalid += (gr / p.Kp < 4 && gr % p.Kp < K) ? 1 : 0;
      }
      mbar_arrive_expect_tx(bar_setup, 4u * H * nvalid);
    }
    fence_mbarrier_init_cluster();
  }
  if constexpr (kTmem) {
    if (warp == 0) {
      tmem_alloc(smem_u32(taddr_s), p.tcols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = kTmem ? *taddr_s : 0u;
  if (lane == 0) {
    // first use of each exchange barrier: every waiting warp arrives once,
    // the first of them with the bytes (tau': the warps of the gate, warp g
    // first; h: all warps, warp 0 first)
    for (int hb = 0; hb < 2; ++hb) {
      const uint32_t bt = smem_u32(&bars[4 * hb + (warp & 3)]);
      const uint32_t bytes = bytes_tau + ((hb == 0 && (warp & 3) == 0 && a.test_stall) ? 16u : 0u);
      if (warp < 4) mbar_arrive_expect_tx(bt, bytes);
      else mbar_arrive(bt);
      const uint32_t bh = smem_u32(&bars[8 + hb]);
      if (warp == 0) mbar_arrive_expect_tx(bh, bytes_h);
      else mbar_arrive(bh);
    }
  }
  for (int i = tid; i < 2 * tau_len; i += kThreads) tau_s[i] = 0.f;
  for (int i = tid; i < h_len; i += kThreads) {
    h_s[i] = (a.h0 != nullptr && i < H) ? a.h0[(long long)b * H + i] : 0.f;
    h_s[h_len + i] = 0.f;
  }

  // V_h rows of this CTA into tensor memory.  Thread (warp w, lane l) holds,
  // for its groups q (group w + 16 q), the values of the group's four rows at
  // the h indices 4*l + 128*e4 + i (e4 < HL/4, i < 4; consecutive lanes read
  // consecutive 16-byte quads of h) in its TMEM lane 32*(w & 3) + l: quad e4
  // of row r at column
  // (w >> 2) * (G*4*HL) + q*4*HL + 16*e4 + 4*r + i, so that one 16-column
  // load brings one h quad of all four rows.
  const int G = (ngroups + kWarps - 1) / kWarps;
  const uint32_t t_lane = tmem_base + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
  const uint32_t t_col0 = static_cast<uint32_t>((warp >> 2) * G * 4 * HL);
  for (int q = 0; kTmem && q < G; ++q) {
    const int grp = warp + kWarps * q;
    const float* rowp[4];  // the group's four rows (null: padding)
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int gr = rank * p.RA + grp * 4 + r;
      const int g = gr / p.Kp, k = gr % p.Kp;
      rowp[r] = (grp < ngroups && g < 4 && k < K) ? a.Vh + ((long long)g * a.Ks + k) * a.ldh : nullptr;
    }
    // all loads of a half (up to 8 h quads x 4 rows) are issued before the
    // first store, so the set-up pays one memory round trip per half
#pragma unroll
    for (int h0 = 0; h0 < HL / 4; h0 += 4) {
      float4 f[4][4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int hi = 4 * lane + 128 * (h0 + e);
#pragma unroll
        for (int r = 0; r < 4; ++r)
          f[e][r] = (rowp[r] != nullptr && hi < H) ? __ldg(reinterpret_cast<const float4*>(rowp[r] + hi))
                                                   : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v[16];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          v[4 * r] = f[e][r].x; v[4 * r + 1] = f[e][r].y; v[4 * r + 2] = f[e][r].z; v[4 * r + 3] = f[e][r].w;
        }
        tmem_st16(t_lane + t_col0 + q * 4 * HL + 16 * (h0 + e), v);
      }
    }
  }
  if constexpr (kTmem) {
    tmem_wait_st();
  } else {
    // V_h rows into shared memory: one bulk copy per row, completing on the
    // set-up barrier; padding rows are cleared with plain stores
    for (int lr = tid; lr < p.RA; lr += kThreads) {
      const int gr = rank * p.RA + lr;
      const int g = gr / p.Kp, k = gr % p.Kp;
      if (g < 4 && k < K) {
        bulk_copy_g2s(smem_u32(vh_s + lr * H), a.Vh + ((long long)g * a.Ks + k) * a.ldh, 4u * H, bar_setup);
      } else {
        float4* dst = reinterpret_cast<float4*>(vh_s + lr * H);
        for (int c4 = 0; c4 < (H >> 2); ++c4) dst[c4] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
  }

  // per-lane row data for phase A: lane 8r + q (tensor memory) or lane
  // 4q + r (shared memory) <-> row r of this warp's group q
  long long p_off = -1;  // offset of this lane's row inside one (t, b) slice of P
  float sig_r = 0.f;
  {
    const int q = kTmem ? (lane & 7) : (lane >> 2), r = kTmem ? (lane >> 3) : (lane & 3);
    const int grp = warp + kWarps * q;
    if (q < kMaxGroups && grp < ngroups) {
      const int gr = rank * p.RA + grp * 4 + r;
      const int g = gr / p.Kp, k = gr % p.Kp;
      if (g < 4 && k < K) {
        p_off = (long long)g * a.Ks + k;
        sig_r = a.sigma[p_off];
      }
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
  // with U in tensor memory: lane l of warp w holds its UW*KT values in
  // columns 16*G*HL + (w >> 2) * UKC + [0, UW*KT)
  const uint32_t u_col = t_lane + static_cast<uint32_t>(16 * G * HL + (warp >> 2) * UKC);
  if constexpr (kUTmem) {
#pragma unroll
    for (int c = 0; c < UKC / 16; ++c) {
      float uv[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int idx = 16 * c + j;
        uv[j] = idx < UW * KT ? ureg[idx / KT][idx % KT] : 0.f;
      }
      tmem_st16(u_col + 16 * c, uv);
    }
    tmem_wait_st();
  }
  // cell state in the unit block's leader, the warp of gate ub (so that the
  // four leaders sit on different SM sub-partitions): lane n*UW + i runs
  // depth set n of unit slot ub*UW + i; lanes i < UW carry c of the full depth
  const bool leader = gw == ub;
  const int ci = lane & (UW - 1);
  const int c_slot = ub * UW + ci;
  const int cj = rank * p.UBv + c_slot;
  const bool unit_ok = c_slot < p.UBv && cj < H;
  float bias_r[4] = {0.f, 0.f, 0.f, 0.f};
  float c_reg = 0.f;
  if (leader && unit_ok) {
#pragma unroll
    for (int g = 0; g < 4; ++g) bias_r[g] = a.bias[g * H + cj];
    if (lane < UW && a.c0 != nullptr) c_reg = a.c0[(long long)b * H + cj];
  }
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
  // everything above only read the factors; P is written by the projection,
  // launched either just before this kernel (which may still be running) or
  // just after it (whose CTAs each raise a flag once their part is stored)
  bool setup_ok = true;
  if (a.proj_flags == nullptr) griddep_wait();
  else if (warp == 0) setup_ok = wait_flags_epoch(a.proj_flags, a.proj_nflags, a.proj_epoch, limit_ns, err);

  // remote addresses of the exchange buffers in CTA (lane mod CS)
  const uint32_t peer = static_cast<uint32_t>(lane) & static_cast<uint32_t>(p.CS - 1);
  const uint32_t bar_tau0 = smem_u32(&bars[0]);
  const uint32_t bar_h0 = smem_u32(&bars[8]);
  const uint32_t r_tau = mapa_shared(smem_u32(tau_s), peer);
  const uint32_t r_bar_tau = mapa_shared(bar_tau0, peer);
  const uint32_t r_h = mapa_shared(smem_u32(h_s), peer);
  const uint32_t r_bar_h = mapa_shared(bar_h0, peer);
  const int lcs = ilog2(p.CS);

  if constexpr (!kTmem) setup_ok = mbar_wait_bounded<false>(bar_setup, 0, limit_ns, err) && setup_ok;
  if (!__syncthreads_and(setup_ok) && tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
  // P through L2 (it may have been written while this kernel ran)
  float p_cur = p_off >= 0 ? __ldcg(a.P + (long long)b * p_stride + p_off) : 0.f;
  cluster_sync_all();  // every CTA's barriers are armed before any st.async

  const int t_end = *err == 0 ? a.T : 0;  // nothing to do after a failed set-up
  bool failed = false;                     // a wait of this unit block ran out
  for (int t = 0; t < t_end; ++t) {
    const int hb = t & 1;
    int fail = 0;  // error code of a wait of this warp that ran out
    // prefetch the next step's projection for this lane's row
    const float p_next = (p_off >= 0 && t + 1 < a.T)
                             ? __ldcg(a.P + ((long long)(t + 1) * a.B + b) * p_stride + p_off)
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
    if constexpr (!kTmem) {
      const float4* h4 = reinterpret_cast<const float4*>(h_s + hb * h_len);
      const int H4 = H >> 2;
      for (int q = 0; fail == 0 && q < kMaxGroups; ++q) {
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
        // transposed reduction: lanes 8r .. 8r+7 then hold row r's full sum;
        // lane 4q + r finishes row r, then the senders gather the four
        float rs[4] = {acc0, acc1, acc2, acc3};
        butterfly_transpose<4>(rs, lane);
        const float mine = __shfl_sync(0xffffffffu, rs[0], (lane & 3) << 3);
        const float tpr = sig_r * (mine + p_cur);
        const float t0 = __shfl_sync(0xffffffffu, tpr, 4 * q + 0);
        const float t1 = __shfl_sync(0xffffffffu, tpr, 4 * q + 1);
        const float t2 = __shfl_sync(0xffffffffu, tpr, 4 * q + 2);
        const float t3 = __shfl_sync(0xffffffffu, tpr, 4 * q + 3);
        const int gr = rank * p.RA + lr0, gg = gr / p.Kp;  // padding rows past gate 3 are not sent
        if (lane < p.CS && gg < 4) {
          const uint32_t off = 4u * (hb * tau_len + tau_pos(gr, p.Kp));
          st_async_v4(r_tau + off, t0, t1, t2, t3, r_bar_tau + 8u * (4 * hb + gg));
        }
      }
    }
    if (kTmem && fail == 0) {
      const float* hsrc = h_s + hb * h_len + 4 * lane;
#pragma unroll 1
      for (int q = 0; q < G; ++q) {
        const int grp = warp + kWarps * q;
        if (grp >= ngroups) break;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        // two h quads per round: two 16-column loads, one wait
#pragma unroll
        for (int e8 = 0; e8 < HL / 8; ++e8) {
          const float4 ha = *reinterpret_cast<const float4*>(hsrc + 256 * e8);
          const float4 hb4 = *reinterpret_cast<const float4*>(hsrc + 256 * e8 + 128);
          float va[16], vb[16];
          const uint32_t col = t_lane + t_col0 + q * 4 * HL + 32 * e8;
          tmem_ld16x2_sync(col, col + 16, va, vb);
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            float s0 = acc[r];
            s0 = fmaf(va[4 * r + 0], ha.x, s0);
            s0 = fmaf(va[4 * r + 1], ha.y, s0);
            s0 = fmaf(va[4 * r + 2], ha.z, s0);
            s0 = fmaf(va[4 * r + 3], ha.w, s0);
            s0 = fmaf(vb[4 * r + 0], hb4.x, s0);
            s0 = fmaf(vb[4 * r + 1], hb4.y, s0);
            s0 = fmaf(vb[4 * r + 2], hb4.z, s0);
            s0 = fmaf(vb[4 * r + 3], hb4.w, s0);
            acc[r] = s0;
          }
        }
        // transposed reduction of the four row sums: afterwards lanes
        // 8r .. 8r+7 hold the full sum of row r of the group
        butterfly_transpose<4>(acc, lane);
        const float tpr = sig_r * (acc[0] + p_cur);  // valid on lane 8r + q
        const float t0 = __shfl_sync(0xffffffffu, tpr, q);
        const float t1 = __shfl_sync(0xffffffffu, tpr, 8 + q);
        const float t2 = __shfl_sync(0xffffffffu, tpr, 16 + q);
        const float t3 = __shfl_sync(0xffffffffu, tpr, 24 + q);
        const int gr = rank * p.RA + grp * 4, gg = gr / p.Kp;  // padding rows past gate 3 are not sent
        if (lane < p.CS && gg < 4) {
          const uint32_t off = 4u * (hb * tau_len + tau_pos(gr, p.Kp));
          st_async_v4(r_tau + off, t0, t1, t2, t3, r_bar_tau + 8u * (4 * hb + gg));
        }
      }
    }

    // U slice of this warp, loaded while tau' is in flight
    uint32_t upre[2][32];
    if constexpr (kPreB) {
      tmem_ld16x2_issue(u_col, u_col + 16, upre[0]);
      if constexpr (kPreNP == 2) tmem_ld16x2_issue(u_col + 32, u_col + 48, upre[1]);
    }
    // ---- wait for this warp's gate of tau' --------------------------------
    if (fail == 0) {
      // only this warp's gate: the four CTAs that hold its rows
      const uint32_t bt = bar_tau0 + 8u * (4 * hb + gw);
      const bool ok = mbar_wait_bounded<true>(bt, (t >> 1) & 1, limit_ns, err);
      if (!__all_sync(0xffffffffu, ok)) {
        fail = kErrWaitTimeoutA;
      } else if (lane == 0) {
        if (warp < 4) mbar_arrive_expect_tx(bt, bytes_tau);
        else mbar_arrive(bt);
      }
    }

    if constexpr (kPreB) {  // also after a failed wait: no load stays outstanding
      tmem_wait_ld_tie32(upre[0]);
      if constexpr (kPreNP == 2) tmem_wait_ld_tie32(upre[1]);
    }

    // ---- phase B: gate sums of this warp's (gate, unit block) -------------
    float* pb = part_s + hb * part_buf;
    if (fail == 0) {
      const float* tau_lane = tau_s + hb * tau_len + gw * tau_gate_len(p.Kp) + k_lane + 4 * (k_lane >> 5);
      float* dst = pb + gw * S4 + ub * UW;
      float v[UW];
      if constexpr (kPreB) lane_partials_pre<UW, KT, kPreNP>(upre, tau_lane, v);
      else if constexpr (kUTmem) lane_partials_tmem<UW, KT>(u_col, tau_lane, KT, v);
      else lane_partials<UW, KT>(ureg, tau_lane, KT, v);
      butterfly_depths<UW>(v, lane, cap, dst, 4 * S4);
      for (uint32_t m = masked; m != 0u; m &= m - 1u) {  // depths of another form
        const int n = __ffs(m) - 1;
        if constexpr (kUTmem) lane_partials_tmem<UW, KT>(u_col, tau_lane, ck_s[n - 1] - k_lane, v);
        else lane_partials<UW, KT>(ureg, tau_lane, ck_s[n - 1] - k_lane, v);
        butterfly_transpose<UW>(v, lane);
        // lane l holds the total of value l >> (5 - log2 UW)
        constexpr int kSh = 5 - ilog2(UW);
        if ((lane & ((1 << kSh) - 1)) == 0) dst[n * 4 * S4 + (lane >> kSh)] = v[0];
      }
    }
    if (fail != 0 && lane == 0) atomicCAS(a.err, 0, fail);
    // the four warps of the unit block meet; a wait that ran out in any of
    // them ends the time loop for the whole block here
    if (block_barrier_or(1 + ub, 128, fail != 0)) {
      failed = true;
      break;
    }

    // ---- cell update (Sec. II) and h_t exchange, in the block's leader ----
    if (leader) {
      const long long tbo = ((long long)t * a.B + b) * H;
      const float cp = __shfl_sync(0xffffffffu, c_reg, ci);  // c_{t-1} of unit ci
      float h_new = 0.f;
      // the cells of the first round (the full depth and the first depth
      // sets) are computed before h_t is sent and stored after it, so that
      // the output stores are not on the path to the next timestep
      const int n_first = lane / UW;
      float hh0 = 0.f, cc0 = 0.f;
      if (n_first < p.nset && unit_ok) {
        const float* src = pb + n_first * 4 * S4 + c_slot;
        lstm_cell_f(src[0] + bias_r[0], src[S4] + bias_r[1], src[2 * S4] + bias_r[2], src[3 * S4] + bias_r[3], cp,
                    hh0, cc0);
        if (n_first == 0) {
          c_reg = cc0;
          h_new = hh0;
        }
      }
      if (t + 1 < a.T) {
        // lane m takes (piece m >> log2 CS, CTA m & (CS-1)), then m + 32
        const int nb = (t + 1) & 1;
        constexpr int kPieces = UW / PIECE;
#pragma unroll
        for (int m0 = 0; m0 < 64; m0 += 32) {
          const int pc = (m0 + lane) >> lcs;
          const int src0 = (pc < kPieces ? pc : 0) * PIECE;
          float hv[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) hv[e] = __shfl_sync(0xffffffffu, h_new, src0 + (e < PIECE ? e : 0));
          const int slot = ub * UW + pc * PIECE;
          if (pc < kPieces && slot < p.UBv) {
            const uint32_t off = 4u * (nb * h_len + rank * p.UBv + slot);
            st_async_piece(r_h + off, hv, PIECE, r_bar_h + 8u * nb);
          }
        }
      }
      if (n_first < p.nset && unit_ok) {
        if (n_first == 0) {
          a.out_h[tbo + cj] = hh0;
        } else {
          const long long o = (long long)(n_first - 1) * a.T * a.B * H + tbo + cj;
          if (a.ckpt_h) a.ckpt_h[o] = hh0;
          if (a.ckpt_c) a.ckpt_c[o] = cc0;
        }
      }
      for (int n0 = 32 / UW; n0 < p.nset; n0 += 32 / UW) {
        const int n = n0 + lane / UW;
        if (n < p.nset && unit_ok) {
          const float* src = pb + n * 4 * S4 + c_slot;
          float hh, cc;
          lstm_cell_f(src[0] + bias_r[0], src[S4] + bias_r[1], src[2 * S4] + bias_r[2], src[3 * S4] + bias_r[3], cp,
                      hh, cc);
          const long long o = (long long)(n - 1) * a.T * a.B * H + tbo + cj;
          if (a.ckpt_h) a.ckpt_h[o] = hh;
          if (a.ckpt_c) a.ckpt_c[o] = cc;
        }
      }
    }
    p_cur = p_next;
  }

  if (leader && lane < UW && unit_ok && a.c_last != nullptr) a.c_last[(long long)b * H + cj] = c_reg;
  tc_fence_before();
  __syncthreads();
  if (kTmem && warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tcols);
  }
  cluster_sync_all();  // no CTA leaves while others may still address its shared memory
  if (__syncthreads_or(failed)) {
    // after a wait ran out, copies and stores issued just before the peers
    // stopped may still be in flight towards this CTA: let them land
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
  }
}

template <int UW, int KT, int HC>
cudaError_t launch_t(const DevPlan& dp, size_t smem, const PersistentArgs& a, cudaStream_t s) {
  auto kern = persistent_kernel<UW, KT, HC>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(dp.CS * a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = dp.CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // may start while the projection before it finishes (set-up overlaps it);
  // with the projection launched after it, an ordinary launch
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = a.proj_flags == nullptr ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
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
  if (H > 1024) {
    *why = "hidden size above 1024";
    return false;
  }
  const int Kp = (K + 3) & ~3;
  const int rows = 4 * Kp;
  int kt = 1;  // terms per lane: the smallest power of two that covers K with 32 lanes
  while (32 * kt < K) kt *= 2;
  const int hc = H <= 256 ? 0 : H <= 512 ? 1 : 2;  // V_h in shared memory (0) or tensor memory
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
    if (hc > 0 && uw < 8) continue;         // the tensor-memory variant is built for UW >= 8
    if (hc == 2 && uw != 16) continue;
    const int groups = (p.RA / 4 + kWarps - 1) / kWarps;
    if (groups > (hc > 0 ? kMaxGroupsTmem : kMaxGroupsSmem)) continue;
    int tcols = 0;
    if (hc > 0) {
      const int ukc = hc == 1 ? (uw * kt + 15) / 16 * 16 : 0;  // U in tensor memory for hc == 1
      const int need = 4 * (groups * 4 * 16 * hc + ukc);
      if (need > 512) continue;
      tcols = 32;
      while (tcols < need) tcols *= 2;
    }
    p.upl = uw;
    p.kpw = kt;
    p.hc = hc;
    p.tcols = tcols;
    DevPlan dp{};
    dp.CS = p.CS; dp.RA = p.RA; dp.UBv = p.UB; dp.Kp = Kp; dp.nset = 1 + ck.n; dp.tcols = tcols;
    p.smem = kHeaderBytes + 4ull * smem_layout(dp, H, hc, 4 * uw).total;
    if (p.smem > 227u * 1024u) continue;
    // at least half of an SM's shared memory, so that no other CTA of this
    // kernel shares the SM (and its tensor memory) with this one
    if (p.smem < kMinSmemBytes) p.smem = kMinSmemBytes;
    best = p;
    found = true;
    if (want_cs != 0) break;
    // automatic choice: the first (smallest) cluster whose V_h slice is small
    if ((size_t)p.RA * H * 4 <= 32u * 1024u) break;
  }
  if (!found) {
    *why = "shape does not fit the persistent kernel (hidden size, K or on-chip memory)";
    return false;
  }
  *plan = best;
  return true;
}

cudaError_t launch_persistent(const PersistentPlan& plan, const PersistentArgs& a, cudaStream_t s) {
  DevPlan dp{};
  dp.CS = plan.CS; dp.RA = plan.RA; dp.UBv = plan.UB; dp.Kp = (a.K + 3) & ~3; dp.nset = 1 + a.ck.n;
  dp.tcols = plan.tcols;
  const int u = plan.upl, k = plan.kpw, h = plan.hc;
#define LA_CASE(U_, K_, H_) \
  if (u == U_ && k == K_ && h == H_) return launch_t<U_, K_, H_>(dp, plan.smem, a, s);
  LA_CASE(1, 1, 0) LA_CASE(1, 2, 0) LA_CASE(1, 4, 0) LA_CASE(1, 8, 0)
  LA_CASE(2, 1, 0) LA_CASE(2, 2, 0) LA_CASE(2, 4, 0) LA_CASE(2, 8, 0)
  LA_CASE(4, 1, 0) LA_CASE(4, 2, 0) LA_CASE(4, 4, 0) LA_CASE(4, 8, 0)
  LA_CASE(8, 1, 0) LA_CASE(8, 2, 0) LA_CASE(8, 4, 0) LA_CASE(8, 8, 0)
  LA_CASE(16, 1, 0) LA_CASE(16, 2, 0) LA_CASE(16, 4, 0)
  LA_CASE(8, 1, 1) LA_CASE(8, 2, 1) LA_CASE(8, 4, 1) LA_CASE(8, 8, 1)
  LA_CASE(16, 1, 1) LA_CASE(16, 2, 1) LA_CASE(16, 4, 1)
  LA_CASE(16, 1, 2) LA_CASE(16, 2, 2) LA_CASE(16, 4, 2)
#undef LA_CASE
  return cudaErrorInvalidValue;
}

}  // namespace lstm_approx_impl
