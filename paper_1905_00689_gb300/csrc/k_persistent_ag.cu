// Persistent small-batch kernel with one exchange per timestep.
//
// Same problem as k_persistent.cu (Eq. 1 for the four gates, then the cell
// update of Sec. II, all T timesteps in one cluster launch), organised so
// that a timestep needs one all-to-all instead of two.  With CS in {4, 8, 16}
// CTAs, each gate's Kp refinement terms are split into CS/4 ranges of RA
// terms and CTA c owns gate g = c / (CS/4) and terms [k0, k0 + RA):
//
//   phase A  tau'_{g,k} = sigma (V_h h_{t-1} + P_t) for the CTA's own RA
//            rows, exactly as in k_persistent.cu (rows of V_h in tensor
//            memory, h from shared memory), written to local shared memory:
//            no exchange, since only this CTA needs them.
//   phase B  thread u (one per hidden unit) forms the CTA's partial gate sum
//            y_c[u] = sum_{k in own range} u_{g,k}[u] tau'_{g,k}, with its RA
//            values of U in tensor memory and tau' read by broadcast, plus a
//            masked sum for every intermediate depth k_j that falls inside
//            the range (progressive inference: the sums below k_j reuse the
//            same products, nothing is recomputed).
//   exchange the partial vectors (H floats each) go to every CTA of the
//            cluster with one bulk copy per destination (TMA engine, shared
//            to distributed shared memory), completing on the receiver's
//            mbarrier.
//   cells    every CTA adds, for each unit and gate, the partials of that
//            gate's CS/4 CTAs in a fixed order and runs all H cells of
//            Sec. II at full depth itself: h_t is then local to every CTA,
//            ready for the next phase A, and the CTAs hold bit-identical
//            states.  CTA c owns the unit block [c UB, (c + 1) UB): it writes
//            those units' outputs and runs their cells at each k_j (from the
//            carried c_{t-1}); a masked partial therefore only travels to the
//            CTA that owns its units.
//
// Receive buffers, send buffers and h are double-buffered by timestep
// parity.  A send buffer is rewritten two steps later, after this CTA has
// received every peer's step t + 1 partials; a peer sends those only after
// its step t wait completed, so every step t copy has landed (and read its
// source) by then.  Every wait is bounded in wall time; a CTA whose wait runs out
// writes the device status word and leaves the time loop at the step's last
// block barrier, the others see the word in their own waits, and the cluster
// meets at one final barrier before any CTA exits.
#include "internal.h"
#include "ptx.cuh"

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr uint32_t kHeaderBytes = 128;  // mbarriers [2], TMEM address, depth table
constexpr size_t kMinSmemBytes = 116 * 1024;

struct AgPlan {
  int CS, RA, Kp, UB;  // UB: units per output block (a multiple of 4)
  int nmask;           // intermediate depths that fall strictly inside some CTA's range
  int tcols;
};

struct AgLayout {
  uint32_t tau, h, send, rfull, rmask, total;  // float offsets after the header
};

// tau_own [RA + 16], h [2][512], send [2][1 + nmask][H],
// recv_full [2][CS][H], recv_mask [2][nmask][4][UB]
__host__ __device__ inline AgLayout ag_layout(const AgPlan& p, int H) {
  AgLayout L;
  uint32_t o = 0;
  L.tau = o;   o += p.RA + 16;
  L.h = o;     o += 2 * 512;
  L.send = o;  o += 2 * (1 + p.nmask) * H;
  L.rfull = o; o += 2 * p.CS * H;
  L.rmask = o; o += 2 * p.nmask * 4 * p.UB;
  L.total = o;
  return L;
}


// Sum of NV values over the 32 lanes, transposed (high lane bits first):
// afterwards lane l holds in v[0] the total of value l >> (5 - log2 NV).
template <int NV>
__device__ __forceinline__ void lanes_sum_transposed(float (&v)[NV], int lane) {
  constexpr int kSteps = NV == 4 ? 2 : NV == 2 ? 1 : 0;
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


// HQ: h quads per lane in phase A (1, 2, 4 for H up to 128, 256, 512)
template <int HQ>
__global__ void __launch_bounds__(kThreads, 1) persistent_ag_kernel(PersistentArgs a, AgPlan p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);          // receive barriers [2]
  uint32_t* taddr_s = reinterpret_cast<uint32_t*>(smem_raw + 16);  // TMEM base address
  // per depth n: the range holding the cut, the cut inside it, the masked slot
  int* cut_part = reinterpret_cast<int*>(smem_raw + 32);
  int* cut_rem = cut_part + kMaxCheckpoints;
  int* cut_slot = cut_rem + kMaxCheckpoints;
  float* sm = reinterpret_cast<float*>(smem_raw + kHeaderBytes);
  const int H = a.H, K = a.K, J = a.ck.n;
  const AgLayout SL = ag_layout(p, H);
  float* tau_s = sm + SL.tau;      // [RA + 16] this CTA's tau' (zero past RA)
  float* h_s = sm + SL.h;          // [2][512] h_{t-1} (zero past H)
  float* send_s = sm + SL.send;    // [2][1 + nmask][H] partial sums to send
  float* rfull_s = sm + SL.rfull;  // [2][CS][H] full-range partials of every CTA
  float* rmask_s = sm + SL.rmask;  // [2][nmask][4][UB] masked partials of the own unit block

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / p.CS;  // one cluster per stream
  // a projection launched after this kernel may start now (it waits for nothing)
  if (a.proj_flags != nullptr) griddep_launch_dependents();
  const int per_gate = p.CS / 4;    // CTAs sharing one gate's terms
  const int gate = (int)rank / per_gate, part = (int)rank % per_gate;
  const int k0 = part * p.RA;       // first own term
  const int RAp = (p.RA + 15) & ~15;
  const uint64_t limit_ns = static_cast<uint64_t>(a.wait_limit_ns);
  const volatile int* err = a.err;
  const int ngroups = p.RA >> 2;  // at most kWarps: warp w computes rows 4w .. 4w+3 of the range
  const int send_len = (1 + p.nmask) * H;
  const int rfull_len = p.CS * H, rmask_len = p.nmask * 4 * p.UB;
  const int ub0 = (int)rank * p.UB;                       // own unit block [ub0, ub0 + my_ub)
  const int my_ub = max(0, min(p.UB, H - ub0));

  // depth n: the range of each gate that holds the cut (per_gate when the
  // depth reaches K), the cut inside it (0 when it falls on a range
  // boundary) and its masked-partial slot (-1: none)
  uint32_t own_slots = 0u;  // slots this CTA computes
  {
    int slot = 0;
    for (int n = 0; n < J; ++n) {
      const int c = a.ck.k[n];
      const bool inside = c < K && (c % p.RA) != 0;
      const int cp = c >= K ? per_gate : c / p.RA;
      if (tid == 0) {
        cut_part[n] = cp;
        cut_rem[n] = inside ? c % p.RA : 0;
        cut_slot[n] = inside ? slot : -1;
      }
      if (inside && cp == part) own_slots |= 1u << slot;
      if (inside) ++slot;
    }
  }
  const uint32_t bytes_in = (uint32_t)(rfull_len + p.nmask * 4 * my_ub) * 4u;

  // ---- set-up ---------------------------------------------------------------
  if (tid == 0) {
    mbar_init(smem_u32(&bars[0]), 1);
    mbar_init(smem_u32(&bars[1]), 1);
    fence_mbarrier_init_cluster();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(taddr_s), p.tcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *taddr_s;
  if (tid == 0) {  // both receive phases armed: step 0 uses barrier 0, step 1 barrier 1
    mbar_arrive_expect_tx(smem_u32(&bars[0]), bytes_in + (a.test_stall ? 16u : 0u));
    mbar_arrive_expect_tx(smem_u32(&bars[1]), bytes_in);
  }
  for (int i = tid; i < p.RA + 16; i += kThreads) tau_s[i] = 0.f;
  for (int i = tid; i < 512; i += kThreads) {
    h_s[i] = (a.h0 != nullptr && i < H) ? a.h0[(long long)b * H + i] : 0.f;
    h_s[512 + i] = 0.f;
  }
  // V_h rows of this CTA in tensor memory (the lane quarter of warp w,
  // columns (w >> 2) * 16 HQ onwards): lane l holds h quads 4l + 128e, and
  // row r of the warp's four at column 16e + 4r + i
  const uint32_t t_lane = tmem_base + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
  const uint32_t t_col0 = static_cast<uint32_t>((warp >> 2) * 16 * HQ);
  {
    const float* rowp[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int k = k0 + warp * 4 + r;
      rowp[r] = (warp < ngroups && k < K) ? a.Vh + ((long long)gate * a.Ks + k) * a.ldh : nullptr;
    }
#pragma unroll 1
    for (int e = 0; e < HQ; ++e) {
      const int hi = 4 * lane + 128 * e;
      float v[16];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const float4 f = (rowp[r] != nullptr && hi < H) ? __ldg(reinterpret_cast<const float4*>(rowp[r] + hi))
                                                        : make_float4(0.f, 0.f, 0.f, 0.f);
        v[4 * r] = f.x; v[4 * r + 1] = f.y; v[4 * r + 2] = f.z; v[4 * r + 3] = f.w;
      }
      tmem_st16(t_lane + t_col0 + 16 * e, v);
    }
  }
  // U of unit tid for this gate's own terms, RAp columns from u_col
  const uint32_t u_col = t_lane + static_cast<uint32_t>(64 * HQ + (warp >> 2) * RAp);
  {
    const bool own = tid < H;
    const float* urow = a.U + ((long long)gate * H + (own ? tid : 0)) * a.Ks + k0;
    const bool u_vec = (a.Ks % 4 == 0) && ((reinterpret_cast<uintptr_t>(a.U) & 15u) == 0);  // k0 % 4 == 0
    for (int c = 0; c < RAp; c += 16) {
      float v[16];
#pragma unroll
      for (int j = 0; j < 16; j += 4) {
        const int k = c + j;  // own-range index; k0 + k < K only for real terms
        float4 f4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (own && k < p.RA && k0 + k < K) {
          if (u_vec) {
            f4 = __ldg(reinterpret_cast<const float4*>(urow + k));
          } else {
            f4.x = __ldg(urow + k);
            f4.y = k0 + k + 1 < K ? __ldg(urow + k + 1) : 0.f;
            f4.z = k0 + k + 2 < K ? __ldg(urow + k + 2) : 0.f;
            f4.w = k0 + k + 3 < K ? __ldg(urow + k + 3) : 0.f;
          }
        }
        v[j] = f4.x;
        v[j + 1] = (k0 + k + 1 < K) ? f4.y : 0.f;
        v[j + 2] = (k0 + k + 2 < K) ? f4.z : 0.f;
        v[j + 3] = (k0 + k + 3 < K) ? f4.w : 0.f;
      }
      tmem_st16(u_col + c, v);
    }
  }
  tmem_wait_st();

  // phase A row data: lane 8r <-> row r of this warp's four
  long long p_off = -1;
  float sig_r = 0.f;
  {
    const int r = lane >> 3;
    const int k = k0 + warp * 4 + r;
    if ((lane & 7) == 0 && warp < ngroups && k < K) {
      p_off = (long long)gate * a.Ks + k;
      sig_r = a.sigma[p_off];
    }
  }
  const long long p_stride = 4LL * a.Ks;
  // cell state: thread tid owns unit tid (in every CTA)
  const bool unit_ok = tid < H;
  float bias_r[4] = {0.f, 0.f, 0.f, 0.f};
  float c_reg = 0.f;
  if (unit_ok) {
#pragma unroll
    for (int g = 0; g < 4; ++g) bias_r[g] = a.bias[g * H + tid];
    if (a.c0 != nullptr) c_reg = a.c0[(long long)b * H + tid];
  }
  // P is written by the projection launched just before this kernel, or just
  // after it (its CTAs then each raise a flag once their part is stored)
  bool setup_ok = true;
  if (a.proj_flags == nullptr) griddep_wait();
  else if (warp == 0) setup_ok = wait_flags_epoch(a.proj_flags, a.proj_nflags, a.proj_epoch, limit_ns, err);
  if (!__syncthreads_and(setup_ok) && tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
  // P through L2 (it may have been written while this kernel ran)
  float p_cur = p_off >= 0 ? __ldcg(a.P + (long long)b * p_stride + p_off) : 0.f;
  const uint32_t bar0 = smem_u32(&bars[0]);
  const bool writer = tid >= ub0 && tid < ub0 + my_ub;
  const bool warp_units = warp * 32 < H;  // tensor-memory loads are warp-wide

  __syncthreads();
  cluster_sync_all();  // every CTA's barriers are armed before any copy reaches them

  const int t_end = *err == 0 ? a.T : 0;  // nothing to do after a failed set-up
  bool failed = false;
  for (int t = 0; t < t_end; ++t) {
    const int hb = t & 1;
    int fail = 0;
    const float p_next = (p_off >= 0 && t + 1 < a.T)
                             ? __ldcg(a.P + ((long long)(t + 1) * a.B + b) * p_stride + p_off)
                             : 0.f;
    // ---- phase A: tau' = sigma (V_h h_{t-1} + P_t), own rows, kept locally --
    if (warp < ngroups) {
      const float* hsrc = h_s + hb * 512 + 4 * lane;
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int e = 0; e < HQ; e += 2) {
        float va[16], vb[16];
        const float4 ha = *reinterpret_cast<const float4*>(hsrc + 128 * e);
        if (e + 1 < HQ) {
          tmem_ld16x2_sync(t_lane + t_col0 + 16 * e, t_lane + t_col0 + 16 * e + 16, va, vb);
        } else {
          tmem_ld16_sync(t_lane + t_col0 + 16 * e, va);
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          float s0 = acc[r];
          s0 = fmaf(va[4 * r + 0], ha.x, s0);
          s0 = fmaf(va[4 * r + 1], ha.y, s0);
          s0 = fmaf(va[4 * r + 2], ha.z, s0);
          s0 = fmaf(va[4 * r + 3], ha.w, s0);
          acc[r] = s0;
        }
        if (e + 1 < HQ) {
          const float4 hb4 = *reinterpret_cast<const float4*>(hsrc + 128 * e + 128);
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            float s0 = acc[r];
            s0 = fmaf(vb[4 * r + 0], hb4.x, s0);
            s0 = fmaf(vb[4 * r + 1], hb4.y, s0);
            s0 = fmaf(vb[4 * r + 2], hb4.z, s0);
            s0 = fmaf(vb[4 * r + 3], hb4.w, s0);
            acc[r] = s0;
          }
        }
      }
      lanes_sum_transposed<4>(acc, lane);          // lanes 8r .. 8r+7: row r's sum
      const float tpr = sig_r * (acc[0] + p_cur);  // valid on lane 8r
      const float t0 = __shfl_sync(0xffffffffu, tpr, 0);
      const float t1 = __shfl_sync(0xffffffffu, tpr, 8);
      const float t2 = __shfl_sync(0xffffffffu, tpr, 16);
      const float t3 = __shfl_sync(0xffffffffu, tpr, 24);
      if (lane == 0) *reinterpret_cast<float4*>(tau_s + warp * 4) = make_float4(t0, t1, t2, t3);
    }
    __syncthreads();

    // ---- phase B: this CTA's partial gate sums for every unit ----------------
    float* sb = send_s + hb * send_len;
    if (warp_units) {
      float y0 = 0.f, y1 = 0.f, y2 = 0.f, y3 = 0.f;  // four chains, summed in a fixed order
#pragma unroll 1
      for (int c = 0; c < RAp; c += 32) {
        float ua[16], ub[16];
        const bool two = c + 16 < RAp;
        if (two) tmem_ld16x2_sync(u_col + c, u_col + c + 16, ua, ub);
        else tmem_ld16_sync(u_col + c, ua);
#pragma unroll
        for (int j = 0; j < 16; j += 4) {
          const float4 tv = *reinterpret_cast<const float4*>(tau_s + c + j);
          y0 = fmaf(ua[j], tv.x, y0);
          y1 = fmaf(ua[j + 1], tv.y, y1);
          y2 = fmaf(ua[j + 2], tv.z, y2);
          y3 = fmaf(ua[j + 3], tv.w, y3);
        }
        if (two) {
#pragma unroll
          for (int j = 0; j < 16; j += 4) {
            const float4 tv = *reinterpret_cast<const float4*>(tau_s + c + 16 + j);
            y0 = fmaf(ub[j], tv.x, y0);
            y1 = fmaf(ub[j + 1], tv.y, y1);
            y2 = fmaf(ub[j + 2], tv.z, y2);
            y3 = fmaf(ub[j + 3], tv.w, y3);
          }
        }
      }
      if (unit_ok) sb[tid] = (y0 + y1) + (y2 + y3);
      // masked sums for the depths inside this range (the same products, cut at lim)
      for (int n = 0; n < J; ++n) {
        if (cut_slot[n] < 0 || cut_part[n] != part) continue;
        const int lim = cut_rem[n];
        float ym = 0.f;
#pragma unroll 1
        for (int c = 0; c < lim; c += 16) {
          float uv[16];
          tmem_ld16_sync(u_col + c, uv);
#pragma unroll
          for (int j = 0; j < 16; ++j) ym = fmaf(c + j < lim ? uv[j] : 0.f, tau_s[c + j], ym);
        }
        if (unit_ok) sb[(1 + cut_slot[n]) * H + tid] = ym;
      }
    }
    fence_proxy_async_shared();  // the generic-proxy writes above, before the copies read them
    __syncthreads();

    // ---- exchange: the partials to every CTA of the cluster ------------------
    const uint32_t bar = bar0 + 8u * hb;
    if (lane == 0 && warp < p.CS) {  // warp d sends to CTA d
      const uint32_t d = static_cast<uint32_t>(warp);
      const uint32_t rbar = mapa_shared(bar, d);
      bulk_copy_s2cluster(mapa_shared(smem_u32(rfull_s + hb * rfull_len + rank * H), d), smem_u32(sb),
                          4u * H, rbar);
      const int d0 = warp * p.UB, dn = min(p.UB, H - d0);  // destination's unit block
      for (uint32_t m = own_slots; m != 0u && dn > 0; m &= m - 1u) {
        const int slot = __ffs(m) - 1;
        bulk_copy_s2cluster(mapa_shared(smem_u32(rmask_s + hb * rmask_len + (slot * 4 + gate) * p.UB), d),
                            smem_u32(sb + (1 + slot) * H + d0), 4u * dn, rbar);
      }
    }
    if (!mbar_wait_bounded<true>(bar, (t >> 1) & 1, limit_ns, err)) fail = kErrWaitTimeoutA;
    else if (tid == 0) mbar_arrive_expect_tx(bar, bytes_in);  // re-arm for step t + 2

    // ---- cells (Sec. II) for every unit and depth --------------------------
    const float* rf = rfull_s + hb * rfull_len;
    const float* rm = rmask_s + hb * rmask_len;
    if (fail == 0 && unit_ok) {
      const long long tbo = ((long long)t * a.B + b) * H + tid;
      const float c_prev = c_reg;
      float y[4];
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (i < per_gate) s += rf[(g * per_gate + i) * H + tid];
        y[g] = s + bias_r[g];
      }
      float hh, cc;
      lstm_cell_f(y[0], y[1], y[2], y[3], c_prev, hh, cc);
      c_reg = cc;
      h_s[(hb ^ 1) * 512 + tid] = hh;
      if (writer) {
        a.out_h[tbo] = hh;
        for (int n = 0; n < J; ++n) {
          float yn[4];
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            float s = 0.f;
            const int np = min(cut_part[n], per_gate);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              if (i < np) s += rf[(g * per_gate + i) * H + tid];
            if (cut_slot[n] >= 0) s += rm[(cut_slot[n] * 4 + g) * p.UB + (tid - ub0)];
            yn[g] = s + bias_r[g];
          }
          float hn, cn;
          lstm_cell_f(yn[0], yn[1], yn[2], yn[3], c_prev, hn, cn);
          const long long o = (long long)n * a.T * a.B * H + tbo;
          if (a.ckpt_h) a.ckpt_h[o] = hn;
          if (a.ckpt_c) a.ckpt_c[o] = cn;
        }
      }
    }
    if (fail != 0) atomicCAS(a.err, 0, fail);
    if (__syncthreads_or(fail != 0)) {
      failed = true;
      break;
    }
    p_cur = p_next;
  }

  if (writer && a.c_last != nullptr) a.c_last[(long long)b * H + tid] = c_reg;
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tcols);
  }
  cluster_sync_all();  // every CTA has left its time loop: no copy is issued after this
  if (failed) {
    // after a wait ran out, copies issued just before the peers stopped may
    // still be in flight towards this CTA: let them land before it exits
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 50000ull) __nanosleep(1000);
  }
}
}  // namespace

bool plan_persistent_ag(int H, int K, const Checkpoints& ck, int want_cs, PersistentAgPlan* plan,
                        std::string* why) {
  if (H % 4 != 0 || H > kThreads) {
    *why = "hidden size not a multiple of 4 or above 512";
    return false;
  }
  if (K < 1 || K > 256) {
    *why = "K outside 1..256";
    return false;
  }
  const int cs_list[] = {4, 8, 16};
  for (int cs : cs_list) {
    if (want_cs != 0 && cs != want_cs) continue;
    AgPlan p{};
    p.CS = cs;
    p.Kp = (K + cs - 1) / cs * cs;          // each gate's terms split into CS/4 ranges of RA (a multiple of 4)
    p.RA = p.Kp / (cs / 4);
    if (p.RA > 4 * kWarps) continue;        // one group of four rows per warp
    p.UB = ((H + cs - 1) / cs + 3) & ~3;
    p.nmask = 0;
    for (int n = 0; n < ck.n; ++n)
      if (ck.k[n] < K && ck.k[n] % p.RA != 0) ++p.nmask;
    const int RAp = (p.RA + 15) & ~15;
    const int hq = H <= 128 ? 1 : H <= 256 ? 2 : 4;
    const int need = 64 * hq + 4 * RAp;  // V_h, then U
    p.tcols = 32;
    while (p.tcols < need) p.tcols *= 2;
    if (p.tcols > 512) continue;
    size_t smem = kHeaderBytes + 4ull * ag_layout(p, H).total;
    if (smem > 227u * 1024u) continue;
    // at least half of an SM's shared memory, so that no other CTA of this
    // kernel shares the SM (and its tensor memory) with this one
    if (smem < kMinSmemBytes) smem = kMinSmemBytes;
    plan->CS = p.CS;
    plan->RA = p.RA;
    plan->Kp = p.Kp;
    plan->UB = p.UB;
    plan->nmask = p.nmask;
    plan->tcols = p.tcols;
    plan->hq = hq;
    plan->smem = smem;
    return true;  // the smallest cluster that fits moves the fewest partials
  }
  *why = "shape does not fit the one-exchange persistent kernel (K, checkpoints or on-chip memory)";
  return false;
}

namespace {

template <int HQ>
cudaError_t launch_ag_t(const AgPlan& p, size_t smem, const PersistentArgs& a, cudaStream_t s) {
  auto kern = persistent_ag_kernel<HQ>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.CS * a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // may start while the projection before it finishes (set-up overlaps it);
  // with the projection launched after it, an ordinary launch
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = a.proj_flags == nullptr ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  static thread_local bool attrs_set = false;
  static thread_local unsigned long long checked[16] = {};
  if (!attrs_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    attrs_set = true;
  }
  const unsigned long long key = (static_cast<unsigned long long>(smem) << 8) | static_cast<unsigned>(p.CS);
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
  return cudaLaunchKernelEx(&cfg, kern, a, p);
}

}  // namespace

cudaError_t launch_persistent_ag(const PersistentAgPlan& plan, const PersistentArgs& a, cudaStream_t s) {
  AgPlan p{};
  p.CS = plan.CS;
  p.RA = plan.RA;
  p.Kp = plan.Kp;
  p.UB = plan.UB;
  p.nmask = plan.nmask;
  p.tcols = plan.tcols;
  switch (plan.hq) {
    case 1: return launch_ag_t<1>(p, plan.smem, a, s);
    case 2: return launch_ag_t<2>(p, plan.smem, a, s);
    case 4: return launch_ag_t<4>(p, plan.smem, a, s);
    default: return cudaErrorInvalidValue;
  }
}

// Work of one CTA of the one-exchange kernel per timestep, H units x RA
// terms, above which the per-unit-block kernel is faster: measured at
// T = 20 on H = 64 .. 512 and K = 16 .. 256, the one-exchange kernel wins
// by 10-40% up to H = 256 and at H = 512 with K = 16, and loses by 15-25%
// at H = 512 with 64 or 256 terms per CTA, where every CTA receives and
// sums 16 partial vectors of 512 floats per step.
constexpr int kAgAutoMaxWork = 16384;

bool choose_persistent(int H, int K, int T, const Checkpoints& ck, int want_cs, int sm_count, int variant,
                       PersistentChoice* c, std::string* why) {
  std::string why_ag;
  if (variant != 1 && plan_persistent_ag(H, K, ck, want_cs, &c->ag, &why_ag) &&
      (variant == 2 || H * c->ag.RA <= kAgAutoMaxWork)) {
    c->variant = 2;
    c->CS = c->ag.CS;
    return true;
  }
  if (variant == 2) {
    *why = why_ag;
    return false;
  }
  if (!plan_persistent(H, K, T, ck, want_cs, sm_count, &c->ub, why)) return false;
  c->variant = 1;
  c->CS = c->ub.CS;
  return true;
}

cudaError_t launch_persistent_choice(const PersistentChoice& c, const PersistentArgs& a, cudaStream_t s) {
  return c.variant == 2 ? launch_persistent_ag(c.ag, a, s) : launch_persistent(c.ub, a, s);
}

}  // namespace lstm_approx_impl
