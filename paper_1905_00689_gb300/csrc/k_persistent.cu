// Persistent small-batch kernel: one cluster launch covers all T timesteps.
//
// The work of one timestep (Eq. 1 for the four gates, then the cell update
// of Sec. II) has two all-to-all dependencies: every refinement coefficient
// tau_{g,k} = prune(v_{g,k})^T [x_t; h_{t-1}] needs all of h_{t-1}, and every
// gate output y_g[j] = sum_k sigma_{g,k} u_{g,k}[j] tau_{g,k} needs all tau.
// One cluster of CS CTAs (CS <= 16) serves one stream:
//
//   phase A  CTA c owns RA coefficient rows (gate-major row g*Kp + k).  Its
//            rows of the pruned V_h (masked-dense, fp32) stay in shared memory
//            for the whole launch; the x part was hoisted into P = V_x X for all
//            t by an earlier launch.  tau' = sigma * (V_h h + P_t) for its rows
//            is pushed into every CTA's tau buffer with st.async, which
//            completes the transaction count of the receiver's mbarrier.
//   phase B  CTA c owns UB hidden units.  Its slice of U (4 gates x K terms x
//            UB units) lives in registers for the whole launch: warp w holds
//            the terms of segment w, lane l the units l, l+32.  Partial sums are
//            reduced across warps in segment order, which yields the prefix
//            sums at the requested depths k_j for free (progressive outputs);
//            the cell update runs on the owning thread, which keeps c_t in a
//            register, and h_t is pushed to every CTA like tau.
//
// Both exchanges are double-buffered by timestep parity.  Every wait is
// bounded in wall time; a wait that runs out writes the device status word,
// all CTAs leave the time loop, and the cluster meets at one final barrier.
#include "internal.h"
#include "ptx.cuh"

#include <algorithm>
#include <cstdio>

namespace lstm_approx_impl {
namespace {

using namespace lstm_approx_dev;

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTauSlack = 32;

struct DevPlan {
  int CS, RA, UB, Kp, nseg, pxc;
  int seg_start[kWarps + 1];
  int ck_seg[kMaxCheckpoints];
};

struct SmemLayout {
  uint32_t vh, sig, px, tau, h, part, y, hsend, total;  // float offsets after the barriers
};

__host__ __device__ inline SmemLayout smem_layout(const DevPlan& p, int H, int J) {
  SmemLayout L;
  uint32_t o = 0;
  L.vh = o;    o += p.RA * H;
  L.sig = o;   o += p.RA;
  L.px = o;    o += p.pxc * p.RA;
  o = (o + 3) & ~3u;
  L.tau = o;   o += 2 * (p.CS * p.RA + kTauSlack);
  L.h = o;     o += 2 * p.CS * p.UB;
  L.part = o;  o += kWarps * 4 * p.UB;
  L.y = o;     o += (J + 1) * 4 * p.UB;
  L.hsend = o; o += p.UB;
  L.total = o;
  return L;
}
constexpr uint32_t kBarrierBytes = 64;

template <int UPL, int KPW>
__global__ void __launch_bounds__(kThreads, 1) persistent_kernel(PersistentArgs a, DevPlan p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw);  // [0,1] tau, [2,3] h
  float* sm = reinterpret_cast<float*>(smem_raw + kBarrierBytes);
  const SmemLayout S = smem_layout(p, a.H, a.ck.n);
  float* vh_s = sm + S.vh;
  float* sig_s = sm + S.sig;
  float* px_s = sm + S.px;
  float* tau_s = sm + S.tau;
  float* h_s = sm + S.h;
  float* part_s = sm + S.part;
  float* y_s = sm + S.y;
  float* hsend_s = sm + S.hsend;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // plan tables indexed at run time live in shared memory (not in a local copy of the parameters)
  __shared__ int seg_tab[kWarps + 1];
  __shared__ int ck_tab[kMaxCheckpoints];
  if (tid == 0) {
#pragma unroll
    for (int i = 0; i <= kWarps; ++i) seg_tab[i] = p.seg_start[i];
#pragma unroll
    for (int i = 0; i < kMaxCheckpoints; ++i) ck_tab[i] = p.ck_seg[i];
  }
  __syncthreads();
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / p.CS;  // one cluster per stream
  const int H = a.H, K = a.K, J = a.ck.n;
  const int tau_len = p.CS * p.RA + kTauSlack;
  const int h_len = p.CS * p.UB;
  const uint32_t bytes_tau = p.CS * p.RA * 4u;
  const uint32_t bytes_h = p.CS * p.UB * 4u;
  const uint64_t limit_ns = static_cast<uint64_t>(a.wait_limit_ns);
  const volatile int* err = a.err;

  // ---- set-up: barriers, resident factors, initial state -----------------
  if (tid == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&bars[i]), 1);
    mbar_arrive_expect_tx(smem_u32(&bars[0]), bytes_tau + (a.test_stall ? 16u : 0u));
    mbar_arrive_expect_tx(smem_u32(&bars[1]), bytes_tau);
    mbar_arrive_expect_tx(smem_u32(&bars[2]), bytes_h);
    mbar_arrive_expect_tx(smem_u32(&bars[3]), bytes_h);
    fence_mbarrier_init_cluster();
  }
  for (int i = tid; i < 2 * tau_len; i += kThreads) tau_s[i] = 0.f;
  for (int i = tid; i < h_len; i += kThreads)
    h_s[i] = (a.h0 != nullptr && i < H) ? a.h0[(long long)b * H + i] : 0.f;

  // coefficient rows owned by this CTA: run row gr = rank*RA + lr = g*Kp + k
  const int H4 = H >> 2;
  for (int lr = warp; lr < p.RA; lr += kWarps) {
    const int gr = rank * p.RA + lr;
    const int g = gr / p.Kp, k = gr % p.Kp;
    const bool valid = g < 4 && k < K;
    const long long srow = (long long)g * a.Ks + k;
    const float4* src = reinterpret_cast<const float4*>(a.Vh + srow * a.ldh);
    float4* dst = reinterpret_cast<float4*>(vh_s + lr * H);
    for (int c4 = lane; c4 < H4; c4 += 32) dst[c4] = valid ? __ldg(src + c4) : make_float4(0.f, 0.f, 0.f, 0.f);
    if (lane == 0) sig_s[lr] = valid ? a.sigma[srow] : 0.f;
  }

  // U slice in registers: warp w <-> terms [seg_start[w], seg_start[w+1]),
  // lane <-> units u = lane + 32 i of this CTA
  float ureg[UPL][4][KPW];
  const int s0 = warp < p.nseg ? seg_tab[warp] : 0;
  const int slen = warp < p.nseg ? seg_tab[warp + 1] - s0 : 0;
#pragma unroll
  for (int i = 0; i < UPL; ++i) {
    const int u = lane + 32 * i;
    const int j = rank * p.UB + u;
    const bool ok = u < p.UB && j < H;
#pragma unroll
    for (int g = 0; g < 4; ++g)
#pragma unroll
      for (int kk = 0; kk < KPW; ++kk)
        ureg[i][g][kk] = (ok && kk < slen) ? __ldg(a.U + ((long long)g * a.Ks + s0 + kk) * H + j) : 0.f;
  }

  // cell-update threads: tid < UB owns unit rank*UB + tid
  const int my_j = rank * p.UB + tid;
  const bool cell_thread = tid < p.UB && my_j < H;
  float bias_r[4] = {0.f, 0.f, 0.f, 0.f};
  float c_reg = 0.f;
  if (cell_thread) {
#pragma unroll
    for (int g = 0; g < 4; ++g) bias_r[g] = a.bias[g * H + my_j];
    c_reg = a.c0 != nullptr ? a.c0[(long long)b * H + my_j] : 0.f;
  }

  __syncthreads();
  cluster_sync_all();  // every CTA's barriers are initialised before any st.async

  const uint32_t bar_tau0 = smem_u32(&bars[0]);
  const uint32_t bar_h0 = smem_u32(&bars[2]);
  const uint32_t tau_base = smem_u32(tau_s);
  const uint32_t h_base = smem_u32(h_s);
  const int vec_tau = (s0 & 3) == 0;
  int pxbase = 0;

  for (int t = 0; t < a.T; ++t) {
    const int hb = t & 1;
    // ---- wait for h_{t-1} (t = 0 uses h0, loaded locally) ----------------
    if (t > 0) {
      const bool ok = mbar_wait_bounded<true>(bar_h0 + 8u * hb, ((t - 1) >> 1) & 1, limit_ns, err);
      if (!__syncthreads_and(ok)) {
        if (tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutB);
        break;
      }
      if (tid == 0) mbar_arrive_expect_tx(bar_h0 + 8u * hb, bytes_h);
    }
    // ---- stage the hoisted input projection for the next timesteps ------
    if (t == pxbase + p.pxc || t == 0) {
      if (t != 0) pxbase = t;
      __syncthreads();
      const int nt = min(p.pxc, a.T - pxbase);
      for (int i = tid; i < nt * p.RA; i += kThreads) {
        const int tt = i / p.RA, lr = i % p.RA;
        const int gr = rank * p.RA + lr;
        const int g = gr / p.Kp, k = gr % p.Kp;
        float v = 0.f;
        if (g < 4 && k < K)
          v = a.P[((long long)(pxbase + tt) * a.B + b) * (4LL * a.Ks) + (long long)g * a.Ks + k];
        px_s[tt * p.RA + lr] = v;
      }
      __syncthreads();
    }

    // ---- phase A: tau' = sigma * (V_h h_{t-1} + P_t) for the owned rows ---
    const float4* h4 = reinterpret_cast<const float4*>(h_s + hb * h_len);
    const float* pxt = px_s + (t - pxbase) * p.RA;
    for (int grp = warp; grp < (p.RA >> 2); grp += kWarps) {
      const int lr0 = grp * 4;
      float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
      const float4* v0 = reinterpret_cast<const float4*>(vh_s + (lr0 + 0) * H);
      const float4* v1 = reinterpret_cast<const float4*>(vh_s + (lr0 + 1) * H);
      const float4* v2 = reinterpret_cast<const float4*>(vh_s + (lr0 + 2) * H);
      const float4* v3 = reinterpret_cast<const float4*>(vh_s + (lr0 + 3) * H);
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
      acc0 = warp_sum(acc0);
      acc1 = warp_sum(acc1);
      acc2 = warp_sum(acc2);
      acc3 = warp_sum(acc3);
      if (lane < p.CS) {
        const float t0 = sig_s[lr0 + 0] * (acc0 + pxt[lr0 + 0]);
        const float t1 = sig_s[lr0 + 1] * (acc1 + pxt[lr0 + 1]);
        const float t2 = sig_s[lr0 + 2] * (acc2 + pxt[lr0 + 2]);
        const float t3 = sig_s[lr0 + 3] * (acc3 + pxt[lr0 + 3]);
        const uint32_t off = 4u * (hb * tau_len + rank * p.RA + lr0);
        st_async_v4(mapa_shared(tau_base + off, lane), t0, t1, t2, t3, mapa_shared(bar_tau0 + 8u * hb, lane));
      }
    }

    // ---- wait for every CTA's tau' ----------------------------------------
    {
      const bool ok = mbar_wait_bounded<true>(bar_tau0 + 8u * hb, (t >> 1) & 1, limit_ns, err);
      if (!__syncthreads_and(ok)) {
        if (tid == 0) atomicCAS(a.err, 0, kErrWaitTimeoutA);
        break;
      }
      if (tid == 0) mbar_arrive_expect_tx(bar_tau0 + 8u * hb, bytes_tau);
    }

    // ---- phase B: partial gate sums over this warp's terms ----------------
    const float* tau = tau_s + hb * tau_len;
    float acc[UPL][4];
#pragma unroll
    for (int i = 0; i < UPL; ++i)
#pragma unroll
      for (int g = 0; g < 4; ++g) acc[i][g] = 0.f;
    if (vec_tau && (KPW % 4) == 0) {
#pragma unroll
      for (int q = 0; q < KPW / 4; ++q) {
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          const float4 tv = *reinterpret_cast<const float4*>(tau + g * p.Kp + s0 + 4 * q);
#pragma unroll
          for (int i = 0; i < UPL; ++i) {
            acc[i][g] = fmaf(ureg[i][g][4 * q + 0], tv.x, acc[i][g]);
            acc[i][g] = fmaf(ureg[i][g][4 * q + 1], tv.y, acc[i][g]);
            acc[i][g] = fmaf(ureg[i][g][4 * q + 2], tv.z, acc[i][g]);
            acc[i][g] = fmaf(ureg[i][g][4 * q + 3], tv.w, acc[i][g]);
          }
        }
      }
    } else {
#pragma unroll
      for (int kk = 0; kk < KPW; ++kk) {
        if (kk < slen) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            const float tv = tau[g * p.Kp + s0 + kk];
#pragma unroll
            for (int i = 0; i < UPL; ++i) acc[i][g] = fmaf(ureg[i][g][kk], tv, acc[i][g]);
          }
        }
      }
    }
#pragma unroll
    for (int i = 0; i < UPL; ++i) {
      const int u = lane + 32 * i;
      if (u < p.UB) {
#pragma unroll
        for (int g = 0; g < 4; ++g) part_s[(warp * 4 + g) * p.UB + u] = acc[i][g];
      }
    }
    __syncthreads();

    // ---- reduce across warps in term order; prefix sums at the depths ----
    if (tid < 4 * p.UB) {
      const int g = tid / p.UB, u = tid % p.UB;
      float s = 0.f;
      int jj = 0;
      for (int w = 0; w < p.nseg; ++w) {
        s += part_s[(w * 4 + g) * p.UB + u];
        while (jj < J && ck_tab[jj] == w + 1) {
          y_s[(jj * 4 + g) * p.UB + u] = s;
          ++jj;
        }
      }
      y_s[(J * 4 + g) * p.UB + u] = s;
    }
    __syncthreads();

    // ---- cell update on the owning threads --------------------------------
    if (tid < p.UB) {
      float hn = 0.f;
      if (cell_thread) {
        const long long tb = ((long long)t * a.B + b) * H + my_j;
        for (int jj = 0; jj < J; ++jj) {
          float hh, cc;
          lstm_cell_f(y_s[(jj * 4 + 0) * p.UB + tid] + bias_r[0], y_s[(jj * 4 + 1) * p.UB + tid] + bias_r[1],
                      y_s[(jj * 4 + 2) * p.UB + tid] + bias_r[2], y_s[(jj * 4 + 3) * p.UB + tid] + bias_r[3],
                      c_reg, hh, cc);
          const long long o = (long long)jj * a.T * a.B * H + tb;
          if (a.ckpt_h) a.ckpt_h[o] = hh;
          if (a.ckpt_c) a.ckpt_c[o] = cc;
        }
        float cn;
        lstm_cell_f(y_s[(J * 4 + 0) * p.UB + tid] + bias_r[0], y_s[(J * 4 + 1) * p.UB + tid] + bias_r[1],
                    y_s[(J * 4 + 2) * p.UB + tid] + bias_r[2], y_s[(J * 4 + 3) * p.UB + tid] + bias_r[3], c_reg,
                    hn, cn);
        c_reg = cn;
        a.out_h[tb] = hn;
      }
      hsend_s[tid] = hn;
    }
    __syncthreads();

    // ---- push h_t to every CTA of the cluster -----------------------------
    if (t + 1 < a.T && warp == 0) {
      const int nb = (t + 1) & 1;
      const int ngroups = p.UB >> 2;
      for (int m = lane; m < ngroups * p.CS; m += 32) {
        const int q = m / p.CS, d = m % p.CS;
        const uint32_t off = 4u * (nb * h_len + rank * p.UB + 4 * q);
        st_async_v4(mapa_shared(h_base + off, d), hsend_s[4 * q + 0], hsend_s[4 * q + 1], hsend_s[4 * q + 2],
                    hsend_s[4 * q + 3], mapa_shared(bar_h0 + 8u * nb, d));
      }
    }
  }

  if (cell_thread && a.c_last != nullptr) a.c_last[(long long)b * H + my_j] = c_reg;
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while others may still address its shared memory
}

template <int UPL, int KPW>
cudaError_t launch_t(const DevPlan& dp, size_t smem, const PersistentArgs& a, cudaStream_t s) {
  auto kern = persistent_kernel<UPL, KPW>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  if (dp.CS > 8) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
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
  int nclusters = 0;
  e = cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg);
  if (e != cudaSuccess) return e;
  if (nclusters < 1) return cudaErrorNotPermitted;
  return cudaLaunchKernelEx(&cfg, kern, a, dp);
}

}  // namespace

bool plan_persistent(int H, int K, int T, const Checkpoints& ck, int want_cs, int sm_count, PersistentPlan* plan,
                     std::string* why) {
  (void)sm_count;
  if (H % 4 != 0) {
    *why = "hidden size not a multiple of 4";
    return false;
  }
  const int Kp = (K + 3) & ~3;
  const int rows = 4 * Kp;
  static const int kpws[] = {1, 2, 4, 8, 16};
  const int cs_list[] = {1, 2, 4, 8, 16};
  PersistentPlan best;
  bool found = false;
  for (int cs : cs_list) {
    if (want_cs != 0 && cs != want_cs) continue;
    PersistentPlan p;
    p.CS = cs;
    p.RA = (((rows + cs - 1) / cs) + 3) & ~3;
    p.UB = (((H + cs - 1) / cs) + 3) & ~3;
    if (p.UB > 64) continue;
    p.upl = p.UB <= 32 ? 1 : 2;
    // split the terms into warp segments, cut at every requested depth
    bool seg_ok = false;
    for (int kpw : kpws) {
      if (p.upl == 2 && kpw > 8) continue;
      int n = 0, a0 = 0, jj = 0;
      int starts[64];
      bool over = false;
      while (a0 < K) {
        int stop = K;
        while (jj < ck.n && ck.k[jj] <= a0) ++jj;
        if (jj < ck.n) stop = std::min(stop, ck.k[jj]);
        const int e = std::min(stop, a0 + kpw);
        if (n >= kWarps) {
          over = true;
          break;
        }
        starts[n++] = a0;
        a0 = e;
      }
      if (over) continue;
      p.kpw = kpw;
      p.nseg = n;
      for (int i = 0; i < n; ++i) p.seg_start[i] = starts[i];
      p.seg_start[n] = K;
      for (int i = n + 1; i <= kWarps; ++i) p.seg_start[i] = K;
      for (int j = 0; j < ck.n; ++j) {
        p.ck_seg[j] = -1;
        for (int i = 0; i < n; ++i)
          if (p.seg_start[i + 1] == ck.k[j]) p.ck_seg[j] = i + 1;
      }
      seg_ok = true;
      break;
    }
    if (!seg_ok) continue;
    p.pxc = std::min(T, 32);
    DevPlan dp{};
    dp.CS = p.CS; dp.RA = p.RA; dp.UB = p.UB; dp.Kp = Kp; dp.nseg = p.nseg; dp.pxc = p.pxc;
    const SmemLayout L = smem_layout(dp, H, ck.n);
    p.smem = kBarrierBytes + 4ull * L.total;
    if (p.smem > 227u * 1024u) continue;
    best = p;
    found = true;
    if (want_cs != 0) break;
    // automatic choice: the first (smallest) cluster whose V_h slice is small
    if ((size_t)p.RA * H * 4 <= 32u * 1024u) break;
  }
  if (!found) {
    *why = "shape does not fit the persistent kernel (K > 256, hidden > 1024 or shared memory)";
    return false;
  }
  *plan = best;
  return true;
}

cudaError_t launch_persistent(const PersistentPlan& plan, const PersistentArgs& a, cudaStream_t s) {
  DevPlan dp{};
  dp.CS = plan.CS; dp.RA = plan.RA; dp.UB = plan.UB; dp.Kp = (a.K + 3) & ~3;
  dp.nseg = plan.nseg; dp.pxc = plan.pxc;
  for (int i = 0; i <= kWarps; ++i) dp.seg_start[i] = plan.seg_start[i];
  for (int i = 0; i < kMaxCheckpoints; ++i) dp.ck_seg[i] = plan.ck_seg[i];
  const int u = plan.upl, k = plan.kpw;
#define LA_CASE(U_, K_) \
  if (u == U_ && k == K_) return launch_t<U_, K_>(dp, plan.smem, a, s);
  LA_CASE(1, 1) LA_CASE(1, 2) LA_CASE(1, 4) LA_CASE(1, 8) LA_CASE(1, 16)
  LA_CASE(2, 1) LA_CASE(2, 2) LA_CASE(2, 4) LA_CASE(2, 8)
#undef LA_CASE
  return cudaErrorInvalidValue;
}

}  // namespace lstm_approx_impl
