// C-ABI of the approximate-LSTM library: handle, factor packing, dispatch.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

using namespace lstm_approx_impl;

namespace {

int fail(lstm_approx_t* h, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (h) h->last_error = buf;
  return code;
}

int cuda_fail(lstm_approx_t* h, cudaError_t e, const char* what) {
  return fail(h, e == cudaErrorMemoryAllocation ? LSTM_APPROX_ENOMEM : LSTM_APPROX_ECUDA, "%s: %s", what,
              cudaGetErrorString(e));
}

#define LA_CUDA(h, call, what)                      \
  do {                                              \
    cudaError_t e_ = (call);                        \
    if (e_ != cudaSuccess) return cuda_fail(h, e_, what); \
  } while (0)

inline int round_up(int v, int m) { return (v + m - 1) / m * m; }

// fp64 -> fp32 -> bf16, both steps round-to-nearest-even; infinities keep
// their sign, every NaN becomes the quiet NaN 0x7FC0.
inline uint16_t to_bf16_bits(double x) {
  const float f = static_cast<float>(x);
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0x7FC0u;                            // nan
  if ((u & 0x7FFFFFFFu) == 0x7F800000u) return static_cast<uint16_t>(u >> 16);  // inf
  const uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return static_cast<uint16_t>(u >> 16);
}

size_t elem_size(int dtype) { return dtype == LSTM_APPROX_BF16 ? 2 : 4; }

int dmalloc(lstm_approx_t* h, void** p, size_t bytes, const char* what) {
  *p = nullptr;
  if (bytes == 0) return LSTM_APPROX_OK;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    *p = nullptr;
    return cuda_fail(h, e, what);
  }
  e = cudaMemset(*p, 0, bytes);
  if (e != cudaSuccess) return cuda_fail(h, e, what);
  h->device_bytes += static_cast<long long>(bytes);
  return LSTM_APPROX_OK;
}

void dfree(lstm_approx_t* h, void* p, size_t bytes) {
  if (p) {
    cudaFree(p);
    h->device_bytes -= static_cast<long long>(bytes);
  }
}

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

size_t layer_bytes_vx(const lstm_approx_t* h, const LayerStore& s) {
  return 4ull * h->Ks * s.ldx * elem_size(h->dtype);
}
size_t layer_bytes_vh(const lstm_approx_t* h) { return 4ull * h->Ks * h->ldh * elem_size(h->dtype); }
size_t layer_bytes_u(const lstm_approx_t* h) { return 4ull * h->Ks * h->H * elem_size(h->dtype); }

// bf16 pair planes (hi, lo) of the tensor path's activations
size_t xbf16_bytes(const lstm_approx_t* h, size_t TB) { return 2 * TB * (size_t)h->layers[0].ldx * 2; }
size_t seqbf16_bytes(const lstm_approx_t* h, size_t TB) { return 2 * TB * (size_t)h->ldh * 2; }

void free_scratch(lstm_approx_t* h) {
  dfree(h, h->Px, h->cap_TB * 4ull * h->Ks * sizeof(float));
  dfree(h, h->seq, h->cap_TB * (size_t)h->H * sizeof(float));
  if (h->x_bf16) dfree(h, h->x_bf16, xbf16_bytes(h, h->cap_TB));
  if (h->seq_bf16) dfree(h, h->seq_bf16, seqbf16_bytes(h, h->cap_TB));
  h->Px = nullptr;
  h->seq = nullptr;
  h->x_bf16 = nullptr;
  h->seq_bf16 = nullptr;
  h->cap_TB = 0;
}

int ensure_scratch(lstm_approx_t* h, size_t TB) {
  if (TB <= h->cap_TB) return LSTM_APPROX_OK;
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "synchronising before growing scratch");
  free_scratch(h);
  int rc = dmalloc(h, reinterpret_cast<void**>(&h->Px), TB * 4ull * h->Ks * sizeof(float), "scratch P");
  if (rc) return rc;
  if (h->L > 1) {
    rc = dmalloc(h, reinterpret_cast<void**>(&h->seq), TB * (size_t)h->H * sizeof(float), "scratch seq");
    if (rc) return rc;
  }
  if (h->dtype == LSTM_APPROX_BF16) {
    rc = dmalloc(h, &h->x_bf16, xbf16_bytes(h, TB), "scratch x bf16");
    if (rc) return rc;
    if (h->L > 1) {
      rc = dmalloc(h, &h->seq_bf16, seqbf16_bytes(h, TB), "scratch seq bf16");
      if (rc) return rc;
    }
  }
  h->cap_TB = TB;
  return LSTM_APPROX_OK;
}

int validate_run(lstm_approx_t* h, const float* x, int T, int B, int K, float* out_h, const int* checkpoints,
                 int J, Checkpoints* ck) {
  if (!x || !out_h) return fail(h, LSTM_APPROX_EINVAL, "x and out_h must not be NULL");
  if (T < 1) return fail(h, LSTM_APPROX_EINVAL, "T=%d must be >= 1", T);
  if (B < 1 || B > h->max_batch) return fail(h, LSTM_APPROX_EINVAL, "B=%d outside [1, %d]", B, h->max_batch);
  if (K < 1 || K > h->Kmax) return fail(h, LSTM_APPROX_EINVAL, "K=%d outside [1, %d]", K, h->Kmax);
  if (J < 0 || J > kMaxCheckpoints) return fail(h, LSTM_APPROX_EINVAL, "J=%d outside [0, %d]", J, kMaxCheckpoints);
  if (J > 0 && !checkpoints) return fail(h, LSTM_APPROX_EINVAL, "checkpoints is NULL with J=%d", J);
  ck->n = J;
  for (int j = 0; j < J; ++j) {
    const int k = checkpoints[j];
    if (k < 1 || k > K) return fail(h, LSTM_APPROX_EINVAL, "checkpoint %d = %d outside [1, K=%d]", j, k, K);
    if (j > 0 && k <= checkpoints[j - 1])
      return fail(h, LSTM_APPROX_EINVAL, "checkpoints must be strictly increasing");
    ck->k[j] = k;
  }
  for (int j = J; j < kMaxCheckpoints; ++j) ck->k[j] = 0;
  for (int l = 0; l < h->L; ++l)
    for (int g = 0; g < 4; ++g)
      if (h->layers[l].Kset[g] < K)
        return fail(h, LSTM_APPROX_ESTATE, "layer %d gate %d has %d terms set, run asks K=%d", l, g,
                    h->layers[l].Kset[g], K);
  return LSTM_APPROX_OK;
}

struct PhaseTimer {
  lstm_approx_t* h;
  int phase;
  cudaEvent_t e1 = nullptr;
  PhaseTimer(lstm_approx_t* hh, int ph) : h(hh), phase(ph) {
    if (!h->timing.on) return;
    cudaEvent_t e0;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    cudaEventRecord(e0, h->stream);
    h->timing.ev.push_back(e0);
    h->timing.ev.push_back(e1);
    h->timing.phase.push_back(phase);
  }
  ~PhaseTimer() {
    if (e1) cudaEventRecord(e1, h->stream);
  }
};

void clear_timing(lstm_approx_t* h) {
  for (cudaEvent_t e : h->timing.ev) cudaEventDestroy(e);
  h->timing.ev.clear();
  h->timing.phase.clear();
}

// The compressed x projection pays when v keeps at most 1/8 of the x columns
// (fp32 factors, few columns).
bool sparse_x_projection(const lstm_approx_t* h, const LayerStore& s, int K, int N) {
  if (h->dtype != LSTM_APPROX_FP32 || N > 32 || h->opt_xproj == 1) return false;
  long long kept = 0;
  for (int g = 0; g < 4; ++g) {
    if (s.xoff[g] == nullptr || (int)s.xoff_h[g].size() <= K) return false;
    kept += s.xoff_h[g][K];
  }
  return h->opt_xproj == 2 || kept * 8 <= 4LL * K * s.D;
}

// The tensor path takes bf16 factors at any depths (a depth off the MMA's
// 16-term slices adds its last terms on the CUDA cores).
bool tensor_path_fits(int dtype) { return dtype == LSTM_APPROX_BF16; }

// Recurrence path of one layer.  Automatic: bf16 factors take the
// tensor-core path; fp32 factors take a persistent
// launch whenever a plan fits, at any batch (one cluster per stream;
// clusters beyond one wave run in the next); everything else takes the
// CUDA-core kernels.  A forced path that cannot take the shape returns 0
// with the reason in *why.  *plan is filled for the persistent path.
int select_path(int dtype, int H, int K, int T, const Checkpoints& ck, int force_path, int want_cs, int sm_count,
                int variant, PersistentChoice* plan, std::string* why) {
  const bool bf16 = dtype == LSTM_APPROX_BF16;
  const bool tensor_ok = tensor_path_fits(dtype);
  if (force_path == 0) {
    if (tensor_ok) return LSTM_APPROX_PATH_TENSOR;
    if (!bf16 && choose_persistent(H, K, T, ck, want_cs, sm_count, variant, plan, why))
      return LSTM_APPROX_PATH_PERSISTENT;
    return LSTM_APPROX_PATH_SIMT;
  }
  if (force_path == LSTM_APPROX_PATH_PERSISTENT) {
    if (bf16) {
      *why = "the persistent path runs fp32 factors only";
      return 0;
    }
    std::string r;
    if (!choose_persistent(H, K, T, ck, want_cs, sm_count, variant, plan, &r)) {
      *why = "persistent path unavailable: " + r;
      return 0;
    }
  } else if (force_path == LSTM_APPROX_PATH_TENSOR && !tensor_ok) {
    *why = "tensor path needs bf16 factors";
    return 0;
  }
  return force_path;
}

struct TensorTiles {
  int bnh = 0, nt = 0, ks = 1, nkb_per = 0;
  int sk = 1, nkb_per_h = 0;  // the tau' GEMM's splits of its reduction axis (H) and 64-chunks per split
  bool raw = false;  // raw gate sums and a reduce kernel (term split, or depths off the 16-term slices)
};

// Tiles of the tensor-core path for one layer: streams per tile of the tau'
// GEMM (bnh) and of the gate GEMM (nt), and the gate GEMM's term-axis
// splits (ks, of nkb_per 64-term chunks each; small grids split the terms
// over more CTAs).
// Rows per gate of the packed factor tile (0: one 128-row tile per gate).
int tensor_rows_per_gate(int K) { return K <= 8 ? 8 : K <= 16 ? 16 : K <= 32 ? 32 : 0; }

TensorTiles tensor_tiles(int H, int B, int K, const Checkpoints& ck) {
  TensorTiles t;
  // packed gates: one row tile, so narrower stream tiles keep more SMs busy
  t.bnh = tensor_rows_per_gate(K) > 0 ? 32 : tc_rows_tile_n(B, 4 * ((K + 127) / 128));
  if (tensor_rows_per_gate(K) == 0) {
    // few tiles of 64 streams over a long reduction axis (H >= 1024): split
    // it over a cluster of 4 CTAs instead of narrowing the stream tiles, so
    // that each CTA streams a quarter of the factor rows.  Measured (whole
    // recurrence): the two-layer D=4096 H=2048 B=64 K=1024 workload 1207 ->
    // 1165 us; splitting in two at D=1024 H=512 B=256 K=512 (383 -> 460 us)
    // and at D=2048 H=1024 B=1024 K=128 (1209 -> 1316 us) cost more in
    // cluster barriers and pushes than the shorter streams save.
    const int row_tiles = 4 * ((K + 127) / 128), nkbh = (H + 63) / 64;
    const long long tiles64 = (long long)row_tiles * ((B + 63) / 64);
    int sk = tiles64 * 4 <= 148 && nkbh >= 16 ? 4 : 1;
    if (sk > 1) {
      t.bnh = 64;
      t.nkb_per_h = (nkbh + sk - 1) / sk;
      t.sk = (nkbh + t.nkb_per_h - 1) / t.nkb_per_h;  // no empty split
    }
  }
  t.nt = tc_gates_tile_n(H, B);
  const int gate_tiles = ((H + 127) / 128) * ((B + t.nt - 1) / t.nt);
  t.ks = tc_gates_splits(gate_tiles, (K + 63) / 64, &t.nkb_per);
  t.raw = t.ks > 1;
  for (int j = 0; j < ck.n; ++j) t.raw = t.raw || ck.k[j] % 16 != 0;
  return t;
}

// The compressed h part of layer l's v on the device, for the compressed
// tau' layout: CSR over the storage rows g*Ks + k of all four gates (rows not
// set: empty), assembled from the per-gate host copies that set_factors
// keeps, when they changed since the last upload.
int ensure_tau_csr(lstm_approx_t* h, int l) {
  LayerStore& s = h->layers[l];
  if (!s.hcsr_dirty && s.hoff != nullptr) return LSTM_APPROX_OK;
  const int Ks = h->Ks;
  std::vector<int> off(4 * (size_t)Ks + 1, 0), allc;
  std::vector<float> allv;
  for (int g = 0; g < 4; ++g) {
    size_t e = 0;
    for (int k = 0; k < Ks; ++k) {
      const int c = k < (int)s.hcount[g].size() ? s.hcount[g][k] : 0;
      for (int i = 0; i < c; ++i) {
        allc.push_back(s.hrows[g][e + i]);
        allv.push_back(s.hvals[g][e + i]);
      }
      e += c;
      off[g * Ks + k + 1] = (int)allc.size();
    }
  }
  const size_t n = allc.empty() ? 1 : allc.size();
  // earlier runs on the handle's stream may still read the old copy
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "synchronising before the factor upload");
  if (s.hoff == nullptr) {
    const int rc = dmalloc(h, reinterpret_cast<void**>(&s.hoff), off.size() * 4, "compressed factor storage");
    if (rc) return rc;
  }
  if (n > s.hcap) {
    dfree(h, s.hcol, s.hcap * 4);
    dfree(h, s.hval, s.hcap * 4);
    s.hcol = nullptr;
    s.hval = nullptr;
    s.hcap = 0;
    int rc = dmalloc(h, reinterpret_cast<void**>(&s.hcol), n * 4, "compressed factor storage");
    if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&s.hval), n * 4, "compressed factor storage");
    if (rc) return rc;
    s.hcap = n;
  }
  LA_CUDA(h, cudaMemcpy(s.hoff, off.data(), off.size() * 4, cudaMemcpyHostToDevice), "factor upload");
  if (!allc.empty()) {
    LA_CUDA(h, cudaMemcpy(s.hcol, allc.data(), allc.size() * 4, cudaMemcpyHostToDevice), "factor upload");
    LA_CUDA(h, cudaMemcpy(s.hval, allv.data(), allv.size() * 4, cudaMemcpyHostToDevice), "factor upload");
  }
  s.hcsr_dirty = false;
  return LSTM_APPROX_OK;
}

int ensure_factor_maps(lstm_approx_t* h, int l) {
  LayerStore& s = h->layers[l];
  if (s.maps_ready) return LSTM_APPROX_OK;
  const uint64_t rows = 4ull * h->Ks;
  if (!tc_make_map(&s.map_vx, s.Vx, s.D, rows, (uint64_t)s.ldx * 2, 128) ||
      !tc_make_map(&s.map_vh, s.Vh, h->H, rows, (uint64_t)h->ldh * 2, 128) ||
      !tc_make_map(&s.map_u, s.U, h->Ks, 4ull * h->H, (uint64_t)h->Ks * 2, 128) ||
      !tc_make_map(&s.map_u64, s.U, h->Ks, 4ull * h->H, (uint64_t)h->Ks * 2, 128, 64))
    return fail(h, LSTM_APPROX_ECUDA, "tensor map encoding failed for layer %d factors", l);
  for (int i = 0; i < 3; ++i)
    if (!tc_make_map(&s.map_vx_p[i], s.Vx, s.D, rows, (uint64_t)s.ldx * 2, 8u << i) ||
        !tc_make_map(&s.map_vh_p[i], s.Vh, h->H, rows, (uint64_t)h->ldh * 2, 8u << i))
      return fail(h, LSTM_APPROX_ECUDA, "tensor map encoding failed for layer %d factors", l);
  s.maps_ready = true;
  return LSTM_APPROX_OK;
}

// One layer on the tensor cores: bf16 input -> (a1) projection -> T x
// [(a2) tau' tile GEMM, (a3, a4, a6) four-gate GEMM with the cell epilogue].
int run_layer_tensor(lstm_approx_t* h, int l, const float* x, int T, int B, int K, const float* h0,
                     const float* c0, float* out_h, float* out_c, const Checkpoints& ck, float* ckpt_h,
                     float* ckpt_c) {
  LayerStore& s = h->layers[l];
  const int H = h->H, D = s.D, TB = T * B;
  const long long ldp = 4LL * h->Ks;
  int rc = ensure_factor_maps(h, l);
  if (rc) return rc;
  if (h->opt_tau_layout == 1 && (rc = ensure_tau_csr(h, l))) return rc;
  const bool top = l == h->L - 1;
  const long long limit_ns = h->opt_wait_limit_us * 1000LL;
  // up to 32 terms the products take one tile of all four gates' rows
  const int rpg = tensor_rows_per_gate(K);
  const int pi = rpg == 8 ? 0 : (rpg == 16 ? 1 : 2);
  __nv_bfloat16* in_bf16 = nullptr;
  int ld_in = 0;
  // packed gates at layer 0: the projection reads x in fp32 and forms its
  // bf16 pair itself (one tile of rows, so x is converted once either way;
  // with several row tiles each would convert it again: at K = 512 the
  // projection took twice as long), where TMA can map x
  const bool x_f32 = l == 0 && rpg > 0 && D % 4 == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  if (l == 0 && !x_f32) {  // operand conversion (outside the timed projection phase)
    LA_CUDA(h, launch_to_bf16(x, TB, D, static_cast<__nv_bfloat16*>(h->x_bf16), s.ldx, h->stream),
            "input conversion launch");
    in_bf16 = static_cast<__nv_bfloat16*>(h->x_bf16);
    ld_in = s.ldx;
    h->launches += 1;
  } else if (l > 0) {
    in_bf16 = static_cast<__nv_bfloat16*>(h->seq_bf16);
    ld_in = h->ldh;
  }
  {
    PhaseTimer pt(h, 0);
    const int kt = (K + 127) / 128;
    const int bnx = tc_rows_tile_n(TB, rpg > 0 ? 1 : 4 * kt);
    TcMap mx;
    const bool mapped = x_f32 ? tc_make_map_f32(&mx, x, D, TB, (uint64_t)D * 4, 64)
                              : tc_make_map(&mx, in_bf16, D, 2ull * TB, (uint64_t)ld_in * 2, bnx);
    if (!mapped) return fail(h, LSTM_APPROX_ECUDA, "tensor map encoding failed for the layer input");
    TcRowsArgs ra{};
    ra.Kdim = D;
    ra.K = K;
    ra.Ks = h->Ks;
    ra.kt_per_gate = (K + 127) / 128;
    ra.rpg = rpg;
    ra.N = TB;
    ra.b_plane = TB;
    ra.mode = 0;
    ra.P = h->Px;
    ra.ldp = (int)ldp;
    ra.err = h->err;
    ra.limit_ns = limit_ns;
    if (x_f32)
      LA_CUDA(h, launch_tc_rows_xf32(s.map_vx_p[pi], mx, ra, TB, h->stream), "input projection launch");
    else
      LA_CUDA(h, launch_tc_rows(rpg > 0 ? s.map_vx_p[pi] : s.map_vx, mx, ra, TB, bnx, h->stream),
              "input projection launch");
    h->launches += 1;
  }
  PhaseTimer pt(h, 1);
  __nv_bfloat16* hb = static_cast<__nv_bfloat16*>(h->h_bf16);
  __nv_bfloat16* tau = static_cast<__nv_bfloat16*>(h->tau);
  float* cs = h->c_state + (size_t)l * h->max_batch * H;
  int ns = 0, utiles = 0;
  if (h->opt_tensor_seq == 0 && h->opt_tau_layout == 0 && (long long)B * ldp < (1LL << 31) &&
      tc_seq_fits(H, B, K, ck, &ns, &utiles, nullptr)) {
    // one launch per tile of streams for all T timesteps
    TcSeqArgs qa{};
    qa.H = H;
    qa.K = K;
    qa.Ks = h->Ks;
    qa.B = B;
    qa.T = T;
    qa.rpg = rpg;
    qa.cs = H / (128 * utiles);
    qa.P = h->Px;
    qa.ldp = (int)ldp;
    qa.sigma = s.sigma;
    qa.bias = s.bias;
    qa.h0 = h0;
    qa.c0 = c0;
    qa.out_h = out_h;
    qa.c_last = out_c;
    qa.seq_bf16 = top ? nullptr : static_cast<__nv_bfloat16*>(h->seq_bf16);
    qa.ldh = h->ldh;
    qa.seq_plane = (long long)TB * h->ldh;
    qa.ck = ck;
    qa.ckpt_h = ckpt_h;
    qa.ckpt_c = ckpt_c;
    qa.ck_stride = (long long)T * B * H;
    qa.err = h->err;
    qa.limit_ns = limit_ns;
    qa.test_stall = h->opt_test_stall;
    h->opt_test_stall = 0;
    LA_CUDA(h, launch_tc_seq(s.map_vh_p[pi], s.map_u64, qa, ns, utiles, h->stream), "recurrence launch");
    h->launches += 1;
    h->last_tensor_seq = 1;
    return LSTM_APPROX_OK;
  }
  h->last_tensor_seq = 0;
  LA_CUDA(h, launch_tc_init_state(h0, c0, B, H, hb, h->ldh, cs, h->stream), "state init launch");
  h->launches += 1;
  // packed gates write only the first rpg terms of each gate's tau' rows; the
  // gate GEMM reads 64-term chunks, so the rest of the pair must be zero
  if (rpg > 0)
    LA_CUDA(h, cudaMemsetAsync(tau, 0, 2ull * B * 4 * h->Ks * sizeof(__nv_bfloat16), h->stream), "tau' clear");
  const TensorTiles tt = tensor_tiles(H, B, K, ck);
  const int bnh = tt.bnh, nt = tt.nt, ks = tt.ks, nkb_per = tt.nkb_per;
  if (tt.raw) {
    const size_t need = (size_t)(ks + ck.n) * 4 * B * H * sizeof(float);
    if (need > h->gpart_bytes) {
      LA_CUDA(h, cudaStreamSynchronize(h->stream), "synchronising before growing the split buffer");
      dfree(h, h->gpart, h->gpart_bytes);
      h->gpart = nullptr;
      h->gpart_bytes = 0;
      rc = dmalloc(h, reinterpret_cast<void**>(&h->gpart), need, "split gate sums");
      if (rc) return rc;
      h->gpart_bytes = need;
    }
  }
  TcMap mh, mt;
  if (!tc_make_map(&mh, hb, H, 2ull * B, (uint64_t)h->ldh * 2, bnh) ||
      !tc_make_map(&mt, tau, ldp, 2ull * B, (uint64_t)ldp * 2, nt))
    return fail(h, LSTM_APPROX_ECUDA, "tensor map encoding failed for the state");
  for (int t = 0; t < T; ++t) {
    TcRowsArgs ra{};
    ra.Kdim = H;
    ra.K = K;
    ra.Ks = h->Ks;
    ra.kt_per_gate = (K + 127) / 128;
    ra.rpg = rpg;
    ra.N = B;
    ra.b_plane = B;
    ra.mode = 1;
    ra.P = h->Px + (size_t)t * B * ldp;
    ra.ldp = (int)ldp;
    ra.sigma = s.sigma;
    ra.tau = tau;
    ra.ldt = (int)ldp;
    ra.tau_plane = (long long)B * ldp;
    ra.err = h->err;
    ra.limit_ns = limit_ns;
    ra.sk = tt.sk;
    ra.nkb_per = tt.nkb_per_h;
    if (h->opt_tau_layout == 1) {  // compressed rows of v's h part on the CUDA cores
      TauSparseArgs sa{};
      sa.off = s.hoff;
      sa.col = s.hcol;
      sa.val = s.hval;
      sa.sigma = s.sigma;
      sa.P = ra.P;
      sa.ldp = (int)ldp;
      sa.h = hb;
      sa.ldh = h->ldh;
      sa.h_plane = (long long)B * h->ldh;
      sa.tau = tau;
      sa.ldt = (int)ldp;
      sa.tau_plane = (long long)B * ldp;
      sa.H = H;
      sa.K = K;
      sa.Ks = h->Ks;
      sa.B = B;
      sa.Rp = (K + 63) / 64 * 64;
      LA_CUDA(h, launch_tau_sparse(sa, h->stream), "recurrent projection launch");
    } else {
      LA_CUDA(h, launch_tc_rows(rpg > 0 ? s.map_vh_p[pi] : s.map_vh, mh, ra, B, bnh, h->stream),
              "recurrent projection launch");
    }
    TcGatesArgs ga{};
    ga.H = H;
    ga.K = K;
    ga.Ks = h->Ks;
    ga.B = B;
    ga.nkb = (K + 63) / 64;
    ga.tau_rows = B;
    ga.U = static_cast<const __nv_bfloat16*>(s.U);
    ga.tau = tau;
    ga.ldt = (int)ldp;
    ga.tau_plane = (long long)B * ldp;
    ga.bias = s.bias;
    ga.c_state = cs;
    ga.h_bf16 = hb;
    ga.ldh = h->ldh;
    ga.h_plane = (long long)B * h->ldh;
    ga.out_h = out_h ? out_h + (size_t)t * B * H : nullptr;
    ga.seq_bf16 = top ? nullptr : static_cast<__nv_bfloat16*>(h->seq_bf16) + (size_t)t * B * h->ldh;
    ga.seq_plane = (long long)TB * h->ldh;
    ga.ck = ck;
    ga.ckpt_h = ckpt_h ? ckpt_h + (size_t)t * B * H : nullptr;
    ga.ckpt_c = ckpt_c ? ckpt_c + (size_t)t * B * H : nullptr;
    ga.ck_stride = (long long)T * B * H;
    ga.err = h->err;
    ga.limit_ns = limit_ns;
    ga.ks = ks;
    ga.nkb_per = nkb_per;
    ga.part = h->gpart;
    ga.raw = tt.raw;
    LA_CUDA(h, launch_tc_gates(s.map_u, mt, ga, nt, h->stream), "gate GEMM launch");
    h->launches += tt.raw ? 3 : 2;
  }
  if (out_c) LA_CUDA(h, cudaMemcpyAsync(out_c, cs, (size_t)B * H * sizeof(float), cudaMemcpyDeviceToDevice, h->stream),
                     "c copy");
  return LSTM_APPROX_OK;
}

int run_device(lstm_approx_t* h, const float* x, int T, int B, int K, const float* h0, const float* c0,
               float* out_h, float* out_c, const Checkpoints& ck, float* ckpt_h, float* ckpt_c) {
  const int H = h->H;
  const bool bf16 = h->dtype == LSTM_APPROX_BF16;
  int rc = ensure_scratch(h, static_cast<size_t>(T) * B);
  if (rc) return rc;
  if (h->timing.on) {
    clear_timing(h);
    if (!h->timing.run0) {
      cudaEventCreate(&h->timing.run0);
      cudaEventCreate(&h->timing.run1);
    }
    cudaEventRecord(h->timing.run0, h->stream);
  }
  const long long ldp = 4LL * h->Ks;
  // A bf16 run takes one path for all its layers, the one its top layer (the
  // only one with intermediate depths) takes: the tensor-core path hands the
  // sequence to the next layer in bf16, the CUDA-core kernels in fp32.
  int run_path = 0;
  if (bf16) {
    PersistentChoice unused;
    std::string why;
    run_path = select_path(h->dtype, H, K, T, ck, h->opt_force_path, h->opt_cluster, h->sm_count,
                           h->opt_persistent_variant, &unused, &why);
    if (run_path == 0) return fail(h, LSTM_APPROX_EINVAL, "%s", why.c_str());
  }
  for (int l = 0; l < h->L; ++l) {
    const LayerStore& s = h->layers[l];
    const bool top = l == h->L - 1;
    const float* in = l == 0 ? x : h->seq;
    float* out = top ? out_h : h->seq;
    const Checkpoints none = {0, {0}};
    const Checkpoints& lck = top ? ck : none;
    // recurrence path
    PersistentChoice plan;
    std::string why;
    const int path = bf16 ? run_path
                          : select_path(h->dtype, H, K, T, lck, h->opt_force_path, h->opt_cluster, h->sm_count,
                                        h->opt_persistent_variant, &plan, &why);
    if (path == 0) return fail(h, LSTM_APPROX_EINVAL, "%s", why.c_str());
    const float* l_h0 = h0 ? h0 + (size_t)l * B * H : nullptr;
    const float* l_c0 = c0 ? c0 + (size_t)l * B * H : nullptr;
    float* l_cout = out_c ? out_c + (size_t)l * B * H : nullptr;
    if (path == LSTM_APPROX_PATH_TENSOR) {
      rc = run_layer_tensor(h, l, x, T, B, K, l_h0, l_c0, top ? out_h : nullptr, l_cout, lck,
                            top ? ckpt_h : nullptr, top ? ckpt_c : nullptr);
      if (rc) return rc;
      h->last_path = path;
      continue;
    }
    // (a1) hoisted input projection P[t][b][(g,k)] = prune(v_{g,k})[0:D]^T x_t,b
    //
    // Order of the two launches.  Ahead of the per-unit-block persistent
    // kernel for one stream, when the few-column projection kernel serves and
    // no phase is being timed, the recurrence is launched first: its cluster
    // takes its SMs at once, the projection follows as its programmatic
    // dependent on the SMs left free and raises one flag per CTA, and the
    // recurrence loads its factors meanwhile and waits for the flags before
    // its first read of P, unless the stream is being captured into a graph
    // (D = 1024, H = 512, T = 20, whole call: K = 256
    // with two intermediate depths 64.1 -> 60.0 us, K = 64 46.8 -> 45.0 us;
    // with the projection split four ways along D, 128 CTAs, 68.7 us).  The
    // one-exchange kernel's short set-up gains nothing from it (K = 16:
    // 41.4 -> 43.0 us), and several streams' clusters need not all be
    // resident at once, which the flags would require.  Otherwise the
    // projection comes first and the recurrence starts as its programmatic
    // dependent; there, before the per-unit-block kernel at K > 128 (a
    // cluster of 16 CTAs whose set-up fills about 256 KB of tensor memory
    // each), the projection runs unsplit along D: its smaller grid leaves a
    // GPC free, so that the recurrence's set-up overlaps it (the run 2%
    // faster although the projection takes 15.8 instead of 10.5 us).
    // Shorter set-ups gain less than the slower projection costs (K = 64: 4%
    // slower, the one-exchange kernel at K = 16: 11%).
    const bool sparse_x = sparse_x_projection(h, s, K, T * B);
    const bool cluster_x = !sparse_x && xproj_cluster_fits(T * B, s.D, s.Vx, s.ldx, in, s.D, bf16);
    // (not while the stream is being captured: a graph would replay the
    // launches with the epoch value of the capture, and the flags of the
    // previous replay would already hold it)
    cudaStreamCaptureStatus capture = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(h->stream, &capture) != cudaSuccess) capture = cudaStreamCaptureStatusActive;
    bool rec_first = path == LSTM_APPROX_PATH_PERSISTENT && plan.variant == 1 && B == 1 && cluster_x &&
                     !h->timing.on && h->opt_launch_order == 0 && h->proj_flags != nullptr &&
                     capture == cudaStreamCaptureStatusNone;
    const int proj_ctas = rec_first ? xproj_cluster_ctas(K, T * B, s.D, 8) : 0;
    rec_first = rec_first && proj_ctas <= kProjFlags && xproj_cluster_prepare(bf16, T * B) == cudaSuccess;
    const int xproj_max_split =
        rec_first ? 8 : (path == LSTM_APPROX_PATH_PERSISTENT && plan.variant == 1 && K > 128) ? 1 : 8;
    XprojSignal sig;
    if (rec_first) {
      if (++h->proj_epoch == 0) ++h->proj_epoch;  // the flags start at zero
      sig.flags = h->proj_flags;
      sig.epoch = h->proj_epoch;
    }
    auto launch_projection = [&]() -> int {
      PhaseTimer pt(h, 0);
      if (sparse_x) {
        SparseXRows sr;
        for (int g = 0; g < 4; ++g) {
          sr.off[g] = s.xoff[g];
          sr.idx[g] = s.xidx[g];
          sr.val[g] = s.xval[g];
        }
        LA_CUDA(h, launch_xproj_sparse(sr, K, h->Ks, in, s.D, T * B, h->Px, (int)ldp, h->stream),
                "input projection launch");
      } else if (cluster_x)
        LA_CUDA(h,
                launch_xproj_cluster(s.Vx, bf16, s.ldx, K, h->Ks, in, s.D, T * B, s.D, h->Px, (int)ldp, h->err,
                                     h->opt_wait_limit_us * 1000LL, h->stream, xproj_max_split,
                                     rec_first ? &sig : nullptr),
                "input projection launch");
      else
        LA_CUDA(h,
                launch_rows_gemm(s.Vx, bf16, s.ldx, K, h->Ks, in, s.D, T * B, s.D, h->Px, (int)ldp, 0, nullptr,
                                 nullptr, 0, h->stream),
                "input projection launch");
      h->launches += 1;
      return LSTM_APPROX_OK;
    };
    if (!rec_first) {
      rc = launch_projection();
      if (rc) return rc;
    }
    if (path == LSTM_APPROX_PATH_PERSISTENT) {
      PhaseTimer pt(h, 1);
      PersistentArgs a{};
      a.Vh = static_cast<const float*>(s.Vh);
      a.U = static_cast<const float*>(s.U);
      a.sigma = s.sigma;
      a.bias = s.bias;
      a.P = h->Px;
      a.h0 = l_h0;
      a.c0 = l_c0;
      a.out_h = out;
      a.c_last = l_cout;
      a.ckpt_h = top ? ckpt_h : nullptr;
      a.ckpt_c = top ? ckpt_c : nullptr;
      a.err = h->err;
      a.H = H;
      a.K = K;
      a.Ks = h->Ks;
      a.ldh = h->ldh;
      a.T = T;
      a.B = B;
      a.ck = lck;
      a.wait_limit_ns = h->opt_wait_limit_us * 1000LL;
      a.test_stall = h->opt_test_stall;
      if (rec_first) {
        a.proj_flags = h->proj_flags;
        a.proj_nflags = proj_ctas;
        a.proj_epoch = sig.epoch;
      }
      h->opt_test_stall = 0;
      LA_CUDA(h, launch_persistent_choice(plan, a, h->stream), "persistent kernel launch");
      h->launches += 1;
      h->last_cluster = plan.CS;
      h->last_variant = plan.variant;
      if (rec_first) {
        rc = launch_projection();
        if (rc) return rc;
      }
    } else {
      PhaseTimer pt(h, 1);
      float* hs = h->h_state + (size_t)l * h->max_batch * H;
      float* cs = h->c_state + (size_t)l * h->max_batch * H;
      const size_t sb = (size_t)B * H * sizeof(float);
      if (l_h0) LA_CUDA(h, cudaMemcpyAsync(hs, l_h0, sb, cudaMemcpyDeviceToDevice, h->stream), "h0 copy");
      else LA_CUDA(h, cudaMemsetAsync(hs, 0, sb, h->stream), "h0 clear");
      if (l_c0) LA_CUDA(h, cudaMemcpyAsync(cs, l_c0, sb, cudaMemcpyDeviceToDevice, h->stream), "c0 copy");
      else LA_CUDA(h, cudaMemsetAsync(cs, 0, sb, h->stream), "c0 clear");
      float* tau = static_cast<float*>(h->tau);
      for (int t = 0; t < T; ++t) {
        // (a2) tau' = sigma * (P_t + prune(v)[D:]^T h_{t-1})
        LA_CUDA(h,
                launch_rows_gemm(s.Vh, bf16, h->ldh, K, h->Ks, hs, H, B, H, tau, (int)ldp, 1, s.sigma,
                                 h->Px + (size_t)t * B * ldp, (int)ldp, h->stream),
                "recurrent projection launch");
        // (a3, a4, a6) sums over u, intermediate outputs, cell update
        CellArgs ca{};
        ca.U = s.U;
        ca.u_bf16 = bf16;
        ca.gs = (long long)H * h->Ks;  // U is [4][H][Ks] for both factor types
        ca.ks = 1;
        ca.js = h->Ks;
        ca.K = K;
        ca.Ks = h->Ks;
        ca.H = H;
        ca.B = B;
        ca.tau = tau;
        ca.ldt = (int)ldp;
        ca.bias = s.bias;
        ca.c_state = cs;
        ca.h_state = hs;
        ca.out_h = out + (size_t)t * B * H;
        ca.ck = lck;
        ca.ckpt_h = (top && ckpt_h) ? ckpt_h + (size_t)t * B * H : nullptr;
        ca.ckpt_c = (top && ckpt_c) ? ckpt_c + (size_t)t * B * H : nullptr;
        ca.ck_stride = (long long)T * B * H;
        LA_CUDA(h, launch_cell_step(ca, h->stream), "cell step launch");
        h->launches += 2;
      }
      if (l_cout) LA_CUDA(h, cudaMemcpyAsync(l_cout, cs, sb, cudaMemcpyDeviceToDevice, h->stream), "c copy");
    }
    h->last_path = path;
  }
  if (h->timing.on) cudaEventRecord(h->timing.run1, h->stream);
  return LSTM_APPROX_OK;
}

// Error text into a caller's buffer (entry points without a handle).
int report(char* msg, int msg_len, int code, const char* fmt, ...) {
  if (msg && msg_len > 0) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(msg, (size_t)msg_len, fmt, ap);
    va_end(ap);
  }
  return code;
}

}  // namespace

extern "C" {

int lstm_approx_create(lstm_approx_t** out, int num_layers, const int* input_dims, int hidden, int max_rank,
                       int max_batch, int dtype, void* cuda_stream) {
  if (!out) return LSTM_APPROX_EINVAL;
  *out = nullptr;
  if (num_layers < 1 || num_layers > 64 || !input_dims || hidden < 1 || max_rank < 1 || max_batch < 1 ||
      (dtype != LSTM_APPROX_FP32 && dtype != LSTM_APPROX_BF16))
    return LSTM_APPROX_EINVAL;
  if (input_dims[0] < 1) return LSTM_APPROX_EINVAL;
  for (int l = 1; l < num_layers; ++l)
    if (input_dims[l] != hidden) return LSTM_APPROX_EINVAL;
  if (hidden > (1 << 20) || input_dims[0] > (1 << 22) || max_rank > (1 << 16) || max_batch > (1 << 20))
    return LSTM_APPROX_EINVAL;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return LSTM_APPROX_ECUDA;
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return LSTM_APPROX_ECUDA;
  if (prop.major != 10 || prop.minor != 3) return LSTM_APPROX_ECUDA;

  lstm_approx_t* h = new (std::nothrow) lstm_approx;
  if (!h) return LSTM_APPROX_ENOMEM;
  h->L = num_layers;
  h->H = hidden;
  h->ldh = round_up(hidden, 8);
  h->Kmax = max_rank;
  h->Ks = dtype == LSTM_APPROX_BF16 ? round_up(max_rank, 128) : round_up(max_rank, 4);
  h->max_batch = max_batch;
  h->dtype = dtype;
  h->stream = static_cast<cudaStream_t>(cuda_stream);
  h->device = dev;
  h->sm_count = prop.multiProcessorCount;
  // with every launch made blocking, the recurrence can never run beside the
  // projection launched after it: start with the projection first
  const char* blocking = std::getenv("CUDA_LAUNCH_BLOCKING");
  if (blocking != nullptr && blocking[0] == '1') h->opt_launch_order = 1;
  h->layers.resize(num_layers);
  int rc = LSTM_APPROX_OK;
  for (int l = 0; l < num_layers && !rc; ++l) {
    LayerStore& s = h->layers[l];
    s.D = input_dims[l];
    s.C = s.D + hidden;
    s.ldx = round_up(s.D, 8);
    s.mask_words = (s.C + 31) / 32;
    if (!rc) rc = dmalloc(h, &s.Vx, layer_bytes_vx(h, s), "factor storage");
    if (!rc) rc = dmalloc(h, &s.Vh, layer_bytes_vh(h), "factor storage");
    if (!rc) rc = dmalloc(h, &s.U, layer_bytes_u(h), "factor storage");
    if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&s.sigma), 4ull * h->Ks * 4, "factor storage");
    if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&s.bias), 4ull * hidden * 4, "factor storage");
    if (!rc)
      rc = dmalloc(h, reinterpret_cast<void**>(&s.mask), 4ull * h->Ks * s.mask_words * 4, "factor storage");
  }
  const size_t state = (size_t)num_layers * max_batch * hidden * sizeof(float);
  if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&h->h_state), state, "state");
  if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&h->c_state), state, "state");
  if (!rc) rc = dmalloc(h, &h->tau, (size_t)max_batch * 4 * h->Ks * sizeof(float), "scratch tau");
  if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&h->err), sizeof(int), "status word");
  if (!rc)
    rc = dmalloc(h, reinterpret_cast<void**>(&h->proj_flags), kProjFlags * sizeof(unsigned), "projection flags");
  if (!rc && cudaHostAlloc(reinterpret_cast<void**>(&h->err_host), sizeof(int), cudaHostAllocDefault) != cudaSuccess)
    rc = fail(h, LSTM_APPROX_ENOMEM, "pinned status word");
  if (!rc && dtype == LSTM_APPROX_BF16)
    rc = dmalloc(h, &h->h_bf16, 2 * (size_t)max_batch * h->ldh * 2, "bf16 state pair");
  if (rc) {
    lstm_approx_destroy(h);
    return rc;
  }
  *out = h;
  return LSTM_APPROX_OK;
}

int lstm_approx_set_factors(lstm_approx_t* h, int layer, int gate, int K, int nz, const double* sigma,
                            const double* u, const int32_t* v_idx, const double* v_val, const double* bias) {
  if (!h) return LSTM_APPROX_EINVAL;
  if (layer < 0 || layer >= h->L) return fail(h, LSTM_APPROX_EINVAL, "layer %d outside [0, %d)", layer, h->L);
  if (gate < 0 || gate > 3) return fail(h, LSTM_APPROX_EINVAL, "gate %d outside [0, 4)", gate);
  LayerStore& s = h->layers[layer];
  if (K < 1 || K > h->Kmax) return fail(h, LSTM_APPROX_EINVAL, "K=%d outside [1, %d]", K, h->Kmax);
  if (nz < 1 || nz > s.C) return fail(h, LSTM_APPROX_EINVAL, "nz=%d outside [1, C=%d]", nz, s.C);
  if (!sigma || !u || !v_idx || !v_val) return fail(h, LSTM_APPROX_EINVAL, "factor pointer is NULL");
  for (int k = 0; k < K; ++k)
    for (int m = 0; m < nz; ++m) {
      const int32_t c = v_idx[(size_t)k * nz + m];
      if (c < 0 || c >= s.C) return fail(h, LSTM_APPROX_EINVAL, "v_idx[%d][%d]=%d outside [0, %d)", k, m, c, s.C);
      if (m > 0 && c <= v_idx[(size_t)k * nz + m - 1])
        return fail(h, LSTM_APPROX_EINVAL, "v_idx row %d not strictly increasing", k);
    }
  DeviceGuard dg(h->device);
  const int H = h->H, D = s.D, Ks = h->Ks;
  const bool bf16 = h->dtype == LSTM_APPROX_BF16;
  const size_t es = elem_size(h->dtype);
  std::vector<unsigned char> vx((size_t)K * s.ldx * es, 0), vh((size_t)K * h->ldh * es, 0),
      uu((size_t)K * H * es, 0);
  std::vector<uint32_t> mask((size_t)K * s.mask_words, 0);
  std::vector<float> sg(K), bs(H, 0.f);
  auto put = [&](std::vector<unsigned char>& buf, size_t i, double v) {
    if (bf16) {
      const uint16_t b = to_bf16_bits(v);
      std::memcpy(buf.data() + 2 * i, &b, 2);
    } else {
      const float f = static_cast<float>(v);
      std::memcpy(buf.data() + 4 * i, &f, 4);
    }
  };
  for (int k = 0; k < K; ++k) {
    sg[k] = static_cast<float>(sigma[k]);
    for (int m = 0; m < nz; ++m) {
      const int c = v_idx[(size_t)k * nz + m];
      const double v = v_val[(size_t)k * nz + m];
      if (c < D) put(vx, (size_t)k * s.ldx + c, v);
      else put(vh, (size_t)k * h->ldh + (c - D), v);
      mask[(size_t)k * s.mask_words + c / 32] |= 1u << (c % 32);
    }
    for (int j = 0; j < H; ++j) put(uu, (size_t)j * K + k, u[(size_t)k * H + j]);  // [H][K], into [H][Ks] below
  }
  if (bias)
    for (int j = 0; j < H; ++j) bs[j] = static_cast<float>(bias[j]);
  const size_t row0 = (size_t)gate * Ks;
  char* Vx = static_cast<char*>(s.Vx);
  char* Vh = static_cast<char*>(s.Vh);
  char* U = static_cast<char*>(s.U);
  LA_CUDA(h, cudaMemcpy(Vx + row0 * s.ldx * es, vx.data(), vx.size(), cudaMemcpyHostToDevice), "factor upload");
  LA_CUDA(h, cudaMemcpy(Vh + row0 * h->ldh * es, vh.data(), vh.size(), cudaMemcpyHostToDevice), "factor upload");
  LA_CUDA(h,
          cudaMemcpy2D(U + (size_t)gate * H * Ks * es, Ks * es, uu.data(), K * es, K * es, H, cudaMemcpyHostToDevice),
          "factor upload");
  LA_CUDA(h, cudaMemcpy(s.sigma + row0, sg.data(), K * sizeof(float), cudaMemcpyHostToDevice), "factor upload");
  LA_CUDA(h, cudaMemcpy(s.bias + (size_t)gate * H, bs.data(), H * sizeof(float), cudaMemcpyHostToDevice),
          "factor upload");
  LA_CUDA(h,
          cudaMemcpy(s.mask + row0 * s.mask_words, mask.data(), mask.size() * sizeof(uint32_t),
                     cudaMemcpyHostToDevice),
          "factor upload");
  if (bf16) {  // the h part again, compressed, for the compressed tau' layout of the tensor path
    std::vector<int>& cols = s.hrows[gate];
    std::vector<float>& vals = s.hvals[gate];
    std::vector<int>& cnt = s.hcount[gate];
    cols.clear();
    vals.clear();
    cnt.assign(K, 0);
    for (int k = 0; k < K; ++k)
      for (int m = 0; m < nz; ++m) {
        const int c = v_idx[(size_t)k * nz + m];
        if (c < D) continue;
        const uint32_t bits = static_cast<uint32_t>(to_bf16_bits(v_val[(size_t)k * nz + m])) << 16;
        float f;
        std::memcpy(&f, &bits, 4);
        cols.push_back(c - D);
        vals.push_back(f);
        ++cnt[k];
      }
    s.hcsr_dirty = true;  // the device copy is rebuilt by the first run that uses it
  }
  if (!bf16) {  // the x part again, compressed: kept (column, value) runs of every row k
    std::vector<int> off(Ks + 1, 0), cols;
    std::vector<float> vals;
    for (int k = 0; k < K; ++k) {
      for (int m = 0; m < nz; ++m) {
        const int c = v_idx[(size_t)k * nz + m];
        if (c >= D) break;  // indices ascend: the h columns follow
        cols.push_back(c);
        vals.push_back(static_cast<float>(v_val[(size_t)k * nz + m]));
      }
      off[k + 1] = static_cast<int>(cols.size());
    }
    for (int k = K; k < Ks; ++k) off[k + 1] = off[K];
    const size_t n = cols.size() > 0 ? cols.size() : 1;
    if (n > s.xcap[gate] || s.xoff[gate] == nullptr) {
      dfree(h, s.xidx[gate], s.xcap[gate] * 4);
      dfree(h, s.xval[gate], s.xcap[gate] * 4);
      s.xidx[gate] = nullptr;
      s.xval[gate] = nullptr;
      s.xcap[gate] = 0;
      int rc = dmalloc(h, reinterpret_cast<void**>(&s.xidx[gate]), n * 4, "compressed factor storage");
      if (!rc) rc = dmalloc(h, reinterpret_cast<void**>(&s.xval[gate]), n * 4, "compressed factor storage");
      if (!rc && s.xoff[gate] == nullptr)
        rc = dmalloc(h, reinterpret_cast<void**>(&s.xoff[gate]), (Ks + 1) * 4ull, "compressed factor storage");
      if (rc) return rc;
      s.xcap[gate] = n;
    }
    LA_CUDA(h, cudaMemcpy(s.xoff[gate], off.data(), off.size() * 4, cudaMemcpyHostToDevice), "factor upload");
    if (!cols.empty()) {
      LA_CUDA(h, cudaMemcpy(s.xidx[gate], cols.data(), cols.size() * 4, cudaMemcpyHostToDevice), "factor upload");
      LA_CUDA(h, cudaMemcpy(s.xval[gate], vals.data(), vals.size() * 4, cudaMemcpyHostToDevice), "factor upload");
    }
    s.xoff_h[gate] = off;
  }
  s.Kset[gate] = K;
  s.nz[gate] = nz;
  return LSTM_APPROX_OK;
}

int lstm_approx_run(lstm_approx_t* h, const float* x, int T, int B, int K, const float* h0, const float* c0,
                    float* out_h, float* out_c, const int* checkpoints, int J, float* ckpt_h, float* ckpt_c) {
  if (!h) return LSTM_APPROX_EINVAL;
  Checkpoints ck;
  int rc = validate_run(h, x, T, B, K, out_h, checkpoints, J, &ck);
  if (rc) return rc;
  DeviceGuard dg(h->device);
  return run_device(h, x, T, B, K, h0, c0, out_h, out_c, ck, ckpt_h, ckpt_c);
}

// Device address of a page-locked, mapped host buffer that the kernels may
// write in place (16-byte aligned), else null: pageable memory goes through
// the staging copies.
static float* mapped_view(const float* p) {
  if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0) return nullptr;
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();  // an unknown pointer: clear the (non-sticky) error
    return nullptr;
  }
  if (at.type != cudaMemoryTypeHost || at.devicePointer == nullptr) return nullptr;
  return static_cast<float*>(at.devicePointer);
}

int lstm_approx_run_host(lstm_approx_t* h, const float* x, int T, int B, int K, const float* h0, const float* c0,
                         float* out_h, float* out_c, const int* checkpoints, int J, float* ckpt_h, float* ckpt_c) {
  if (!h) return LSTM_APPROX_EINVAL;
  Checkpoints ck;
  int rc = validate_run(h, x, T, B, K, out_h, checkpoints, J, &ck);
  if (rc) return rc;
  DeviceGuard dg(h->device);
  const size_t H = h->H, L = h->L, D = h->layers[0].D;
  const size_t nx = (size_t)T * B * D, ns = L * B * H, no = (size_t)T * B * H, nk = (size_t)J * T * B * H;
  const size_t off_x = 0, off_h0 = off_x + nx, off_c0 = off_h0 + ns, off_oh = off_c0 + ns, off_oc = off_oh + no,
               off_kh = off_oc + ns, off_kc = off_kh + nk, total = (off_kc + nk) * sizeof(float);
  if (total > h->stage_bytes) {
    LA_CUDA(h, cudaStreamSynchronize(h->stream), "synchronising before growing staging");
    dfree(h, h->stage, h->stage_bytes);
    h->stage = nullptr;
    h->stage_bytes = 0;
    rc = dmalloc(h, reinterpret_cast<void**>(&h->stage), total, "host-call staging");
    if (rc) return rc;
    h->stage_bytes = total;
  }
  float* st = reinterpret_cast<float*>(h->stage);
  // page-locked out_h and checkpoint buffers are written in place by the
  // kernels over the host link (the stores are posted; 3% off a batch-1
  // call).  The inputs are staged: a kernel reading x from host memory waits
  // on the link, which costs more than one copy.  The states, which the run
  // copies between device buffers, are staged too.
  const float* dx = nullptr;
  const float* dh0 = nullptr;
  const float* dc0 = nullptr;
  float* doh = mapped_view(out_h);
  float* doc = nullptr;
  float* dkh = nk ? mapped_view(ckpt_h) : nullptr;
  float* dkc = nk ? mapped_view(ckpt_c) : nullptr;
  if (!dx) {
    LA_CUDA(h, cudaMemcpyAsync(st + off_x, x, nx * 4, cudaMemcpyHostToDevice, h->stream), "input copy");
    dx = st + off_x;
  }
  if (h0 && !dh0) {
    LA_CUDA(h, cudaMemcpyAsync(st + off_h0, h0, ns * 4, cudaMemcpyHostToDevice, h->stream), "h0 copy");
    dh0 = st + off_h0;
  }
  if (c0 && !dc0) {
    LA_CUDA(h, cudaMemcpyAsync(st + off_c0, c0, ns * 4, cudaMemcpyHostToDevice, h->stream), "c0 copy");
    dc0 = st + off_c0;
  }
  rc = run_device(h, dx, T, B, K, dh0, dc0, doh ? doh : st + off_oh, out_c ? (doc ? doc : st + off_oc) : nullptr, ck,
                  (ckpt_h && nk) ? (dkh ? dkh : st + off_kh) : nullptr,
                  (ckpt_c && nk) ? (dkc ? dkc : st + off_kc) : nullptr);
  if (rc) return rc;
  if (!doh) LA_CUDA(h, cudaMemcpyAsync(out_h, st + off_oh, no * 4, cudaMemcpyDeviceToHost, h->stream), "output copy");
  if (out_c && !doc)
    LA_CUDA(h, cudaMemcpyAsync(out_c, st + off_oc, ns * 4, cudaMemcpyDeviceToHost, h->stream), "c copy");
  if (ckpt_h && nk && !dkh)
    LA_CUDA(h, cudaMemcpyAsync(ckpt_h, st + off_kh, nk * 4, cudaMemcpyDeviceToHost, h->stream), "ckpt copy");
  if (ckpt_c && nk && !dkc)
    LA_CUDA(h, cudaMemcpyAsync(ckpt_c, st + off_kc, nk * 4, cudaMemcpyDeviceToHost, h->stream), "ckpt copy");
  return lstm_approx_sync(h);
}

int lstm_approx_sync(lstm_approx_t* h) {
  if (!h) return LSTM_APPROX_EINVAL;
  DeviceGuard dg(h->device);
  // the status word rides on the stream into pinned memory: one synchronisation
  LA_CUDA(h, cudaMemcpyAsync(h->err_host, h->err, sizeof(int), cudaMemcpyDeviceToHost, h->stream), "status read");
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "stream synchronise");
  const int code = *h->err_host;
  if (code != 0) {
    LA_CUDA(h, cudaMemsetAsync(h->err, 0, sizeof(int), h->stream), "status clear");
    LA_CUDA(h, cudaStreamSynchronize(h->stream), "stream synchronise");
    return fail(h, LSTM_APPROX_ETIMEOUT, "a bounded in-kernel wait ran out (code %d); outputs are invalid", code);
  }
  return LSTM_APPROX_OK;
}

int lstm_approx_get_mask(lstm_approx_t* h, int layer, int gate, int k, int32_t* idx_out, int* nz_out) {
  if (!h) return LSTM_APPROX_EINVAL;
  if (layer < 0 || layer >= h->L || gate < 0 || gate > 3 || !idx_out || !nz_out)
    return fail(h, LSTM_APPROX_EINVAL, "bad layer/gate/pointer");
  const LayerStore& s = h->layers[layer];
  if (k < 0 || k >= s.Kset[gate]) return fail(h, LSTM_APPROX_EINVAL, "term %d not set", k);
  DeviceGuard dg(h->device);
  std::vector<uint32_t> words(s.mask_words);
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "stream synchronise");
  LA_CUDA(h,
          cudaMemcpy(words.data(), s.mask + ((size_t)gate * h->Ks + k) * s.mask_words,
                     s.mask_words * sizeof(uint32_t), cudaMemcpyDeviceToHost),
          "mask read");
  int n = 0;
  for (int c = 0; c < s.C; ++c)
    if (words[c / 32] >> (c % 32) & 1u) idx_out[n++] = c;
  *nz_out = n;
  return LSTM_APPROX_OK;
}

int lstm_approx_get_term(lstm_approx_t* h, int layer, int gate, int k, float* sigma_out, float* u_out,
                         float* v_out) {
  if (!h) return LSTM_APPROX_EINVAL;
  if (layer < 0 || layer >= h->L || gate < 0 || gate > 3 || !sigma_out || !u_out || !v_out)
    return fail(h, LSTM_APPROX_EINVAL, "bad layer/gate/pointer");
  const LayerStore& s = h->layers[layer];
  if (k < 0 || k >= s.Kset[gate]) return fail(h, LSTM_APPROX_EINVAL, "term %d not set", k);
  DeviceGuard dg(h->device);
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "stream synchronise");
  const int H = h->H, D = s.D, Ks = h->Ks;
  const bool bf16 = h->dtype == LSTM_APPROX_BF16;
  const size_t es = elem_size(h->dtype);
  const size_t row = (size_t)gate * Ks + k;
  std::vector<unsigned char> vx((size_t)D * es), vh((size_t)H * es), uu((size_t)H * es);
  LA_CUDA(h, cudaMemcpy(vx.data(), static_cast<const char*>(s.Vx) + row * s.ldx * es, vx.size(), cudaMemcpyDeviceToHost),
          "factor read");
  LA_CUDA(h, cudaMemcpy(vh.data(), static_cast<const char*>(s.Vh) + row * h->ldh * es, vh.size(), cudaMemcpyDeviceToHost),
          "factor read");
  // u_k[j] sits at (gate*H + j)*Ks + k: one strided column of U
  LA_CUDA(h,
          cudaMemcpy2D(uu.data(), es, static_cast<const char*>(s.U) + ((size_t)gate * H * Ks + k) * es, Ks * es, es, H,
                       cudaMemcpyDeviceToHost),
          "factor read");
  LA_CUDA(h, cudaMemcpy(sigma_out, s.sigma + row, sizeof(float), cudaMemcpyDeviceToHost), "factor read");
  auto widen = [&](const std::vector<unsigned char>& buf, size_t i) {
    float f;
    if (bf16) {
      uint16_t b;
      std::memcpy(&b, buf.data() + 2 * i, 2);
      const uint32_t u = static_cast<uint32_t>(b) << 16;
      std::memcpy(&f, &u, 4);
    } else {
      std::memcpy(&f, buf.data() + 4 * i, 4);
    }
    return f;
  };
  for (int j = 0; j < H; ++j) u_out[j] = widen(uu, j);
  for (int c = 0; c < D; ++c) v_out[c] = widen(vx, c);
  for (int c = 0; c < H; ++c) v_out[D + c] = widen(vh, c);
  return LSTM_APPROX_OK;
}

const char* lstm_approx_last_error(const lstm_approx_t* h) {
  if (!h) return "invalid handle (NULL)";
  return h->last_error.c_str();
}

void lstm_approx_destroy(lstm_approx_t* h) {
  if (!h) return;
  DeviceGuard dg(h->device);
  cudaStreamSynchronize(h->stream);
  clear_timing(h);
  if (h->timing.run0) cudaEventDestroy(h->timing.run0);
  if (h->timing.run1) cudaEventDestroy(h->timing.run1);
  for (LayerStore& s : h->layers) {
    cudaFree(s.Vx);
    cudaFree(s.Vh);
    cudaFree(s.U);
    cudaFree(s.sigma);
    cudaFree(s.bias);
    cudaFree(s.mask);
    for (int g = 0; g < 4; ++g) {
      cudaFree(s.xoff[g]);
      cudaFree(s.xidx[g]);
      cudaFree(s.xval[g]);
    }
    cudaFree(s.hoff);
    cudaFree(s.hcol);
    cudaFree(s.hval);
  }
  cudaFree(h->h_state);
  cudaFree(h->c_state);
  cudaFree(h->Px);
  cudaFree(h->seq);
  cudaFree(h->tau);
  cudaFree(h->err);
  cudaFree(h->proj_flags);
  if (h->err_host) cudaFreeHost(h->err_host);
  cudaFree(h->stage);
  cudaFree(h->gpart);
  cudaFree(h->x_bf16);
  cudaFree(h->seq_bf16);
  cudaFree(h->h_bf16);
  delete h;
}

int lstm_approx_query(const lstm_approx_t* h, int key, long long* value) {
  if (!h || !value) return LSTM_APPROX_EINVAL;
  switch (key) {
    case LSTM_APPROX_Q_LAUNCHES: *value = h->launches; return LSTM_APPROX_OK;
    case LSTM_APPROX_Q_LAST_PATH: *value = h->last_path; return LSTM_APPROX_OK;
    case LSTM_APPROX_Q_CLUSTER: *value = h->last_cluster; return LSTM_APPROX_OK;
    case LSTM_APPROX_Q_DEVICE_BYTES: *value = h->device_bytes; return LSTM_APPROX_OK;
    case LSTM_APPROX_Q_PERSISTENT_VARIANT: *value = h->last_variant; return LSTM_APPROX_OK;
    case LSTM_APPROX_Q_TENSOR_SEQ: *value = h->last_tensor_seq; return LSTM_APPROX_OK;
    default: return LSTM_APPROX_EINVAL;
  }
}

int lstm_approx_set_option(lstm_approx_t* h, int key, long long value) {
  if (!h) return LSTM_APPROX_EINVAL;
  switch (key) {
    case LSTM_APPROX_OPT_FORCE_PATH:
      if (value < 0 || value > 3) return fail(h, LSTM_APPROX_EINVAL, "bad path %lld", value);
      h->opt_force_path = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_CLUSTER:
      if (value != 0 && value != 1 && value != 2 && value != 4 && value != 8 && value != 16)
        return fail(h, LSTM_APPROX_EINVAL, "bad cluster size %lld", value);
      h->opt_cluster = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_TIMING:
      h->timing.on = value != 0;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_WAIT_LIMIT:
      if (value < 1) return fail(h, LSTM_APPROX_EINVAL, "wait limit must be >= 1 us");
      h->opt_wait_limit_us = value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_TEST_STALL:
      h->opt_test_stall = value != 0;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_XPROJ:
      if (value < 0 || value > 2) return fail(h, LSTM_APPROX_EINVAL, "bad projection choice %lld", value);
      h->opt_xproj = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_TAU_LAYOUT:
      if (value < 0 || value > 1) return fail(h, LSTM_APPROX_EINVAL, "bad tau' layout %lld", value);
      if (value == 1 && h->dtype != LSTM_APPROX_BF16)
        return fail(h, LSTM_APPROX_EINVAL, "the compressed tau' layout is for bf16 factors (the tensor path)");
      if (value == 1 && h->H > tau_sparse_max_h())
        return fail(h, LSTM_APPROX_EINVAL, "the compressed tau' layout takes H <= %d", tau_sparse_max_h());
      h->opt_tau_layout = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_TENSOR_SEQ:
      if (value < 0 || value > 1) return fail(h, LSTM_APPROX_EINVAL, "bad tensor launch choice %lld", value);
      h->opt_tensor_seq = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_LAUNCH_ORDER:
      if (value < 0 || value > 1) return fail(h, LSTM_APPROX_EINVAL, "bad launch order %lld", value);
      h->opt_launch_order = (int)value;
      return LSTM_APPROX_OK;
    case LSTM_APPROX_OPT_PERSISTENT_VARIANT:
      if (value < 0 || value > 2) return fail(h, LSTM_APPROX_EINVAL, "bad persistent variant %lld", value);
      h->opt_persistent_variant = (int)value;
      return LSTM_APPROX_OK;
    default: return fail(h, LSTM_APPROX_EINVAL, "unknown option %d", key);
  }
}

int lstm_approx_phase_times(lstm_approx_t* h, float* ms_out) {
  if (!h || !ms_out) return LSTM_APPROX_EINVAL;
  if (!h->timing.on || !h->timing.run0) return fail(h, LSTM_APPROX_ESTATE, "timing was not enabled for the last run");
  DeviceGuard dg(h->device);
  LA_CUDA(h, cudaStreamSynchronize(h->stream), "stream synchronise");
  ms_out[0] = ms_out[1] = ms_out[2] = 0.f;
  for (size_t i = 0; i + 1 < h->timing.ev.size(); i += 2) {
    float ms = 0.f;
    LA_CUDA(h, cudaEventElapsedTime(&ms, h->timing.ev[i], h->timing.ev[i + 1]), "event time");
    ms_out[h->timing.phase[i / 2]] += ms;
  }
  LA_CUDA(h, cudaEventElapsedTime(&ms_out[2], h->timing.run0, h->timing.run1), "event time");
  return LSTM_APPROX_OK;
}

int lstm_approx_plan(int dtype, int hidden, int T, int B, int K, const int* checkpoints, int J, int force_path,
                     int cluster, int persistent_variant, int* out, int n_out, char* msg, int msg_len) {
  if (msg && msg_len > 0) msg[0] = '\0';
  const int E = LSTM_APPROX_EINVAL;
  if (dtype != LSTM_APPROX_FP32 && dtype != LSTM_APPROX_BF16) return report(msg, msg_len, E, "bad dtype %d", dtype);
  if (hidden < 1 || T < 1 || B < 1 || K < 1)
    return report(msg, msg_len, E, "hidden=%d, T=%d, B=%d and K=%d must be >= 1", hidden, T, B, K);
  if (J < 0 || J > kMaxCheckpoints) return report(msg, msg_len, E, "J=%d outside [0, %d]", J, kMaxCheckpoints);
  if (J > 0 && !checkpoints) return report(msg, msg_len, E, "checkpoints is NULL with J=%d", J);
  Checkpoints ck;
  ck.n = J;
  for (int j = 0; j < kMaxCheckpoints; ++j) ck.k[j] = 0;
  for (int j = 0; j < J; ++j) {
    const int k = checkpoints[j];
    if (k < 1 || k > K) return report(msg, msg_len, E, "checkpoint %d = %d outside [1, K=%d]", j, k, K);
    if (j > 0 && k <= checkpoints[j - 1]) return report(msg, msg_len, E, "checkpoints must be strictly increasing");
    ck.k[j] = k;
  }
  if (force_path < 0 || force_path > 3) return report(msg, msg_len, E, "bad path %d", force_path);
  if (cluster != 0 && cluster != 1 && cluster != 2 && cluster != 4 && cluster != 8 && cluster != 16)
    return report(msg, msg_len, E, "bad cluster size %d", cluster);
  if (persistent_variant < 0 || persistent_variant > 2)
    return report(msg, msg_len, E, "bad persistent variant %d", persistent_variant);
  if (n_out < 0 || (n_out > 0 && !out)) return report(msg, msg_len, E, "out is NULL with n_out=%d", n_out);
  PersistentChoice pc;
  std::string why;
  const int path = select_path(dtype, hidden, K, T, ck, force_path, cluster, 0, persistent_variant, &pc, &why);
  if (path == 0) return report(msg, msg_len, E, "%s", why.c_str());
  int v[LSTM_APPROX_PLAN_ITEMS] = {};
  v[LSTM_APPROX_PLAN_PATH] = path;
  if (path == LSTM_APPROX_PATH_PERSISTENT) {
    v[LSTM_APPROX_PLAN_PERSISTENT_VARIANT] = pc.variant;
    v[LSTM_APPROX_PLAN_CLUSTER] = pc.CS;
    if (pc.variant == 1) {
      v[LSTM_APPROX_PLAN_TERMS_PER_CTA] = pc.ub.RA;
      v[LSTM_APPROX_PLAN_UNITS_PER_WARP] = pc.ub.upl;
      v[LSTM_APPROX_PLAN_TERMS_PER_LANE] = pc.ub.kpw;
      v[LSTM_APPROX_PLAN_VH_LAYOUT] = pc.ub.hc;
      v[LSTM_APPROX_PLAN_SMEM_BYTES] = (int)pc.ub.smem;
      v[LSTM_APPROX_PLAN_TMEM_COLUMNS] = pc.ub.tcols;
    } else {
      v[LSTM_APPROX_PLAN_TERMS_PER_CTA] = pc.ag.RA;
      v[LSTM_APPROX_PLAN_H_QUADS] = pc.ag.hq;
      v[LSTM_APPROX_PLAN_SMEM_BYTES] = (int)pc.ag.smem;
      v[LSTM_APPROX_PLAN_TMEM_COLUMNS] = pc.ag.tcols;
    }
  } else if (path == LSTM_APPROX_PATH_TENSOR) {
    int ns = 0, mt = 0;
    if (tc_seq_fits(hidden, B, K, ck, &ns, &mt, nullptr)) {
      v[LSTM_APPROX_PLAN_TENSOR_SEQ] = 1;
      v[LSTM_APPROX_PLAN_CLUSTER] = hidden / (128 * mt);
      v[LSTM_APPROX_PLAN_TAU_TILE_STREAMS] = ns;
      v[LSTM_APPROX_PLAN_GATE_TILE_STREAMS] = ns;
      v[LSTM_APPROX_PLAN_GATE_SPLITS] = 1;
      v[LSTM_APPROX_PLAN_TAU_SPLITS] = 1;
    } else {
      const TensorTiles tt = tensor_tiles(hidden, B, K, ck);
      v[LSTM_APPROX_PLAN_TAU_TILE_STREAMS] = tt.bnh;
      v[LSTM_APPROX_PLAN_GATE_TILE_STREAMS] = tt.nt;
      v[LSTM_APPROX_PLAN_GATE_SPLITS] = tt.ks;
      v[LSTM_APPROX_PLAN_TAU_SPLITS] = tt.sk;
    }
  }
  for (int i = 0; i < n_out; ++i) out[i] = i < LSTM_APPROX_PLAN_ITEMS ? v[i] : 0;
  return LSTM_APPROX_OK;
}

}  // extern "C"
