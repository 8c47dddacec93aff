// Internal declarations shared by the C-ABI implementation and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <string>
#include <vector>

#include "../../include/lstm_approx.h"

namespace lstm_approx_impl {

constexpr int kMaxCheckpoints = 8;

struct Checkpoints {
  int n;
  int k[kMaxCheckpoints];
};

// Opaque storage of one CUtensorMap (128 bytes, 64-byte aligned).
struct alignas(64) TcMap {
  unsigned char bytes[128];
};

// Device factor storage of one layer.  Row (g, k) of the packed matrices is
// storage row g * Ks + k ("gate-major"), rows k >= K_set are zero.
//   Vx   [4*Ks][ldx]  masked-dense pruned v over the x columns (ldx >= D)
//   Vh   [4*Ks][ldh]  masked-dense pruned v over the h columns (ldh >= H)
//   U    [4][H][Ks] (u_k[j] at (g*H + j)*Ks + k): K-major, so the terms a
//        lane or an MMA operand needs are contiguous
//   sigma [4][Ks] fp32, bias [4][H] fp32
//   mask [4*Ks][mask_words] bit c set <=> column c of x~ is kept
struct LayerStore {
  int D = 0, C = 0, ldx = 0;
  void* Vx = nullptr;
  void* Vh = nullptr;
  void* U = nullptr;
  float* sigma = nullptr;
  float* bias = nullptr;
  uint32_t* mask = nullptr;
  int mask_words = 0;
  int Kset[4] = {0, 0, 0, 0};
  int nz[4] = {0, 0, 0, 0};
  // compressed x part (fp32 factors): device CSR per gate and its host offsets
  int* xoff[4] = {nullptr, nullptr, nullptr, nullptr};
  int* xidx[4] = {nullptr, nullptr, nullptr, nullptr};
  float* xval[4] = {nullptr, nullptr, nullptr, nullptr};
  size_t xcap[4] = {0, 0, 0, 0};  // entries allocated in xidx / xval
  std::vector<int> xoff_h[4];
  bool maps_ready = false;  // tensor maps of Vx, Vh, U (bf16 path), built on first use
  TcMap map_vx, map_vh, map_u;
  TcMap map_vx_p[3], map_vh_p[3];  // the same with boxes of 8, 16, 32 rows (packed gates)
  TcMap map_u64;                   // U as 32-term boxes of 128 rows, 64-byte swizzled (one-launch kernel)
  // compressed recurrent part of v (bf16 factors): CSR over storage rows g*Ks + k
  int* hoff = nullptr;
  int* hcol = nullptr;
  float* hval = nullptr;
  size_t hcap = 0;                 // entries allocated
  bool hcsr_dirty = false;         // the host copies below changed since the last upload
  std::vector<int> hrows[4];       // per gate: host copy of its rows' kept h columns, counts per row
  std::vector<float> hvals[4];
  std::vector<int> hcount[4];
};

struct Timing {
  bool on = false;
  std::vector<cudaEvent_t> ev;  // pairs (start, stop) per phase launch
  std::vector<int> phase;       // 0 = input projection, 1 = recurrence
  cudaEvent_t run0 = nullptr, run1 = nullptr;
};

}  // namespace lstm_approx_impl

struct lstm_approx {
  int L = 0, H = 0, ldh = 0, Kmax = 0, Ks = 0, max_batch = 0, dtype = 0;
  cudaStream_t stream = nullptr;
  int device = 0, sm_count = 0;
  std::vector<lstm_approx_impl::LayerStore> layers;

  // state and scratch
  float* h_state = nullptr;   // [L][max_batch][H]
  float* c_state = nullptr;   // [L][max_batch][H]
  size_t cap_TB = 0;          // capacity (T*B) of the T-dependent scratch
  float* Px = nullptr;        // [T*B][4*Ks] hoisted input projection
  float* seq = nullptr;       // [T*B][H] output sequence of a lower layer
  void* tau = nullptr;        // [max_batch][4*Ks] refinement coefficients (fp32; on the tensor path
                              // the bf16 pair planes [2][B][4*Ks], the same bytes)
  void* x_bf16 = nullptr;     // [2][T*B][ldx of layer 0] bf16 pair of the input (tensor path)
  void* seq_bf16 = nullptr;   // [2][T*B][ldh] bf16 pair of the sequence between layers (tensor path)
  void* h_bf16 = nullptr;     // [2][B][ldh] bf16 pair of the h operand (tensor path)
  int* err = nullptr;         // device status word (0 = ok)
  int* err_host = nullptr;    // pinned host copy of it, read after the stream synchronises
  unsigned* proj_flags = nullptr;  // [kProjFlags] completion flags of a projection launched after the recurrence
  unsigned proj_epoch = 0;         // the value the last such launch wrote

  // staging for lstm_approx_run_host
  size_t stage_bytes = 0;
  float* gpart = nullptr;     // raw gate sums of a term-split gate GEMM (tensor path), grown on demand
  size_t gpart_bytes = 0;
  char* stage = nullptr;

  // options and counters
  int opt_force_path = 0, opt_cluster = 0, opt_persistent_variant = 0;
  int opt_xproj = 0;  // 0 automatic, 1 masked-dense, 2 compressed (fp32, T*B <= 32)
  int opt_tau_layout = 0;  // tensor path's tau': 0 masked-dense (tensor cores), 1 compressed (CUDA cores)
  int opt_tensor_seq = 0;  // tensor path: 0 one launch for all timesteps where the layer fits, 1 per-step launches
  int opt_launch_order = 0;  // batch-1 persistent path: 0 recurrence before its projection where it applies, 1 after
  long long opt_wait_limit_us = 2000000;
  int opt_test_stall = 0;
  long long launches = 0;
  int last_path = 0, last_cluster = 0, last_variant = 0;
  int last_tensor_seq = 0;  // 1 if the last tensor-path layer ran as one launch for all timesteps
  long long device_bytes = 0;
  lstm_approx_impl::Timing timing;
  std::string last_error;
};

namespace lstm_approx_impl {

// ---- generic CUDA-core kernels (any size, both factor types) -------------

// out[n][srow(r)] = sum_c A[srow(r)][c] * Bm[n][c] for run rows r < 4K, where
// srow(r) = (r / K) * Ks + r % K.  mode 0 stores the sum; mode 1 stores
// sigma[srow] * (sum + P[n][srow]).
cudaError_t launch_rows_gemm(const void* A, bool a_bf16, int lda, int K, int Ks, const float* Bm, int ldb,
                             int N, int Kdim, float* out, int ldo, int mode, const float* sigma,
                             const float* P, int ldp, cudaStream_t s);

// Same product for few columns (N = T*B <= 256, in chunks of 32): clusters
// split the D axis, rows are staged by asynchronous copies and the chunk
// sums pushed to their owner CTA (deterministic).  Needs D % 8 == 0 and
// 16-byte aligned base pointers and rows; a push that does not arrive
// within limit_ns sets *err.  max_split caps the CTAs per cluster along D
// (1: one CTA per row tile and column chunk).
bool xproj_cluster_fits(int N, int D, const void* A, int lda, const float* X, int ldxin, bool a_bf16);

// Compressed x part of the pruned v (fp32 factors): per gate, the kept x
// columns of row k are entries off[g][k] .. off[g][k+1] of idx[g] / val[g].
struct SparseXRows {
  const int* off[4];
  const int* idx[4];
  const float* val[4];
};
// The same product from the compressed rows, for T*B <= 32 columns.
cudaError_t launch_xproj_sparse(const SparseXRows& sr, int K, int Ks, const float* X, int ldxin, int N, float* out,
                                int ldo, cudaStream_t s);
// Launched after the recurrence kernel that reads its output (see
// run_device): the projection then starts as a programmatic dependent of
// that kernel, may take every SM the recurrence leaves free, and each of its
// CTAs writes `epoch` to flags[its linear index] (release, GPU scope) once
// its outputs are stored; the recurrence waits for all of them before its
// first read of P.
struct XprojSignal {
  unsigned* flags = nullptr;
  unsigned epoch = 0;
};
cudaError_t launch_xproj_cluster(const void* A, bool a_bf16, int lda, int K, int Ks, const float* X, int ldxin,
                                 int N, int D, float* out, int ldo, int* err, long long limit_ns, cudaStream_t s,
                                 int max_split, const XprojSignal* sig = nullptr);
// CTAs of that launch (one flag each when it signals).
int xproj_cluster_ctas(int K, int N, int D, int max_split);
// Loads the kernel that launch_xproj_cluster would launch for N columns
// (lazy module loading would otherwise delay a launch made while the
// recurrence runs until that recurrence has finished).
cudaError_t xproj_cluster_prepare(bool a_bf16, int N);
constexpr int kProjFlags = 2048;  // flags of one signalling projection launch

// One timestep of the refinement sums over u (a3), the intermediate outputs
// (a6) and the cell update (a4) for B streams.
struct CellArgs {
  const void* U;
  bool u_bf16;
  long long gs, ks, js;  // element strides of U over (gate, k, unit)
  int K, Ks, H, B;
  const float* tau;      // [B][ldt], coefficient of (g, k) at g*Ks + k
  int ldt;
  const float* bias;     // [4][H]
  float* c_state;        // [B][H], read then overwritten
  float* h_state;        // [B][H], overwritten
  float* out_h;          // [B][H] or null
  Checkpoints ck;
  float* ckpt_h;         // element (j, b, unit) at j*ck_stride + b*H + unit, or null
  float* ckpt_c;
  long long ck_stride;
};
cudaError_t launch_cell_step(const CellArgs& a, cudaStream_t s);

// ---- persistent cluster kernels (fp32 factors, one cluster per stream) -----

struct PersistentPlan {
  int CS = 0;        // CTAs per cluster
  int RA = 0;        // coefficient rows per CTA (multiple of 4)
  int UB = 0;        // hidden units per CTA (ceil(H / CS) rounded up to 4)
  int upl = 0;       // hidden units per warp (1, 2, 4, 8 or 16; four warps per gate)
  int kpw = 0;       // refinement terms per lane (1, 2, 4 or 8)
  int hc = 0;        // 16-value chunks of h per lane in the recurrent product (1 or 2)
  int tcols = 0;     // tensor-memory columns holding the CTA's V_h rows
  size_t smem = 0;   // dynamic shared memory bytes
};

// Chooses a plan; returns false (with a reason) if the shape does not fit.
bool plan_persistent(int H, int K, int T, const Checkpoints& ck, int want_cs, int sm_count,
                     PersistentPlan* plan, std::string* why);

struct PersistentArgs {
  const float* Vh;     // [4*Ks][ldh]
  const float* U;      // [4][H][Ks]
  const float* sigma;  // [4][Ks]
  const float* bias;   // [4][H]
  const float* P;      // [T][B][4*Ks]
  const float* h0;     // [B][H] or null
  const float* c0;     // [B][H] or null
  float* out_h;        // [T][B][H]
  float* c_last;       // [B][H] or null
  float* ckpt_h;       // [J][T][B][H] or null
  float* ckpt_c;
  int* err;
  int H, K, Ks, ldh, T, B;
  Checkpoints ck;
  long long wait_limit_ns;
  int test_stall;
  // Non-null when the projection that writes P is launched after this kernel
  // (XprojSignal): the kernel then waits until proj_flags[0, proj_nflags)
  // all hold proj_epoch instead of waiting for the grid before it.
  const unsigned* proj_flags;
  int proj_nflags;
  unsigned proj_epoch;
};
cudaError_t launch_persistent(const PersistentPlan& plan, const PersistentArgs& a, cudaStream_t s);

// One-exchange variant (H <= 512, K <= 256): each CTA owns a range of one
// gate's terms, and the CTAs swap partial gate sums once per timestep.
struct PersistentAgPlan {
  int CS = 0;       // CTAs per cluster (4, 8 or 16)
  int RA = 0;       // terms per CTA (a multiple of 4, at most 64)
  int Kp = 0;       // terms per gate rounded up to CS
  int UB = 0;       // units per output block (a multiple of 4)
  int nmask = 0;    // intermediate depths that cut a CTA's range
  int tcols = 0;    // tensor-memory columns (V_h rows, then U)
  int hq = 0;       // h quads per lane in the recurrent product (1, 2 or 4)
  size_t smem = 0;  // dynamic shared memory bytes
};
bool plan_persistent_ag(int H, int K, const Checkpoints& ck, int want_cs, PersistentAgPlan* plan,
                        std::string* why);
cudaError_t launch_persistent_ag(const PersistentAgPlan& plan, const PersistentArgs& a, cudaStream_t s);

// Either persistent kernel: variant 1 = per-unit-block kernel (two
// exchanges per step), 2 = one-exchange kernel; 0 picks the one-exchange
// kernel where it fits and a CTA's share (H x terms per CTA) is small, else
// the per-unit-block one.
struct PersistentChoice {
  int variant = 0;
  int CS = 0;
  PersistentPlan ub;
  PersistentAgPlan ag;
};
bool choose_persistent(int H, int K, int T, const Checkpoints& ck, int want_cs, int sm_count, int variant,
                       PersistentChoice* c, std::string* why);
cudaError_t launch_persistent_choice(const PersistentChoice& c, const PersistentArgs& a, cudaStream_t s);

// ---- tensor-core path (bf16, tcgen05 / TMEM / TMA) -----------------------
// Activations (x, h, tau') enter the MMAs as bf16 pairs hi = bf16(a),
// lo = bf16(a - hi), stored as two planes: the hi plane of R rows, then the
// lo plane of R rows, so one tensor map of 2R rows covers both.

// 2-D K-major bf16 tensor [rows][inner] with `pitch_bytes` between rows, as
// TMA tiles of box_rows rows of one swizzled row each: 64 inner elements
// with 128-byte swizzling, or 32 with 64-byte swizzling.
bool tc_make_map(TcMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t pitch_bytes,
                 uint32_t box_rows, uint32_t swizzle_bytes = 128);
int tc_rows_tile_n(int n_cols, int row_tiles);  // column tile of launch_tc_rows
int tc_gates_tile_n(int H, int B);               // stream tile of launch_tc_gates

struct TcRowsArgs {
  int Kdim;          // reduction length (D of the layer, or H)
  int K, Ks;         // refinement depth of the run; gate stride of the packed rows
  int kt_per_gate;   // 128-row tiles per gate: ceil(K / 128)
  int rpg;           // 0, or packed gates (K <= rpg, rpg 8, 16 or 32): one tile of the four gates'
                     // first rpg rows, whose factor map has boxes of rpg rows
  int N;             // valid columns (T*B for the projection, B for tau')
  int b_plane;       // rows of one plane of the activation's map (its lo plane starts there)
  int mode;          // 0: P[n][row] = sum; 1: tau[n][row] = pair of sigma[row] (sum + P[n][row]), 0 for k >= K
  float* P;          // [N][ldp]
  int ldp;
  const float* sigma;
  __nv_bfloat16* tau;  // planes [2][N][ldt]: hi, then lo at tau + tau_plane
  int ldt;
  long long tau_plane;
  int* err;
  long long limit_ns;
  // mode 1 only: the reduction axis split over the sk CTAs of a cluster
  // (grid z), nkb_per 64-element chunks each; each CTA then finishes
  // 128 / sk rows of the tile from all sk partial sums (1: no split)
  int sk;
  int nkb_per;
};
// `bn` (64, 128 or 256) must match the box rows of Bm's map.
cudaError_t launch_tc_rows(const TcMap& A, const TcMap& Bm, const TcRowsArgs& a, int n_cols, int bn, cudaStream_t s);
// The projection (mode 0) with packed gates from fp32 activations: Xf maps
// the fp32 [N][Kdim] input in boxes of 32 columns x 64 rows (tc_make_map_f32),
// and the kernel forms the bf16 pair itself (64 columns per tile).
cudaError_t launch_tc_rows_xf32(const TcMap& A, const TcMap& Xf, const TcRowsArgs& a, int n_cols, cudaStream_t s);
// 2-D fp32 tensor [rows][inner] as unswizzled TMA boxes of 32 inner elements x box_rows rows.
bool tc_make_map_f32(TcMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t pitch_bytes,
                     uint32_t box_rows);

struct TcGatesArgs {
  int H, K, Ks, B;
  int nkb;                  // 64-term chunks: ceil(K / 64)
  int tau_rows;             // rows of one plane of tau's map (B: the lo plane starts there)
  const __nv_bfloat16* U;   // factor U [4][H][Ks] and the stored tau' pair [2][B][ldt]: the reduce kernel
  const __nv_bfloat16* tau; // adds the terms of an intermediate depth past its last 16-term slice boundary
  int ldt;                  // from these on the CUDA cores
  long long tau_plane;
  const float* bias;        // [4][H]
  float* c_state;           // [B][H] fp32, c_{t-1} in, c_t out
  __nv_bfloat16* h_bf16;    // planes [2][B][ldh]: h_t out (next step's operand), lo at h_bf16 + h_plane
  int ldh;
  long long h_plane;
  float* out_h;             // [B][H] fp32 h_t (this timestep) or null
  __nv_bfloat16* seq_bf16;  // [B][ldh] h_t for the next layer (this timestep; lo at seq_bf16 + seq_plane) or null
  long long seq_plane;
  Checkpoints ck;           // intermediate depths
  float* ckpt_h;            // element (j, n, unit) at j*ck_stride + n*H + unit (this timestep) or null
  float* ckpt_c;
  long long ck_stride;
  int* err;
  long long limit_ns;
  // split over the term axis (ks > 1, grid z = ks): CTA z accumulates the
  // 64-term chunks [z nkb_per, (z+1) nkb_per) and writes its raw gate sums,
  // element (slot, g, n, unit) at ((slot*4 + g)*B + n)*H + unit of `part`:
  // slot z for its whole range, slot ks + j at an intermediate depth k_j that
  // ends inside it.  launch_tc_gates then runs the sum over the splits and
  // the cell update of Sec. II in a second kernel.
  int ks, nkb_per;
  float* part;
  bool raw;                 // raw-sum mode: ks > 1, or an intermediate depth that is not a multiple of 16
};
// `nt` (32, 64 or 128) must match the box rows of Tau's map.
cudaError_t launch_tc_gates(const TcMap& U, const TcMap& Tau, const TcGatesArgs& a, int nt, cudaStream_t s);
// Term-axis splits for a gate GEMM of `tiles` CTAs over nkb 64-term chunks
// (1: no split); *nkb_per receives the chunks per split.
int tc_gates_splits(int tiles, int nkb, int* nkb_per);

// One launch per tile of NS streams for all T timesteps of a layer (bf16
// factors, K <= 32, H = 256, 512 or 1024): a cluster of CS CTAs, CTA r
// owning hidden units [UC r, UC r + UC) (UC = 128 or 256), keeps its columns of
// the packed V_h, its rows of U, its h_t and c_t on chip; per step the CTAs
// add their partial tau' over distributed shared memory and exchange the
// bf16 pair of tau'.
struct TcSeqArgs {
  int H, K, Ks, B, T;
  int rpg;                  // packed rows per gate: 8, 16 or 32 (K <= rpg)
  int cs;                   // CTAs per cluster, H / (128 units per tile x unit tiles per CTA)
  const float* P;           // [T*B][ldp] hoisted input projection, column g*Ks + k
  int ldp;
  const float* sigma;       // [4][Ks]
  const float* bias;        // [4][H]
  const float* h0;          // [B][H] or null (zero)
  const float* c0;          // [B][H] or null (zero)
  float* out_h;             // element (t, n, unit) at (t*B + n)*H + unit, or null
  float* c_last;            // [B][H] c after the last step, or null
  __nv_bfloat16* seq_bf16;  // pair of h_t for the next layer: (t*B + n)*ldh + unit, lo plane at + seq_plane; or null
  int ldh;
  long long seq_plane;
  Checkpoints ck;           // intermediate depths: multiples of 16, or >= K
  float* ckpt_h;            // element (j, t, n, unit) at j*ck_stride + (t*B + n)*H + unit, or null
  float* ckpt_c;
  long long ck_stride;
  int* err;
  long long limit_ns;
  int test_stall;           // 1: CTA 0 of the first tile withholds its first partial tau' (the waits run out)
};
// Whether a layer of this shape takes the one-launch kernel; *ns receives
// its streams per tile (32 or 64), *mt its 128-unit tiles per CTA (1 or 2).
bool tc_seq_fits(int H, int B, int K, const Checkpoints& ck, int* ns, int* mt, std::string* why);
// Vh_p: the packed V_h map with boxes of rpg rows; U64: U as 32-term boxes of
// 128 rows with 64-byte swizzling.
cudaError_t launch_tc_seq(const TcMap& Vh_p, const TcMap& U64, const TcSeqArgs& a, int ns, int mt, cudaStream_t s);

// Compressed tau' (the recurrent part of the pruned v as (column, value)
// entries per storage row g*Ks + k, entries off[row] .. off[row + 1]) on the
// CUDA cores, for the tensor path; H <= tau_sparse_max_h().
struct TauSparseArgs {
  const int* off;
  const int* col;            // h column of each entry
  const float* val;          // the entry (the bf16-stored value, widened)
  const float* sigma;        // [4][Ks]
  const float* P;            // [B][ldp] P_t
  int ldp;
  const __nv_bfloat16* h;    // pair planes [2][B][ldh] of h_{t-1}
  int ldh;
  long long h_plane;
  __nv_bfloat16* tau;        // pair planes [2][B][ldt]
  int ldt;
  long long tau_plane;
  int H, K, Ks, B;
  int Rp;                    // K rounded up to 64: rows [K, Rp) of each gate store zero
};
cudaError_t launch_tau_sparse(const TauSparseArgs& a, cudaStream_t s);
int tau_sparse_max_h();

cudaError_t launch_to_bf16(const float* x, int N, int D, __nv_bfloat16* out, int ld, cudaStream_t s);
cudaError_t launch_tc_init_state(const float* h0, const float* c0, int B, int H, __nv_bfloat16* h_bf16, int ldh,
                                 float* c_state, cudaStream_t s);

// ---- error codes written to the device status word -----------------------
constexpr int kErrWaitTimeoutA = 1;
constexpr int kErrWaitTimeoutB = 2;
constexpr int kErrTcTimeout = 3;

}  // namespace lstm_approx_impl
