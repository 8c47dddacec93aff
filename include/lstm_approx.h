/*
 * lstm_approx.h -- progressive approximate-LSTM inference on sm_103a (GB300).
 *
 * The method (arXiv 1905.00689, Sec. III, Eq. 1): each LSTM gate's augmented
 * matrix W = [Wx Wh] (R x C, R = hidden size H, C = D + H) is replaced by a
 * sum of K pruned rank-1 terms sigma^(n) u^(n) prune(v^(n), NZ)^T taken from
 * the residual of the previous terms.  One timestep of one stream computes,
 * per gate g and with x~ = [x_t ; h_{t-1}] (Sec. III):
 *
 *     t_g[n] = prune(v_g^(n))^T x~                    (dot products, 2 NZ ops)
 *     y_g    = sum_{n<=K} sigma_g^(n) u_g^(n) t_g[n]    (2R + 1 ops per n)
 *
 * followed by the gate nonlinearities and the cell update of Sec. II
 * (i, f, o: logistic sigmoid; cell gate: tanh; c_t = f c_{t-1} + i g;
 * h_t = o tanh(c_t)).  Prefix sums over n <= k_j give the intermediate
 * ("progressive", Sec. I and Fig. 1b) outputs for a refinement depth k_j.
 *
 * Gate order everywhere in this interface: 0 = input (i), 1 = forget (f),
 * 2 = cell candidate (g), 3 = output (o).
 *
 * Conventions for every entry point:
 *   - returns an lstm_approx_status; nothing aborts, throws or prints;
 *   - arguments are checked before anything is launched; a call that
 *     returns LSTM_APPROX_EINVAL or LSTM_APPROX_ESTATE changes no state;
 *   - the text of the last error of a handle is lstm_approx_last_error();
 *   - there is no CPU fallback: without a usable sm_103a device every call
 *     that needs one returns LSTM_APPROX_ECUDA.
 */
#ifndef LSTM_APPROX_H
#define LSTM_APPROX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct lstm_approx lstm_approx_t; /* opaque; owned by the library */

enum lstm_approx_status {
  LSTM_APPROX_OK = 0,
  LSTM_APPROX_EINVAL = 1,   /* invalid argument (size, pointer, range) */
  LSTM_APPROX_ENOMEM = 2,   /* device or host allocation failed */
  LSTM_APPROX_ECUDA = 3,    /* CUDA error, or no usable sm_103a device */
  LSTM_APPROX_ETIMEOUT = 4, /* a bounded in-kernel wait ran out */
  LSTM_APPROX_ESTATE = 5    /* factors not set, or K above the depth set */
};

/* Storage/operand type of the factors u, v.  sigma, bias, the state and all
 * accumulation are fp32 in both.  BF16 is the tensor-core path. */
enum lstm_approx_dtype { LSTM_APPROX_FP32 = 0, LSTM_APPROX_BF16 = 1 };

/*
 * Create a handle for an L-layer stack (layer l >= 1 consumes layer l-1's
 * h_t as its input, so input_dims[l] must equal `hidden` for l >= 1).
 *
 *   out         receives the handle (set to NULL on failure)
 *   num_layers  L >= 1
 *   input_dims  host array [L]; input_dims[0] = D >= 1
 *   hidden      H = R >= 1 (Sec. III: W is R x C, C = D + H)
 *   max_rank    largest refinement depth K (N_steps, Sec. III) ever set
 *   max_batch   largest number of independent streams B passed to run
 *   dtype       enum lstm_approx_dtype
 *   cuda_stream cudaStream_t every launch and copy of this handle goes to;
 *               NULL = the legacy default stream.  Not owned.
 *
 * Allocates the device factor storage and per-stream state.  Errors:
 * EINVAL (sizes), ECUDA (no sm_103a device), ENOMEM.
 */
int lstm_approx_create(lstm_approx_t **out, int num_layers, const int *input_dims, int hidden,
                       int max_rank, int max_batch, int dtype, void *cuda_stream);

/*
 * Set the first K refinement terms of one gate (Eq. 1): for n < K,
 * sigma[n] u[n][:] prune(v[n])^T, where prune(v[n]) has the nz entries
 * v_val[n][m] at columns v_idx[n][m] of the augmented input x~ = [x; h]
 * (columns 0..D-1 multiply x_t, columns D..D+H-1 multiply h_{t-1}).
 *
 *   layer, gate  0 <= layer < L, 0 <= gate < 4 (i, f, g, o)
 *   K            1 <= K <= max_rank; later runs may use any depth <= K
 *   nz           1 <= nz <= C (the paper's NZ; may differ between gates)
 *   sigma        host [K] (fp64)
 *   u            host [K][H] row-major (fp64); u is not pruned
 *   v_idx        host [K][nz]; each row strictly increasing, in [0, C)
 *   v_val        host [K][nz] (fp64)
 *   bias         host [H] added to the gate pre-activation, or NULL = 0
 *                (the paper writes no bias; it is exact, not approximated)
 *
 * The library copies the arrays (the caller keeps ownership), rounds sigma
 * and bias to fp32 and u, v to the handle's dtype (fp64 -> fp32 -> bf16,
 * each round-to-nearest-even), packs them and uploads them with one
 * synchronous copy.  Errors: EINVAL (ranges, unsorted or out-of-range
 * indices), ECUDA.
 */
int lstm_approx_set_factors(lstm_approx_t *h, int layer, int gate, int K, int nz, const double *sigma,
                            const double *u, const int32_t *v_idx, const double *v_val,
                            const double *bias);

/*
 * Run the stack over a sequence: T timesteps of B independent streams at
 * refinement depth K, asynchronously on the handle's stream.
 *
 * All tensors are caller-owned DEVICE pointers, fp32, row-major:
 *   x        [T][B][D]          input sequence of layer 0
 *   h0, c0   [L][B][H] or NULL  initial state (NULL = zeros)
 *   out_h    [T][B][H]          top layer's h_t at depth K
 *   out_c    [L][B][H] or NULL  each layer's final c_T (for resuming)
 *   checkpoints host [J], strictly increasing, each in [1, K], J <= 8
 *            (may be NULL when J = 0)
 *   ckpt_h, ckpt_c [J][T][B][H] or NULL: the top layer's h_t, c_t when its
 *            refinement sums stop at depth k_j.  h_{t-1} and c_{t-1} always
 *            come from the full-depth chain, so one run yields every depth
 *            without recomputing shared prefixes (computation cut short as
 *            the time budget is hit, Sec. VI-B.1).
 *
 * 1 <= T, 1 <= B <= max_batch, 1 <= K <= the depth set for every gate.
 * Errors: EINVAL, ESTATE (a gate's factors missing or shallower than K),
 * ENOMEM (growing the T-dependent scratch), ECUDA (launch failure).
 * Kernel-side failures (a bounded wait that ran out) are reported by the
 * next lstm_approx_sync().  The first run at a new largest T*B (and, on
 * the bf16 tensor-core path with few streams, at a new largest B * H with
 * intermediate depths) may allocate scratch, synchronising the stream;
 * lstm_approx_run_static never allocates.
 */
int lstm_approx_run(lstm_approx_t *h, const float *x, int T, int B, int K, const float *h0,
                    const float *c0, float *out_h, float *out_c, const int *checkpoints, int J,
                    float *ckpt_h, float *ckpt_c);

/*
 * lstm_approx_run with every tensor a HOST pointer (same shapes and
 * meaning).  out_h, ckpt_h and ckpt_c in page-locked, mapped host memory
 * (cudaHostAlloc / cudaHostRegister, 16-byte aligned) are written in place
 * by the kernels; every other buffer is copied through device staging
 * buffers owned by the handle.  Waits for the stream before it
 * returns.  Returns what lstm_approx_run or lstm_approx_sync would.
 */
int lstm_approx_run_host(lstm_approx_t *h, const float *x, int T, int B, int K, const float *h0,
                         const float *c0, float *out_h, float *out_c, const int *checkpoints, int J,
                         float *ckpt_h, float *ckpt_c);

/*
 * Allocation-free variant of lstm_approx_run for one fp32 layer.  The paper
 * has no counterpart: this entry point exists for callers that must not
 * allocate device memory once running -- hard real-time control loops,
 * where cudaMalloc's unbounded latency (and device synchronisation) is not
 * acceptable and safety rules often forbid allocation after start-up, and
 * plug-ins inside a host framework whose own allocator owns all device
 * memory.  Such callers allocate factors, inputs and outputs up front and
 * pass them here; no handle is involved and nothing is allocated.
 *
 * Factors are caller-owned DEVICE arrays, fp32, in the library's packed
 * layout (row (g, k) = g*K + k, gate order i, f, g, o):
 *   Vx [4][K][D]  masked-dense pruned v over the x columns (zeros elsewhere)
 *   Vh [4][K][H]  masked-dense pruned v over the h columns (16-byte aligned)
 *   U  [4][H][K]  u_k[j] at (g*H + j)*K + k (16-byte aligned);  sigma [4][K];
 *                 bias [4][H] or NULL
 * x, h0, c0, out_h, out_c, checkpoints, J, ckpt_h, ckpt_c: as for
 * lstm_approx_run with L = 1 (device pointers, checkpoints on the host).
 * cuda_stream: cudaStream_t to run on (NULL = legacy default stream).
 * msg: optional host buffer of msg_len bytes that receives an error text.
 *
 * The scratch (the hoisted input projection, a status word, a zero bias)
 * is a fixed 4 MiB __device__ array inside the library, held by every GPU
 * that loads it until the process exits; calls needing more than
 * T*B*4*K + 4*H (rounded up to 64) + 64 <= 1048576 floats are rejected with
 * EINVAL.  The first call on a device looks up the array's address (do it
 * before any stream capture).  Every call shares the array and it keeps the
 * last call's contents, so calls that overlap on the GPU race.  The call is
 * synchronous: it waits for the stream and returns OK, EINVAL (sizes,
 * alignment, a shape the persistent kernel cannot hold), ECUDA or ETIMEOUT.
 */
int lstm_approx_run_static(const float *Vx, const float *Vh, const float *U, const float *sigma,
                           const float *bias, int D, int H, int K, const float *x, int T, int B,
                           const float *h0, const float *c0, float *out_h, float *out_c,
                           const int *checkpoints, int J, float *ckpt_h, float *ckpt_c,
                           void *cuda_stream, char *msg, int msg_len);

/*
 * Dense comparator: the LSTM of Sec. II with the full gate matrices
 * W_g = [Wx_g Wh_g] (no approximation), for one fp32 layer, on the same kind
 * of persistent cluster kernel as the approximate path (one cluster per
 * stream; Wh held in tensor memory for the whole launch; one h exchange per
 * timestep).  It serves as the dense baseline against which the speed-up of
 * the approximation is measured (the paper compares its approximate design
 * with dense designs on each platform, Sec. VI-B, Table I).
 *
 *   Wx    DEVICE [4H][D] fp32, row g*H + j = the input part of row j of W_g
 *   Wh    DEVICE [4H][H] fp32, row g*H + j = the recurrent part of that row
 *   bias  DEVICE [4][H] or NULL;  D >= 1, 1 <= H <= 512
 *   x, h0, c0, out_h, out_c: as lstm_approx_run with L = 1 (DEVICE, fp32)
 *   workspace  DEVICE buffer of at least
 *              lstm_approx_dense_workspace_bytes(H, T, B) bytes, 256-byte
 *              aligned, owned by the caller (the hoisted Wx x_t, a status
 *              word and the projection's completion flags); it must not be
 *              used by another call in flight
 *
 * For one stream the recurrence is launched before the input projection and
 * waits (bounded) for flags the projection raises, as lstm_approx_run does
 * (LSTM_APPROX_OPT_LAUNCH_ORDER): the two kernels must be able to run at the
 * same time, which tools that run one kernel at a time do not allow.
 *   cuda_stream  cudaStream_t (NULL = legacy default stream)
 *   msg   optional host buffer of msg_len bytes for an error text
 *
 * Synchronous: waits for the stream.  Returns OK, EINVAL (sizes, NULL,
 * workspace too small or misaligned), ECUDA or ETIMEOUT (a bounded
 * in-kernel wait ran out).  Allocates nothing.
 */
int lstm_approx_dense_run(const float *Wx, const float *Wh, const float *bias, int D, int H,
                          const float *x, int T, int B, const float *h0, const float *c0,
                          float *out_h, float *out_c, void *workspace, size_t workspace_bytes,
                          void *cuda_stream, char *msg, int msg_len);
/* Workspace bytes lstm_approx_dense_run needs for (H, T, B); 0 for invalid sizes. */
size_t lstm_approx_dense_workspace_bytes(int H, int T, int B);
/* Launch order of lstm_approx_dense_run for every later call in the process,
 * as LSTM_APPROX_OPT_LAUNCH_ORDER: 0 = automatic (recurrence first for one
 * stream), 1 = projection first (what tools that run one kernel at a time
 * need).  Returns OK or EINVAL (another value). */
int lstm_approx_dense_set_launch_order(int order);

/*
 * Wait for the handle's stream and report kernel-side status: OK, or
 * ETIMEOUT when a bounded in-kernel wait ran out since the last sync (the
 * outputs of that run are then invalid; the status word is cleared), or
 * ECUDA.
 */
int lstm_approx_sync(lstm_approx_t *h);

/*
 * Read back the pruning mask of term k (0 <= k < K set) of (layer, gate)
 * from the device-resident packed representation.  idx_out: host [C]
 * (capacity C = D_layer + H); *nz_out receives the count.  The indices are
 * ascending and must equal the v_idx row passed to set_factors bit for bit.
 */
int lstm_approx_get_mask(lstm_approx_t *h, int layer, int gate, int k, int32_t *idx_out, int *nz_out);

/*
 * Read back term k (0 <= k < K set) of (layer, gate) as the device storage
 * holds it, i.e. after the rounding of lstm_approx_set_factors: sigma, u
 * and prune(v) of Eq. 1 (Sec. III), each stored value widened exactly to
 * fp32 (a bf16 value is the upper half of its fp32 pattern).
 *
 *   sigma_out  host [1]
 *   u_out      host [H]
 *   v_out      host [C] (C = D_layer + H): dense, zero at pruned columns
 *
 * Synchronises the handle's stream.  Errors: EINVAL (range, NULL), ECUDA.
 * Used to check the stored values bit for bit against the rounding rule.
 */
int lstm_approx_get_term(lstm_approx_t *h, int layer, int gate, int k, float *sigma_out, float *u_out,
                         float *v_out);

/* Text of the handle's last error ("" if none).  Static text for NULL. */
const char *lstm_approx_last_error(const lstm_approx_t *h);

/* Free the handle and everything it owns (waits for its stream).  NULL-safe. */
void lstm_approx_destroy(lstm_approx_t *h);

/* ---- introspection and tuning (tests, benchmarks) ---------------------- */

enum lstm_approx_query_key {
  LSTM_APPROX_Q_LAUNCHES = 0,    /* kernels launched by this handle so far */
  LSTM_APPROX_Q_LAST_PATH = 1,   /* recurrence path of the last run (enum below) */
  LSTM_APPROX_Q_CLUSTER = 2,     /* CTAs per cluster of the last persistent run */
  LSTM_APPROX_Q_DEVICE_BYTES = 3, /* device bytes currently held by the handle */
  LSTM_APPROX_Q_PERSISTENT_VARIANT = 4, /* persistent kernel of the last persistent run
                                          (1 or 2, see LSTM_APPROX_OPT_PERSISTENT_VARIANT) */
  LSTM_APPROX_Q_TENSOR_SEQ = 5   /* 1 if the last tensor-path layer ran as one launch
                                    for all timesteps (see LSTM_APPROX_OPT_TENSOR_SEQ) */
};
enum lstm_approx_path {
  LSTM_APPROX_PATH_NONE = 0,
  LSTM_APPROX_PATH_SIMT = 1,       /* per-timestep CUDA-core kernels */
  LSTM_APPROX_PATH_PERSISTENT = 2, /* one persistent cluster launch over all T (fp32) */
  LSTM_APPROX_PATH_TENSOR = 3      /* tcgen05/TMEM GEMMs with fused epilogues (bf16) */
};
int lstm_approx_query(const lstm_approx_t *h, int key, long long *value);

enum lstm_approx_option_key {
  LSTM_APPROX_OPT_FORCE_PATH = 0,   /* 0 = automatic, else an lstm_approx_path */
  LSTM_APPROX_OPT_CLUSTER = 1,      /* 0 = automatic, else 1, 2, 4, 8 or 16 */
  LSTM_APPROX_OPT_TIMING = 2,       /* 1 = record CUDA events around each phase */
  LSTM_APPROX_OPT_WAIT_LIMIT = 3,   /* wall-time limit of every bounded in-kernel
                                       wait, in microseconds (default 2000000) */
  LSTM_APPROX_OPT_TEST_STALL = 4,   /* 1 = next persistent run waits on a signal
                                       nobody sends (exercises ETIMEOUT) */
  LSTM_APPROX_OPT_PERSISTENT_VARIANT = 5, /* persistent kernel: 0 = automatic (the
                                       one-exchange kernel where it fits and
                                       H x terms per CTA <= 16384, else the
                                       per-unit-block one),
                                       1 = per-unit-block kernel (two cluster
                                       exchanges per timestep, any H <= 1024),
                                       2 = one-exchange kernel (H <= 512,
                                       K <= 256, cluster of 4, 8 or 16) */
  LSTM_APPROX_OPT_XPROJ = 6, /* input projection of the small-batch fp32 path
                               (T*B <= 32): 0 = automatic (compressed when v
                               keeps at most 1/8 of the x columns), 1 =
                               masked-dense rows, 2 = compressed rows */
  LSTM_APPROX_OPT_TAU_LAYOUT = 7, /* the tensor path's recurrent projection tau'
                               (bf16 factors): 0 = masked-dense v rows on the
                               tensor cores (default: faster at every shape
                               measured), 1 = v's kept h entries (compressed
                               rows) on the CUDA cores, H <= 1280 */
  LSTM_APPROX_OPT_TENSOR_SEQ = 8, /* tensor path: 0 = automatic (one launch per
                               tile of streams for all T timesteps where the
                               layer fits: K <= 32, H = 256, 512 or 1024,
                               intermediate depths multiples of 16 or >= K,
                               masked-dense tau'), 1 = two launches per
                               timestep */
  LSTM_APPROX_OPT_LAUNCH_ORDER = 9 /* batch-1 fp32 path with the per-unit-block
                               kernel: 0 = automatic (the recurrence is
                               launched before its input projection and
                               waits, bounded, for flags the projection
                               raises: the two kernels must be able to run
                               at the same time), 1 = projection first,
                               recurrence as its programmatic dependent.
                               Tools that run kernels one at a time (kernel
                               profilers, memory checkers) need 1; with 0
                               under such a tool each run ends in
                               LSTM_APPROX_ETIMEOUT after the wait limit.
                               Phase timing (LSTM_APPROX_OPT_TIMING) and
                               runs on a stream being captured into a CUDA
                               graph use 1; a handle created with
                               CUDA_LAUNCH_BLOCKING=1 in the environment
                               starts at 1. */
};
int lstm_approx_set_option(lstm_approx_t *h, int key, long long value);

/*
 * Device milliseconds of the last run's phases, from CUDA events recorded
 * on the handle's stream when LSTM_APPROX_OPT_TIMING is 1 (waits for the
 * stream).  ms_out[0] = input projection (hoisted over all T), ms_out[1] =
 * recurrence (all layers, all T), ms_out[2] = whole run.
 */
int lstm_approx_phase_times(lstm_approx_t *h, float *ms_out);

/*
 * Which kernels lstm_approx_run takes for one layer of this shape, by the
 * same rules as the run: the path, the persistent kernel with its cluster
 * size and on-chip layout, and the tensor-core tiles and term splits.  Host
 * only: no handle, no device, nothing launched.
 *
 *   dtype        enum lstm_approx_dtype of the factors
 *   hidden       H >= 1;  T, B, K >= 1: timesteps, streams, refinement depth
 *   checkpoints  host array [J] of the layer's intermediate depths k_j
 *                (strictly increasing, in [1, K]); NULL when J = 0
 *   force_path, cluster, persistent_variant
 *                the values of LSTM_APPROX_OPT_FORCE_PATH, _CLUSTER and
 *                _PERSISTENT_VARIANT (0 = automatic)
 *   out          host array [n_out]; out[i] receives item i of enum
 *                lstm_approx_plan_item (0 where an item does not apply to
 *                the chosen path, and for i >= LSTM_APPROX_PLAN_ITEMS)
 *   msg          optional host buffer of msg_len bytes for an error text
 *
 * Returns OK, or EINVAL for invalid arguments and for a forced path or
 * kernel that cannot take the shape (where lstm_approx_run returns EINVAL).
 * The input projection's kernel, which also depends on the factors' masks,
 * is not reported.
 */
enum lstm_approx_plan_item {
  LSTM_APPROX_PLAN_PATH = 0,               /* enum lstm_approx_path */
  LSTM_APPROX_PLAN_PERSISTENT_VARIANT = 1, /* 1 per-unit-block, 2 one-exchange kernel */
  LSTM_APPROX_PLAN_CLUSTER = 2,            /* CTAs per stream */
  LSTM_APPROX_PLAN_TERMS_PER_CTA = 3,      /* coefficient rows a CTA owns (per-unit-block:
                                              gate-major rows of all four gates; one-exchange:
                                              terms of one gate) */
  LSTM_APPROX_PLAN_UNITS_PER_WARP = 4,     /* per-unit-block: hidden units per warp, 1..16 */
  LSTM_APPROX_PLAN_TERMS_PER_LANE = 5,     /* per-unit-block: terms per lane, 1..8 */
  LSTM_APPROX_PLAN_VH_LAYOUT = 6,          /* per-unit-block: 0 V_h in shared memory, 1 V_h and
                                              U in tensor memory, 2 V_h in tensor memory at 32
                                              values per lane */
  LSTM_APPROX_PLAN_H_QUADS = 7,            /* one-exchange: h quads per lane, 1, 2 or 4 */
  LSTM_APPROX_PLAN_SMEM_BYTES = 8,         /* persistent: dynamic shared memory per CTA */
  LSTM_APPROX_PLAN_TMEM_COLUMNS = 9,       /* persistent: tensor-memory columns per CTA */
  LSTM_APPROX_PLAN_TAU_TILE_STREAMS = 10,  /* tensor path: streams per tile of the tau' GEMM */
  LSTM_APPROX_PLAN_GATE_TILE_STREAMS = 11, /* tensor path: streams per tile of the gate GEMM */
  LSTM_APPROX_PLAN_GATE_SPLITS = 12,       /* tensor path: term-axis splits of the gate GEMM */
  LSTM_APPROX_PLAN_TENSOR_SEQ = 13,        /* tensor path: 1 = one launch per tile of streams for
                                              all T (then CLUSTER = H / 128 CTAs per tile and both
                                              tile items = the streams per tile), 0 = two launches
                                              per timestep */
  LSTM_APPROX_PLAN_TAU_SPLITS = 14,        /* tensor path: CTAs of a cluster over which the tau'
                                              GEMM splits its reduction axis (H), 1 = none */
  LSTM_APPROX_PLAN_ITEMS = 15
};
int lstm_approx_plan(int dtype, int hidden, int T, int B, int K, const int *checkpoints, int J,
                     int force_path, int cluster, int persistent_variant, int *out, int n_out,
                     char *msg, int msg_len);

#ifdef __cplusplus
}
#endif
#endif /* LSTM_APPROX_H */
