/*
 * lionmuon.h -- C ABI of the GB300 (sm_103a) LionMuon optimizer-step library.
 *
 * LionMuon (arXiv 2605.19811, Algorithm 1) keeps one momentum buffer M per
 * parameter.  At step t it forms the interpolated direction
 *     G_hat = beta1 * M_{t-1} + (1 - beta1) * G_t
 * and, when t mod P == 0, takes the Muon step
 *     W <- W - eta_M * (0.2 sqrt(max(m,n)) * NS_K(G_hat) + lambda * W)
 * (Table 5 gives K_NS = 5 and the 0.2 sqrt(max(m,n)) scaling), otherwise the
 * Lion step
 *     W <- W - eta_L * (sign(G_hat) + lambda * W);
 * every step then updates M_t = beta2 * M_{t-1} + (1 - beta2) * G_t.
 * Vectors (rows == 1 or cols == 1) take the Lion step on every step.
 * NS_K is the odd-polynomial Newton-Schulz approximation of msign(X) = U V^T
 * (Section 2): X <- X / (||X||_F + eps), then K times
 *     A = X X^T ;  B = b A + c A A ;  X <- a X + B X
 * run on the wide orientation (X^T for a tall matrix).
 *
 * Conventions for every call:
 *   - Device pointers are CUDA device memory of the current device; host
 *     pointers are ordinary host memory.  Tensors are dense, row-major,
 *     contiguous and 16-byte aligned (LM_ERR_ALIGN otherwise).  A tensor
 *     whose data is host memory (page-locked or not) or another device's
 *     memory is refused with LM_ERR_INVALID_ARG (managed memory is
 *     accepted); lm_step checks each gradient pointer the first time it
 *     sees it.
 *   - Calls return an lm_status; nothing unwinds across the ABI.  Arguments
 *     are validated before any work is enqueued: on an error return nothing
 *     was enqueued and no state changed.  An asynchronous CUDA error surfaces
 *     as LM_ERR_CUDA from a later call.  lm_last_error() gives a one-line
 *     description of the most recent error on the calling thread.
 *   - Work is enqueued on the caller's stream (a cudaStream_t passed as
 *     void*, NULL = legacy default stream).  lm_step never synchronises and
 *     never copies device to host.  One state is driven by one stream at a
 *     time.
 */
#ifndef LIONMUON_H
#define LIONMUON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LM_OK = 0,
  LM_ERR_INVALID_ARG = 1, /* bad count, shape, hyper-parameter or NULL pointer */
  LM_ERR_DTYPE = 2,       /* unsupported dtype or grads/params dtype mismatch */
  LM_ERR_ALIGN = 3,       /* a data pointer is not 16-byte aligned */
  LM_ERR_OOM = 4,         /* device allocation failed */
  LM_ERR_CUDA = 5,        /* a CUDA runtime/driver call failed */
  LM_ERR_UNSUPPORTED = 6, /* no sm_103a device, or a size beyond a stated limit */
  LM_ERR_TIMEOUT = 7      /* a bounded device-side wait gave up */
} lm_status;

typedef enum { LM_F32 = 0, LM_BF16 = 1 } lm_dtype;

/* A dense row-major tensor.  rows == 1 or cols == 1 means a vector.
 * rows * cols may be 0 (an empty parameter is accepted and skipped). */
typedef struct {
  void* data;
  int64_t rows;
  int64_t cols;
  lm_dtype dtype;
} lm_tensor;

/* Device status flags read by lm_get_status. */
#define LM_FLAG_NONFINITE 0x1u /* a matrix direction had a non-finite Frobenius norm */
#define LM_FLAG_TIMEOUT 0x2u   /* a bounded device wait gave up */
#define LM_FLAG_GUARD 0x4u     /* states created with LM_DEBUG=1: a workspace guard band was overwritten */

/* Environment switches, read by lm_create for that state (host side; the
 * device code is the same):
 *   LM_DEBUG=1          a 256-byte guard band after every part of the state's
 *                       workspace, filled with a fixed pattern and compared by
 *                       lm_get_status (LM_FLAG_GUARD if one was overwritten)
 *   LM_NVTX=1           NVTX ranges named after the kernel families around the
 *                       library's launches
 *   LM_FAULT=oom        lm_create returns LM_ERR_OOM as if the device allocation
 *                       had failed (to exercise callers' error paths)
 *   LM_NS_FORCE_FP32=1  the fp32 Newton-Schulz path whatever ns_precision says
 *   LM_NS_TILES=wide    bf16 Newton-Schulz tiles of two 256-column blocks per
 *                       CTA pair (the default is one block); same results bit
 *                       for bit, slower on the GPT-style parameter sets
 *   LM_PDL=0            no programmatic dependent launch between the
 *                       Newton-Schulz launches (same results)
 *   LM_NS_FOLD=0        bf16 Newton-Schulz keeps a X as a separate term of
 *                       X' = a X + B X; by default an iteration with |a| < 4
 *                       folds a into the diagonal of the stored B (results
 *                       within the same tolerance, slightly closer to the
 *                       fp64 iteration for the constant quintic)
 *   LM_WAIT_LIMIT_NS=n  limit of every bounded device wait in ns (default 5 s;
 *                       also read by lm_msign_ns and lm_msign_ns_noalloc).  A
 *                       wait that runs out raises LM_FLAG_TIMEOUT; every kernel
 *                       of this state (or call) launched after it reads the
 *                       flag at entry and does nothing, so a step stops within
 *                       about one limit and writes no parameter after the
 *                       give-up, until lm_get_status clears the flag. */

/* Hyper-parameters: the Require line of Algorithm 1 plus the NS reading.
 * beta1, beta2 in [0, 1); eta_* >= 0; weight_decay >= 0;
 * period >= 1, or 0 for P = infinity (never Muon);
 * ns_steps in [0, 64]; ns_eps >= 0; shape_scale >= 0;
 * ns_precision LM_BF16 (tensor-core bf16 GEMMs, fp32 accumulate), LM_F32
 * (fp32 CUDA-core GEMMs) or LM_NS_F32_TC (fp32 values on the tensor cores:
 * each fp32 operand is stored exactly as three bf16 pieces hi + mid + lo and
 * a product sums the six piece products down to order 2^-16, accumulated in
 * fp32; the fast fp32 mode, at the cost of six bf16 products per product).
 * ns_coeffs: NULL for the same (ns_a, ns_b, ns_c) in every NS iteration, or
 * 3 * ns_steps finite values (a_k, b_k, c_k), k = 0 .. ns_steps - 1, for
 * iteration-dependent odd polynomials X <- a_k X + (b_k A + c_k A^2) X, the
 * form of the minimax (Polar Express) and Chebyshev-type msign iterations
 * Section 2 names.  The table is caller memory read only by lm_create, which
 * copies it; ns_a/ns_b/ns_c are then ignored. */
typedef struct {
  double beta1, beta2;
  double eta_muon, eta_lion;
  double weight_decay;
  int64_t period;
  int ns_steps;
  double ns_a, ns_b, ns_c;
  double ns_eps;
  double shape_scale;
  int ns_precision;
  const double* ns_coeffs;
  /* Update rule of 1-D parameters (rows == 1 or cols == 1): LM_VECTOR_LION
   * (Algorithm 1's Lion step on every step, the default) or LM_VECTOR_ADAMW,
   * the AdamW fallback Section 3 uses for biases and norm gains:
   *   m = b1 m + (1-b1) g;  v = b2 v + (1-b2) g^2;  w -= lr wd w;
   *   w -= lr / (1 - b1^(t+1)) * m / (sqrt(v) / sqrt(1 - b2^(t+1)) + eps)
   * with the momentum buffer as m, one more fp32 buffer v per 1-D parameter,
   * and t the step index passed to lm_step (t + 1 updates so far).
   * adamw_lr >= 0 (Table 5: 1e-3), adamw_beta1/2 in [0, 1) (Table 5:
   * 0.8, 0.999), adamw_eps > 0 (1e-8), adamw_weight_decay >= 0 (0.1). */
  int vector_rule;
  double adamw_lr, adamw_beta1, adamw_beta2, adamw_eps, adamw_weight_decay;
  /* Choice between the Muon and Lion step for matrices: LM_SCHEDULE_PERIOD
   * (Algorithm 1: Muon iff t mod period == 0, the default) or
   * LM_SCHEDULE_STABLE_RANK, the adaptive rule of Appendix G: on every step
   * a matrix takes the Muon step iff the stable rank of its momentum buffer
   * M_{t-1}, ||M||_F^2 / sigma_1_hat^2, is at most srank_alpha * min(m, n)
   * (a zero buffer takes Muon); sigma_1_hat^2 is the Rayleigh quotient of
   * M^T M after srank_iters - 1 power-iteration steps from a SplitMix64
   * start vector (seed srank_seed), srank_iters reads of M in all.
   * srank_alpha > 0 (Appendix G sweeps 0.002 .. 0.01; default 0.01),
   * srank_iters in [1, 64] (default 5); period is then ignored, and matrices
   * may have at most 16384 columns.  When the matrices' column counts need
   * more than one power-iteration launch per pass, lm_create also creates
   * two non-blocking streams (freed by lm_destroy) on which lm_step runs
   * those launches, forked from and joined back to the caller's stream by
   * events: work enqueued on the caller's stream after lm_step still sees
   * all of it. */
  int schedule;
  double srank_alpha;
  int srank_iters;
  uint64_t srank_seed;
  /* Layer-sharded Muon (Section 5.4: a Muon step needs each matrix whole,
   * a Lion step is element-wise).  With shard_world > 1 this state is rank
   * shard_rank of shard_world ranks that each hold all parameters, the
   * (already reduced) gradients and the momentum.  Every matrix has one owner
   * rank (lm_shard_owners).  On a Muon step a rank runs the momentum, Newton-
   * Schulz and parameter write only for the matrices it owns, and for the
   * others the momentum update M = beta2 M + (1 - beta2) G alone; the caller
   * then copies each matrix from its owner to the other ranks (a broadcast
   * per matrix, on Muon steps only).  Lion steps and 1-D parameters run the
   * same on every rank and exchange nothing.  The Newton-Schulz workspace
   * covers the owned matrices only.  shard_world 0 or 1: no sharding (the
   * default 1); otherwise shard_world <= 4096, 0 <= shard_rank < shard_world,
   * and schedule must be LM_SCHEDULE_PERIOD. */
  int shard_rank;
  int shard_world;
} lm_config;

#define LM_SCHEDULE_PERIOD 0
#define LM_SCHEDULE_STABLE_RANK 1

/* ns_precision / precision value for the three-piece tensor-core fp32 mode
 * (LM_BF16 and LM_F32 are the other two). */
#define LM_NS_F32_TC 2

#define LM_VECTOR_LION 0
#define LM_VECTOR_ADAMW 1

typedef struct lm_state lm_state; /* opaque */

/* Fill *cfg with the paper's defaults: beta (0.9, 0.99) (Table 5, Lion),
 * (eta_M, eta_L) = (3e-3, 2e-5) (Appendix E, LionMuon P=2), lambda = 0.1
 * (Table 5), P = 2, K_NS = 5 (Table 5), quintic NS coefficients
 * (3.4445, -4.7750, 2.0315) with eps 1e-7 (the paper gives none; this is the
 * stated reading), shape_scale 0.2 (Table 5), ns_precision LM_BF16. */
void lm_config_default(lm_config* cfg);

/* sizeof(lm_config) as this library was built: a binding that lays the
 * struct out itself compares it with its own size before any call that
 * takes an lm_config (a mismatch would make those calls read or write past
 * the caller's struct). */
size_t lm_config_size(void);

/* Owner rank of each parameter under layer sharding over `world` ranks
 * (lm_config::shard_world, Section 5.4): matrices (rows, cols >= 2) are
 * dealt out whole, largest Newton-Schulz cost 3 s^2 l + s^3 first (s, l the
 * smaller and larger dimension; the FLOPs of one iteration counting the
 * symmetric products once), each to the rank with the least cost so far (the
 * lowest such rank), ties in cost taken in parameter order; 1-D parameters
 * get -1 (every rank updates them).  The same inputs give the same owners on
 * every rank.  Reads only the shapes (no device access; usable without a
 * GPU).  owner: n ints of host memory.
 * Errors: LM_ERR_INVALID_ARG (NULL, n < 1, world outside [1, 4096]). */
lm_status lm_shard_owners(const lm_tensor* params, int n, int world, int* owner);

/* Create an optimizer state over n parameter tensors (Algorithm 1, Require:
 * W_0 given, M_{-1} = 0).  params[i].data is caller-owned device memory that
 * the state borrows for its lifetime and updates in place; dtype LM_BF16 or
 * LM_F32.  The state allocates and zeroes one fp32 momentum buffer per
 * parameter plus the Newton-Schulz workspace, and records the shapes.
 * Errors: LM_ERR_INVALID_ARG (n < 1, NULL, bad cfg), LM_ERR_DTYPE,
 * LM_ERR_ALIGN, LM_ERR_OOM, LM_ERR_CUDA, LM_ERR_UNSUPPORTED (device is not
 * sm_103). */
lm_status lm_create(const lm_tensor* params, int n, const lm_config* cfg,
                    void* cuda_stream, lm_state** out);

/* One LionMuon step t >= 0 (Algorithm 1 body).  grads[i] must have the shape
 * and dtype of params[i]; they are read-only device memory borrowed until the
 * enqueued work completes.  Muon iff period != 0 and t % period == 0.
 * The work may be captured into a CUDA graph (stream capture on a non-NULL
 * stream): the graph keeps the gradient pointers, the learning rates and t
 * of the capture.  Under the Lion/Muon rules t matters only mod period, so
 * a graph of step k (0 <= k < period) serves every later step t with
 * t % period == k; the AdamW rule for vectors uses t itself (bias
 * correction).
 * After a captured step every later lm_step re-uploads its gradient pointers.
 * Replays and lm_step calls on one state must not overlap on the GPU.
 * Errors: LM_ERR_INVALID_ARG (n mismatch, t < 0, shape mismatch, NULL),
 * LM_ERR_DTYPE, LM_ERR_ALIGN, LM_ERR_CUDA. */
lm_status lm_step(lm_state* s, const lm_tensor* grads, int n, int64_t t,
                  void* cuda_stream);

/* Change the two learning rates (a caller-driven schedule); takes effect for
 * the next lm_step.  Errors: LM_ERR_INVALID_ARG (NULL, negative, non-finite). */
lm_status lm_set_lr(lm_state* s, double eta_muon, double eta_lion);

/* The branch each parameter took in the last lm_step, and under
 * LM_SCHEDULE_STABLE_RANK the stable-rank estimate behind it (Appendix G).
 * took_muon (n entries, or NULL): 1 where parameter i took the Muon step.
 * srank (n entries, or NULL): ||M_{t-1}||_F^2 / sigma_1_hat^2 of matrix i
 * (0 for a zero buffer), NaN for 1-D parameters and under the fixed period.
 * Host memory; synchronises the state's last stream.  Errors:
 * LM_ERR_INVALID_ARG (NULL state, n differs from the parameter count, no
 * step taken yet), LM_ERR_CUDA. */
lm_status lm_get_selection(lm_state* s, int n, unsigned char* took_muon, double* srank);

/* Change the AdamW learning rate of 1-D parameters (LM_VECTOR_ADAMW); takes
 * effect for the next lm_step.  Errors: LM_ERR_INVALID_ARG (NULL, negative,
 * non-finite). */
lm_status lm_set_adamw_lr(lm_state* s, double lr);

/* AdamW second moment v of 1-D parameter i (LM_VECTOR_ADAMW only): a
 * read-only fp32 device view of the parameter's shape, owned by the state;
 * lm_set_second_moment copies src (fp32 device memory of that shape) into it
 * on cuda_stream, for checkpoint / resume together with lm_set_momentum.
 * Errors: LM_ERR_INVALID_ARG (NULL, index out of range, parameter i has no
 * second moment, shape mismatch), LM_ERR_DTYPE, LM_ERR_ALIGN, LM_ERR_CUDA. */
lm_status lm_get_second_moment(const lm_state* s, int i, lm_tensor* view);
lm_status lm_set_second_moment(lm_state* s, int i, const lm_tensor* src,
                               void* cuda_stream);

/* Newton-Schulz approximation of msign (Section 2): out = NS_steps(in) with
 * coefficients (a, b, c), normalisation X / (||X||_F + eps), iterated on the
 * wide orientation, with no 0.2 sqrt(max(m,n)) scaling.  in and out are
 * device tensors of equal shape (rows, cols >= 2 each), dtype LM_BF16 or
 * LM_F32 (may differ).  precision LM_BF16 uses the tensor-core path, LM_F32
 * the fp32 CUDA-core path, LM_NS_F32_TC fp32 values on the tensor cores (as
 * for lm_config::ns_precision).  Allocates its workspace with stream-ordered
 * allocation on cuda_stream and frees it the same way.  A testing entry
 * point: it synchronises cuda_stream before it returns, to read its own
 * status word.
 * Errors: LM_ERR_INVALID_ARG, LM_ERR_DTYPE, LM_ERR_ALIGN, LM_ERR_OOM,
 * LM_ERR_CUDA, LM_ERR_TIMEOUT (a bounded device wait gave up; the kernels
 * after it did nothing and out holds no result). */
lm_status lm_msign_ns(const lm_tensor* in, lm_tensor* out, int steps, double a,
                      double b, double c, double eps, int precision,
                      void* cuda_stream);

/* lm_msign_ns with iteration-dependent coefficients: iteration k uses
 * (coeffs[3k], coeffs[3k+1], coeffs[3k+2]); coeffs holds 3 * steps finite
 * host values, read before the call returns (NULL is allowed only for
 * steps == 0).  Everything else as lm_msign_ns. */
lm_status lm_msign_ns_coeffs(const lm_tensor* in, lm_tensor* out, int steps,
                             const double* coeffs, double eps, int precision,
                             void* cuda_stream);

/* The same computation as lm_msign_ns, for callers that cannot allocate
 * device memory while they run: for example a program whose device memory is
 * fully budgeted up front by its own allocator, or a latency-critical loop in
 * which cudaMalloc/cudaFree (cudaFree synchronises the device) are not
 * acceptable.  This entry point allocates nothing.  Its workspace is a fixed
 * 64 MiB area inside the library (a static device array that every GPU which
 * loads the library holds until the process exits); a matrix whose workspace
 * does not fit is rejected with LM_ERR_UNSUPPORTED and a message giving the
 * bytes needed.  The workspace is (2 s_p l_p + 2 s_p^2) e bytes plus about
 * 1 KB of descriptors, 24 bytes per 32768 elements of the matrix and 16
 * bytes per tile, where s = min(rows, cols), l = max(rows, cols); with
 * precision LM_BF16: e = 2, s_p = s rounded up to 128, l_p = l rounded up
 * to 256 (so 2048 x 5120 fits, 2048 x 8192 does not); with LM_F32: e = 4 and
 * both rounded up to 128.  The caller still provides in and out.
 * The first call on a device (and the first after its context was
 * destroyed and made again, as by cudaDeviceReset) looks up the area's
 * device address on that device (cudaGetSymbolAddress); make that first call
 * before any stream capture.  All calls share the one area, which keeps the
 * last call's data: each call clears what must start at zero, and calls
 * whose GPU work may overlap (unordered streams or threads) race on the area
 * and must be serialised by the caller.  Unlike lm_msign_ns the call does not
 * synchronise: lm_msign_ns_noalloc_status reports its status word.
 * Arguments and errors as for lm_msign_ns, except that precision is LM_BF16
 * or LM_F32 only.
 * The paper has no counterpart of this call; it is a deployment variant. */
lm_status lm_msign_ns_noalloc(const lm_tensor* in, lm_tensor* out, int steps,
                              double a, double b, double c, double eps,
                              int precision, void* cuda_stream);

/* Status of the last lm_msign_ns_noalloc call on the current device:
 * synchronises cuda_stream (the stream of that call), then stores its status
 * word (LM_FLAG_*) in *device_flags, without allocating.  Returns
 * LM_ERR_TIMEOUT when a bounded device wait of that call gave up (out then
 * holds no result).  The paper has no counterpart; deployment variant.
 * Errors: LM_ERR_INVALID_ARG (NULL), LM_ERR_CUDA, LM_ERR_TIMEOUT. */
lm_status lm_msign_ns_noalloc_status(uint32_t* device_flags, void* cuda_stream);

/* A read-only view of parameter i's momentum buffer (fp32, the shape of
 * params[i], device memory owned by the state).  For checkpointing and tests.
 * Errors: LM_ERR_INVALID_ARG (NULL, i out of range). */
lm_status lm_get_momentum(const lm_state* s, int i, lm_tensor* view);

/* Overwrite parameter i's momentum from src (device, fp32, same shape),
 * enqueued on cuda_stream (resume from a checkpoint: restore M and pass the
 * same t).  Errors: LM_ERR_INVALID_ARG, LM_ERR_DTYPE, LM_ERR_ALIGN,
 * LM_ERR_CUDA. */
lm_status lm_set_momentum(lm_state* s, int i, const lm_tensor* src,
                          void* cuda_stream);

/* Synchronise the state's last stream, then return and clear the device
 * status flags (LM_FLAG_*).  Errors: LM_ERR_INVALID_ARG, LM_ERR_CUDA. */
lm_status lm_get_status(lm_state* s, uint32_t* device_flags);

/* Bytes of persisted optimizer state: exactly 4 * sum |W_i| (one fp32
 * momentum buffer per parameter, Section 3 Implementation notes), plus
 * 4 * sum |w| over 1-D parameters with LM_VECTOR_ADAMW (their second
 * moments).  Returns 0 for NULL. */
size_t lm_state_bytes(const lm_state* s);

/* Bytes of transient device workspace the state holds (Newton-Schulz
 * buffers, tables).  Returns 0 for NULL. */
size_t lm_workspace_bytes(const lm_state* s);

/* Synchronise the state's last stream and free everything it owns.  NULL is
 * a no-op. */
void lm_destroy(lm_state* s);

/* Static text for a status code. */
const char* lm_status_string(lm_status st);

/* Description of the most recent error returned on the calling thread
 * (static storage of the library; "" if none). */
const char* lm_last_error(void);

/* Number of CUDA kernels this library has launched in this process (a
 * monotonically increasing counter, for launch accounting by benchmarks). */
uint64_t lm_kernel_launch_count(void);

/* Failure-detection probe: launches one thread that waits, with the bounded
 * wait every device-side wait of this library uses, on a barrier that nothing
 * signals.  When limit_ns passes the kernel records LM_FLAG_TIMEOUT and
 * returns normally, leaving the context usable.  Synchronises cuda_stream and
 * stores the flags in *device_flags.  Returns LM_ERR_TIMEOUT when the wait gave
 * up (the expected outcome), LM_OK otherwise.  The paper has no counterpart;
 * it tests the library's own error path.  Errors: LM_ERR_INVALID_ARG (NULL,
 * limit_ns outside (0, 1e10]), LM_ERR_UNSUPPORTED, LM_ERR_CUDA. */
lm_status lm_probe_bounded_wait(uint64_t limit_ns, uint32_t* device_flags,
                                void* cuda_stream);

/* Per-kernel-family timing, measured with CUDA events recorded on the
 * launching stream around every kernel launch of lm_step while enabled. */
typedef enum {
  LM_KERNEL_LION = 0,          /* Lion step (all params, or vectors on Muon steps) */
  LM_KERNEL_MOMENTUM_NORM = 1, /* Muon: G_hat, ||G_hat||_F^2, M update, X0 */
  LM_KERNEL_NS_GRAM = 2,       /* Newton-Schulz: A = X X^T */
  LM_KERNEL_NS_POLY = 3,       /* Newton-Schulz: B = b A + c A A */
  LM_KERNEL_NS_APPLY = 4,      /* Newton-Schulz: X <- a X + B X */
  LM_KERNEL_FINALIZE = 5,      /* Muon: parameter write */
  LM_KERNEL_OTHER = 6,         /* gradient-pointer upload, norm reset */
  LM_KERNEL_ADAMW = 7,         /* AdamW on 1-D parameters (LM_VECTOR_ADAMW) */
  LM_KERNEL_SRANK = 8,         /* stable-rank selection: power iteration, decision */
  LM_KERNEL_FAMILIES = 9
} lm_kernel_family;

typedef struct {
  double ms[LM_KERNEL_FAMILIES];          /* summed event-to-event time */
  uint64_t launches[LM_KERNEL_FAMILIES];  /* launches timed */
} lm_profile;

/* Turn event timing on (on != 0) or off for the state's later lm_step calls
 * (steps captured into a CUDA graph are not timed).
 * Errors: LM_ERR_INVALID_ARG. */
lm_status lm_profile_enable(lm_state* s, int on);

/* Synchronise the state's last stream, add up the recorded events into *out
 * and, if reset != 0, clear them.  Errors: LM_ERR_INVALID_ARG, LM_ERR_CUDA. */
lm_status lm_profile_read(lm_state* s, lm_profile* out, int reset);

#ifdef __cplusplus
}
#endif

#endif /* LIONMUON_H */
