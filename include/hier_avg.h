/*
 * hier_avg.h - C ABI of the Hier-AVG data-parallel hot path on one GPU.
 *
 * Hier-AVG is Algorithm 1 (Sec. 3.1) of Zhou & Cong, "A Distributed Hierarchical
 * Averaging SGD Algorithm: Trading Local Reductions for Global Reductions".  All
 * P learners live on one GPU as rows of a learner-indexed fp32 parameter matrix
 * [P, ld]; the paper's local and global reductions become in-memory segmented and
 * full means over the learner axis.
 *
 * Conventions shared by every call
 *   - Every pointer argument named *_dev is a device pointer on the current CUDA
 *     device; *_host pointers are host memory.  Nothing is freed by the library
 *     that the caller passed in; the caller keeps ownership of all buffers and
 *     must keep them alive while work that uses them is in flight.
 *   - All compute calls are asynchronous on the CUDA stream given to them (or
 *     bound to the handle); a NULL stream is the legacy default stream.  Only
 *     hier_avg_losses, hier_avg_check, hier_avg_round_host and the profile read
 *     synchronise.
 *   - No call changes the calling thread's current CUDA device: a call that runs
 *     work on the handle's device makes it current and restores the caller's.
 *   - Every call returns HA_OK (0) or a negative status; nothing aborts.
 *     hier_avg_strerror() names a status, hier_avg_last_error() gives the
 *     message of the handle's last failure.
 *   - K2 counts LOCAL AVERAGES per global average (the paper's beta, Sec. 3.1);
 *     the paper's global interval in local steps is K1 * K2.
 */
#ifndef HIER_AVG_H
#define HIER_AVG_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define HA_OK            0
#define HA_EINVAL       (-1)  /* an argument is out of range or inconsistent        */
#define HA_ENOMEM       (-2)  /* a caller-provided buffer is too small              */
#define HA_ECUDA        (-3)  /* a CUDA runtime or driver call failed               */
#define HA_ESTATE       (-4)  /* call out of order (e.g. a step before bind)        */
#define HA_ETIMEOUT     (-5)  /* a bounded device-side wait expired; see check      */
#define HA_EUNSUPPORTED (-6)  /* valid request the library does not implement       */

#define HA_PREC_FP32 0        /* every product in fp32 on CUDA cores                */
#define HA_PREC_BF16 1        /* bf16 GEMM operands, fp32 accumulate, fp32 master   */

/* ---------------------------------------------------------------------------
 * Stateless averaging on a caller's learner-indexed buffer.
 *
 * w_dev: P rows of D fp32 values, row j starting at w_dev + j * ld (ld >= D).
 * The mean of n rows is their sum in the canonical adjacent-pair tree order
 * (levels h = 1, 2, 4, ...: v[i] += v[i+h] for i = 0, 2h, ..., an unpaired
 * element carried up), then one correctly rounded fp32 division by n; no FMA,
 * no flush of subnormals.  The result is therefore bit-reproducible.
 * Errors: HA_EINVAL if P < 1, D < 0, ld < D, S < 1, P % S != 0 or w_dev is NULL
 * with D > 0; HA_ECUDA if the launch fails.  D = 0 is a no-op.
 * ------------------------------------------------------------------------- */

/* Local average, Algorithm 1 (Sec. 3.1) "locally average and synchronize":
 * every row of cluster g (rows [g*S, (g+1)*S)) is replaced by the cluster mean. */
int hier_avg_local_average_buffer(float* w_dev, int64_t P, int64_t S, int64_t D,
                                  int64_t ld, void* stream);

/* Global average, Algorithm 1 (Sec. 3.1) "globally average and synchronize"
 * together with the synchronisation at the top of the next round: every row is
 * replaced by the mean over all P rows. */
int hier_avg_global_average_buffer(float* w_dev, int64_t P, int64_t D, int64_t ld,
                                   void* stream);

/* The last local average of a round followed by the global average (Algorithm 1,
 * end of the b-loop then the global step), in one pass over memory.  Bit-identical
 * to hier_avg_local_average_buffer followed by hier_avg_global_average_buffer. */
int hier_avg_local_global_average_buffer(float* w_dev, int64_t P, int64_t S, int64_t D,
                                         int64_t ld, void* stream);

/* ---------------------------------------------------------------------------
 * Handle API: P learners of a ReLU MLP d_0 -> d_1 -> ... -> d_L trained with
 * mean softmax cross-entropy (the learner objective; Algorithm 1 leaves F open).
 * ------------------------------------------------------------------------- */
typedef struct hier_avg hier_avg;

/* Validate a configuration and create a handle (host memory only, no GPU work).
 *   P, S, K1, K2, lr, B : Sec. 2 notation (K2 = local averages per round), S | P
 *   dims[0..n_dims-1]   : d_0 .. d_L, n_dims = L + 1 >= 2, every d >= 1
 *   precision           : HA_PREC_FP32 or HA_PREC_BF16
 * Errors: HA_EINVAL for P, S, K1, K2, B < 1, P % S != 0, non-finite lr, bad dims or
 * precision; HA_EUNSUPPORTED for a shape the kernels do not cover (BF16: B > 64 or
 * an input width d_0 .. d_{L-1} not a multiple of 8; either: P > 65535). */
int hier_avg_create(int P, int S, int K1, int K2, float lr, int B, const int* dims,
                    int n_dims, int precision, hier_avg** out);

/* Free the handle (never the caller's buffers).  NULL is a no-op. */
void hier_avg_destroy(hier_avg* h);

/* Parameter layout of one learner row.  *D = parameters per learner,
 * *ld = padded row length in floats (multiple of 64; padding stays zero).
 * offsets (2 * L entries, may be NULL): offsets[2l] = start of W_{l+1}
 * ([d_{l+1}, d_l] row-major), offsets[2l+1] = start of b_{l+1} ([d_{l+1}]). */
int hier_avg_param_layout(const hier_avg* h, int64_t* D, int64_t* ld, int64_t* offsets);

/* Bytes of device workspace hier_avg_bind needs: a step's scratch and, for the bf16
 * path with S > 1, the cluster means [P / S, ld] fp32 that hier_avg_round's local
 * averages write. */
int hier_avg_workspace_bytes(const hier_avg* h, int64_t* bytes);

/* Attach device memory (all borrowed, caller-owned) and the stream:
 *   params_dev    [P, ld] fp32, the learner replicas (initialised by the caller,
 *                 e.g. one w0 copied to every row: Algorithm 1 starts from one
 *                 global parameter)
 *   workspace_dev >= hier_avg_workspace_bytes bytes, 256-byte aligned; zeroed here
 *   X_dev         [P, N, d_0] per-learner samples, bf16 for HA_PREC_BF16, fp32
 *                 for HA_PREC_FP32; y_dev [P, N] int32 labels in [0, d_L)
 * Builds the TMA descriptors.  Resets the step counter to 0.
 * Errors: HA_EINVAL (NULL pointer, N < 1, misaligned params or workspace),
 * HA_ENOMEM (workspace too small), HA_ECUDA. */
int hier_avg_bind(hier_avg* h, float* params_dev, void* workspace_dev,
                  int64_t workspace_bytes, const void* X_dev, const int32_t* y_dev,
                  int64_t N, void* stream);

/* One local SGD step of every learner, Algorithm 1 inner loop (Sec. 3.1):
 * w_j <- w_j - (lr / B) * sum_s grad f(w_j; xi_{j,s}).  Learner j at step t uses
 * rows (t*B + s) mod N of its own data.  Then t <- t + 1.  HA_ESTATE before bind. */
int hier_avg_step(hier_avg* h);

/* Local average of the bound parameters (see hier_avg_local_average_buffer). */
int hier_avg_local_average(hier_avg* h);

/* Global average of the bound parameters (see hier_avg_global_average_buffer). */
int hier_avg_global_average(hier_avg* h);

/* One global round of Algorithm 1: K2 x (K1 x step, local average), then the
 * global average; the last local average is fused with the global one
 * (bit-identical to doing them in turn).  The other local averages write each
 * cluster's mean once, into the workspace, and the step that follows reads every
 * learner's parameters from its cluster's mean (forwarding groups of a cluster's
 * learners with one product per weight tile) and writes the learner's row.  With S
 * even (bf16 path), the step before each average stores, instead of every learner's
 * updated weights, the sums of pairs or quads of a cluster's learners (the first
 * levels of the averaging tree) in the first learner row of each pair or quad, and the
 * average finishes the tree from them.  So within a round the rows of params_dev are
 * scratch; the values every step and average computes are those of the literal
 * sequence, and when the round returns every row holds its learner's parameters.
 * Within the round, a step whose successor starts no local block and reads a
 * contiguous batch also computes that successor's first-layer output from the weights
 * it has just updated (bf16 path, two or more layers), so W_1 is read once per step;
 * the results are those of calling hier_avg_step, hier_avg_local_average and
 * hier_avg_global_average in turn, bit for bit. */
int hier_avg_round(hier_avg* h);

/* Global averaging interval in local steps: hier_avg_round then runs `steps` local
 * steps, a local average after every K1-th of them, and the global average after the
 * last, preceded by a local average exactly when K1 divides `steps`.  Sec. 3.1 takes
 * the interval K1 * beta with beta an integer for the analysis and leaves it free in
 * practice (Sec. 4's ImageNet run: K1 = 20, 43 steps).  0 restores K1 * K2 (the
 * default).  HA_EINVAL for steps < 0 or a NULL handle. */
int hier_avg_set_global_steps(hier_avg* h, int steps);

/* Step size of the following local steps (the gamma_n of round n; Theorem 3.3's
 * diminishing schedules set it between rounds).  HA_EINVAL if lr is not finite. */
int hier_avg_set_lr(hier_avg* h, float lr);

/* Mini-batch size of the following local steps (the B_n of round n; Theorem 3.3's
 * growing batches), 1 <= B <= the B given at create (which sizes the buffers).  Each
 * learner reads its data sequentially: a step's batch starts where the previous one
 * ended, at row (rows read so far) mod N, which is t * B for a constant B.
 * HA_EINVAL outside that range; HA_ECUDA if clearing device buffers fails. */
int hier_avg_set_batch(hier_avg* h, int B);

/* One round end to end from host memory: copies the rows of X_host [P, N, d_0] that
 * this round reads, and all of y_host [P, N] (P * N * 4 bytes, one copy), into the
 * bound device data set (pinned host memory recommended), runs hier_avg_round, and
 * copies the per-learner loss of the round's last step into loss_host [P].  The rows
 * of X go in chunks of steps that double in length, on a stream of the library's own,
 * issued between the kernel launches, and overlap the kernels: a step waits only for
 * the chunk holding the rows it reads (bf16 path; the fp32 path copies the round's
 * rows first).  A chunk whose rows span at least 512 KB per learner is one copy per
 * learner when a learner's parameter row holds at least 4 Mi values, otherwise a
 * single pitched copy for all learners.  Synchronises. */
int hier_avg_round_host(hier_avg* h, const void* X_host, const int32_t* y_host,
                        float* loss_host);

/* One local step, exactly as hier_avg_step, for callers that cannot allocate
 * device memory (no cudaMalloc in their environment, an allocator they do not
 * own, or a binding that only passes existing buffers).  The paper has no
 * counterpart: this is a property of the library, not of the method.
 * The caller passes the inputs and outputs (params_dev [P, ld] updated in place,
 * X_dev, y_dev, N as for hier_avg_bind); the step's scratch lives in one 32 MiB
 * array that the library holds in every GPU's memory until the process exits.
 * The call binds the handle to these buffers and to that array, clears the part
 * of the array the step uses, takes the step at the handle's counter t and
 * advances t.  It calls no device allocator.
 *   - The first call in each CUDA context of a device (so once per device, and
 *     again after a device reset) looks up the array's device address; make that
 *     first call before any stream capture on that device.
 *   - Every call, from any handle, shares the one array and leaves its contents
 *     behind; calls whose work overlaps on the GPU (other streams, other
 *     threads) race on it.  After a call, later hier_avg_step / round calls of
 *     the same handle also use the array until hier_avg_bind is called again.
 * Errors: HA_ENOMEM (with a message naming both sizes) when one step of the
 * configuration needs more than 32 MiB of scratch (hier_avg_workspace_bytes less
 * the cluster means, which only rounds use; a round of a handle bound this way
 * averages in place), HA_EINVAL for NULL or misaligned buffers or N < 1, HA_ECUDA. */
int hier_avg_step_static(hier_avg* h, float* params_dev, const void* X_dev,
                         const int32_t* y_dev, int64_t N, void* stream);

/* Step counter t (local SGD steps taken); setting it resumes a run whose
 * parameters were saved: it also sets the rows read so far to t * B (the current
 * batch size), which is where a run with a constant batch size stands. */
int hier_avg_get_step(const hier_avg* h, int64_t* t);
int hier_avg_set_step(hier_avg* h, int64_t t);

/* Per-learner mean cross-entropy of the last step's mini-batch -> loss_host [P].
 * Synchronises the bound stream. */
int hier_avg_losses(hier_avg* h, float* loss_host);

/* Synchronise the bound stream and report a device-side failure:
 * HA_ETIMEOUT if a bounded wait inside a kernel expired (that kernel stopped
 * early and its outputs are invalid), HA_ECUDA on an asynchronous CUDA error. */
int hier_avg_check(hier_avg* h);

/* Failure-detection self-test (the paper has no counterpart: this checks the
 * library's own failure detection).  Launches one kernel on the bound stream that
 * runs the library's two kinds of bounded device wait -- an acquire spin on a global
 * flag and an mbarrier phase wait, the waits that order split-K reductions and the
 * TMA / tensor-core pipelines -- on conditions nothing will satisfy, each with a limit
 * of limit_us microseconds at the device's peak SM clock (longer at a lower clock).
 * Both expire; the kernel records the timeout in the handle's error word and returns
 * with nothing in flight, so the CUDA context stays usable.  The next hier_avg_check
 * returns HA_ETIMEOUT and clears the word; later calls work as before.
 * Errors: HA_ESTATE before bind, HA_EINVAL for limit_us outside [1, 1e7], HA_ECUDA. */
int hier_avg_wait_selftest(hier_avg* h, int64_t limit_us);

/* Kernel timing with CUDA events recorded on the bound stream around every
 * launch of the handle.  enable = 1 starts (and clears) it, 0 stops it. */
#define HA_KERNEL_GATHER        0   /* mini-batch fetch (+ transpose)        */
#define HA_KERNEL_FORWARD       1   /* per-layer forward GEMM + epilogue     */
#define HA_KERNEL_XENT          2   /* softmax cross-entropy gradient        */
#define HA_KERNEL_BACKWARD      3   /* fused dX + dW + SGD update            */
#define HA_KERNEL_LOCAL_AVG     4
#define HA_KERNEL_GLOBAL_AVG    5   /* fused last local + global average     */
#define HA_KERNEL_HEAD          6   /* fused last layer (<= 16 classes)      */
#define HA_KERNEL_UPDATE_FORWARD 7  /* first-layer update + next forward     */
#define HA_KERNEL_KINDS         8
int hier_avg_profile(hier_avg* h, int enable);

/* The same for a subset: kinds is a bitmask of (1 << HA_KERNEL_*); 0 stops.
 * Each timed launch costs two event records that separate it from its
 * neighbours on the stream, so a throughput measurement times only the kinds it
 * reports.  HA_EINVAL for bits beyond HA_KERNEL_KINDS. */
int hier_avg_profile_kinds(hier_avg* h, unsigned kinds);

/* Kernels this handle has launched since it was created (every launch of the step,
 * averaging and round calls, one per kernel).  HA_EINVAL for NULL arguments. */
int hier_avg_launches(const hier_avg* h, int64_t* launches);

/* Time only every n-th launch of each enabled kind (n >= 1, default 1; counted from
 * the last hier_avg_profile / hier_avg_profile_kinds), so that a throughput
 * measurement perturbs few launches.  hier_avg_profile_read then reports the
 * sampled launches.  HA_EINVAL for n < 1. */
int hier_avg_profile_every(hier_avg* h, int every);

/* Synchronise and read kind's totals since profiling was enabled: summed event
 * time in ms, number of launches, the algorithmic bytes moved by them (fp32 master
 * read and written, activations read and written once) and their algorithmic flops
 * (2 per multiply-add of the step's products: forward, dW and dX of every learner;
 * P * ld additions per average).  Any output pointer may be NULL. */
int hier_avg_profile_read(hier_avg* h, int kind, double* total_ms, int64_t* launches,
                          double* bytes, double* flops);

const char* hier_avg_strerror(int status);
const char* hier_avg_last_error(const hier_avg* h);

#ifdef __cplusplus
}
#endif

#endif /* HIER_AVG_H */
