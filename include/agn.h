/*
 * agn.h - C ABI of the GB300 implementation of the hot path of Accumulated
 * Gradient Normalization (Hermans, Spanakis & Moeckel, ACML 2017).
 *
 * What the library computes (all of it in CUDA kernels on one GPU):
 *   n workers, each a resident replica theta_k of the parameters, pull the
 *   central variable theta~, take lambda local minibatch-SGD steps on their own
 *   data shard while accumulating the gradients (Algorithm 1), and commit the
 *   accumulated update normalised by lambda,
 *       Delta theta^k = -(eta / lambda) * sum_i (1/m) sum_j grad L(theta_i; x_ij, y_ij)   (Eq. 1)
 *   which the parameter server adds to theta~ in FIFO order (Eq. 2).  The
 *   asynchrony is an explicit, seeded schedule: commit c belongs to worker w_c
 *   and was computed from theta~ after v_c = c - tau_c commits (Fig. 1).
 *
 * Conventions for every entry point:
 *   - Return 0 (AGN_OK) on success, a negative AGN_E_* code on failure; the
 *     message of the last failure on a handle is agn_last_error(handle), and
 *     that of a handle-less call is agn_last_error(NULL) (per thread).
 *   - Host buffers are owned by the caller and given with a capacity in
 *     elements; a short buffer gives AGN_E_INVALID and writes nothing.
 *   - Device buffers passed in are owned by the caller and must stay valid
 *     until the work queued on the given stream completes.
 *   - A handle must not be used by two threads at once.
 *   - Flat parameter order (the paper fixes none): for l = 1..L, W_l row-major
 *     [d_l][d_{l-1}], then b_l [d_l].  P = sum_l (d_l d_{l-1} + d_l).
 *   - The loss is softmax cross-entropy over the last layer's d_L outputs; the
 *     hidden layers use ReLU.
 */
#ifndef AGN_H
#define AGN_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AGN_OK 0
#define AGN_E_INVALID (-1)     /* bad sizes, pointers or options            */
#define AGN_E_SCHEDULE (-2)    /* infeasible (worker, staleness) pair       */
#define AGN_E_OOM (-3)         /* device or host allocation failed          */
#define AGN_E_CUDA (-4)        /* a CUDA call failed (message has details)   */
#define AGN_E_TIMEOUT (-5)     /* a bounded device wait gave up              */
#define AGN_E_NONFINITE (-6)   /* a loss or a commit was not finite; the run
                                  still completed and theta~ is readable     */
#define AGN_E_UNSUPPORTED (-7) /* valid request this build cannot serve      */
#define AGN_E_BOUNDS (-8)      /* bounds-checked build only: a kernel access
                                  outside every known device buffer was
                                  refused (not performed); see agn_last_error */

#define AGN_PREC_FP32 0        /* fp32 parameters, activations and GEMMs    */
#define AGN_PREC_BF16 1        /* bf16 GEMM operands, fp32 accumulation, fp32
                                  master replicas and accumulators            */

#define AGN_DIST_UNIFORM 0     /* x ~ U[0,1)^d0 */
#define AGN_DIST_NORMAL 1      /* x ~ N(0,1)^d0 */

#define AGN_GEMM_AUTO 0        /* tcgen05 where eligible, else CUDA cores   */
#define AGN_GEMM_SIMT 1        /* CUDA-core GEMM kernels only                */
#define AGN_GEMM_TCGEN05 2     /* tcgen05/TMEM GEMMs for the hidden layers in
                                  either precision (fp32 mode feeds every fp32
                                  operand as three exact bf16 pieces, fp32
                                  accumulation); needs at least one hidden
                                  layer, batch <= 256 and d_0 .. d_{L-1}
                                  multiples of 8 (else AGN_E_UNSUPPORTED).
                                  The d_L-wide output layer's forward,
                                  softmax-CE and dX run on CUDA cores; its dW
                                  joins the tensor-core dW launch          */

/* Local optimizers (agn_options.local_optimizer) */
#define AGN_OPT_SGD 0
#define AGN_OPT_ADAM 1

/* Commit rules (agn_options.commit_rule) */
#define AGN_COMMIT_AGN 0       /* Delta = -eta a / lambda (Eq. 1)            */
#define AGN_COMMIT_DYNSGD 1    /* Delta = -eta a / (tau_c + 1), Section 4     */

typedef struct agn_handle agn_handle;

/* Options of agn_create.  Fill with agn_default_options, then override. */
typedef struct agn_options {
  int32_t precision;            /* AGN_PREC_*, default fp32                    */
  int32_t batch;                /* m, samples per minibatch per worker (32)    */
  int64_t n_samples;            /* N, dataset rows, split into n equal shards of
                                   S = N / n rows (the last N mod n unused)    */
  int32_t input_dist;           /* AGN_DIST_*, default uniform                 */
  const int32_t* teacher_dims;  /* labelling network dims (d_0 .. 10); NULL =
                                   {d_0, 64, d_L}                             */
  int32_t n_teacher_dims;
  int32_t normalize;            /* 1 = AGN (divide by lambda, Eq. 1); 0 = the
                                   un-normalised ablation (Fig. 3)            */
  int32_t gemm;                 /* AGN_GEMM_*                                  */
  int32_t tau_lo, tau_hi;       /* staleness range of the built-in schedule    */
  void* stream;                 /* cudaStream_t for all work; NULL = a stream
                                   the handle creates and owns                 */
  /* Optional caller inputs (host, copied at create); NULL = generate from the
     seed.  x: [n_samples][d_0] fp32 row-major, y: [n_samples] int32 in
     [0, d_L), theta0: [P] fp32 flat order. */
  const float* x_init;
  const int32_t* y_init;
  const float* theta_init;
  /* Diagnostic: which hidden-layer GEMMs use the tcgen05 kernels when they
     are on (bit 0 forward, bit 1 dX, bit 2 dW; none of bits 0-2 = all three).  Bit 3 runs the
     dW GEMMs on the earlier non-persistent tcgen05 kernel (one tile per CTA)
     instead of the persistent one, for comparison.  Bit 4 runs the forward
     and dX GEMMs without split K (one CTA per output tile).  Bit 5 runs the
     output layer (forward, softmax-CE, dX) as a kernel of its own instead of
     in the epilogue of the last hidden layer's forward GEMM.  Bit 6 gathers
     each local step's minibatch into a buffer of its own (one launch per
     step) instead of reading it from the padded shards in place.  Bit 7
     runs the bf16 forward and dX GEMMs of full waves with one 128-row tile
     per CTA instead of two that share each B stage.  Bit 8 makes the
     persistent dW kernel read each accumulator chunk into shared memory and
     store a_k + g even for waves whose accumulators fit well within the L2,
     where it otherwise adds g to a_k in the L2 (red.add).  Bit 9 makes the
     forward of layer 1 request no weight stage before its dependency wait.
     Any other bit: AGN_E_INVALID. */
  int32_t tc_mask;
  /* Commit rule (AGN_COMMIT_*): AGN_COMMIT_AGN (default) commits
     Delta = -eta a / lambda (Eq. 1; -eta a with normalize = 0);
     AGN_COMMIT_DYNSGD commits the accumulated update scaled by staleness,
     Delta = -eta a / (tau_c + 1), tau_c the schedule's staleness of commit c
     (the DynSGD comparison of Section 4; normalize is ignored). */
  int32_t commit_rule;
  /* 1: keep no gradient accumulator.  Each worker keeps the theta~ it
     pulled (theta_pull) and a commit adds (theta_k - theta_pull) scaled by
     1/lambda (1/(tau_c + 1) for DynSGD, 1 without normalisation), which
     equals -eta a / lambda in exact arithmetic (the sum of the local updates,
     Algorithm 1).  Saves the accumulator's 8 bytes per parameter and local
     step; the paper has no such variant.  Not with tc_mask bit 3. */
  int32_t elide_accumulator;
  /* Held-out evaluation set for agn_evaluate: rows [N, N + n_eval) of the
     seeded generator, labelled by the same teacher (0 = none; not with
     x_init / y_init). */
  int64_t n_eval;
  /* Local optimizer (AGN_OPT_*): AGN_OPT_SGD (default), g = -eta grad; or
     AGN_OPT_ADAM (Algorithm 1 names Adam as an example), g = -eta m^/(sqrt(v^)
     + eps) with per-worker moments that persist across commits and bias
     corrections at the worker's step count (never reset).  The accumulator
     then sums the steps g, and a commit adds a/lambda (a/(tau_c+1), a).
     adam_beta1, adam_beta2, adam_eps: 0 = 0.9, 0.999, 1e-8.  Not with
     tc_mask bit 3. */
  int32_t local_optimizer;
  float adam_beta1, adam_beta2, adam_eps;
} agn_options;

void agn_default_options(agn_options* opt);

/*
 * Create a handle: allocate theta~ [P], replicas theta_k [n][P] and
 * accumulators a_k [n][P] (fp32; plus bf16 working copies [n][P] in bf16
 * mode), the dataset and activation workspaces on the current device;
 * generate (or copy) the dataset, teacher labels and theta~^0 (Glorot-uniform
 * weights, zero biases); every replica pulls version 0.
 *   dims     : d_0 .. d_L (n_dims = L + 1 >= 2), all > 0; d_L = classes.
 *   n_workers: n >= 1;  lambda: local steps per commit >= 1 (Algorithm 1);
 *   eta      : learning rate > 0 (constant: Section 4 uses no decay);
 *   seed     : seeds every generated input;  opt: NULL = defaults.
 * Errors: AGN_E_INVALID, AGN_E_OOM, AGN_E_CUDA, AGN_E_UNSUPPORTED.
 */
int agn_create(const int32_t* dims, int32_t n_dims, int32_t n_workers, int32_t lambda,
               double eta, uint64_t seed, const agn_options* opt, agn_handle** out);

/*
 * Run the next n_commits commits (Algorithm 1 workers, Eq. 2 server).
 * worker[i], staleness[i] (host, length n_schedule >= n_commits) describe
 * commits V .. V+n_schedule-1, V = commits applied so far: commit c belongs
 * to worker[c-V] and reads theta~ after c - staleness[c-V] commits.  Entries
 * past n_commits are look-ahead: they tell the handle which version each
 * worker must pull during this call.  Feasible iff prev(w) < v_c <= c with
 * prev(w) the worker's previous commit (-1 before its first); a commit whose
 * version was passed in an earlier call must match the pull made then.
 * worker == NULL and staleness == NULL: use the built-in seeded round-robin
 * schedule (agn_make_schedule with the handle's tau_lo/tau_hi and seed).
 * Cumulative: repeated calls continue the commit index and the step counters.
 * Queues the work on the handle's stream and waits for it.
 * Errors: AGN_E_INVALID, AGN_E_SCHEDULE (nothing run), AGN_E_CUDA,
 * AGN_E_NONFINITE (run completed; results readable), AGN_E_TIMEOUT (a
 * tensor-core kernel gave up on a bounded wait; results are not valid).
 */
int agn_run(agn_handle* h, int32_t n_commits, const int32_t* worker,
            const int32_t* staleness, int32_t n_schedule);

/*
 * The central variable theta~ after the commits run so far: theta~^0 plus
 * every commit Delta theta^k added in FIFO order by the parameter server
 * (Eq. 2; Algorithm 1's Commit).  fp32, flat order, into host out[P]
 * (cap >= P, else AGN_E_INVALID).  Waits for the handle's queued work.
 */
int agn_central(agn_handle* h, float* out, int64_t cap);

/* Replica theta_k (fp32 master), flat order, into host out[P]. */
int agn_replica(agn_handle* h, int32_t k, float* out, int64_t cap);

/*
 * Per commit c so far (index order): the mean over the worker's lambda local
 * steps of the minibatch loss (1/m) sum_j L(theta_i; x_ij, y_ij), the
 * objective whose gradient Eq. 1 sums, L being softmax cross-entropy.  fp32
 * into host out[C], C = agn_num_commits (cap >= C, else AGN_E_INVALID).
 * Waits for the handle's queued work.
 */
int agn_loss(agn_handle* h, float* out, int64_t cap);

/*
 * Loss and accuracy of the current theta~ on the held-out set (the training-
 * accuracy curves of Section 4): softmax cross-entropy mean and the fraction
 * of samples whose argmax (lowest index on ties) is the label.  Forward pass in
 * fp32 on the device (CUDA-core GEMMs), fixed-order reductions; blocks until
 * done.  loss, accuracy: host floats (nullable); pred: host int32 [n_eval]
 * predictions (nullable), cap its length.  AGN_E_INVALID without an
 * evaluation set or with a short pred buffer.  No counterpart call in the
 * paper, which reports these metrics.
 */
int agn_evaluate(agn_handle* h, float* loss, float* accuracy, int32_t* pred, int64_t cap);

/*
 * Temporal efficiency, Eq. 4: E(a, b) = int_0^m f_a dt / int_0^m f_b dt with m
 * the shorter of the two curves' end times.  Curve x is sampled at times
 * tx[0..nx) (non-decreasing, >= 0) with values fx; it is the piecewise-linear
 * interpolation of its samples, constant at fx[0] on [0, tx[0]] (the paper
 * does not fix the quadrature).  Host arrays; result in *out.  AGN_E_INVALID
 * for empty or decreasing curves, no shared time, or a zero denominator.
 */
int agn_temporal_efficiency(const double* ta, const double* fa, int64_t na, const double* tb,
                            const double* fb, int64_t nb, double* out);

/* Per commit so far: ||Delta_c||_2 (host out[C]). */
int agn_delta_norm(agn_handle* h, float* out, int64_t cap);

int64_t agn_num_params(const agn_handle* h);   /* P, or -1 for NULL */
int64_t agn_num_commits(const agn_handle* h);  /* commits applied so far */

/*
 * Statistics of the last agn_run: [0] waves, [1] kernel launches, [2] GPU
 * milliseconds (CUDA events around the queued work), [3] worker-steps, and,
 * when cap >= 5, [4] host milliseconds from the call's start until all of its
 * work was queued (planning and launches, before the final wait).
 */
int agn_last_run_stats(const agn_handle* h, double* out, int64_t cap);

/*
 * Pure host helper: the inputs agn_create generates for these arguments,
 * restricted to dataset rows [row0, row0 + n_rows): x [n_rows][d_0] fp32,
 * y [n_rows] int32 (teacher labels), theta0 [P] fp32 flat (any may be NULL).
 * teacher_dims NULL = {d_0, 64, d_L}.  Needs no GPU.
 */
int agn_generate_inputs(const int32_t* dims, int32_t n_dims, int32_t input_dist,
                        const int32_t* teacher_dims, int32_t n_teacher_dims, uint64_t seed,
                        int64_t row0, int64_t n_rows, float* x, int32_t* y, float* theta0);

/*
 * Per-kernel profiling.  agn_profile(h, 1) makes every later agn_run record a
 * CUDA event pair around each kernel launch (on the handle's stream) and
 * accumulate, per kernel class, the launches, the device milliseconds and
 * the algorithmic flops and DRAM bytes of those launches; agn_profile(h, 0)
 * stops and agn_profile(h, 2) clears the totals.  agn_kernel_stats writes
 * AGN_KERNEL_CLASSES rows of 4 doubles {launches, ms, flops, bytes}, row i
 * for class i below, into out (cap >= 4 * AGN_KERNEL_CLASSES).
 */
#define AGN_K_GATHER 0       /* minibatch gather (FetchNextMiniBatch)            */
#define AGN_K_FORWARD 1      /* forward GEMM + bias + ReLU                       */
#define AGN_K_SOFTMAX 2      /* softmax cross-entropy; with a narrow output layer
                                the fused output head (forward, softmax-CE, dX)  */
#define AGN_K_BACKWARD_DX 3  /* dX GEMM + ReLU mask                              */
#define AGN_K_BACKWARD_DW 4  /* dW GEMM + local step + accumulation              */
#define AGN_K_COMMIT 5       /* fused commit + pull                              */
#define AGN_K_NORMS 6        /* per-commit norm reduction                        */
#define AGN_K_OTHER 7        /* pulls outside commits, loss means                */
#define AGN_K_FORWARD_HEAD 8 /* the last hidden layer's forward GEMM with the
                                output layer in its epilogue (forward,
                                softmax-CE, dX of the last hidden layer)         */
#define AGN_KERNEL_CLASSES 9
int agn_profile(agn_handle* h, int32_t mode);
int agn_kernel_stats(const agn_handle* h, double* out, int64_t cap);

/* Copy the generated inputs (host, caller-owned, any may be NULL):
   x [n_samples][d_0] fp32, y [n_samples] int32, theta0 [P] fp32 flat. */
int agn_export_inputs(agn_handle* h, float* x, int32_t* y, float* theta0);

const char* agn_last_error(const agn_handle* h);
void agn_destroy(agn_handle* h);

/*
 * Seeded round-robin schedule (pure host helper): commit c belongs to worker
 * c mod n, staleness tau_c = tau_lo + ((d_c >> 40)(tau_hi - tau_lo + 1)) >> 24
 * with d_c the c-th draw of the schedule stream, clamped to c - prev(w_c) - 1.
 * Outputs are host arrays of n_commits int32.
 */
int agn_make_schedule(int32_t n, int32_t n_commits, int32_t tau_lo, int32_t tau_hi,
                      uint64_t seed, int32_t* worker_out, int32_t* tau_out);

/*
 * The plan agn_run follows for the first n_commits commits of a fresh handle
 * with n_workers workers (1 .. 256, as agn_create) and lambda local steps
 * (pure host helper, no device).  Commit c reads theta~ after v_c = c - staleness[c] commits
 * (Figure 1's FIFO server; Algorithm 1's Pull before its local steps), so
 * the local steps of every commit whose version is already applied can run
 * together: a wave takes, per worker, its next commit if v_c <= V (V = commits
 * applied so far); then the longest run of computed commits from V on is
 * applied in order, and the replicas pull the versions their next commits
 * read as those versions appear.  worker / staleness as for agn_run
 * (n_schedule >= n_commits entries; entries past n_commits are look-ahead).
 * Outputs (host, caller-owned):
 *   n_waves_out            : number of waves;
 *   wave_slots[w], wave_end[w] (capacity n_commits each): the commits whose
 *                            local steps wave w runs, and the number of
 *                            commits applied once it is done;
 *   slot_commit[s], slot_t0[s] (capacity n_commits): the commits in wave
 *                            order, and the worker's step counter t (Algorithm
 *                            1; never reset) when that commit's steps start;
 *   pull_version[p], pull_worker[p] (capacity pull_cap; *n_pulls_out entries):
 *                            the pulls, in order: the worker pulls theta~ right
 *                            after pull_version commits are applied.
 * Errors: AGN_E_INVALID (bad sizes or a short buffer), AGN_E_SCHEDULE.
 */
int agn_plan_waves(int32_t n_workers, int32_t lambda, int32_t n_commits, const int32_t* worker,
                   const int32_t* staleness, int32_t n_schedule, int32_t* n_waves_out,
                   int32_t* wave_slots, int32_t* wave_end, int32_t* slot_commit,
                   int64_t* slot_t0, int64_t pull_cap, int32_t* pull_version,
                   int32_t* pull_worker, int64_t* n_pulls_out);

/*
 * Standalone commit + pull (the parameter-server step, Eq. 1-2 and the
 * Commit/Pull of Algorithm 1) on caller device buffers.  For c = 0 .. C-1 in
 * order: k = commit_worker[c];
 *     Delta = fp32(acc[k] * s), s = fp32(-eta/lambda) (fp32(-eta) when
 *     normalize == 0), computed in double; theta_c = fp32(theta_c + Delta)
 *     (no fused multiply-add, so results are bit-reproducible);
 *     acc[k] = 0;  replica[p] = theta_c for every p in
 *     pull_workers[pull_offsets[c] .. pull_offsets[c+1]).
 *   theta_c   : device fp32 [P];  acc, replicas: device fp32 [n][ld],
 *               ld >= P, ld % 4 == 0, all three 16-byte aligned.
 *   replicas_bf16: optional device bf16 [n][ld] that receives bf16(theta_c)
 *               (round to nearest even) at each pull; NULL = none.
 *   commit_worker [C], pull_offsets [C+1], pull_workers: host int32.
 *   delta_norm: optional device fp32 [C] receiving ||Delta_c||_2 (the
 *               per-block partial sums are reduced in a fixed order).
 *   stream    : cudaStream_t or NULL (legacy default stream).
 * Queues the work and returns without waiting.  Scratch memory (the schedule
 * and the norm partials) comes from the stream-ordered allocator.
 * Errors: AGN_E_INVALID, AGN_E_OOM, AGN_E_CUDA.
 */
int agn_commit_pull(float* theta_c, float* acc, float* replicas, void* replicas_bf16,
                    int64_t P, int64_t ld, int32_t n, int32_t C,
                    const int32_t* commit_worker, const int32_t* pull_offsets,
                    const int32_t* pull_workers, double eta, int32_t lambda,
                    int32_t normalize, float* delta_norm, void* stream);

/*
 * agn_commit_pull_noalloc: agn_commit_pull for callers that may not allocate
 * device memory.  The paper has no counterpart; it is a deployment variant.
 * Some callers cannot call cudaMalloc on this path: a host framework that
 * owns all device memory through its own pool and forbids allocations
 * outside it, or a latency-bound loop where an allocation, which can
 * synchronise the device or fail under memory pressure, is not allowed.
 * Same arguments, same kernels and bit-identical results as agn_commit_pull
 * (theta~, accumulators and replicas always; the norms too whenever the
 * commit kernel's grid fits the fixed array, i.e. on every GPU with at most
 * 256 SMs, GB300 included: they are then reduced in the same fixed order).  It allocates nothing: its scratch (the per-block
 * partial sums of the norms) is a fixed array of 16 x 1024 doubles
 * (128 KiB) in device global memory that every GPU loading the library holds
 * until the process exits.
 *   - Limit: each commit may have at most 256 pulls (more gives
 *     AGN_E_INVALID with a message saying so); P, C and n are otherwise free.
 *   - The first call on a device looks up the array's device address (with
 *     that device current) and caches it; make that first call before any
 *     stream capture.
 *   - Every call shares the one array, which keeps the last call's contents
 *     (nothing in it needs to start at zero).  Calls that overlap on the GPU
 *     (other streams, other host threads) race on it and give wrong norms:
 *     order them on one stream or with events.
 * Errors: AGN_E_INVALID, AGN_E_CUDA, AGN_E_UNSUPPORTED (device ordinal > 63).
 */
int agn_commit_pull_noalloc(float* theta_c, float* acc, float* replicas, void* replicas_bf16,
                            int64_t P, int64_t ld, int32_t n, int32_t C,
                            const int32_t* commit_worker, const int32_t* pull_offsets,
                            const int32_t* pull_workers, double eta, int32_t lambda,
                            int32_t normalize, float* delta_norm, void* stream);

/*
 * Test hook of the failure path of the bounded device waits (the paper has no
 * counterpart).  The tensor-core GEMMs' split-K exchange and the fused output
 * layer wait, on the device, for the other CTAs of their launch; every such
 * wait gives up after a time limit, the kernel then returns without its
 * results and agn_run reports AGN_E_TIMEOUT.  wait_ns > 0 sets that limit for
 * this handle's later runs (0 = the default, 2 s); withhold_rank >= 0 makes
 * split-K rank withhold_rank of every split-K launch skip its arrival on the
 * tile counter, so that the ranks waiting for it give up after wait_ns
 * (-1 = none).  After a run that timed out, the handle's results are not
 * valid: destroy it.  Errors: AGN_E_INVALID.
 */
int agn_debug_waits(agn_handle* h, int64_t wait_ns, int32_t withhold_rank);

/*
 * Fill the inputs of the standalone commit workload on the device with the
 * seeded generator: theta_c[i] = fp32(N(0,1) number i of the commit-theta
 * stream); acc[k][i] = fp32(0.1 * N(0,1) number k*P + i of the commit-acc
 * stream) for k < n; replicas [n][ld] (optional) = theta_c.  Asynchronous.
 */
int agn_fill_commit_inputs(float* theta_c, float* acc, float* replicas, int64_t P,
                           int64_t ld, int32_t n, uint64_t seed, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AGN_H */
