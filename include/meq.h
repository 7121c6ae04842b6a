/*
 * meq.h -- C ABI of the GB300 (sm_103a) MeqMuon optimizer step for 2D
 * hidden-layer weights.
 *
 * The step follows the paper "MeqMuon: Matrix-Equilibrating Muon for LLM
 * Pretraining", Algorithm 1 (hidden-weight branch), for every matrix W_i:
 *
 *   B_t   = mu B_{t-1} + G_t                                   Eq. (10)
 *   U_t   = NS_K(B_t)  (X_0 = B/||B||_F;
 *           X_{k+1} = a X_k + (b A_k + c A_k^2) X_k, A_k = X_k X_k^T)  Eq. (5)
 *   r_i = ||U_{i,:}||/sqrt(n), c_j = ||U_{:,j}||/sqrt(m)       Eq. (7)
 *   gamma = std/mean over entries > eps                        Eq. (8)
 *   U~  = diag(r^-1) U  if gamma_r >= gamma_c, else U diag(c^-1)  Eqs. (9), (11)
 *   W  <- (1 - lr*wd) W - rho*lr*U~                            Eq. (14)
 *
 * Everything runs in the library's own CUDA kernels, asynchronously on the
 * caller's stream. Newton-Schulz runs on the tensor cores (tcgen05, TMA, TMEM)
 * with 16-bit operands and fp32 accumulation; all other arithmetic is fp32.
 *
 * Conventions shared by every call:
 *   - Matrices are fp32, row-major, contiguous, rows = output features and
 *     columns = input features (the PyTorch layout the paper uses, Section 3.1).
 *   - Device pointers must be 16-byte aligned.
 *   - A meq_state is not thread-safe: one host thread drives it at a time.
 *   - Validation errors are returned synchronously and nothing is enqueued.
 *     Errors raised on the device (a bounded wait that expired) are reported
 *     by the next meq_sync() as MEQ_ERR_TIMEOUT / MEQ_ERR_CUDA.
 */
#ifndef MEQ_H
#define MEQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MEQ_OK = 0,
  MEQ_ERR_INVALID_ARG = 1,   /* null pointer, bad size, misaligned pointer, shape list differs from init */
  MEQ_ERR_OOM = 2,           /* device allocation failed or the workspace limit was exceeded */
  MEQ_ERR_CUDA = 3,          /* a CUDA runtime call failed (see meq_last_error) */
  MEQ_ERR_NONFINITE = 4,     /* a step's momentum had a non-finite norm (reported by meq_sync) */
  MEQ_ERR_TIMEOUT = 5,       /* a device-side bounded wait expired; the kernel returned early */
  MEQ_ERR_UNSUPPORTED = 6,   /* no sm_103a device, or a size beyond the library's limits */
  MEQ_ERR_CORRUPTED = 7      /* meq_check_canaries found a workspace guard band overwritten */
} meq_status;

/* One matrix: rows = out features (m), cols = in features (n). */
typedef struct {
  int64_t rows;
  int64_t cols;
} meq_shape;

/* Options fixed at init. meq_default_options() fills the paper's values. */
typedef struct {
  float rho;              /* RMS alignment coefficient, Eq. (14); 0.2 (Section 4) */
  int ns_steps;           /* K of Eq. (5); 5 (Sections 2 and 4); 1..32 */
  float ns_a, ns_b, ns_c; /* (3.4445, -4.7750, 2.0315), Section 2 */
  int nesterov;           /* 0: NS input B_t (Eq. (10), Algorithm 1);
                             1: NS input G_t + mu B_t (Nesterov look-ahead, Section 4) */
  uint32_t ns_fp16_mask;  /* bit k set: NS iteration k uses fp16 operands, else bf16.
                             Default 0xFFFFFFFF (all fp16; same tensor-core rate as bf16,
                             three more mantissa bits). 0 = all bf16. */
  float tie_atol;         /* Eq. (11) chooses row when gamma_r >= gamma_c - tie_atol; 1e-6 */
  int use_graph;          /* 1: the step's kernels are replayed from a CUDA graph (default) */
  int64_t workspace_limit_bytes; /* 0 = no limit; else init fails with MEQ_ERR_OOM above it */
  float wait_timeout_ms;  /* bound of every device-side spin wait; default 4000. An NS kernel's
                             MMA thread starts waiting for its first operands while the kernel
                             before it may still run, so the bound must exceed the longest kernel
                             of a step (about 20 ms per NS product at Llama-7B-class sizes) */
  int ns_cta_pair;        /* 1 (default): NS GEMMs run on CTA pairs (tcgen05 cta_group::2,
                             256 x 256 tiles on two SMs); 0: one CTA per 128 x 256 tile */
  int ns_x0_fused;        /* 1 (default): the momentum pass also writes X_0, unnormalised in
                             bf16, and the first NS products apply 1/||B||_F; iteration 0
                             then runs its X and P operands in bf16. 0: a separate pass
                             writes the normalised X_0 in the format ns_fp16_mask gives it. */
  int update_rule;        /* meq_update_rule; default MEQ_RULE_MEQMUON */
  int debug_canaries;     /* 1: guard bands of a fixed byte pattern surround every workspace
                             buffer (meq_check_canaries); default 0 */
  int debug_skip_load;    /* 1 (tests only): in every step's first NS launch, the leader
                             CTA of the first CTA pair arms its first operand stage but
                             does not load its half, so that stage never completes: the
                             MMA issuer's bounded wait expires, every role of the launch
                             stops and drains, and meq_sync reports MEQ_ERR_TIMEOUT (the
                             results of that step are not meaningful). Requires
                             ns_cta_pair = 1. Default 0. */
} meq_options;

/* Update applied to the hidden 2D weights after momentum and Newton-Schulz. */
typedef enum {
  MEQ_RULE_MEQMUON = 0, /* Eq. (11) equilibration, then Eq. (14) (Algorithm 1) */
  MEQ_RULE_MUON = 1     /* Muon with decoupled weight decay and RMS alignment, Eq. (6)
                           (the comparison baseline of Section 4): W <- (1 - lr wd) W
                           - lr rho sqrt(max(m, n)) U, no equilibration. Every entry must
                           be MEQ_KIND_HIDDEN (that baseline updates the others with
                           AdamW, which this library does not provide). */
} meq_update_rule;

/* Parameter type, selecting the branch of Algorithm 1 applied to it. */
typedef enum {
  MEQ_KIND_HIDDEN = 0,       /* 2D weight in a hidden layer: NS, then Eq. (11) (default) */
  MEQ_KIND_REMAINING_2D = 1, /* token embedding / LM head: N_c(N_r(B_t)), Eq. (12) */
  MEQ_KIND_VECTOR = 2        /* 1D parameter, given as shape (1, d): B_t / (||B_t||/sqrt(d)), Eq. (13) */
} meq_kind;

typedef struct meq_state meq_state; /* opaque */

void meq_default_options(meq_options* opt);

/* Bytes the state would allocate for this shape list, computed on the host
 * without touching the GPU. persistent = momentum buffers (4 bytes per
 * element: the only state MeqMuon keeps, Section 4 "Memory overhead");
 * workspace = transient NS / statistics buffers. Either output may be NULL. */
meq_status meq_state_bytes(const meq_shape* shapes, int n, const meq_options* opt,
                           size_t* persistent_bytes, size_t* workspace_bytes);

/* As meq_state_bytes, with a parameter type per entry (kinds may be NULL:
 * all MEQ_KIND_HIDDEN). MEQ_KIND_VECTOR entries must have rows == 1. */
meq_status meq_state_bytes_kinds(const meq_shape* shapes, const int* kinds, int n, const meq_options* opt,
                                 size_t* persistent_bytes, size_t* workspace_bytes);

/* Create the state for n matrices: zeroed momentum (B_{-1} = 0, Algorithm 1)
 * and the workspace, on the current CUDA device. opt may be NULL (defaults).
 * cuda_stream (cudaStream_t, may be NULL) orders the zero-fill. The shape
 * list is copied. On success *out owns device memory until meq_free. */
meq_status meq_init_state(const meq_shape* shapes, int n, const meq_options* opt,
                          void* cuda_stream, meq_state** out);

/* As meq_init_state, with a parameter type (meq_kind) per entry, so one state
 * runs Algorithm 1 over every trainable parameter of a model: hidden 2D
 * weights, the other 2D parameters, and vectors (shape (1, d)).
 * kinds is copied; NULL means all MEQ_KIND_HIDDEN. */
meq_status meq_init_state_kinds(const meq_shape* shapes, const int* kinds, int n,
                                const meq_options* opt, void* cuda_stream, meq_state** out);

/* One MeqMuon step over all n matrices (Algorithm 1, hidden branch).
 *   params[i]: device fp32 W_i (rows x cols), updated in place.
 *   grads[i] : device fp32 G_i, read only.
 *   shapes/n : must equal the list given to meq_init_state.
 *   lr = eta_t (the caller applies warm-up / decay), momentum = mu,
 *   weight_decay = lambda, eps = delta of Section 3.1 (1e-7).
 * All work is enqueued on cuda_stream (cudaStream_t; NULL = legacy default
 * stream) with no host synchronisation. params/grads must stay valid until
 * the enqueued work has run. */
meq_status meq_step(float* const* params, const float* const* grads, meq_state* st,
                    const meq_shape* shapes, int n, float lr, float momentum,
                    float weight_decay, float eps, void* cuda_stream);

/* The same step in two calls, split before the parameter update, so that a
 * caller can overlap work on the parameters of the previous step (a copy
 * to the host, an all-gather) with this step's momentum, Newton-Schulz and
 * statistics, which do not touch the parameters:
 *   meq_step_prepare: Eq. (10), Eq. (5) and the statistics of Eqs. (7)-(9)
 *     and (11) (Algorithm 1 up to the update), for the gradients and scalars
 *     given (the arguments of meq_step without params);
 *   meq_step_apply: the update (Eq. (14); Eqs. (12) and (13) for the other
 *     kinds) of params with the scalars of the pending prepare.
 * meq_step(params, grads, ...) equals meq_step_prepare(grads, ...) then
 * meq_step_apply(params, ...), bit for bit. Each call enqueues on its
 * cuda_stream; the apply must be ordered after its prepare and before the
 * next prepare (for example, one stream, with a cudaStreamWaitEvent on the
 * caller's copy before the apply). A second prepare before the apply, an
 * apply without a prepare, or meq_step while a prepare is pending returns
 * MEQ_ERR_INVALID_ARG. With use_graph, each part replays its own graph. */
meq_status meq_step_prepare(const float* const* grads, meq_state* st, const meq_shape* shapes, int n,
                            float lr, float momentum, float weight_decay, float eps, void* cuda_stream);
meq_status meq_step_apply(float* const* params, meq_state* st, void* cuda_stream);

/* Wait for the state's enqueued work and report device-side errors
 * (MEQ_ERR_TIMEOUT for an expired bounded wait, MEQ_ERR_CUDA otherwise), then
 * MEQ_ERR_NONFINITE if, in a step since the last meq_sync, the momentum of
 * some entry had a NaN or infinite sum of squares (a non-finite gradient, or
 * a momentum already non-finite); meq_last_error names the first such entry.
 * Each report clears the condition. Such an entry's momentum and parameters
 * take the non-finite values (no step is skipped); every other entry's step
 * is unaffected, since entries are updated independently. */
meq_status meq_sync(meq_state* st);

/* Release all device memory of the state (synchronises first). NULL is a no-op. */
meq_status meq_free(meq_state* st);

/* Human-readable text of the last error of st; with st NULL, of the last
 * failed call made without a state (meq_init_state[_kinds],
 * meq_state_bytes[_kinds], meq_ns_cv_trajectory, meq_row_col_stats_noalloc).
 * Valid until the next such call. */
const char* meq_last_error(const meq_state* st);
const char* meq_status_string(meq_status s);

/* ---- inspection and checkpointing (synchronise the state first) ---------- */

/* Copy momentum B_i (rows x cols fp32) to dst (host or device memory). */
meq_status meq_read_momentum(meq_state* st, int i, float* dst);
/* Overwrite momentum B_i from src (host or device), e.g. to resume. */
meq_status meq_write_momentum(meq_state* st, int i, const float* src);
/* Copy the last step's Newton-Schulz output U_i (rows x cols fp32, before
 * equilibration) to dst (host or device). Hidden weights only. U is held on
 * the device in fp16 (scaled by 2^14, so every entry above 4e-9 keeps 11
 * significant bits); the values returned are those fp16 values, from which
 * the row and column statistics are taken and which the update applies. */
meq_status meq_read_ns_output(meq_state* st, int i, float* dst);
/* Copy the normalised update U~_i of the last step (rows x cols fp32) to
 * dst (host or device): the matrix that step applied as
 * W <- (1 - lr wd) W - rho lr U~ (Eq. (14)). Hidden weight: diag(r^-1) U or
 * U diag(c^-1) (Eqs. (9), (11); rows or columns with RMS <= eps scaled by 0),
 * or sqrt(max(m, n)) U under MEQ_RULE_MUON (Eq. (6)); remaining 2D
 * parameter: N_c(N_r(B_t)) (Eq. (12)); vector: B_t / RMS(B_t) (Eq. (13)).
 * Computed by a kernel on the state's device (whichever device is current;
 * the current device is restored) from the operands and scale factors of
 * the update kernel; a host dst goes through a temporary device buffer of the
 * same size (MEQ_ERR_OOM if that allocation fails). Synchronises the state's
 * stream. */
meq_status meq_read_update(meq_state* st, int i, float* dst);
/* Last step's statistics of entry i. Hidden weight: r (rows floats), c (cols
 * floats) of Eq. (7) for U, gamma_r, gamma_c of Eq. (8) and the direction of
 * Eq. (11) (0 = row, 1 = column; 4 under MEQ_RULE_MUON, whose update is
 * the uniform sqrt(max(m, n)) U of Eq. (6) while r, c and the CVs still
 * describe U). Remaining 2D parameter: r = row RMS of B_t, c = column RMS
 * of N_r(B_t), their CVs, direction 2. Vector: r[0] = RMS of B_t, gammas 0,
 * direction 3. Any output may be NULL; r and c are host or device memory. */
meq_status meq_read_stats(meq_state* st, int i, float* r, float* c,
                          double* gamma_r, double* gamma_c, int* direction);
/* How often Eq. (11) chose row-wise (*rows) and column-wise (*cols)
 * normalisation for hidden weight i since the state was created or the
 * counts were last reset (both 0 for other entries and under MEQ_RULE_MUON).
 * The counts are kept on the device by the statistics kernel. */
meq_status meq_read_direction_counts(meq_state* st, int i, int64_t* rows, int64_t* cols);
/* Zero every entry's direction counts (enqueued on the state's stream). */
meq_status meq_reset_direction_counts(meq_state* st);

/* ---- diagnostics -------------------------------------------------------- */

/* With debug_canaries set at init: synchronise the state's stream and check
 * that every guard band still holds its pattern. MEQ_OK, or
 * MEQ_ERR_CORRUPTED with *bad_offset (may be NULL) = the arena offset of the
 * first changed byte (-1 otherwise); MEQ_ERR_INVALID_ARG without guards. */
meq_status meq_check_canaries(meq_state* st, int64_t* bad_offset);
/* Number of guard bands (0 without debug_canaries). */
int meq_canary_count(const meq_state* st);
/* Test hook: overwrite one byte of guard band `index` from the host
 * (cudaMemset), so that tests can check meq_check_canaries. */
meq_status meq_debug_corrupt_canary(meq_state* st, int index);

/* Row / column CV trajectory of the Newton-Schulz iterates (Section 3.1
 * replays Eq. (5) on saved pre-NS matrices this way): gamma_r[k] and
 * gamma_c[k] are the Eq. (8) CVs (over entries > eps) of the row and column
 * RMS (Eq. (7)) of X_k, k = 0..steps, computed by this library's CUDA path
 * with the NS options of opt (NULL: defaults; its ns_steps and update_rule
 * are ignored). k = 0 is X_0 = h / ||h||_F: its RMS values, like those of
 * every later iterate, are compared with eps after the normalisation. h:
 * device fp32, rows x cols row-major, 16-byte aligned, read only. gamma_r,
 * gamma_c: host arrays of steps + 1 doubles. steps: 0..32. Synchronous;
 * allocates and frees its own device scratch (about rows x cols x 4 bytes
 * plus one optimizer state per k), so concurrent calls do not share memory;
 * every shape meq_init_state accepts is accepted. Errors:
 * MEQ_ERR_INVALID_ARG (NULL, misaligned, bad sizes), MEQ_ERR_OOM, or the
 * error of the step it runs (text in meq_last_error(NULL)). */
meq_status meq_ns_cv_trajectory(const float* h, int64_t rows, int64_t cols, int steps, float eps,
                                const meq_options* opt, double* gamma_r, double* gamma_c, void* cuda_stream);
/* Number of kernels one meq_step launches (for launch accounting), and how
 * many of them are Newton-Schulz GEMM launches. */
int meq_kernels_per_step(const meq_state* st);
int meq_ns_gemm_launches_per_step(const meq_state* st);

/* Per-phase timing with CUDA events on the launch stream. While enabled,
 * meq_step runs the same kernels with an event recorded between phases:
 * with use_graph, by replaying a second graph that holds event-record nodes
 * between the phases, then waiting for the stream and adding up that step's
 * phase times (so profiled steps are not pipelined with the host); without
 * use_graph, by launching directly. meq_read_profile synchronises and returns
 * the summed milliseconds of each phase since profiling was enabled:
 *   phase_ms[0] momentum update + norms (all kinds), [1] X_0 cast,
 *   [2] all NS GEMMs, [3] statistics + direction / scales, [4] apply;
 *   *steps = profiled steps. */
meq_status meq_set_profiling(meq_state* st, int enable);
meq_status meq_read_profile(meq_state* st, double* phase_ms /* 5 */, int64_t* steps);

/* Failure-path self test of the device-side bounded waits: launches one
 * kernel that spins on a flag nothing ever sets, with the given limit
 * (0 < timeout_ms <= 10000), then synchronises. The kernel gives up when the
 * limit expires, records the timeout and returns, so the expected result is
 * MEQ_ERR_TIMEOUT with the context still usable. The paper has no
 * counterpart; this exists to test error reporting without faulting a GPU. */
meq_status meq_debug_wait_selftest(meq_state* st, float timeout_ms);

/* ---- allocation-free statistics ------------------------------------------
 * The paper has no counterpart to this entry point; it exists for callers
 * that cannot call cudaMalloc (code running inside a framework that owns all
 * device memory through its own pool, or a latency-critical path that must
 * not allocate after start-up, since cudaMalloc may synchronise the device).
 *
 * meq_row_col_stats_noalloc computes, for one fp32 row-major matrix U
 * (rows x cols, device memory, read only), the statistics step of the
 * optimizer: r (rows floats) and c (cols floats) of Eq. (7), gammas[0] =
 * gamma_r and gammas[1] = gamma_c of Eq. (8) over entries > eps, and
 * *direction of Eq. (11) (0 = row, 1 = column; row when gamma_r >= gamma_c -
 * tie_atol). All outputs are caller-provided device memory. The definitions
 * and precision (fp32 sums of squares and two-pass fp32 CVs) are those of
 * meq_step's statistics, so results agree with meq_read_stats for the same U
 * up to fp32 summation order.
 *
 * It allocates nothing. Its scratch is a fixed 8 MiB __device__ array inside
 * the library, held by every GPU that loads the library until the process
 * exits. A matrix fits when rows * ceil(cols / 1024) + ceil(rows / 32) * cols
 * <= 2,097,152 floats (e.g. 4096 x 11008 and 11008 x 4096, but not 8192 x
 * 8192); larger ones, NULL pointers or
 * non-positive sizes return MEQ_ERR_INVALID_ARG before anything is enqueued
 * and before any CUDA call; meq_last_error(NULL) then says why.
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any CUDA
 * stream capture. Every call shares the one array and overwrites all of the
 * scratch it reads, so nothing needs clearing between calls, but calls whose
 * kernels overlap on the GPU (different streams without ordering) race on
 * it. Work is enqueued on cuda_stream (cudaStream_t, NULL = legacy stream)
 * as three kernel launches; MEQ_ERR_CUDA reports a failed launch or address
 * lookup of this call (its own status, with the CUDA error text in
 * meq_last_error(NULL)). */
meq_status meq_row_col_stats_noalloc(const float* U, int64_t rows, int64_t cols, float eps,
                                     float tie_atol, float* r, float* c, double* gammas,
                                     int* direction, void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* MEQ_H */
