/*
 * paraanya.h -- C ABI of the GB300 (sm_103a) cached Picard solver step.
 *
 * The library implements one Picard iteration of sliding-window parallel DDIM
 * sampling (ParaDiGMS-style) with ParaAnya's output cache:
 *
 *   Sec. 2.1, Eq. 1   Picard update  x_{t+j+1} <- x_t + sum_{i=t}^{t+j} s(x_i, eps_i)
 *   Sec. 2.1, Eq. 2   convergence    (1/D) ||x^{k+1}_i - x^k_i||^2 <= tau
 *   Sec. 2.2, Eq. 3   cache map      C: t -> (xhat_t, ehat_t)
 *   Sec. 2.2, Eq. 4   cache distance delta_t = (1/D) ||x_t - xhat_t||_1
 *   Sec. 2.2, Eq. 5   hit iff delta_t < tau_cache; first entry is a miss
 *   Sec. 2.2, Eq. 6   eps_t = ehat_t (hit) or eps_theta(x_t, t) (miss)
 *   Sec. 2.2, Eq. 7   cache update for misses only
 *
 * Call order:  pa_create -> pa_init -> ( pa_step -> denoise -> pa_submit_eps )*
 *              -> pa_step returns PA_DONE -> pa_result -> pa_destroy.
 * pa_step_async / pa_poll are the host-sync-free variant of pa_step for
 * denoisers that read the miss count on the device (e.g. pa_gmm_eps).
 * Any other order returns PA_ERR_STATE and changes nothing.
 *
 * Conventions
 *  - Latents are fp32, contiguous, NCHW-flattened: one row of D = prod(shape)
 *    floats per timestep.
 *  - Sampling index 0 is the noisiest state (x_0 of Eq. 1 is the initial
 *    noise); alphas_cumprod has T+1 entries and entry T is the clean end (1.0).
 *  - Misses are ordered trajectory-major, then by ascending timestep; the
 *    miss list holds int32 pairs (b, i): trajectory b, absolute timestep i.
 *  - Device memory: the caller owns every buffer. The solver's internal state
 *    lives in a caller-allocated device workspace of pa_workspace_bytes()
 *    bytes (256-byte aligned); the library never calls cudaMalloc. Pointers
 *    returned by pa_step stay valid until the next pa_submit_eps/pa_destroy.
 *  - Streams: every kernel and copy of a solver is issued on the stream given
 *    to pa_create (NULL = legacy default stream). A replay of a CUDA graph
 *    captured from that stream must be launched on it too: work of one handle
 *    running on two streams at once races on its workspace (torn plans and
 *    miss lists, which the kernels do not guard against).
 *  - Errors: every call returns a pa_status; nothing throws across the ABI.
 *    Device-side failures (a bounded wait that ran out, an index check) are
 *    recorded in a device status word and reported by the next call that
 *    synchronises (pa_step, pa_poll, pa_result, pa_stats).
 */
#ifndef PARAANYA_H
#define PARAANYA_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define PA_API __attribute__((visibility("default")))
#else
#define PA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pa_solver pa_solver;   /* opaque, owned by the library */
typedef struct pa_gmm pa_gmm;         /* opaque, owned by the library */

typedef enum {
  PA_OK = 0,
  PA_DONE = 1,           /* every trajectory reached t = T */
  PA_ERR_ARG = -1,       /* bad argument (size, pointer, alignment) */
  PA_ERR_STATE = -2,     /* call out of order */
  PA_ERR_CUDA = -3,      /* a CUDA runtime call failed */
  PA_ERR_WORKSPACE = -4, /* workspace too small or misaligned */
  PA_ERR_TIMEOUT = -5,   /* a device-side bounded wait ran out */
  PA_ERR_DEVICE = -6     /* a device-side consistency check failed */
} pa_status;

typedef struct {
  int64_t iters;         /* Picard iterations completed (global loop count) */
  int64_t nfe;           /* sum over iterations of misses (network evaluations) */
  int64_t hits;          /* sum over iterations of cache hits */
  int64_t launches;      /* kernels this handle launched since pa_create */
  int32_t n_active;      /* trajectories with t < T */
  int32_t n_miss;        /* misses planned for the next iteration */
  int32_t device_status; /* 0, or the first device-side error code */
  int32_t update_kernel; /* kernel of the last pa_submit_eps: 0 plain loads, 1 bulk forms,
                            2 lean register form, 3 fused step, 4 Anderson mixing
                            (pa_set_anderson), -1 none yet */
} pa_stats_t;

/* ---- solver ------------------------------------------------------------ */

/* Bytes of device workspace a solver of these sizes needs (0 on bad sizes).
 * T: DDIM steps (>= 1); window: P, evaluation points per iteration (1..1024);
 * D: latent size (>= 1); batch: independent trajectories (1..64). */
PA_API size_t pa_workspace_bytes(int T, int window, int64_t D, int batch);

/* Create a solver. latent_shape[ndim] gives D = prod(latent_shape).
 * alphas_cumprod: HOST array, T+1 doubles, sampling order (see above), each in
 *   (0, 1], non-decreasing not required. The DDIM drift coefficients of Sec. 2.1
 *   are derived from it on the host in fp64 and stored in fp32.
 * tol: tau of Eq. 2 (>= 0). cache_thresh: tau_cache of Eq. 5 (>= 0; 0 disables
 *   hits because the comparison is strict).
 * workspace_dev: device pointer, 256-byte aligned, >= pa_workspace_bytes().
 * stream: a cudaStream_t (may be NULL). The handle is written to *out. */
PA_API pa_status pa_create(pa_solver** out, int T, int window,
                    const int64_t* latent_shape, int ndim,
                    const double* alphas_cumprod, double tol, double cache_thresh,
                    int batch, void* workspace_dev, size_t workspace_bytes,
                    void* stream);

/* Stochastic steps (an extension beyond the paper's DDIM runs; eta = 1 over the
 * full 1000-step schedule is DDPM, the sampler of Table 2). Step i becomes
 * x_{i+1} = c_i x_i + e_i eps + sigma_i z_i with
 * sigma_i = eta sqrt((1 - a_{i+1}) / (1 - a_i)) sqrt(1 - a_i / a_{i+1}) and
 * e_i = sqrt(1 - a_{i+1} - sigma_i^2) - sqrt(a_{i+1} (1 - a_i) / a_i), so the
 * Picard drift (Eq. 1) gains sigma_i z_i. The draws z_i are fixed before
 * sampling (the paper is silent on stochastic samplers; this is the reading
 * that keeps Eq. 1 a deterministic recursion): noise_dev is a DEVICE array
 * [batch][T][D] fp32 of N(0, 1) draws, 16-byte aligned (else PA_ERR_ARG),
 * caller-owned, read by every following
 * iteration until the next pa_set_noise -- it must stay valid and unchanged
 * that long. eta = 0 (noise_dev may be NULL) restores plain DDIM. eta must be
 * in [0, 1]. Not allowed between pa_step and pa_submit_eps (PA_ERR_STATE);
 * takes effect from the next iteration (call pa_init to restart cleanly).
 * With draws the default update is the register-resident bulk form (or the
 * staged bulk form, which copies the draws into shared memory) when
 * D % 4 == 0 and the window fits; otherwise the plain-load kernel runs.
 * Synchronises the solver's stream. */
PA_API pa_status pa_set_noise(pa_solver* s, double eta, const float* noise_dev);

/* Start a generation: x_init [batch][D] fp32, HOST or DEVICE pointer (the copy
 * direction is inferred from the address). All states of the first window are
 * x_init (Sec. 2.1 initial trajectory estimate); every first-window timestep is
 * a first entry, hence a miss (Sec. 2.2). Clears the cache and counters,
 * plans the first iteration and gathers its batch (two kernels), all
 * asynchronous on the solver's stream. May be called again at any time to
 * restart. */
PA_API pa_status pa_init(pa_solver* s, const float* x_init);

/* The planned iteration: returns in *n_miss the number of misses M (Eq. 5),
 * in *batch_x_dev the contiguous batch [M][D] of their latents and in
 * *miss_bt_dev the (b, i) list [M][2]. The plan and the batch were made on
 * the device by pa_init (first iteration) or by the previous pa_submit_eps;
 * pa_step launches nothing and synchronises the solver's stream once (to read
 * M). Returns PA_DONE (and M = 0) when every trajectory has finished. */
PA_API pa_status pa_step(pa_solver* s, int* n_miss, const float** batch_x_dev,
                  const int32_t** miss_bt_dev);

/* As pa_step without synchronising: *n_miss_dev points to the device int32
 * holding M. The batch has room for batch*window rows; rows >= M are stale.
 * Iterating a finished solver is a no-op on the device. */
PA_API pa_status pa_step_async(pa_solver* s, const float** batch_x_dev,
                        const int32_t** miss_bt_dev, const int32_t** n_miss_dev);

/* Device address of the int32 holding the planned miss count M (the value
 * pa_step returns); valid for the solver's lifetime. NULL for a NULL solver. */
PA_API const int32_t* pa_n_miss_dev(const pa_solver* s);

/* Hand back eps_theta for the planned misses: batch_eps_dev [M][D] fp32,
 * DEVICE pointer, 16-byte aligned for the fused, lean and bulk update forms
 * (otherwise the plain-load kernel runs). Runs Eq. 6 (assembly), Eq. 7 (cache update),
 * the drift and the Picard prefix sum (Eq. 1), the errors of Eq. 2 and the
 * cache distances of the next iteration (Eq. 4), then the window advance
 * (Sec. 2.1), the hit-miss plan of the next iteration (Eq. 5) and the gather
 * of its batch (Sec. 2.2, one batched pass): by default in an update kernel
 * followed by a planning kernel, or (pa_set_update_kernel 3) in one fused
 * kernel when all of its CTAs fit on the GPU at once -- a cooperative launch
 * with a bounded grid barrier. Asynchronous on the solver's stream;
 * batch_eps_dev must stay valid until the update has run. */
PA_API pa_status pa_submit_eps(pa_solver* s, const float* batch_eps_dev);

/* Synchronise and report: *n_active = trajectories not yet at t = T.
 * Returns PA_DONE when it is 0, or a device error status. */
PA_API pa_status pa_poll(pa_solver* s, int* n_active);

/* Final states x_T [batch][D] fp32 into a HOST or DEVICE pointer: the end
 * point of Eq. 1's trajectory once the sliding window has reached T
 * (Sec. 2.1: the window advances until every state has converged by Eq. 2).
 * Valid once pa_step/pa_poll returned PA_DONE; PA_ERR_STATE before.
 * Synchronises. */
PA_API pa_status pa_result(pa_solver* s, float* x_out);

/* pa_poll and pa_result behind one synchronisation, for callers that poll in
 * a loop (Solver.generate): enqueues the copy of the counters and the copy of
 * the states at t = T into x_out (HOST or DEVICE, [batch][D] fp32), waits for
 * the stream once, then reports like pa_poll. When it returns PA_DONE, x_out
 * holds x_T (Eq. 1's end point, Sec. 2.1) exactly as pa_result would write it;
 * with PA_OK (trajectories still active) x_out holds the states then stored
 * in the slot of x_T, which the caller overwrites by a later call. A device
 * error status as pa_poll. PA_ERR_STATE before pa_init or between
 * pa_step_async and pa_submit_eps. */
PA_API pa_status pa_poll_result(pa_solver* s, float* x_out, int* n_active);

/* pa_poll_result split in two so that the caller can enqueue more work
 * before it waits (Solver.generate without waiting enqueues the next
 * generation behind the poll of the previous one, so the GPU does not idle
 * while the host reads the counters). pa_poll_begin enqueues, on the solver's
 * stream, the copy of the
 * states at t = T into x_out (HOST or DEVICE, [batch][D] fp32; NULL: no copy)
 * and of the counters into one of two pinned mirrors, and returns without
 * waiting; x_out must stay allocated and unread until the matching
 * pa_poll_end. pa_poll_end waits for the OLDEST pending pa_poll_begin's
 * copies and reports its counters like pa_poll: PA_DONE when no trajectory
 * was active at that point (x_out of that poll holds x_T, Eq. 1's end point,
 * Sec. 2.1, exactly as pa_result writes it), PA_OK otherwise, or a device
 * error status. Iterations enqueued after every trajectory reached T change
 * nothing, so a later pending poll copies the same x_T. At most two polls
 * pending: a third pa_poll_begin returns PA_ERR_STATE, as does pa_poll_end
 * with none pending, pa_poll_begin before pa_init, between pa_step_async and
 * pa_submit_eps, or while the stream is being captured. Pending polls
 * survive pa_init: each reports the counters as they stood at its own
 * pa_poll_begin in stream order. */
PA_API pa_status pa_poll_begin(pa_solver* s, float* x_out);
PA_API pa_status pa_poll_end(pa_solver* s, int* n_active);

/* The device-driven generation loop: Sec. 2.1's outer loop (slide the window
 * until every trajectory has reached T, Eq. 1 and 2) run by the GPU itself,
 * with no host round trip per iteration or per chunk. pa_loop_capture_begin
 * (after pa_init or any even number of iterations) builds a CUDA graph of one
 * conditional WHILE node and starts capturing the solver's stream into the
 * node's body; the caller then
 * issues an even number n >= 2 of iterations (pa_step_async, its denoiser's
 * launches on the solver's stream reading the miss count on the device,
 * pa_submit_eps; an even number because the iterations alternate two plan
 * copies); pa_loop_capture_end appends a one-thread kernel that sets the
 * node's condition (repeat while a trajectory is active, the device status is
 * clean and fewer than T / n + 2 passes have run: the window advances at
 * least one step per iteration, so T iterations always suffice, and the pass
 * limit bounds the loop whatever the counters say; iterations after the end
 * do nothing), closes the capture and instantiates the graph. Nothing runs
 * during the capture, and the host state returns to what it was at
 * pa_loop_capture_begin. pa_loop_launch(s, x_init) is pa_init followed by the
 * whole loop: it enqueues the copy of x_init ([batch][D] fp32, HOST or
 * DEVICE) into state 0, pa_init's kernel (the first plan, its batch, cleared
 * sums and counters, the loop's pass counter among them) and one launch of
 * the graph, and returns; then
 * pa_poll_begin (or pa_poll_result) reads the outcome. Host stepping
 * (pa_step_async) is refused until the next pa_init. The captured launches
 * carry the settings of the capture: every setter of this handle drops the
 * loop (and is refused while a capture is open). One loop per handle; a new
 * capture replaces it. Errors: PA_ERR_ARG for NULL arguments; PA_ERR_STATE
 * for a call out of order (no capture open, a body of an odd number of
 * iterations or none, kernel timing enabled: its events cannot sit in a loop
 * body, a stream already being captured, a launch between pa_step_async and
 * pa_submit_eps or with nothing captured); PA_ERR_CUDA where the driver
 * refuses the conditional node or its instantiation, or where the capture
 * was invalidated (a synchronisation of the solver's stream during it, say);
 * the capture is closed either way, nothing is kept, and the stream stays
 * usable. The capture is relaxed: CUDA calls the thread makes meanwhile on
 * other work do not invalidate it. */
PA_API pa_status pa_loop_capture_begin(pa_solver* s);
PA_API pa_status pa_loop_capture_end(pa_solver* s);
PA_API pa_status pa_loop_launch(pa_solver* s, const float* x_init);

/* Network evaluations so far: the sum over iterations of the misses, i.e. of
 * |M| of Eq. 5 (hits reuse the cached eps of Eq. 6 and cost no evaluation),
 * the NFE that Table 1 and Table 3 count per image. Synchronises; -1 on
 * error. */
PA_API int64_t pa_nfe(pa_solver* s);

/* Counters, see pa_stats_t: the iterations, NFE and cache hits that the
 * paper reports (Table 1: NFE; Table 3: iterations, NFE and hits per image),
 * plus bookkeeping (launches, active trajectories, device status).
 * Synchronises. */
PA_API pa_status pa_stats(pa_solver* s, pa_stats_t* out);

/* Per-iteration log, HOST buffer out[max_iters][batch][8] int32:
 * (window start t, evaluation points p, misses of trajectory b, stride,
 *  evaluated frontier e before the iteration (states > e were lazy copies of
 *  state e), hits among window positions 1..p-1, window positions that had a
 *  cache entry, hits among them).
 * *n_iters receives the number of logged iterations. Synchronises. */
PA_API pa_status pa_iter_log(pa_solver* s, int32_t* out, int max_iters, int* n_iters);

/* The reductions of the most recent pa_submit_eps, HOST buffers [batch][window]
 * fp32: err_out[b][j] is Eq. 2's error of state t+j+1 and delta_out[b][j] the
 * Eq. 4 distance of timestep t+j+1 against its cache entry (valid for j < p-1).
 * Either pointer may be NULL. Synchronises. */
PA_API pa_status pa_last_reductions(pa_solver* s, float* err_out, float* delta_out);

/* Select the Picard-update kernel (all forms compute Eq. 1, 2, 4, 6 and 7 of
 * one iteration; they differ in rounding order only, never in a decision
 * beyond the decision-margin guard):
 *   3       the fused step: the lean register form's update, a grid barrier,
 *           the decision in every CTA and the next batch written from
 *           registers, one kernel per iteration; used when every CTA of its
 *           grid (ceil(D / 128) x batch) is resident at once and
 *           batch * window <= 1024, else form 2 runs;
 *   300 + n the fused step with lean launch shape n (0, 1, 4, 5 below; with
 *           stochastic steps 0, 1, 3, 4);
 *   0       plain loads (one thread per column; any D);
 *   1       the bulk forms: register-resident rows, or rows staged in shared
 *           memory by bulk copies for windows the registers cannot hold;
 *   2       the lean register form followed by the planning kernel (default
 *           when D % 4 == 0): 16-byte rows
 *           straight into registers, plain fp32 prefix sums, coefficients and
 *           ranks staged in shared memory; windows up to 112 points with
 *           deterministic steps, else it falls back to 1;
 *   100 + n bulk forms with launch shape n (0..12; columns per lane, warps per
 *           CTA, pipeline depth; 112 = the register-resident form);
 *   200 + n lean form with launch shape n: 0 by window, 1 = 16 warps x 7
 *           positions, 2 = 12 x 9, 3 = 8 x 4 and 4 = 8 x 8 (two CTAs per SM),
 *           5 = 8 x 4 (three CTAs per SM), 6 = 4 x 8 (four CTAs per SM);
 *           210 + n (n <= 4) the same with compensated (TwoSum) sums,
 *           deterministic steps only. Shapes 5 and 6 take deterministic steps
 *           only. A shape that cannot hold the window falls back to 1.
 * Forms 1 and 2 fall back to plain loads for a batch_eps pointer that is not
 * 16-byte aligned. A tuning aid; returns PA_ERR_ARG for an unknown value. */
PA_API pa_status pa_set_update_kernel(pa_solver* s, int kind);

/* ---- triangular Anderson mixing (ParaTAA-style update) ------------------
 * Sec. 2.1 names ParaTAA among the Picard-family samplers the cache plugs
 * into and Sec. 2.2 leaves the sampler's own update to it; the paper states
 * no formula for ParaTAA. This library's reading: every iteration first forms
 * the Picard map's value G_s (Eq. 1) and the residual R_s = G_s - X_s of each
 * window state s = t + j + 1, then mixes with the previous iteration's G'_s,
 * R'_s (history depth 1):
 *   gamma_j = sum_{j' <= j} <dR, R> / sum_{j' <= j} <dR, dR>, dR = R - R'
 *   (sums over D and over window positions up to j: a least-squares fit
 *   that is lower triangular in time; 0 for a zero denominator),
 *   X_s <- G_s - gamma_j (G_s - G'_s)
 * for states that were computed in the previous iteration, except window
 * position 0, whose Picard value is already exact (it depends only on the
 * converged window start); other states take X_s <- G_s. The cache test
 * (Eq. 4-5), the batch, Eq. 6-7, the convergence error (Eq. 2) of the mixed
 * iterate, the stride rule and the window advance are unchanged. Depth 0 is
 * plain Picard. One iteration is then three kernels (the mixing form of the
 * lean update, the mix kernel, the planning kernel) besides the denoiser.
 * ------------------------------------------------------------------------ */

/* Bytes of the second device workspace that mixing needs: G and R of every
 * window state by iteration parity (4 x batch x (window+1) x D fp32), the
 * Gram sums and one row per trajectory (the frontier state before the
 * iteration); 0 on bad sizes. */
PA_API size_t pa_anderson_workspace_bytes(int T, int window, int64_t D, int batch);

/* depth 1: mix every iteration, using workspace_dev (DEVICE, 256-byte
 * aligned, >= pa_anderson_workspace_bytes(), caller-owned, valid until depth
 * 0 is set or the solver is destroyed); depth 0: plain Picard (workspace
 * ignored). Needs D % 4 == 0, a window of at most 112 points and fp32 cache
 * entries (PA_ERR_ARG otherwise). Not between pa_step and pa_submit_eps
 * (PA_ERR_STATE); pa_init must follow. While mixing, pa_set_update_kernel's
 * choice does not apply and pa_stats reports update_kernel 4. */
PA_API pa_status pa_set_anderson(pa_solver* s, int depth, void* workspace_dev, size_t workspace_bytes);

/* ---- online adaptation of tau_cache ---------------------------------------
 * The paper's conclusion names an online adaptive tau_cache as future work and
 * states no rule. This library's reading: every trajectory keeps its own
 * tau_cache, starting at pa_create's cache_thresh; after each iteration, with
 * n_e of its window positions that had a cache entry and n_h hits among them
 * (Eq. 5):
 *   n_h / n_e <  target:  tau <- min(tau * (1 + rate), tau_max) if the window
 *                         advanced beyond its first position (stride > 1),
 *                         else tau holds (reuse is not raised while the window
 *                         stalls);
 *   n_h / n_e >= target:  tau <- max(tau / (1 + rate), tau_min);
 *   n_e = 0:              tau holds;
 * and the next iteration's hit test (Eq. 5) uses the new tau. All of it runs
 * in the planning kernel's decision (fp64 on the device, exactly as on the
 * host). rate = 0 switches adaptation off (tau_cache fixed, the default).
 * ------------------------------------------------------------------------ */

/* rate >= 0 (0: off), 0 <= target <= 1, 0 <= tau_min <= tau_max (tau_max may
 * be +inf). Needs batch * window <= 1024 when rate > 0. PA_ERR_ARG otherwise;
 * PA_ERR_STATE between pa_step and pa_submit_eps; pa_init must follow. */
PA_API pa_status pa_set_cache_adaptation(pa_solver* s, double rate, double target, double tau_min, double tau_max);

/* The tau_cache of the planned iteration's hit test, per trajectory, into a
 * HOST array of batch doubles (cache_thresh for every trajectory when
 * adaptation is off). PA_ERR_STATE before pa_init. Synchronises. */
PA_API pa_status pa_cache_thresholds(pa_solver* s, double* tau_out);

/* Storage precision of the cache entries (xhat, ehat of Eq. 3): 32 = fp32
 * (default), 16 = bfloat16, rounded to nearest even when an entry is written
 * (Eq. 7) and widened exactly when read. Not from the paper: a storage option
 * that halves the entries' bytes; the states, the fresh eps of a miss and all
 * arithmetic stay fp32, so a hit reuses the rounded eps and Eq. 4 measures the
 * distance to the rounded input. With 16 the update runs in the lean register
 * form (windows up to 112, deterministic steps; selecting 1 or 112 gives the
 * register-resident bulk form) or the plain-load kernel. Any time
 * except between pa_step and pa_submit_eps; the next call must be pa_init.
 * Returns PA_ERR_ARG for another value, PA_ERR_STATE in the wrong state. */
PA_API pa_status pa_set_cache_precision(pa_solver* s, int bits);

/* Fault-handling test hook: the number of tries (each may suspend for about
 * 10 us) after which an mbarrier wait of the bulk-copy update kernel counts
 * as timed out (default 2^17, about a second); the fused step's grid barrier
 * polls 16 times this many times. With 0 every such wait gives up at once:
 * the kernel records PA_ERR_TIMEOUT (read by the next synchronising call),
 * still drains its in-flight copies with the default bound, and leaves the
 * solver's numbers meaningless until pa_init. */
PA_API pa_status pa_debug_set_wait_limit(pa_solver* s, uint32_t polls);

/* Enable (1) or disable (0) CUDA-event timing of every Picard-update kernel
 * launch, recorded on the solver's stream directly around the launch. Inside
 * a stream capture the records become event nodes of the graph, recorded
 * again at every replay. */
PA_API pa_status pa_set_kernel_timing(pa_solver* s, int enable);

/* Sum of the update-kernel durations in ms, and how many launches were timed,
 * since the last reset. reset != 0 starts a new count. For a captured graph,
 * read with reset = 0 after each replay: the captured records hold that
 * replay's times. Synchronises. */
PA_API pa_status pa_kernel_timing(pa_solver* s, double* update_ms, int64_t* n_launches, int reset);

/* Timing aid: launches one kernel that does no work, with the programmatic
 * dependent launch attribute that the library's own kernels carry, on a
 * cudaStream_t (may be NULL). Placed between pa_submit_eps calls where the
 * denoiser would run (eps replayed from a recorded run), it keeps the solver
 * kernels' dependency structure -- each kernel reads before its dependency
 * wait only what was written two or more kernels back -- so that the solver
 * step can be timed alone. Not part of the method. */
PA_API pa_status pa_debug_gap(void* stream);

/* Release the solver handle (the host-side state machine of Sec. 2.1-2.2's
 * iteration: the window, the plan and the counters). The caller-owned
 * workspace, and with it the cache of Eq. 3, is not freed. Synchronises the
 * solver's stream first; NULL is a no-op. */
PA_API void pa_destroy(pa_solver* s);

/* ---- Parareal (SRDS-style) sampling with the same cache ------------------
 * Sec. 2.1 names Parareal-based samplers (SRDS: a coarse solver initialises,
 * fine solvers refine); Sec. 2.2 applies the output cache to their network
 * evaluations and leaves the Parareal update unchanged. The paper states no
 * more; this library's reading: blocks of s = ceil(sqrt(T)) DDIM steps
 * (N = ceil(T / s) blocks); coarse solver G_n = one DDIM jump across block n
 * from eps at its start; fine solver F_n = the block's DDIM steps;
 * iteration 0: U_{n+1} = G_n(U_n); iteration k: F_n(U_n^{k-1}) for all n, then
 * U_{n+1}^k = G_n(U_n^k) + F_n(U_n^{k-1}) - G_n(U_n^{k-1}) in block order;
 * converged when max_n (1/D) ||U_n^k - U_n^{k-1}||^2 <= tol (Eq. 2 on the block
 * boundaries) or k = N (Parareal is then exact); converged trajectories freeze.
 * One cache entry per (trajectory, sampling index), shared by coarse and fine
 * evaluations: hit iff an entry exists and its Eq. 4 distance < cache_thresh
 * (Eq. 5); misses are evaluated and stored (Eq. 7). Each evaluation stage (a
 * fine step of every block, or one coarse block) is one pa_srds_step /
 * denoise / pa_srds_submit_eps round, with the same batch_x / miss_bt
 * conventions as pa_step (misses trajectory-major, then by block).
 * ------------------------------------------------------------------------ */
typedef struct pa_srds pa_srds;

typedef struct {
  int64_t iters;         /* Parareal iterations completed (0 = coarse initialisation only) */
  int64_t nfe;           /* network evaluations (misses) */
  int64_t hits;          /* evaluations served by the cache */
  int64_t launches;      /* kernels this handle launched */
  int32_t n_active;      /* trajectories not yet converged */
  int32_t n_miss;        /* misses of the current stage */
  int32_t device_status;
  int32_t blocks;        /* N */
  int32_t block_steps;   /* s */
  int32_t reserved;
} pa_srds_stats_t;

/* Device workspace bytes (0 on bad sizes; batch <= 64, batch * N <= 2048). */
PA_API size_t pa_srds_workspace_bytes(int T, int64_t D, int batch);

/* Same conventions as pa_create (alphas_cumprod HOST [T+1], sampling order;
 * caller-owned 256-byte aligned DEVICE workspace; stream may be NULL). */
PA_API pa_status pa_srds_create(pa_srds** out, int T, const int64_t* latent_shape, int ndim,
                                const double* alphas_cumprod, double tol, double cache_thresh,
                                int batch, void* workspace_dev, size_t workspace_bytes, void* stream);

/* x_init [batch][D] fp32, HOST or DEVICE; clears the cache; restarts. */
PA_API pa_status pa_srds_init(pa_srds* h, const float* x_init);

/* Plan the next evaluation stage: cache test of its rows, compaction of the
 * misses into batch_x [n_miss][D] (library-owned, valid until the next
 * submit), miss_bt [n_miss][2] = (trajectory, sampling index). Synchronises
 * to read n_miss; PA_DONE once every trajectory has converged. */
PA_API pa_status pa_srds_step(pa_srds* h, int* n_miss, const float** batch_x, const int32_t** miss_bt);

/* pa_srds_step without host synchronisation: *n_miss_dev is the device
 * address of the miss count (for device-side denoisers such as pa_gmm_eps).
 * Stages issued after the last trajectory converged do nothing. */
PA_API pa_status pa_srds_step_async(pa_srds* h, const float** batch_x, const int32_t** miss_bt,
                                    const int32_t** n_miss_dev);

/* Device address of the current stage's miss count (NULL for a NULL handle). */
PA_API const int32_t* pa_srds_n_miss_dev(const pa_srds* h);

/* batch_eps [n_miss][D] fp32 DEVICE for the planned misses: applies the
 * stage (fine steps or coarse jump + correction), and after the last stage of
 * an iteration the convergence test. */
PA_API pa_status pa_srds_submit_eps(pa_srds* h, const float* batch_eps);

/* Synchronise; *n_active = trajectories still refining; PA_DONE when none. */
PA_API pa_status pa_srds_poll(pa_srds* h, int* n_active);

/* x_out [batch][D] (HOST or DEVICE) = U_N; only after PA_DONE. Synchronises. */
PA_API pa_status pa_srds_result(pa_srds* h, float* x_out);

PA_API pa_status pa_srds_stats(pa_srds* h, pa_srds_stats_t* out);

/* err_out [N][batch] fp32 HOST: the block-boundary error of every iteration
 * (rows of iterations not run are unspecified). Synchronises. */
PA_API pa_status pa_srds_errors(pa_srds* h, float* err_out);

/* A whole Parareal generation as one CUDA graph (the outer loop of Sec. 2.1's
 * SRDS-style sampler run by the GPU, no host round trip between stages): a
 * chain of conditional IF nodes, one per Parareal iteration 0..N, each body
 * that iteration's stages; iteration 0 always runs, iteration k only when the
 * finishing kernel of iteration k-1 (the convergence test above) found a
 * trajectory still active. pa_srds_loop_capture_begin, right after
 * pa_srds_init, starts capturing the sampler's stream; the caller then issues
 * every stage (pa_srds_step_async, its denoiser's launches on the same stream
 * reading the miss count on the device, pa_srds_submit_eps) until
 * pa_srds_step_async returns PA_DONE, i.e. all N + 1 iterations; the library
 * moves the capture from one IF body to the next at each iteration's end.
 * pa_srds_loop_capture_end instantiates the graph; nothing runs during the
 * capture, and the handle is back in its state after pa_srds_init.
 * pa_srds_loop_launch, after a pa_srds_init, enqueues the graph: on return
 * pa_srds_result (or pa_srds_poll) reads the outcome. No IF node loops, so
 * the graph always ends. The captured launches carry the settings of the
 * capture. Errors: PA_ERR_ARG for a NULL handle; PA_ERR_STATE for a call out
 * of order (capture_begin not right after pa_srds_init or with a capture
 * open; capture_end with none open or before every stage was issued: the
 * capture is then closed and dropped and pa_srds_init must follow; launch
 * with nothing captured or not right after pa_srds_init); synchronising calls
 * (pa_srds_step, _poll, _result, _stats, _init) are refused while a capture
 * is open; PA_ERR_CUDA where the driver refuses a conditional node (the
 * capture is closed either way). */
PA_API pa_status pa_srds_loop_capture_begin(pa_srds* h);
PA_API pa_status pa_srds_loop_capture_end(pa_srds* h);
PA_API pa_status pa_srds_loop_launch(pa_srds* h);

PA_API void pa_srds_destroy(pa_srds* h);

/* ---- synthetic denoiser: posterior-mean eps of an isotropic Gaussian mixture
 * (stand-in for the SD v1.5 UNet of Sec. 3.2; not part of the paper's method).
 * eps*(x) = sqrt(1-a)/v * (x - sqrt(a) * sum_k r_k mu_k),
 * v = a s^2 + 1 - a, r = softmax_k(-||x - sqrt(a) mu_k||^2 / (2v)), equal weights.
 * ------------------------------------------------------------------------ */

/* Bytes of device workspace for K components (1..128), latent size D, at most
 * max_rows rows per call and T sampling steps (0 on bad sizes). */
PA_API size_t pa_gmm_workspace_bytes(int K, int64_t D, int max_rows, int T);

/* means_dev: DEVICE [K][D] fp32, caller-owned, must outlive the handle.
 * alphas_cumprod: HOST [T+1] doubles (same array as the solver's).
 * max_rows: largest batch ever passed (the solver's batch * window). */
PA_API pa_status pa_gmm_create(pa_gmm** out, int K, int64_t D, const float* means_dev,
                        double std, const double* alphas_cumprod, int T,
                        int max_rows, void* workspace_dev, size_t workspace_bytes,
                        void* stream);

/* eps for rows r < *n_rows_dev (DEVICE int32) of batch_x_dev [max_rows][D]:
 * the timestep of row r is miss_bt_dev[2r+1]. Writes batch_eps_dev [.][D].
 * Asynchronous on the handle's stream. */
PA_API pa_status pa_gmm_eps(pa_gmm* g, const float* batch_x_dev, const int32_t* miss_bt_dev,
                     const int32_t* n_rows_dev, float* batch_eps_dev);

/* Synchronise the handle's stream and report a device-side failure of the
 * denoiser kernels (a bounded bulk-copy wait that ran out): PA_ERR_TIMEOUT.
 * The failure also shows in the output: the output kernel writes NaN into
 * every tile of a call whose waits ran out, and, the handle's accumulators
 * being incomplete from then on, into every later call's output; create a
 * new handle after a timeout. */
PA_API pa_status pa_gmm_check(pa_gmm* g);

/* Kernels launched by this handle since pa_gmm_create. */
PA_API int64_t pa_gmm_launches(const pa_gmm* g);

/* How pa_gmm_eps computes (a choice of this library; the paper has no
 * counterpart). form 2 (the default for K <= 16 when D is a multiple of 64):
 * one kernel -- a thread-block cluster of 16 CTAs per block of 8 rows, each CTA
 * one sixteenth of the columns; the partial dot products x . mu_k are summed
 * across the cluster through distributed shared memory and every CTA writes
 * its columns of eps from the row and mean tiles it staged once. form 1: the
 * dot products on the tensor cores (tcgen05, kind::tf32, every operand split
 * into two tf32 parts and three products summed, which keeps fp32 accuracy),
 * 128 rows x 64 columns per CTA, then an output kernel -- for 16 < K <= 64
 * and D % 128 == 0 the output contraction R M on the tensor cores as well (a
 * kernel that forms the responsibilities' split image, then 128 rows x 128
 * columns per CTA with the accumulators in TMEM); available when the GPU
 * is of the sm_100 family, D % 4 == 0 and the means are 16-byte aligned, and
 * the default when K > 16. form 0: fp32 FMA dot products on the CUDA cores,
 * then the output kernel. A call whose batch_x or batch_eps is not 16-byte
 * aligned uses form 0 (form 2 falls back to it). The forms agree to fp32
 * rounding; each is bitwise reproducible. Returns PA_ERR_ARG for a form that
 * is not available. */
PA_API pa_status pa_gmm_set_form(pa_gmm* g, int form);

/* The form pa_gmm_eps uses: 2, 1 or 0, -1 for NULL. */
PA_API int pa_gmm_form(const pa_gmm* g);

PA_API void pa_gmm_destroy(pa_gmm* g);

/* pa_gmm_eps without a handle and without any device allocation (the paper
 * has no counterpart; this is a deployment convenience).
 *
 * For callers that cannot allocate device memory when they run the denoiser:
 * plugins that only get buffers from their host framework, real-time loops
 * that forbid cudaMalloc/cudaFree after start-up, code that does not own the
 * device's allocator. The caller passes the inputs (means_dev [K][D],
 * alphas_cumprod on the HOST [T+1], batch_x_dev [n_rows][D], miss_bt_dev
 * [n_rows][2] whose second entries are sampling indices < T) and the output
 * batch_eps_dev [n_rows][D]; the dot products are formed on the CUDA cores
 * (pa_gmm_set_form's form 0), and results agree with pa_gmm_eps's to fp32
 * rounding.
 *
 * Scratch lives in one fixed 4 MiB device array inside this library (every
 * GPU that loads the library holds it until the process exits). Sizes whose
 * scratch (3T coefficients, K norms, two sets of n_rows*K int64 dot-product
 * accumulators) would exceed 4 MiB are rejected with PA_ERR_ARG and a message
 * naming the bytes needed; use pa_gmm_create/pa_gmm_eps then.
 *
 * Every call looks up the array's device address (cudaGetSymbolAddress) with
 * the caller's device current; the first call on a device also makes the
 * library's device code resident there, so make that first call before any
 * stream capture. Every call on a device shares the one array and overwrites
 * it (the status word, the accumulators and the row count are set afresh at
 * the start of each call), so calls whose work overlaps on the GPU -- on
 * different streams, or from different host threads without ordering -- race
 * and give wrong results. The call is asynchronous on `stream`: the
 * per-timestep scalars are formed on the device from alphas that travel in
 * the parameters of small set-up launches (one per 3000 timesteps), so
 * nothing on the host has to outlive the call and no host-to-device copy
 * blocks it. It calls no cudaMalloc, cudaFree or other allocating routine. A
 * bounded-wait timeout inside its kernels is recorded in the array's status
 * word, and the output rows of the tiles it affected are written as NaN. */
PA_API pa_status pa_gmm_eps_noalloc(const float* means_dev, int K, int64_t D, double std,
                                    const double* alphas_cumprod, int T,
                                    const float* batch_x_dev, const int32_t* miss_bt_dev,
                                    int n_rows, float* batch_eps_dev, void* stream);

/* ---- misc -------------------------------------------------------------- */

PA_API const char* pa_status_string(int status);
/* Last host-side error message of this thread ("" if none). */
PA_API const char* pa_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* PARAANYA_H */
