/*
 * lipz.h -- C ABI of the GB300 grid-iteration engine for Lipizzaner-style coevolutionary GAN
 * training (arXiv 1811.12843, Section 3 "Coevolutionary GAN Training", steps 1-3 and 5).
 *
 * A grid is an R x C torus of cells. Every cell holds one generator G (parameters u, learning
 * rate delta) and one discriminator D (parameters v, learning rate gamma), each with its Adam
 * state (Table 1: population size 1 per cell, Adam, tournament size 2). One grid iteration is
 *   1. lipz_eval_neighborhoods: every G of a cell's 5-cell von Neumann neighbourhood (centre,
 *      north, south, west, east; Section 2) is scored against every D of that neighbourhood on
 *      the cell's minibatch (Section 3, step 2);
 *   2. lipz_select_replace: size-2 tournaments on those fitnesses choose the individuals that
 *      become the cell's new centre (Section 3, step 3, first half);
 *   3. lipz_train_step: one gradient/Adam update of every cell's new centre pair (step 3,
 *      second half), written to the next population snapshot.
 * lipz_iterate runs the three calls n times. All device memory is owned by the grid; every
 * host pointer argument is owned by the caller and only read or written during the call.
 *
 * Conventions
 *   - Every call returns LIPZ_OK (0) or an error code; the message of the last failure of a
 *     grid is lipz_last_error(grid). No call throws, aborts or exits.
 *   - Calls are asynchronous on the grid's CUDA stream (lipz_set_stream) unless a host output
 *     pointer is given, in which case the call waits for the stream before returning.
 *   - One grid must not be used by two host threads at the same time.
 *   - Cells are numbered c = r * cols + q. Slot s of cell c is nbr[c][s] with s = 0 centre,
 *     1 north (r-1), 2 south (r+1), 3 west (q-1), 4 east (q+1), indices wrapping around.
 *   - Fitness is a loss for both populations (lower is better):
 *       L_D(i, j) = mean_b BCE(D_j(x_b), 1) + mean_b BCE(D_j(G_i(z_b)), 0)
 *       L_G(i, j) = mean_b BCE(D_j(G_i(z_b)), 1)
 *       f_G[c][i] = mean_j L_G(i, j),   f_D[c][j] = mean_i L_D(i, j).
 *   - Random draws: Philox4x32-10 (Salmon et al., SC'11) with key (seed lo, seed hi) and
 *     counter (block, cell, iteration, stream); the stream ids are LIPZ_STREAM_*.
 */
#ifndef LIPZ_H
#define LIPZ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define LIPZ_API __attribute__((visibility("default")))
#else
#define LIPZ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
enum {
  LIPZ_OK = 0,
  LIPZ_ERR_INVALID = 1,   /* bad argument (null grid, size mismatch, out-of-range field) */
  LIPZ_ERR_CUDA = 2,      /* a CUDA runtime/driver call failed; see lipz_last_error */
  LIPZ_ERR_OOM = 3,       /* device or pinned allocation failed */
  LIPZ_ERR_NONFINITE = 4, /* a loss or fitness came out NaN/Inf (first such cell in the message) */
  LIPZ_ERR_TIMEOUT = 5,   /* a bounded device-side wait expired (the kernel stopped early) */
  LIPZ_ERR_STATE = 6      /* call out of order (e.g. train before select) */
};

enum { LIPZ_MLP = 0, LIPZ_DCGAN64 = 1 };           /* network family */
enum { LIPZ_FP32 = 0, LIPZ_BF16 = 1 };              /* arithmetic of the matrix products */
enum { LIPZ_REPLACE_IF_BETTER = 0, LIPZ_REPLACE_ALWAYS = 1 };

/* Philox stream ids (fourth counter word). */
enum {
  LIPZ_STREAM_INIT_G = 1, LIPZ_STREAM_INIT_D = 2, LIPZ_STREAM_BATCH = 3, LIPZ_STREAM_NOISE = 4,
  LIPZ_STREAM_TOUR_G = 5, LIPZ_STREAM_TOUR_D = 6, LIPZ_STREAM_MUT_G = 7, LIPZ_STREAM_MUT_D = 8,
  LIPZ_STREAM_MIX = 9
};
/* Minibatch step k of an iteration draws its batch from stream LIPZ_STREAM_BATCH + stride * k and
 * its noise from LIPZ_STREAM_NOISE + stride * k (k = 0 is the evaluation minibatch). */
enum { LIPZ_STEP_STREAM_STRIDE = 256 };

/*
 * Architecture and hyper-parameters (Table 1, MLP column). Fill with lipz_arch_default and
 * change fields; struct_size must be sizeof(lipz_arch).
 *   G: z_dim -> hidden (ReLU) -> hidden (ReLU) -> x_dim (tanh)
 *   D: x_dim -> hidden (LeakyReLU leaky_slope) -> hidden (LeakyReLU) -> 1 (sigmoid in the loss)
 * precision LIPZ_BF16: weights, activations and back-propagated deltas enter every matrix
 * product rounded to bfloat16 (nearest even), products accumulate in fp32; biases, logits,
 * losses, gradients and the Adam state (fp32 master weights, m, v) stay fp32.
 * LIPZ_FP32: everything fp32. Constraints: z_dim, hidden, x_dim, batch >= 1; hidden <= 1024;
 * tournament_size in 1..5; the tensor-core path additionally needs hidden == 256 and z_dim,
 * x_dim multiples of 16 (other shapes run on the CUDA-core kernels).
 */
typedef struct lipz_arch {
  uint32_t struct_size;
  int32_t kind;            /* LIPZ_MLP, or LIPZ_DCGAN64 (see ngf) */
  int32_t precision;       /* LIPZ_FP32 or LIPZ_BF16 */
  int32_t z_dim;           /* 64 */
  int32_t hidden;          /* 256 */
  int32_t x_dim;           /* 784 */
  int32_t batch;           /* 100 */
  float lr;                /* 2e-4, initial learning rate of every G and D */
  float beta1;             /* 0.5 */
  float beta2;             /* 0.999 */
  float eps;               /* 1e-8 */
  int32_t tournament_size; /* 2 */
  int32_t replace_mode;    /* LIPZ_REPLACE_IF_BETTER */
  int32_t lr_mutation;     /* 0: off; 1: Gaussian lr mutation at selection */
  float lr_mut_std;        /* 1e-4 */
  float lr_mut_prob;       /* 0.5 */
  float leaky_slope;       /* 0.2 */
  int32_t keep_grads;      /* 1: keep the last train step's gradients for lipz_get_gradients */
  int32_t force_simt;      /* 1: run the forward on the CUDA-core kernels even where the
                              tensor-core kernels apply (for comparisons) */
  int32_t train_steps;     /* K >= 1 (default 1): Adam steps of each cell's new centre pair per
                              iteration. Step 0 uses the evaluation minibatch; step k >= 1
                              trains the pair again, in place, on a fresh minibatch drawn from
                              the pool with stream ids + LIPZ_STEP_STREAM_STRIDE * k (also when
                              the caller supplied step 0's real rows); selection and the lr
                              mutation happen once, before step 0. K <= 65536. */
  int32_t mixture;         /* 1: every evaluation also takes one ES-(1+1) step of each cell's
                              generator-mixture weights (Section 3 step 4); see
                              lipz_get_mixture. Default 0. */
  float mix_sigma;         /* 0.01: mixture mutation scale (Table 1) */
  int32_t stale_neighbors; /* 1: the asynchronous cells of Section 3, emulated deterministically:
                              an evaluation sees each cell's own centre as of the iteration and
                              its four neighbours as they were one iteration earlier (the first
                              iteration after create or lipz_import_state sees them as they
                              are); a selected neighbour brings that older individual with its
                              optimiser state. Needs train_steps == 1. Default 0. */
  int32_t ngf;             /* LIPZ_DCGAN64 (Table 1, CelebA column; the DCGAN architecture):
                              G: z_dim -> ConvT 4x4 -> 8ngf x 4 x 4 -> ConvT 4x4 /2 ->
                              4ngf x 8 x 8 -> 2ngf x 16 x 16 -> ngf x 32 x 32 (each batch norm in
                              training mode + ReLU) -> 3 x 64 x 64 tanh; weights [in][out][4][4] */
  int32_t ndf;             /* D: 3 x 64 x 64 -> Conv 4x4 /2 -> ndf x 32 x 32 -> 2ndf x 16 x 16 ->
                              4ndf x 8 x 8 -> 8ndf x 4 x 4 (each LeakyReLU) -> Conv 4x4 -> logit;
                              weights [out][in][4][4], no biases. Needs x_dim == 12288 (CHW
                              images), train_steps == 1. bf16 with ngf, ndf multiples of 64 runs
                              the convolutions on the tensor cores; fp32 and other widths on
                              the CUDA-core kernels. Layout
                              per generator: W1, gamma1, beta1, ..., W4, gamma4, beta4, W5;
                              initial weights N(0, 0.02^2), scales 1 + N(0, 0.02^2), shifts 0.
                              Default 64 (the 512/256/128/64 configuration). */
} lipz_arch;

typedef struct lipz_grid lipz_grid;

/* Writes the Table 1 MLP defaults (values in the comments above) into *arch. */
LIPZ_API int lipz_arch_default(lipz_arch* arch);

/*
 * Creates a rows x cols grid on the current CUDA device (Section 3, step 1): every G and D
 * gets Xavier-uniform weights (bound sqrt(6/(fan_in+fan_out)); element k of a weight tensor
 * from word k of its stream: w = a * (2 (word >> 8) + 1 - 2^24) / 2^24), zero biases, zero
 * Adam moments, step 0, lr = arch->lr. Needs rows, cols >= 1. The real-data pool starts
 * empty: call lipz_set_data before lipz_eval_neighborhoods / lipz_iterate.
 * Returns LIPZ_ERR_OOM if device memory runs out (nothing is leaked).
 */
LIPZ_API int lipz_grid_create(int rows, int cols, const lipz_arch* arch, uint64_t seed, lipz_grid** out);

/* Frees everything the grid owns. Null is accepted. */
LIPZ_API int lipz_grid_destroy(lipz_grid* g);

/* Runs the grid's work on `stream` (a cudaStream_t, owned by the caller), or on the grid's own
 * non-blocking stream (the default, created with the grid) when `stream` is null. Work already
 * queued completes first. On a created stream consecutive kernels use programmatic dependent
 * launch; on the legacy or per-thread default stream they keep plain stream order. */
LIPZ_API int lipz_set_stream(lipz_grid* g, void* stream);

/* Blocks until the grid's stream is idle; reports a non-finite loss or an expired bounded wait
 * seen since the last check, and completes a pending lipz_iterate_batch_async call (its
 * fitnesses are copied to the caller's buffers). */
LIPZ_API int lipz_synchronize(lipz_grid* g);

/*
 * Copies the real-data pool from host memory: n_rows rows of dim == x_dim fp32 values,
 * row-major, values expected in [-1, 1]. A minibatch row b of cell c at iteration t is pool
 * row mulhi(word_b, n_rows) of stream LIPZ_STREAM_BATCH (mulhi(w, n) = (w * n) >> 32).
 */
LIPZ_API int lipz_set_data(lipz_grid* g, const float* host_pool, int64_t n_rows, int32_t dim);

/*
 * Step 2 for every cell at the current iteration t: draws the cell's minibatch (x from the
 * pool, z: batch x z_dim normals by Box-Muller from stream LIPZ_STREAM_NOISE, block i's words
 * (w0..w3) giving normals 4i..4i+3), runs every (generator slot i, discriminator slot j) pair
 * and reduces the fitnesses. Host outputs (each may be null; any non-null output makes the
 * call synchronous): fit_g, fit_d [cells][5] fp32; pair_lg, pair_ld [cells][5 (i)][5 (j)].
 */
LIPZ_API int lipz_eval_neighborhoods(lipz_grid* g, float* fit_g, float* fit_d, float* pair_lg,
                            float* pair_ld);

/*
 * Step 3 (selection) for every cell: a tournament of arch->tournament_size distinct slots per
 * population (entrant m = the mulhi(word_m, 5 - m)-th slot not yet drawn, ascending; words
 * from LIPZ_STREAM_TOUR_G / _D), lowest fitness wins, the lower slot on a tie. The new centre
 * is the winner if it is strictly fitter than the centre (LIPZ_REPLACE_IF_BETTER) or always
 * (LIPZ_REPLACE_ALWAYS); it brings its weights, Adam moments, step count and learning rate.
 * With lr_mutation, the new centre's lr becomes max(lr + lr_mut_std * N(0,1), 1e-8) with
 * probability lr_mut_prob (words from LIPZ_STREAM_MUT_G / _D). Host outputs sel_g, sel_d
 * [cells] int32: the chosen slot (0 = centre kept); null allowed.
 * Must follow lipz_eval_neighborhoods of the same iteration, else LIPZ_ERR_STATE.
 */
LIPZ_API int lipz_select_replace(lipz_grid* g, int32_t* sel_g, int32_t* sel_d);

/*
 * Step 3 (training) for every cell: gradients of the new centre pair on the cell's minibatch
 * from the evaluation (dL_D/dv with the fake batch detached, dL_G/du through D, both at the
 * pre-update parameters), one Adam step (Kingma & Ba 2015, Algorithm 1) per individual, into
 * the next snapshot; the iteration counter advances. Must follow lipz_select_replace.
 */
LIPZ_API int lipz_train_step(lipz_grid* g);

/* n_iters times: eval, select, train (asynchronous on the grid's stream). */
LIPZ_API int lipz_iterate(lipz_grid* g, int n_iters);

/*
 * One grid iteration whose real minibatches come from the caller: x_host is [cells][batch]
 * [x_dim] fp32 in host memory (pinned memory makes the copy asynchronous-capable); z is still
 * drawn from LIPZ_STREAM_NOISE. fit_g / fit_d (host, [cells][5], nullable) receive the
 * iteration's fitnesses; the call returns after the iteration is complete.
 */
LIPZ_API int lipz_iterate_batch(lipz_grid* g, const float* x_host, float* fit_g, float* fit_d);

/*
 * The same, pipelined across calls: while this iteration computes, x_next (host, the same
 * shape, nullable) is uploaded into a second device staging buffer (allocated on the first
 * call, cells x batch x x_dim fp32), and the next call whose x_host is that same address
 * skips its upload. The caller must keep x_next's contents unchanged until that call; a call
 * with another x_host (or lipz_iterate_batch) uploads as usual and the early copy is dropped.
 * Results, errors and synchronisation as lipz_iterate_batch.
 */
LIPZ_API int lipz_iterate_batch_next(lipz_grid* g, const float* x_host, const float* x_next,
                                     float* fit_g, float* fit_d);

/*
 * The same one call ahead (a pipeline one iteration deep), for a caller that keeps the GPU
 * busy across calls: the call enqueues this iteration (and x_next's upload) and then waits
 * only for the PREVIOUS call's iteration. When it returns, the previous call's fit_g / fit_d
 * hold that iteration's fitnesses, and the return code reports the previous iteration's device
 * status (LIPZ_ERR_NONFINITE, LIPZ_ERR_TIMEOUT) or an error in enqueueing this one; the first
 * call returns without waiting. This call's fit_g / fit_d are written when the next call (or
 * lipz_synchronize) returns: the caller must leave them, x_host and x_next alone until then,
 * so two sets of result buffers alternate. lipz_synchronize completes the last call (its
 * fitnesses included) and reports its
 * status; any other call on the grid may report it instead. After an error the pipeline is
 * drained (this call's iteration has completed too and is not reported separately). An upload
 * into a staging buffer waits on the device for the iteration that last read it. Results are
 * bit-identical to lipz_iterate_batch on the same minibatches. Per iteration the fitnesses
 * and device status words are gathered on the device and come back in one copy into a pinned
 * slot of the grid; the fitnesses are copied into fit_g / fit_d (any host memory) when the
 * call completes.
 */
LIPZ_API int lipz_iterate_batch_async(lipz_grid* g, const float* x_host, const float* x_next,
                                      float* fit_g, float* fit_d);

/*
 * State I/O (checkpoint / resume, and state exchange with other implementations). Layout,
 * little-endian: a 64-byte header {u32 magic 0x5A50494C, u32 version 2, i32 rows, cols, z_dim,
 * hidden, x_dim, batch, precision, 0, i64 t, u64 seed, 8 zero bytes}, then f32 Gw[cells][PG],
 * Gm, Gv, Dw[cells][PD], Dm, Dv, i32 Gstep[cells], Dstep[cells], f32 Glr[cells], Dlr[cells],
 * f32 mix[cells][5] (generator-mixture weights).
 * PG, PD = parameter counts; each individual's vector is, in order, W1 [out][in], b1, W2, b2,
 * W3, b3 (PyTorch Linear layout). Import requires the same rows, cols and arch sizes; it
 * replaces the seed and iteration counter too. Both calls are synchronous.
 */
LIPZ_API int lipz_state_bytes(const lipz_grid* g, size_t* bytes);
LIPZ_API int lipz_export_state(lipz_grid* g, void* host, size_t bytes);
LIPZ_API int lipz_import_state(lipz_grid* g, const void* host, size_t bytes);

/* Current iteration counter t (number of completed train steps since creation/import). */
LIPZ_API int lipz_get_iteration(const lipz_grid* g, int64_t* t);

/* Inspection of the last evaluation (synchronous; valid after lipz_eval_neighborhoods):
 * x [cells][batch][x_dim] and z [cells][batch][z_dim] as fp32 (bf16 mode: the rounded values
 * the products used); logits [cells][5 (j)][6 * batch]: discriminator slot j on the cell's
 * real rows, then the fakes of generator slots 0..4. */
LIPZ_API int lipz_get_batch(lipz_grid* g, float* x, float* z);
LIPZ_API int lipz_get_logits(lipz_grid* g, float* logits);

/*
 * Generator mixtures (Section 3 step 4; synchronous, host pointers, each may be null).
 * weights [cells][5]: every neighbourhood's mixture weights over its generator slots 0..4
 * (initially 1/5; with arch.mixture each evaluation takes one ES-(1+1) step). blocks
 * [cells][6][6] and score [cells] (need arch.mixture, else LIPZ_ERR_STATE): of the last
 * evaluation, S[a][b] = mean over the rows r of block a and s of block b of
 * exp(-||e_r - e_s||^2 / x_dim), the blocks being the B real rows (0) and the fakes of
 * generator slots 0..4 (1..5) as the discriminators received them; score = the squared MMD
 * sum_ij w_i w_j S[1+i][1+j] - 2 sum_i w_i S[1+i][0] + S[0][0] of the weights kept. The step:
 * w' = max(w + mix_sigma n, 0) / sum (n: the first five normals of stream LIPZ_STREAM_MIX at
 * the iteration; w kept if the sum is 0) replaces w iff its squared MMD is lower. The score
 * stands in for the paper's FID (no Inception network here).
 */
LIPZ_API int lipz_get_mixture(lipz_grid* g, float* weights, float* blocks, float* score);

/* Gradients of the last train step (needs arch.keep_grads): gG [cells][PG], gD [cells][PD]. */
LIPZ_API int lipz_get_gradients(lipz_grid* g, float* grad_g, float* grad_d);

/*
 * Per-phase device timing (tracing). Phases: LIPZ_PHASE_BATCH (minibatch draw), _G_FWD and
 * _D_FWD (evaluation forward of all generator / discriminator slots), _FITNESS (BCE losses and
 * fitness), _SELECT, _TRAIN_FWD (forward of the selected pairs and the logit deltas),
 * _TRAIN_BWD (their backward; on the tensor-core path one kernel, which also applies Adam to
 * the weight matrices unless arch.keep_grads is set), _ADAM (bias gradients, then the rest of
 * the update and replacement), _MIXTURE (with arch.mixture: the mixture step at the end of
 * an evaluation). While enabled, every phase is bracketed by CUDA events on
 * the grid's stream. lipz_profile_read waits for the stream and writes, per phase, the summed
 * device milliseconds (ms[n]), the number of phase executions (count[n]) and of kernel launches
 * (launches[n]) since the last read (any pointer may be null; n <= LIPZ_N_PHASES), then resets.
 */
enum {
  LIPZ_PHASE_BATCH = 0, LIPZ_PHASE_G_FWD = 1, LIPZ_PHASE_D_FWD = 2, LIPZ_PHASE_FITNESS = 3,
  LIPZ_PHASE_SELECT = 4, LIPZ_PHASE_TRAIN_FWD = 5, LIPZ_PHASE_TRAIN_BWD = 6,
  LIPZ_PHASE_ADAM = 7, LIPZ_PHASE_MIXTURE = 8, LIPZ_N_PHASES = 9
};
LIPZ_API int lipz_profile_enable(lipz_grid* g, int enable);
LIPZ_API int lipz_profile_read(lipz_grid* g, double* ms, int64_t* count, int64_t* launches, int n);

/*
 * Fitness of every cell from logits already in device memory, allocating nothing.
 * Not part of the method: the paper has no counterpart. It is for callers that cannot call
 * cudaMalloc when they need the fitness: a serving loop whose device memory is fully reserved
 * by another allocator (a new allocation would fail), or a latency-critical path that cannot
 * afford the implicit synchronisation of cudaMalloc / cudaFree. The per-pair losses that the
 * computation needs go to one file-scope device array of about 800 KB, which every GPU that
 * loads this library holds until the process exits.
 *   logits: device, [cells][5 (j)][6 * batch] fp32, laid out as lipz_get_logits returns it;
 *   fit_g, fit_d: device outputs [cells][5] fp32 (as lipz_eval_neighborhoods computes them);
 *   stream: the cudaStream_t to run on (0 = legacy default). The call is asynchronous.
 * The library cannot check device buffers: they must hold the sizes above.
 * Limits: 1 <= cells <= LIPZ_NOALLOC_MAX_CELLS and batch >= 1, else LIPZ_ERR_INVALID with
 * nothing launched; a null pointer also gives LIPZ_ERR_INVALID. LIPZ_ERR_CUDA if a CUDA call
 * fails. The first call on a device looks up the array's device address (once per device,
 * with that device current) and keeps it for the life of the process: make that first call
 * before any stream capture, and do not use the call across a cudaDeviceReset (the array
 * moves with the device's primary context). All calls share the array, and each call
 * overwrites what it uses, so two calls whose work overlaps on the GPU (different streams,
 * no ordering) race. Non-finite losses are reported only through NaN/Inf fitness values
 * (lipz_eval_neighborhoods returns LIPZ_ERR_NONFINITE for them; this call has no channel).
 */
#define LIPZ_NOALLOC_MAX_CELLS 4096
LIPZ_API int lipz_fitness_from_logits_noalloc(const float* logits, int32_t cells, int32_t batch,
                                             float* fit_g, float* fit_d, void* stream);

/* Message of the grid's last failure ("" if none); for a null grid, of the last failed
 * lipz_grid_create on this thread. The pointer stays valid until the next call on the grid. */
LIPZ_API const char* lipz_last_error(const lipz_grid* g);

/* Static text for a status code. */
LIPZ_API const char* lipz_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif /* LIPZ_H */
