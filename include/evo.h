/*
 * evo.h -- C ABI of the GB300 schedule-driven cached denoiser (EVO hot path).
 *
 * The library runs the reverse diffusion loop of a transformer diffusion
 * policy on one GPU.  For every cacheable unit b (self-attention,
 * cross-attention and FFN residual branch of each decoder layer; B = 3L units,
 * Sec. 3.1) and every loop step t in {0..T-1}, a binary lattice S decides
 * whether the unit is recomputed -- its residual output r_{b,t} is written to
 * the unit's activation cache c_b -- or replaced by the cached c_b (Eq. 1).
 * Caches are reset at the start of every action query (Sec. 3.1, Sec. 3.4).
 * The sampler, weights and action interface are those of the policy and do
 * not change with S (Sec. 3.4).
 *
 * Conventions for every entry point:
 *  - Return value: an evo_status.  Argument and shape errors are detected on
 *    the host before anything is launched and nothing is written.
 *  - Device pointers are plain CUDA device addresses (for example from
 *    torch tensors); "stream" is a cudaStream_t passed as void* (NULL = the
 *    legacy default stream).  Work is asynchronous on that stream.
 *  - All floating-point buffers are float32, C-contiguous, in the layouts
 *    given below.  The caller owns every buffer it passes; the handle owns
 *    the packed weights, the activation caches and its workspace.
 *  - Errors found on the device (a schedule read from device memory with an
 *    entry outside {0,1}, or a wait that timed out) are recorded in the
 *    handle's status word; evo_get_status() reads and clears it.  With
 *    cfg.debug_sync = 1 every call synchronizes and returns that status.
 *  - A handle may be used from one stream at a time.
 */
#ifndef EVO_H
#define EVO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct evo_handle evo_handle;

typedef enum {
  EVO_OK = 0,
  EVO_ERR_ARG = 1,          /* null pointer, bad enum value, non-positive size */
  EVO_ERR_SHAPE = 2,        /* shape not supported or batch above max_batch */
  EVO_ERR_SCHEDULE = 3,     /* lattice entry outside {0,1}, wrong row count, duplicate position */
  EVO_ERR_CUDA = 4,         /* a CUDA runtime call failed */
  EVO_ERR_TIMEOUT = 5,      /* a device-side wait exceeded its iteration limit */
  EVO_ERR_OOM = 6,          /* device allocation failed */
  EVO_ERR_UNSUPPORTED = 7,  /* no GPU with cluster launch, or the shape does not fit on chip */
  EVO_ERR_CORRUPT = 8       /* a guard band around an activation buffer was overwritten, or (debug
                               build) a device-side index check failed */
} evo_status;

enum { EVO_SAMPLER_DDPM = 0, EVO_SAMPLER_DDIM = 1 };
enum { EVO_DTYPE_F32 = 0, EVO_DTYPE_BF16 = 1 };
/* Empty-cache policy for a unit that has not been refreshed yet in the
 * current query: ZERO adds nothing (the reset cache is a zero tensor);
 * FORCE computes the unit at that first use even if S skips it. */
enum { EVO_EMPTY_ZERO = 0, EVO_EMPTY_FORCE = 1 };

typedef struct evo_config {
  int32_t n_layer;      /* L decoder layers; B = 3L cacheable units */
  int32_t n_emb;        /* E */
  int32_t n_head;       /* attention heads, E % n_head == 0 */
  int32_t horizon;      /* H action tokens per sample (<= 32) */
  int32_t action_dim;   /* A */
  int32_t n_obs;        /* observation tokens; memory = 1 timestep token + n_obs */
  int32_t obs_dim;      /* D */
  int32_t n_steps;      /* T loop steps (lattice columns) */
  int32_t train_steps;  /* diffusion training steps of the noise schedule (n_steps divides it) */
  int32_t sampler;      /* EVO_SAMPLER_* */
  int32_t dtype;        /* EVO_DTYPE_*: arithmetic/storage type of weights, GEMM operands and caches */
  int32_t empty_cache;  /* EVO_EMPTY_* */
  int32_t cluster;      /* CTAs that cooperate on one job; 0 = choose per call: the handle packs every
                           compiled decomposition of the model (16, 8, 4 CTAs) and a call takes the one
                           with the fewest estimated rounds of jobs for its batch */
  int32_t job_samples;  /* samples per job (rows = job_samples * horizon); 0 = choose */
  int32_t debug_sync;   /* 1: synchronize after each call and return the device status */
  int32_t wide_rows;    /* batch-wide tensor-core path for calls of at least this many action-token
                           rows (samples x horizon); 0 = 1024; < 0 = never.  bf16 with n_emb 256 or
                           512, head size 64, horizon 16 or 32, action dim <= 16, at most 7
                           observation tokens */
} evo_config;

/* Number of float32 values in the weight blob for cfg (0 if cfg is invalid).
 * Blob order (matrices are [in][out], y = x W):
 *   obs_w[D][E] obs_b[E] cond_pos[1+n_obs][E] cm_w1[E][4E] cm_b1[4E] cm_w2[4E][E] cm_b2[E]
 *   in_w[A][E] in_b[E] pos[H][E]
 *   per layer l = 0..L-1:
 *     ln1_g[E] ln1_b[E] sa_wqkv[E][3E] sa_bqkv[3E] sa_wo[E][E] sa_bo[E]
 *     ln2_g[E] ln2_b[E] ca_wq[E][E] ca_bq[E] ca_wkv[E][2E] ca_bkv[2E] ca_wo[E][E] ca_bo[E]
 *     ln3_g[E] ln3_b[E] ff_w1[E][4E] ff_b1[4E] ff_w2[4E][E] ff_b2[E]
 *   lnf_g[E] lnf_b[E] head_w[E][A] head_b[A]
 * (sa_wqkv columns are [q | k | v], ca_wkv columns are [k | v], each E wide.) */
size_t evo_weight_count(const evo_config* cfg);

/* Create a handle: copies the HOST weight blob (n_floats values, layout of
 * evo_weight_count) to the device, packs it for the kernels, precomputes the
 * timestep-token keys/values of every step, and sizes caches and workspace
 * for up to max_batch samples per call (evo_denoise: N; population: (P+1)*N_obs).
 * The current CUDA device at the time of the call is the handle's device. */
evo_status evo_create(const float* weights, size_t n_floats, const evo_config* cfg,
                      int32_t max_batch, evo_handle** out);

evo_status evo_destroy(evo_handle* h);

/* One action query per sample (Sec. 3.4 deployment, Eq. 1 inside the sampler loop).
 *   obs    device [N][n_obs][obs_dim]   observation condition features
 *   noise  device [n_noise][N][H][A]    slot 0 = initial x; DDPM: slot 1+t = z of loop step t
 *                                       (n_noise = T+1); DDIM: n_noise = 1
 *   S      [S_rows][T] uint8 lattice, host or device memory.  S_rows = 3L (unit rows
 *          b = 3l + {0 SA, 1 CA, 2 FFN}) or L (row l covers the three units of layer l).
 *          A host lattice is validated before launch; a device lattice is checked on the
 *          device (EVO_ERR_SCHEDULE in the status word, outputs untouched), except on
 *          the batch-wide path, which copies it to the host (one synchronisation) and
 *          returns EVO_ERR_SCHEDULE before any launch.
 *   out    device [N][H][A]             final actions (normalised space, after T steps)
 */
evo_status evo_denoise(evo_handle* h, const float* obs, const float* noise,
                       const uint8_t* S, int32_t S_rows, int32_t N,
                       float* out_actions, void* stream);

/* Batched candidate evaluation in one launch: P schedules, each applied to the
 * same N_obs observations and noise, plus the all-refresh schedule as a
 * reference.  dev_l2[p] = mean_n || x_{p,n} - x_full,n ||_2 over the H*A action
 * values (the candidates' cost for the search of Sec. 3.2).
 *   obs    device [N_obs][n_obs][obs_dim]
 *   noise  device [n_noise][N_obs][H][A]
 *   S_pop  [P][S_rows][T] uint8, host or device
 *   out_actions device [P][N_obs][H][A] or NULL
 *   dev_l2 device [P]
 */
evo_status evo_denoise_population(evo_handle* h, const float* obs, const float* noise,
                                  const uint8_t* S_pop, int32_t P, int32_t S_rows, int32_t N_obs,
                                  float* out_actions, float* dev_l2, void* stream);

/* Exact per-sample FLOPs of one action query under S (host memory), in the
 * convention 2 FLOPs per multiply-accumulate of every matmul (attention score
 * and value products over the full H x H / H x (1+n_obs) matrices): T times the
 * fixed per-step work (observation embedding, condition MLP, input and output
 * projections) plus, for every refreshed lattice cell (Eq. 2's |S| cells), the
 * FLOPs of that unit.  Under EVO_EMPTY_FORCE a row whose first entry is 0 adds
 * one refresh. */
evo_status evo_flops(const evo_handle* h, const uint8_t* S, int32_t S_rows, int64_t* flops_per_sample);
/* The same count for a configuration without a handle; only the shape fields
 * (and empty_cache) matter, and any positive model is accepted. */
evo_status evo_flops_cfg(const evo_config* cfg, const uint8_t* S, int32_t S_rows, int64_t* flops_per_sample);

/* Individual encoding of Eq. 3 -> lattice.  bt: K pairs (b, t) in host memory;
 * writes S_out[n_units][T] (host).  Rejects positions outside the lattice and
 * duplicates (EVO_ERR_SCHEDULE); S_out is written only on success. */
evo_status evo_schedule_from_positions(const int16_t* bt, int32_t K, int32_t n_units, int32_t T,
                                       uint8_t* S_out);

/* Fixed-interval baseline schedule (EfficientVLA, as the paper describes it:
 * every unit refreshed synchronously at a fixed temporal interval, M refreshes
 * per unit): S_out[n_units][T] (host) has ones at t_i = floor(i * T / M),
 * i = 0..M-1, in every row.  1 <= M <= T. */
evo_status evo_schedule_fixed_interval(int32_t n_units, int32_t T, int32_t M, uint8_t* S_out);

/* Debug variant of evo_denoise that also records the residual added at every
 * lattice cell: trace device [T][3L][N][H][E] float32 (refreshed cells: r_{b,t};
 * skipped cells: the cached c_b as stored; empty cache under ZERO: 0).  Takes
 * the same path (one cluster per job, or batch-wide) as evo_denoise would. */
evo_status evo_denoise_trace(evo_handle* h, const float* obs, const float* noise,
                             const uint8_t* S, int32_t S_rows, int32_t N,
                             float* out_actions, float* trace, void* stream);

/* Profiling hook: when both events are non-NULL (cudaEvent_t passed as void*),
 * every launch of the denoising-loop kernel is bracketed by cudaEventRecord
 * of `start` and `stop` on the call's stream, so a caller can read that
 * kernel's own duration.  Pass NULL, NULL to turn it off. */
evo_status evo_set_profile_events(evo_handle* h, void* start, void* stop);

/* evo_denoise for callers that cannot allocate device memory when they run a
 * query: a real-time control loop that forbids allocation once it has
 * started (an allocation can block for an unbounded time), or an application
 * whose own allocator reserved the device's memory up front, so that a
 * cudaMalloc behind its back would fail or fragment that pool.  The paper has
 * no counterpart; this is an interface choice.  Arguments, layouts and
 * results are those of evo_denoise, and it always takes the one-cluster-per-job
 * path, so its output is bit-identical to an evo_denoise call that takes that
 * path.  The per-call scratch (the observation tokens' cross-attention
 * keys/values and the condition MLP's intermediates) lives in one file-scope
 * device array of 8 MiB that every GPU which loads this library holds until
 * the process exits; N * n_obs * (2 * n_layer + 6) * n_emb * 4 bytes must fit
 * in it (186 samples of the Push-T-shaped model), else EVO_ERR_SHAPE and
 * nothing is launched.  No cudaMalloc, cudaFree or allocating library routine
 * is called.  The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) and keeps it for later calls.  All calls share the
 * array and every call overwrites all of it
 * that it reads, so nothing needs clearing; calls that overlap on the GPU
 * (other streams, other handles) race on it.  The handle's device must be the
 * current device (EVO_ERR_ARG otherwise). */
evo_status evo_denoise_noalloc(evo_handle* h, const float* obs, const float* noise,
                               const uint8_t* S, int32_t S_rows, int32_t N,
                               float* out_actions, void* stream);

/* Diagnostic of the device-side failure path (the paper has no counterpart).
 * Every wait in the library's kernels is bounded: when it gives up, the kernel
 * records EVO_ERR_TIMEOUT in the handle's status word and ends instead of
 * hanging.  This entry point exercises that path safely: one thread of one
 * block (no cluster, no asynchronous copy, no tensor memory) waits on a
 * barrier that nothing arrives at, through the same wait helper as the
 * denoising-loop kernel (helper 0, limit in SM cycles, 1..10^7) or the
 * tensor-core kernels (helper 1, limit in polls, 1..10^5), so the wait runs
 * out.  Afterwards evo_get_status() returns EVO_ERR_TIMEOUT once (and clears
 * it); the handle stays usable.  EVO_ERR_ARG for other helpers or limits. */
evo_status evo_test_wait_timeout(evo_handle* h, int32_t helper, int64_t limit, void* stream);

/* Diagnostic of the feed-forward activation (the paper has no counterpart).
 * The FFN units of both paths apply GELU in its erf form, x·Phi(x) =
 * x/2 (1 + erf(x / sqrt 2)) (the denoiser of Sec. 3.1), evaluating erf with
 * formula 7.1.26 of Abramowitz & Stegun (absolute error <= 1.5e-7).  This
 * entry point applies that same device code to n fp32 values: y[i] =
 * GELU(x[i]), x and y DEVICE pointers (caller-owned, n floats each; they may be
 * the same buffer), asynchronous on `stream`.  packed = 0 runs the scalar form
 * of the denoising-loop kernel, packed = 1 the two-value (f32x2) form of the
 * tensor-core GEMM epilogue; the two give identical bits.  EVO_ERR_ARG for
 * n < 0, another `packed`, or host / null pointers; n = 0 launches nothing. */
evo_status evo_test_gelu(const float* x, float* y, int64_t n, int32_t packed, void* stream);

/* Debug aid (the paper has no counterpart): every activation buffer of the
 * handle (unit caches, and on the batch-wide path the residual stream and the
 * GEMM operands) is allocated with a 4 KiB guard band of a fixed pattern on
 * each side.  Synchronizes the handle's last stream and checks every band:
 * EVO_OK if all are intact, EVO_ERR_CORRUPT if a kernel wrote past a buffer. */
evo_status evo_check_guards(evo_handle* h);

/* Synchronizes the handle's last stream, returns and clears the device status word. */
evo_status evo_get_status(evo_handle* h);

/* Launch geometry chosen at create: CTAs per job cluster, samples per job,
 * clusters resident at once, dynamic shared memory per CTA (bytes). */
evo_status evo_get_launch_info(const evo_handle* h, int32_t* cluster, int32_t* job_samples,
                               int32_t* max_clusters, int32_t* smem_bytes);

/* How the handle's last call ran: path 0 = one cluster per job (the persistent
 * denoising-loop kernel), 1 = batch-wide (step-synchronous over all samples,
 * tensor-core GEMMs); kernels = kernel launches of that call. */
evo_status evo_get_last_call(const evo_handle* h, int32_t* path, int64_t* kernels);

/* Redundancy-aware initialisation (Sec. 3.3).
 *
 * Dissimilarity map of Eq. 6 and its variants from the residual activations of
 * the uncached policy: trace = the device output of evo_denoise_trace with the
 * all-refresh lattice, [T][U][N][n] fp32 (n = H*E entries per activation).
 * For every unit b and step t, d[b][t] = mean over the N samples of
 * 1/(T-1) sum_{t' != t} D(a_t, a_t'), with D by metric:
 *   EVO_METRIC_COSINE  1 - cosine similarity (Eq. 6; a zero activation counts as 1)
 *   EVO_METRIC_MSE     mean squared difference of the entries
 *   EVO_METRIC_L1      mean absolute difference of the entries
 *   EVO_METRIC_W1      Wasserstein-1 distance between the entries' empirical
 *                      distributions (mean |sorted a_t - sorted a_t'|); n a power of two <= 16384
 *   d       device [U][T] fp32 (output)
 *   scratch device, evo_redundancy_scratch_bytes(...) bytes, caller-owned
 * 2 <= T <= 128.  Asynchronous on the stream; deterministic. */
enum { EVO_METRIC_COSINE = 0, EVO_METRIC_MSE = 1, EVO_METRIC_L1 = 2, EVO_METRIC_W1 = 3 };
size_t evo_redundancy_scratch_bytes(int32_t T, int32_t U, int32_t N, int32_t n, int32_t metric);
evo_status evo_redundancy_map(const float* trace, int32_t T, int32_t U, int32_t N, int32_t n, int32_t metric,
                              float* d, void* scratch, void* stream);

/* Guided sampling of P fixed-budget schedules (Eq. 7): K distinct lattice
 * cells each, drawn without replacement with probability proportional to
 * (eps + w)^gamma, w = d / max d (d > 0).  The weights are taken in fixed
 * point, q = floor((eps + w)^gamma * 2^40) (double precision, gamma a positive
 * integer <= 16), and draw k of schedule p takes, among the cells not yet
 * drawn in index order (b * T + t), the first whose running sum of q exceeds
 * rnd[p][k] mod (sum of the remaining q), or the first cell not yet drawn
 * when only zero weights remain -- exact integer arithmetic, so the
 * result is reproducible bit for bit.
 *   d    device [U][T] fp32, U * T <= 4096
 *   rnd  device [P][K] unsigned 64-bit random integers (caller-drawn)
 *   S    device [P][U][T] uint8 (output, 0/1)
 * Asynchronous on the stream. */
evo_status evo_guided_schedules(const float* d, int32_t U, int32_t T, int32_t K, float eps, int32_t gamma,
                                const uint64_t* rnd, int32_t P, uint8_t* S, void* stream);

/* Schedule search (Sec. 3.2 genetic algorithm, Sec. 3.3 redundancy-guided
 * initialisation and target-conditioned early stopping, Eq. 8 and 9).  Host
 * code; fitness comes from the caller:
 *   evo_fitness_fn(user, S [P][n_units][T] uint8 host, P, n_units, T, fitness[P])
 * returns 0 on success (e.g. -dev_l2 of evo_denoise_population; higher is better).
 * The search keeps every individual at exactly `budget` unique positions
 * (block_wise: `budget` steps in every unit row, the ablation's Block-wise GA),
 * evaluates each distinct schedule once (signature memo), carries `elites`
 * over, breeds the rest by tournament selection, set-level crossover (common
 * positions kept, each other one with probability 1/2), mutation (each
 * position resampled with probability mutation_rate) and repair; `guided` of
 * the initial individuals follow Eq. 7 (d_map host [n_units][T], as from
 * evo_redundancy_map), the others are uniform.  With early_stop, candidates
 * whose quick fitness reaches q_base are evaluated by `formal`; the first (in
 * fitness order) whose formal fitness is at least q_base - delta_acc is
 * returned and the search stops.  Every random choice draws from one
 * SplitMix64 stream seeded by `seed`: the search is reproducible.
 * best_S: host [n_units][T] uint8 (the accepted schedule, else the best seen). */
typedef int32_t (*evo_fitness_fn)(void* user, const uint8_t* S, int32_t P, int32_t n_units, int32_t T,
                                  double* fitness);
typedef struct evo_search_config {
  int32_t n_units, n_steps;
  int32_t budget;            /* K (block_wise = 0) or refresh steps per unit (block_wise = 1) */
  int32_t block_wise;
  int32_t population, elites, generations, tournament;
  int32_t guided;            /* initial individuals drawn by Eq. 7 (needs d_map) */
  int32_t gamma;             /* Eq. 7 exponent (positive integer) */
  float eps;                 /* Eq. 7 offset */
  float pad_;
  double crossover_rate, mutation_rate;
  int32_t early_stop;
  int32_t pad2_;
  double q_base, delta_acc;  /* Eq. 8 / Eq. 9 */
  uint64_t seed;
} evo_search_config;
typedef struct evo_search_result {
  double best_fitness;
  int32_t generations, evaluations, formal_evaluations, memo_hits, stopped_early, pad_;
} evo_search_result;
evo_status evo_search(const evo_search_config* cfg, const float* d_map, evo_fitness_fn quick, evo_fitness_fn formal,
                      void* user, uint8_t* best_S, evo_search_result* result);

/* The cudaError_t of the most recent CUDA runtime failure behind an
 * EVO_ERR_CUDA on the calling thread (0 if none): the detail a caller needs to
 * tell, for instance, a launch-configuration error from a device fault. */
int32_t evo_last_cuda_error(void);

const char* evo_status_string(evo_status s);

#ifdef __cplusplus
}
#endif

#endif /* EVO_H */
