/*
 * bkmoo.h -- C ABI of the Bucket-Level MOO resolve library for GB300 (sm_103a).
 *
 * The method ("Multilingual Fine-Tuning via Localized Gradient Conflict
 * Resolution", arXiv 2606.05613, Section 3.2 and Algorithm 1) splits the
 * parameters into disjoint buckets and, for every bucket, resolves the K
 * per-language gradients restricted to that bucket into one update
 * direction with a multi-objective rule (MGDA, CAGrad or PCGrad).  The global
 * update is the concatenation of the bucket directions (Section 3.2).
 *
 * Every rule needs the gradients only through the bucket's K x K Gram matrix
 * G[i][j] = <g_i, g_j> (Eq. 3, Eq. 4, Eq. 5 are functions of inner products),
 * and every rule's result is a linear combination d_b = sum_k beta_k g_k.  So
 * one resolve is three device passes: Gram, per-bucket solve for beta, and
 * combination.
 *
 * Notation: K = number of languages (the paper's T), B = number of buckets
 * (the paper's K), N = elements per language gradient.
 *
 * Conventions common to every entry point:
 *  - Every buffer is owned by the caller.  No entry point allocates device
 *    memory; scratch lives in a caller-supplied workspace.
 *  - Device work is asynchronous on the caller's `stream` (a cudaStream_t
 *    passed as void*; NULL = the legacy default stream).  Argument errors are
 *    returned synchronously; conditions found on the device are written to
 *    per-bucket status words and to the workspace status word
 *    (bkmoo_workspace_status).
 *  - Gradients are K separate device buffers, each the flat per-language
 *    gradient in the layout the plan describes, N elements, fp32 or bf16,
 *    16-byte aligned.
 *  - Offsets are int64 element offsets: offsets[0] = 0, strictly
 *    increasing, offsets[B] = N.  Bucket b is [offsets[b], offsets[b+1]).
 *  - 1 <= K <= 16.
 */
#ifndef BKMOO_H
#define BKMOO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes and per-bucket status values. */
typedef enum {
  BKMOO_OK = 0,
  BKMOO_ERR_INVALID = 1,          /* bad argument; nothing was launched    */
  BKMOO_ERR_CUDA = 2,             /* a CUDA call failed                    */
  BKMOO_ERR_NONFINITE = 3,        /* per bucket: Gram not finite, beta=1/K */
  BKMOO_ERR_WORKSPACE = 4,        /* workspace not initialised for this
                                     plan, or too small                    */
  BKMOO_ERR_TIMEOUT = 5,          /* a bounded device wait gave up         */
  BKMOO_ERR_BUFFER_TOO_SMALL = 6, /* an output array is too short          */
  BKMOO_ERR_NOT_CONVERGED = 7     /* per bucket: the solver hit its
                                     iteration cap without meeting the
                                     stopping test; beta is the last
                                     iterate                               */
} bkmoo_status;

/* The multi-objective rule applied to every bucket (Algorithm 1). */
typedef enum {
  BKMOO_MGDA = 0,   /* Eq. 3 / Eq. 6: min-norm point of the convex hull     */
  BKMOO_PCGRAD = 1, /* Eq. 5 / Eq. 8: sequential projection of conflicts   */
  BKMOO_CAGRAD = 2, /* Eq. 4 / Eq. 7: conflict-averse direction            */
  BKMOO_MEAN = 3    /* the averaged gradient of plain fine-tuning          */
} bkmoo_rule;

typedef enum { BKMOO_F32 = 0, BKMOO_BF16 = 1 } bkmoo_dtype;

/* bkmoo_params.flags */
#define BKMOO_FLAG_CLOSED_FORM_K2 0x1u /* K = 2 MGDA by its closed form      */
#define BKMOO_FLAG_POLISH 0x2u         /* exact active-set completion after
                                          the Frank-Wolfe phase (MGDA and
                                          CAGrad)                            */
#define BKMOO_FLAG_FUSED 0x4u          /* one launch that resolves bucket
                                          after bucket while the bucket is
                                          still in L2: a thread-block cluster
                                          per bucket for K <= 4, groups of
                                          CTAs for K = 5..8; above, ignored
                                          (three passes).  On a GB300 the
                                          cluster kernel is faster than three
                                          passes for K = 2..4 with buckets of
                                          2-6 MiB (the per-plan choice takes
                                          it there, see bkmoo_resolve_path),
                                          slower for 1 MiB buckets, large
                                          buckets and K = 1 or 8.  The
                                          cluster kernel's look-ahead into
                                          the next bucket can be overridden
                                          with the environment variable
                                          BKMOO_CLUSTER_HEAD (items per
                                          thread).  Results agree
                                          with the three-pass path to
                                          rounding, not bit for bit.  The
                                          groups kernel's L2 budget and
                                          look-ahead can be overridden with
                                          the environment variables
                                          BKMOO_FUSED_L2_BUDGET (bytes) and
                                          BKMOO_FUSED_LOOKAHEAD (buckets).   */
#define BKMOO_FLAG_THREE_PASS 0x8u     /* always the three-launch path (Gram,
                                          solve, combination); without it and
                                          without BKMOO_FLAG_FUSED the path is
                                          chosen per plan, see
                                          bkmoo_resolve_path                 */
#define BKMOO_FLAG_TEST_WITHHOLD 0x100u /* testing failure detection, with
                                          BKMOO_FLAG_FUSED only (it selects
                                          the grid-synchronised fused
                                          kernel): that kernel never
                                          publishes bucket 0's
                                          coefficients, so its bounded waits
                                          (about 1 s) run out and the call
                                          ends with BKMOO_ERR_TIMEOUT in the
                                          workspace status word; the output
                                          is then undefined                 */
#define BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE 0x200u /* testing failure detection,
                                          with BKMOO_FLAG_FUSED and K <= 4
                                          only (the cluster kernel): CTA 0
                                          of every cluster never hands its
                                          partial Gram of the cluster's
                                          first bucket to its peers, so the
                                          peers' bounded exchange waits
                                          (about 1 s) run out, every later
                                          wait gives up at once, and the
                                          call ends with BKMOO_ERR_TIMEOUT
                                          in the workspace status word; the
                                          output is then undefined          */

typedef struct {
  int32_t max_iter; /* Frank-Wolfe iterations per bucket (MGDA, CAGrad)     */
  double tol;       /* relative duality-gap stop of the Frank-Wolfe phase   */
  double cagrad_c;  /* CAGrad c in [0, 1) (Eq. 4); the paper uses 0.5       */
  uint64_t seed;    /* PCGrad "random order" (Algorithm 1) is a function of */
  uint64_t step;    /*   (seed, step, bucket, task), see bkmoo_resolve      */
  uint32_t flags;   /* BKMOO_FLAG_*                                         */
  void* events;     /* tracing: NULL, or an array of 4 cudaEvent_t that
                       bkmoo_resolve records on `stream` before the Gram pass,
                       after it, after the solve and after the combination
                       (one persistent launch: the middle two are recorded
                       together after it).  Owned by the caller.           */
} bkmoo_params;

/* Fill *p with the defaults: max_iter 256, tol 1e-12, cagrad_c 0.5, seed 0,
 * step 0, flags CLOSED_FORM_K2 | POLISH, events NULL. */
void bkmoo_default_params(bkmoo_params* p);

/*
 * bkmoo_plan -- bucket partition (Section 3.2, Figure 4 caption: fixed-size
 * buckets filled during the backward pass starting from the last
 * parameters).  Host only, pure.
 *
 * param_sizes[n_params]: element counts of the model's tensors in
 * registration order.  The flat gradient the other calls read lists them in
 * REVERSE registration order, each tensor in its own flat order.  A bucket
 * holds at most cap = floor(bucket_bytes / elem_bytes) elements: a tensor
 * that does not fit in the open bucket closes it; a tensor larger than cap is
 * cut into cap-sized pieces; the rest joins the open bucket.  Empty tensors
 * are skipped.
 *
 * Two-call use: with out_offsets == NULL only *n_buckets is set.  Otherwise
 * out_offsets[0 .. *n_buckets] is written; out_cap is its length (>= B + 1,
 * else BKMOO_ERR_BUFFER_TOO_SMALL).  BKMOO_ERR_INVALID on a NULL pointer,
 * negative size, elem_bytes <= 0 or cap < 1.
 */
int bkmoo_plan(const int64_t* param_sizes, int32_t n_params, int32_t elem_bytes,
               int64_t bucket_bytes, int64_t* out_offsets, int64_t out_cap,
               int64_t* n_buckets);

/*
 * bkmoo_workspace_size -- bytes of device workspace that bkmoo_gram and
 * bkmoo_resolve need for K languages of `in_dtype` over the buckets given by
 * offsets[0 .. n_buckets] (host array).  Writes *bytes.  The workspace holds
 * the device copy of the bucket table, per-block Gram partials (fp64), the
 * per-bucket coefficients and a status word.
 */
int bkmoo_workspace_size(int32_t K, int32_t in_dtype, const int64_t* offsets,
                         int64_t n_buckets, size_t* bytes);

/*
 * bkmoo_workspace_init -- write the bucket table for (K, in_dtype, offsets)
 * into the workspace `ws` (device, ws_bytes >= bkmoo_workspace_size, 256-byte
 * aligned).  Call once per plan and workspace, before the first bkmoo_gram or
 * bkmoo_resolve with them.  Copies from host memory and synchronises
 * `stream`.  Later calls must pass the same offsets: a different plan is
 * detected on the device and reported as BKMOO_ERR_WORKSPACE.
 */
int bkmoo_workspace_init(int32_t K, int32_t in_dtype, const int64_t* offsets,
                         int64_t n_buckets, void* ws, size_t ws_bytes,
                         void* stream);

/*
 * bkmoo_gram -- per-bucket Gram matrices, the inner products every rule is
 * built on (Eq. 2, the QP of Eq. 3 / Eq. 6 and the tests of Eq. 8 depend on
 * the gradients only through them).
 *
 * grads: host array of K device pointers.  out_gram: device, fp64,
 * [n_buckets][K][K], row-major, both triangles written.  Results are
 * deterministic: each element is summed in fp32 within a thread over at most
 * 128 elements, then reduced in a fixed order (warp tree in fp32, CTA and
 * cross-CTA in fp64); no atomics.
 */
int bkmoo_gram(const void* const* grads, int32_t K, int32_t in_dtype,
               const int64_t* offsets, int64_t n_buckets, double* out_gram,
               void* ws, size_t ws_bytes, void* stream);

/*
 * bkmoo_conflicts -- the gradient-conflict statistics of Figure 1, per
 * bucket, from Gram matrices (bkmoo_gram's out_gram): the pairwise cosines
 * cos_ij = G_ij / sqrt(G_ii G_jj) -- a pair conflicts when its cosine is
 * negative (Eq. 2, Definition A.4) -- their mean, population standard
 * deviation and minimum over the K(K-1)/2 pairs, and a flag for "at least
 * one pair conflicts" (the event whose per-layer frequency over training
 * steps Figure 1 plots).  A pair with a zero-norm gradient has cosine 0.
 *
 * gram: device fp64 [n_buckets][K][K].  Outputs (device, each may be NULL):
 * out_cos fp32 [n_buckets][K][K] (diagonal 1, or 0 for a zero gradient),
 * out_stats fp32 [n_buckets][3] = (mean, std, min), out_conflict int32
 * [n_buckets] in {0, 1}.  2 <= K <= 16, else BKMOO_ERR_INVALID.
 */
int bkmoo_conflicts(const double* gram, int32_t K, int64_t n_buckets, float* out_cos,
                    float* out_stats, int32_t* out_conflict, void* stream);

/*
 * bkmoo_gram_noalloc -- bkmoo_gram without a workspace argument; it allocates
 * no memory at all.  The paper has no counterpart: this is a service for
 * callers that hold their input and output buffers but cannot get more
 * device memory, for instance a hook inside a training framework whose
 * device memory all belongs to the framework's caching allocator, or a C
 * caller in a process where another component owns device allocation.
 *
 * Same arguments, results and determinism as bkmoo_gram (the same kernels
 * run).  The scratch (bucket table and per-chunk partial sums) lives in a
 * static device array of BKMOO_NOALLOC_SCRATCH_BYTES that every GPU which
 * loads this library keeps until the process exits; the bucket table reaches
 * it through kernel parameters, so no copy or allocating call is made.
 * Limits: at most BKMOO_NOALLOC_MAX_BUCKETS buckets and a problem whose
 * workspace (bkmoo_workspace_size) fits the array -- about 13 billion
 * elements per language for K = 4 and 1 billion for K = 16 with bf16
 * gradients (half as many with fp32); larger problems return
 * BKMOO_ERR_WORKSPACE.
 *
 * Each call made outside stream capture looks up the array's device address
 * in the current context (cudaGetSymbolAddress, with the device current);
 * a call made while its stream is being captured reuses the last address
 * seen on that device, so make the first call on each device before any
 * stream capture.  Every call shares the one array and rewrites
 * the parts it reads, so results never depend on an earlier call; but calls
 * whose work overlaps on the GPU (other streams or host threads on the same
 * device) race on it and must be serialised by the caller.
 */
#define BKMOO_NOALLOC_SCRATCH_BYTES (32u << 20)
#define BKMOO_NOALLOC_MAX_BUCKETS 4096
int bkmoo_gram_noalloc(const void* const* grads, int32_t K, int32_t in_dtype,
                       const int64_t* offsets, int64_t n_buckets, double* out_gram,
                       void* stream);

/*
 * bkmoo_resolve -- the resolve of Algorithm 1 for every bucket: Gram ->
 * rule -> d_b = sum_k beta_k g_k, written into the flat direction out_dir
 * (the concatenation of Section 3.2).
 *
 * grads / K / in_dtype / offsets / n_buckets as in bkmoo_gram.
 * rule: bkmoo_rule.  p: parameters (NULL = defaults).
 *  - MGDA: Frank-Wolfe on the simplex QP from the best pair (exact line
 *    search, at most p->max_iter steps, stop at duality gap <= p->tol
 *    relative to max_k G_kk), then, with BKMOO_FLAG_POLISH, an exact
 *    active-set (Wolfe minimum-norm-point) completion.  K = 2 with
 *    BKMOO_FLAG_CLOSED_FORM_K2 uses
 *    gamma = clamp(<g2 - g1, g2> / ||g1 - g2||^2, 0, 1).  beta = alpha.
 *  - CAGrad: the dual min_{w in simplex} <g0, g_w> + c ||g0|| ||g_w||
 *    (g0 the mean) by Frank-Wolfe with exact line search, then the same
 *    active-set completion; beta = 1/K + c ||g0|| w / ||g_w||.  No rescaling.
 *  - PCGrad: for each task t, other tasks j in t's order, project the
 *    running d_t off the ORIGINAL g_j when <d_t, g_j> < 0; d = sum_t d_t.
 *    The order of task t in bucket b is a Fisher-Yates shuffle of the
 *    ascending list [0..K-1] without t, slot i = m-1 .. 1 (m = K-1) swapped
 *    with slot r mod (i+1), r the draws mix64(k3 + (n+1) * 0x9E3779B97F4A7C15)
 *    for n = 0, 1, ..., where k1 = mix64(seed + (step+1) * G),
 *    k2 = mix64(k1 + (b+1) * G), k3 = mix64(k2 + (t+1) * G),
 *    G = 0x9E3779B97F4A7C15 and mix64 is the SplitMix64 output function.
 *  - MEAN: beta = 1/K.
 * out_dir: device, N elements of out_dtype (fp32 or bf16, round to nearest
 *   even).  It may be exactly one of the grads buffers when the dtypes match
 *   (in-place); any other overlap with a gradient is BKMOO_ERR_INVALID.
 * out_weights: device fp32 [n_buckets][K] = beta, or NULL.
 * out_status: device int32 [n_buckets] = BKMOO_OK, BKMOO_ERR_NONFINITE (the
 *   Gram had a NaN/Inf; beta = 1/K), BKMOO_ERR_NOT_CONVERGED or
 *   BKMOO_ERR_WORKSPACE; or NULL.
 * ws / ws_bytes: the workspace after bkmoo_workspace_init with the same
 *   K, in_dtype and offsets.
 * Path: three launches (Gram, solve, combination) or one fused launch, as
 *   bkmoo_resolve_path gives for the plan, rule and p->flags.  Each path is
 *   deterministic; the two agree to rounding.
 * Returns BKMOO_OK once the work is queued on `stream`.
 */
int bkmoo_resolve(const void* const* grads, int32_t K, int32_t in_dtype,
                  const int64_t* offsets, int64_t n_buckets, int32_t rule,
                  const bkmoo_params* p, void* out_dir, int32_t out_dtype,
                  float* out_weights, int32_t* out_status, void* ws,
                  size_t ws_bytes, void* stream);

/*
 * bkmoo_resolve_buckets -- bkmoo_resolve for the buckets b_lo .. b_hi-1 of
 * the plan only.  Algorithm 1 resolves bucket k as soon as the backward pass
 * has filled it (its interception "when bucket k is full", Figure 4), while
 * the rest of the backward pass still runs: this entry point lets a caller
 * resolve each bucket as it completes, on any stream.
 *
 * Arguments as in bkmoo_resolve (the whole plan's offsets and workspace),
 * plus 0 <= b_lo <= b_hi <= n_buckets (else BKMOO_ERR_INVALID; b_lo == b_hi
 * queues nothing).  Only those buckets' Gram, rule and combination run: the
 * elements of out_dir, the rows of out_weights / out_status and the
 * workspace partials of other buckets are not touched, so calls for disjoint
 * bucket ranges may run concurrently on different streams.  Results are
 * bit-identical to those of bkmoo_resolve's three-launch path for the same
 * buckets.  The workspace
 * status word is not cleared (other calls may be in flight); device-side
 * errors are recorded into it.  BKMOO_FLAG_FUSED and p->events are ignored.
 */
int bkmoo_resolve_buckets(const void* const* grads, int32_t K, int32_t in_dtype,
                          const int64_t* offsets, int64_t n_buckets, int64_t b_lo, int64_t b_hi,
                          int32_t rule, const bkmoo_params* p, void* out_dir, int32_t out_dtype,
                          float* out_weights, int32_t* out_status, void* ws, size_t ws_bytes,
                          void* stream);

/*
 * bkmoo_host_staging_size -- device staging bytes bkmoo_resolve_host needs
 * so that every window holds at least max(window_elems, the largest bucket)
 * elements per language.  Host only, pure.  Writes *bytes.
 */
int bkmoo_host_staging_size(int32_t K, int32_t in_dtype, int32_t out_dtype,
                            const int64_t* offsets, int64_t n_buckets, int64_t window_elems,
                            size_t* bytes);

/*
 * bkmoo_resolve_host -- bkmoo_resolve for gradients held in HOST memory, the
 * direction written back to host memory.  It follows the per-bucket loop of
 * Algorithm 1 -- bring a bucket's K gradients to the device, resolve it,
 * send its direction on and free the bucket's device copy -- so that device
 * memory holds only a bounded window of buckets, not the K full gradients.
 *
 * Buckets go through three device staging slots in windows of whole buckets:
 * while window w is resolved (Gram -> rule -> combination on `stream`, the
 * same kernels and the same per-chunk arithmetic as bkmoo_resolve's
 * three-launch path, so beta and the direction are bit-identical to it),
 * the next windows are copied
 * in and earlier windows' directions copied out on two internal copy
 * streams, created and destroyed by the call.  Work already queued on `stream` comes first;
 * `stream` completes only after the last byte reaches host_out.
 *
 * host_grads: host array of K host pointers (16-byte aligned), N elements
 *   each.  Page-locked memory (cudaHostAlloc / cudaHostRegister) lets the
 *   copies overlap; pageable memory gives the same results more slowly.
 * host_out: host, N elements of out_dtype; may be exactly one of host_grads
 *   (same dtype); any other overlap is BKMOO_ERR_INVALID.
 * out_weights, out_status, ws, ws_bytes, rule, p: as in bkmoo_resolve (device
 *   buffers; ws initialised for this plan).  p->events and
 *   BKMOO_FLAG_FUSED are ignored.
 * staging: device, 256-byte aligned, staging_bytes long.  It holds three
 *   slots of K input regions and one output region of
 *   round_up(cap e + 16, 256) bytes each (e the region's element size); cap,
 *   the window length in elements per language, is the largest that fits.
 *   A bucket longer than cap is BKMOO_ERR_WORKSPACE (bkmoo_host_staging_size
 *   gives the size for a chosen cap).  Larger staging means fewer, longer
 *   windows.  Calls that share a staging buffer or a workspace must not
 *   overlap on the GPU.
 * Returns BKMOO_OK once everything is queued.
 */
int bkmoo_resolve_host(const void* const* host_grads, int32_t K, int32_t in_dtype,
                       const int64_t* offsets, int64_t n_buckets, int32_t rule,
                       const bkmoo_params* p, void* host_out, int32_t out_dtype,
                       float* out_weights, int32_t* out_status, void* ws, size_t ws_bytes,
                       void* staging, size_t staging_bytes, void* stream);

/*
 * bkmoo_workspace_status -- synchronise `stream` and read the workspace
 * status word: BKMOO_OK, or the first device-side error recorded since the
 * last bkmoo_gram / bkmoo_resolve started (BKMOO_ERR_WORKSPACE,
 * BKMOO_ERR_TIMEOUT).  Writes *status.
 */
int bkmoo_workspace_status(const void* ws, void* stream, int32_t* status);

/*
 * bkmoo_resolve_path -- which path bkmoo_resolve takes for this plan, rule
 * and flags: *path = 0 for the three launches (Gram, solve, combination), 1
 * for the cluster-per-bucket fused kernel (one bucket per thread-block
 * cluster, its re-read served from L2), 2 for the grid-synchronised fused
 * kernel.  BKMOO_FLAG_THREE_PASS gives 0; BKMOO_FLAG_FUSED gives 1 for
 * K <= 4 (2 with BKMOO_FLAG_TEST_WITHHOLD), 2 for K = 5..8, 0 above.
 * Without either flag the choice follows measurements on GB300 (sweeps of
 * 1e9 elements per language, fp32 and bf16, and small plans): 1 when K <= 2
 * and the plan has at most 8 buckets and 4 Mi elements per language (one
 * launch instead of three), or when 2 <= K <= 4, the largest bucket holds at
 * least 2 MiB per language and its K gradients together at most 12 MiB
 * (and at least 6 MiB for bf16; for CAGrad, whose per-bucket solve is
 * longer, fp32 only and at least 8 MiB), and at least 90 % of the
 * elements lie in buckets of at least half the largest; 0 otherwise.  Host only; BKMOO_ERR_INVALID on bad arguments.
 * bkmoo_resolve_buckets and bkmoo_resolve_host always take path 0.
 */
int bkmoo_resolve_path(int32_t K, int32_t in_dtype, int32_t rule, const int64_t* offsets,
                       int64_t n_buckets, uint32_t flags, int32_t* path);

/* Static English text for a bkmoo_status value. */
const char* bkmoo_status_string(int32_t status);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t bkmoo_version(void);

/*
 * bkmoo_selftest_fp64 -- runs, element by element on the device, the fp64
 * division and square root that the fast per-bucket solvers use for the
 * CAGrad and PCGrad coefficients (Eq. 4 / Eq. 7, Eq. 5 / Eq. 8): an fp32
 * seed refined by one Newton-Raphson step with a residual correction
 * (q = a r, q + (a - b q) r with r = 1/b rounded to fp32; s + (x - s^2) / (2 s)
 * with s = sqrt(x) rounded to fp32), relative error at most about 2^-46;
 * arguments outside [1e-30, 1e30] take the correctly rounded operation.
 * A test entry point, so that its accuracy can be checked against the
 * correctly rounded fp64 operations.
 * op 0: out[i] = a[i] / b[i]; op 1: out[i] = sqrt(a[i]) (0 for a[i] <= 0;
 * b unused, may be NULL).  a, b, out: device fp64 [n].  Asynchronous on
 * `stream`.  Returns BKMOO_ERR_INVALID for another op, n < 0 or a NULL
 * array, BKMOO_ERR_CUDA if the launch fails.
 */
int bkmoo_selftest_fp64(int32_t op, const double* a, const double* b, double* out, int64_t n,
                        void* stream);

#ifdef __cplusplus
}
#endif

#endif /* BKMOO_H */
