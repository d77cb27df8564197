/*
 * asymspec.h -- C ABI of the AsymSpec per-step fuse-and-verify path on GB300.
 *
 * The operation (paper: "AsymSpec: Context-Asymmetric Speculative Decoding for
 * Agentic LLMs", Section 3 and Algorithm 1).  Each speculation step produces,
 * for every batch element b and each of its K+1 positions k (row k predicts
 * the token at position k+1; row K is the position after the last draft),
 * three vocabulary-wide logit rows:
 *   logits_full  a = drafter S on the full context        (Section 3.2, item 1)
 *   logits_comp  b = drafter S on the compressed context  (Section 3.2, item 2)
 *   logits_ver   t = verifier L on the compressed context (Section 3.2, item 3)
 * and the drafter's K draft tokens d.  Per row the library computes the
 * log-softmax normalisers of a, b, t and of the fused scores
 * s = t + beta * (a - b) (Eqs. 1-2), the Jensen-Shannon divergence
 * D = JSD(softmax a || softmax b) and the threshold gamma_eff = gamma exp(-D)
 * (Eq. 3), the acceptance test of Eq. 4, and then, per batch element, the
 * sequential accept scan of Algorithm 1:
 *   greedy mode: accept d_k iff softmax(t_k)[d_k] > gamma_eff(k) softmax(b_k)[d_k];
 *     the first rejected position emits argmax(s_k); if all K pass, the bonus
 *     position emits argmax(t_K) (argmax(s_K) with fuse_bonus);
 *   stochastic mode (an extension; the paper decodes greedily): accept d_k iff
 *     q_k(d_k) / draft_probs[k] > u_k gamma_eff(k) with q_k = softmax(s_k); the
 *     first rejected position draws from max(0, q_k - softmax(a_k)) normalised
 *     (from q_k if that residual is identically zero) by inverse CDF at u_K;
 *     if all K pass, the bonus position draws from q_K at u_K.
 * Ties in an argmax resolve to the lowest index; inverse-CDF draws return the
 * smallest index whose cumulative mass (in index order) exceeds the target.
 *
 * Conventions for every entry point below:
 *  - Array arguments are caller-owned DEVICE pointers unless stated; the
 *    library never frees or retains them.  Logit tensors are [B, K+1, V]
 *    row-major in the dtype given (fp32, or bf16 as 16-bit words), with rows
 *    16-byte aligned for the fast path (any element-aligned pointer works; a
 *    slower path handles the rest).
 *  - All work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream) and is asynchronous: results are valid once the stream has
 *    completed.  Calls on different streams are independent and may run
 *    concurrently if their workspaces differ.
 *  - Return values are ASYMSPEC_* status codes; host-detectable errors are
 *    reported before anything is enqueued.  Problems in the DATA (found on the
 *    device) never trap: the affected batch element gets accept_len = -1 and
 *    next_token = -1 and a bit is OR-ed into the optional device error word.
 *  - Inputs must be finite.  A NaN or +inf logit is detected (the element's
 *    normalisers become non-finite); a -inf logit is outside the contract.
 */
#ifndef ASYMSPEC_H
#define ASYMSPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define ASYMSPEC_OK 0
#define ASYMSPEC_ERR_INVALID_ARG (-1)   /* null pointer, B<1, K<1, V<2, gamma or beta out of range */
#define ASYMSPEC_ERR_UNSUPPORTED (-2)   /* unknown dtype, mode or divergence */
#define ASYMSPEC_ERR_MISALIGNED (-3)    /* a pointer not aligned to its element size */
#define ASYMSPEC_ERR_WORKSPACE (-4)     /* workspace missing or smaller than asymspec_workspace_bytes() */
#define ASYMSPEC_ERR_CUDA (-5)          /* a CUDA call failed; see asymspec_last_cuda_error() */
#define ASYMSPEC_ERR_TOO_LARGE (-6)     /* V too large for the row slices of any cluster (see asymspec_plan) */
#define ASYMSPEC_ERR_SCRATCH_LIMIT (-7) /* B*(K+1) above ASYMSPEC_STATIC_MAX_ROWS (asymspec_fuse_verify_static) */

/* ---- device error-word bits (data errors, per batch element) ----------- */
#define ASYMSPEC_DATA_BAD_TOKEN 0x1u    /* a draft token outside [0, V) */
#define ASYMSPEC_DATA_NONFINITE 0x2u    /* a non-finite normaliser or divergence (NaN/inf logits) */
#define ASYMSPEC_DATA_BAD_PROB 0x4u     /* stochastic: draft probability outside (0, 1] */
#define ASYMSPEC_DATA_BAD_UNIFORM 0x8u  /* stochastic: uniform outside [0, 1) */
#define ASYMSPEC_DATA_TIMEOUT 0x10u     /* a bulk copy into shared memory (staged row kernel) or the
                                           exchange of the cluster's pass-1 records (production row
                                           kernel) did not complete within its time limit (the
                                           kernel gave up instead of hanging) */
#define ASYMSPEC_DATA_BAD_MAP 0x20u     /* cross-family step: a map entry outside its vocabulary */

typedef enum { ASYMSPEC_FP32 = 0, ASYMSPEC_BF16 = 1 } asymspec_dtype_t;

typedef enum {
  ASYMSPEC_MODE_GREEDY = 0,      /* Algorithm 1 (tau = 0, the paper's setting) */
  ASYMSPEC_MODE_STOCHASTIC = 1   /* speculative sampling with the CDA-relaxed threshold */
} asymspec_mode_t;

typedef enum {
  ASYMSPEC_DIV_JSD = 0,    /* Eq. 3: D = JSD(softmax a || softmax b), natural log (default) */
  ASYMSPEC_DIV_NONE = 1,   /* fixed-gamma gate: gamma_eff = gamma (Appendix B baseline) */
  ASYMSPEC_DIV_KL = 2,     /* D = KL(softmax a || softmax b) (Table "JSD vs KL") */
  ASYMSPEC_DIV_LAMBDA = 3  /* gamma_eff = gamma exp(-lambda (log p_a(d) - log p_b(d))) (Appendix B) */
} asymspec_div_t;

/* Hyper-parameters of the step (host struct, read during the call). */
typedef struct {
  float gamma;         /* base threshold, in (0, 1]; paper default 0.5 (Algorithm 1, Section 4.2) */
  float beta;          /* fusion weight, finite and >= 0; paper default 1.0 (Eq. 2) */
  float lambda;        /* only for ASYMSPEC_DIV_LAMBDA; paper default 0.1 (Appendix B) */
  int32_t mode;        /* asymspec_mode_t */
  int32_t divergence;  /* asymspec_div_t */
  int32_t fuse_bonus;  /* greedy: 0 = bonus emits argmax(t_K) as in Algorithm 1; 1 = argmax(s_K) */
  int32_t flags;       /* bits 0-1: the delta source (ASYMSPEC_DELTA_*); other bits reserved, 0 */
} asymspec_gate_params;

/* The signal fused into the emission, s = t + beta * delta (Eq. 2), in
 * gate_params.flags & ASYMSPEC_FLAG_DELTA_MASK: the paper's delta = a - b
 * (Eq. 1), or one of the alternatives its mechanism ablation compares,
 * delta = a (raw-augmented) and delta = t - b (SCD-style).  Only the fused
 * scores change: the gate (Eq. 3) and the acceptance test (Eq. 4) keep their
 * own a, b and t. */
#define ASYMSPEC_DELTA_AB 0
#define ASYMSPEC_DELTA_A 1
#define ASYMSPEC_DELTA_TB 2
#define ASYMSPEC_FLAG_DELTA_MASK 3

/* Optional launch overrides (host struct); zero fields mean "automatic". */
typedef struct {
  int32_t cluster_size;   /* CTAs per row triple: 1 to 16 */
  int32_t block_threads;  /* 0 (automatic) or 256: every kernel runs 256-thread CTAs;
                             other values are reserved (ASYMSPEC_ERR_INVALID_ARG) */
  int32_t kernel;         /* 0 automatic; ASYMSPEC_KERNEL_GENERIC or ASYMSPEC_KERNEL_TMA */
  int32_t test_flags;     /* 0, or test hooks (ASYMSPEC_TEST_*); other bits reserved, 0 */
  /* Optional cudaEvent_t handles (or NULL): recorded on the call's stream
   * immediately before and after the launch of the fused row kernel (not
   * around the decision kernel that follows it), so that a caller can time
   * that kernel alone with cudaEventElapsedTime.  Both or neither. */
  void* timing_begin;
  void* timing_end;
} asymspec_launch_opts;

/* Test hook (asymspec_launch_opts.test_flags), for tests of the timeout
 * path only: every bulk-copy wait of the staged row kernel of
 * ASYMSPEC_KERNEL_TMA (fuse_verify_tma) gives up at once, as if its time
 * limit (200 ms) had passed, while the copies still land.
 * Each CTA then takes its timeout branch: it marks its row, still reaches
 * every cluster barrier, and before it exits waits (with the normal limit)
 * for its copies in flight; every batch element comes back as a data error
 * (accept_len = next_token = -1) with ASYMSPEC_DATA_TIMEOUT in the error
 * word.  The generic kernel waits on no copies and ignores it; so does the
 * production row kernel (fuse_verify_row), whose one bounded wait (the
 * record exchange, 200 ms) the hook does not shorten. */
#define ASYMSPEC_TEST_COPY_GIVE_UP 1

/* Kernels (asymspec_launch_opts.kernel, asymspec_launch_info.kernel). */
#define ASYMSPEC_KERNEL_GENERIC 1  /* one cluster per row; any element-aligned input */
#define ASYMSPEC_KERNEL_TMA 2      /* one cluster per row, then a decision kernel; rows
                                      16-byte aligned.  The stochastic JSD step without debug
                                      outputs runs the production row kernel (slices read
                                      from HBM, then again from the L2; C chosen so that the
                                      rows in flight stay within an L2 budget once a batch
                                      fills a wave of clusters of 8); every other program
                                      stages its slices by chunked 1-D bulk copies */

/* What a launch would use (filled by asymspec_plan). */
typedef struct {
  int32_t cluster_size;    /* CTAs that split one row triple, combined over DSMEM */
  int32_t block_threads;   /* threads per CTA */
  int32_t slice_elems;     /* vocabulary entries per CTA (its slice of each row) */
  int32_t smem_bytes;      /* dynamic shared memory per CTA */
  int64_t ctas;            /* CTAs in the grid */
  int32_t vector_path;     /* 1 if rows qualify for 16-byte copies (V * element size % 16 == 0) */
  int32_t max_active_clusters; /* clusters the device can hold at once (0 if unknown) */
  int32_t kernel;          /* ASYMSPEC_KERNEL_GENERIC or ASYMSPEC_KERNEL_TMA */
  int32_t launches;        /* kernel launches of one call: 1 (the generic kernel) or 2
                              (a cluster row kernel and its decision kernel) */
  int32_t row_kernel;      /* 1 if ASYMSPEC_KERNEL_TMA runs its production row kernel
                              (fuse_verify_row: the stochastic JSD step without debug
                              outputs), 0 otherwise */
} asymspec_launch_info;

/* Fills *p with the paper's defaults: gamma 0.5, beta 1.0, lambda 0.1,
 * greedy mode, JSD gate, unfused bonus (Section 4.2, Appendix B). */
void asymspec_default_gate_params(asymspec_gate_params* p);

/* Bytes of device workspace asymspec_fuse_verify_ex needs for a batch of
 * B elements with K drafts and V vocabulary entries (enough for every kernel,
 * cluster size and dtype).  Layout, each part 256-byte aligned: 16 B of row
 * record per row and 4 B of ticket per element (all the generic kernel
 * needs); then, for ASYMSPEC_KERNEL_TMA with clusters of C CTAs, 48 B of
 * pass-1 results per row and 352 B per row and CTA of pass-2 record and
 * inverse-CDF group masses, which its decision kernel reads.  With less than
 * the TMA part the automatic choice falls back to the generic kernel.  The tickets
 * must be zero before the first use (cudaMemset or
 * asymspec_workspace_reset); every call that completes leaves them zero
 * again, and every other part is written before it is read.  Two calls in
 * flight at the same time must not share a workspace. */
size_t asymspec_workspace_bytes(int B, int K, int V);

/* Enqueues a zero fill of a workspace on `stream`. */
int asymspec_workspace_reset(void* workspace, size_t workspace_bytes, void* stream);

/*
 * The step with the paper's problem statement as arguments (Section 3).
 *   logits_full, logits_comp, logits_ver: [B, K+1, V] device, dtype `dtype`
 *   draft_tokens: [B, K] int32 device
 *   draft_probs:  [B, K] fp32 device, the drafter's probability of each draft
 *                 (stochastic mode; may be NULL in greedy mode)
 *   uniforms:     [B, K+1] fp32 device in [0, 1): u[b][k] for the k-th test,
 *                 u[b][K] for the one non-draft draw (stochastic; NULL in greedy)
 *   gate_params:  host pointer, NULL = asymspec_default_gate_params
 *   out_accept_len, out_next_token: [B] int32 device outputs
 * Obtains its workspace with cudaMallocAsync/cudaFreeAsync on `stream`.
 */
int asymspec_fuse_verify(const void* logits_full, const void* logits_comp,
                         const void* logits_ver, const int32_t* draft_tokens,
                         const float* draft_probs, const float* uniforms, int B, int K,
                         int V, int dtype, const asymspec_gate_params* gate_params,
                         int32_t* out_accept_len, int32_t* out_next_token, void* stream);

/*
 * As asymspec_fuse_verify, with a caller-owned workspace and optional outputs:
 *   workspace, workspace_bytes: device scratch of asymspec_workspace_bytes()
 *       bytes, zeroed before first use (see above)
 *   out_row_stats:  [B, K+1, 8] fp32 device or NULL: per row LSE(a), LSE(b),
 *       LSE(t), LSE(s), D, gamma_eff, acceptance margin (greedy
 *       1 - ratio/gamma_eff, stochastic u - ratio/gamma_eff; NaN on row K) and
 *       the inverse-CDF mass used (stochastic) or NaN
 *   out_row_tokens: [B, K+1, 2] int32 device or NULL: per row argmax(s) and
 *       the token emitted if the scan stops at that row
 *   out_fused_logprobs: [B, K+1, V] fp32 device or NULL: log softmax(s), the
 *       fused target (a debug output that adds 4 V bytes of writes per row)
 *   out_error_word: one uint32 device word or NULL; ASYMSPEC_DATA_* bits are
 *       OR-ed into it (the caller clears it)
 *   opts: NULL for automatic launch parameters
 */
int asymspec_fuse_verify_ex(const void* logits_full, const void* logits_comp,
                            const void* logits_ver, const int32_t* draft_tokens,
                            const float* draft_probs, const float* uniforms, int B, int K,
                            int V, int dtype, const asymspec_gate_params* gate_params,
                            int32_t* out_accept_len, int32_t* out_next_token,
                            void* workspace, size_t workspace_bytes, float* out_row_stats,
                            int32_t* out_row_tokens, float* out_fused_logprobs,
                            uint32_t* out_error_word, const asymspec_launch_opts* opts,
                            void* stream);

/*
 * The step of asymspec_fuse_verify without any allocation.  The paper has no
 * counterpart: this is a deployment variant of the same launch.
 *
 * Callers that cannot allocate device memory per step use it: a serving loop
 * that has reserved all free HBM up front for its own allocator (KV cache,
 * activations), where a per-step cudaMallocAsync can fail or make the pool
 * grow and trim, and plain C hosts that have no device allocator to provide
 * the workspace asymspec_fuse_verify_ex wants.
 *
 * Scratch: one file-scope static __device__ array of the library
 * (ASYMSPEC_STATIC_SCRATCH_BYTES, 4 MiB),
 * used as asymspec_fuse_verify_ex uses a workspace.  It holds the generic
 * kernel's records and tickets for B*(K+1) <= 8192 rows (16 bytes per row
 * and 4 per batch element); larger batches return ASYMSPEC_ERR_SCRATCH_LIMIT
 * before anything is enqueued.  Aligned rows run ASYMSPEC_KERNEL_TMA when
 * the array also holds its per-row results (48 + 576 C bytes a row for
 * clusters of C: about 890 rows at C = 8, 1190 at C = 6), else the generic
 * kernel.  Each call enqueues on `stream` a zero fill
 * of the B tickets (the only part that must start at zero), then the
 * launches of asymspec_fuse_verify_ex.  Nothing is allocated: no
 * cudaMalloc, cudaMallocAsync, cudaFree or library call that allocates.
 *
 * Set-up: every call looks up the array's device address in the current
 * device's context with cudaGetSymbolAddress (return code checked,
 * ASYMSPEC_ERR_CUDA on failure), so the address stays right after a
 * cudaDeviceReset.  The first call in a context may load the module: make it
 * before any stream capture begins on that device.
 *
 * Concurrency: there is one scratch array per device.  Calls that overlap in
 * time on one device (several streams, or several host threads) share it and
 * race, with undefined results; order them (one stream, or events).
 *
 * Arguments, outputs and status codes are those of asymspec_fuse_verify.
 */
#define ASYMSPEC_STATIC_MAX_ROWS 8192
#define ASYMSPEC_STATIC_SCRATCH_BYTES (4u << 20)
int asymspec_fuse_verify_static(const void* logits_full, const void* logits_comp,
                                const void* logits_ver, const int32_t* draft_tokens,
                                const float* draft_probs, const float* uniforms, int B, int K,
                                int V, int dtype, const asymspec_gate_params* gate_params,
                                int32_t* out_accept_len, int32_t* out_next_token,
                                void* stream);

/*
 * The step from host memory: asymspec_fuse_verify_ex's computation for
 * callers whose logits are in host memory (no counterpart in the paper: a
 * deployment variant).  The batch is cut into at most ASYMSPEC_HOST_CHUNKS
 * chunks of whole batch elements.  Every chunk's inputs are copied host to
 * device on a copy stream the library keeps per device; the step of chunk c
 * runs on `stream` as soon as chunk c's copies have landed, while later
 * chunks are still being copied, and each chunk's two outputs are copied
 * back on `stream`.
 *   h_logits_full, h_logits_comp, h_logits_ver: [B, K+1, V] host, dtype `dtype`
 *   h_draft_tokens [B, K] int32, h_draft_probs [B, K] fp32 and
 *   h_uniforms [B, K+1] fp32: host (probabilities and uniforms may be NULL in
 *       greedy mode), laid out as for asymspec_fuse_verify
 *   h_out_accept_len, h_out_next_token: [B] int32 host, written once `stream`
 *       reaches the end of the call (synchronise on it before reading them)
 *   d_scratch, scratch_bytes: device memory of at least
 *       asymspec_host_scratch_bytes(B, K, V, dtype) bytes, 256-byte aligned:
 *       device copies of the inputs and outputs, then one workspace per
 *       chunk.  It needs no zeroing (each chunk's tickets are cleared on
 *       `stream` before its step).
 * Host buffers should be page-locked (cudaMallocHost or cudaHostRegister)
 * for the copies to run asynchronously and overlap the kernels; pageable
 * buffers give the same results with the copies staged by the driver.
 * Calls that overlap in time must not share a scratch, and calls from
 * several host threads on one device must be serialised by the caller
 * (they share the copy stream's events).  Status codes are those of
 * asymspec_fuse_verify_ex; ASYMSPEC_ERR_WORKSPACE when the scratch is
 * missing, unaligned or too small.  On a status other than ASYMSPEC_OK
 * returned after copies were enqueued, the call waits for the copy stream
 * before returning.
 */
#define ASYMSPEC_HOST_CHUNKS 8
size_t asymspec_host_scratch_bytes(int B, int K, int V, int dtype);
int asymspec_fuse_verify_host(const void* h_logits_full, const void* h_logits_comp,
                              const void* h_logits_ver, const int32_t* h_draft_tokens,
                              const float* h_draft_probs, const float* h_uniforms, int B, int K,
                              int V, int dtype, const asymspec_gate_params* gate_params,
                              int32_t* h_out_accept_len, int32_t* h_out_next_token,
                              void* d_scratch, size_t scratch_bytes, void* stream);

/* ---- the drafter's draw ---------------------------------------------------
 * The step upstream of fuse-and-verify (Section 3.2, item 1: the augmented
 * drafter S run on the full context; the drafting step of Algorithm 1): for
 * each of `rows` positions, the draft token d drawn from the drafter's
 * full-context logits a, and the drafter's probability of it, softmax(a)[d]
 * (the draft_probs that the stochastic acceptance test of Eq. 4 divides by).
 *   mode ASYMSPEC_MODE_GREEDY:     d = argmax a, the lowest index on ties;
 *                                  uniforms is not read (may be NULL).
 *   mode ASYMSPEC_MODE_STOCHASTIC: d = the smallest index whose cumulative
 *                                  softmax(a) mass, in index order, exceeds
 *                                  uniforms[r] (inverse CDF); if rounding
 *                                  leaves no such index, the last index of
 *                                  positive mass.
 * Arguments (device pointers, caller-owned, not retained):
 *   logits      [rows, V] row-major, fp32 or bf16 (dtype), element-aligned;
 *               16-byte aligned with V * element size a multiple of 16 takes
 *               the vector path (same results)
 *   uniforms    [rows] float32, stochastic mode only
 *   out_tokens  [rows] int32; out_probs [rows] float32
 *   cluster_size  CTAs that share a row (1, 2, 4 or 8; each reads one
 *               contiguous slice of it), or 0 for the library's choice: the
 *               smallest that gives at least 4 CTAs per SM, up to 8, while a
 *               slice keeps at least 512 vectors.  Results do not depend on it
 *               beyond fp32 rounding of the sums.
 * One kernel launch on `stream` (rows x cluster_size CTAs), no workspace,
 * nothing allocated.  rows = 0 is a no-op.  Host-detectable errors, returned
 * before anything is enqueued: ASYMSPEC_ERR_INVALID_ARG (a null pointer,
 * rows < 0, V < 2, a cluster_size other than 0, 1, 2, 4, 8),
 * ASYMSPEC_ERR_UNSUPPORTED (dtype or mode), ASYMSPEC_ERR_MISALIGNED,
 * ASYMSPEC_ERR_TOO_LARGE (V > ASYMSPEC_DRAFT_MAX_V or rows above 2^27).  In the data: a row with
 * a non-finite logit (NaN, +inf or -inf) or, stochastic, a uniform outside
 * [0, 1) gets token -1 and probability NaN; the other rows are unaffected.
 */
#define ASYMSPEC_DRAFT_MAX_V (1 << 20)
int asymspec_draft_sample(const void* logits, int rows, int V, int dtype, int mode,
                          const float* uniforms, int32_t* out_tokens, float* out_probs,
                          int cluster_size, void* stream);

/* ---- cross-family vocabularies -------------------------------------------
 * The step for a drafter and a verifier that tokenise differently (Section 4,
 * "Cross-family portability", and the appendix of the same name: delta is
 * computed in the drafter's vocabulary and carried to the verifier through
 * the S string-identical tokens; committed tokens are restricted to that
 * shared set).  The S pairs are (map_d[j], map_v[j]): drafter token map_d[j]
 * and verifier token map_v[j] spell the same string.  The step runs, exactly
 * as asymspec_fuse_verify_ex defines it, on the rows restricted to the pairs
 * in pair order, a'_j = a[map_d[j]], b'_j = b[map_d[j]], t'_j = t[map_v[j]]:
 * every softmax, the divergence of Eq. 3, the acceptance test of Eq. 4 and
 * the emission are taken over the S pairs.  Draft tokens are given as pair
 * indices in [0, S); the emitted pair index j is committed as the verifier
 * token map_v[j].
 *
 * asymspec_xvocab_gather: the restriction alone.  For each of `rows` rows,
 *   out_full[r][j] = logits_full[r][map_d[j]], out_comp likewise, and
 *   out_ver[r][j] = logits_ver[r][map_v[j]]; outputs [rows, S] row-major in
 *   `dtype`, caller-owned device memory.  logits_full and logits_comp are
 *   [rows, V_d], logits_ver [rows, V_v], all device, element-aligned.
 *   map_d, map_v: [S] int32 device.  out_error_word: device word or NULL.
 *   scratch, scratch_bytes: device memory of at least
 *   asymspec_xvocab_gather_scratch_bytes(V_d, V_v) bytes, 256-byte aligned,
 *   no zeroing needed, or NULL.  With a scratch the maps are checked: the
 *   inverse maps of the pairs are built in it (atomicCAS), and a map entry
 *   outside its vocabulary or a token that appears in two pairs sets
 *   ASYMSPEC_DATA_BAD_MAP in *out_error_word and a map-error word in the
 *   scratch.  Without one, an entry outside its vocabulary is still never
 *   dereferenced (its values read NaN, and ASYMSPEC_DATA_BAD_MAP is set) but
 *   a repeated token is not detected.  a and b are read through map_d (one
 *   thread per pair and row).  With a scratch, logits_ver 16-byte aligned,
 *   V_v * element size a multiple of 16 and S * element size at most
 *   227 KB, t is gathered by a second kernel, one CTA per row, that builds
 *   the restricted row in shared memory through the inverse map of the
 *   check, so that a map_v in any order costs no DRAM sector per entry;
 *   otherwise t too is read through map_v by the first kernel.  One launch
 *   on `stream` (four with a scratch), nothing allocated.  Host-detectable errors:
 *   ASYMSPEC_ERR_INVALID_ARG (a null pointer, rows < 0, S < 2, V_d < 1,
 *   V_v < 1), ASYMSPEC_ERR_UNSUPPORTED (dtype), ASYMSPEC_ERR_MISALIGNED,
 *   ASYMSPEC_ERR_WORKSPACE (scratch unaligned or too small),
 *   ASYMSPEC_ERR_TOO_LARGE (rows above 524,280).
 *
 * asymspec_fuse_verify_xvocab: map check, gather, step and emission, up to
 *   seven launches on `stream` (the gather's four, the step's one or two,
 *   the emission): logits_full, logits_comp
 *   [B, K+1, V_d]; logits_ver [B, K+1, V_v]; draft_index [B, K] int32 pair indices; draft_probs,
 *   uniforms, gate_params as for asymspec_fuse_verify (draft_probs[b][k] is
 *   the drafter's probability of pair draft_index[b][k] under the restricted
 *   softmax); out_accept_len, out_next_token [B] int32 (verifier tokens);
 *   out_next_index [B] int32 or NULL: the emitted pair index (-1 on a data
 *   error); workspace of
 *   asymspec_xvocab_workspace_bytes(B, K, S, V_d, V_v, dtype) bytes,
 *   256-byte aligned and zeroed before its first use
 *   (asymspec_workspace_reset; every call that completes leaves it fit for
 *   the next); out_error_word as for asymspec_fuse_verify_ex.  A map entry
 *   outside its vocabulary or a token in two pairs makes every batch element
 *   a data error (accept_len = next_token = -1, ASYMSPEC_DATA_BAD_MAP).  The
 *   restricted rows are laid out with a stride of S entries, so the fast
 *   step kernel runs when S * element size is a multiple of 16 and the
 *   generic one otherwise.  Status codes are those of
 *   asymspec_fuse_verify_ex and asymspec_xvocab_gather; a pair index outside
 *   [0, S) is the data error ASYMSPEC_DATA_BAD_TOKEN of that element.
 */
size_t asymspec_xvocab_gather_scratch_bytes(int V_d, int V_v);
size_t asymspec_xvocab_workspace_bytes(int B, int K, int S, int V_d, int V_v, int dtype);
int asymspec_xvocab_gather(const void* logits_full, const void* logits_comp, int V_d,
                           const void* logits_ver, int V_v, const int32_t* map_d,
                           const int32_t* map_v, int S, int rows, int dtype, void* out_full,
                           void* out_comp, void* out_ver, uint32_t* out_error_word,
                           void* scratch, size_t scratch_bytes, void* stream);
int asymspec_fuse_verify_xvocab(const void* logits_full, const void* logits_comp, int V_d,
                                const void* logits_ver, int V_v, const int32_t* map_d,
                                const int32_t* map_v, int S, const int32_t* draft_index,
                                const float* draft_probs, const float* uniforms, int B, int K,
                                int dtype, const asymspec_gate_params* gate_params,
                                int32_t* out_accept_len, int32_t* out_next_token,
                                int32_t* out_next_index, void* workspace,
                                size_t workspace_bytes, uint32_t* out_error_word, void* stream);

/* Launch parameters a call with these sizes would use, without launching.
 * Uses the current CUDA device. */
int asymspec_plan(int B, int K, int V, int dtype, const asymspec_gate_params* gate_params,
                  const asymspec_launch_opts* opts, asymspec_launch_info* out);

/* Static description of a status code. */
const char* asymspec_status_string(int status);

/* The cudaError_t of the last ASYMSPEC_ERR_CUDA returned on this thread. */
int asymspec_last_cuda_error(void);

/* Library version: major * 10000 + minor * 100 + patch. */
int asymspec_version(void);

#ifdef __cplusplus
}
#endif

#endif /* ASYMSPEC_H */
