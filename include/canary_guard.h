/*
 * canary_guard.h -- C ABI of the GB300 (sm_103a) canary-trap hot path.
 *
 * The library implements the verifier-side hot path of arxiv 2607.19490,
 * "Integrity of peer-to-peer distributed LLM inference under malicious
 * nodes":
 *   - a synthetic k-stage pipeline: fp32 hop references and fp16 live
 *     activations, benign (Eq. 2) or tampered (Eq. 3, Sec. 3.2);
 *   - the drift scores of every (stage, canary) pair: the relative-L2
 *     mismatch (Eq. 4), the max-abs deviation and the cosine mismatch of the
 *     cosine-metric ablation (Sec. 4.4);
 *   - the per-canary AUROC (Eq. 5) as exact Mann-Whitney counts, its mean
 *     over canaries (Eq. 6) and the scrambled-label control (Sec. 4.5).
 *
 * Conventions shared by every entry point:
 *   - Every buffer argument named d_* is caller-owned device memory; h_*
 *     is host memory.  The library allocates no device memory, creates no
 *     stream and never synchronises, except cg_read_status.
 *   - Calls are asynchronous and ordered on `stream` (a cudaStream_t; NULL
 *     is the legacy default stream).
 *   - All arguments are validated on the host before any launch; a rejected
 *     call launches nothing and returns the error.  CG_ERR_CUDA reports a
 *     launch error (the CUDA error is left for the caller to inspect).
 *   - Conditions only the device can see (a NaN score, a control canary
 *     without a benign stage, a bounded wait that gave up) are OR-ed as
 *     CG_DEVFLAG_* bits into an optional caller-owned int32 device word
 *     d_status (may be NULL).  cg_read_status synchronises the stream and
 *     maps the word to a cg_status.
 *   - Results are deterministic run to run on one GPU: fixed reduction
 *     order, no floating-point atomics.
 *   - The library keeps per-device set-up (kernel attributes, occupancy)
 *     for the life of the process; after cudaDeviceReset, calls on that
 *     device may fail with CG_ERR_CUDA.
 *   - fp16 tensors are passed as uint16_t binary16 bit patterns.
 *   - Layouts: live activations and references are [S][N][T][d] row-major
 *     (one (stage, canary) segment = T*d contiguous elements); drift
 *     scores are [stat][N][S] with stat 0 = rel_l2, 1 = max_abs,
 *     2 = cos_dev; labels and AUROC inputs are [C][N][S] per configuration.
 */
#ifndef CANARY_GUARD_H
#define CANARY_GUARD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *cg_stream_t;

typedef enum {
  CG_OK = 0,
  CG_ERR_INVALID_ARG = 1,   /* a NULL, zero or out-of-range argument */
  CG_ERR_ALIGNMENT = 2,     /* a device pointer below its required alignment */
  CG_ERR_WORKSPACE = 3,     /* workspace missing or smaller than the size query */
  CG_ERR_NAN_SCORE = 4,     /* a labelled score is NaN (device flag) */
  CG_ERR_CUDA = 5,          /* a CUDA launch or runtime call failed */
  CG_ERR_TIMEOUT = 6,       /* a bounded device wait gave up (device flag) */
  CG_ERR_UNSUPPORTED = 7,   /* a size beyond what this build handles */
  CG_ERR_NO_BENIGN = 8      /* a control canary had no benign stage (device flag) */
} cg_status;

/* Bits of the device status word. */
#define CG_DEVFLAG_NAN_SCORE 1
#define CG_DEVFLAG_TIMEOUT 2
#define CG_DEVFLAG_NO_BENIGN 4

/* Benign noise of a stage outside the malicious set (Eq. 2). */
typedef enum {
  CG_NOISE_MULT = 0,   /* h = fp16(a (1 + sigma_s z)): relative per-element noise */
  CG_NOISE_PAPER = 1   /* h = fp16(a + sigma_s mu z), mu = ||a||_1 / (T d) (Eq. 2) */
} cg_noise_model;

/* Tamper applied by a malicious stage (Eq. 3 and the strategies of Sec. 3.2). */
typedef enum {
  CG_TAMPER_ADDITIVE = 0,          /* a + eps ||a||_F g / ||g||_F, eps = tamper_param */
  CG_TAMPER_SIGNFLIP_CHANNELS = 1, /* negate max(1, round(p d)) channels, p = tamper_param */
  CG_TAMPER_SIGNFLIP_FULL = 2,     /* -a */
  CG_TAMPER_SCALE = 3              /* beta a, beta = tamper_param */
} cg_tamper_kind;

/*
 * One synthetic pipeline configuration: k = n_shards stages of hidden size
 * d, n canaries of T tokens (Sec. 3.1, Sec. 3.3), the malicious set M
 * (Sec. 3.2), sigma_hw (Eq. 2) and the tamper parameter.  Random draws use
 * Philox4x32-10 (Salmon et al., SC'11) keyed by `seed` with config_id in the
 * counter, so every value is a pure function of the description.
 */
typedef struct {
  uint32_t n_shards;             /* k >= 1 stages (shards), at most 1024 */
  uint32_t hidden;               /* d >= 1 */
  uint32_t n_canaries;           /* n >= 1 */
  uint32_t tokens;               /* T >= 1; T * d < 2^34 */
  const int32_t *malicious;      /* host array of n_malicious distinct 0-based stage ids */
  uint32_t n_malicious;          /* c = |M|, 0 <= c < k */
  int32_t noise;                 /* cg_noise_model */
  float benign_sigma;            /* sigma_hw >= 0 */
  float shard_sigma_lognormal;   /* lambda >= 0: sigma_s = sigma exp(lambda z_s); 0 = same sigma */
  uint32_t n_outlier;            /* outlier channels per configuration, <= min(d, 256) */
  float outlier_scale;           /* reference multiplier on outlier channels */
  int32_t tamper;                /* cg_tamper_kind */
  float tamper_param;            /* eps | channel fraction in (0, 1] | scale factor */
  uint64_t seed;                 /* Philox key */
  uint32_t config_id;            /* < 2^30; separates the draws of configurations */
} cg_pipeline_desc;

/* Human-readable name of a status code (static storage). */
const char *cg_status_string(cg_status status);

/* ABI version of this header (incremented on incompatible changes). */
int cg_abi_version(void);

/*
 * Philox4x32-10 blocks first_block .. first_block + n_blocks - 1 with
 * counter (block, c1, c2, c3) and key (seed lo, seed hi) (SC'11), written
 * block-major to d_out (4 * n_blocks words, 16-byte aligned).  This is the
 * stream every generator draw is taken from (seed semantics, Sec. 4.4).
 */
cg_status cg_philox_words(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                          uint32_t first_block, uint32_t n_blocks,
                          uint32_t *d_out, cg_stream_t stream);

/*
 * The Box-Muller normals of the same blocks (the Gaussians of Eq. 2 and of
 * the Gaussian tamper, Sec. 3.2): per block, (x0, x1) -> normals 0, 1 and
 * (x2, x3) -> normals 2, 3 with u1 = ((x >> 8) + 1) 2^-24,
 * u2 = (x >> 8) 2^-24, z = sqrt(-2 ln u1) (cos, sin)(2 pi u2), in fp32.
 * d_out: 4 * n_blocks floats, 16-byte aligned.
 */
cg_status cg_philox_normals(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                            uint32_t first_block, uint32_t n_blocks,
                            float *d_out, cg_stream_t stream);

/*
 * The Box-Muller transform alone, on caller-given word pairs: pair i =
 * (d_words[2i], d_words[2i+1]) -> d_out[2i], d_out[2i+1] = sqrt(-2 ln u1)
 * (cos, sin)(2 pi u2) with u1 = ((x0 >> 8) + 1) 2^-24 and u2 = (x1 >> 8)
 * 2^-24, in fp32, by the same device code every generator normal goes
 * through.  It lets a test sweep each factor over all 2^24 values of its
 * word.  d_words: 2 * n_pairs words, d_out: 2 * n_pairs floats, both device
 * memory, 8-byte aligned.  n_pairs = 0 or a null pointer -> INVALID_ARG.
 */
cg_status cg_box_muller_pairs(const uint32_t *d_words, uint64_t n_pairs, float *d_out,
                              cg_stream_t stream);

/* Workspace bytes cg_generate_pipeline needs for `desc`. */
cg_status cg_generate_workspace_size(const cg_pipeline_desc *desc, size_t *bytes);

/*
 * Materialise one pipeline configuration (Eq. 1-3 stand-in, Sec. 3.3):
 *   d_refs   fp32 [S][N][T][d]  reference a (stored fp32 references)
 *   d_acts   fp16 [S][N][T][d]  live h: benign stages per `noise` (Eq. 2),
 *                               malicious stages per `tamper` (Eq. 3)
 *   d_labels int8 [N][S] or NULL: 1 on malicious stages, else 0
 *   d_ws     workspace of ws_bytes >= cg_generate_workspace_size, 16-byte
 *            aligned; its contents are scratch.
 * d_acts and d_refs must be 16-byte aligned.  A distinct-channel draw that
 * exhausts its draw cap (not expected for valid descriptions) raises
 * CG_DEVFLAG_TIMEOUT in d_status.
 */
cg_status cg_generate_pipeline(const cg_pipeline_desc *desc, uint16_t *d_acts,
                               float *d_refs, int8_t *d_labels, void *d_ws,
                               size_t ws_bytes, int32_t *d_status,
                               cg_stream_t stream);

/*
 * An independent benign recompute of every stage, for the
 * redundant-recompute ceiling (Sec. 4.5) and the noisy-reference ablation
 * (Sec. 4.4): d_out (fp32 [S][N][T][d], 16-byte aligned) receives the fp16
 * output of the benign computation of each stage -- malicious stages
 * included, since the recompute is honest -- with its noise drawn from
 * replica `replica` (Philox counter word 3).  Replica 0 reproduces the live
 * benign draw of cg_generate_pipeline; passing d_out as the references of
 * cg_drift_scores scores the live pipeline against the recompute.  The
 * workspace is cg_generate_workspace_size(desc).
 */
cg_status cg_generate_recompute(const cg_pipeline_desc *desc, uint32_t replica,
                                float *d_out, void *d_ws, size_t ws_bytes,
                                int32_t *d_status, cg_stream_t stream);

/*
 * A pipeline whose stages inherit the upstream deviation (Eq. 2's recursion
 * h_i = f_i(h_{i-1}) + delta_i), with each block's response to its input
 * linearised as f_i(h_{i-1}) = a_i + gain (h_{i-1} - a_{i-1}); the first
 * stage sees the exact embedding.  Benign stages add Eq. 2 noise to
 * v_i = f_i(h_{i-1}) (mu_i = ||v_i||_1 / (T d)); malicious stages output
 * fp16(tau(v_i)) (Eq. 3).  gain = 0 gives cg_generate_pipeline's output.
 * Arguments, layouts and workspace as cg_generate_pipeline; the stages are
 * produced in order (3 launches per stage).
 */
cg_status cg_generate_propagating(const cg_pipeline_desc *desc, float gain,
                                  uint16_t *d_acts, float *d_refs, int8_t *d_labels,
                                  void *d_ws, size_t ws_bytes, int32_t *d_status,
                                  cg_stream_t stream);

/*
 * Random-baseline scores (Sec. 4.5): d_scores[c][n][s] ~ Uniform(0, 1),
 * the top 24 bits of word s of Philox aux stream 5 (canary n, config id
 * config_id0 + c) times 2^-24.  fp32 [C][N][S], 4-byte aligned.
 */
cg_status cg_random_scores(uint64_t seed, uint32_t config_id0, uint32_t n_configs,
                           uint32_t n_canaries, uint32_t n_shards, float *d_scores,
                           cg_stream_t stream);

/* Workspace bytes cg_drift_scores needs for S * N segments of seg_len. */
cg_status cg_drift_workspace_size(uint32_t n_shards, uint32_t n_canaries,
                                  uint64_t seg_len, size_t *bytes);

/*
 * Drift scores of every (stage s, canary n) segment (Eq. 4 and Sec. 4.4):
 *   rel_l2  = ||h - a||_F / ||a||_F (0 if both are zero, +inf if only a is)
 *   max_abs = max |h - a|           (computed in fp32, exact)
 *   cos_dev = 1 - h.a / (||h|| ||a||) (0 when either norm is zero)
 * d_acts fp16 and d_refs fp32 are [S][N][seg_len], 16-byte aligned; any
 * seg_len >= 1 (ragged tails handled).  Scores are written to
 * d_scores[stat * stat_stride + n * S + s] (stat_stride >= N * S; pass
 * N * S for a dense [3][N][S] block).  Each element of d_acts and d_refs is
 * read once from HBM.  Sums are accumulated in fp32 per work item of at
 * most 16384 elements and combined in fp64, so the scores hold their
 * tolerance (rel_l2 within 1e-5 relative) for finite element magnitudes
 * between about 1e-18 and 1e17: above, the squared sums overflow; below
 * about 1e-19 the squares fall into fp32's subnormal range and lose
 * precision, and below about 4e-23 they underflow to zero.  A segment
 * whose every squared difference underflows while some difference is
 * nonzero (all |h - a| < 2^-74.5) gets rel_l2 and cos_dev NaN, never a
 * wrong finite value.  A NaN element makes rel_l2 and cos_dev NaN
 * (max_abs skips it); an infinite live element (fp16 +-inf, which an
 * untrusted hop may send) makes rel_l2 and max_abs +inf and cos_dev NaN.
 * d_ws: >= cg_drift_workspace_size bytes, 16-byte aligned, scratch.
 */
cg_status cg_drift_scores(const uint16_t *d_acts, const float *d_refs,
                          uint32_t n_shards, uint32_t n_canaries,
                          uint64_t seg_len, float *d_scores,
                          uint64_t stat_stride, void *d_ws, size_t ws_bytes,
                          int32_t *d_status, cg_stream_t stream);

/* Kernel choice for cg_drift_scores_ex. */
typedef enum {
  CG_DRIFT_AUTO = 0,       /* CG_DRIFT_BULK when both inputs are device memory and
                              seg_len % 8 == 0, else CG_DRIFT_STREAM (cg_drift_scores) */
  CG_DRIFT_STREAM = 1,     /* register-streaming kernel, any seg_len */
  CG_DRIFT_BULK = 2,       /* TMA bulk-copy pipeline, 6 shared-memory stages, 1 block per SM;
                              needs device memory and seg_len % 8 == 0
                              (else CG_ERR_UNSUPPORTED) */
  CG_DRIFT_BULK_2CTA = 3   /* TMA bulk-copy pipeline, 4 stages, 2 blocks per SM; same need */
} cg_drift_algo;

/*
 * cg_drift_scores with an explicit kernel choice (same results up to the
 * order of fp32 additions).  The bulk-copy kernels report a wait that gave
 * up as CG_DEVFLAG_TIMEOUT in d_status.
 */
cg_status cg_drift_scores_ex(const uint16_t *d_acts, const float *d_refs,
                             uint32_t n_shards, uint32_t n_canaries,
                             uint64_t seg_len, float *d_scores,
                             uint64_t stat_stride, void *d_ws, size_t ws_bytes,
                             int32_t *d_status, int32_t algo, cg_stream_t stream);

/*
 * cg_drift_scores over a batch of C = n_configs configurations of the same
 * shape in one launch pair (the factorial and the substudies score many
 * configurations of equal shape, Sec. 4.4; a launch over several of them
 * amortises the pipeline's fill and drain).  d_acts fp16 and d_refs fp32
 * are [C][S][N][seg_len], 16-byte aligned; the scores of configuration c go
 * to d_scores[stat * stat_stride + c * N * S + n * S + s] (stat_stride >=
 * C * N * S; pass C * N * S for a dense [3][C][N][S] block, whose per-stat
 * [C][N][S] slices are cg_auroc's input).  d_ws: >= cg_drift_workspace_size(
 * C * S, N, seg_len) bytes, 16-byte aligned, scratch.  Kernel choice,
 * numerics and every other rule are those of cg_drift_scores; C = 1 is
 * cg_drift_scores itself.
 */
cg_status cg_drift_scores_batch(const uint16_t *d_acts, const float *d_refs,
                                uint32_t n_configs, uint32_t n_shards,
                                uint32_t n_canaries, uint64_t seg_len,
                                float *d_scores, uint64_t stat_stride, void *d_ws,
                                size_t ws_bytes, int32_t *d_status,
                                cg_stream_t stream);

/*
 * cg_drift_scores with the live activations in pinned host memory: the
 * drift kernel reads h_acts directly over the host-GPU link (one pass, no
 * staging copy in HBM) while the references stay resident in device memory,
 * as the verifier's stored fp32 references do (Sec. 3.3).  h_acts must be
 * page-locked host memory known to CUDA (cudaHostAlloc or cudaHostRegister);
 * anything else returns CG_ERR_INVALID_ARG before any launch.  It must stay
 * unmodified until the call's work on `stream` completes.  All other
 * arguments, layouts and results are those of cg_drift_scores.
 */
cg_status cg_drift_scores_host(const uint16_t *h_acts, const float *d_refs,
                               uint32_t n_shards, uint32_t n_canaries,
                               uint64_t seg_len, float *d_scores,
                               uint64_t stat_stride, void *d_ws, size_t ws_bytes,
                               int32_t *d_status, cg_stream_t stream);

/*
 * cg_drift_scores without a workspace: same arguments, layouts and results
 * as cg_drift_scores, but the per-chunk partial sums go to a fixed 4 MiB
 * array of device memory inside the library, so the call allocates nothing
 * and needs no scratch buffer from the caller.  The paper has no
 * counterpart; this exists for callers that cannot allocate device memory
 * on their scoring path: a verifier embedded in an inference server whose
 * memory pool already holds nearly all of HBM (weights and KV cache) and
 * gives plug-ins no allocator, or a serving loop that cannot afford the
 * device-wide synchronisation cudaMalloc/cudaFree may cause.
 *   Limit: n_shards * n_canaries * ceil(seg_len / CG_NOALLOC_CHUNK_ELEMENTS)
 *   <= CG_NOALLOC_MAX_WORK_ITEMS (e.g. 4096 segments of 2^20 elements);
 *   larger problems return CG_ERR_UNSUPPORTED before any launch.
 *   The 4 MiB are held on each device where the library's device code is
 *   loaded (its first kernel launch or first call of this entry point on
 *   that device, under CUDA's default lazy module loading) until the
 *   process exits.  Every call looks up the array's device address
 *   (cudaGetSymbolAddress) with the current device; the first such lookup on
 *   a device loads the module there, so make that first call before any
 *   stream capture.
 *   Every call shares the array: calls that overlap on the GPU (on
 *   different streams or from different host threads) race and corrupt
 *   each other's results; serialise them on one stream.  Nothing in it
 *   needs to start at zero: every partial is written before it is read.
 *   d_status is checked for alignment and otherwise unused: this path runs
 *   the register-streaming kernel, which has no wait that could give up
 *   (a NaN element shows in the scores, as with cg_drift_scores).
 */
#define CG_NOALLOC_CHUNK_ELEMENTS 16384u
#define CG_NOALLOC_MAX_WORK_ITEMS 262144u
cg_status cg_drift_scores_noalloc(const uint16_t *d_acts, const float *d_refs,
                                  uint32_t n_shards, uint32_t n_canaries,
                                  uint64_t seg_len, float *d_scores,
                                  uint64_t stat_stride, int32_t *d_status,
                                  cg_stream_t stream);

/*
 * Scrambled-label negative control (Sec. 4.5).  For every configuration c
 * and canary n, a stage j* is drawn uniformly from the stages labelled 0 in
 * d_labels (ascending order; Philox aux stream 4 with config id
 * config_id0 + c) and labelled 1; the stages labelled 1 in d_labels become
 * -1 (left out); the other benign stages stay 0.
 * d_labels, d_ctrl: int8 [C][N][S].  A canary with no benign stage gets no
 * j* and raises CG_DEVFLAG_NO_BENIGN.
 */
cg_status cg_make_control_labels(const int8_t *d_labels, uint32_t n_configs,
                                 uint32_t n_canaries, uint32_t n_shards,
                                 uint64_t seed, uint32_t config_id0,
                                 int8_t *d_ctrl, int32_t *d_status,
                                 cg_stream_t stream);

/*
 * Exact Mann-Whitney counts and AUROC (Eq. 5, Eq. 6).
 *   d_scores fp32 [C][N][S] (one statistic), d_labels int8 [C][N][S]:
 *   1 = malicious, 0 = benign, anything else = left out.
 * Per (c, n): gt = #{(i, j): label 1, label 0, m_i > m_j},
 *             eq = #{same pairs with m_i == m_j},
 *             d_u2[c][n] = 2 gt + eq (twice U; ties count one half).
 * Per c: d_auroc[c] = mean over canaries with at least one pair of
 * U / (c_t b_t); when every such canary has the same pair count P this is
 * sum(u2) / (2 P N_valid), one fp64 division of exact integers; otherwise
 * the per-canary ratios are added in canary order.  NaN when no canary has
 * a pair.  d_u2 and d_auroc are required; d_gt, d_eq may be NULL.  A NaN
 * labelled score raises CG_DEVFLAG_NAN_SCORE (its comparisons count as
 * neither greater nor equal).  S up to 1024.
 */
cg_status cg_auroc(const float *d_scores, const int8_t *d_labels,
                   uint32_t n_configs, uint32_t n_canaries, uint32_t n_shards,
                   int64_t *d_u2, int64_t *d_gt, int64_t *d_eq,
                   double *d_auroc, int32_t *d_status, cg_stream_t stream);

/*
 * Pooled Mann-Whitney AUROC: per configuration, every malicious score of
 * every canary against every benign score of every canary (the U statistic
 * the paper names as equivalent to its ranking test, Sec. 3.4; the
 * per-canary mean of cg_auroc is Eq. 6 itself).  d_scores fp32 / d_labels
 * int8 [C][N][S] as in cg_auroc.  Per configuration: d_u2[c] = 2 U (ties
 * count one half), d_n_mal[c], d_n_ben[c] (may be NULL) and
 * d_auroc[c] = u2 / (2 n_mal n_ben), one fp64 division of exact integers
 * (NaN without a pair).  NaN scores are left out of the pool and raise
 * CG_DEVFLAG_NAN_SCORE.  N * S up to 16384.
 */
cg_status cg_auroc_pooled(const float *d_scores, const int8_t *d_labels,
                          uint32_t n_configs, uint32_t n_canaries, uint32_t n_shards,
                          int64_t *d_u2, int64_t *d_n_mal, int64_t *d_n_ben,
                          double *d_auroc, int32_t *d_status, cg_stream_t stream);

/*
 * Diagnostic of the failure path of the library's device waits (the
 * bulk-copy drift pipeline waits on mbarriers with a time limit): one warp
 * waits on an mbarrier phase that nothing completes, gives up after
 * limit_us microseconds (1 .. 10^7) and raises CG_DEVFLAG_TIMEOUT in
 * d_status (required), which cg_read_status then reports as
 * CG_ERR_TIMEOUT.  The device stays usable afterwards.
 */
cg_status cg_selftest_bounded_wait(uint32_t limit_us, int32_t *d_status, cg_stream_t stream);

/*
 * Synchronise `stream`, read the device status word and map it: 0 ->
 * CG_OK, else the first of CG_ERR_TIMEOUT, CG_ERR_NAN_SCORE,
 * CG_ERR_NO_BENIGN that is set.  The raw word goes to *h_word if non-NULL.
 * The word is not cleared.
 */
cg_status cg_read_status(const int32_t *d_status, cg_stream_t stream,
                         int32_t *h_word);

#ifdef __cplusplus
}
#endif

#endif /* CANARY_GUARD_H */
