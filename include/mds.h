/*
 * mds.h -- C ABI of the GB300 multi-draft speculative verification library.
 *
 * The library verifies K draft branches of L tokens per sequence against a
 * target model, as in "Multi-Draft Speculative Sampling: Canonical
 * Decomposition and Theoretical Limits" (arXiv 2410.18234).  For every depth
 * j of every sequence b it computes the temperature softmax of the target row
 * and of one row per distinct draft model (Section 3), chooses one
 * intermediate token Y among the valid draft tokens with an importance step
 * (Definition 1; Theorem 1's canonical decomposition), applies the
 * single-draft speculative step to Y (Appendix A, Algorithm 1: accept with
 * probability min(1, q(Y)/p_I(Y)), else resample the normalised residual
 * max(0, q - p_I)), and walks the draft tree: the walk continues while the
 * output token is one of the valid draft tokens (the event Z in S of
 * Problem 1), and after L accepted positions a bonus token is drawn from the
 * target row at depth L.
 *
 * Notation follows the paper: q is the target distribution, p a draft
 * distribution, p_I the law of the intermediate token.
 *
 * Random numbers: Philox4x32-10 (Salmon et al., SC'11) with counter
 * (b, j, draw, 0) and key (seed low 32 bits, seed high 32 bits); the uniform
 * is (word0 >> 8) * 2^-24.  Draw ids: 0..15 importance-step selection (stage
 * m of the pairwise stages uses m), 16..31 accept (the sequential-rejection
 * baseline's round i uses 16 + i), 32 residual, 33 bonus, 34 truncated
 * alphabet keep test, 35 truncated alphabet replacement.
 *
 * Threading: a context may be used from one host thread at a time and its
 * calls must not overlap on the GPU (they share a work counter and a status
 * word).  All device work is issued on the caller's stream; mds_verify does
 * not synchronise.
 */
#ifndef MDS_H
#define MDS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes (synchronous argument/launch errors) ---------------- */
#define MDS_OK 0
#define MDS_EINVAL (-1)   /* null pointer, bad enum, misaligned pointer     */
#define MDS_ESHAPE (-2)   /* B, K, L or V outside the supported range       */
#define MDS_EVOCAB (-3)   /* V does not fit the shared-memory budget        */
#define MDS_ECUDA (-4)    /* a CUDA runtime call failed                     */
#define MDS_EUNSUP (-5)   /* unsupported combination (see mds_verify)       */

/* ---- device status bits (read and cleared by mds_status) -------------- */
#define MDS_ST_NONFINITE 1u   /* a row had NaN logits or a zero/inf normaliser */
#define MDS_ST_BADTEMP 2u     /* a temperature was <= 0 or not finite          */
#define MDS_ST_ZERO_RESID 4u  /* residual mass was 0 after a rejection (only by
                                 rounding); the target row was sampled instead */
#define MDS_ST_TIMEOUT 8u     /* a bounded wait on a bulk copy gave up         */
#define MDS_ST_LP_CAP 16u     /* the stage LP hit its augmentation cap         */
#define MDS_ST_BADTOKEN 32u   /* a draft token was outside [0, V) (token 0 used) */
#define MDS_ST_OMEGA0 64u     /* MDS_WIS0: the candidate list could not certify the
                                 cut of Omega_0 (ties around its last entries); the
                                 tokens above the certified bound formed Omega_0.
                                 The output still follows the target; only the
                                 acceptance rate can differ from the exact cut. */

/* ---- limits ------------------------------------------------------------ */
#define MDS_MAX_K 16      /* draft branches per sequence                    */
#define MDS_MAX_L 64      /* draft positions per branch                     */
#define MDS_MAX_S 8       /* LP truncation threshold s (|Omega_1|)          */
#define MDS_MAX_IS_MODELS 4  /* distinct draft models for plain IS          */
#define MDS_MAX_OMEGA0 62 /* |Omega_0| of the truncated alphabet, MDS_WIS0  */
#define MDS_MAX_OMEGA0_CLUSTER 30 /* ... with a cluster size set (per-sequence engine) */
#define MDS_MAX_TOPK 16   /* top_k of the top-k restriction                 */

typedef struct mds_ctx mds_ctx;

/* Importance step.  MDS_SINGLE: Algorithm 1 on the lowest valid branch.
 * MDS_IS: classical importance sampling, Pr(I = i) proportional to
 * q(X_i)/p(X_i) (Section 3, after Definition 1).  MDS_WIS: the paper's
 * weighted importance sampling with the variant truncated LP (appendix
 * "Variant of Truncated LP", Eq. heur2), pairwise stages for K > 2
 * (Remark 4) and the non-iid key q - p_1 p_2 (non-iid appendix).
 * MDS_SPECTR: sequential-rejection baseline (Algorithm 1 applied to the
 * valid drafts in turn against the running residual target).
 * MDS_WIS0: the truncated-alphabet scheme (Section 4) around MDS_WIS.
 * Omega_0 is the set of target tokens whose logit is above the (M+1)-th
 * largest target logit, M = omega0 (at most M tokens; tokens tied at the cut
 * are all left out).  With p_a = q(Omega_0), the WIS stages run on the
 * alphabet Omega_0 against q / p_a, using only the valid draft tokens that
 * lie in Omega_0 with their draft laws restricted to Omega_0 and
 * renormalised (the non-iid appendix's remark); Algorithm 1 against q / p_a
 * gives Y' (drawn from q / p_a directly when no draft token lies in
 * Omega_0).  Y' is kept with probability p_a (draw 34), otherwise the output
 * is drawn from the tokens outside Omega_0 in proportion to q (draw 35).
 * MDS_WISSORT: MDS_WIS with the sorted rule on Omega_2 (Section 4, Eq. heur
 * and Eq. p_Ieq; the non-iid appendix): a pair of tokens outside Omega_1
 * selects the one earlier in key order (larger q - a b, then lower id).
 * Served with top_k > 0 only (MDS_EUNSUP otherwise). */
typedef enum { MDS_SINGLE = 0, MDS_IS = 1, MDS_WIS = 2, MDS_SPECTR = 3, MDS_WIS0 = 4, MDS_WISSORT = 5 } mds_scheme;

/* Storage type of the logits. */
typedef enum { MDS_F32 = 0, MDS_BF16 = 1 } mds_dtype;

typedef struct {
  int max_B;       /* largest batch a call may pass (>= 1)                    */
  int K;           /* draft branches, 1..MDS_MAX_K                            */
  int L;           /* draft positions per branch, 1..MDS_MAX_L                */
  int V;           /* vocabulary size, 1..2^24                                */
  mds_dtype dtype; /* storage type of every logit buffer                      */
  int wis_s;       /* LP truncation threshold s, 1..MDS_MAX_S (0: 5, the value
                      of the paper's experiments, Section 5)                  */
  float is_h;      /* trapezoid step in ln t for plain IS (0: 0.25)           */
  int cluster;     /* CTAs per sequence: 1, 2, 4, 8 or 16 (0: chosen from max_B and the device) */
  int omega0;      /* |Omega_0| for MDS_WIS0, 1..MDS_MAX_OMEGA0 (0: 20; the paper's
                      runs use 10 to 50, Section 5, Table "Effect of LP
                      Truncation and Alphabet Truncation").  Sizes above
                      MDS_MAX_OMEGA0_CLUSTER run on the slice-dataflow engine
                      only: an MDS_WIS0 call that engine does not serve (a
                      cluster size set, see mds_cluster_size) returns
                      MDS_EUNSUP.                                             */
  int acc_prob;    /* 1: out_diag[b][j][2] holds the residual mass R = sum_k
                      max(0, q_k - p_I(k)) at every visited depth below L, so
                      that 1 - R = sum_k min(q_k, p_I(k)) is the depth's
                      acceptance probability (Theorem 1's objective for the
                      depth's draft laws); costs one more pass over the rows
                      at accepted depths.  0: R only after a rejection (0 when
                      accepted).  Used by MDS_SINGLE, MDS_IS and MDS_WIS; for
                      MDS_SPECTR out_diag[b][j][2] is prod_i R_i, the
                      probability that every round rejects (with 1 the rounds
                      after an acceptance are computed too).                  */
  int top_k;       /* 0: off.  1..MDS_MAX_TOPK: every row (target and drafts)
                      is restricted to its top_k largest logits (ties: lower
                      token id first) and renormalised before verification
                      (Section 5's top-k runs, Tables 2 and 3); the caller's
                      draft tokens should come from the restricted draft rows
                      (a token outside them has p_I = 0 and is accepted, as
                      Algorithm 1 reads a zero denominator).  Served for
                      MDS_SINGLE, MDS_WIS, MDS_SPECTR and MDS_WISSORT by the top-k kernel
                      (one CTA per sequence, no cluster); MDS_IS and MDS_WIS0
                      return MDS_EUNSUP.  acc_prob and out_diag as above.     */
} mds_config;

/* Create a context on CUDA device `device`.  Allocates the context's device
 * workspace (a work counter and the status word) and, lazily, the staging
 * buffers of mds_verify_host.  Returns MDS_OK and stores the context in *out,
 * or a negative code (nothing allocated). */
int mds_create(mds_ctx** out, const mds_config* cfg, int device);

/* Verify B sequences (0 <= B <= max_B) on `stream` (a cudaStream_t; NULL for
 * the legacy default stream).  All buffers are caller-owned DEVICE memory in
 * row-major layout:
 *   target_logits  [B][K][L+1][V] dtype: target logits of the node reached by
 *                  branch k after j draft tokens (branches with equal prefixes
 *                  must hold equal rows; the walk reads the lowest valid one)
 *   draft_logits   HOST array of K device pointers, each [B][L][V] dtype:
 *                  branch k's draft-model logits at depth j
 *   draft_model_id HOST array [K] of ids in 0..MDS_MAX_K-1: branches with equal
 *                  ids are i.i.d. drafts of one model (equal rows at equal
 *                  prefixes, equal temperatures)
 *   draft_tokens   [B][K][L] int32 in [0, V)
 *   temperatures   [B][1+K] float32 > 0: target, then one per branch
 *   out_tokens     [B][L+1] int32: the emitted tokens (accepted tokens then the
 *                  correction or bonus token), -1 after them
 *   out_accept_len [B] int32 in [0, L]: accepted draft positions
 *   out_diag       optional [B][L+1][4] float32: per depth q(Y), p_I(Y), the
 *                  residual mass (0 if accepted, unless acc_prob) and Y; NULL
 *                  to skip
 * Pointers must be aligned to the element size; rows whose byte length is a
 * multiple of 16 at 16-byte-aligned bases are fetched with bulk copies.
 * Plain IS supports at most MDS_MAX_IS_MODELS distinct draft models
 * (MDS_EUNSUP otherwise).  For MDS_WIS0, out_diag holds q(Y)/p_a and p_I(Y)
 * of the inner step on Omega_0 (Y = -1 when no draft token lies in it).  Returns MDS_OK after the launch was issued, or a
 * negative code with nothing launched.  Data-dependent anomalies are reported
 * through the status word (mds_status). */
int mds_verify(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits,
               const int32_t* draft_model_id, const int32_t* draft_tokens, const float* temperatures,
               int scheme, uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len,
               float* out_diag, int B, void* stream);

/* Same as mds_verify with every buffer in HOST memory.  When the target and
 * every draft logits buffer are page-locked host memory mapped into the
 * device's address space (cudaHostAlloc / cudaHostRegister with mapping,
 * e.g. torch pin_memory()), the kernel reads the logits in place with plain
 * loads, so only the rows the walk visits cross the host link; otherwise the
 * context first copies them into device buffers it owns (allocated on first
 * use, grown as needed).  Tokens and temperatures are always staged, and the
 * outputs copied back, all on `stream`; the call synchronises the stream
 * before returning. */
int mds_verify_host(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits,
                    const int32_t* draft_model_id, const int32_t* draft_tokens, const float* temperatures,
                    int scheme, uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len,
                    float* out_diag, int B, void* stream);

/* Variant of mds_verify for callers that cannot allocate device memory:
 * code that runs where cudaMalloc is not allowed (for example inside a
 * serving loop whose memory is fixed at start-up, or under an allocator that
 * forbids growth after warm-up) and so cannot create a context.  It takes
 * the configuration directly and the same buffers as mds_verify (caller-
 * owned device memory; same layouts, alignment rules and return codes) and
 * runs the same kernel as mds_verify would for that configuration, so its
 * outputs are the same.  It allocates nothing: the kernels' scratch (a status
 * word, and for single, WIS and WIS0 the slice engine's control words, task
 * ring, per-sequence state and slice records, which grow with B and with the
 * number of slices per row, about V / 8192) lives in a file-scope device
 * array of MDS_NOALLOC_SCRATCH_BYTES (8 MiB) that every GPU loading the
 * library holds until the process exits; a call whose scratch exceeds it
 * (for llama3-like rows of 128k bf16 logits, beyond roughly 1,500 sequences
 * per call) is rejected
 * with MDS_ESHAPE before any launch.  The first call on a device looks up
 * that array's device address and sets kernel attributes, so make it before
 * any stream capture.  Every call clears the parts of the scratch that must
 * start at zero on `stream`, then launches; all calls share the one array,
 * so calls that overlap on the GPU race.  The status word is not reported
 * (use mds_noalloc_status).  The paper has no counterpart to this entry
 * point: it exists only for callers that cannot allocate. */
#define MDS_NOALLOC_SCRATCH_BYTES (8u << 20)
int mds_verify_noalloc(const mds_config* cfg, int device, const void* target_logits,
                       const void* const* draft_logits, const int32_t* draft_model_id,
                       const int32_t* draft_tokens, const float* temperatures, int scheme,
                       uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len, float* out_diag,
                       int B, void* stream);

/* The status word of the last mds_verify_noalloc call on `device`: copies it
 * to the host on `stream` (after that call's kernel) and synchronises the
 * stream, allocating nothing.  Returns the MDS_ST_* bits (>= 0) or a negative
 * code; *msg (if not NULL) as for mds_status.  The word is cleared by the
 * next mds_verify_noalloc call on the device, not by this one. */
int mds_noalloc_status(int device, void* stream, const char** msg);

/* Synchronise the device, read and clear the status word.  Returns the
 * MDS_ST_* bits (>= 0) or a negative code; *msg (if not NULL) receives a
 * static description of the highest set bit. */
int mds_status(mds_ctx* ctx, const char** msg);

/* CTAs per sequence of the context's last launch (for reporting): the
 * cluster size of the per-sequence engine, or 0 when the call ran on the
 * slice-dataflow engine, where every CTA works on every sequence's slices. */
int mds_cluster_size(const mds_ctx* ctx);

/* Softmax export for tests (Sec. 3: q = softmax of the target row, p = of a
 * draft row, both at their temperatures, Sec. 5).  mds_debug_row_stats
 * makes the context's later calls served by the slice-dataflow engine
 * (single, WIS, WIS0; see mds_cluster_size) write, for every depth a
 * sequence's walk visits with a statistics pass, the statistics the kernel
 * derived for each row of that pass: `row_stats` is caller-owned device
 * memory of max_B * (L + 1) * MDS_DEBUG_ROWS * 4 floats, laid out
 * [b][j][r][4] = {M, 1/Z, c = log2(e) / T, source}, source = k for the target
 * row of branch k (r = 0) and 100 + k for the draft row of branch k (r > 0);
 * entries of depths and rows not visited are left untouched.  NULL turns it
 * off.  The per-sequence engine (IS, SpecTr, cluster sizes > 0) writes
 * nothing.  mds_debug_probs then writes, for one row of V logits of
 * `dtype` in device memory, the probability the kernel assigns to every
 * token under such statistics: out[x] = 2^(l_x c - M c) / Z, evaluated by the
 * same device function as every probability on the verification path.
 * Asynchronous on `stream`; MDS_EINVAL for bad arguments. */
#define MDS_DEBUG_ROWS 4
int mds_debug_row_stats(mds_ctx* ctx, float* row_stats);

/* Measurement export for classical IS (Sec. 3, the law p_I of the selected
 * token by the quadrature of its Laplace identity): mds_debug_exp_count
 * makes the context's later IS calls add to *counter (caller-owned device
 * memory, one unsigned 64-bit word) the exponentials of their quadrature
 * node sums, nodes x V x draft rows per visited depth and per residual draw,
 * with the node count each depth chose on the device.  NULL turns it off. */
int mds_debug_exp_count(mds_ctx* ctx, unsigned long long* counter);
int mds_debug_probs(const void* row, int dtype, int V, float M, float invZ, float c, float* out, void* stream);

/* Diagnostics of an instrumented build (compiled with MDS_PHASE_TIMERS; the
 * default build returns MDS_EUNSUP): synchronises device `device`, copies
 * up to n phase counters of the slice-dataflow engine (SM cycles summed over
 * CTAs, and task and decision counts, in the order the library's source
 * lists them) to cycles, clears them and returns how many counters exist. */
int mds_phase_timers(int device, unsigned long long* cycles, int n);

/* Static text for a return code. */
const char* mds_error_string(int code);

/* Free the context and everything it allocated. */
void mds_destroy(mds_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* MDS_H */
