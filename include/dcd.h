/*
 * dcd.h -- C ABI of the GB300 (sm_103a) contrastive-decoding verification library.
 *
 * The library implements the verification step of Decoupled Contrastive Decoding
 * (arxiv 2608.12913, Algorithm 1): for every node of a drafted token tree it turns
 * the expert's and the amateur's vocabulary-wide logits into the CD target
 *
 *     log pi_CD(x) = (1 + alpha) log pi_p(x) - alpha log pi_q(x) - log Z_CD      (Eq. 1)
 *
 * optionally restricted to the expert-plausibility set
 *     P_beta = { x : pi_p(x) >= beta * max_x' pi_p(x') }                          (Sec. 2.1)
 * and sharpened by a temperature T (pi_CD,T proportional to exp(score / T) on P_beta),
 * applies the greedy (T = 0) or the speculative-sampling acceptance rule, and walks
 * the tree to the longest accepted path and its bonus token.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - B sequences, N tree nodes per sequence (the root included), vocabulary V.
 *   Rows are numbered g = b * N + n; row g of a logit matrix holds the next-token
 *   logits after node n of sequence b, i.e. the distribution node n's children
 *   were drafted from.  The root's own token is context and is not verified.
 * - parents[b*N + 0] = -1 and 0 <= parents[b*N + n] < n for n >= 1 (BFS-compatible
 *   order); tokens[b*N + n] in [0, V) for n >= 1.  These device-resident arrays are
 *   checked on the device: a violation sets a bit of the device error word (read
 *   it with dcd_get_device_error) and that sequence reports accept_len = 0,
 *   bonus = -1; nothing traps.
 * - Siblings are tried in ascending node id.  Greedy: a child is accepted iff its
 *   token equals the argmax of the CD score over P_beta (ties -> lowest token id;
 *   duplicate sibling tokens -> lowest node id).  Sampled (T > 0): with r_0 = pi_CD,T
 *   child j is accepted iff u_j <= r_{j-1}(t_j) / q(t_j); after a rejection
 *   r_j = normalise(max(0, r_{j-1} - q)) (Algorithm 1, generalised to sibling lists);
 *   a node with no accepted child draws its terminal token from its last residual r
 *   (pi_CD,T at a leaf) by a two-level exponential race: the block k of 1024
 *   consecutive tokens maximising log R_k - log(-log v_k), R_k = sum of r over the
 *   block, then the token x of that block maximising log r(x) - log(-log u_x).  The
 *   two levels together draw x with probability r(x) (Algorithm 1 leaves the sampling
 *   method open).
 * - Randomness: Philox4x32-10 (Salmon et al., SC'11), key = (seed_lo, seed_hi).
 *   The acceptance uniform of node c uses counter (b*N + c, 0, offset_lo, offset_hi)
 *   word 0; in row g the block uniform v_k uses counter (g, 2^31 + k/4, offset_lo,
 *   offset_hi) word k%4 and the token uniform u_x counter (g, 1 + x/4, offset_lo,
 *   offset_hi) word x%4; a word w maps to u = ((w >> 9) + 0.5) * 2^-23 in (0, 1).
 *   One call consumes one offset value: advance `offset` by one per call.
 * - accept_len[b] counts accepted drafted tokens (the bonus token is excluded, as in
 *   the paper's mean accepted length L, App. D).  accept_path[b*N + i] lists the
 *   accepted node ids from the root (accept_path[b*N] = 0), padded with -1.
 * - Optional outputs (may be NULL): cd_logprob[b*N + n] = log pi_CD,T_eff(token_n)
 *   under the parent's row (root: 0; -inf outside P_beta), cd_argmax[g] = argmax of
 *   the CD score of row g, cd_lse[g] = log sum_{x in P_beta} exp(s'(x) / T_eff) with
 *   the raw-logit score s' = (1 + alpha) z_p - alpha z_q (so log pi_CD,T(x) =
 *   s'(x) / T_eff - cd_lse[g]); T_eff = T, or 1 for greedy sequences.
 * - Memory: every array pointer is a DEVICE pointer owned by the caller.  The
 *   library allocates nothing per call; scratch lives in the caller's workspace
 *   (dcd_workspace_bytes: 256 bytes plus, per row, 532 bytes and 16 bytes per
 *   residual piece -- a piece covers 16384 vocabulary tokens with bf16 logits, 8192
 *   with fp32, half that in calls of at most 256 rows -- rounded up to 256; 660 bytes
 *   a row at V = 128256 in bf16; its contents need no initialisation).  Calls are asynchronous and ordered on
 *   `stream`; host-side argument checks return a negative status before anything is
 *   launched.  Two calls that share a workspace must not overlap on the device.
 * - Vocabulary limit: the streaming kernel keeps 8 bytes per 1024 vocabulary tokens
 *   (per 512 with fp32 logits) of the row in flight in shared memory, next to its
 *   64 KB ring.  A shape for which that does not fit in a CTA's 227 KB -- V above
 *   about 18 million tokens with bf16 logits, 9 million with fp32, at N = 1024; a
 *   little more for smaller trees -- returns DCD_ERR_UNSUPPORTED (the one-launch
 *   greedy path of small calls has no such limit).
 * - Thread safety: entry points may be called from several host threads, each with
 *   its own workspace.
 */
#ifndef DCD_H_
#define DCD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* dcd_stream_t;

/* Status codes returned by every entry point. */
enum {
  DCD_OK = 0,
  DCD_ERR_INVALID_ARG = -1, /* null pointer, bad size, stride or dtype */
  DCD_ERR_BAD_TREE = -2,    /* reserved: tree checks run on the device (see error word) */
  DCD_ERR_UNSUPPORTED = -3, /* valid request this build cannot serve (e.g. N > DCD_MAX_NODES) */
  DCD_ERR_CUDA = -4,        /* a CUDA runtime call or kernel launch failed */
  DCD_ERR_TIMEOUT = -5,     /* a bounded device wait gave up (reported via the error word) */
  DCD_ERR_DEVICE_INPUT = -6,/* dcd_get_device_error found a nonzero error word */
  DCD_ERR_WORKSPACE = -7    /* workspace missing, misaligned (256 B) or too small */
};

/* Logit element types. */
enum { DCD_F32 = 0, DCD_BF16 = 1 };

/*
 * dcd_shape.flags: DCD_SIBLINGS_DISTINCT selects the sampled rule for sibling lists drawn
 * WITHOUT replacement from q (distinct drafted tokens, EAGLE-style top-k sampling): sibling j
 * is tested against r_{j-1} with its actual proposal q_{j-1} = q without the tokens of siblings
 * 1..j-1, renormalised, which also replaces q in the residual step r_j = normalise(max(0,
 * r_{j-1} - q_{j-1})).  Without the flag siblings are taken as i.i.d. draws from q.  The flag
 * supports nodes with at most 32 children (more: DCD_DEVERR_UNSUPPORTED for the sequence).  q
 * is taken as given: the first sibling's proposal is q itself, and a renormalised proposal
 * divides by the mass that remains, q's own sum (measured in the first residual pass; a
 * top-k-truncated drafter's rows sum to less than 1) less the removed tokens' q.
 */
#define DCD_SIBLINGS_DISTINCT 0x1

/* Bits of the device error word (dcd_get_device_error). */
#define DCD_DEVERR_BAD_PARENT 0x1u  /* parents[] violates the ordering rule */
#define DCD_DEVERR_BAD_TOKEN 0x2u   /* a drafted token is outside [0, V) */
#define DCD_DEVERR_NONFINITE 0x4u   /* NaN / +inf reached a row's max or normaliser */
#define DCD_DEVERR_TIMEOUT 0x8u     /* a bounded wait on an asynchronous copy expired */
#define DCD_DEVERR_BAD_PARAM 0x10u  /* alpha < 0, beta outside [0, 1], T < 0 or non-finite */
#define DCD_DEVERR_UNSUPPORTED 0x20u /* a node has more children than the call supports (fused
                                        LM-head: 8; DCD_SIBLINGS_DISTINCT: 32) */

/* Largest tree (nodes per sequence, root included) the library accepts. */
#define DCD_MAX_NODES 1024

typedef struct {
  int32_t B;            /* sequences (>= 0) */
  int32_t N;            /* nodes per sequence, root included (1 .. DCD_MAX_NODES) */
  int64_t V;            /* vocabulary size (1 .. 2^31 - 1; see the shared-memory limit below) */
  int32_t logits_dtype; /* DCD_F32 or DCD_BF16, for z_exp and z_ama */
  int32_t flags;        /* 0, or DCD_SIBLINGS_DISTINCT (sampled calls); other bits must be 0 */
  int64_t ld_logits;    /* row stride of z_exp / z_ama in elements (>= V) */
  int64_t ld_q;         /* row stride of q in fp32 elements (>= V; sampled calls only) */
} dcd_shape;

/*
 * Bytes of device workspace a call with this shape needs (the same value serves
 * greedy and sampled calls).  Returns 0 for an invalid shape.
 */
size_t dcd_workspace_bytes(const dcd_shape* shape);

/*
 * Greedy CD verification (T = 0 for every sequence).  Eq. 1 with the plausibility
 * mask of Sec. 2.1; acceptance is the T -> 0 limit of Algorithm 1.
 *   z_exp, z_ama : [B*N rows, ld_logits] logits of the expert M_p and amateur M_q.
 *   tokens, parents : int32 [B, N] draft tree (see conventions).
 *   alpha : fp32 [B], contrastive strength alpha >= 0 (Eq. 1).
 *   beta  : fp32 [B] plausibility threshold in [0, 1], or NULL for beta = 0.
 *   accept_len [B], accept_path [B, N], bonus [B] : int32 outputs.
 *   cd_logprob [B, N], cd_argmax [B, N], cd_lse [B, N] : optional outputs (NULL skips).
 *   workspace : device scratch of at least dcd_workspace_bytes(shape), 256-byte aligned.
 * A small call (B*N <= 512 rows and N <= 256: chains and small trees of single-request
 * decoding) runs as one kernel after a memset of the workspace counters; larger calls run the
 * streaming kernel and the tree walk (dcd_score_rows + dcd_tree_walk).  Both give the same
 * accepted paths; the scores differ only by the order of fp32 summation.
 */
int dcd_verify_greedy(const dcd_shape* shape, const void* z_exp, const void* z_ama, const int32_t* tokens,
                      const int32_t* parents, const float* alpha, const float* beta, int32_t* accept_len,
                      int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax,
                      float* cd_lse, void* workspace, size_t workspace_bytes, dcd_stream_t stream);

/*
 * Speculative-sampling CD verification (Algorithm 1 on trees); sequences whose
 * temperature is 0 follow the greedy rule within the same call.
 *   q : fp32 [B*N rows, ld_q]; row g is the draft distribution pi_e that node n's
 *       children were drawn from.  Read only for non-leaf rows of T > 0 sequences.
 *   temperature : fp32 [B], T >= 0.
 *   seed, offset : Philox key and stream position (see conventions).
 *   residual : optional fp32 [B, V]; receives the distribution each sequence's bonus
 *       token was drawn from (the last node's final residual; one-hot at the bonus
 *       for greedy sequences).  Meant for tests; costs one extra pass per sequence.
 * Other arguments as for dcd_verify_greedy.
 */
int dcd_verify_sample(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                      const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                      const float* temperature, uint64_t seed, uint64_t offset, int32_t* accept_len,
                      int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax,
                      float* cd_lse, float* residual, void* workspace, size_t workspace_bytes,
                      dcd_stream_t stream);

/*
 * The two steps dcd_verify_sample is made of, exposed for step-level timing.
 * dcd_score_rows runs the per-row work (Eq. 1 target, row reductions, sibling
 * acceptance tests, terminal draws) and leaves one record per row in the workspace;
 * q and temperature may be NULL for an all-greedy call.  dcd_tree_walk then
 * follows the accepted children from each root and writes accept_len, accept_path
 * and bonus.  Calling them back to back equals one dcd_verify_sample call with
 * residual = NULL.
 */
int dcd_score_rows(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                   const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                   const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob,
                   int32_t* cd_argmax, float* cd_lse, void* workspace, size_t workspace_bytes,
                   dcd_stream_t stream);

int dcd_tree_walk(const dcd_shape* shape, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                  void* workspace, size_t workspace_bytes, dcd_stream_t stream);

/*
 * Capacity of the scratch array inside the library used by dcd_verify_sample_noalloc:
 * enough for dcd_workspace_bytes(shape) <= 4 MiB, e.g. B * N up to 6,354 rows at
 * V = 128256 with bf16 logits.
 */
#define DCD_STATIC_SCRATCH_BYTES (4u * 1024u * 1024u)

/*
 * dcd_verify_sample without a workspace argument, for callers that cannot allocate
 * device memory: for example a plugin inside an inference engine that reserves all
 * device memory for its own allocator, or a hook that must not call cudaMalloc or
 * cudaFree because they can synchronise the device or fail under a fixed budget.
 * (The paper has no counterpart; this is a deployment convenience of the library.)
 * The caller still passes every input and output; the scratch lives in one array of
 * DCD_STATIC_SCRATCH_BYTES compiled into the library, which every GPU that loads the
 * library holds until the process exits.  Shapes needing more scratch return
 * DCD_ERR_UNSUPPORTED.  Nothing is allocated: no cudaMalloc, cudaFree or allocating
 * library call.  The first call on a device, and the first after the device gets a new
 * context (e.g. after cudaDeviceReset), looks up the array's device address (with that
 * device current) and caches it for that context; make that first call before any stream
 * capture.  All calls share the one array and it keeps the last call's contents (each call
 * resets the error word before its kernels run), so calls that overlap on the GPU, from any
 * stream or thread, race and must be serialised by the caller.  dcd_get_device_error
 * cannot read this scratch; device-side input errors still show as accept_len = 0 and
 * bonus = -1 for the affected sequences, and a bounded device wait that gave up
 * (DCD_DEVERR_TIMEOUT) shows as accept_len = 0 and bonus = -1 for every sequence of the
 * call, so a record left by an earlier call is never reported as this call's result.
 * Arguments and results otherwise as dcd_verify_sample.
 */
int dcd_verify_sample_noalloc(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                              const int32_t* tokens, const int32_t* parents, const float* alpha,
                              const float* beta, const float* temperature, uint64_t seed, uint64_t offset,
                              int32_t* accept_len, int32_t* accept_path, int32_t* bonus, float* cd_logprob,
                              int32_t* cd_argmax, float* cd_lse, float* residual, dcd_stream_t stream);

/*
 * Staging of a sampled call's draft distributions from host memory: copies into q_dev the
 * rows of q_host that dcd_verify_sample reads -- the rows of sequences with a positive
 * temperature whose node has at least one child (the sibling test reads q at the
 * children's tokens and a residual pass the whole row, Algorithm 1; a leaf draws its
 * terminal token from pi_CD alone).  Every other row of q_dev keeps its contents.
 *   shape       : B, N, V and ld_q (the row stride, in floats, of both q_host and q_dev;
 *                 >= V); logits_dtype and ld_logits as for dcd_verify_sample.
 *   q_host      : fp32 [B*N, ld_q] in page-locked host memory mapped into the device's
 *                 address space (cudaHostAlloc, or cudaHostRegister with the mapped flag);
 *                 the GPU reads it directly, in one launch, at the host link's rate.
 *   q_dev       : fp32 [B*N, ld_q] device memory.
 *   parents, temperature : the call's DEVICE arrays as for dcd_verify_sample (already on
 *                 the device: the copy is ordered after them on `stream`).
 * Returns DCD_ERR_INVALID_ARG for a bad shape, a null pointer, or a q_host whose first or
 * last element is not mapped page-locked host memory (nothing is launched).  Asynchronous
 * on `stream`; the caller keeps q_host unchanged until the copy completes.
 */
int dcd_upload_q_rows(const dcd_shape* shape, const float* q_host, float* q_dev, const int32_t* parents,
                      const float* temperature, dcd_stream_t stream);

/*
 * dcd_score_rows with an explicit launch geometry, for tests and tuning: `stages` is
 * the depth of each CTA's ring of shared-memory stages (0 = automatic, else 2 .. 8)
 * and `plain_loads` = 1 stages rows with ordinary loads instead of bulk asynchronous
 * copies.  Results equal dcd_score_rows up to fp32 summation order.
 * `poll_limit_cycles` bounds, in SM clock cycles, the wait of a CTA whose rows are all
 * claimed for residual passes that other CTAs may still publish (0 = the default bound of
 * about two seconds; negative values are rejected).  No copy is in flight during that wait,
 * so a short bound exercises the timeout path safely: the CTA stops, the call sets
 * DCD_DEVERR_TIMEOUT in the error word, every sequence of a following dcd_tree_walk reports
 * accept_len = 0 and bonus = -1, and the device stays usable.  Meant for tests.
 */
int dcd_score_rows_ex(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                      const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                      const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob,
                      int32_t* cd_argmax, float* cd_lse, void* workspace, size_t workspace_bytes,
                      dcd_stream_t stream, int stages, int plain_loads, int64_t poll_limit_cycles);

/*
 * Greedy CD verification fused with the two models' output projections (LM heads): the
 * logits z_p = h_exp W_exp^T and z_q = h_ama W_ama^T of Eq. 1 are computed on the tensor
 * cores tile by tile and reduced in place, never written to memory.  The target is Eq. 1
 * with beta = 0 (the untruncated target, Sec. 2.1) and the greedy rule (the T -> 0 limit of
 * Algorithm 1), exactly as dcd_verify_greedy with beta = NULL on the logits
 * h W^T computed with fp32 accumulation of the bf16 products.
 *   shape : B, N, V as for dcd_verify_greedy; logits_dtype must be DCD_BF16 (the type of
 *       h and W); ld_logits and ld_q are not used.
 *   h_exp : bf16 [B*N, H_exp] row-major, the expert's final hidden state after each node
 *       (row g = b*N + n, the same row convention as the logits).
 *   w_exp : bf16 [V, H_exp] row-major, the expert's output embedding (the layout of an
 *       nn.Linear weight: row v produces logit v).
 *   h_ama, w_ama : the amateur's, [B*N, H_ama] and [V, H_ama].
 *   H_exp, H_ama : hidden sizes, >= 1 and multiples of 8 (16-byte rows); every matrix base
 *       16-byte aligned.
 *   tokens, parents, alpha, accept_len, accept_path, bonus, cd_logprob, cd_argmax,
 *       cd_lse : as for dcd_verify_greedy (beta is 0 here; dcd_verify_fused_lmhead_ex takes it).  A node may have at most 8 children
 *       (else its sequence reports DCD_DEVERR_UNSUPPORTED and accept_len = 0).
 *   workspace : device scratch of at least dcd_fused_workspace_bytes(shape), 256-byte
 *       aligned; about 16 * B * N * ceil(V / 256) bytes.
 * Returns DCD_ERR_UNSUPPORTED if the driver cannot describe the matrices to the tensor
 * memory accelerator.  Errors found on the device are read with dcd_get_device_error.
 */
size_t dcd_fused_workspace_bytes(const dcd_shape* shape);

int dcd_verify_fused_lmhead(const dcd_shape* shape, const void* h_exp, int32_t H_exp, const void* w_exp,
                            const void* h_ama, int32_t H_ama, const void* w_ama, const int32_t* tokens,
                            const int32_t* parents, const float* alpha, int32_t* accept_len,
                            int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax,
                            float* cd_lse, void* workspace, size_t workspace_bytes, dcd_stream_t stream);

/*
 * dcd_verify_fused_lmhead with the plausibility mask and timing events.
 *   beta : fp32 [B] device plausibility thresholds in [0, 1] (Sec. 2.1), or NULL for beta = 0.
 *       With beta, the tensor-core kernel runs twice: a first sweep over the expert's hidden
 *       size only finds each row's max z_p (the same MMAs in the same order as the second sweep,
 *       so both see bit-identical logits), and the second scores only the tokens with
 *       z_p - max z_p >= log beta.  That costs the expert GEMM once more (about 1.8x the FLOPs
 *       of a call without beta at H_exp = 4 H_ama); a sequence with beta = 0 is not masked.
 *   gemm_start, gemm_stop : two CUDA events (cudaEvent_t handles, or NULL) recorded on
 *       `stream` immediately before the first and after the last tensor-core sweep, for timing
 *       them alone.
 * With beta NULL the results equal dcd_verify_fused_lmhead.
 */
int dcd_verify_fused_lmhead_ex(const dcd_shape* shape, const void* h_exp, int32_t H_exp, const void* w_exp,
                               const void* h_ama, int32_t H_ama, const void* w_ama, const int32_t* tokens,
                               const int32_t* parents, const float* alpha, const float* beta,
                               int32_t* accept_len, int32_t* accept_path, int32_t* bonus, float* cd_logprob,
                               int32_t* cd_argmax, float* cd_lse, void* workspace, size_t workspace_bytes,
                               dcd_stream_t stream, void* gemm_start, void* gemm_stop);

/*
 * Per-row diagnostics of contrastive verification: the quantities behind the signal versus
 * proposal-error analysis (Sec. 3.1), the alignment-gap estimator (App. C) and the KL
 * decomposition of the CD target (App. B, Lemma kl_decomposition).  For every row r of the B*N
 * rows, with pi_p = softmax(z_exp[r]), pi_q = softmax(z_ama[r]) over the full vocabulary (no
 * temperature, no plausibility mask) and e = q[r] (the drafter's distribution):
 *   diag[r][0] = lse_p = log sum_x exp(z_exp[r][x])
 *   diag[r][1] = lse_q = log sum_x exp(z_ama[r][x])
 *   diag[r][2] = signal = |log pi_p(x*) - log pi_q(x*)| at x* = xstar[r] (the CD argmax, e.g.
 *                the cd_argmax output of a verification call); NaN if xstar is NULL or
 *                xstar[r] is outside [0, V)
 *   diag[r][3] = E_{pi_q}[log pi_p - log pi_q]   (= -D_KL(pi_q || pi_p))
 *   diag[r][4] = E_e[log pi_p - log pi_q]         (NaN if q is NULL)
 *   diag[r][5] = D_KL(e || pi_p), 0 log 0 = 0     (NaN if q is NULL)
 *   diag[r][6] = D_KL(pi_p || pi_q)               (= E_{pi_p}[log pi_p - log pi_q])
 *   diag[r][7] = D_KL(pi_p || pi_CD) = log Z_CD - alpha D_KL(pi_p || pi_q), the lemma of App. B
 *                for the untruncated target at T = 1, pi_CD = pi_p^(1+alpha) pi_q^(-alpha) / Z_CD,
 *                with log Z_CD = cd_lse[r] - (1 + alpha) lse_p + alpha lse_q taken from the
 *                cd_lse output of a verification call on the same logits.  NaN if cd_lse is NULL,
 *                or if the row's sequence has beta > 0 or a temperature other than 0 or 1 (the
 *                lemma does not hold for a masked or tempered target).
 * The alignment gap of App. C is diag[4] - diag[3] averaged over the rows a caller selects.
 *   shape : B, N, V, logits_dtype, ld_logits as for the verification calls; ld_q (>= V) when q
 *       is given; flags must be 0.
 *   z_exp, z_ama : [B*N, ld_logits] device logits; q : [B*N, ld_q] fp32 device probabilities or
 *       NULL; xstar : int32 [B*N] device tokens or NULL; diag : fp32 [B*N, 8] device output.
 *   cd_lse : fp32 [B*N] device values (the verification call's cd_lse output), or NULL;
 *   alpha, beta, temperature : fp32 [B] device arrays of that verification call (alpha is
 *       required with cd_lse and must be NULL without it; beta and temperature may be NULL for
 *       0, i.e. unmasked and greedy).
 *   workspace : device scratch of at least dcd_diagnostics_workspace_bytes(shape) bytes,
 *       256-byte aligned (about 48 * B * N * ceil(V / 2048) bytes).
 * Logits must be finite (non-finite inputs give NaN or inf results; no error word is kept).
 * One pass over the inputs (fp32 accumulation) and a per-row combine, stream-ordered on
 * `stream`.  Returns DCD_ERR_INVALID_ARG or DCD_ERR_WORKSPACE for bad arguments, DCD_ERR_CUDA
 * if a launch fails.
 */
#define DCD_DIAG_COLS 8

size_t dcd_diagnostics_workspace_bytes(const dcd_shape* shape);

int dcd_row_diagnostics(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                        const int32_t* xstar, const float* cd_lse, const float* alpha, const float* beta,
                        const float* temperature, float* diag, void* workspace, size_t workspace_bytes,
                        dcd_stream_t stream);

/* dcd_row_diagnostics that also records two CUDA events (cudaEvent_t, or NULL) on `stream`
 * immediately before and after the streaming pass (the per-row combine follows it). */
int dcd_row_diagnostics_ex(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                           const int32_t* xstar, const float* cd_lse, const float* alpha, const float* beta,
                           const float* temperature, float* diag, void* workspace, size_t workspace_bytes,
                           dcd_stream_t stream, void* pass_start, void* pass_stop);

/*
 * Synchronises `stream`, then copies the device error word of `workspace` (the OR of
 * the DCD_DEVERR_* bits raised by the last call that used it) into *bits.  Returns
 * DCD_OK when the word is zero, DCD_ERR_DEVICE_INPUT when it is not, DCD_ERR_CUDA if
 * the copy fails.
 */
int dcd_get_device_error(const void* workspace, dcd_stream_t stream, uint32_t* bits);

/* Static English text for a status code. */
const char* dcd_status_string(int status);

/* Library version, major * 10000 + minor * 100 + patch. */
int dcd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DCD_H_ */
