/*
 * acespec.h -- C ABI of the AceSpec verify / sparsify / state-cache path on
 * one GB300 GPU (sm_103a).
 *
 * AceSpec (arXiv 2609.02514) splits speculative decoding between an edge
 * device and a cloud server.  The cloud verifies a drafted main chain of K
 * tokens against the target model and answers with the first-rejection index
 * pi and a sparse target distribution (Sec. III-B); the edge turns a
 * rejection into an O(1) lookup in a probabilistic cache of alternative
 * branches built per draft depth (Sec. III-C, Algorithm 1).  This library
 * implements the vocabulary-wide per-position arithmetic of those steps.
 * Verification follows the modified rejection sampling the paper relies on
 * (Sec. II-A, Chen et al.), whose output has exactly the target distribution.
 *
 * Conventions shared by every entry point
 *   - All array arguments are DEVICE pointers owned by the caller; the
 *     library never allocates, frees or retains them, and allocates no
 *     device memory of its own (aces_cloud_step creates one stream and two
 *     events per device on its first call there).  F_host is the one host
 *     array.
 *   - Work is enqueued on `stream` (aces_cloud_step also on its own stream,
 *     forked from and joined back to `stream`) and the call returns before
 *     it finishes.  A call returns ACES_OK once its kernels are launched.
 *   - Arguments are validated before anything is launched; on
 *     ACES_ERR_INVALID_ARG / ACES_ERR_UNSUPPORTED nothing is enqueued and no
 *     output is touched.  ACES_ERR_CUDA reports a failed launch.
 *   - Layouts are dense row-major with the vocabulary (V) contiguous.
 *     Row r = b * (K + 1) + i addresses position i of sequence b.
 *   - Order of a distribution: ids by (logit desc, id asc); exactly equal
 *     logits are ordered by the lower id.  -0.0 equals +0.0.
 *   - Data errors never trap: they are reported per row in row_status.
 *
 * Reading of points the paper leaves open (the library's contract):
 *   - nucleus: the shortest prefix of the order whose softmax(z/T) mass
 *     reaches top_p (the crossing id is kept); top_p = 1 keeps every id
 *     with a finite logit; p is renormalised over the kept set.
 *   - accept: a_i = [u_i < min(1, p_i(x~_i) / q_i(x~_i))]; q_i(x~_i) <= 0,
 *     NaN, or an out-of-range draft token forces a reject (ACES_ROW_BAD_Q).
 *   - residual: max(0, p - q) is 0 wherever p = 0 for any valid q, so the
 *     draft row q_pi is read only at ids with p > 0; a NaN or negative q at
 *     one of those ids marks row pi ACES_ROW_BAD_Q (out_token -1).
 *   - pi_b = first i with a_i = 0, else K.  When pi < K the emitted token is
 *     drawn from norm(max(0, p_pi - q_pi)) (from p_pi if that is all zero);
 *     when pi = K the bonus token is drawn from p_K.  The draw is the
 *     smallest id j whose prefix sum over ids 0..j exceeds u[b, K] times the
 *     total.
 *   - -inf logits are allowed (probability 0).  NaN or +inf logits, or a row
 *     whose logits are all -inf, mark the row ACES_ROW_NONFINITE.
 */
#ifndef ACESPEC_H
#define ACESPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    ACES_OK = 0,
    ACES_ERR_INVALID_ARG = 1,
    ACES_ERR_UNSUPPORTED = 2,
    ACES_ERR_CUDA = 3
} aces_status;

typedef enum { ACES_F32 = 0, ACES_BF16 = 1 } aces_dtype;

/* bits of row_status */
#define ACES_ROW_NONFINITE 1 /* NaN / +inf logits, or all logits -inf      */
#define ACES_ROW_BAD_Q 2     /* invalid draft probability or draft token   */
#define ACES_ROW_TIMEOUT 4   /* reserved for a kernel that gives up a bounded
                                wait; no current kernel waits on another */

/* The CUDA runtime's cudaStream_t (NULL = legacy default stream). */
typedef struct CUstream_st *aces_stream_t;

/* Limits checked by every entry point. */
#define ACES_MAX_K 16        /* draft length gamma                        */
#define ACES_MAX_V (1 << 20) /* vocabulary                                */
#define ACES_MAX_TOPK 256    /* payload entries per row                   */
#define ACES_MAX_BRANCH 1024 /* branches per depth                        */

/*
 * Bytes of device scratch that aces_verify (B sequences, K >= 1) or
 * aces_sparsify (B rows, K = 0) needs: about 4.2 KiB per target row for
 * aces_verify (almost all of it the row's nucleus, kept for the residual
 * draw when it has at most 512 ids), under 100 bytes per row for
 * aces_sparsify.  The caller allocates it, passes it to the call and must
 * not use it while the call's work is in flight; it needs no
 * initialisation.  Its first 256 bytes keep, from one aces_verify call to
 * the next on the same workspace, statistics of the rows (how deep below
 * their max their nucleus ended, how many were short) that let the row
 * kernel pick its pass before enough of the new call's rows have finished;
 * they choose a pass only, never a result, so any content there (a fresh
 * allocation, another shape's call) gives the same outputs.  Returns 0 for
 * invalid sizes.
 */
size_t aces_workspace_bytes(int B, int K, int V, int k);

/*
 * Cloud-side lossless verification of B drafted chains, fused with the
 * sparse downlink payload (Sec. III-B; Algorithm 1 RECEIVE_WAIT / RESAMPLE
 * inputs; Sec. V-C for the compact payload).
 *
 *   target_logits [B, K+1, V]  float32 or bfloat16 (dt); row K is the bonus
 *                              position after the last draft token
 *   draft_probs   [B, K, V]    float32, the edge model's distributions Q
 *   draft_tokens  [B, K]       int32, the uploaded main chain x~
 *   uniforms      [B, K+1]     float32 in (0,1); u[:, i<K] drive the accept
 *                              tests, u[:, K] the single residual/bonus draw
 *   T > 0, 0 < top_p <= 1      temperature and nucleus mass
 * Outputs:
 *   accept_len    [B]  int32   pi_b, accepted draft tokens (0..K)
 *   out_token     [B]  int32   corrected (pi < K) or bonus (pi = K) token;
 *                              -1 when that row is NONFINITE or its draft
 *                              row holds a NaN / negative probability at an
 *                              id with p > 0
 *   row_status    [B, K+1]     int32 ACES_ROW_* bits per row
 * Sparse payload (k >= 1; k = 0 skips it and the three pointers may be NULL):
 *   topk_ids      [B, K+1, k]  int32   first k ids of every row's nucleus
 *                              in order, -1 padding
 *   topk_probs    [B, K+1, k]  float32 their renormalised p, 0 padding
 *   tail_mass     [B, K+1]     float32 1 - sum of the row's topk_probs
 * workspace / workspace_bytes: device scratch of at least
 *   aces_workspace_bytes(B, K, V, k) bytes, 16-byte aligned.  It includes
 *   4 KiB per row to keep each row's nucleus (when it has at most 512 ids)
 *   for the residual draw, which then reads q at those ids only.
 * Limits: 1 <= B, 1 <= K <= ACES_MAX_K, 2 <= V <= ACES_MAX_V,
 *   0 <= k <= min(V, ACES_MAX_TOPK).
 */
aces_status aces_verify(const void *target_logits, aces_dtype dt, const float *draft_probs,
                        const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                        float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                        int32_t *topk_ids, float *topk_probs, float *tail_mass,
                        int32_t *row_status, void *workspace, size_t workspace_bytes,
                        aces_stream_t stream);

/*
 * aces_verify for callers that cannot allocate device memory themselves.
 * The paper has no counterpart; this is a library convenience.
 *
 * Who needs it: a caller with no device allocator on its serving path.
 * cudaMalloc synchronizes the whole device, which a latency-bound verify loop
 * cannot afford, and some host runtimes that embed this library own all
 * device memory.  Such callers cannot supply aces_verify's workspace.
 *
 * Same arguments, outputs and errors as aces_verify, without the workspace:
 * the scratch is a fixed array of ACES_NOALLOC_SCRATCH_BYTES bytes inside the
 * library, kept on every GPU that loads the library until the process exits.
 * This call allocates nothing.
 *   - Size limit: returns ACES_ERR_UNSUPPORTED (nothing launched) when
 *     B > 876 at K = 16, B > 1196 at K = 8, B > 1463 at K = 4 (the limit
 *     does not depend on V or k).  The scratch keeps nucleus lists only for
 *     B <= 14 at K = 16 (27 at K = 8, 49 at K = 4); without them the
 *     residual draw scans its whole row.  The results are the same either
 *     way.
 *   - Set-up: the first call on each device looks up the array's device
 *     address (cudaGetSymbolAddress) with that device current; make that
 *     first call before any stream capture on the device.
 *   - Sharing: every call on a device uses the same scratch, which keeps the
 *     last call's contents (each call clears what it needs).  Calls whose
 *     work overlaps on the GPU race on it: serialize them (one stream, or
 *     events between streams).
 *   - The looked-up address is kept for the life of the process: no
 *     cudaDeviceReset may come between two calls on a device.
 */
#define ACES_NOALLOC_SCRATCH_BYTES (1 << 20)
aces_status aces_verify_noalloc(const void *target_logits, aces_dtype dt, const float *draft_probs,
                                const int32_t *draft_tokens, const float *uniforms, int B, int K,
                                int V, float T, float top_p, int32_t *accept_len,
                                int32_t *out_token, int k, int32_t *topk_ids, float *topk_probs,
                                float *tail_mass, int32_t *row_status, aces_stream_t stream);

/*
 * aces_verify on the library's exact general row kernel alone: the same
 * arguments, outputs, limits, errors and results (bit for bit), but every
 * row takes the slow path that aces_verify keeps for rows its single-pass
 * kernel cannot settle (it reads each row two to four times).  A reference
 * for checking the fast path; not meant for serving.
 */
aces_status aces_verify_exact(const void *target_logits, aces_dtype dt, const float *draft_probs,
                              const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                              float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                              int32_t *topk_ids, float *topk_probs, float *tail_mass,
                              int32_t *row_status, void *workspace, size_t workspace_bytes,
                              aces_stream_t stream);

/*
 * Sparse payload alone for `rows` independent target rows (the COMPRESS of
 * the downlink distribution, Sec. III-B and Sec. V-C): temperature softmax,
 * nucleus, then the first k ids of the nucleus with their renormalised
 * probabilities and the tail mass.
 *   target_logits [rows, V]; outputs topk_ids / topk_probs [rows, k],
 *   tail_mass [rows], row_status [rows].
 * workspace: at least aces_workspace_bytes(rows, 0, V, k) bytes.
 * Limits: rows >= 1, 2 <= V <= ACES_MAX_V, 1 <= k <= min(V, ACES_MAX_TOPK).
 */
aces_status aces_sparsify(const void *target_logits, aces_dtype dt, int rows, int V, float T,
                          float top_p, int k, int32_t *topk_ids, float *topk_probs,
                          float *tail_mass, int32_t *row_status, void *workspace,
                          size_t workspace_bytes, aces_stream_t stream);

/*
 * Edge-side probabilistic state cache (Sec. III-C; Algorithm 1 TREE_DRAFT):
 * at every draft depth d < K, the F_d most probable alternative tokens of
 * the draft distribution q[b, d, :] other than the main-chain token
 * x~[b, d], ordered by (q desc, id asc), among ids with q > 0, with branch
 * probability q(x) / (1 - q(x~[b, d])).
 *   draft_probs  [B, K, V] float32, draft_tokens [B, K] int32
 *   F_host       [K] host int32 fan-out vector (Sec. IV-B), 0 <= F_d <=
 *                min(V - 1, ACES_MAX_BRANCH)
 * Outputs, S = sum F:  branch_tok [B, S] int32 (-1 padding when fewer ids
 *   qualify, or when 1 - q(x~) <= 0 or x~ is out of range),
 *   branch_prob [B, S] float32 (0 padding).  Depth d occupies columns
 *   [off_d, off_d + F_d) with off_d = F_0 + ... + F_{d-1}.
 */
aces_status aces_cache_build(const float *draft_probs, const int32_t *draft_tokens,
                             const int32_t *F_host, int B, int K, int V, int32_t *branch_tok,
                             float *branch_prob, aces_stream_t stream);

/*
 * The cloud side of one speculation cycle in one call (Sec. III-B/C;
 * Algorithm 1): aces_verify and aces_cache_build of the same batch, with the
 * arguments, outputs, limits and errors of both.  The workspace must hold
 * aces_workspace_bytes(B, K, V, k) bytes.  The two stream different tensors
 * (the logits and the draft distributions), so the cache build runs on a
 * stream of the library's own, forked from `stream` (it waits for the work
 * queued there before the call) and joined back to it (work queued on
 * `stream` after the call waits for both).  Results are bit-identical to the
 * two separate calls.
 *   - Arguments of both calls are checked before anything is launched.
 *   - The first call on each device creates that stream and two events
 *     (kept until the process exits); make it before any stream capture on
 *     the device.  Calls from several host threads are serialised while they
 *     queue their work.
 */
aces_status aces_cloud_step(const void *target_logits, aces_dtype dt, const float *draft_probs,
                            const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                            float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                            int32_t *topk_ids, float *topk_probs, float *tail_mass, int32_t *row_status,
                            const int32_t *F_host, int32_t *branch_tok, float *branch_prob, void *workspace,
                            size_t workspace_bytes, aces_stream_t stream);

/*
 * O(1) state recovery lookup (Sec. III-B, Algorithm 1: w = (pi, x_resampled),
 * w in dom(T)).  For each sequence: slot[b] = off_pi + j when
 * branch_tok[b, off_pi + j] == token[b] (the first such j); -1 on a miss or
 * when token[b] < 0; -2 when accept_len[b] == K (the whole chain was
 * accepted and the main chain continues).
 *   branch_tok [B, sum F], accept_len [B], token [B] -> slot [B] (int32).
 */
aces_status aces_cache_lookup(const int32_t *branch_tok, const int32_t *F_host, int B, int K,
                              const int32_t *accept_len, const int32_t *token, int32_t *slot,
                              aces_stream_t stream);

/*
 * Edge-side resample from the sparse downlink payload (Alg. 1
 * RESAMPLE(P^_target, Q); Sec. III-B): the edge receives pi and the payload
 * of row pi and draws the corrected (pi < K) or bonus (pi = K) token itself,
 * with its own draft row q_pi.
 *
 * The target p is known only on the payload ids I (probs p^_I) plus the
 * mass tau = tail_mass outside them.  For pi < K the tail is spread like
 * the draft, p^(x) = tau * q(x) / q_rest outside I (q_rest = draft mass
 * outside I), and the token is drawn from norm(max(0, p^ - q)) with the
 * rule of aces_verify (smallest id j whose prefix sum over ids 0..j
 * exceeds u[b, K] times the total); if that is all zero, from p^_I.  For
 * pi = K the token is drawn from p^_I.  When the nucleus of row pi has at
 * most k ids, tau = 0 and the token equals aces_verify's out_token.
 *
 *   accept_len  [B]          int32 pi_b from aces_verify
 *   topk_ids    [B, K+1, k]  int32, topk_probs [B, K+1, k] float32,
 *   tail_mass   [B, K+1]     float32, row_status [B, K+1]: aces_verify's
 *                            payload and status (only row pi_b is read)
 *   draft_probs [B, K, V]    float32; row pi_b is read on the payload ids,
 *                            and entirely when its tail_mass > 0
 *   uniforms    [B, K+1]     float32; u[b, K] is the draw
 * Outputs: token [B] int32 (-1 when row pi is NONFINITE, the payload is
 *   empty, or q is NaN/negative where it is read); status [B] int32
 *   (ACES_ROW_NONFINITE / ACES_ROW_BAD_Q for those cases, else 0).
 * Limits: 1 <= B, 1 <= K <= ACES_MAX_K, 2 <= V <= ACES_MAX_V,
 *   1 <= k <= min(V, ACES_MAX_TOPK).
 */
aces_status aces_resample_sparse(const int32_t *accept_len, const int32_t *topk_ids, const float *topk_probs,
                                 const float *tail_mass, const int32_t *row_status, const float *draft_probs,
                                 const float *uniforms, int B, int K, int V, int k, int32_t *token,
                                 int32_t *status, aces_stream_t stream);

/*
 * COMPACT_KV / ROLLBACK_KV of the edge pipeline (Alg. 1; Sec. III-C): after
 * aces_cache_lookup, realign each sequence's KV cache so that the next cycle
 * continues from contiguous rows.
 *   kv [planes, B, H, S, D]  device array of elem_bytes-sized elements
 *                            (planes = layers x {K, V}); 16-byte aligned,
 *                            D * elem_bytes a multiple of 16.  Updated in place.
 * Tree layout of sequence b: its prefix of prefix_len[b] positions, then
 * the main chain (K positions), then the branches in slot order (the slots
 * of aces_cache_lookup), branch_len positions each (the branch token and
 * its drafted continuation).  With pi = accept_len[b] and s = slot[b]:
 *   s >= 0 (hit):   rows [t+K+s*branch_len, +branch_len) move to [t+pi, ...),
 *                   new_len[b] = t + pi + branch_len;
 *   s == -2 (whole chain accepted): nothing moves, new_len[b] = t + K;
 *   s == -1 (miss, ROLLBACK_KV): nothing moves, new_len[b] = t + pi (the
 *                   rejected drafts and every branch are dropped).
 * A sequence whose tree would pass position S, or with t < 0 or pi outside
 * 0..K, gets new_len[b] = -1 and nothing moves.  Rows outside the moved
 * block keep their contents.  prefix_len, accept_len, slot, new_len: [B]
 * int32 device arrays.
 */
aces_status aces_compact_kv(void *kv, int elem_bytes, int planes, int B, int H, int S, int D,
                            const int32_t *prefix_len, const int32_t *accept_len, const int32_t *slot, int K,
                            int branch_len, int32_t *new_len, aces_stream_t stream);

/*
 * Tree attention mask of the packed branch forward (Sec. III-C): every tree
 * token attends to the shared prefix (all of it; not part of this mask),
 * to the main-chain tokens before its branch point (main-path block) and to
 * its own branch up to itself (suffix-diagonal block).  Packed order: the
 * main chain (K tokens), then the branches in slot order (depth 0's F_0
 * branches first, as in aces_cache_build), branch_len tokens each (the
 * alternative token and its drafted continuation); the same layout as
 * aces_compact_kv.
 *   n = aces_tree_tokens(F_host, K, branch_len) = K + sum(F) * branch_len
 *   mask  [n, ceil(n / 32)] uint32 device: bit j of word w of row q is set
 *         when tree token q may attend to tree token 32 w + j
 *   depth [n] int32 device: the token's depth (its position is prefix + depth)
 * aces_tree_tokens returns -1 for invalid sizes (n above 2^20 included).
 */
int aces_tree_tokens(const int32_t *F_host, int K, int branch_len);
aces_status aces_tree_mask(const int32_t *F_host, int K, int branch_len, uint32_t *mask, int32_t *depth,
                           aces_stream_t stream);

/*
 * Network-aware tree budget (Sec. IV-B, Eq. for B*(t)): the largest tree
 * size B whose edge drafting time fits in the cloud turnaround,
 * draft_latency_s[B - 1] <= rtt_s + verify_s, capped by B_max.  The host
 * array draft_latency_s [n] is the measured tree-drafting time of sizes
 * 1..n (non-decreasing; this tabulates the inverse latency function).
 * *B_star = 0 when even one token does not fit.  The branch budget is then
 * B_alloc = B* - gamma (Sec. IV-C).  Host-only; launches nothing.
 */
aces_status aces_tree_budget(const double *draft_latency_s, int n, double rtt_s, double verify_s, int B_max,
                             int *B_star);

/*
 * Geometric-decay branch allocation (Sec. IV-C): with eta = alpha^(1/(beta+1)),
 * F*_k = B_alloc (1 - eta) / (1 - eta^gamma) eta^k (uniform when eta = 1),
 * rounded to integers summing to B_alloc: floor, then one more branch for
 * each of the largest fractional parts, ties to the shallower depth.
 * F_out [gamma] host int32.  0 < alpha <= 1, beta > 0, B_alloc >= 0,
 * 1 <= gamma <= ACES_MAX_K.  Host-only; launches nothing.
 */
aces_status aces_branch_alloc(int B_alloc, int gamma, double alpha, double beta, int32_t *F_out);

#ifdef ACES_CHECKED
/*
 * Checked build only (compiled with -DACES_CHECKED; a test aid, not part of
 * the product library): every kernel checks its data-dependent shared- and
 * global-memory indices and records the first index out of range instead of
 * making the access.  This returns that record since the last call:
 * out[0] = site (source file number * 10000 + line; 0 when none), out[1] =
 * the index, out[2] = its bound.  It waits for the device and clears the
 * record.  The paper has no counterpart.
 */
aces_status aces_checked_violation(unsigned long long out[3]);
#endif

/* Static English text for a status code. */
const char *aces_status_string(aces_status s);

#ifdef __cplusplus
}
#endif
#endif /* ACESPEC_H */
