/*
 * osd.h -- C ABI of the GB300 (sm_103a) hot path of Online Speculative
 * Decoding (Liu et al., "Online Speculative Decoding", ICML 2024).
 *
 * The operations of every serving step of the paper's Algorithm 1:
 *
 *   osd_verify   speculative-sampling verification of k draft tokens against
 *                k+1 target distributions (Section 3 and Appendix A.1; the
 *                "determine number of accepted tokens and sample one more
 *                token" step of Algorithm 1), which also emits the mismatch
 *                mask that feeds the temporary buffer R of Algorithm 1.
 *   osd_distill  the per-position distillation loss D(p || q_theta) of Eq. 2
 *                with D one of the distances of Eq. 3 (forward KL, reverse
 *                KL, JSD[beta]), total variation distance or the label
 *                cross-entropy, and its gradient with respect to the draft
 *                logits (the analytic update step of Algorithm 1).
 *   osd_distill_accepted  the same on the rows osd_verify rejected, selected
 *                and compacted on the device from its accepted counts.
 *   osd_mixed_sample  one token per position from beta p + (1 - beta) q
 *                (Section 4.1, mixed sampling).
 *   osd_verify_tree  verification of several candidates per position laid
 *                out as a token tree (the paper's Medusa combination).
 *
 * Conventions shared by every entry point:
 *   - All array arguments are DEVICE pointers to caller-owned memory on the
 *     current CUDA device; the library allocates nothing itself.  Apart from
 *     the fixed array behind osd_verify_noalloc it keeps no device memory.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued asynchronously on it; outputs are valid once
 *     the stream reaches that point.  Argument errors are detected on the
 *     host and returned before anything is enqueued.
 *   - No C++ exception crosses this boundary.  Functions are thread-safe as
 *     long as concurrent calls do not share output or workspace buffers.
 *   - Logits are row-major with the vocabulary innermost and contiguous, in
 *     fp32 or bf16 (OSD_F32 / OSD_BF16).  Any alignment to the element size
 *     is accepted; rows that start on 16-byte boundaries take the fast
 *     vectorised path.
 *   - Accumulation is fp32 inside a thread.  Where a sum decides a sample
 *     position it is carried exactly, in 64-bit fixed point with 60
 *     fraction bits (verification, tree verification), or in fp64 (mixed
 *     sampling); exponentials use the hardware ex2 unit.
 */
#ifndef OSD_H_
#define OSD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum osd_status {
    OSD_OK = 0,
    OSD_ERR_INVALID_ARG = 1,  /* a null pointer, size, alignment or value out of range */
    OSD_ERR_UNSUPPORTED = 2,  /* valid arguments beyond the library's limits (e.g. V) */
    OSD_ERR_CUDA = 3,         /* a CUDA launch or API call failed                        */
    OSD_ERR_TIMEOUT = 4       /* a bounded device-side wait gave up (see osd_distill)    */
} osd_status;

typedef enum osd_dtype { OSD_F32 = 0, OSD_BF16 = 1 } osd_dtype;

/* Distances of Eq. 3 (Section 4.1), total variation distance, and the
 * label fine-tuning baseline of Table 1 (FT). */
typedef enum osd_loss {
    OSD_FKL = 0,  /* KL(p || q)                                               */
    OSD_RKL = 1,  /* KL(q || p)                                               */
    OSD_JSD = 2,  /* beta KL(p || m) + (1 - beta) KL(q || m), m = beta p + (1-beta) q */
    OSD_TVD = 3,  /* 1/2 sum |p - q|                                          */
    OSD_CE = 4    /* -log q(y*), y* = argmax of the target logits (lowest index on ties) */
} osd_loss;

/* Largest vocabulary osd_verify accepts. */
#define OSD_VERIFY_MAX_V (1 << 21)
/* Largest number of draft tokens osd_verify accepts. */
#define OSD_VERIFY_MAX_K 64

/* Human-readable name of a status code (static string, never NULL). */
const char *osd_status_string(osd_status status);

/* ABI version of this library: (major << 16) | minor.  2.0 added the
 * temperature argument of osd_distill and the OSD_CE loss; 2.1 added
 * osd_distill_accepted; 2.2 added osd_mixed_sample; 2.3 added
 * osd_verify_tree; 2.4 added osd_check_bounded_wait; 2.5 raised
 * osd_mixed_sample's vocabulary limit to OSD_VERIFY_MAX_V. */
int osd_abi_version(void);

/*
 * Bytes of device workspace osd_verify needs for B sequences of k draft
 * tokens over a vocabulary of V (per-row softmax statistics).  Writes the
 * size to *bytes.  Returns OSD_ERR_INVALID_ARG for a null `bytes` or sizes
 * out of range, OSD_ERR_UNSUPPORTED beyond OSD_VERIFY_MAX_K/_MAX_V.
 */
osd_status osd_verify_workspace_size(int B, int k, int V, size_t *bytes);

/*
 * Speculative-sampling verification (Section 3, Appendix A.1, Algorithm 1).
 *
 * For each sequence b, with q_i = softmax(draft_logits[b,i,:] / T) and
 * p_i = softmax(target_logits[b,i,:] / T):
 *   - tests i = 0..k-1 in order and accepts draft_tokens[b,i] iff
 *     uniforms[b,i] < p_i(y_i) / q_i(y_i) (strict; q(y) = 0 < p(y) accepts),
 *     stopping at the first rejection; a = number accepted;
 *   - samples one more token by inverse CDF with uniforms[b,k]: from
 *     norm(max(0, p_a - q_a)) if a < k, from p_k if a = k.  The CDF runs in
 *     ascending vocabulary order and picks min{ j : C_j > u W }.
 *   - T == 0 is greedy: accept while y_i == argmax p_i (lowest index on
 *     ties), then emit argmax p_a; uniforms and draft logits are not read.
 *
 * draft_logits   [B, k, V]    dtype, contiguous (not read when T == 0)
 * target_logits  [B, k+1, V]  dtype, contiguous
 * draft_tokens   [B, k]       int32
 * uniforms       [B, k+1]     fp32 in [0, 1) (not read when T == 0)
 * temperature    >= 0 and finite, else OSD_ERR_INVALID_ARG
 * accepted       [B]          out: a in 0..k; -1 if any draft token of the
 *                             sequence lies outside [0, V), or (small batches
 *                             at T > 0, whose rows are staged by bulk copy) if
 *                             the GPU did not deliver the sequence's rows within
 *                             a one-second bound
 * out_tokens     [B, k+1]     out: y_0..y_{a-1}, the sampled token at a, then -1
 * mismatch_mask  [B, k]       out: 1 at i == a when a < k, else 0 (the first
 *                             rejected position, the rows Algorithm 1 keeps
 *                             for distillation)
 * diag_margin    [B, k]       out, nullable: |u_i - r_i| for decided
 *                             positions, NaN after the decision and when T == 0
 * diag_cdf_gap   [B]          out, nullable: distance of u W to the nearest
 *                             edge of the chosen CDF step, divided by W (NaN
 *                             when T == 0)
 * workspace      device scratch of at least osd_verify_workspace_size()
 *                bytes, 16-byte aligned; contents need no initialisation and
 *                are garbage afterwards.  Calls that overlap on the GPU
 *                must not share it.
 * Limits: 1 <= k <= OSD_VERIFY_MAX_K, 1 <= V <= OSD_VERIFY_MAX_V, B >= 0.
 */
osd_status osd_verify(const void *draft_logits, const void *target_logits,
                      osd_dtype dtype, int B, int k, int V,
                      const int32_t *draft_tokens, const float *uniforms,
                      float temperature,
                      int32_t *accepted, int32_t *out_tokens, uint8_t *mismatch_mask,
                      float *diag_margin, float *diag_cdf_gap,
                      void *workspace, size_t workspace_bytes, void *stream);

/*
 * osd_verify without a caller-supplied workspace (no counterpart in the paper).
 *
 * For callers that must not allocate device memory while serving: engines
 * that reserve all free device memory for their KV cache at start-up, plugins
 * running inside such an engine without an allocator of their own, and
 * latency-critical loops where cudaMalloc, which may synchronise the device,
 * would stall the other streams.  Arguments and results are those of
 * osd_verify; the workspace is a 4 MiB array inside the library (one per GPU
 * that loads it, kept until the process exits).  This function allocates
 * nothing: no cudaMalloc, cudaFree or allocating library call.
 *   - The first call on a device looks up that device's copy of the array
 *     (cudaGetSymbolAddress, with the device current); make that first call
 *     before any stream capture.  The address is kept per device together with
 *     the ID of the context it was found in, and looked up again when the
 *     current context changes (after cudaDeviceReset, for instance); make the
 *     first call after such a change before any stream capture too.
 *   - Returns OSD_ERR_UNSUPPORTED when osd_verify_workspace_size(B, k, V)
 *     exceeds 4 MiB, or when the current device ordinal is 64 or more.  That
 *     size is B * (2k+1) * ceil(V / L) * 16 bytes, rounded up to 256, with
 *     slices of L = 8192 entries below 512 rows B * (2k+1), 16384 below
 *     2048 rows and 32768 from 2048 rows on (B = 256, k = 8, V = 128256 needs
 *     0.28 MB).
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents (every entry is rewritten before it is read, so nothing needs
 *     clearing).  Calls that overlap on the GPU, on different streams or from
 *     different threads, race on it: serialise them.
 */
osd_status osd_verify_noalloc(const void *draft_logits, const void *target_logits,
                              osd_dtype dtype, int B, int k, int V,
                              const int32_t *draft_tokens, const float *uniforms,
                              float temperature,
                              int32_t *accepted, int32_t *out_tokens, uint8_t *mismatch_mask,
                              float *diag_margin, float *diag_cdf_gap, void *stream);

/*
 * Per-position distillation loss and gradient (Eq. 2-3, Section 4.1) over
 * rows laid out as [G, P, V] with element strides (the [N, V] case is G = N,
 * P = 1, d_stride_g = t_stride_g = V).  q = softmax(draft row / tau),
 * p = softmax(target row / tau), tau = `temperature` (Section 4.1's tunable
 * softmax temperature; 1 is the plain softmax).
 *
 * draft_logits, target_logits  row (g, p) starts at base + g*stride_g +
 *                p*stride_p elements; the V entries of a row are contiguous.
 * mask           [G, P] uint8, nullable (NULL = every row active).
 * kind, beta     the distance; beta in [0, 1] is used by OSD_JSD only.
 * temperature    tau > 0 and finite, else OSD_ERR_INVALID_ARG.
 * loss           [G, P] fp32 out: the per-position loss (the 1/n_B batch
 *                mean of Eq. 2 is left to the caller); 0 for inactive rows.
 * dlogits        [G, P, V] fp32 contiguous out: d loss / d draft logits
 *                (the raw logits, so including the factor 1/tau), unscaled
 *                by any batch size; rows of inactive positions are NOT written.
 * status         nullable device int32: set to 0 by this call, then to
 *                OSD_ERR_TIMEOUT if a bounded wait for a bulk copy gave up
 *                (that row's loss is then NaN and its gradient not written).
 * Limits: V <= 393216 (bf16) or 196608 (fp32), else OSD_ERR_UNSUPPORTED.
 * Rows whose logits are all -inf, or that hold +inf or NaN, are outside the
 * domain: their results are unspecified.
 */
osd_status osd_distill(const void *draft_logits, const void *target_logits,
                       osd_dtype dtype, int G, int P, int V,
                       int64_t d_stride_g, int64_t d_stride_p,
                       int64_t t_stride_g, int64_t t_stride_p,
                       const uint8_t *mask, osd_loss kind, float beta, float temperature,
                       float *loss, float *dlogits, int32_t *status, void *stream);

/*
 * Distillation of the rows that verification rejected, chosen on the device
 * (Algorithm 1: the first rejected position of each step and the target's
 * distribution there go into the buffer R; Eq. 2-3 give the loss on them).
 *
 * Sequence b contributes the row at position a = accepted[b] when 0 <= a < k,
 * the first draft token osd_verify rejected (where its mismatch_mask is 1):
 * draft row (b, a) of draft_logits [B, k, V] and target row (b, a) of
 * target_logits [B, k+1, V], both contiguous, the layouts osd_verify reads.
 * Sequences with a == k (all accepted) or a == -1 (bad tokens) contribute
 * nothing.  Loss, gradient and temperature are those of osd_distill.
 *
 * Results go to a stable partition of the sequences: the n active ones
 * first, in increasing b, then the inactive ones, in increasing b.
 *
 * accepted      [B] int32 device, as osd_verify writes it; read on the device,
 *               so the call can follow osd_verify on the same stream with no
 *               host synchronisation (and be captured in the same graph).
 * loss          [B] fp32 out: slot r < n holds the loss of sequence
 *               seq_of_row[r]; slots r >= n are set to 0.
 * dlogits       [B, V] fp32 out: rows r < n hold the gradients; rows r >= n
 *               are not written.
 * seq_of_row    [B] int32 out, nullable: the sequence b behind slot r.
 * count         device int32 out, nullable: n.
 * status        as in osd_distill.
 * Returns OSD_ERR_INVALID_ARG for k < 1, B < 0, a null `accepted` with
 * B > 0, and the osd_distill argument errors.  B = 0 only sets *count = 0.
 */
osd_status osd_distill_accepted(const void *draft_logits, const void *target_logits,
                                osd_dtype dtype, int B, int k, int V, const int32_t *accepted,
                                osd_loss kind, float beta, float temperature,
                                float *loss, float *dlogits, int32_t *seq_of_row, int32_t *count,
                                int32_t *status, void *stream);

/* Largest token tree osd_verify_tree accepts (nodes, root included). */
#define OSD_TREE_MAX_NODES 64

/*
 * Bytes of device workspace osd_verify_tree needs for B trees of n_nodes
 * nodes over a vocabulary of V (per-row softmax statistics).  Errors as
 * osd_verify_workspace_size; OSD_ERR_UNSUPPORTED beyond OSD_TREE_MAX_NODES.
 */
osd_status osd_verify_tree_workspace_size(int B, int n_nodes, int V, size_t *bytes);

/*
 * Multi-candidate verification over a token tree: the tree-style speculative
 * decoding the paper combines OSD with (its Medusa study), where several
 * candidates are proposed per position.  Node i > 0 carries one candidate
 * token; its children are the alternatives for the next position.
 *
 * At the current node (the root first), with q = softmax(draft row / T) and
 * p = softmax(target row / T) of that node, the children are tried in
 * increasing index order: child y passes iff u < r(y) / q(y), with r the
 * current residual, starting from r = p; a rejection replaces r by
 * norm(max(0, r - q)) (multi-candidate speculative sampling, which keeps the
 * output distributed as p); a pass moves the walk to that child.  When every
 * child is rejected, or the node has none, one more token is drawn from r by
 * the inverse CDF of osd_verify's extra token (u = uniforms[b, 0]).
 * T == 0 is greedy: the first child equal to argmax p (lowest index) passes;
 * otherwise the extra token is argmax p.
 *
 * draft_logits   [B, n_nodes, V] dtype, contiguous: row i is the draft
 *                distribution the children of node i were proposed from
 *                (not read at T == 0; leaves' rows are not read)
 * target_logits  [B, n_nodes, V] dtype, contiguous: row i is the target
 *                distribution after the path to node i
 * parent         [n_nodes] int32 HOST array, the static tree shared by the
 *                batch: parent[0] = -1, 0 <= parent[i] < i
 * tokens         [B, n_nodes] int32: candidate of node i (entry 0 unused)
 * uniforms       [B, n_nodes] fp32 in [0, 1): u[b, i] tests node i, u[b, 0]
 *                drives the extra draw (not read at T == 0)
 * accepted       [B] out: accepted tokens (the depth reached), -1 if a token
 *                lies outside [0, V)
 * path           [B, n_nodes] out: the accepted nodes, root excluded, then -1
 * out_tokens     [B, n_nodes] out: the accepted tokens, the extra token, then -1
 * last_node      [B] out: the node where the walk stopped (its rows are the
 *                ones a distillation step keeps when it has children)
 * diag_margin    [B, n_nodes] out, nullable: |u - r(y)/q(y)| of every test made
 *                (at node i's entry), NaN elsewhere and when T == 0
 * diag_cdf_gap   [B] out, nullable: as in osd_verify
 * workspace      >= osd_verify_tree_workspace_size() bytes, 16-byte aligned
 * Limits: 1 <= n_nodes <= OSD_TREE_MAX_NODES, 1 <= V <= OSD_VERIFY_MAX_V.
 * Returns OSD_ERR_INVALID_ARG for a malformed tree or the argument errors of
 * osd_verify.
 */
osd_status osd_verify_tree(const void *draft_logits, const void *target_logits, osd_dtype dtype,
                           int B, int n_nodes, int V, const int32_t *parent,
                           const int32_t *tokens, const float *uniforms, float temperature,
                           int32_t *accepted, int32_t *path, int32_t *out_tokens,
                           int32_t *last_node, float *diag_margin, float *diag_cdf_gap,
                           void *workspace, size_t workspace_bytes, void *stream);

/*
 * Mixed-token sampling (Section 4.1): one token per position from the mixture
 * beta p + (1 - beta) q, p = softmax(target row / tau), q = softmax(draft row
 * / tau), the sampling the paper borrows to pick the tokens y the distillation
 * loss is evaluated on.  The draw is one inverse-CDF step over the mixture
 * weights w_j = beta p_j + (1 - beta) q_j in ascending vocabulary order:
 * j* = min{ j : C_j > u W }, W = sum_j w_j, with the largest j with w_j > 0
 * if rounding leaves none (the convention of osd_verify's extra token).
 *
 * draft_logits, target_logits  row n starts at base + n * stride elements
 *                (stride 0 repeats one row); the V entries of a row are
 *                contiguous; dtype as in osd_distill.
 * uniforms       [N] fp32 in [0, 1), one per row.
 * beta           in [0, 1]: 1 samples the target, 0 the draft.
 * temperature    tau > 0 and finite.
 * tokens         [N] int32 out.
 * cdf_gap        [N] fp32 out, nullable: distance of u W to the nearest edge of
 *                the chosen CDF step, divided by W (<= 0 when rounding left
 *                no step above u W).
 * status         nullable device int32, set to 0 (OSD_OK): the kernel
 *                streams both rows with plain loads and has no wait that can
 *                run out; kept so that every staging entry point reports the
 *                same way.
 * Limits: 1 <= V <= OSD_VERIFY_MAX_V, N >= 0.
 * Argument errors: OSD_ERR_INVALID_ARG (null pointers with N > 0, negative
 * sizes or strides, beta outside [0, 1], bad temperature, misalignment).
 */
osd_status osd_mixed_sample(const void *draft_logits, const void *target_logits, osd_dtype dtype,
                            int N, int V, int64_t d_stride, int64_t t_stride,
                            const float *uniforms, float beta, float temperature,
                            int32_t *tokens, float *cdf_gap, int32_t *status, void *stream);

/*
 * Health check of the failure path every staging kernel shares: a bounded
 * wait on an mbarrier (the one that guards the bulk copies of osd_distill
 * and osd_distill_accepted) is run against a barrier that
 * nothing completes.  When limit_us microseconds have passed it writes
 * OSD_ERR_TIMEOUT to the device int32 *status (OSD_OK would mean the wait
 * completed, which cannot happen) and the nanoseconds it waited to the device
 * uint64 *waited_ns (nullable).  The kernel then exits
 * normally, so the context stays usable; no logits are read.
 * Returns OSD_ERR_INVALID_ARG for a null `status`, misalignment, or limit_us
 * outside [1, 10^7].
 */
osd_status osd_check_bounded_wait(uint32_t limit_us, int32_t *status, uint64_t *waited_ns, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* OSD_H_ */
