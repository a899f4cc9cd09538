/*
 * nld.h -- C ABI of libnld: block attention over a paged bf16 KV cache and
 * the token decisions of tri-mode decoding, on one sm_103a GPU.
 *
 * Method (Nemotron-Labs-Diffusion, tri-mode decoding):
 *   - Sec. 2.2 (attention pattern): noisy block tokens attend bidirectionally
 *     inside their block and to the whole clean prefix; the clean stream is
 *     strictly causal.
 *   - Sec. 3, Mode 2 (block-wise diffusion): a block of mask tokens is
 *     denoised in parallel against the cached prefix; confident positions are
 *     committed step by step.
 *   - Sec. 3, Mode 3 (linear self-speculation): a diffusion draft pass over
 *     k mask positions, then a causal AR verify pass over the drafts, both
 *     reusing the prefix KV cache; the longest matching draft prefix is
 *     accepted.
 *
 * Conventions shared by every entry point:
 *   - All tensor pointers are DEVICE pointers, row-major and contiguous, owned
 *     by the caller. The library never allocates, frees or synchronises; each
 *     call enqueues its kernels on `stream` and returns.
 *   - Arguments that can be checked on the host are checked before anything
 *     is launched; a failed check returns NLD_ERR_INVALID_ARG,
 *     NLD_ERR_UNSUPPORTED or NLD_ERR_WORKSPACE and launches nothing. A failed
 *     launch returns NLD_ERR_CUDA.
 *   - Values that live on the device (prefix lengths, page ids) are not read
 *     by the host. Kernels clamp out-of-range values into range (so no access
 *     leaves the caller's buffers) and record the event in a device error
 *     word, readable with nld_device_error().
 *   - Pointers to bf16 and fp32 tensor data and the workspace must be 16-byte
 *     aligned; int32 arrays must be 4-byte aligned.
 */
#ifndef NLD_H
#define NLD_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    NLD_OK = 0,
    NLD_ERR_INVALID_ARG = 1, /* null/misaligned pointer, bad size or shape   */
    NLD_ERR_UNSUPPORTED = 2, /* valid but not built: head_dim, block, group  */
    NLD_ERR_WORKSPACE = 3,   /* workspace missing or smaller than required   */
    NLD_ERR_CUDA = 4         /* a CUDA runtime/driver call or launch failed  */
} nld_status_t;

/* Mask inside the block (Sec. 2.2, Sec. 3). The prefix is visible in both. */
typedef enum {
    NLD_MODE_DIFFUSION = 0, /* diffusion draft: bidirectional inside the block */
    NLD_MODE_VERIFY = 1     /* AR verify: causal inside the block, self included */
} nld_mode_t;

/* Bits of the device error word (nld_device_error). */
#define NLD_DEVERR_PREFIX_RANGE 0x1u /* a prefix length outside [0, max_pages*P - bl] was clamped */
#define NLD_DEVERR_PAGE_RANGE 0x2u   /* a page id outside [0, num_pages) was clamped              */
#define NLD_DEVERR_WAIT_TIMEOUT 0x4u /* a pipeline wait passed its time limit; output is invalid  */

/*
 * Shape of one block-attention call.
 *   batch             B, number of sequences (>= 1)
 *   num_q_heads       Hq; query head h reads KV head h / (Hq / Hkv)
 *   num_kv_heads      Hkv; Hq % Hkv == 0
 *   head_dim          D, 64 or 128
 *   page_size         P, tokens per page: a power of two in [16, 256]
 *   num_pages         pages in the pool (first dim of k_pages / v_pages)
 *   max_pages_per_seq second dim of page_table
 *   num_splits        pieces the KV range of each (sequence, KV head) is cut
 *                     into; 0 = choose from the SM count. Values above 128
 *                     are rejected.
 *   softmax_scale     score scale; 0 = 1/sqrt(head_dim)
 *   flags             0, or an OR of NLD_ATTN_PREFIX_READY and
 *                     NLD_ATTN_NO_CLUSTER
 */
typedef struct {
    int batch;
    int num_q_heads;
    int num_kv_heads;
    int head_dim;
    int page_size;
    int num_pages;
    int max_pages_per_seq;
    int num_splits;
    float softmax_scale;
    unsigned int flags;
} nld_attn_params_t;

/*
 * NLD_ATTN_PREFIX_READY: the caller guarantees that page_table, prefix_lens
 * and the cached prefix K/V (slots below L_b) are not written by kernels
 * that were enqueued earlier on the same stream and may still be running.
 * The attention kernels are launched with programmatic stream serialization;
 * with this flag they start streaming the prefix K/V before waiting for
 * those earlier kernels, overlapping the load ramp with them. The block's
 * own K/V slots, q_block and the outputs are still accessed only after the
 * wait. Without the flag nothing is read before the wait.
 */
#define NLD_ATTN_PREFIX_READY 0x1u

/*
 * NLD_ATTN_NO_CLUSTER: never run the splits of a (sequence, KV head) as a
 * thread-block cluster; every split writes its own partial. With explicit
 * split counts this makes num_splits the number of partials.
 */
#define NLD_ATTN_NO_CLUSTER 0x4u

/*
 * Number of split partials per output row that nld_block_attn leaves in the
 * workspace and merges with the split combine (1: the call writes the final
 * output directly and needs no workspace), or -1 if the parameters are
 * invalid. The KV range of each (sequence, KV head) is cut into
 * params->num_splits pieces (0: chosen from the current device's SM count);
 * pieces that run as one thread-block cluster merge on chip into a single
 * partial, so this count can be smaller than the number of pieces.
 */
int nld_block_attn_num_splits(const nld_attn_params_t *params, int block_len);

/*
 * Kernels one nld_block_attn call with these parameters launches on the
 * current device: 1 (unsplit, or split and merged in a thread-block
 * cluster) or 2 (attention, then the split combine), or -1 if the
 * parameters are invalid. Host-side query; launches nothing.
 */
int nld_block_attn_kernels(const nld_attn_params_t *params, int block_len);

/*
 * Host-only view of the split plan for a device with sm_count SMs: plan[0]
 * splits per (sequence, KV head), plan[1] tokens per split, plan[2] cluster
 * size, plan[3] partials per output row. An explicit params->num_splits
 * divisible by 8, 4 or 2 runs as clusters of that size (plan[2] = 8, 4 or
 * 2), exactly as nld_block_attn launches it. An automatic plan
 * (num_splits = 0) is given as if no cluster were resident: on a device
 * where the plan's 2..8 pieces per (sequence, KV head) fit as resident
 * clusters, the launched plan instead uses one cluster of 2, 4 or 8 per
 * (sequence, KV head) and one partial, and nld_block_attn_num_splits
 * reports that. Returns 0, or -1 for invalid parameters. Touches no device;
 * for tests and capacity planning.
 */
int nld_block_attn_plan(const nld_attn_params_t *params, int block_len, int sm_count, int32_t plan[4]);

/*
 * Workspace bytes nld_block_attn needs (0 when it runs unsplit). The
 * workspace holds the split partials: O_part bf16 [S, B, Hq, bl, D] (each
 * row the partial output normalised by its own sum, so its values lie within
 * the range of V) then LSE_part fp32 [S, B, Hq, bl] at the next 256-byte
 * boundary. Its contents need no initialisation. Calls whose kernels may overlap on the GPU need
 * separate workspaces.
 * Returns (size_t)-1 if the parameters are invalid.
 */
size_t nld_block_attn_workspace_size(const nld_attn_params_t *params, int block_len);

/*
 * Block attention of a block of `block_len` tokens per sequence against the
 * paged KV cache (Sec. 2.2 mask; Sec. 3 Modes 2 and 3).
 *
 * For sequence b with prefix length L_b = prefix_lens[b], query head h,
 * block row i (0 <= i < block_len), key t is visible when t < L_b, or
 * t = L_b + j with j < block_len and (mode == DIFFUSION or j <= i). Key t is
 * read from physical page page_table[b][t / P], slot t % P, KV head
 * h / (Hq / Hkv). Then, with s_t = softmax_scale * <q, k_t>:
 *   out[b, i, h, :] = sum_t softmax(s)_t v_t,   lse[b, h, i] = ln sum_t exp(s_t).
 *
 *   q_block     bf16 [B, block_len, Hq, D]
 *   k_pages     bf16 [num_pages, Hkv, P, D]
 *   v_pages     bf16 [num_pages, Hkv, P, D]
 *   page_table  int32 [B, max_pages_per_seq]; entries for logical pages
 *               0 .. ceil((L_b + block_len) / P) - 1 must be valid page ids
 *   prefix_lens int32 [B], L_b >= 0 and L_b + block_len <= max_pages_per_seq * P
 *   block_len   1 .. 32, with (Hq / Hkv) * block_len <= 256
 *   mode        NLD_MODE_DIFFUSION or NLD_MODE_VERIFY
 *   out         bf16 [B, block_len, Hq, D]
 *   lse         fp32 [B, Hq, block_len] (natural log), or NULL
 *   workspace   device scratch of nld_block_attn_workspace_size() bytes
 *               (may be NULL when that size is 0)
 *
 * The block's own K/V must already be in the paged slots L_b .. L_b+bl-1.
 * When the plan splits the KV range into S > 1 partials (the workspace
 * holds them), the attention kernel is followed by the split combine (the
 * kernel nld_split_kv_combine runs).
 */
nld_status_t nld_block_attn(const nld_attn_params_t *params, const void *q_block,
                            const void *k_pages, const void *v_pages,
                            const int32_t *page_table, const int32_t *prefix_lens,
                            int block_len, nld_mode_t mode, void *out, float *lse,
                            void *workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * The attention kernel of nld_block_attn alone, same arguments. When the
 * split plan has one split it writes out and lse exactly as nld_block_attn
 * does. With S > 1 splits it writes only the partials into the workspace
 * (bf16 O_part at offset 0, fp32 LSE_part at the next 256-byte boundary
 * after S*B*Hq*bl*D*2 bytes) and leaves out/lse untouched; the caller then
 * merges them with nld_split_kv_combine (S = nld_block_attn_num_splits()).
 * This lets a caller time, overlap or reorder the two kernels.
 */
nld_status_t nld_block_attn_partials(const nld_attn_params_t *params, const void *q_block,
                                     const void *k_pages, const void *v_pages,
                                     const int32_t *page_table, const int32_t *prefix_lens,
                                     int block_len, nld_mode_t mode, void *out, float *lse,
                                     void *workspace, size_t workspace_bytes,
                                     cudaStream_t stream);

/*
 * nld_block_attn with the block part of the mask from a table, for
 * structured masks such as quadratic self-speculation's (Sec. 3 variant):
 * key t is visible to block row i when t < L_b (the prefix, as always), or
 * t = L_b + j with bit j of block_mask[i] set. A row that sees no key (no
 * prefix and an empty table entry) gets out = 0 and lse = -inf.
 *
 *   block_mask  uint32 [block_len] on the device (block_len <= 32)
 *   other arguments as for nld_block_attn
 */
nld_status_t nld_block_attn_masked(const nld_attn_params_t *params, const void *q_block,
                                   const void *k_pages, const void *v_pages,
                                   const int32_t *page_table, const int32_t *prefix_lens,
                                   int block_len, const uint32_t *block_mask, void *out, float *lse,
                                   void *workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * The block layout and table mask of quadratic self-speculation (Sec. 3
 * variant; appendix Eq. quad_input), host side: after the prefix come the AR
 * token x_{n+1} (slot 0) and k groups, each a speculative token followed by
 * k fresh mask tokens (slots 1+g(k+1) .. 1+g(k+1)+k): 1 + k + k^2 slots.
 * The speculative chain (the AR token and the speculative tokens) is causal
 * and sees no mask token (its predictions verify the previous drafts); the
 * masks of a group see the chain up to their speculative token and their
 * own group's masks (they draft the next block in case verification accepts
 * up to that token). Writes masks[0 .. 1+k+k^2-1]; returns 1+k+k^2, or -1
 * when k < 1 or the block would exceed 32 slots (k > 5).
 */
int nld_quadss_block_mask(int k, uint32_t *masks);

/*
 * nld_block_attn for callers that cannot allocate device memory (the paper
 * has no counterpart: this is a deployment convenience of this library).
 * Plugins running inside another runtime's enqueue step, code bound to a
 * fixed memory budget, or callers holding only raw input/output pointers may
 * have no way to provide a workspace. This entry point takes the same
 * arguments as nld_block_attn minus the workspace and keeps the split
 * partials in a 16 MiB array compiled into the library (held by every GPU
 * that loads it until exit). It allocates and frees nothing.
 *   - Returns NLD_ERR_WORKSPACE, launching nothing, when the split plan
 *     needs more than 16 MiB of partials (nld_block_attn_workspace_size()
 *     > 16 MiB); ask for fewer splits (params->num_splits) or use
 *     nld_block_attn with your own workspace.
 *   - The first call made with a device current looks up the array's device
 *     address on that device; make it before any stream capture.
 *   - All calls on a device share the array. Calls whose kernels may overlap
 *     on the GPU (unordered streams) race on it; order them on one stream.
 */
nld_status_t nld_block_attn_static_scratch(const nld_attn_params_t *params, const void *q_block,
                                           const void *k_pages, const void *v_pages,
                                           const int32_t *page_table, const int32_t *prefix_lens,
                                           int block_len, nld_mode_t mode, void *out, float *lse,
                                           cudaStream_t stream);

/*
 * Merge split-KV partials (each a softmax-normalised partial output and its
 * log-sum-exp over one key range) into the full result:
 *   m = max_s lse_s, c_s = exp(lse_s - m),
 *   out = sum_s c_s o_s / sum_s c_s,  lse = m + ln sum_s c_s.
 * A partial with lse_s = -inf carries no keys: it gets weight 0 and its
 * o_s is not read. A row whose partials are all -inf gets out = 0 and
 * lse = -inf. Weights, sums and the merged row are computed in fp32 from the
 * bf16 partials; out is rounded to bf16 once.
 *
 *   o_part   bf16 [S, B, Hq, bl, D] (16-byte aligned)
 *   lse_part fp32 [S, B, Hq, bl]
 *   out      bf16 [B, bl, Hq, D]
 *   lse      fp32 [B, Hq, bl], or NULL
 *   1 <= num_splits <= 128, head_dim 64 or 128, 1 <= block_len <= 32
 */
nld_status_t nld_split_kv_combine(const void *o_part, const float *lse_part, int num_splits,
                                  int batch, int num_q_heads, int block_len, int head_dim,
                                  void *out, float *lse, cudaStream_t stream);

/*
 * Longest-prefix acceptance of linear self-speculation (Sec. 3, Mode 3):
 * accepted_len[b] = the first j with draft_ids[b][j] != verify_ids[b][j],
 * or n when all n positions agree. The caller commits draft[0:acc] plus the
 * verifier's token at the first mismatch, so a step yields 1..n+1 tokens.
 *
 *   draft_ids, verify_ids int32 [B, n];  accepted_len int32 [B];  1 <= n <= 32
 */
nld_status_t nld_accept(const int32_t *draft_ids, const int32_t *verify_ids, int batch, int n,
                        int32_t *accepted_len, cudaStream_t stream);

/*
 * Confidence-ranked unmasking of the diffusion mode (Sec. 3, Mode 2; the
 * serial denoising of Sec. 4 commits the single most confident position):
 * the k eligible positions with the largest fp32 confidence, written in rank
 * order (confidence descending; equal values, +0 and -0 included, by
 * position ascending). -inf and NaN mark ineligible (already committed)
 * positions. When fewer than k are eligible the tail of `positions` is -1.
 *
 *   confidences fp32 [B, n];  positions int32 [B, k];
 *   num_selected int32 [B] or NULL;  1 <= k <= n <= 32
 */
nld_status_t nld_unmask(const float *confidences, int batch, int n, int k, int32_t *positions,
                        int32_t *num_selected, cudaStream_t stream);

/*
 * Threshold unmasking with a top-1 fallback (Sec. 2, confidence-based
 * sampling: a denoising step commits every masked position whose
 * confidence exceeds the threshold). Commits every eligible position whose
 * confidence is strictly greater than `threshold` (fp32 comparison); if none
 * is, commits the single highest-confidence eligible position (the lower
 * position on ties; +0 and -0 tie), so that a step commits at least one
 * position while any remains masked. -inf and NaN mark positions already
 * committed (not eligible).
 *
 *   confidences  fp32 [B, n], 1 <= n <= 32
 *   positions    int32 [B, n]: the committed positions in ascending order,
 *                then -1
 *   num_selected int32 [B] (may be NULL): committed count (0 only when no
 *                position is eligible)
 */
nld_status_t nld_unmask_threshold(const float *confidences, int batch, int n, float threshold,
                                  int32_t *positions, int32_t *num_selected, cudaStream_t stream);

/*
 * Greedy parallel acceptance against a serial target (Sec. 5, diffusion SOL
 * construction): one iteration commits every masked position j whose argmax
 * prediction equals the target, pred_ids[b][j] == target_ids[b][j]; if none
 * does, the single highest-confidence masked position (lower position on
 * ties). A position is masked when its confidence is neither -inf nor NaN;
 * the confidences also rank the fallback.
 *
 *   pred_ids, target_ids int32 [B, n]; confidences fp32 [B, n], 1 <= n <= 32
 *   positions, num_selected as for nld_unmask_threshold
 */
nld_status_t nld_greedy_accept(const int32_t *pred_ids, const int32_t *target_ids,
                               const float *confidences, int batch, int n, int32_t *positions,
                               int32_t *num_selected, cudaStream_t stream);

/*
 * Logits -> (argmax id, confidence) per position, the inputs of the token
 * decisions above (the confidence of Sec. 2 confidence-based sampling; Sec. 5
 * serial denoising commits the position with the highest peak probability):
 *   m = max_v logits[r][v],  ids[r] = the lowest v with logits[r][v] = m,
 *   conf[r] = max_v softmax(logits[r])_v = 1 / sum_v exp(logits[r][v] - m).
 * A NaN logit never wins the argmax and makes conf NaN; a row with nothing
 * above -inf gets id 0 and conf 0. fp32 arithmetic (relative error of conf
 * within a few 1e-6 at vocab 131072).
 *
 *   logits  bf16 [rows, ld], the first `vocab` entries of each row used;
 *           ld >= vocab and a multiple of 8, base 16-byte aligned
 *   ids     int32 [rows]
 *   conf    fp32 [rows]
 */
nld_status_t nld_logits_argmax(const void *logits, int rows, int vocab, int ld, int32_t *ids,
                               float *conf, cudaStream_t stream);

/*
 * AR-diffusion ensemble verifier (appendix, quadratic self-speculation:
 * verification with the ensemble): per row r,
 *   p = lambda softmax(ar_logits[r]) + (1 - lambda) softmax(diff_logits[r]),
 *   ids[r] = the lowest v with p_v = max p,  conf[r] = max p,
 * from the causal logits at a speculative token and the denoising logits at
 * the mask that follows it. A row whose logits are all -inf contributes
 * nothing; logits are finite or -inf. fp32 arithmetic: two rows whose
 * mixture values lie within a few 1e-6 (relative) of each other may be taken
 * in either order.
 *
 *   ar_logits, diff_logits  bf16 [rows, ld], first `vocab` entries used;
 *                           ld >= vocab, a multiple of 8; 16-byte aligned
 *   lambda                  in [0, 1]
 *   ids int32 [rows], conf fp32 [rows]
 */
nld_status_t nld_logits_ensemble_argmax(const void *ar_logits, const void *diff_logits, int rows,
                                        int vocab, int ld, float lambda, int32_t *ids, float *conf,
                                        cudaStream_t stream);

/*
 * Block KV commit into the paged cache (Sec. 3 Mode 3: the accepted drafts
 * are committed to the verified prefix and the verifier's cache is rebuilt
 * at the rejection point; Sec. 2: a completed diffusion block's KV cache is
 * refreshed). Row j < count_b of the new block K/V is written to logical
 * slot L_b + j, i.e. page page_table[b][(L_b + j) / P], slot (L_b + j) % P,
 * for every KV head; with advance != 0, prefix_lens[b] then grows by
 * count_b. Slots past the committed rows are left untouched (they are no
 * longer part of the prefix: that is the rollback).
 *
 * Uses:
 *   - before an attention pass, stage the block's own K/V in slots
 *     [L_b, L_b + bl): counts = NULL, advance = 0;
 *   - after verification, commit the accepted drafts (the verify pass's K/V
 *     of those positions): counts = accepted_len from nld_accept, advance = 1
 *     (the bonus token's K/V comes from the next forward pass);
 *   - when a diffusion block completes, commit its refreshed K/V:
 *     counts = NULL, advance = 1.
 *
 *   params      shapes as for nld_block_attn (batch, num_kv_heads, head_dim,
 *               page_size, num_pages, max_pages_per_seq)
 *   k_new, v_new bf16 [B, block_len, Hkv, D]
 *   counts      int32 [B] on the device, 0 .. block_len, or NULL (= block_len)
 *   page_table  int32 [B, max_pages_per_seq], covering the written slots
 *   prefix_lens int32 [B] on the device (read; updated when advance != 0)
 *   k_pages, v_pages bf16 [num_pages, Hkv, P, D], written
 *
 * Device-side range errors (a count outside 0..block_len, a slot past the
 * page table, a page id outside the pool) are flagged in nld_device_error
 * and the row is skipped. The call writes the cache and prefix_lens: an
 * attention call enqueued after it must not pass NLD_ATTN_PREFIX_READY.
 */
nld_status_t nld_kv_commit(const nld_attn_params_t *params, const void *k_new, const void *v_new,
                           const int32_t *counts, const int32_t *page_table, int32_t *prefix_lens,
                           int block_len, int advance, void *k_pages, void *v_pages,
                           cudaStream_t stream);

/*
 * Failure-detection check: launches one thread that waits, with the same
 * bounded wait every pipeline uses, on an mbarrier nothing ever arrives on.
 * After limit_ns nanoseconds (1 .. 1e9) the wait gives up, sets
 * NLD_DEVERR_WAIT_TIMEOUT in the device error word and the kernel returns;
 * the context stays usable. For tests and diagnostics.
 * Errors: NLD_ERR_INVALID_ARG (limit out of range), NLD_ERR_CUDA (launch).
 */
nld_status_t nld_check_wait_timeout(uint64_t limit_ns, cudaStream_t stream);

/* A static, human-readable name for a status code. */
const char *nld_status_string(nld_status_t status);

/*
 * Read the current device's error word (NLD_DEVERR_* bits) into *bits;
 * with clear != 0 reset it to 0. Synchronises the device; meant for tests
 * and diagnostics, not for the decode loop.
 */
nld_status_t nld_device_error(uint32_t *bits, int clear);

/*
 * Read the current device's count of running-max rescale events into
 * *count; with clear != 0 reset it to 0. The attention kernels keep a
 * row's running softmax maximum lazily (the online softmax of the scaled
 * scores, Sec. 2.2 attention): the accumulated output is rescaled in tensor
 * memory only when a later tile raises the row maximum by more than 2^8
 * (base 2). Each warp that performs such a rescale adds 1. The count tells
 * tests and diagnostics that this path ran; it does not change any result.
 * Synchronises the device; not for the decode loop.
 */
nld_status_t nld_rescale_count(uint64_t *count, int clear);

#ifdef __cplusplus
}
#endif

#endif /* NLD_H */
