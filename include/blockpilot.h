/*
 * blockpilot.h -- C ABI of the GB300 (sm_103a) block-verify hot path of BlockPilot
 * (instance-adaptive block sizes for diffusion-based speculative decoding,
 * arxiv 2606.31315).
 *
 * Three operations, one per stage of the per-request pipeline of Section 2.4:
 *
 *   bp_policy_select    once per request: the block-size predictor (Sections 2.3, 2.4)
 *   bp_block_attention  every step: block attention of the drafter (bidirectional within
 *                       the block) and of the target's verify pass (causal within the block)
 *                       over the KV cache (Section 2.1, Figure 1)
 *   bp_spec_accept      every step: lossless acceptance of the drafted block over the full
 *                       vocabulary -- the longest accepted prefix plus one corrected or bonus
 *                       token (Figure 1; Section 1)
 *
 * bp_block_attention_paged and bp_kv_append run the attention over a paged KV cache (pages of
 * a shared pool named by a per-sequence block table) and append a block's K/V to it.
 * bp_verify_epilogue fuses the LM head that produces the logits with bp_spec_accept: it takes
 * the final hidden states of the verified and drafted positions instead of their logits.
 * bp_tau_select evaluates Appendix A's acceptance-length model for a batch of requests.
 * bp_verify_commit rolls the KV lengths back to the accepted prefix on the device, closing the loop.
 *
 * Conventions shared by every entry point
 *   - Pointers to tensors are DEVICE pointers (cudaMalloc / torch allocations), owned by
 *     the caller; the library never allocates, frees or retains them after the call.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls only enqueue work:
 *     they return before the GPU has run it and never synchronize, except bp_get_status.
 *   - `workspace` is caller-owned device scratch of at least the size the matching
 *     *_workspace_size function returns, 256-byte aligned, ZERO-FILLED BEFORE ITS FIRST
 *     USE.  Every call puts its own counters back at zero, so the next call of the same
 *     entry point with the same *_workspace_size arguments can follow on it directly.  Its
 *     other scratch keeps data, and the counters of a call with other size arguments (or of
 *     another entry point) may lie where that data is: zero-fill the workspace again before
 *     such a call (spec_accept's per-sequence tickets come first, in 256-byte units of 64
 *     sequences, so there only a call with more of those units than an earlier one needs
 *     this).  Its first 16 bytes hold a sticky device error word read by bp_get_status.  Two
 *     calls that may run concurrently need distinct workspaces.
 *   - Host-checkable problems (NULL pointers, unsupported shapes, a workspace that is too
 *     small) return an error code immediately and enqueue nothing.  Problems only the GPU
 *     sees (a draft token id outside [0, V), a bounded wait that timed out) set the
 *     workspace error word; the outputs of that call are then undefined.
 *   - There is no CPU fallback: without a usable sm_103a device the calls return
 *     BP_ERR_CUDA.
 */
#ifndef BLOCKPILOT_H
#define BLOCKPILOT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BP_ABI_VERSION 3

/* Symbols of the ABI are exported; everything else in the library is hidden. */
#if defined(__GNUC__)
#define BP_API __attribute__((visibility("default")))
#else
#define BP_API
#endif

typedef enum {
    BP_OK = 0,
    BP_ERR_INVALID_ARG = 1, /* NULL pointer, negative size, inconsistent shape */
    BP_ERR_UNSUPPORTED = 2, /* valid but not implemented (e.g. bf16 attention with head_dim != 128) */
    BP_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed (no device, launch failure) */
    BP_ERR_WORKSPACE = 4,   /* workspace NULL, misaligned or smaller than required */
    BP_ERR_TIMEOUT = 5,     /* a device-side bounded wait expired (from bp_get_status) */
    BP_ERR_DEVICE_FLAG = 6  /* a device-side argument check failed (from bp_get_status) */
} bp_status;

typedef enum {
    BP_MASK_CAUSAL_BLOCK = 0, /* target verify: block query i sees context + block keys 0..i */
    BP_MASK_BIDIR_BLOCK = 1   /* dLLM drafter: every block query sees context + whole block */
} bp_mask;

typedef enum { BP_F32 = 0, BP_BF16 = 1 } bp_dtype;

/* ---------------------------------------------------------------------------------
 * Block attention.  Section 2.1 (the drafter proposes B tokens in one forward pass and
 * the target verifies them in one parallel pass) and the Figure 1 caption.
 *
 * For every sequence s, query head h and block position i:
 *   O[i,h] = sum_j softmax_j(scale * <q_{i,h}, k_{j,h/g}> + M_ij) v_{j,h/g},  g = Hq/Hkv
 * Sequence s owns query rows [cu_q[s], cu_q[s+1]) -- its block, B_s = cu_q[s+1]-cu_q[s]
 * rows -- and key/value rows [cu_kv[s], cu_kv[s+1]): its L_s context rows followed by the
 * block's own B_s rows (so cu_kv[s+1]-cu_kv[s] = L_s + B_s >= B_s).
 * Mask: BP_MASK_CAUSAL_BLOCK lets block query i see keys 0 .. L_s+i; BP_MASK_BIDIR_BLOCK
 * lets every block query see all L_s+B_s keys.
 *
 *   q, o     [total_q][num_q_heads][head_dim]   dtype (o written in dtype)
 *   k, v     [total_kv][num_kv_heads][head_dim] dtype; 16-byte aligned base addresses
 *   lse      [total_q][num_q_heads] float32, natural-log log-sum-exp of the scaled masked
 *            scores of each output row; may be NULL
 *   cu_q, cu_kv  [num_seqs+1] int32 device arrays, non-decreasing, cu_*[0] = 0,
 *            cu_q[num_seqs] = total_q, cu_kv[num_seqs] = total_kv
 *   max_q_len, max_kv_len  host-side upper bounds of B_s and L_s+B_s
 *   dtype    BP_BF16 (tensor-core path, head_dim 128) or BP_F32 (head_dim <= 128)
 *   softmax_scale  0 selects 1/sqrt(head_dim)
 * Limits: 1 <= num_kv_heads, num_q_heads % num_kv_heads == 0, max_q_len <= 64,
 * max_q_len <= max_kv_len.  Every key row must be finite (bf16 or fp32 values).
 * ------------------------------------------------------------------------------- */
BP_API size_t bp_block_attention_workspace_size(int num_seqs, int max_q_len, int num_q_heads, int num_kv_heads,
                                         int head_dim);
BP_API int bp_block_attention(const void* q, const void* k, const void* v, void* o, float* lse, const int32_t* cu_q,
                       const int32_t* cu_kv, int num_seqs, int total_q, int total_kv, int max_q_len,
                       int max_kv_len, int num_q_heads, int num_kv_heads, int head_dim, int dtype, int mask,
                       float softmax_scale, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------------
 * Block attention over a paged KV cache.  The same operation as bp_block_attention
 * (Section 2.1, Figure 1 caption), with the keys and values of every sequence held in
 * fixed-size pages of a shared pool, as a serving engine keeps them:
 *
 *   key/value j of sequence s  =  pool row  block_table[s*pages_per_seq + j/page_size]*page_size
 *                                           + j % page_size
 *
 *   k_cache, v_cache  [num_pages*page_size][num_kv_heads][128] bf16, 16-byte aligned
 *   block_table  [num_seqs][pages_per_seq] int32 device array of page ids (< num_pages);
 *            the first ceil((cu_kv[s+1]-cu_kv[s]) / page_size) entries of row s are used
 *   cu_kv    [num_seqs+1] prefix sums of the sequences' key counts L_s + B_s (only the
 *            counts matter here: the rows come from the pages); total_kv = cu_kv[num_seqs]
 *   page_size  a power of two >= 16; pages_per_seq * page_size >= max_kv_len
 *   everything else as bp_block_attention (bf16, head_dim 128 only; same workspace size).
 * The pages of a sequence may be anywhere in the pool and in any order; every row of every
 * page the block table names must be finite.
 * ------------------------------------------------------------------------------- */
BP_API int bp_block_attention_paged(const void* q, const void* k_cache, const void* v_cache, void* o, float* lse,
                                    const int32_t* cu_q, const int32_t* cu_kv, const int32_t* block_table,
                                    int pages_per_seq, int page_size, int num_pages, int num_seqs, int total_q,
                                    int total_kv, int max_q_len, int max_kv_len, int num_q_heads, int num_kv_heads,
                                    int head_dim, int dtype, int mask, float softmax_scale, void* workspace,
                                    size_t workspace_bytes, void* stream);

/* Appends the new K/V rows of every sequence (its block) to its pages: new row i of sequence
 * s, rows [cu_new[s], cu_new[s+1]) of k_new / v_new, becomes key L_s + i, with
 * L_s = (cu_kv[s+1]-cu_kv[s]) - (cu_new[s+1]-cu_new[s]) -- cu_kv already counts the block.
 *   k_new, v_new  [total_new][num_kv_heads][head_dim] dtype (bf16 or fp32),
 *                 head_dim * element size a multiple of 16 bytes
 *   k_cache, v_cache, block_table, pages_per_seq, page_size as bp_block_attention_paged
 * The pages that receive the rows must already be in the block table.  No workspace. */
BP_API int bp_kv_append(void* k_cache, void* v_cache, const void* k_new, const void* v_new, const int32_t* cu_new,
                        const int32_t* cu_kv, const int32_t* block_table, int pages_per_seq, int page_size,
                        int num_pages, int num_seqs, int total_new, int num_kv_heads, int head_dim, int dtype,
                        void* stream);
/* ---------------------------------------------------------------------------------
 * Lossless speculative acceptance over the full vocabulary.  Figure 1 caption (the
 * target accepts the longest consistent prefix of the drafted block), Section 1 and
 * Section 3.1 Metrics (the target's output distribution is preserved exactly).  The
 * paper leaves the rule to standard speculative sampling; this library implements:
 *
 *   p_i = softmax(target_row_i / T), q_i = softmax(draft_row_i / T)
 *   a_i = min(1, p_i(x_i) / q_i(x_i))         (q=0<p gives 1; p=q=0 gives 0)
 *   k   = first i < gamma_s with u_accept_i >= a_i, else gamma_s
 *   emitted token at slot k: the smallest t with C_t > u_sample_s * Z, C_t = sum_{j<=t} w_j,
 *   Z = sum_j w_j, where w = max(0, p_k - q_k) when k < gamma_s (w = p_k if that residual
 *   is identically zero) and w = p_gamma (the bonus row) when every draft was accepted.
 * temperature == 0 is greedy: accept iff x_i == argmax(target_row_i) (lowest index on
 * ties), emit argmax(target_row_k); draft_logits, u_accept and u_sample are not read.
 *
 *   Sequence s has gamma_s = cu_draft[s+1] - cu_draft[s] >= 0 drafted tokens.
 *   target_logits  [total_draft + num_seqs][vocab] fp32; the gamma_s + 1 target rows of s
 *                  start at row cu_draft[s] + s
 *   draft_logits   [total_draft][vocab] fp32; NULL allowed iff temperature == 0
 *   draft_tokens   [total_draft] int32, each in [0, vocab) (else BP_ERR_DEVICE_FLAG)
 *   cu_draft       [num_seqs+1] int32 device array, non-decreasing, cu_draft[0] = 0
 *   u_accept       [total_draft] fp32 uniforms in [0,1); u_sample [num_seqs] in [0,1)
 *   n_accepted     [num_seqs] int32 out: k
 *   out_tokens     [total_draft + num_seqs] int32 out: slots cu_draft[s]+s .. +gamma_s hold
 *                  x_0..x_{k-1}, the emitted token, then -1
 *   accept_prob    [total_draft] fp32 out: a_i for every drafted position; may be NULL
 * Row addresses must be 16-byte aligned for the vectorised path (vocab % 4 == 0 and
 * 16-byte aligned bases); other vocabularies take a scalar path.
 * Small problems run as one latency-bound kernel (a thread-block cluster per row); from 2.5M
 * logits read at T = 0 ((total_draft + num_seqs) x vocab) and 6.5M at T > 0 ((2 total_draft +
 * num_seqs) x vocab) on, as three throughput kernels (chunk statistics, decisions, draw).  The
 * rule and the result's bars are the same; the workspace of the larger problems grows by about
 * 16 bytes per row and 16K vocabulary entries, plus 4 KB per sequence and 16K entries.
 * ------------------------------------------------------------------------------- */
BP_API size_t bp_spec_accept_workspace_size(int num_seqs, int total_draft, int vocab);
BP_API int bp_spec_accept(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                   const int32_t* cu_draft, int num_seqs, int total_draft, int vocab, float temperature,
                   const float* u_accept, const float* u_sample, int32_t* n_accepted, int32_t* out_tokens,
                   float* accept_prob, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------------
 * bp_spec_accept without a workspace.  The paper has no counterpart: this entry point exists
 * for callers that cannot allocate device memory -- e.g. a plugin running inside another
 * inference engine that only hands it input and output buffers, or a serving loop that must
 * not call cudaMalloc while requests are in flight (it can synchronize the device).
 *
 * Same arguments, results and errors as bp_spec_accept, except:
 *   - no workspace: the scratch is a fixed array of BP_NOALLOC_SCRATCH_BYTES inside the
 *     library, held on every GPU that loads the library until the process exits;
 *   - the three throughput kernels run only when their scratch fits in the array too; other
 *     problems large enough for them run on the single kernel;
 *   - problems whose single-kernel scratch would exceed it return BP_ERR_WORKSPACE (8 bytes per
 *     target row, i.e. per total_draft + num_seqs, so about a million target rows fit);
 *   - device-detected errors are OR-ed into *device_error (a caller-owned device word, may be
 *     NULL to drop them) instead of a workspace: 1 = a wait timed out, 2 = a draft token id
 *     outside [0, vocab);
 *   - the first call on each device may load the library's acceptance module (placing the
 *     array in device memory) and looks up the array's device address (cached afterwards): make
 *     that first call during set-up, before any stream capture;
 *   - every call clears the array's per-sequence counters on `stream` before its kernel runs (the
 *     kernels leave them at zero, so this only matters after a call that did not finish normally);
 *     calls that run concurrently on the GPU (unordered streams) share the array and race.
 * ------------------------------------------------------------------------------- */
#define BP_NOALLOC_SCRATCH_BYTES (8u << 20)
BP_API int bp_spec_accept_noalloc(const float* target_logits, const float* draft_logits,
                                  const int32_t* draft_tokens, const int32_t* cu_draft, int num_seqs,
                                  int total_draft, int vocab, float temperature, const float* u_accept,
                                  const float* u_sample, int32_t* n_accepted, int32_t* out_tokens,
                                  float* accept_prob, unsigned int* device_error, void* stream);

/* ---------------------------------------------------------------------------------
 * Block-size policy head, run once per request after prefill.  Sections 2.3 and 2.4:
 * an MLP maps the request's prefill representation to one logit per candidate block
 * size and B_hat = argmax over the candidates, fixed for the whole request; Section 3.1
 * fixes two layers (hidden width 2048 by default).  With ReLU as the activation:
 *
 *   h = max(0, W1 x + b1),  o = W2 h + b2,  block_size_out[n] = candidates[argmax o]
 *
 * (lowest index on ties).  Pooling: request n reads feature row row_index[n] (e.g. its
 * last prefill token), or row n when row_index is NULL.  No preprocessing of x (Table 5).
 *
 *   feats       rows of d_in values of type wdtype, row_stride elements apart (>= d_in)
 *   w1 [hidden][d_in], w2 [num_cand][hidden] of type wdtype; b1 [hidden], b2 [num_cand] fp32
 *   candidates  [num_cand] int32 device array of block sizes
 *   logits_out  [num_reqs][num_cand] fp32 out, may be NULL; block_size_out [num_reqs] int32 out
 * Limits: d_in % 8 == 0 and 16-byte aligned rows for bf16 (d_in % 4 == 0 for fp32),
 * num_cand <= 64.  Any d_in: wide inputs (such as the V-sized logit vector of Section 3.1) are
 * streamed; the workspace then also holds the gathered bf16 rows (num_reqs rounded up to 64) x d_in,
 * which is why its size depends on d_in.
 * ------------------------------------------------------------------------------- */
BP_API size_t bp_policy_select_workspace_size(int num_reqs, int d_in, int hidden, int num_cand);
BP_API int bp_policy_select(const void* feats, int64_t feat_row_stride, const int32_t* row_index, int num_reqs, int d_in,
                     const void* w1, const float* b1, int hidden, const void* w2, const float* b2, int num_cand,
                     const int32_t* candidates, int wdtype, float* logits_out, int32_t* block_size_out,
                     void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------------
 * Verify epilogue: the LM-head projection of the final hidden states fused with the lossless
 * acceptance of bp_spec_accept; up to 64 rows without writing the logits to memory.  Section 2.1 and the
 * Figure 1 caption: the target scores every position of the drafted block in one pass and
 * keeps the longest accepted prefix; the distributions it compares are
 *
 *   p_i = softmax(W h_target_i / T),  q_i = softmax(W h_draft_i / T)
 *
 * with W the [vocab][hidden] LM head shared by the target and the drafter.  The acceptance,
 * its outputs and its conventions are those of bp_spec_accept applied to target_logits =
 * h_target W^T and draft_logits = h_draft W^T (fp32 accumulation of bf16 products).
 *
 *   lm_head      [vocab][hidden] bf16, 16-byte aligned
 *   h_target     [total_draft + num_seqs][hidden] bf16: the target's final states, rows in the
 *                target-row order of bp_spec_accept; 16-byte aligned
 *   h_draft      [total_draft][hidden] bf16: the drafter's final states at its drafted
 *                positions; NULL allowed iff temperature == 0
 *   draft_tokens, cu_draft, u_accept, u_sample, n_accepted, out_tokens, accept_prob: as in
 *                bp_spec_accept
 *   logits_out   [rows][vocab] fp32, may be NULL: if given, the logits are also written (rows:
 *                the target rows, then at T > 0 the drafter rows)
 * Two paths, chosen by rows = total_draft + num_seqs (+ total_draft at T > 0):
 *   rows <= 64: one cooperative launch of one CTA per SM keeps every logit in tensor memory; the
 *     logits never reach memory unless logits_out asks for them (then for testing: it adds the write
 *     traffic the fusion exists to avoid).  Limits: the vocabulary split over the SMs must leave each
 *     CTA at most 16 tiles of 128 entries and tiles x (32 if rows <= 32 else 64) <= 512 tensor-memory
 *     columns (152 SMs: vocab <= 155,648 at rows <= 64, 311,296 at rows <= 32).
 *   rows > 64: the logits of that many rows do not fit on chip (the GPU's tensor memory holds about
 *     39 MB; 248 rows of a 151,936-entry vocabulary take 151 MB), so the LM head is streamed in
 *     256-entry passes, groups of at most 256 rows per pass over W, and every row's statistics are
 *     formed in the projection's epilogue.  At T = 0 only the statistics leave the chip.  At T > 0
 *     the logits are written once (into logits_out if given, else into the workspace) and only the
 *     draw's row pair of each sequence and the logits at the drafted tokens are read back.  Any
 *     vocabulary; W is read once per group of 256 rows.
 * Limits (else BP_ERR_UNSUPPORTED): hidden % 64 == 0; the rows <= 64 limits above.
 * Workspace: bp_verify_epilogue_workspace_size(num_seqs, total_draft, vocab), sized for T > 0 (at
 * more than 64 rows it holds the [rows][vocab] fp32 logits; logits_out given, that part is unused).
 * ------------------------------------------------------------------------------- */
BP_API size_t bp_verify_epilogue_workspace_size(int num_seqs, int total_draft, int vocab);
BP_API int bp_verify_epilogue(const void* lm_head, const void* h_target, const void* h_draft, int hidden, int vocab,
                              const int32_t* draft_tokens, const int32_t* cu_draft, int num_seqs, int total_draft,
                              float temperature, const float* u_accept, const float* u_sample,
                              int32_t* n_accepted, int32_t* out_tokens, float* accept_prob, float* logits_out,
                              void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------------
 * Appendix A's model of the expected acceptance length over a batch of requests, the
 * optimal block size of each request and the regret of a predicted one.  Appendix A.1-A.2:
 *
 *   tau(b; x) = sum_{i=1}^{b} r(b; B)^i prod_{j<=i} gamma_j(x),   r(b; B) = exp(-alpha (b - B)^2)
 *
 * (gamma_j(x): predictability of request x at drafted position j; B = train_block, the block
 * size the drafter was trained with); B*(x) = argmax over the candidates of tau(b; x), lowest
 * index on ties.  Appendix A.3: R(x) = tau(B*) - tau(B_hat) <= L(x) |B* - B_hat| with L(x) the
 * largest |tau(b1) - tau(b2)| / |b1 - b2| over the candidates, so E[R] <= L_tau E|B* - B_hat|.
 *
 *   gamma        [num_reqs][jmax] fp32 device array; jmax == 1: one gamma_x per request
 *                (constant predictability, the geometric form of Appendix A.2)
 *   candidates   [num_cand] int32 HOST array (read during the call; the sizes and r(b; B) travel
 *                to the GPU with the launch), strictly increasing, each in [1, 64] and <= jmax
 *                when jmax > 1 (else BP_ERR_INVALID_ARG)
 *   predicted    [num_reqs] int32 device array of predicted sizes, each one of the candidates
 *                (else BP_ERR_DEVICE_FLAG), or NULL
 *   tau_out      [num_reqs][num_cand] fp32 out, may be NULL; best_out [num_reqs] int32 out: B*
 *   regret_out   [num_reqs] fp32 out, may be NULL (needs predicted)
 *   summary_out  [4] fp64 out, may be NULL: mean R, mean |B* - B_hat| (both 0 without
 *                predicted), L_tau, L_tau * mean |B* - B_hat| (the bound on mean R)
 * Limits: jmax <= 64, num_cand <= 32 (else BP_ERR_UNSUPPORTED).  Sums of the summary are formed
 * in a fixed order: the result does not depend on scheduling.
 * ------------------------------------------------------------------------------- */
BP_API size_t bp_tau_select_workspace_size(int num_reqs);
BP_API int bp_tau_select(const float* gamma, int num_reqs, int jmax, const int32_t* candidates, int num_cand,
                         int train_block, float alpha, const int32_t* predicted, float* tau_out, int32_t* best_out,
                         float* regret_out, double* summary_out, void* workspace, size_t workspace_bytes,
                         void* stream);

/* ---------------------------------------------------------------------------------
 * Commit of a verify step: the decoding loop's bookkeeping after the acceptance, on the device,
 * so that a step -- bp_kv_append of the block's K/V, bp_block_attention_paged, bp_spec_accept,
 * bp_verify_commit -- needs no host round trip and can be captured once in a CUDA graph.  Section
 * 2.1 / Figure 1: the verify pass appends the rows of all B_s = gamma_s + 1 block positions (the
 * anchor and the drafts); the rows that stay are the anchor's and the accepted drafts', the
 * rejected drafts' rows are dropped (the next block overwrites them):
 *
 *   ctx_lens[s]   += 1 + n_accepted[s]
 *   anchor_out[s]  = out_tokens[cu_draft[s] + s + n_accepted[s]]     (the next block's anchor)
 *   cu_kv_next     = prefix sums of ctx_lens[s] + gamma_s + 1        (the next pass's keys)
 *
 *   ctx_lens     [num_seqs] int32 device array, in/out: committed rows per sequence
 *   n_accepted, out_tokens, cu_draft: as bp_spec_accept writes / reads them
 *   capacity     rows a sequence's cache can hold (pages_per_seq * page_size)
 *   anchor_out   [num_seqs] int32 out, may be NULL; cu_kv_next [num_seqs+1] int32 out (may be the
 *                cu_kv array the next step's append and attention read)
 *   workspace    at least 256 bytes (the error word)
 * If some n_accepted is outside [0, gamma_s] or a next pass would exceed capacity, the device error
 * word is set (BP_ERR_DEVICE_FLAG) and nothing is changed.  One CTA; num_seqs is not limited.
 * ------------------------------------------------------------------------------- */
BP_API int bp_verify_commit(int32_t* ctx_lens, const int32_t* n_accepted, const int32_t* out_tokens,
                            const int32_t* cu_draft, int num_seqs, int capacity, int32_t* anchor_out,
                            int32_t* cu_kv_next, void* workspace, size_t workspace_bytes, void* stream);

/* Reads and clears the sticky device error word of `workspace` (synchronizes `stream`).
 * Returns BP_OK, BP_ERR_TIMEOUT or BP_ERR_DEVICE_FLAG (or BP_ERR_CUDA if the read fails). */
BP_API int bp_get_status(void* workspace, void* stream);

/* Human-readable name of a bp_status value (static string, never NULL). */
BP_API const char* bp_error_string(int status);

/* BP_ABI_VERSION of the loaded library. */
BP_API int bp_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BLOCKPILOT_H */
