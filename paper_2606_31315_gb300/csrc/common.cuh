// Internal declarations shared by the translation units of libblockpilot.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/blockpilot.h"

namespace bp {

// Workspace header: the first 256 bytes of every workspace.
//   word 0: sticky error bits (kErrTimeout | kErrDeviceArg), cleared by bp_get_status
struct WorkspaceHeader {
    unsigned int error_bits;
    unsigned int pad[63];
};
static_assert(sizeof(WorkspaceHeader) == 256, "workspace header is 256 bytes");

enum : unsigned int { kErrTimeout = 1u, kErrDeviceArg = 2u };

// Cycle budget of every bounded device-side wait for work to arrive (about one second at 2 GHz).  A
// wait that expires records kErrTimeout and the kernel winds down; before a CTA leaves it waits out its
// own copies and tensor-core operations still in flight with kDrainBudget, so nothing writes into its
// shared or tensor memory after it.  BP_TEST_SHORT_WAITS (a test-only build of the library) makes every
// such wait a single non-blocking test, so that the tests can take the wind-down path on purpose; the
// drains keep their budget.
#ifdef BP_TEST_SHORT_WAITS
constexpr long long kWaitBudget = 0;
#else
constexpr long long kWaitBudget = 2000000000LL;
#endif
constexpr long long kDrainBudget = 2000000000LL;

__device__ __forceinline__ void raise_error(unsigned int* err_word, unsigned int bits) {
    if (err_word) atomicOr(err_word, bits);
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Properties of the current device, cached once per device.
struct DeviceInfo {
    int device = -1;
    int sm_count = 0;
    int cc_major = 0, cc_minor = 0;
    int max_smem_optin = 0;
};
int device_info(DeviceInfo* out);  // BP_OK or BP_ERR_CUDA

// Encodes a tiled TMA descriptor (driver entry point resolved once).
int encode_tensor_map(CUtensorMap* map, CUtensorMapDataType dt, cuuint32_t rank, void* base, const cuuint64_t* dims,
                      const cuuint64_t* strides_bytes, const cuuint32_t* box, CUtensorMapSwizzle swizzle);

// Launchers (host side).  They assume the arguments were validated by the API layer.
struct AttentionArgs {
    const void* q;
    const void* k;
    const void* v;
    void* o;
    float* lse;
    const int32_t* cu_q;
    const int32_t* cu_kv;
    int num_seqs, total_q, total_kv, max_q_len, max_kv_len;
    int num_q_heads, num_kv_heads, head_dim;
    int mask;
    float scale;
    unsigned int* err_word;
    // paged KV cache (NULL block_table: contiguous rows from cu_kv); pool of num_pages pages
    const int32_t* block_table;
    int pages_per_seq, page_size, num_pages;
    void* scratch;  // workspace past the header (the flat split's partial slots)
    size_t scratch_bytes;
};
int launch_attention_bf16(const AttentionArgs& a, const DeviceInfo& dev, cudaStream_t stream);
// The flat split of the bf16 attention runs on at most this many CTAs (one per SM) and keeps two
// partial (O, m, l) slots per CTA in the workspace; a workspace without room for them keeps the
// cluster split.
constexpr int kAttnFlatMaxGrid = 192;
size_t attention_flat_scratch_bytes(int max_q_len, int group);

struct KvAppendArgs {
    void* k_cache;
    void* v_cache;
    const void* k_new;
    const void* v_new;
    const int32_t* cu_new;
    const int32_t* cu_kv;
    const int32_t* block_table;
    int pages_per_seq, page_size, num_seqs, total_new, num_kv_heads, row_bytes;  // row_bytes = head_dim * elt
};
int launch_kv_append(const KvAppendArgs& a, cudaStream_t stream);
int launch_attention_f32(const AttentionArgs& a, cudaStream_t stream);

struct AcceptArgs {
    const float* target;
    const float* draft;
    const int32_t* tokens;
    const int32_t* cu_draft;
    int num_seqs, total_draft, vocab;
    float temperature;
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    void* scratch;  // workspace past the header
    unsigned int* err_word;
};
size_t accept_scratch_bytes(int num_seqs, int total_draft, int vocab);
// allow_batch = false keeps every call on the cluster kernel (its scratch alone suffices)
int launch_accept(const AcceptArgs& a, const DeviceInfo& dev, cudaStream_t stream, bool allow_batch = true);
// The acceptance runs as the throughput kernels of accept_batch.cu from this many logits read on (the
// per-row cluster kernel below it): target rows x vocab at T = 0, target and drafter rows x vocab at
// T > 0.  Set at the measured crossover of the two on GB300.
constexpr long long kAcceptBatchLogitsT0 = 2500000;
constexpr long long kAcceptBatchLogitsT1 = 6500000;
inline bool accept_use_batch(int num_seqs, int total_draft, int vocab, bool greedy) {
    const long long rows = greedy ? (long long)total_draft + num_seqs : 2LL * total_draft + num_seqs;
    return rows * vocab >= (greedy ? kAcceptBatchLogitsT0 : kAcceptBatchLogitsT1);
}
// The workspace is sized for the throughput kernels when either temperature may use them.
inline bool accept_may_batch(int num_seqs, int total_draft, int vocab) {
    return accept_use_batch(num_seqs, total_draft, vocab, true) || accept_use_batch(num_seqs, total_draft, vocab, false);
}
size_t accept_batch_scratch_bytes(int num_seqs, int total_draft, int vocab);
int launch_accept_batch(const AcceptArgs& a, int sm_count, int* tickets, void* scratch, cudaStream_t stream);
// The throughput path's decisions and draw alone, from statistics merged beforehand: row_stats[r] is row
// r's (scaled max, sum of 2^(l*log2e/T - max)) over the whole vocabulary, at T = 0 its (max, lowest
// index bits); rows in the stacked order (target rows, then the drafter's).  At T = 0 no logits are read.
size_t accept_draw_scratch_bytes(int num_seqs, int vocab);
int launch_accept_rows(const AcceptArgs& a, const float2* row_stats, int sm_count, int* tickets, void* draw_scratch,
                       cudaStream_t stream);
// Same kernel, scratch taken from the library's own static device array (no workspace).
int launch_accept_noalloc(const AcceptArgs& a, const DeviceInfo& dev, cudaStream_t stream);

struct PolicyArgs {
    const void* feats;
    int64_t row_stride;
    const int32_t* row_index;
    int num_reqs, d_in;
    const void* w1;
    const float* b1;
    int hidden;
    const void* w2;
    const float* b2;
    int num_cand;
    const int32_t* candidates;
    int wdtype;
    float* logits_out;
    int32_t* block_size_out;
    void* scratch;
    unsigned int* err_word;
};
size_t policy_scratch_bytes(int num_reqs, int d_in, int hidden, int num_cand);
int launch_policy(const PolicyArgs& a, const DeviceInfo& dev, cudaStream_t stream);

struct VerifyEpilogueArgs {
    const void* lm_head;   // [vocab][hidden] bf16
    const void* h_target;  // [total_draft + num_seqs][hidden] bf16
    const void* h_draft;   // [total_draft][hidden] bf16 (unused at T = 0)
    int hidden, vocab, num_seqs, total_draft;
    float temperature;
    const int32_t* tokens;
    const int32_t* cu_draft;
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    float* logits_out;
    void* scratch;
    unsigned int* err_word;
};
// Rows (target + drafter) above which the verify epilogue streams the LM head (verify_stream.cu)
// instead of keeping every logit in tensor memory (verify_epilogue.cu).
constexpr int kVerifyResidentRows = 64;
size_t verify_epilogue_scratch_bytes(int num_seqs, int total_draft, int vocab);
// Grid size, padded row count (MMA N) and tiles per CTA; BP_ERR_UNSUPPORTED outside the limits.
int verify_epilogue_config(int rows, int vocab, int hidden, int sm_count, int* grid, int* np, int* tiles_per_cta);
int launch_verify_epilogue(const VerifyEpilogueArgs& a, const DeviceInfo& dev, cudaStream_t stream);
// The streamed path's scratch, carved from the verify epilogue's workspace.
struct VerifyStreamScratch {
    float* logits;      // [rows][vocab] fp32: the logits at T > 0 when the caller gives no logits_out
    float2* part;       // [rows][slices] slice statistics
    float2* row_stats;  // [rows] merged statistics
    int* tickets;       // [num_seqs], zero between calls
    void* draw;         // accept_draw_scratch_bytes(num_seqs, vocab)
};
int verify_stream_grid(int vocab, int sm_count);  // slices of the vocabulary (CTAs); < 1: unsupported
int launch_verify_stream(const VerifyEpilogueArgs& a, const VerifyStreamScratch& s, const DeviceInfo& dev,
                         cudaStream_t stream);

struct TauArgs {
    const float* gamma;         // [num_reqs][jmax]
    int num_reqs, jmax;
    const int32_t* candidates;  // [num_cand] HOST array, strictly increasing
    int num_cand, train_block;
    float alpha;
    const int32_t* predicted;   // [num_reqs] or null
    float* tau_out;             // [num_reqs][num_cand] or null
    int32_t* best_out;          // [num_reqs]
    float* regret_out;          // [num_reqs] or null
    double* summary_out;        // [4] or null
    void* scratch;
    unsigned int* err_word;
};
size_t tau_scratch_bytes(int num_reqs);
int launch_tau(const TauArgs& a, const DeviceInfo& dev, cudaStream_t stream);

struct CommitArgs {
    int32_t* ctx_lens;            // [num_seqs] in/out
    const int32_t* n_accepted;    // [num_seqs]
    const int32_t* out_tokens;    // [total_draft + num_seqs]
    const int32_t* cu_draft;      // [num_seqs + 1]
    int num_seqs, capacity;
    int32_t* anchor_out;          // [num_seqs] or null
    int32_t* cu_kv_next;          // [num_seqs + 1]
    unsigned int* err_word;
};
int launch_verify_commit(const CommitArgs& a, cudaStream_t stream);

}  // namespace bp
