// The C ABI of libblockpilot: argument validation, workspace bookkeeping, device
// properties and TMA descriptor encoding.  Every entry point only enqueues work on the
// caller's stream (bp_get_status excepted) and never allocates.
#include <limits.h>
#include <math.h>
#include <mutex>

#include "common.cuh"

namespace bp {

int device_info(DeviceInfo* out) {
    static DeviceInfo cache[64];
    static std::mutex mu;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return BP_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(mu);
    DeviceInfo& d = cache[dev];
    if (d.device != dev) {
        DeviceInfo n;
        n.device = dev;
        if (cudaDeviceGetAttribute(&n.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n.cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
            cudaGetLastError();
            return BP_ERR_CUDA;
        }
        d = n;
    }
    if (d.cc_major != 10 || d.cc_minor != 3) return BP_ERR_CUDA;  // built for sm_103a only
    *out = d;
    return BP_OK;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int encode_tensor_map(CUtensorMap* map, CUtensorMapDataType dt, cuuint32_t rank, void* base, const cuuint64_t* dims,
                      const cuuint64_t* strides_bytes, const cuuint32_t* box, CUtensorMapSwizzle swizzle) {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
        cudaGetLastError();
    });
    if (!fn) return BP_ERR_CUDA;
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    const CUresult r = fn(map, dt, rank, base, dims, strides_bytes, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? BP_OK : BP_ERR_INVALID_ARG;
}

namespace {
bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_workspace(void* ws, size_t bytes, size_t need) {
    if (!ws || !aligned(ws, 256) || bytes < need) return BP_ERR_WORKSPACE;
    return BP_OK;
}
unsigned int* err_word(void* ws) { return &static_cast<WorkspaceHeader*>(ws)->error_bits; }
void* scratch(void* ws) { return static_cast<uint8_t*>(ws) + sizeof(WorkspaceHeader); }
}  // namespace

}  // namespace bp

using namespace bp;

extern "C" {

int bp_abi_version(void) { return BP_ABI_VERSION; }

const char* bp_error_string(int status) {
    switch (status) {
        case BP_OK: return "BP_OK";
        case BP_ERR_INVALID_ARG: return "BP_ERR_INVALID_ARG: invalid argument";
        case BP_ERR_UNSUPPORTED: return "BP_ERR_UNSUPPORTED: valid but unsupported shape or type";
        case BP_ERR_CUDA: return "BP_ERR_CUDA: CUDA call failed or no sm_103 device";
        case BP_ERR_WORKSPACE: return "BP_ERR_WORKSPACE: workspace missing, misaligned or too small";
        case BP_ERR_TIMEOUT: return "BP_ERR_TIMEOUT: a device-side bounded wait expired";
        case BP_ERR_DEVICE_FLAG: return "BP_ERR_DEVICE_FLAG: a device-side argument check failed";
        default: return "unknown bp_status";
    }
}

size_t bp_block_attention_workspace_size(int num_seqs, int max_q_len, int num_q_heads, int num_kv_heads,
                                         int head_dim) {
    (void)num_seqs; (void)head_dim;
    if (max_q_len < 1 || num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads != 0)
        return sizeof(WorkspaceHeader);
    return sizeof(WorkspaceHeader) + attention_flat_scratch_bytes(max_q_len, num_q_heads / num_kv_heads);
}

int bp_block_attention(const void* q, const void* k, const void* v, void* o, float* lse, const int32_t* cu_q,
                       const int32_t* cu_kv, int num_seqs, int total_q, int total_kv, int max_q_len,
                       int max_kv_len, int num_q_heads, int num_kv_heads, int head_dim, int dtype, int mask,
                       float softmax_scale, void* workspace, size_t workspace_bytes, void* stream) {
    if (num_seqs < 0 || total_q < 0 || total_kv < 0 || max_q_len < 0 || max_kv_len < 0) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0 || total_q == 0) return BP_OK;  // nothing to compute (empty tensors may be NULL)
    if (!q || !k || !v || !o || !cu_q || !cu_kv) return BP_ERR_INVALID_ARG;
    if (num_q_heads < 1 || num_kv_heads < 1 || head_dim < 1 || num_q_heads % num_kv_heads != 0)
        return BP_ERR_INVALID_ARG;
    if (mask != BP_MASK_CAUSAL_BLOCK && mask != BP_MASK_BIDIR_BLOCK) return BP_ERR_INVALID_ARG;
    if (dtype != BP_F32 && dtype != BP_BF16) return BP_ERR_INVALID_ARG;
    if (!(softmax_scale >= 0.f) || isinf(softmax_scale)) return BP_ERR_INVALID_ARG;
    if (max_q_len > max_kv_len || total_q > total_kv) return BP_ERR_INVALID_ARG;
    if (max_q_len > 64) return BP_ERR_UNSUPPORTED;
    if (dtype == BP_BF16 && head_dim != 128) return BP_ERR_UNSUPPORTED;
    if (dtype == BP_F32 && head_dim > 128) return BP_ERR_UNSUPPORTED;
    if (dtype == BP_BF16 && (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(o, 16)))
        return BP_ERR_INVALID_ARG;
    // the header is the minimum; a workspace of bp_block_attention_workspace_size bytes also holds the
    // flat split's partial slots (a smaller one keeps the cluster split)
    int rc = check_workspace(workspace, workspace_bytes, sizeof(WorkspaceHeader));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    AttentionArgs a;
    a.q = q; a.k = k; a.v = v; a.o = o; a.lse = lse; a.cu_q = cu_q; a.cu_kv = cu_kv;
    a.num_seqs = num_seqs; a.total_q = total_q; a.total_kv = total_kv;
    a.max_q_len = max_q_len; a.max_kv_len = max_kv_len;
    a.num_q_heads = num_q_heads; a.num_kv_heads = num_kv_heads; a.head_dim = head_dim;
    a.mask = mask;
    a.scale = softmax_scale == 0.f ? 1.f / sqrtf((float)head_dim) : softmax_scale;
    a.err_word = err_word(workspace);
    a.block_table = nullptr;
    a.pages_per_seq = a.page_size = a.num_pages = 0;
    a.scratch = scratch(workspace);
    a.scratch_bytes = workspace_bytes - sizeof(WorkspaceHeader);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    rc = dtype == BP_BF16 ? launch_attention_bf16(a, dev, st) : launch_attention_f32(a, st);
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

namespace {
bool valid_page_size(int page_size) { return page_size >= 16 && page_size <= (1 << 20) && (page_size & (page_size - 1)) == 0; }
}  // namespace

int bp_block_attention_paged(const void* q, const void* k_cache, const void* v_cache, void* o, float* lse,
                             const int32_t* cu_q, const int32_t* cu_kv, const int32_t* block_table,
                             int pages_per_seq, int page_size, int num_pages, int num_seqs, int total_q,
                             int total_kv, int max_q_len, int max_kv_len, int num_q_heads, int num_kv_heads,
                             int head_dim,
                             int dtype, int mask, float softmax_scale, void* workspace, size_t workspace_bytes,
                             void* stream) {
    if (num_seqs < 0 || total_q < 0 || total_kv < 0 || max_q_len < 0 || max_kv_len < 0) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0 || total_q == 0) return BP_OK;  // nothing to compute
    if (!q || !k_cache || !v_cache || !o || !cu_q || !cu_kv || !block_table) return BP_ERR_INVALID_ARG;
    if (num_q_heads < 1 || num_kv_heads < 1 || head_dim < 1 || num_q_heads % num_kv_heads != 0)
        return BP_ERR_INVALID_ARG;
    if (mask != BP_MASK_CAUSAL_BLOCK && mask != BP_MASK_BIDIR_BLOCK) return BP_ERR_INVALID_ARG;
    if (dtype != BP_F32 && dtype != BP_BF16) return BP_ERR_INVALID_ARG;
    if (!(softmax_scale >= 0.f) || isinf(softmax_scale)) return BP_ERR_INVALID_ARG;
    if (max_q_len > max_kv_len || total_q > total_kv || !valid_page_size(page_size) || num_pages < 1)
        return BP_ERR_INVALID_ARG;
    if ((long long)pages_per_seq * page_size < max_kv_len || (long long)num_pages * page_size > INT32_MAX)
        return BP_ERR_INVALID_ARG;
    if (max_q_len > 64) return BP_ERR_UNSUPPORTED;
    if (dtype != BP_BF16 || head_dim != 128) return BP_ERR_UNSUPPORTED;  // tensor-core path only
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(o, 16)) return BP_ERR_INVALID_ARG;
    // the header is the minimum; a workspace of bp_block_attention_workspace_size bytes also holds the
    // flat split's partial slots (a smaller one keeps the cluster split)
    int rc = check_workspace(workspace, workspace_bytes, sizeof(WorkspaceHeader));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    AttentionArgs a;
    a.q = q; a.k = k_cache; a.v = v_cache; a.o = o; a.lse = lse; a.cu_q = cu_q; a.cu_kv = cu_kv;
    a.num_seqs = num_seqs; a.total_q = total_q; a.total_kv = total_kv;
    a.max_q_len = max_q_len; a.max_kv_len = max_kv_len;
    a.num_q_heads = num_q_heads; a.num_kv_heads = num_kv_heads; a.head_dim = head_dim;
    a.mask = mask;
    a.scale = softmax_scale == 0.f ? 1.f / sqrtf((float)head_dim) : softmax_scale;
    a.err_word = err_word(workspace);
    a.block_table = block_table;
    a.pages_per_seq = pages_per_seq;
    a.page_size = page_size;
    a.num_pages = num_pages;
    a.scratch = scratch(workspace);
    a.scratch_bytes = workspace_bytes - sizeof(WorkspaceHeader);
    rc = launch_attention_bf16(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

int bp_kv_append(void* k_cache, void* v_cache, const void* k_new, const void* v_new, const int32_t* cu_new,
                 const int32_t* cu_kv, const int32_t* block_table, int pages_per_seq, int page_size, int num_pages,
                 int num_seqs, int total_new, int num_kv_heads, int head_dim, int dtype, void* stream) {
    if (num_seqs < 0 || total_new < 0) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0 || total_new == 0) return BP_OK;
    if (!k_cache || !v_cache || !k_new || !v_new || !cu_new || !cu_kv || !block_table) return BP_ERR_INVALID_ARG;
    if (num_kv_heads < 1 || head_dim < 1 || pages_per_seq < 1 || num_pages < 1 || !valid_page_size(page_size))
        return BP_ERR_INVALID_ARG;
    if (dtype != BP_F32 && dtype != BP_BF16) return BP_ERR_INVALID_ARG;
    const int row_bytes = head_dim * (dtype == BP_BF16 ? 2 : 4);
    if (row_bytes % 16 != 0) return BP_ERR_UNSUPPORTED;
    if (!aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(k_new, 16) || !aligned(v_new, 16))
        return BP_ERR_INVALID_ARG;
    DeviceInfo dev;
    int rc = device_info(&dev);
    if (rc != BP_OK) return rc;
    KvAppendArgs a;
    a.k_cache = k_cache; a.v_cache = v_cache; a.k_new = k_new; a.v_new = v_new;
    a.cu_new = cu_new; a.cu_kv = cu_kv; a.block_table = block_table;
    a.pages_per_seq = pages_per_seq; a.page_size = page_size; a.num_seqs = num_seqs; a.total_new = total_new;
    a.num_kv_heads = num_kv_heads; a.row_bytes = row_bytes;
    rc = launch_kv_append(a, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

size_t bp_spec_accept_workspace_size(int num_seqs, int total_draft, int vocab) {
    if (num_seqs < 0 || total_draft < 0 || vocab < 1) return 0;
    const size_t s = accept_scratch_bytes(num_seqs, total_draft, vocab);
    return s == 0 && num_seqs > 0 ? 0 : sizeof(WorkspaceHeader) + s;
}

int bp_spec_accept(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                   const int32_t* cu_draft, int num_seqs, int total_draft, int vocab, float temperature,
                   const float* u_accept, const float* u_sample, int32_t* n_accepted, int32_t* out_tokens,
                   float* accept_prob, void* workspace, size_t workspace_bytes, void* stream) {
    if (num_seqs < 0 || total_draft < 0 || vocab < 1) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0) return BP_OK;  // nothing to compute (empty tensors may be NULL)
    if (!target_logits || !cu_draft || !n_accepted || !out_tokens || (total_draft > 0 && !draft_tokens))
        return BP_ERR_INVALID_ARG;
    if (!(temperature >= 0.f) || isinf(temperature)) return BP_ERR_INVALID_ARG;
    if (temperature > 0.f && (!u_sample || (total_draft > 0 && (!draft_logits || !u_accept))))
        return BP_ERR_INVALID_ARG;
    if ((long long)(total_draft + (long long)num_seqs) * vocab > (1LL << 40)) return BP_ERR_UNSUPPORTED;
    const size_t need = bp_spec_accept_workspace_size(num_seqs, total_draft, vocab);
    if (need == 0 && num_seqs > 0) return BP_ERR_UNSUPPORTED;
    int rc = check_workspace(workspace, workspace_bytes, need);
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    AcceptArgs a;
    a.target = target_logits; a.draft = draft_logits; a.tokens = draft_tokens; a.cu_draft = cu_draft;
    a.num_seqs = num_seqs; a.total_draft = total_draft; a.vocab = vocab; a.temperature = temperature;
    a.u_accept = u_accept; a.u_sample = u_sample;
    a.n_accepted = n_accepted; a.out_tokens = out_tokens; a.accept_prob = accept_prob;
    a.scratch = scratch(workspace);
    a.err_word = err_word(workspace);
    rc = launch_accept(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

int bp_spec_accept_noalloc(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                           const int32_t* cu_draft, int num_seqs, int total_draft, int vocab, float temperature,
                           const float* u_accept, const float* u_sample, int32_t* n_accepted, int32_t* out_tokens,
                           float* accept_prob, unsigned int* device_error, void* stream) {
    if (num_seqs < 0 || total_draft < 0 || vocab < 1) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0) return BP_OK;
    if (!target_logits || !cu_draft || !n_accepted || !out_tokens || (total_draft > 0 && !draft_tokens))
        return BP_ERR_INVALID_ARG;
    if (!(temperature >= 0.f) || isinf(temperature)) return BP_ERR_INVALID_ARG;
    if (temperature > 0.f && (!u_sample || (total_draft > 0 && (!draft_logits || !u_accept))))
        return BP_ERR_INVALID_ARG;
    if ((long long)(total_draft + (long long)num_seqs) * vocab > (1LL << 40)) return BP_ERR_UNSUPPORTED;
    DeviceInfo dev;
    int rc = device_info(&dev);
    if (rc != BP_OK) return rc;
    AcceptArgs a;
    a.target = target_logits; a.draft = draft_logits; a.tokens = draft_tokens; a.cu_draft = cu_draft;
    a.num_seqs = num_seqs; a.total_draft = total_draft; a.vocab = vocab; a.temperature = temperature;
    a.u_accept = u_accept; a.u_sample = u_sample;
    a.n_accepted = n_accepted; a.out_tokens = out_tokens; a.accept_prob = accept_prob;
    a.scratch = nullptr;
    a.err_word = device_error;
    rc = launch_accept_noalloc(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

size_t bp_verify_epilogue_workspace_size(int num_seqs, int total_draft, int vocab) {
    if (num_seqs < 0 || total_draft < 0 || vocab < 1) return 0;
    return sizeof(WorkspaceHeader) + verify_epilogue_scratch_bytes(num_seqs, total_draft, vocab);
}

int bp_verify_epilogue(const void* lm_head, const void* h_target, const void* h_draft, int hidden, int vocab,
                       const int32_t* draft_tokens, const int32_t* cu_draft, int num_seqs, int total_draft,
                       float temperature, const float* u_accept, const float* u_sample, int32_t* n_accepted,
                       int32_t* out_tokens, float* accept_prob, float* logits_out, void* workspace,
                       size_t workspace_bytes, void* stream) {
    if (num_seqs < 0 || total_draft < 0 || vocab < 1 || hidden < 1) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0) return BP_OK;
    if (!lm_head || !h_target || !cu_draft || !n_accepted || !out_tokens || (total_draft > 0 && !draft_tokens))
        return BP_ERR_INVALID_ARG;
    if (!(temperature >= 0.f) || isinf(temperature)) return BP_ERR_INVALID_ARG;
    const bool greedy = temperature == 0.f;
    if (!greedy && (!u_sample || (total_draft > 0 && (!h_draft || !u_accept)))) return BP_ERR_INVALID_ARG;
    if (hidden % 64 != 0) return BP_ERR_UNSUPPORTED;
    if (!aligned(lm_head, 16) || !aligned(h_target, 16) || (!greedy && h_draft && !aligned(h_draft, 16)))
        return BP_ERR_UNSUPPORTED;
    const long long rows = (long long)total_draft + num_seqs + (greedy ? 0 : total_draft);
    if (2LL * total_draft + num_seqs > INT_MAX / 2) return BP_ERR_UNSUPPORTED;
    int rc = check_workspace(workspace, workspace_bytes,
                             bp_verify_epilogue_workspace_size(num_seqs, total_draft, vocab));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    if (rows > kVerifyResidentRows) {  // streamed: any vocabulary the SMs can be given a slice of
        if (verify_stream_grid(vocab, dev.sm_count) < 1) return BP_ERR_UNSUPPORTED;
    } else {
        int grid, np, per;
        if ((rc = verify_epilogue_config((int)rows, vocab, hidden, dev.sm_count, &grid, &np, &per)) != BP_OK)
            return rc;
    }
    VerifyEpilogueArgs a;
    a.lm_head = lm_head; a.h_target = h_target; a.h_draft = h_draft;
    a.hidden = hidden; a.vocab = vocab; a.num_seqs = num_seqs; a.total_draft = total_draft;
    a.temperature = temperature;
    a.tokens = draft_tokens; a.cu_draft = cu_draft; a.u_accept = u_accept; a.u_sample = u_sample;
    a.n_accepted = n_accepted; a.out_tokens = out_tokens; a.accept_prob = accept_prob; a.logits_out = logits_out;
    a.scratch = scratch(workspace);
    a.err_word = err_word(workspace);
    rc = launch_verify_epilogue(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

size_t bp_tau_select_workspace_size(int num_reqs) {
    if (num_reqs < 0) return 0;
    return sizeof(WorkspaceHeader) + tau_scratch_bytes(num_reqs);
}

int bp_tau_select(const float* gamma, int num_reqs, int jmax, const int32_t* candidates, int num_cand, int train_block,
                  float alpha, const int32_t* predicted, float* tau_out, int32_t* best_out, float* regret_out,
                  double* summary_out, void* workspace, size_t workspace_bytes, void* stream) {
    if (num_reqs < 0 || jmax < 1 || num_cand < 1 || !(alpha >= 0.f) || isinf(alpha)) return BP_ERR_INVALID_ARG;
    if (num_reqs == 0) return BP_OK;
    if (!gamma || !candidates || !best_out || (regret_out && !predicted)) return BP_ERR_INVALID_ARG;
    if (num_cand > 32 || jmax > 64) return BP_ERR_UNSUPPORTED;
    for (int c = 0; c < num_cand; ++c) {  // strictly increasing sizes within the rows (a host array)
        const int b = candidates[c];
        if (b < 1 || b > 64 || (jmax > 1 && b > jmax) || (c > 0 && b <= candidates[c - 1])) return BP_ERR_INVALID_ARG;
    }
    int rc = check_workspace(workspace, workspace_bytes, bp_tau_select_workspace_size(num_reqs));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    TauArgs a;
    a.gamma = gamma; a.num_reqs = num_reqs; a.jmax = jmax; a.candidates = candidates; a.num_cand = num_cand;
    a.train_block = train_block; a.alpha = alpha; a.predicted = predicted; a.tau_out = tau_out;
    a.best_out = best_out; a.regret_out = regret_out; a.summary_out = summary_out;
    a.scratch = scratch(workspace);
    a.err_word = err_word(workspace);
    rc = launch_tau(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

int bp_verify_commit(int32_t* ctx_lens, const int32_t* n_accepted, const int32_t* out_tokens, const int32_t* cu_draft,
                     int num_seqs, int capacity, int32_t* anchor_out, int32_t* cu_kv_next, void* workspace,
                     size_t workspace_bytes, void* stream) {
    if (num_seqs < 0 || capacity < 1) return BP_ERR_INVALID_ARG;
    if (num_seqs == 0) return BP_OK;
    if (!ctx_lens || !n_accepted || !out_tokens || !cu_draft || !cu_kv_next) return BP_ERR_INVALID_ARG;
    int rc = check_workspace(workspace, workspace_bytes, sizeof(WorkspaceHeader));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    CommitArgs a;
    a.ctx_lens = ctx_lens; a.n_accepted = n_accepted; a.out_tokens = out_tokens; a.cu_draft = cu_draft;
    a.num_seqs = num_seqs; a.capacity = capacity; a.anchor_out = anchor_out; a.cu_kv_next = cu_kv_next;
    a.err_word = err_word(workspace);
    rc = launch_verify_commit(a, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

size_t bp_policy_select_workspace_size(int num_reqs, int d_in, int hidden, int num_cand) {
    if (num_reqs < 0 || d_in < 1 || hidden < 1 || num_cand < 1) return 0;
    return sizeof(WorkspaceHeader) + policy_scratch_bytes(num_reqs, d_in, hidden, num_cand);
}

int bp_policy_select(const void* feats, int64_t feat_row_stride, const int32_t* row_index, int num_reqs, int d_in,
                     const void* w1, const float* b1, int hidden, const void* w2, const float* b2, int num_cand,
                     const int32_t* candidates, int wdtype, float* logits_out, int32_t* block_size_out,
                     void* workspace, size_t workspace_bytes, void* stream) {
    if (num_reqs < 0 || d_in < 1 || hidden < 1 || num_cand < 1 || feat_row_stride < d_in) return BP_ERR_INVALID_ARG;
    if (num_reqs == 0) return BP_OK;  // nothing to compute
    if (!feats || !w1 || !b1 || !w2 || !b2 || !candidates || !block_size_out) return BP_ERR_INVALID_ARG;
    if (wdtype != BP_F32 && wdtype != BP_BF16) return BP_ERR_INVALID_ARG;
    if (num_cand > 64) return BP_ERR_UNSUPPORTED;
    const int elt = wdtype == BP_BF16 ? 2 : 4;
    if ((d_in * elt) % 16 != 0 || (feat_row_stride * elt) % 16 != 0 || !aligned(feats, 16) || !aligned(w1, 16))
        return BP_ERR_UNSUPPORTED;
    int rc = check_workspace(workspace, workspace_bytes, bp_policy_select_workspace_size(num_reqs, d_in, hidden, num_cand));
    if (rc != BP_OK) return rc;
    DeviceInfo dev;
    if ((rc = device_info(&dev)) != BP_OK) return rc;
    PolicyArgs a;
    a.feats = feats; a.row_stride = feat_row_stride; a.row_index = row_index; a.num_reqs = num_reqs; a.d_in = d_in;
    a.w1 = w1; a.b1 = b1; a.hidden = hidden; a.w2 = w2; a.b2 = b2; a.num_cand = num_cand;
    a.candidates = candidates; a.wdtype = wdtype; a.logits_out = logits_out; a.block_size_out = block_size_out;
    a.scratch = scratch(workspace);
    a.err_word = err_word(workspace);
    rc = launch_policy(a, dev, static_cast<cudaStream_t>(stream));
    if (rc == BP_ERR_CUDA) cudaGetLastError();
    return rc;
}

int bp_get_status(void* workspace, void* stream) {
    if (!workspace) return BP_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int bits = 0;
    if (cudaStreamSynchronize(st) != cudaSuccess ||
        cudaMemcpy(&bits, err_word(workspace), sizeof(bits), cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemset(err_word(workspace), 0, sizeof(bits)) != cudaSuccess) {
        cudaGetLastError();
        return BP_ERR_CUDA;
    }
    if (bits & kErrTimeout) return BP_ERR_TIMEOUT;
    if (bits & kErrDeviceArg) return BP_ERR_DEVICE_FLAG;
    return BP_OK;
}

}  // extern "C"
