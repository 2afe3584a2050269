// Commit of a verify step: the decoding loop's bookkeeping after the acceptance, on the device, so that
// a whole step (append the block's K/V, attend, accept, commit) runs without a host round trip and can
// be captured once in a CUDA graph and replayed.
//
// Section 2.1 / Figure 1 and Section 2.4: a step drafts a block of B_s = gamma_s + 1 positions (the
// anchor -- the last emitted token -- and gamma_s drafts); the verify pass appends all B_s rows to the
// KV cache; the target keeps the longest accepted prefix and emits one token.  The rows that stay are
// the anchor's and the accepted drafts', so the committed length grows by 1 + n_acc and the rejected
// drafts' rows are dropped (the next block overwrites them).  The next pass attends over ctx + B_s keys
// (the block size is fixed for the request), and its anchor is the token just emitted.
//
// One CTA: every sequence is checked first (a commit with n_acc outside [0, gamma] or a next pass
// beyond the cache's capacity raises the device flag and changes nothing), then the lengths advance
// and a chunked block scan writes the next key offsets.
#include <cuda_runtime.h>

#include "common.cuh"

namespace bp {
namespace {

constexpr int kCommitThreads = 1024;

__global__ void __launch_bounds__(kCommitThreads) verify_commit_kernel(int32_t* __restrict__ ctx,
                                                                       const int32_t* __restrict__ n_acc,
                                                                       const int32_t* __restrict__ out_tokens,
                                                                       const int32_t* __restrict__ cu_draft,
                                                                       int num_seqs, int capacity,
                                                                       int32_t* __restrict__ anchor,
                                                                       int32_t* __restrict__ cu_kv,
                                                                       unsigned int* err) {
    __shared__ int warp_tot[kCommitThreads / 32];
    __shared__ int carry_sh;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int bad = 0;
    for (int s = tid; s < num_seqs; s += kCommitThreads) {
        const int g = cu_draft[s + 1] - cu_draft[s];
        const int k = n_acc[s];
        if (g < 0 || k < 0 || k > g || (long long)ctx[s] + 1 + k + g + 1 > capacity) bad = 1;
    }
    if (__syncthreads_or(bad)) {
        if (tid == 0) raise_error(err, kErrDeviceArg);
        return;
    }
    if (tid == 0) {
        carry_sh = 0;
        cu_kv[0] = 0;
    }
    for (int base = 0; base < num_seqs; base += kCommitThreads) {
        const int s = base + tid;
        int len = 0;
        if (s < num_seqs) {
            const int d0 = cu_draft[s], g = cu_draft[s + 1] - d0, k = n_acc[s];
            const int c = ctx[s] + 1 + k;  // the anchor and the accepted drafts stay
            ctx[s] = c;
            if (anchor) anchor[s] = out_tokens[d0 + s + k];
            len = c + g + 1;  // keys of the next verify pass
        }
        int incl = len;  // inclusive scan over the block: warps, then the warp totals
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        __syncthreads();  // the previous chunk is done with warp_tot and carry_sh
        if (lane == 31) warp_tot[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int w = warp_tot[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            warp_tot[lane] = w;  // inclusive over the warps
        }
        __syncthreads();
        const int before = carry_sh + (warp > 0 ? warp_tot[warp - 1] : 0);
        if (s < num_seqs) cu_kv[s + 1] = before + incl;
        __syncthreads();
        if (tid == 0) carry_sh += warp_tot[kCommitThreads / 32 - 1];
    }
}

}  // namespace

int launch_verify_commit(const CommitArgs& a, cudaStream_t stream) {
    verify_commit_kernel<<<1, kCommitThreads, 0, stream>>>(a.ctx_lens, a.n_accepted, a.out_tokens, a.cu_draft,
                                                           a.num_seqs, a.capacity, a.anchor_out, a.cu_kv_next,
                                                           a.err_word);
    return cudaGetLastError() == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

}  // namespace bp
