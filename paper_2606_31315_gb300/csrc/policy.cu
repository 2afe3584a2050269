// Block-size policy head (Sections 2.3-2.4 of the BlockPilot paper): once per request,
//   h = max(0, W1 x + b1),  o = W2 h + b2,  block size = candidates[argmax o].
//
// Kernel 1 streams W1 exactly once for a group of up to 32 requests: the pooled feature
// rows of the group are staged in shared memory (gathered by row_index), every warp owns
// hidden rows and reads them with 16-byte loads, fp32 accumulation, warp-shuffle
// reduction, bias and ReLU fused into the store of h.  Kernel 2 (one CTA per request)
// applies the small output layer and takes the argmax with the lowest index on ties.
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx_sm103.cuh"

namespace bp {
namespace {

constexpr int kGroup = 32;       // requests per pass over W1
constexpr int kThreads1 = 256;   // 8 warps
constexpr int kRowsPerWarp = 2;
constexpr int kSmemBudget = 160 * 1024;

template <typename T>
struct Vec8;  // 8 consecutive elements as fp32
template <>
struct Vec8<__nv_bfloat16> {
    __device__ __forceinline__ static void load(const __nv_bfloat16* p, float (&f)[8]) {
        const uint4 u = *reinterpret_cast<const uint4*>(p);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
};
template <>
struct Vec8<float> {
    __device__ __forceinline__ static void load(const float* p, float (&f)[8]) {
        const float4 a = *reinterpret_cast<const float4*>(p);
        const float4 b = *reinterpret_cast<const float4*>(p + 4);
        f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
        f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
    }
};

template <typename T>
__global__ void __launch_bounds__(kThreads1) policy_hidden_kernel(const T* __restrict__ feats, int64_t row_stride,
                                                                  const int32_t* __restrict__ row_index, int n0,
                                                                  int ng, int d_in, const T* __restrict__ w1,
                                                                  const float* __restrict__ b1, int hidden,
                                                                  float* __restrict__ hbuf) {
    extern __shared__ uint8_t smem_raw[];
    T* xs = reinterpret_cast<T*>(smem_raw);  // [ng][d_in]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    griddep_launch_dependents();
    griddep_wait();
    // stage the pooled rows of this request group (16-byte copies)
    const int per_row = d_in * (int)sizeof(T) / 16;
    for (int idx = tid; idx < ng * per_row; idx += kThreads1) {
        const int n = idx / per_row, c = idx % per_row;
        const long long row = row_index ? (long long)row_index[n0 + n] : (long long)(n0 + n);
        reinterpret_cast<uint4*>(xs + (size_t)n * d_in)[c] =
            reinterpret_cast<const uint4*>(feats + row * row_stride)[c];
    }
    __syncthreads();
    const int row_base = (blockIdx.x * (kThreads1 / 32) + warp) * kRowsPerWarp;
    for (int rr = 0; rr < kRowsPerWarp; ++rr) {
        const int j = row_base + rr;
        if (j >= hidden) break;
        float acc[kGroup];
#pragma unroll
        for (int n = 0; n < kGroup; ++n) acc[n] = 0.f;
        const T* wr = w1 + (size_t)j * d_in;
        for (int d = lane * 8; d < d_in; d += 256) {
            float w8[8];
            Vec8<T>::load(wr + d, w8);
#pragma unroll
            for (int n = 0; n < kGroup; ++n) {
                if (n < ng) {
                    float x8[8];
                    Vec8<T>::load(xs + (size_t)n * d_in + d, x8);
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[n] = fmaf(w8[e], x8[e], acc[n]);
                }
            }
        }
        float mine = 0.f;
#pragma unroll
        for (int n = 0; n < kGroup; ++n) {
            float v = acc[n];
#pragma unroll
            for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == n) mine = v;
        }
        if (lane < ng) hbuf[(size_t)(n0 + lane) * hidden + j] = fmaxf(0.f, mine + b1[j]);
    }
}

template <typename T>
__global__ void __launch_bounds__(256) policy_out_kernel(const float* __restrict__ hbuf, int hidden,
                                                         const T* __restrict__ w2, const float* __restrict__ b2,
                                                         int num_cand, const int32_t* __restrict__ candidates,
                                                         float* __restrict__ logits_out,
                                                         int32_t* __restrict__ block_size_out) {
    __shared__ float red[8];
    __shared__ float logits[64];
    const int n = blockIdx.x, tid = threadIdx.x;
    griddep_launch_dependents();
    griddep_wait();
    const float* h = hbuf + (size_t)n * hidden;
    for (int c = 0; c < num_cand; ++c) {
        float acc = 0.f;
        for (int j = tid; j < hidden; j += 256) acc = fmaf(static_cast<float>(w2[(size_t)c * hidden + j]), h[j], acc);
#pragma unroll
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if ((tid & 31) == 0) red[tid >> 5] = acc;
        __syncthreads();
        if (tid == 0) {
            float t = 0.f;
            for (int w = 0; w < 8; ++w) t += red[w];
            logits[c] = t + b2[c];
        }
        __syncthreads();
    }
    if (tid == 0) {
        int best = 0;
        for (int c = 1; c < num_cand; ++c)
            if (logits[c] > logits[best]) best = c;
        block_size_out[n] = candidates[best];
        if (logits_out)
            for (int c = 0; c < num_cand; ++c) logits_out[(size_t)n * num_cand + c] = logits[c];
    }
}

template <typename T>
int run(const PolicyArgs& a, cudaStream_t stream) {
    float* hbuf = static_cast<float*>(a.scratch);
    const int max_group = kSmemBudget / (a.d_in * (int)sizeof(T));
    if (max_group < 1) return BP_ERR_UNSUPPORTED;
    const int group = max_group < kGroup ? max_group : kGroup;
    const int rows_per_block = (kThreads1 / 32) * kRowsPerWarp;
    const unsigned blocks = (unsigned)((a.hidden + rows_per_block - 1) / rows_per_block);
    static int configured = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured != dev) {
        if (cudaFuncSetAttribute(policy_hidden_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget) !=
                cudaSuccess ||
            cudaFuncSetAttribute(policy_hidden_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared) != cudaSuccess ||
            cudaFuncSetAttribute(policy_out_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared) != cudaSuccess)
            return BP_ERR_CUDA;
        configured = dev;
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    for (int n0 = 0; n0 < a.num_reqs; n0 += group) {
        const int ng = a.num_reqs - n0 < group ? a.num_reqs - n0 : group;
        cfg.gridDim = dim3(blocks, 1, 1);
        cfg.blockDim = dim3(kThreads1, 1, 1);
        cfg.dynamicSmemBytes = (size_t)ng * a.d_in * sizeof(T);
        if (cudaLaunchKernelEx(&cfg, policy_hidden_kernel<T>, static_cast<const T*>(a.feats), a.row_stride,
                               a.row_index, n0, ng, a.d_in, static_cast<const T*>(a.w1), a.b1, a.hidden,
                               hbuf) != cudaSuccess)
            return BP_ERR_CUDA;
    }
    cfg.gridDim = dim3((unsigned)a.num_reqs, 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = 0;
    if (cudaLaunchKernelEx(&cfg, policy_out_kernel<T>, (const float*)hbuf, a.hidden, static_cast<const T*>(a.w2), a.b2,
                           a.num_cand, a.candidates, a.logits_out, a.block_size_out) != cudaSuccess)
        return BP_ERR_CUDA;
    return BP_OK;
}

}  // namespace

size_t policy_scratch_bytes(int num_reqs, int hidden, int num_cand) {
    (void)num_cand;
    return align_up(sizeof(float) * (size_t)num_reqs * hidden, 256);
}

int launch_policy(const PolicyArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    (void)dev;
    if (a.num_reqs == 0) return BP_OK;
    return a.wdtype == BP_BF16 ? run<__nv_bfloat16>(a, stream) : run<float>(a, stream);
}

}  // namespace bp
