// Appendix A's acceptance-length model over a batch of requests: tau(b; x) for every candidate block
// size, the optimal size B*(x), and the regret of a predicted size with its Lipschitz bound.
//
// Appendix A.1-A.2: tau(b; x) = sum_{i=1}^{b} r(b; B)^i prod_{j<=i} gamma_j(x) with retention
// r(b; B) = exp(-alpha (b - B)^2); B*(x) = argmax over the candidates (lowest index on ties).
// Appendix A.3: R(x) = tau(B*) - tau(B_hat) <= L(x) |B* - B_hat| with L(x) the largest slope of tau
// between adjacent candidates, so E[R] <= L_tau E|B* - B_hat| with L_tau = max_x L(x).
//
// One thread per request; a warp takes 32 consecutive requests (a grid of resident blocks strides over
// them).  The warp copies its 32 gamma rows into shared memory with coalesced 16-byte loads, each
// thread turns its row into the prefix products P_i = prod_{j<=i} gamma_j in registers and forms all
// candidates' tau at once as the product of P with the table R[i][c] = r_c^(i+1) (i < b_c) -- static
// fused multiply-adds with independent accumulators -- and the warp writes its tau rows back
// coalesced.  Only warp-level synchronisation inside the loop.
// Each block writes its regret sums and largest slope to the workspace; a one-CTA kernel folds them
// in block order, so the summary is deterministic.
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "ptx_sm103.cuh"

namespace bp {
namespace {

constexpr int kTauThreads = 256;
constexpr int kTauMaxCand = 32;
constexpr int kTauMaxJ = 64;
constexpr int kTauMaxBlocks = 4096;  // partials in the workspace

struct TauParams {
    const float* gamma;  // [n][jmax]
    int n, jmax;
    int nc;
    const int32_t* predicted;  // [n] or null
    float* tau;                // [n][nc] or null
    int32_t* best;             // [n]
    float* regret;             // [n] or null
    double* summary;           // [4] or null
    double* part;              // [blocks][4]: regret sum, |B* - B_hat| sum, largest slope, unused
    unsigned int* err;
};

// Per-warp staging area: two buffers of the warp's 32 gamma rows (ldr floats each) -- the next 32
// requests' rows stream in (cp.async) while the current ones are computed -- then its 32 tau rows.
__host__ __device__ inline int tau_ldr(int jmax) { return (jmax & 3) == 0 ? jmax + 4 : jmax + 1; }
__host__ __device__ inline int tau_warp_floats(int jmax, int nc) { return 32 * (2 * tau_ldr(jmax) + nc); }

// tau_c = sum_{i=1}^{b_c} r_c^i P_i is the product of the request's prefix products P with the table
// R[i][c] = r_c^(i+1) for i < b_c (0 past b_c and for padding candidates), the same for every request.
// The table travels as a kernel parameter: the fused multiply-adds read it from the constant bank.
template <int JM, int NCB>
struct TauTable {
    float R[JM * NCB];
    int cand[NCB];   // candidate sizes (padding: 0)
    float inv[NCB];  // 1 / (b_c - b_{c-1}); 0 for c = 0 and padding
};

template <int JM, int NCB>
__global__ void __launch_bounds__(kTauThreads) tau_kernel(const __grid_constant__ TauTable<JM, NCB> tab,
                                                          const TauParams p) {
    extern __shared__ float4 dyn4[];  // per-warp staging areas
    __shared__ double red_sh[kTauThreads / 32][3];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ldr = tau_ldr(p.jmax);
    float* rows_buf = reinterpret_cast<float*>(dyn4) + warp * tau_warp_floats(p.jmax, p.nc);
    float* out_sh = rows_buf + 2 * 32 * ldr;
    const bool vec = (p.jmax & 3) == 0 && (reinterpret_cast<uintptr_t>(p.gamma) & 15) == 0;
    const int q4 = p.jmax >> 2;
    const unsigned magic = vec ? (unsigned)((0x100000000ull + q4 - 1) / q4) : 0u;  // f / q4 = umulhi(f, magic)
    // a warp's tau rows start 32 * nc floats apart: 16-byte aligned whenever the array is
    const bool vout = p.tau && (reinterpret_cast<uintptr_t>(p.tau) & 15) == 0;
    float rsum_t = 0.f, lmax_t = 0.f;  // this thread's requests, in order (fp32: the FP64 pipe is slow)
    long long dsum_t = 0;
    // the warp's 32 rows of requests x0.. are contiguous: coalesced 16-byte asynchronous copies
    const auto prefetch = [&](long long xp, float* dst) {
        const int nrows = (int)min(32LL, (long long)p.n - xp);
        const float4* s4 = reinterpret_cast<const float4*>(p.gamma + (size_t)xp * p.jmax);
        for (int f = lane; f < nrows * q4; f += 32) {
            const int r = (int)__umulhi((unsigned)f, magic), q = f - r * q4;
            cp_async16(dst + r * ldr + 4 * q, s4 + f, true);
        }
    };
    // each warp takes 32 consecutive requests; the grid strides over them
    const long long xstride = (long long)gridDim.x * kTauThreads;
    long long x0 = ((long long)blockIdx.x * (kTauThreads / 32) + warp) * 32;
    if (vec && x0 < p.n) prefetch(x0, rows_buf);
    cp_async_commit();
    for (int buf = 0; x0 < p.n; x0 += xstride, buf ^= (vec ? 1 : 0)) {
        const int rows = (int)min(32LL, (long long)p.n - x0);
        float* rows_sh = rows_buf + buf * 32 * ldr;
        if (vec) {  // the next 32 requests' rows start streaming; this iteration's have landed
            if (x0 + xstride < p.n) prefetch(x0 + xstride, rows_buf + (buf ^ 1) * 32 * ldr);
            cp_async_commit();
            cp_async_wait_group<1>();
        } else {
            const float* src = p.gamma + (size_t)x0 * p.jmax;
            for (int f = lane; f < rows * p.jmax; f += 32) rows_sh[(f / p.jmax) * ldr + f % p.jmax] = __ldg(src + f);
        }
        __syncwarp();
        if (lane < rows) {
            const long long x = x0 + lane;
            const int bh = p.predicted ? __ldg(p.predicted + x) : -1;
            const float* row = rows_sh + lane * ldr;
            float P[JM];
            if (p.jmax == 1) {  // one gamma_x per request: P_i = gamma_x^i
                P[0] = row[0];
#pragma unroll
                for (int j = 1; j < JM; ++j) P[j] = P[j - 1] * row[0];
            } else {  // prefix products P_i = prod_{j<=i} gamma_j (rows shorter than JM padded with 0)
                if (vec) {  // 16-byte reads: eight consecutive lanes' rows fall on distinct banks
#pragma unroll
                    for (int q = 0; q < JM / 4; ++q) {
                        const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
                        const float4 v = 4 * q < p.jmax ? *reinterpret_cast<const float4*>(row + 4 * q) : z;
                        P[4 * q] = v.x;
                        P[4 * q + 1] = v.y;
                        P[4 * q + 2] = v.z;
                        P[4 * q + 3] = v.w;
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < JM; ++j) P[j] = j < p.jmax ? row[j] : 0.f;
                }
#pragma unroll
                for (int j = 1; j < JM; ++j) P[j] *= P[j - 1];
            }
            float t[NCB];
#pragma unroll
            for (int c = 0; c < NCB; ++c) t[c] = 0.f;
#pragma unroll
            for (int i = 0; i < JM; ++i) {
#pragma unroll
                for (int c = 0; c < NCB; ++c) t[c] = __fmaf_rn(P[i], tab.R[i * NCB + c], t[c]);
            }
            int bb = tab.cand[0], pi = -1;
            float l = 0.f, tb = t[0], tp = 0.f;
#pragma unroll
            for (int c = 0; c < NCB; ++c) {
                if (c < p.nc) {
                    if (t[c] > tb) {  // strictly greater: ties keep the lowest index
                        tb = t[c];
                        bb = tab.cand[c];
                    }
                    if (c > 0) l = fmaxf(l, fabsf(t[c] - t[c - 1]) * tab.inv[c]);
                    if (tab.cand[c] == bh) {
                        pi = c;
                        tp = t[c];
                    }
                    if (vout) out_sh[lane * p.nc + c] = t[c];
                    else if (p.tau) p.tau[(size_t)x * p.nc + c] = t[c];
                }
            }
            p.best[x] = bb;
            lmax_t = fmaxf(lmax_t, l);
            if (p.predicted) {
                if (pi < 0) raise_error(p.err, kErrDeviceArg);  // not a candidate
                const float rx = pi < 0 ? 0.f : tb - tp;
                if (p.regret) p.regret[x] = rx;
                rsum_t += rx;
                dsum_t += pi < 0 ? 0 : abs(bb - bh);
            }
        }
        __syncwarp();
        if (vout) {  // the warp's tau rows are contiguous in memory: coalesced 16-byte stores
            float* dst = p.tau + (size_t)x0 * p.nc;
            const int nf = rows * p.nc;
            for (int f = lane; f < nf / 4; f += 32)
                reinterpret_cast<float4*>(dst)[f] = reinterpret_cast<const float4*>(out_sh)[f];
            for (int f = (nf & ~3) + lane; f < nf; f += 32) dst[f] = out_sh[f];  // a ragged last chunk
        }
        __syncwarp();
    }
    // ---- this block's partials, reduced in a fixed order
    double rsum = rsum_t, dsum = (double)dsum_t, lmax = lmax_t;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
        dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
        lmax = fmax(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
    }
    if (lane == 0) {
        red_sh[warp][0] = rsum;
        red_sh[warp][1] = dsum;
        red_sh[warp][2] = lmax;
    }
    __syncthreads();
    if (tid == 0) {
        double a = 0.0, b = 0.0, c = 0.0;
        for (int w = 0; w < kTauThreads / 32; ++w) {
            a += red_sh[w][0];
            b += red_sh[w][1];
            c = fmax(c, red_sh[w][2]);
        }
        double* pp = p.part + (size_t)blockIdx.x * 4;
        pp[0] = a;
        pp[1] = b;
        pp[2] = c;
    }
}

// The blocks' partials in block order (one CTA; runs after tau_kernel on the same stream).
__global__ void __launch_bounds__(kTauThreads) tau_finish_kernel(const double* __restrict__ part, int blocks, int n,
                                                                 double* __restrict__ summary) {
    __shared__ double fin[kTauThreads][3];
    const int tid = threadIdx.x;
    double a = 0.0, b = 0.0, c = 0.0;
    for (int k = tid; k < blocks; k += kTauThreads) {  // thread tid: blocks tid, tid + 256, ...
        a += part[(size_t)k * 4];
        b += part[(size_t)k * 4 + 1];
        c = fmax(c, part[(size_t)k * 4 + 2]);
    }
    fin[tid][0] = a;
    fin[tid][1] = b;
    fin[tid][2] = c;
    for (int h = kTauThreads / 2; h >= 1; h >>= 1) {  // a fixed-order tree
        __syncthreads();
        if (tid < h) {
            fin[tid][0] += fin[tid + h][0];
            fin[tid][1] += fin[tid + h][1];
            fin[tid][2] = fmax(fin[tid][2], fin[tid + h][2]);
        }
    }
    if (tid == 0) {
        summary[0] = fin[0][0] / (double)n;
        summary[1] = fin[0][1] / (double)n;
        summary[2] = fin[0][2];
        summary[3] = fin[0][2] * (fin[0][1] / (double)n);
    }
}

}  // namespace

size_t tau_scratch_bytes(int num_reqs) {
    (void)num_reqs;
    return align_up((size_t)kTauMaxBlocks * 4 * sizeof(double), 256);
}

// Shared memory of one block: each warp's staging area (the JM x NCB table is a kernel parameter).
size_t tau_smem_bytes(int JM, int NCB, int jmax, int nc) {
    (void)JM;
    (void)NCB;
    return (size_t)(kTauThreads / 32) * tau_warp_floats(jmax, nc) * sizeof(float);
}

template <int JM, int NCB>
int tau_launch(const TauArgs& a, const TauParams& p, const DeviceInfo& dev, cudaStream_t stream) {
    static std::mutex cfg_mu;
    static int configured[64] = {};
    if (dev.device < 0 || dev.device >= 64) return BP_ERR_UNSUPPORTED;
    {
        std::lock_guard<std::mutex> cfg_lock(cfg_mu);  // once per device, from any host thread
        if (!configured[dev.device]) {
            const int most = (int)tau_smem_bytes(JM, NCB, kTauMaxJ, kTauMaxCand);
            if (cudaFuncSetAttribute(tau_kernel<JM, NCB>, cudaFuncAttributeMaxDynamicSharedMemorySize, most) !=
                cudaSuccess)
                return BP_ERR_CUDA;
            configured[dev.device] = 1;
        }
    }
    // the table: r_c = exp(-alpha (b_c - B)^2) and its powers as running products
    TauTable<JM, NCB> tab;
    for (int c = 0; c < NCB; ++c) {
        const bool live = c < a.num_cand;
        const int b = live ? a.candidates[c] : 0;
        const float d = (float)(b - a.train_block);
        const float r = live ? expf(-a.alpha * d * d) : 0.f;
        float pw = 1.f;
        for (int i = 0; i < JM; ++i) {
            pw *= r;
            tab.R[i * NCB + c] = i < b ? pw : 0.f;
        }
        tab.cand[c] = b;
        tab.inv[c] = live && c > 0 ? 1.f / (float)(b - a.candidates[c - 1]) : 0.f;
    }
    const size_t smem = tau_smem_bytes(0, 0, p.jmax, p.nc);
    int occ = 0;
    const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, tau_kernel<JM, NCB>, kTauThreads, smem);
    if (e != cudaSuccess || occ < 1) return BP_ERR_CUDA;
    const long long need = ((long long)p.n + kTauThreads - 1) / kTauThreads;
    long long blocks = (long long)dev.sm_count * occ;  // one wave; warps stride over the requests
    blocks = blocks < need ? blocks : need;
    blocks = blocks < kTauMaxBlocks ? blocks : kTauMaxBlocks;
    tau_kernel<JM, NCB><<<(unsigned)blocks, kTauThreads, smem, stream>>>(tab, p);
    if (p.summary) tau_finish_kernel<<<1, kTauThreads, 0, stream>>>(p.part, (int)blocks, p.n, p.summary);
    return cudaGetLastError() == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

int launch_tau(const TauArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    if (a.num_cand > kTauMaxCand || a.jmax > kTauMaxJ) return BP_ERR_UNSUPPORTED;
    for (int c = 0; c < a.num_cand; ++c) {  // strictly increasing sizes within the rows
        const int b = a.candidates[c];
        if (b < 1 || b > kTauMaxJ || (a.jmax > 1 && b > a.jmax) || (c > 0 && b <= a.candidates[c - 1]))
            return BP_ERR_INVALID_ARG;
    }
    TauParams p;
    p.gamma = a.gamma;
    p.n = a.num_reqs;
    p.jmax = a.jmax;
    p.nc = a.num_cand;
    p.predicted = a.predicted;
    p.tau = a.tau_out;
    p.best = a.best_out;
    p.regret = a.regret_out;
    p.summary = a.summary_out;
    p.part = reinterpret_cast<double*>(a.scratch);
    p.err = a.err_word;
    // register rows of 24, 32 or 64 prefix products (64 for one gamma per request: sizes up to 64),
    // 9, 16 or 32 candidate columns
    // (9 columns: the nine candidate sizes 8, 10, ..., 24 of the paper's setting; padding columns cost
    // a multiply-add each)
    const int nc = a.num_cand;
    if (a.jmax > 1 && a.jmax <= 24) {
        if (nc <= 9) return tau_launch<24, 9>(a, p, dev, stream);
        return nc <= 16 ? tau_launch<24, 16>(a, p, dev, stream) : tau_launch<24, 32>(a, p, dev, stream);
    }
    if (a.jmax > 1 && a.jmax <= 32) {
        if (nc <= 9) return tau_launch<32, 9>(a, p, dev, stream);
        return nc <= 16 ? tau_launch<32, 16>(a, p, dev, stream) : tau_launch<32, 32>(a, p, dev, stream);
    }
    if (nc <= 9) return tau_launch<64, 9>(a, p, dev, stream);
    return nc <= 16 ? tau_launch<64, 16>(a, p, dev, stream) : tau_launch<64, 32>(a, p, dev, stream);
}

}  // namespace bp
