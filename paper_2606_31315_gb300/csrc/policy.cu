// Block-size policy head (Sections 2.3-2.4 of the BlockPilot paper): once per request,
//   h = max(0, W1 x + b1),  o = W2 h + b2,  block size = candidates[argmax o].
//
// bf16 weights -- tensor cores (sm_103a), one launch:
//   * W1 [hidden x d_in] is cut into 128-row tiles; a thread-block cluster of KS CTAs splits one
//     tile's d_in into 64-column swizzle atoms.  Each CTA brings its W1 atoms in with TMA
//     (SWIZZLE_128B), gathers the requests' pooled rows x (row_index) into the matching
//     K-major layout, and one thread issues M=128 x N=requests tcgen05 MMAs (bf16 in, fp32
//     accumulated in tensor memory): W1 is read from HBM exactly once for up to 64 requests.
//   * The KS partial tiles are summed through distributed shared memory; each CTA takes a
//     share of the rows, adds b1 and applies ReLU, and folds its rows of h straight into the
//     output layer (W2 columns of those rows), so h never goes to global memory.
//   * The cluster's output-layer partials go to the workspace; the last tile to finish (an
//     atomic ticket, no waiting) adds them in tile order with b2 and takes the argmax (lowest
//     index on ties).  Every sum runs in a fixed order: the result is deterministic.
// fp32 weights (and bf16 shapes outside the tensor-core limits) -- CUDA cores:
//   kernel 1 streams W1 once for a group of up to 32 requests (rows staged in shared memory,
//   a warp per hidden row, fp32 accumulation, bias and ReLU fused into the store of h);
//   kernel 2 (one CTA per request) applies the output layer and takes the argmax.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <mutex>

#include "common.cuh"
#include "ptx_sm103.cuh"

namespace cg = cooperative_groups;

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

// ---------------------------------------------------------------- tensor-core path (bf16)
constexpr int kTcM = 128;          // hidden rows per tile: the MMA M
constexpr int kTcMaxN = 64;        // requests per group: the MMA N (padded to a multiple of 16)
constexpr int kTcAtom = 64;        // d_in columns per 128-byte swizzle atom
constexpr int kTcAtomBytes = kTcM * kTcAtom * 2;  // 16 KB of W1 per atom
constexpr int kTcMaxAtoms = 8;     // atoms per CTA when all of them are loaded at once
constexpr int kTcStages = 5;       // ring depth at most, when the atoms of a CTA are streamed (large d_in)
constexpr int kTcMaxKS = 9;        // CTAs per cluster (non-portable above 8)
constexpr int kTcThreads = 128;    // thread t = tile row t = TMEM lane t
constexpr uint32_t kTcTmemCols = 64;
constexpr int kTcMaxSmem = 200 * 1024;

struct PolicyTcParams {
    const __nv_bfloat16* feats;
    int64_t row_stride;
    const int32_t* row_index;
    int num_reqs, d_in, hidden, num_cand;
    int atoms_total, atoms_per_cta, tiles, npad;
    int w_bytes, x_bytes, h_bytes, op_bytes;  // dynamic shared-memory regions
    const float* b1;
    const __nv_bfloat16* w2;
    const float* b2;
    const int32_t* candidates;
    float* logits_out;
    int32_t* block_size_out;
    float* part;    // [groups][tiles][kTcMaxN][num_cand] output-layer partials of each tile
    int* counters;  // [groups] tickets, zero between calls
    unsigned int* err;
};

__device__ __forceinline__ int atomic_add_acq_rel_gpu(int* addr, int v) {
    int old;
    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], %2;" : "=r"(old) : "l"(addr), "r"(v) : "memory");
    return old;
}

// Gathers the pooled rows of every request group into a contiguous [groups*64][d_in] buffer (rows
// past the last request zero), so that the streamed path can load x with TMA like W1.
__global__ void __launch_bounds__(256) policy_gather_kernel(const __nv_bfloat16* __restrict__ feats,
                                                            int64_t row_stride, const int32_t* __restrict__ row_index,
                                                            int num_reqs, int d_in, int groups, int npad,
                                                            __nv_bfloat16* __restrict__ xg) {
    griddep_launch_dependents();
    griddep_wait();
    const int chunks = d_in / 8;
    const long long total = (long long)groups * npad * chunks;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx % chunks);
        const long long gn = idx / chunks;
        const int n = (int)(gn % npad), g = (int)(gn / npad);
        const int req = g * kTcMaxN + n;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (req < num_reqs) {
            const long long row = row_index ? (long long)row_index[req] : (long long)req;
            v = *reinterpret_cast<const uint4*>(feats + row * row_stride + c * 8);
        }
        *reinterpret_cast<uint4*>(xg + (size_t)req * d_in + c * 8) = v;
    }
}

// RING = false: every W1 and x atom of the CTA is loaded at once (x gathered by the CTA itself).
// RING = true: the atoms stream through a ring of S stages of one atom (W1 and the gathered x by TMA),
// for any d_in; thread 0 produces, thread 32 issues the MMAs.  S is compile-time: the producer and the
// issuer are single threads on the critical path of every stage (with S and the atoms per stage as
// runtime values the same ring ran 127.0 instead of 116.8 us at 32 requests x 151936 -> 2048; two
// atoms per stage at half the depth, 256-byte row fetches, measured 127.4 us).
template <bool RING, int S>
__global__ void __launch_bounds__(kTcThreads) policy_tc_kernel(const __grid_constant__ CUtensorMap w1map,
                                                              const __grid_constant__ CUtensorMap xmap,
                                                              const PolicyTcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sW = base;                                         // W1 atoms, later the partial tile
    uint8_t* sX = base + p.w_bytes;                             // x atoms
    float* hs = reinterpret_cast<float*>(sX + p.x_bytes);       // h of the owned rows [rows][npad]
    float* op = reinterpret_cast<float*>(sX + p.x_bytes + p.h_bytes);  // output-layer partial [n][c]
    float* w2s = op + p.op_bytes / 4;  // W2 columns of the owned rows [c][row]
    __shared__ float b1s[kTcM], b2s[64];
    __shared__ int cands[64];
    __shared__ long long row_sh[kTcMaxN];  // feature row of each request of the group
    __shared__ uint64_t bar_w[kTcMaxAtoms], bar_mma;  // one-shot: an atom's landing; ring: full stages
    __shared__ uint64_t bar_empty[kTcStages];
    __shared__ uint32_t tmem_sh;
    __shared__ int last_sh;

    cg::cluster_group cluster = cg::this_cluster();
    const int KS = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x, warp = tid >> 5;
    const int tile = blockIdx.x / KS, g = blockIdx.y;
    const int m0 = tile * kTcM, n0 = g * kTcMaxN;
    const int ng = min(kTcMaxN, p.num_reqs - n0);
    const int npad = p.npad;
    const int a0 = rank * p.atoms_per_cta;
    const int na = max(0, min(p.atoms_total, a0 + p.atoms_per_cta) - a0);
    const int C = p.num_cand;
    const int rpr = (kTcM + KS - 1) / KS;  // rows of the tile owned by each CTA after the split-K sum
    const int rb = rank * rpr;
    const int nr = max(0, min(kTcM, rb + rpr) - rb);

    cluster_arrive_relaxed();  // peers must be running before any distributed shared memory access
    if (tid == 0) {
        prefetch_tensormap(&w1map);
        if (RING) prefetch_tensormap(&xmap);
        const int nb = RING ? S : na;
        for (int a = 0; a < nb; ++a) mbar_init(&bar_w[a], 1);
        if (RING)
            for (int st = 0; st < S; ++st) mbar_init(&bar_empty[st], 1);
        mbar_init(&bar_mma, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(&tmem_sh, kTcTmemCols);
        tmem_relinquish();
    }
    griddep_launch_dependents();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    griddep_wait();  // inputs may come from the previous kernel on the stream
    if (RING) {
        static_assert(!RING || (S >= 2 && S <= kTcStages && S <= kTcMaxAtoms), "ring depth");
        const uint32_t stage_bytes = (uint32_t)(kTcAtomBytes + npad * 128);
        if (tid == 0) {  // producer: W1 and x atoms through the ring
            int j = 0;
            for (; j < na; ++j) {
                const int st = j % S;
                if (j >= S && !mbar_wait(&bar_empty[st], ((j / S) - 1) & 1, kWaitBudget)) {
                    raise_error(p.err, kErrTimeout);
                    break;
                }
                mbar_arrive_expect_tx(&bar_w[st], stage_bytes);
                tma_load_2d(sW + st * kTcAtomBytes, &w1map, &bar_w[st], (a0 + j) * kTcAtom, m0);
                tma_load_2d(sX + st * npad * 128, &xmap, &bar_w[st], (a0 + j) * kTcAtom, n0);
            }
            if (j < na)  // wound down early: the copies still in flight land before the CTA moves on
                for (int jj = max(0, j - S); jj < j; ++jj) mbar_wait(&bar_w[jj % S], (jj / S) & 1, kDrainBudget);
        } else if (tid == 32) {  // MMA issuer
            if (na > 0) {
                const uint32_t idesc = idesc_bf16_f32(kTcM, npad, false, false);
                bool ok = true;
                for (int j = 0; j < na; ++j) {
                    const int st = j % S;
                    if (!mbar_wait(&bar_w[st], (j / S) & 1, kWaitBudget)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t wa = smem_addr(sW + st * kTcAtomBytes), xa = smem_addr(sX + st * npad * 128);
#pragma unroll
                    for (int kk = 0; kk < kTcAtom / 16; ++kk)
                        umma_ss(tmem, smem_desc(wa + kk * 32, 16, 1024, kSwizzle128B),
                                smem_desc(xa + kk * 32, 16, 1024, kSwizzle128B), idesc, (j | kk) ? 1u : 0u);
                    umma_commit(&bar_empty[st]);  // the stage is free once these MMAs have read it
                }
                if (!ok) raise_error(p.err, kErrTimeout);
                umma_commit(&bar_mma);
            }
        } else if (warp >= 2) {  // the small operands of the epilogue, while the ring runs
            const int t = tid - 64;
            for (int i = t; i < C * nr; i += kTcThreads - 64) {
                const int c = i / nr, rr = i % nr;
                const int j = m0 + rb + rr;
                w2s[c * rpr + rr] = j < p.hidden ? __bfloat162float(p.w2[(size_t)c * p.hidden + j]) : 0.f;
            }
            for (int rr = t; rr < nr; rr += kTcThreads - 64) b1s[rr] = m0 + rb + rr < p.hidden ? p.b1[m0 + rb + rr] : 0.f;
            if (rank == 0)
                for (int c = t; c < C; c += kTcThreads - 64) {
                    b2s[c] = p.b2[c];
                    cands[c] = p.candidates[c];
                }
        }
        __syncthreads();  // the epilogue operands
    } else {
        if (tid < ng) row_sh[tid] = p.row_index ? (long long)p.row_index[n0 + tid] : (long long)(n0 + tid);
        if (tid == 0)
            for (int a = 0; a < na; ++a) {
                mbar_arrive_expect_tx(&bar_w[a], kTcAtomBytes);
                tma_load_2d(sW + a * kTcAtomBytes, &w1map, &bar_w[a], (a0 + a) * kTcAtom, m0);
            }
        __syncthreads();  // row_sh
        // x of the group, K-major SWIZZLE_128B: atom a holds rows n of 128 bytes, 16-byte chunk c of
        // row n stored at chunk c ^ (n & 7); rows past the group and columns past d_in are zero.
        // Asynchronous 16-byte copies: every copy of a thread is in flight at once.
        for (int idx = tid; idx < npad * na * 8; idx += kTcThreads) {
            const int n = idx / (na * 8), rem = idx % (na * 8);
            const int a = rem >> 3, c = rem & 7;
            const int k = (a0 + a) * kTcAtom + c * 8;
            const bool valid = n < ng && k < p.d_in;
            const long long row = valid ? row_sh[n] : 0;
            cp_async16(sX + a * npad * 128 + n * 128 + ((c ^ (n & 7)) << 4), p.feats + row * p.row_stride + (valid ? k : 0),
                       valid);
        }
        // the small operands of the epilogue, read while the copies are in flight
        for (int i = tid; i < C * nr; i += kTcThreads) {
            const int c = i / nr, rr = i % nr;
            const int j = m0 + rb + rr;
            w2s[c * rpr + rr] = j < p.hidden ? __bfloat162float(p.w2[(size_t)c * p.hidden + j]) : 0.f;
        }
        for (int rr = tid; rr < nr; rr += kTcThreads) b1s[rr] = m0 + rb + rr < p.hidden ? p.b1[m0 + rb + rr] : 0.f;
        if (rank == 0)
            for (int c = tid; c < C; c += kTcThreads) {
                b2s[c] = p.b2[c];
                cands[c] = p.candidates[c];
            }
        cp_async_wait_all();
        fence_proxy_async_smem();  // the MMAs read x through the async proxy
        __syncthreads();
        if (tid == 0 && na > 0) {
            const uint32_t idesc = idesc_bf16_f32(kTcM, npad, false, false);
            bool ok = true;
            for (int a = 0; a < na && ok; ++a) {
                if (!mbar_wait(&bar_w[a], 0, kWaitBudget)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t wa = smem_addr(sW + a * kTcAtomBytes), xa = smem_addr(sX + a * npad * 128);
#pragma unroll
                for (int kk = 0; kk < kTcAtom / 16; ++kk)
                    umma_ss(tmem, smem_desc(wa + kk * 32, 16, 1024, kSwizzle128B),
                            smem_desc(xa + kk * 32, 16, 1024, kSwizzle128B), idesc, (a | kk) ? 1u : 0u);
            }
            if (!ok) {  // every W1 atom's copy lands before the CTA moves on
                raise_error(p.err, kErrTimeout);
                for (int a = 0; a < na; ++a) mbar_wait(&bar_w[a], 0, kDrainBudget);
            }
            umma_commit(&bar_mma);
        }
    }
    // ---- this CTA's partial tile row (thread = row = TMEM lane)
    float d[kTcMaxN];
#pragma unroll
    for (int e = 0; e < kTcMaxN; ++e) d[e] = 0.f;
    if (na > 0) {
        if (!mbar_wait(&bar_mma, 0, kDrainBudget)) raise_error(p.err, kErrTimeout);
        tc_fence_after();
#pragma unroll
        for (int c0 = 0; c0 < kTcMaxN; c0 += 16) {
            if (c0 < npad) {  // uniform: npad is the same in every thread
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) d[c0 + e] = __uint_as_float(v[e]);
            }
        }
    }
    // the W1 atoms are consumed: the partial tile takes their place, rows npad + 4 floats apart
    // (an odd number of 16-byte chunks, so the row writes of 8 consecutive threads do not collide)
    float* pd = reinterpret_cast<float*>(sW);
    const int ldp = npad + 4;
#pragma unroll
    for (int c = 0; c < kTcMaxN / 4; ++c)
        if (4 * c < npad)
            *reinterpret_cast<float4*>(pd + tid * ldp + 4 * c) = make_float4(d[4 * c], d[4 * c + 1], d[4 * c + 2], d[4 * c + 3]);
    cluster_wait();  // every peer is running
    cluster_sync_all();  // partial tiles complete and visible
    // ---- owned rows: sum of the KS partials, + b1, ReLU
    for (int item = tid; item < nr * (npad / 4); item += kTcThreads) {
        const int rr = item / (npad / 4), c4 = item % (npad / 4);
        const int row = rb + rr;
        const float4* src = reinterpret_cast<const float4*>(pd + row * ldp + 4 * c4);
        float4 v[kTcMaxKS];  // every remote load in flight at once, then summed in rank order
#pragma unroll
        for (int pr = 0; pr < kTcMaxKS; ++pr)
            v[pr] = pr < KS ? *cluster.map_shared_rank(src, pr) : make_float4(0.f, 0.f, 0.f, 0.f);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int pr = 0; pr < kTcMaxKS; ++pr) {
            acc.x += v[pr].x;
            acc.y += v[pr].y;
            acc.z += v[pr].z;
            acc.w += v[pr].w;
        }
        const int j = m0 + row;
        float4 h = make_float4(0.f, 0.f, 0.f, 0.f);
        if (j < p.hidden) {
            const float bj = b1s[rr];
            h = make_float4(fmaxf(0.f, acc.x + bj), fmaxf(0.f, acc.y + bj), fmaxf(0.f, acc.z + bj),
                            fmaxf(0.f, acc.w + bj));
        }
        *reinterpret_cast<float4*>(hs + rr * npad + 4 * c4) = h;
    }
    __syncthreads();
    // ---- the owned rows' share of the output layer: op[n][c] = sum_j W2[c][j] h[j][n]
    for (int item = tid; item < ng * C; item += kTcThreads) {
        const int n = item / C, c = item % C;
        const float* w2r = w2s + c * rpr;
        float acc = 0.f;
        for (int rr = 0; rr < nr; ++rr) acc = fmaf(w2r[rr], hs[rr * npad + n], acc);  // zero past hidden
        op[item] = acc;
    }
    cluster_sync_all();  // every CTA's share visible to rank 0
    if (rank == 0) {
        float* dst = p.part + ((size_t)g * p.tiles + tile) * (kTcMaxN * C);
        for (int item = tid; item < ng * C; item += kTcThreads) {
            float v[kTcMaxKS];
#pragma unroll
            for (int pr = 0; pr < kTcMaxKS; ++pr) v[pr] = pr < KS ? *cluster.map_shared_rank(op + item, pr) : 0.f;
            float sum = 0.f;
#pragma unroll
            for (int pr = 0; pr < kTcMaxKS; ++pr) sum += v[pr];
            dst[item] = sum;
        }
        // the CTA barrier orders every thread's partial before thread 0's release (cumulative); its
        // acquire makes the other tiles' partials visible to this CTA once it holds the last ticket
        __syncthreads();
        if (tid == 0) last_sh = atomic_add_acq_rel_gpu(p.counters + g, 1) == p.tiles - 1;
        __syncthreads();
        if (last_sh) {
            // every tile has published: logits in tile order, then the argmax per request
            float* logits = hs;  // this CTA's h is no longer needed (ng * C <= npad * rpr floats)
            const float* base = p.part + (size_t)g * p.tiles * (kTcMaxN * C);
            constexpr int kItems = 3;  // items per thread per round: 48 loads in flight
            for (int i0 = 0; i0 < ng * C; i0 += kItems * kTcThreads) {
                for (int t0 = 0; t0 < p.tiles; t0 += 16) {
                    float v[kItems][16];
#pragma unroll
                    for (int k = 0; k < kItems; ++k) {
                        const int item = i0 + tid + k * kTcThreads;
#pragma unroll
                        for (int u = 0; u < 16; ++u)
                            v[k][u] = item < ng * C && t0 + u < p.tiles
                                          ? __ldcg(base + (size_t)(t0 + u) * (kTcMaxN * C) + item) : 0.f;
                    }
#pragma unroll
                    for (int k = 0; k < kItems; ++k) {
                        const int item = i0 + tid + k * kTcThreads;
                        if (item < ng * C) {
                            float sum = t0 == 0 ? b2s[item % C] : logits[item];
#pragma unroll
                            for (int u = 0; u < 16; ++u) sum += v[k][u];  // tile order
                            logits[item] = sum;
                        }
                    }
                }
            }
            if (p.logits_out)  // the same items as above: each thread reads back its own sums
                for (int item = tid; item < ng * C; item += kTcThreads)
                    p.logits_out[(size_t)n0 * C + item] = logits[item];
            __syncthreads();
            for (int n = tid; n < ng; n += kTcThreads) {
                int best = 0;
                for (int c = 1; c < C; ++c)
                    if (logits[n * C + c] > logits[n * C + best]) best = c;
                p.block_size_out[n0 + n] = cands[best];
            }
            if (tid == 0) p.counters[g] = 0;  // ready for the next call
        }
    }
    cluster_sync_all();  // no CTA leaves while a peer may still read its shared memory
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, kTcTmemCols);
}

// Scratch of the tensor-core path: partials and tickets (after the CUDA-core path's h buffer).
size_t tc_part_bytes(int num_reqs, int hidden, int num_cand) {
    const size_t groups = ((size_t)num_reqs + kTcMaxN - 1) / kTcMaxN;
    const size_t tiles = ((size_t)hidden + kTcM - 1) / kTcM;
    return align_up(sizeof(float) * groups * tiles * kTcMaxN * (size_t)num_cand, 256) +
           align_up(sizeof(int) * groups, 256);
}
// The gathered x of the streamed path: [groups * 64][d_in] bf16.
size_t tc_x_bytes(int num_reqs, int d_in) {
    const size_t groups = ((size_t)num_reqs + kTcMaxN - 1) / kTcMaxN;
    return align_up(groups * kTcMaxN * (size_t)d_in * 2, 256);
}

// The instantiations: the one-shot kernel, then the rings, deepest first (the order of preference).
using TcFn = void (*)(CUtensorMap, CUtensorMap, PolicyTcParams);
struct TcKernel {
    TcFn fn;
    int stages;
};
constexpr int kTcRings = 4;
const TcKernel kTcKernels[1 + kTcRings] = {{policy_tc_kernel<false, 1>, 0}, {policy_tc_kernel<true, 5>, 5},
                                           {policy_tc_kernel<true, 4>, 4}, {policy_tc_kernel<true, 3>, 3},
                                           {policy_tc_kernel<true, 2>, 2}};

// Opt-in shared memory and non-portable cluster sizes, once per device.
int configure_tc(int device) {
    static std::mutex mu;
    static bool configured[64] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (device >= 0 && device < 64 && configured[device]) return BP_OK;
    for (const TcKernel k : kTcKernels)
        if (cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcMaxSmem) != cudaSuccess ||
            cudaFuncSetAttribute(k.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
            return BP_ERR_CUDA;
    if (device >= 0 && device < 64) configured[device] = true;
    return BP_OK;
}

// Clusters of ks streaming CTAs with smem bytes of dynamic shared memory each that the device holds at
// once (cached per device, cluster size and size).  The occupancy query counts clusters at one CTA per
// SM (on this GB300 it answers 15 nine-CTA clusters at every size); clusters also share SMs when the
// shared memory lets several CTAs fit, so its count is scaled by the CTAs per SM (measured: 16 such
// clusters ran at once at two CTAs per SM, not at one).
int active_ring_clusters(int device, int ks, int smem) {
    struct Entry {
        int device, ks, smem, n;
    };
    static std::mutex mu;
    static Entry cache[64];
    static int used = 0;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < used; ++i)
        if (cache[i].device == device && cache[i].ks == ks && cache[i].smem == smem) return cache[i].n;
    cudaLaunchConfig_t probe = {};
    cudaLaunchAttribute pa[1];
    probe.gridDim = dim3((unsigned)ks, 1, 1);
    probe.blockDim = dim3(kTcThreads, 1, 1);
    probe.dynamicSmemBytes = (size_t)smem;
    pa[0].id = cudaLaunchAttributeClusterDimension;
    pa[0].val.clusterDim.x = (unsigned)ks;
    pa[0].val.clusterDim.y = 1;
    pa[0].val.clusterDim.z = 1;
    probe.attrs = pa;
    probe.numAttrs = 1;
    int n = 0, per_sm = 0, reserved = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kTcKernels[1].fn, &probe) != cudaSuccess ||
        cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, device) != cudaSuccess ||
        cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, device) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    const int ctas_per_sm = per_sm / (smem + reserved);
    n *= ctas_per_sm > 1 ? ctas_per_sm : 1;
    if (used < 64) cache[used++] = Entry{device, ks, smem, n};
    return n;
}

// Launches the tensor-core path; returns -1 when the shape is outside its limits.
int run_tc(const PolicyArgs& a, const DeviceInfo& dev, float* part, int* counters, __nv_bfloat16* xg,
           cudaStream_t stream) {
    if (reinterpret_cast<uintptr_t>(a.w1) % 16 != 0 || a.num_cand > 64) return -1;
    const int atoms_total = (a.d_in + kTcAtom - 1) / kTcAtom;
    const int tiles = (a.hidden + kTcM - 1) / kTcM;
    const int groups = (a.num_reqs + kTcMaxN - 1) / kTcMaxN;
    const int npad = ((a.num_reqs < kTcMaxN ? a.num_reqs : kTcMaxN) + 15) / 16 * 16;
    // split d_in over as many CTAs as one wave of SMs holds, kTcMaxKS at most
    int ks = dev.sm_count / (tiles * groups);
    ks = ks < 1 ? 1 : ks;
    ks = ks > kTcMaxKS ? kTcMaxKS : ks;
    ks = ks > atoms_total ? atoms_total : ks;
    const int per = (atoms_total + ks - 1) / ks;
    const bool ring = per > kTcMaxAtoms;  // too many atoms to hold at once: stream them
    const int pd_bytes = kTcM * (npad + 4) * 4;
    const int rpr = (kTcM + ks - 1) / ks;
    int h_bytes = rpr * npad * 4;
    const int lg_bytes = kTcMaxN * a.num_cand * 4;  // the last tile's logits reuse the h region
    h_bytes = h_bytes > lg_bytes ? h_bytes : lg_bytes;
    const int op_bytes = kTcMaxN * a.num_cand * 4;
    const int w2s_bytes = a.num_cand * rpr * 4;
    const auto smem_for = [&](int slots) {  // atoms held at once
        const int wb = slots * kTcAtomBytes > pd_bytes ? slots * kTcAtomBytes : pd_bytes;
        return 1024 + wb + slots * npad * 128 + h_bytes + op_bytes + w2s_bytes;
    };
    if (configure_tc(dev.device) != BP_OK) return BP_ERR_CUDA;
    // ring: the deepest under which every cluster of the grid is resident at once -- a cluster left for
    // a second wave streams its tile alone at a fraction of the bandwidth (measured at 64 requests x
    // 151936 -> 2048: 16 tiles of 9-CTA clusters took 200 us with the 5-stage ring at one CTA per SM);
    // if none, the deepest that fits
    int kernel = 0;  // index into kTcKernels
    if (ring) {
        for (int i = 1; i <= kTcRings; ++i) {
            const int sm = smem_for(kTcKernels[i].stages);
            if (sm > kTcMaxSmem) continue;
            if (kernel == 0) kernel = i;
            if (active_ring_clusters(dev.device, ks, sm) >= tiles * groups) {
                kernel = i;
                break;
            }
        }
        if (kernel == 0) return -1;
    }
    const int slots = ring ? kTcKernels[kernel].stages : per;
    const int w_bytes = slots * kTcAtomBytes > pd_bytes ? slots * kTcAtomBytes : pd_bytes;
    const int x_bytes = slots * npad * 128;
    const int smem = smem_for(slots);
    if (smem > kTcMaxSmem) return -1;

    CUtensorMap w1map, xmap;
    const cuuint64_t dims[2] = {(cuuint64_t)a.d_in, (cuuint64_t)a.hidden};
    const cuuint64_t strides[1] = {(cuuint64_t)a.d_in * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kTcAtom, (cuuint32_t)kTcM};
    if (encode_tensor_map(&w1map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a.w1), dims, strides, box,
                          CU_TENSOR_MAP_SWIZZLE_128B) != BP_OK)
        return -1;
    xmap = w1map;  // not read by the one-shot kernel
    if (ring) {
        const cuuint64_t xdims[2] = {(cuuint64_t)a.d_in, (cuuint64_t)groups * kTcMaxN};
        const cuuint32_t xbox[2] = {(cuuint32_t)kTcAtom, (cuuint32_t)npad};
        if (encode_tensor_map(&xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, xg, xdims, strides, xbox,
                              CU_TENSOR_MAP_SWIZZLE_128B) != BP_OK)
            return -1;
    }
    PolicyTcParams p;
    p.feats = static_cast<const __nv_bfloat16*>(a.feats);
    p.row_stride = a.row_stride;
    p.row_index = a.row_index;
    p.num_reqs = a.num_reqs;
    p.d_in = a.d_in;
    p.hidden = a.hidden;
    p.num_cand = a.num_cand;
    p.atoms_total = atoms_total;
    p.atoms_per_cta = per;
    p.tiles = tiles;
    p.npad = npad;
    p.w_bytes = w_bytes;
    p.x_bytes = x_bytes;
    p.h_bytes = h_bytes;
    p.op_bytes = op_bytes;
    p.b1 = a.b1;
    p.w2 = static_cast<const __nv_bfloat16*>(a.w2);
    p.b2 = a.b2;
    p.candidates = a.candidates;
    p.logits_out = a.logits_out;
    p.block_size_out = a.block_size_out;
    p.part = part;
    p.counters = counters;
    p.err = a.err_word;
    cudaLaunchAttribute pdl[1];
    pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    pdl[0].val.programmaticStreamSerializationAllowed = 1;
    if (ring) {
        const long long total = (long long)groups * npad * (a.d_in / 8);
        long long blocks = (total + 255) / 256;
        const long long cap = 4LL * dev.sm_count;
        cudaLaunchConfig_t gcfg = {};
        gcfg.gridDim = dim3((unsigned)(blocks < cap ? blocks : cap), 1, 1);
        gcfg.blockDim = dim3(256, 1, 1);
        gcfg.stream = stream;
        gcfg.attrs = pdl;
        gcfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&gcfg, policy_gather_kernel, p.feats, a.row_stride, a.row_index, a.num_reqs, a.d_in,
                               groups, npad, xg) != cudaSuccess)
            return BP_ERR_CUDA;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3((unsigned)(tiles * ks), (unsigned)groups, 1);
    cfg.blockDim = dim3(kTcThreads, 1, 1);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)ks;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1] = pdl[0];
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kTcKernels[kernel].fn, w1map, xmap, p);
    return e == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

template <typename T>
int run(const PolicyArgs& a, cudaStream_t stream) {
    float* hbuf = static_cast<float*>(a.scratch);
    const int max_group = kSmemBudget / (a.d_in * (int)sizeof(T));
    if (max_group < 1) return BP_ERR_UNSUPPORTED;
    const int group = max_group < kGroup ? max_group : kGroup;
    const int rows_per_block = (kThreads1 / 32) * kRowsPerWarp;
    const unsigned blocks = (unsigned)((a.hidden + rows_per_block - 1) / rows_per_block);
    static std::mutex cfg_mu;
    static bool configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return BP_ERR_CUDA;
    std::lock_guard<std::mutex> cfg_lock(cfg_mu);  // once per device, from any host thread
    if (!configured[dev]) {
        if (cudaFuncSetAttribute(policy_hidden_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget) !=
                cudaSuccess ||
            cudaFuncSetAttribute(policy_hidden_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared) != cudaSuccess ||
            cudaFuncSetAttribute(policy_out_kernel<T>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared) != cudaSuccess)
            return BP_ERR_CUDA;
        configured[dev] = true;
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

size_t policy_scratch_bytes(int num_reqs, int d_in, int hidden, int num_cand) {
    return align_up(sizeof(float) * (size_t)num_reqs * hidden, 256) + tc_part_bytes(num_reqs, hidden, num_cand) +
           tc_x_bytes(num_reqs, d_in);
}

int launch_policy(const PolicyArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    if (a.num_reqs == 0) return BP_OK;
    if (a.wdtype == BP_BF16) {
        uint8_t* w = static_cast<uint8_t*>(a.scratch) + align_up(sizeof(float) * (size_t)a.num_reqs * a.hidden, 256);
        float* part = reinterpret_cast<float*>(w);
        const size_t groups = ((size_t)a.num_reqs + kTcMaxN - 1) / kTcMaxN;
        const size_t tiles = ((size_t)a.hidden + kTcM - 1) / kTcM;
        int* counters = reinterpret_cast<int*>(w + align_up(sizeof(float) * groups * tiles * kTcMaxN * (size_t)a.num_cand, 256));
        __nv_bfloat16* xg = reinterpret_cast<__nv_bfloat16*>(w + tc_part_bytes(a.num_reqs, a.hidden, a.num_cand));
        const int rc = run_tc(a, dev, part, counters, xg, stream);
        if (rc != -1) return rc;
        return run<__nv_bfloat16>(a, stream);
    }
    return run<float>(a, stream);
}

}  // namespace bp
