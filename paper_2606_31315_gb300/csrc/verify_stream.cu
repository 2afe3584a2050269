// Verify epilogue for batches whose logits cannot stay on chip: the LM-head projection of the
// verified (and drafted) positions streamed through tensor memory, with every row's softmax
// statistics formed in the GEMM's epilogue, followed by the throughput acceptance.
//
// Section 2.1 / Figure 1: the target scores every drafted position in one pass and keeps the longest
// prefix the acceptance rule admits; the rule reads p = softmax(W h_t / T) and q = softmax(W h_d / T)
// over the whole vocabulary.  The resident kernel (verify_epilogue.cu) keeps a batch's whole
// [rows, V] accumulator in tensor memory, which bounds it to 64 rows: the GPU's tensor memory holds
// about 39 MB, and 248 rows of a 151,936-entry vocabulary take 151 MB in fp32.  Here:
//   1. lm_head_stream_kernel: one CTA per SM owns a contiguous run of 256-entry passes of the
//      vocabulary.  Per pass, its W rows (256 entries x 64 hidden columns per stage) and the states of
//      up to 256 rows stream through a TMA ring; one thread issues M=128 (state rows) x N=256 (entries)
//      x K=16 tcgen05 MMAs, one per 128-row half of the states.  Tensor-memory lane = state row, so each
//      epilogue thread owns one row and folds the pass's 256 logits into its row's running (max, sum of
//      2^(l*log2e/T - max)) -- at T = 0 its (max, lowest index) -- with one exponential per logit and no
//      exchange between threads.  At T > 0 it also writes the logits once (each warp's 32 x 32 chunk
//      staged in shared memory and sent by one TMA store): the draw at the first rejection needs a
//      whole row pair again, and no on-chip store can hold every row until the decisions are known.
//      At T = 0 nothing but the statistics leaves the chip.  Each CTA writes its slice's statistics
//      of every row.
//   2. lm_head_row_merge_kernel: one warp per row merges the slices' statistics in a fixed order.
//   3. The decisions and the draw of accept_batch.cu on those row statistics: only the draw's row pair
//      per sequence (and the logits at the drafted tokens) is read back.
// Rows beyond 256 go in groups of at most 256, one projection launch per group (W is read once per
// group).  Every wait is bounded; an expired wait sets the workspace error word and the kernel winds
// down after its own copies and MMAs have completed.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <limits.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "ptx_sm103.cuh"
#include "softmax_math.cuh"

namespace bp {
namespace {

constexpr int kVsN = 256;                // vocabulary entries per pass: the MMA N
constexpr int kVsWBytes = kVsN * 128;    // W of one stage: 256 entries x 128 bytes
constexpr int kVsM = 128;                // state rows per half: the MMA M, tensor-memory lanes
constexpr int kVsAtom = 64;              // hidden columns per 128-byte swizzle atom
constexpr int kVsHBytes = kVsM * 128;    // states of one stage and half: 128 rows x 128 bytes
constexpr int kVsThreads = 320;          // warps 0-7 epilogue, 8 TMA producer, 9 MMA issuer
constexpr int kVsEpiWarps = 8;
constexpr int kVsProducer = 8, kVsIssuer = 9;
constexpr int kVsMaxSlices = 160;        // slices (CTAs) per row in the statistics array

// MT halves of 128 state rows.  Tensor memory (512 columns) holds two passes' accumulators with one
// half -- the epilogue of one pass overlaps the MMAs of the next -- or one pass with two.  (Passes of
// 128 entries would let two halves double-buffer too, but the MMAs' operand reads and the ring's
// fills then ask more of shared memory per entry than it serves: measured slower.)  Stages
// of W and states together: 4 x 48 KB with one half, 3 x 64 KB with two; then the store staging.
__host__ __device__ constexpr int vs_stages(int MT) { return MT == 2 ? 3 : 4; }
constexpr int kVsStageBytes = 32 * 128;  // per epilogue warp: one chunk of 32 rows x 32 fp32 logits
template <int MT, bool WRITE>
constexpr size_t vs_smem_bytes() {
    return 1024 + (size_t)vs_stages(MT) * (kVsWBytes + MT * kVsHBytes) + (WRITE ? kVsEpiWarps * kVsStageBytes : 0);
}

struct VsParams {
    int vocab, atoms;
    int passes_base, passes_extra;  // CTA c: passes_base + (c < passes_extra) passes of 256 entries
    int nt, nt8, nd;                // the group's target rows, nt rounded up to 8, its drafter rows
    int ht0, hd0;                   // first target / drafter state of the group (TMA row coordinates)
    int row_t0, row_d0;             // their stacked rows (target rows first, then the drafter's)
    float c2;                       // log2(e) / T (0 at T = 0)
    float* logits;                  // [rows][vocab] fp32, or null
    int vec;                        // logits rows start 16-byte aligned
    int tma_store;                  // the group's rows are contiguous stacked rows: chunks go out by TMA
    int grows;                      // stacked rows of the group
    float2* part;                   // [rows][nslices] slice statistics
    int nslices;
    unsigned int* err;
};

// Named barrier among `count` threads (a multiple of 32) of the CTA.
__device__ __forceinline__ void named_barrier_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Stacked row of row `srow` of the group's state tile (-1: a padding row).
__device__ __forceinline__ int stacked_row(const VsParams& p, int srow) {
    if (srow < p.nt) return p.row_t0 + srow;
    return srow >= p.nt8 && srow < p.nt8 + p.nd ? p.row_d0 + (srow - p.nt8) : -1;
}

// The 32 logits of one chunk of columns folded into a row's running statistics; n valid entries.
// Four interleaved partial results shorten the dependency chains; they merge in a fixed order.
template <bool GREEDY>
__device__ __forceinline__ void fold_chunk(const uint32_t (&r)[32], int n, int v0, float c2, float& a0, float& a1) {
    if (GREEDY) {
        float bv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        int bi[4] = {INT_MAX, INT_MAX, INT_MAX, INT_MAX};
#pragma unroll
        for (int e = 0; e < 32; ++e) {  // increasing entries per partial: strict > keeps the lowest index
            const float l = __uint_as_float(r[e]);
            if (e < n && l > bv[e & 3]) {
                bv[e & 3] = l;
                bi[e & 3] = v0 + e;
            }
        }
        int ai = __float_as_int(a1);
#pragma unroll
        for (int k = 0; k < 4; ++k) amax_merge(a0, ai, bv[k], bi[k]);
        a1 = __int_as_float(ai);
    } else {
        float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int e = 0; e < 32; ++e)
            if (e < n) mx[e & 3] = fmaxf(mx[e & 3], __uint_as_float(r[e]));
        const float lm = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        const float mn = fmaxf(a0, __fmul_rn(lm, c2));
        float sm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int e = 0; e < 32; ++e)
            if (e < n) sm[e & 3] += ex2(__fmaf_rn(__uint_as_float(r[e]), c2, -mn));
        a1 = __fmaf_rn(a1, ex2d(a0, mn), (sm[0] + sm[1]) + (sm[2] + sm[3]));
        a0 = mn;
    }
}

// The warp's 32 rows x 32 entries of one chunk written to the logits.  Each lane puts its row into the
// warp's 4 KB staging buffer, 16-byte chunk i of row l at chunk i ^ (l & 7) -- the 128-byte swizzle of
// a TMA box of 32 rows x 32 fp32, and a layout in which neither row-wise writes nor column-wise reads
// conflict.  Where the group's rows are contiguous stacked rows (lmap: the group's rows of the logits),
// one TMA store sends the box and the warp goes on (it waits only, before the next chunk, until the
// copy has read the buffer); otherwise every store instruction covers whole 128-byte rows: four rows
// per 16-byte store, one per 4-byte store where rows are not 16-byte aligned.  srow0: the state-tile
// row of lane 0; n valid entries from v0.  Warp-collective.
__device__ __forceinline__ void store_chunk(uint8_t* stage, const uint32_t (&r)[32], int lane, int srow0,
                                            const VsParams& p, const CUtensorMap* lmap, int v0, int n) {
    if (p.tma_store) {
        if (lane == 0) bulk_wait_group_read<0>();  // the previous chunk's copy has read the buffer
        __syncwarp();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i)
        *reinterpret_cast<uint4*>(stage + lane * 128 + ((i ^ (lane & 7)) << 4)) =
            make_uint4(r[4 * i], r[4 * i + 1], r[4 * i + 2], r[4 * i + 3]);
    if (p.tma_store) {
        fence_proxy_async_smem();  // the copy reads the buffer through the async proxy
        __syncwarp();
        if (lane == 0 && srow0 < p.grows) {  // rows past the group, entries past the vocabulary: clipped
            tma_store_2d(lmap, stage, v0, srow0);
            bulk_commit_group();
        }
        return;
    }
    __syncwarp();
    if (p.vec && n == 32) {
        const int c = lane & 7;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int j = 4 * k + (lane >> 3);
            const int row = stacked_row(p, srow0 + j);
            const float4 x = *reinterpret_cast<const float4*>(stage + j * 128 + ((c ^ (j & 7)) << 4));
            if (row >= 0) __stcs(reinterpret_cast<float4*>(p.logits + (size_t)row * p.vocab + v0) + c, x);
        }
    } else {
#pragma unroll 4
        for (int j = 0; j < 32; ++j) {
            const int row = stacked_row(p, srow0 + j);
            const float x =
                *reinterpret_cast<const float*>(stage + j * 128 + (((lane >> 2) ^ (j & 7)) << 4) + ((lane & 3) << 2));
            if (row >= 0 && lane < n) __stcs(p.logits + (size_t)row * p.vocab + v0 + lane, x);
        }
    }
    __syncwarp();  // the buffer is free for the next chunk
}

template <bool GREEDY, int MT, bool WRITE>
__global__ void __launch_bounds__(kVsThreads, 1)
    lm_head_stream_kernel(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap htmap,
                          const __grid_constant__ CUtensorMap hdmap, const __grid_constant__ CUtensorMap lmap,
                          const VsParams p) {
    constexpr int STG = vs_stages(MT);
    constexpr int NB = 2 / MT;                     // accumulator buffers of MT x 256 columns
    constexpr int STAGE = kVsWBytes + MT * kVsHBytes;
    constexpr int CW = MT == 2 ? kVsN : kVsN / 2;  // columns (entries) per epilogue warp and pass
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sbase = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t full[STG], empty[STG], acc_full[NB], acc_empty[NB], mma_done;
    __shared__ uint32_t tmem_sh;
    __shared__ float2 half_sh[kVsM];              // MT = 1: the second column half's statistics per row

    griddep_launch_dependents();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int c = (int)blockIdx.x;
    const int npass = p.passes_base + (c < p.passes_extra ? 1 : 0);
    const int pass0 = c * p.passes_base + min(c, p.passes_extra);
    const int J = npass * p.atoms;  // ring stages of this CTA
    const uint32_t stage_tx = (uint32_t)(kVsWBytes + (p.nt + p.nd) * 128);

    if (tid == 0) {
        prefetch_tensormap(&wmap);
        if (p.nt) prefetch_tensormap(&htmap);
        if (p.nd) prefetch_tensormap(&hdmap);
        if (WRITE && p.tma_store) prefetch_tensormap(&lmap);
        for (int st = 0; st < STG; ++st) {
            mbar_init(&full[st], 1);
            mbar_init(&empty[st], 1);
        }
        for (int b = 0; b < NB; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], kVsEpiWarps);
        }
        mbar_init(&mma_done, 1);
        fence_mbar_init();
    }
    if (warp == kVsIssuer) {
        tmem_alloc(&tmem_sh, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;

    if (warp == kVsProducer) {
        // ---- TMA producer: stage j = (pass j / atoms, hidden atom j % atoms): 256 W rows, the group's states
        if (lane == 0) {
            int issued = 0;
            for (int j = 0; j < J; ++j) {
                const int st = j % STG;
                if (j >= STG && !mbar_wait(&empty[st], ((j / STG) - 1) & 1, kWaitBudget)) {
                    raise_error(p.err, kErrTimeout);
                    break;
                }
                const int pp = j / p.atoms, a = j - pp * p.atoms;
                uint8_t* sw = sbase + st * STAGE;
                uint8_t* sh = sw + kVsWBytes;
                mbar_arrive_expect_tx(&full[st], stage_tx);
                tma_load_2d(sw, &wmap, &full[st], a * kVsAtom, (pass0 + pp) * kVsN);
                if (p.nt) tma_load_2d(sh, &htmap, &full[st], a * kVsAtom, p.ht0);
                if (p.nd) tma_load_2d(sh + p.nt8 * 128, &hdmap, &full[st], a * kVsAtom, p.hd0);
                issued = j + 1;
            }
            if (issued < J)  // wound down early: let the copies still in flight land before exiting
                for (int j = max(0, issued - STG); j < issued; ++j)
                    mbar_wait(&full[j % STG], (j / STG) & 1, kDrainBudget);
        }
    } else if (warp == kVsIssuer) {
        // ---- MMA issuer: pass pp accumulates into buffer pp % NB; half m of the states into its own 256 columns
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(kVsM, kVsN, false, false);
            bool ok = true;
            int j = 0;
            for (int pp = 0; pp < npass && ok; ++pp) {
                const int b = pp % NB;
                if (pp >= NB && !mbar_wait(&acc_empty[b], ((pp / NB) - 1) & 1, kWaitBudget)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t dcol = tmem + (uint32_t)(b * MT * kVsN);
                for (int a = 0; a < p.atoms; ++a, ++j) {
                    const int st = j % STG;
                    if (!mbar_wait(&full[st], (j / STG) & 1, kWaitBudget)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t wa = smem_addr(sbase + st * STAGE), ha = wa + kVsWBytes;
#pragma unroll
                    for (int m = 0; m < MT; ++m)
#pragma unroll
                        for (int kk = 0; kk < kVsAtom / 16; ++kk)
                            umma_ss(dcol + (uint32_t)(m * kVsN),
                                    smem_desc(ha + m * kVsHBytes + kk * 32, 16, 1024, kSwizzle128B),
                                    smem_desc(wa + kk * 32, 16, 1024, kSwizzle128B), idesc, (a | kk) ? 1u : 0u);
                    umma_commit(&empty[st]);  // the stage is free once these MMAs have read it
                }
                if (ok) umma_commit(&acc_full[b]);
            }
            if (!ok) raise_error(p.err, kErrTimeout);
            umma_commit(&mma_done);  // every MMA issued is complete before tensor memory is released
            mbar_wait(&mma_done, 0, kDrainBudget);
        }
    } else {
        // ---- epilogue: thread = state row (tensor-memory lane); warp w reads lane quarter w % 4 of half
        // w / 4 (MT = 2: all 256 columns of a pass) or of the only half (MT = 1: column half w / 4)
        const int q = warp & 3, h = warp >> 2;
        const int m = MT == 2 ? h : 0, cb = MT == 2 ? 0 : h * CW;
        const int srow0 = m * kVsM + q * 32;  // state-tile row of lane 0
        const int row = stacked_row(p, srow0 + lane);
        float a0 = -INFINITY, a1 = GREEDY ? __int_as_float(INT_MAX) : 0.f;
        const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(m * kVsN + cb);
        uint8_t* stage = sbase + STG * STAGE + warp * kVsStageBytes;  // WRITE only
        bool ok = true;
        for (int pp = 0; pp < npass; ++pp) {
            const int b = pp % NB;
            ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[b], (pp / NB) & 1, kWaitBudget));
            if (!ok) break;
            tc_fence_after();
            const int vb = (pass0 + pp) * kVsN + cb;  // entry of the warp's first column
#pragma unroll 1
            for (int c0 = 0; c0 < CW; c0 += 64) {  // two chunks of 32 columns per wait
                uint32_t r0[32], r1[32];
                tmem_ld32(tq + (uint32_t)(b * MT * kVsN + c0), r0);
                tmem_ld32(tq + (uint32_t)(b * MT * kVsN + c0 + 32), r1);
                tmem_ld_wait();
                const int v0 = vb + c0, n0 = min(32, p.vocab - v0), n1 = min(32, p.vocab - v0 - 32);
                if (n0 > 0) {
                    if (WRITE) store_chunk(stage, r0, lane, srow0, p, &lmap, v0, n0);
                    if (row >= 0) fold_chunk<GREEDY>(r0, n0, v0, p.c2, a0, a1);
                }
                if (n1 > 0) {
                    if (WRITE) store_chunk(stage, r1, lane, srow0, p, &lmap, v0 + 32, n1);
                    if (row >= 0) fold_chunk<GREEDY>(r1, n1, v0 + 32, p.c2, a0, a1);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
        }
        if (WRITE && p.tma_store && lane == 0) bulk_wait_group<0>();  // this warp's logits are written
        if (!ok && lane == 0) raise_error(p.err, kErrTimeout);
        if (MT == 1) {  // the two column halves of a row, merged in entry order
            if (h == 1) half_sh[q * 32 + lane] = make_float2(a0, a1);
            named_barrier_sync(1, kVsEpiWarps * 32);
            if (h == 0) {
                const float2 o = half_sh[q * 32 + lane];
                if (GREEDY) {
                    int bi = __float_as_int(a1);
                    amax_merge(a0, bi, o.x, __float_as_int(o.y));
                    a1 = __int_as_float(bi);
                } else {
                    lse_merge(a0, a1, o.x, o.y);
                }
            }
        }
        if (row >= 0 && (MT == 2 || h == 0)) p.part[(size_t)row * p.nslices + c] = make_float2(a0, a1);
    }

    // ---- release tensor memory
    tc_fence_before();
    __syncthreads();
    if (warp == kVsIssuer) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// One warp per stacked row: the slices' statistics merged in a fixed order (each lane its slices in
// increasing order, then a butterfly), so every call gives bit-identical row statistics.
template <bool GREEDY>
__global__ void __launch_bounds__(256) lm_head_row_merge_kernel(const float2* __restrict__ part, int nslices,
                                                                int rows, float2* __restrict__ out) {
    griddep_launch_dependents();
    griddep_wait();
    const int r = (int)blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (r >= rows) return;
    constexpr int K = kVsMaxSlices / 32;
    float2 x[K];
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const int i = lane + 32 * k;
        x[k] = i < nslices ? __ldcg(&part[(size_t)r * nslices + i])
                           : make_float2(-INFINITY, GREEDY ? __int_as_float(INT_MAX) : 0.f);
    }
    float a0 = x[0].x, a1 = x[0].y;
    int ai = __float_as_int(a1);
#pragma unroll
    for (int k = 1; k < K; ++k) {
        if (GREEDY) amax_merge(a0, ai, x[k].x, __float_as_int(x[k].y));
        else lse_merge(a0, a1, x[k].x, x[k].y);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const float b0 = __shfl_xor_sync(0xffffffffu, a0, o);
        if (GREEDY) {
            amax_merge(a0, ai, b0, __shfl_xor_sync(0xffffffffu, ai, o));
        } else {
            const float b1 = __shfl_xor_sync(0xffffffffu, a1, o);
            lse_merge(a0, a1, b0, b1);
        }
    }
    if (lane == 0) out[r] = make_float2(a0, GREEDY ? __int_as_float(ai) : a1);
}

template <bool GREEDY, int MT, bool WRITE>
int vs_launch(const CUtensorMap& wmap, const CUtensorMap& htmap, const CUtensorMap& hdmap, const CUtensorMap& lmap,
              const VsParams& p, int grid, const DeviceInfo& dev, cudaStream_t stream) {
    static std::mutex cfg_mu;  // per instantiation (a template's own statics)
    static int configured[64] = {};
    const size_t smem = vs_smem_bytes<MT, WRITE>();
    if (dev.device >= 0 && dev.device < 64) {
        std::lock_guard<std::mutex> cfg_lock(cfg_mu);  // once per device, from any host thread
        if (!configured[dev.device]) {
            if (cudaFuncSetAttribute(lm_head_stream_kernel<GREEDY, MT, WRITE>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
                return BP_ERR_CUDA;
            configured[dev.device] = 1;
        }
    }
    lm_head_stream_kernel<GREEDY, MT, WRITE><<<grid, kVsThreads, smem, stream>>>(wmap, htmap, hdmap, lmap, p);
    return cudaGetLastError() == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

template <bool GREEDY>
int vs_dispatch(int mt, bool write, const CUtensorMap& wmap, const CUtensorMap& htmap, const CUtensorMap& hdmap,
                const CUtensorMap& lmap, const VsParams& p, int grid, const DeviceInfo& dev, cudaStream_t stream) {
    if (mt == 2)
        return write ? vs_launch<GREEDY, 2, true>(wmap, htmap, hdmap, lmap, p, grid, dev, stream)
                     : vs_launch<GREEDY, 2, false>(wmap, htmap, hdmap, lmap, p, grid, dev, stream);
    return write ? vs_launch<GREEDY, 1, true>(wmap, htmap, hdmap, lmap, p, grid, dev, stream)
                 : vs_launch<GREEDY, 1, false>(wmap, htmap, hdmap, lmap, p, grid, dev, stream);
}

int encode_rows(CUtensorMap* map, const void* base, int hidden, int rows, int box_rows) {
    const cuuint64_t dims[2] = {(cuuint64_t)hidden, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)hidden * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kVsAtom, (cuuint32_t)box_rows};
    return encode_tensor_map(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                             CU_TENSOR_MAP_SWIZZLE_128B);
}

}  // namespace

int verify_stream_grid(int vocab, int sm_count) {
    const int passes = (vocab + kVsN - 1) / kVsN;
    return min(min(sm_count, kVsMaxSlices), passes);
}

int launch_verify_stream(const VerifyEpilogueArgs& a, const VerifyStreamScratch& s, const DeviceInfo& dev,
                         cudaStream_t stream) {
    const bool greedy = a.temperature == 0.f;
    const int rows_t = a.total_draft + a.num_seqs;
    const int rows = rows_t + (greedy ? 0 : a.total_draft);
    float* logits = a.logits_out ? a.logits_out : (greedy ? nullptr : s.logits);
    const bool write = logits != nullptr;
    const int grid = verify_stream_grid(a.vocab, dev.sm_count);
    if (grid < 1 || a.hidden % kVsAtom != 0) return BP_ERR_UNSUPPORTED;

    const int passes = (a.vocab + kVsN - 1) / kVsN;
    CUtensorMap wmap, htmap, hdmap, lmap;
    if (encode_rows(&wmap, a.lm_head, a.hidden, a.vocab, kVsN) != BP_OK) return BP_ERR_CUDA;
    VsParams p;
    p.vocab = a.vocab;
    p.atoms = a.hidden / kVsAtom;
    p.passes_base = passes / grid;
    p.passes_extra = passes % grid;
    p.c2 = greedy ? 0.f : 1.4426950408889634f / a.temperature;
    p.logits = logits;
    p.vec = write && a.vocab % 4 == 0 && reinterpret_cast<uintptr_t>(logits) % 16 == 0;
    p.part = s.part;
    p.nslices = grid;
    p.err = a.err_word;
    // groups of at most 256 stacked rows; a group that holds both kinds keeps its drafter rows at an
    // 8-row boundary of the state tile (the 1024-byte swizzle atom), so it may hold a few rows less
    for (int r0 = 0; r0 < rows;) {
        int r1 = min(rows, r0 + 2 * kVsM);
        if (r0 < rows_t && r1 > rows_t) {
            const int nt = rows_t - r0, nt8 = (nt + 7) & ~7;
            if (nt8 + (r1 - rows_t) > 2 * kVsM) r1 -= nt8 - nt;
        }
        p.nt = max(0, min(r1, rows_t) - r0);
        p.nt8 = (p.nt + 7) & ~7;
        p.nd = max(0, r1 - max(r0, rows_t));
        p.ht0 = r0;
        p.row_t0 = r0;
        p.hd0 = max(r0, rows_t) - rows_t;
        p.row_d0 = max(r0, rows_t);
        if (p.nt && encode_rows(&htmap, a.h_target, a.hidden, rows_t, p.nt) != BP_OK) return BP_ERR_CUDA;
        if (p.nd && encode_rows(&hdmap, a.h_draft, a.hidden, a.total_draft, p.nd) != BP_OK) return BP_ERR_CUDA;
        const int mt = p.nt8 + p.nd > kVsM ? 2 : 1;
        // TMA stores where state-tile row i is stacked row r0 + i for every row the group holds
        p.tma_store = p.vec && (p.nt % 8 == 0 || p.nd == 0);
        p.grows = r1 - r0;
        if (p.tma_store) {
            const cuuint64_t dims[2] = {(cuuint64_t)a.vocab, (cuuint64_t)(r1 - r0)};
            const cuuint64_t strides[1] = {(cuuint64_t)a.vocab * 4};
            const cuuint32_t box[2] = {32, 32};
            if (encode_tensor_map(&lmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, logits + (size_t)r0 * a.vocab, dims,
                                  strides, box, CU_TENSOR_MAP_SWIZZLE_128B) != BP_OK)
                return BP_ERR_CUDA;
        }
        const CUtensorMap& ht = p.nt ? htmap : wmap;  // an unused map slot holds any valid map
        const CUtensorMap& hd = p.nd ? hdmap : wmap;
        const CUtensorMap& lm = p.tma_store ? lmap : wmap;
        const int rc = greedy ? vs_dispatch<true>(mt, write, wmap, ht, hd, lm, p, grid, dev, stream)
                              : vs_dispatch<false>(mt, write, wmap, ht, hd, lm, p, grid, dev, stream);
        if (rc != BP_OK) return rc;
        r0 = r1;
    }

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((rows + 7) / 8));
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const float2* part = s.part;
    const cudaError_t e = greedy ? cudaLaunchKernelEx(&cfg, lm_head_row_merge_kernel<true>, part, grid, rows, s.row_stats)
                                 : cudaLaunchKernelEx(&cfg, lm_head_row_merge_kernel<false>, part, grid, rows,
                                                      s.row_stats);
    if (e != cudaSuccess) return BP_ERR_CUDA;

    AcceptArgs aa;
    aa.target = logits;
    aa.draft = logits ? logits + (size_t)rows_t * a.vocab : nullptr;
    aa.tokens = a.tokens;
    aa.cu_draft = a.cu_draft;
    aa.num_seqs = a.num_seqs;
    aa.total_draft = a.total_draft;
    aa.vocab = a.vocab;
    aa.temperature = a.temperature;
    aa.u_accept = a.u_accept;
    aa.u_sample = a.u_sample;
    aa.n_accepted = a.n_accepted;
    aa.out_tokens = a.out_tokens;
    aa.accept_prob = a.accept_prob;
    aa.scratch = nullptr;
    aa.err_word = a.err_word;
    return launch_accept_rows(aa, s.row_stats, dev.sm_count, s.tickets, s.draw, stream);
}

}  // namespace bp
