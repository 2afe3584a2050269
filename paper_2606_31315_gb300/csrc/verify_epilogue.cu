// Fused verify epilogue: the LM-head projection of the verified positions (and of the drafter's
// positions) with the lossless acceptance of Section 2.1 applied to it on the fly.  The logits
// never leave the chip.
//
// Section 2.1 / Figure 1: the target scores every position of a drafted block in one pass and
// keeps the longest prefix the acceptance rule admits; that rule (standard speculative sampling:
// accept x_i with probability min(1, p_i(x_i) / q_i(x_i)), redraw from norm(max(0, p_k - q_k)) at
// the first rejection k, a bonus draw from p_gamma when every draft is accepted; greedy at T = 0)
// reads p = softmax(W h_t / T) and q = softmax(W h_d / T) over the whole vocabulary, W being the
// [V, H] LM head.  Unfused, the LM-head GEMM writes [rows, V] fp32 logits to HBM and the
// acceptance reads them back; here the GEMM's accumulators stay in tensor memory until the
// acceptance has used them, so the only HBM stream is W itself (read once).
//
// One persistent cooperative launch, one CTA per SM (every CTA co-resident):
//   * CTA c owns a contiguous slice of the vocabulary, at most 16 tiles of 128 LM-head rows.  Its
//     W rows stream once through an 8-stage TMA ring (one 128 x 64 bf16 box per stage, 128-byte
//     swizzle); warp 2 gathers the same 64 columns of every state row (target rows, then drafter
//     rows, zero rows up to NP) into the stage with 16-byte cp.async copies; one thread of warp 1
//     issues M=128 x N=NP x K=16 tcgen05 MMAs into the tile's own NP columns of tensor memory.
//   * Warps 4-7 read each finished tile (TMEM lane = vocabulary entry, column = row) while the next
//     one streams: every row's running max and sum of 2^(l*log2e/T - max) (T = 0: running argmax,
//     lowest index first), and the scaled logits at the draft tokens the slice holds.
//   * Grid barrier 1.  Every CTA merges the slices' statistics of every row in the same fixed
//     order, so all CTAs hold bit-identical normalisers, ratios a_i and first rejections k_s; CTA 0
//     writes n_accepted, the accepted drafts and accept_prob (T = 0: the emitted argmax too).
//   * T > 0: every CTA sums its slice's mass of max(0, p_k - q_k) (p_gamma for a bonus draw) per
//     sequence in exact 2^-52 fixed point; grid barrier 2; the CTA whose slice holds the crossing of
//     u_s * total recomputes its 32-entry chunks, finds the entry and writes the emitted token.
//   * The last CTA out clears the grid-barrier counters for the next call.
// Every wait is bounded; an expired wait sets the workspace error word and the kernel winds down.
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

constexpr int kVeM = 128;                        // vocabulary entries per tile: the MMA M, TMEM lanes
constexpr int kVeAtom = 64;                      // hidden columns per 128-byte swizzle atom
constexpr int kVeWBytes = kVeM * kVeAtom * 2;    // 16 KB of W per atom
constexpr int kVeMaxStages = 8;
constexpr int kVeLag = 2;                        // state copies kept in flight before a stage is published
constexpr int kVeThreads = 256;
constexpr int kVeEpi = 4;                        // first epilogue warp (lane quarter = warp % 4)
constexpr int kVeMaxTiles = 16;
constexpr int kVeMaxGrid = 160;

// Ring geometry: APS atoms (64 hidden columns each) per stage -- two atoms fetch 256 contiguous
// bytes of every W row at once, which HBM serves far better than 128 -- and as many stages as
// fit beside the states (NP rows per atom) in shared memory.
__host__ __device__ constexpr int ve_stages(int NP, int APS) { return APS == 1 ? 8 : (NP == 32 ? 5 : 4); }

struct VeParams {
    const __nv_bfloat16* h_target;  // [rows_t][hidden]
    const __nv_bfloat16* h_draft;   // [rows - rows_t][hidden]
    int hidden, vocab, atoms;
    int num_seqs, total_draft, rows_t, rows;
    int tiles_base, tiles_extra;    // CTA c: tiles_base + (c < tiles_extra) tiles
    uint32_t tmem_cols;
    float c2;                       // log2(e) / T
    const int32_t* tokens;
    const int32_t* cu_draft;
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    float* logits_out;              // [rows][vocab] or null
    float2* part;                   // [rows][grid] slice statistics (T = 0: value, index bits)
    float2* xg;                     // [total_draft] scaled (target, drafter) logits at the draft token
    ulonglong2* tot;                // [num_seqs][grid] slice masses of r and p, 2^-52 units
    unsigned int* sync;             // [0] grid-barrier arrivals, [1] exits; zero between calls
    unsigned int* err;
};

__device__ __forceinline__ void red_release_gpu(unsigned int* a, unsigned int v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(a), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned int ld_acquire_gpu(const unsigned int* a) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
    return v;
}
__device__ __forceinline__ unsigned int atom_add_acq_rel_gpu(unsigned int* a, unsigned int v) {
    unsigned int old;
    asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
    return old;
}
// Named barrier among `count` threads (a multiple of 32) of the CTA.
__device__ __forceinline__ void named_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void named_arrive(int id, int count) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Every CTA of the (co-resident) grid arrives, then waits until `target` arrivals are counted.
// False in every thread if they were not within the wait budget.  The CTA barrier orders the block's
// writes before thread 0's gpu-scope release, and its acquire before the block's later reads (release
// and acquire are cumulative): no separate fences.
__device__ bool grid_barrier(unsigned int* count, unsigned int target, int* ok_sh) {
    __syncthreads();
    if (threadIdx.x == 0) {
        red_release_gpu(count, 1u);
        const long long t0 = clock64();
        int ok = 1;
        while (ld_acquire_gpu(count) < target) {
            if (clock64() - t0 > kWaitBudget) {
                ok = 0;
                break;
            }
            __nanosleep(64);
        }
        *ok_sh = ok;
    }
    __syncthreads();
    return *ok_sh != 0;
}

// Value of column `col` among the NP columns a thread loaded (a select chain: no dynamic indexing).
template <int NP>
__device__ __forceinline__ float pick(const uint32_t (&r)[NP], int col) {
    float x = 0.f;
#pragma unroll
    for (int e = 0; e < NP; ++e)
        if (e == col) x = __uint_as_float(r[e]);
    return x;
}

// Lane `lane` ends with the warp-wide merge of column `lane` of the (max, sum) pairs: a butterfly
// that halves the columns it carries at every step (31 exchanges).
__device__ __forceinline__ float2 lse_reduce_scatter32(float (&m)[32], float (&s)[32], int lane) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int j = 0; j < o; ++j) {
            const float sm = up ? m[j] : m[j + o], ss = up ? s[j] : s[j + o];
            float km = up ? m[j + o] : m[j], ks = up ? s[j + o] : s[j];
            lse_merge(km, ks, __shfl_xor_sync(0xffffffffu, sm, o), __shfl_xor_sync(0xffffffffu, ss, o));
            m[j] = km;
            s[j] = ks;
        }
    }
    return make_float2(m[0], s[0]);
}
// The same for (value, index) argmax pairs.
__device__ __forceinline__ float2 amax_reduce_scatter32(float (&v)[32], int (&ix)[32], int lane) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int j = 0; j < o; ++j) {
            const float sv = up ? v[j] : v[j + o];
            const int si = up ? ix[j] : ix[j + o];
            float kv = up ? v[j + o] : v[j];
            int ki = up ? ix[j + o] : ix[j];
            amax_merge(kv, ki, __shfl_xor_sync(0xffffffffu, sv, o), __shfl_xor_sync(0xffffffffu, si, o));
            v[j] = kv;
            ix[j] = ki;
        }
    }
    return make_float2(v[0], __int_as_float(ix[0]));
}

// Weights of this lane's entry in tile t of the slice for one sequence's draw: x.x = r = max(0, p - q)
// (0 without a draft row), x.y = p.  The crossing search recomputes them with this same code.
struct DrawRow {
    int ct, cd;        // TMEM columns of the target row and the drafter row (cd < 0: none)
    float Mt, izt, Md, izd;
};
__device__ __forceinline__ float2 draw_weights(float lt, float ld, const DrawRow& d, bool in_vocab, float c2) {
    if (!in_vocab) return make_float2(0.f, 0.f);
    const float pv = __fmul_rn(ex2(__fsub_rn(__fmul_rn(lt, c2), d.Mt)), d.izt);
    float rv = 0.f;
    if (d.cd >= 0) rv = fmaxf(0.f, __fsub_rn(pv, __fmul_rn(ex2(__fsub_rn(__fmul_rn(ld, c2), d.Md)), d.izd)));
    return make_float2(rv, pv);
}
template <int NP>
__device__ __forceinline__ float2 entry_weights(uint32_t tmem_q, int t, const DrawRow& d, bool in_vocab, float c2) {
    const uint32_t col = (uint32_t)(t * NP);
    const float lt = __uint_as_float(tmem_ld1(tmem_q + col + (uint32_t)d.ct));
    const float ld = d.cd >= 0 ? __uint_as_float(tmem_ld1(tmem_q + col + (uint32_t)d.cd)) : 0.f;
    tmem_ld_wait();
    return draw_weights(lt, ld, d, in_vocab, c2);
}

template <bool GREEDY, int NP, int APS>
__global__ void __launch_bounds__(kVeThreads, 1)
    verify_epilogue_kernel(const __grid_constant__ CUtensorMap wmap, const VeParams p) {
    constexpr int STG = ve_stages(NP, APS);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sW = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sH = sW + STG * APS * kVeWBytes;  // state rows of each stage: APS x NP rows of 128 bytes
    __shared__ uint64_t wfull[kVeMaxStages], hfull[kVeMaxStages], empty[kVeMaxStages], acc_full[kVeMaxTiles], mma_done;
    __shared__ uint32_t tmem_sh;
    __shared__ int ok_sh, own_n, find_sh, sel_sh;
    __shared__ float2 wst[4][64];      // per epilogue warp: statistics of each row over its lanes
    __shared__ float2 rst[64];         // statistics of each row over the whole vocabulary
    __shared__ int own_v[64], own_ct[64], own_cd[64], own_i[64];  // draft tokens held by the slice
    __shared__ int cu_sh[65], k_sh[64], tok_sh[64];
    __shared__ float ua_sh[64];
    __shared__ ulonglong2 wtot[4][64];
    __shared__ unsigned long long off_sh, base_sh;
    __shared__ int use_r_sh;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int c = (int)blockIdx.x, grid = (int)gridDim.x;
    const int ntile = p.tiles_base + (c < p.tiles_extra ? 1 : 0);
    const int tile0 = c * p.tiles_base + min(c, p.tiles_extra);
    const int v0 = tile0 * kVeM;                        // first vocabulary entry of the slice
    const int v1 = min(p.vocab, v0 + ntile * kVeM);
    const int spt = p.atoms / APS;                   // ring stages per tile
    const int J = ntile * spt;                          // ring stages of this CTA
    const int S = p.num_seqs;

    // stage j of the ring: atoms a0 .. a0 + APS - 1 of tile t, both found from j
    auto issue_w = [&](int j) {
        const int st = j % STG, t = j / spt, a0 = (j - t * spt) * APS;
        mbar_arrive_expect_tx(&wfull[st], APS * kVeWBytes);
#pragma unroll
        for (int u = 0; u < APS; ++u)
            tma_load_2d(sW + (st * APS + u) * kVeWBytes, &wmap, &wfull[st], (a0 + u) * kVeAtom, (tile0 + t) * kVeM);
    };
    const int j_first = min(STG, J);  // stages issued before the block-wide set-up completes
    if (tid == 0) {
        prefetch_tensormap(&wmap);
        for (int st = 0; st < STG; ++st) {
            mbar_init(&wfull[st], 1);
            mbar_init(&hfull[st], 1);
            mbar_init(&empty[st], 1);
        }
        for (int t = 0; t < kVeMaxTiles; ++t) mbar_init(&acc_full[t], 1);
        mbar_init(&mma_done, 1);
        fence_mbar_init();
        own_n = 0;
        for (int j = 0; j < j_first; ++j) issue_w(j);  // the W stream starts at once
    }
    if (warp == 1) {
        tmem_alloc(&tmem_sh, p.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;

    if (warp == 0) {
        // ---- W producer: the slice's LM-head rows, tile by tile, APS x 64 hidden columns per stage
        if (lane == 0) {
            int issued = j_first;
            for (int j = j_first; j < J; ++j) {
                const int st = j % STG;
                if (!mbar_wait(&empty[st], ((j / STG) - 1) & 1, kWaitBudget)) {
                    raise_error(p.err, kErrTimeout);
                    break;
                }
                issue_w(j);
                issued = j + 1;
            }
            if (issued < J)  // wound down early: let the copies still in flight land before exiting
                for (int j = max(0, issued - STG); j < issued; ++j)
                    mbar_wait(&wfull[j % STG], (j / STG) & 1, kDrainBudget);
        }
    } else if (warp == 2) {
        // ---- state producer: row n's 16-byte chunk ch of atom a goes to chunk ch ^ (n & 7) of row n
        int j = 0;
        for (; j < J; ++j) {
            const int st = j % STG;
            const bool ok = j < STG || mbar_wait(&empty[st], ((j / STG) - 1) & 1, kWaitBudget);
            if (!__all_sync(0xffffffffu, ok)) {
                if (lane == 0) raise_error(p.err, kErrTimeout);
                break;
            }
            const int a0 = (j % spt) * APS;
#pragma unroll
            for (int it = 0; it < APS * NP * 8 / 32; ++it) {
                const int idx = it * 32 + lane;
                const int u = idx / (NP * 8), n = (idx >> 3) % NP, ch = idx & 7;
                const int a = a0 + u;
                uint8_t* dst = sH + (st * APS + u) * (NP * 128);
                const bool valid = n < p.rows;
                const __nv_bfloat16* row = n < p.rows_t ? p.h_target + (size_t)n * p.hidden
                                                        : p.h_draft + (size_t)(valid ? n - p.rows_t : 0) * p.hidden;
                cp_async16(dst + n * 128 + ((ch ^ (n & 7)) << 4), valid ? row + a * kVeAtom + ch * 8 : p.h_target,
                           valid);
            }
            cp_async_commit();
            if (j >= kVeLag) {
                cp_async_wait_group<kVeLag>();
                fence_proxy_async_smem();  // the MMAs read the states through the async proxy
                __syncwarp();
                if (lane == 0) mbar_arrive(&hfull[(j - kVeLag) % STG]);
            }
        }
        cp_async_wait_group<0>();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0)
            for (int jj = max(0, j - kVeLag); jj < j; ++jj) mbar_arrive(&hfull[jj % STG]);
    } else if (warp == 1) {
        // ---- MMA issuer: tile t accumulates into TMEM columns [t * NP, t * NP + NP)
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(kVeM, NP, false, false);
            for (int j = 0; j < J; ++j) {
                const int st = j % STG;
                const uint32_t par = (j / STG) & 1;
                if (!mbar_wait(&wfull[st], par, kWaitBudget) || !mbar_wait(&hfull[st], par, kWaitBudget)) {
                    raise_error(p.err, kErrTimeout);
                    break;
                }
                tc_fence_after();
                const int t = j / spt, a0 = (j - t * spt) * APS;
#pragma unroll
                for (int u = 0; u < APS; ++u) {
                    const uint32_t wa = smem_addr(sW + (st * APS + u) * kVeWBytes);
                    const uint32_t ha = smem_addr(sH + (st * APS + u) * (NP * 128));
#pragma unroll
                    for (int kk = 0; kk < kVeAtom / 16; ++kk)
                        umma_ss(tmem + (uint32_t)(t * NP), smem_desc(wa + kk * 32, 16, 1024, kSwizzle128B),
                                smem_desc(ha + kk * 32, 16, 1024, kSwizzle128B), idesc, ((a0 + u) | kk) ? 1u : 0u);
                }
                umma_commit(&empty[st]);  // the stage is free once these MMAs have read it
                if (a0 + APS == p.atoms) umma_commit(&acc_full[t]);
            }
            umma_commit(&mma_done);  // every MMA issued is complete before tensor memory is released
            mbar_wait(&mma_done, 0, kDrainBudget);
        }
    } else if (warp == 3) {
        // ---- sequence offsets (read by every warp after grid barrier 1), then the draft tokens held
        // by this slice (their logits are captured by the epilogue)
        for (int i = lane; i <= S; i += 32) cu_sh[i] = p.cu_draft[i];
        for (int i = lane; i < p.total_draft; i += 32) {  // inputs of the decisions, read before they are due
            tok_sh[i] = p.tokens[i];
            ua_sh[i] = GREEDY ? 0.f : p.u_accept[i];
        }
        __syncwarp();
        if (!GREEDY) {
            for (int i = lane; i < p.total_draft; i += 32) {
                const int x = tok_sh[i];
                if (x >= v0 && x < v1) {
                    int lo = 0, hi = S;  // sequence of draft i: cu[lo] <= i < cu[lo + 1]
                    while (hi - lo > 1) {
                        const int mid = (lo + hi) >> 1;
                        if (cu_sh[mid] <= i) lo = mid; else hi = mid;
                    }
                    const int o = atomicAdd(&own_n, 1);
                    own_v[o] = x - v0;
                    own_i[o] = i;
                    own_ct[o] = i + lo;           // target row of draft i
                    own_cd[o] = p.rows_t + i;     // its drafter row
                }
            }
            __threadfence_block();
            named_arrive(2, 160);
        }
        if (c == 0)
            for (int i = lane; i < p.total_draft; i += 32) {
                const int x = tok_sh[i];
                if (x < 0 || x >= p.vocab) raise_error(p.err, kErrDeviceArg);
            }
    } else {
        // ---- epilogue: the running statistics of every row over this lane's entries, tile by tile
        const int q = warp & 3;
        const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16);
        float m[NP], s[NP];
        int ix[NP];
#pragma unroll
        for (int e = 0; e < NP; ++e) {
            m[e] = -INFINITY;
            s[e] = 0.f;
            ix[e] = INT_MAX;
        }
        int nown = 0;
        if (!GREEDY) {
            named_sync(2, 160);
            nown = own_n;
        }
        for (int t = 0; t < ntile; ++t) {
            if (!mbar_wait(&acc_full[t], 0, kWaitBudget)) {
                raise_error(p.err, kErrTimeout);
                break;
            }
            tc_fence_after();
            const int vl = t * kVeM + q * 32 + lane;  // entry within the slice
            const int v = v0 + vl;
#pragma unroll
            for (int h0 = 0; h0 < NP; h0 += 32) {  // 32 columns at a time
                if (h0 >= p.rows) break;
                uint32_t r[32];
                tmem_ld32(tq + (uint32_t)(t * NP + h0), r);
                tmem_ld_wait();
                if (v < v1) {
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        if (h0 + e < p.rows) {
                            const float l = __uint_as_float(r[e]);
                            if (GREEDY) {
                                if (l > m[h0 + e]) {  // entries arrive in increasing index: ties keep the first
                                    m[h0 + e] = l;
                                    ix[h0 + e] = v;
                                }
                            } else {
                                const float x = __fmul_rn(l, p.c2);
                                const float d = __fsub_rn(x, m[h0 + e]);
                                const float w = ex2(-fabsf(d));
                                s[h0 + e] = d > 0.f ? __fmaf_rn(s[h0 + e], w, 1.f) : __fadd_rn(s[h0 + e], w);
                                m[h0 + e] = fmaxf(m[h0 + e], x);
                            }
                            if (p.logits_out) p.logits_out[(size_t)(h0 + e) * p.vocab + v] = l;
                        }
                    }
                    for (int o = 0; o < nown; ++o)
                        if (own_v[o] == vl) {  // scaled logits of the draft token (each owned by one thread)
                            const int ct = own_ct[o] - h0, cd = own_cd[o] - h0;
                            if (ct >= 0 && ct < 32) p.xg[own_i[o]].x = __fmul_rn(pick<32>(r, ct), p.c2);
                            if (cd >= 0 && cd < 32) p.xg[own_i[o]].y = __fmul_rn(pick<32>(r, cd), p.c2);
                        }
                }
            }
        }
        // the statistics of every row over the warp's 32 lanes, then over the four warps
#pragma unroll
        for (int h0 = 0; h0 < NP; h0 += 32) {
            float2 res;
            if (GREEDY) {
                float vv[32];
                int ii[32];
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    vv[e] = m[h0 + e];
                    ii[e] = ix[h0 + e];
                }
                res = amax_reduce_scatter32(vv, ii, lane);
            } else {
                float mm[32], ss[32];
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    mm[e] = m[h0 + e];
                    ss[e] = s[h0 + e];
                }
                res = lse_reduce_scatter32(mm, ss, lane);
            }
            wst[q][h0 + lane] = res;
        }
        named_sync(1, 128);
        for (int r = tid - kVeEpi * 32; r < p.rows; r += 128) {
            float2 a = wst[0][r];
            for (int w = 1; w < 4; ++w) {
                if (GREEDY) {
                    int ai = __float_as_int(a.y);
                    amax_merge(a.x, ai, wst[w][r].x, __float_as_int(wst[w][r].y));
                    a.y = __int_as_float(ai);
                } else {
                    lse_merge(a.x, a.y, wst[w][r].x, wst[w][r].y);
                }
            }
            p.part[(size_t)r * grid + c] = a;
        }
    }

    // ================= grid barrier 1: every slice's statistics and draft-token logits are out
    if (!grid_barrier(p.sync, (unsigned)grid, &ok_sh)) raise_error(p.err, kErrTimeout);

    for (int sq = tid; sq < S; sq += kVeThreads) k_sh[sq] = cu_sh[sq + 1] - cu_sh[sq];  // no rejection yet
    // ---- row statistics over the whole vocabulary, merged in one fixed order in every CTA; a warp
    // takes rows warp, warp + 8, ... and keeps the loads of four rows in flight at once
    for (int r0 = warp; r0 < p.rows; r0 += 4 * (kVeThreads / 32)) {
        float2 x[4][kVeMaxGrid / 32];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int r = r0 + b * (kVeThreads / 32);
#pragma unroll
            for (int m = 0; m < kVeMaxGrid / 32; ++m) {
                const int cc = m * 32 + lane;
                const float2 none = make_float2(-INFINITY, GREEDY ? __int_as_float(INT_MAX) : 0.f);
                x[b][m] = (r < p.rows && cc < grid) ? __ldcg(&p.part[(size_t)r * grid + cc]) : none;
            }
        }
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int r = r0 + b * (kVeThreads / 32);
            float a0 = -INFINITY, a1 = 0.f;
            int ai = INT_MAX;
#pragma unroll
            for (int m = 0; m < kVeMaxGrid / 32; ++m) {
                if (GREEDY) amax_merge(a0, ai, x[b][m].x, __float_as_int(x[b][m].y));
                else lse_merge(a0, a1, x[b][m].x, x[b][m].y);
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) {
                const float b0 = __shfl_xor_sync(0xffffffffu, a0, o);
                if (GREEDY) {
                    amax_merge(a0, ai, b0, __shfl_xor_sync(0xffffffffu, ai, o));
                } else {
                    lse_merge(a0, a1, b0, __shfl_xor_sync(0xffffffffu, a1, o));
                }
            }
            if (lane == 0 && r < p.rows) rst[r] = GREEDY ? make_float2(a0, __int_as_float(ai)) : make_float2(a0, a1);
        }
    }
    __syncthreads();
    // ---- ratios of every drafted position (one thread each) and the first rejection of every
    // sequence (identical in every CTA)
    for (int i = tid; i < p.total_draft; i += kVeThreads) {
        int sq = 0, hi = S;  // sequence of draft i: cu[sq] <= i < cu[sq + 1]
        while (hi - sq > 1) {
            const int mid = (sq + hi) >> 1;
            if (cu_sh[mid] <= i) sq = mid; else hi = mid;
        }
        const int ct = i + sq;
        const int x = tok_sh[i];
        float a;
        if (GREEDY) {
            a = (x == __float_as_int(rst[ct].y)) ? 1.f : 0.f;
        } else if (x < 0 || x >= p.vocab) {
            a = 0.f;
        } else {
            const float2 xx = __ldcg(&p.xg[i]);
            const float2 st = rst[ct], sd = rst[p.rows_t + i];
            // a = min(1, p(x)/q(x)) in the log domain: 2^((xt - Mt) - (xd - Md)) * Zd / Zt
            const float lr = __fsub_rn(__fsub_rn(xx.x, st.x), __fsub_rn(xx.y, sd.x));
            a = fminf(1.f, ex2(lr) * __fdiv_rn(sd.y, st.y));
        }
        if (c == 0 && p.accept_prob) p.accept_prob[i] = a;
        const bool rej = GREEDY ? (a == 0.f) : !(ua_sh[i] < a);
        if (rej) atomicMin(&k_sh[sq], i - cu_sh[sq]);
    }
    __syncthreads();
    if (c == 0) {  // n_accepted, the accepted drafts, -1 past the emitted slot (T = 0: the emitted argmax)
        for (int sq = warp; sq < S; sq += kVeThreads / 32) {
            const int d0 = cu_sh[sq], g = cu_sh[sq + 1] - d0, k = k_sh[sq], t0 = d0 + sq;
            for (int j = lane; j <= g; j += 32) {
                if (j < k) p.out_tokens[t0 + j] = tok_sh[d0 + j];
                else if (j > k) p.out_tokens[t0 + j] = -1;
                else if (GREEDY) p.out_tokens[t0 + j] = __float_as_int(rst[t0 + k].y);
            }
            if (lane == 0) p.n_accepted[sq] = k;
        }
    }

    if (!GREEDY) {
        // ---- this slice's mass of each sequence's draw distribution, exact fixed point; the masses of
        // its 32-entry chunks are kept (in the ring's shared memory, idle now) for the crossing search
        ulonglong2* chunk = reinterpret_cast<ulonglong2*>(sW);  // [sequence][tile][lane quarter]
        const int q = warp & 3;
        const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16);
        if (warp >= kVeEpi) {
            for (int sq = 0; sq < S; ++sq) {
                const int d0 = cu_sh[sq], g = cu_sh[sq + 1] - d0, k = k_sh[sq];
                DrawRow d;
                d.ct = d0 + sq + k;
                d.cd = k < g ? p.rows_t + d0 + k : -1;
                d.Mt = rst[d.ct].x;
                d.izt = __fdiv_rn(1.f, rst[d.ct].y);
                d.Md = d.cd >= 0 ? rst[d.cd].x : 0.f;
                d.izd = d.cd >= 0 ? __fdiv_rn(1.f, rst[d.cd].y) : 0.f;
                // every tile's two columns first (one wait), then the weights of this lane's entries
                uint32_t rt[kVeMaxTiles], rd[kVeMaxTiles];
#pragma unroll
                for (int t = 0; t < kVeMaxTiles; ++t) {
                    if (t < ntile) {
                        rt[t] = tmem_ld1(tq + (uint32_t)(t * NP + d.ct));
                        rd[t] = d.cd >= 0 ? tmem_ld1(tq + (uint32_t)(t * NP + d.cd)) : 0u;
                    }
                }
                tmem_ld_wait();
                // lane t ends with the r-mass of tile t's chunk, lane 16 + t with its p-mass (31 shuffles)
                float v[32];
#pragma unroll
                for (int t = 0; t < kVeMaxTiles; ++t) {
                    float2 w = make_float2(0.f, 0.f);
                    if (t < ntile)
                        w = draw_weights(__uint_as_float(rt[t]), __uint_as_float(rd[t]), d,
                                         v0 + t * kVeM + q * 32 + lane < v1, p.c2);
                    v[t] = w.x;
                    v[kVeMaxTiles + t] = w.y;
                }
                const unsigned long long f = to_fix(reduce_scatter32(v, lane));
                const int tl = lane & (kVeMaxTiles - 1);
                unsigned long long* cf = reinterpret_cast<unsigned long long*>(chunk);
                if (tl < ntile) cf[((sq * ntile + tl) * 4 + q) * 2 + (lane >> 4)] = f;  // .x = r, .y = p
                unsigned long long tot = tl < ntile ? f : 0ull;  // lanes 0-15 sum r, lanes 16-31 sum p
#pragma unroll
                for (int o = kVeMaxTiles / 2; o >= 1; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
                if (lane == 0) wtot[q][sq].x = tot;
                if (lane == kVeMaxTiles) wtot[q][sq].y = tot;
            }
            named_sync(1, 128);
            for (int sq = tid - kVeEpi * 32; sq < S; sq += 128) {
                ulonglong2 a = wtot[0][sq];
                for (int w = 1; w < 4; ++w) {
                    a.x += wtot[w][sq].x;
                    a.y += wtot[w][sq].y;
                }
                p.tot[(size_t)sq * grid + c] = a;
            }
        }

        // ================= grid barrier 2: every slice's masses are out
        if (!grid_barrier(p.sync, 2u * (unsigned)grid, &ok_sh)) raise_error(p.err, kErrTimeout);

        for (int sq = 0; sq < S; ++sq) {
            const int d0 = cu_sh[sq], g = cu_sh[sq + 1] - d0, k = k_sh[sq];
            if (warp == 0) {
                unsigned long long R = 0, P = 0, Rb = 0, Pb = 0;
                for (int cc = lane; cc < grid; cc += 32) {
                    const ulonglong2 x = __ldcg(&p.tot[(size_t)sq * grid + cc]);
                    R += x.x;
                    P += x.y;
                    if (cc < c) {
                        Rb += x.x;
                        Pb += x.y;
                    }
                }
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) {
                    R += __shfl_xor_sync(0xffffffffu, R, o);
                    P += __shfl_xor_sync(0xffffffffu, P, o);
                    Rb += __shfl_xor_sync(0xffffffffu, Rb, o);
                    Pb += __shfl_xor_sync(0xffffffffu, Pb, o);
                }
                if (lane == 0) {
                    const ulonglong2 own = __ldcg(&p.tot[(size_t)sq * grid + c]);
                    const bool use_r = k < g && R > 0;  // a vanishing residual (p == q) draws from p
                    const unsigned long long total = use_r ? R : P, below = use_r ? Rb : Pb;
                    const unsigned long long mine = use_r ? own.x : own.y;
                    float u = __ldg(p.u_sample + sq);
                    if (!(u >= 0.f)) u = 0.f;
                    u = fminf(u, 0.99999994f);  // u in [0, 1): the crossing always exists
                    const unsigned long long thr = __umul64hi(__float2ull_rn(u * 18446744073709551616.f), total);
                    int find = 0;
                    if (total == 0) {  // no positive mass at all: report, emit 0
                        if (c == 0) {
                            raise_error(p.err, kErrDeviceArg);
                            p.out_tokens[d0 + sq + k] = 0;
                        }
                    } else if (below <= thr && thr < below + mine) {
                        find = 1;
                        off_sh = thr - below;
                    }
                    find_sh = find;
                    use_r_sh = use_r;
                }
            }
            __syncthreads();
            if (find_sh && warp >= kVeEpi) {
                // ---- the crossing is in this slice: chunk masses in entry order, then the entry
                DrawRow d;
                d.ct = d0 + sq + k;
                d.cd = k < g ? p.rows_t + d0 + k : -1;
                d.Mt = rst[d.ct].x;
                d.izt = __fdiv_rn(1.f, rst[d.ct].y);
                d.Md = d.cd >= 0 ? rst[d.cd].x : 0.f;
                d.izd = d.cd >= 0 ? __fdiv_rn(1.f, rst[d.cd].y) : 0.f;
                const bool use_r = use_r_sh != 0;
                if (warp == kVeEpi) {  // one warp scans the chunk masses in entry order (tile, then quarter)
                    const unsigned long long off = off_sh;
                    const int n = ntile * 4, i0 = 2 * lane;  // lane l holds chunks 2l and 2l + 1
                    const ulonglong2 c0 = i0 < n ? chunk[sq * n + i0] : make_ulonglong2(0ull, 0ull);
                    const ulonglong2 c1 = i0 + 1 < n ? chunk[sq * n + i0 + 1] : make_ulonglong2(0ull, 0ull);
                    const unsigned long long x0 = use_r ? c0.x : c0.y, x1 = use_r ? c1.x : c1.y;
                    const unsigned long long incl = warp_incl_scan(x0 + x1, lane);
                    const unsigned long long b0 = incl - x1 - x0, b1 = incl - x1;
                    const bool h0 = x0 > 0 && b0 <= off && off < b1, h1 = x1 > 0 && b1 <= off && off < incl;
                    const unsigned hits = __ballot_sync(0xffffffffu, h0 || h1);  // exactly one with exact sums
                    if (hits == 0u) {
                        if (lane == 0) sel_sh = -1;
                    } else if (lane == __ffs(hits) - 1) {
                        sel_sh = h0 ? i0 : i0 + 1;
                        base_sh = h0 ? b0 : b1;
                    }
                }
                named_sync(1, 128);
                const int sel = sel_sh;
                if (sel < 0) {  // unreachable with exact sums: report, emit the slice's first entry
                    if (tid == kVeEpi * 32) {
                        raise_error(p.err, kErrDeviceArg);
                        p.out_tokens[d0 + sq + k] = v0;
                    }
                } else if ((sel & 3) == q) {
                    const int t = sel >> 2;
                    const int v = v0 + t * kVeM + q * 32 + lane;
                    const float2 w2 = entry_weights<NP>(tq, t, d, v < v1, p.c2);
                    const float w = use_r ? w2.x : w2.y;
                    // offset of the threshold inside the chunk, back in probability units
                    const float off = __ull2float_rn(off_sh - base_sh) * 2.220446049250313e-16f;
                    const float run = warp_incl_scan_f(w, lane);
                    const unsigned hit = __ballot_sync(0xffffffffu, w > 0.f && run > off);
                    const unsigned pos = __ballot_sync(0xffffffffu, w > 0.f);
                    // fp32 rounding inside the chunk can leave the crossing just past its end: then
                    // the chunk's last entry with positive weight
                    const int ln = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
                    if (lane == 0) p.out_tokens[d0 + sq + k] = v0 + t * kVeM + q * 32 + ln;
                }
            }
            __syncthreads();
        }
    }

    // ---- release tensor memory; the last CTA out clears the grid-barrier counters
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, p.tmem_cols);
    }
    if (tid == 0) {
        const unsigned int old = atom_add_acq_rel_gpu(p.sync + 1, 1u);
        if (old == (unsigned)grid - 1u) {
            atomicExch(p.sync, 0u);
            atomicExch(p.sync + 1, 0u);
        }
    }
}

template <int NP, int APS>
size_t ve_smem_bytes() {
    return 1024 + (size_t)ve_stages(NP, APS) * APS * (kVeWBytes + NP * 128);
}

struct VeLayout {
    size_t sync_off, part_off, xg_off, tot_off, total;
    size_t rowst_off, tickets_off, draw_off, logits_off;  // the streamed path (more than 64 rows at T > 0)
};
VeLayout ve_layout(int num_seqs, int total_draft, int vocab) {
    VeLayout l;
    const int rows = 2 * total_draft + num_seqs;
    l.sync_off = 0;
    l.part_off = 256;
    l.xg_off = l.part_off + align_up((size_t)(rows > 0 ? rows : 1) * kVeMaxGrid * sizeof(float2), 256);
    l.tot_off = l.xg_off + align_up((size_t)(total_draft > 0 ? total_draft : 1) * sizeof(float2), 256);
    l.total = l.tot_off + align_up((size_t)(num_seqs > 0 ? num_seqs : 1) * kVeMaxGrid * sizeof(ulonglong2), 256);
    l.rowst_off = l.tickets_off = l.draw_off = l.logits_off = 0;
    if (rows > kVerifyResidentRows) {
        l.rowst_off = l.total;
        l.tickets_off = l.rowst_off + align_up((size_t)rows * sizeof(float2), 256);
        l.draw_off = l.tickets_off + align_up((size_t)num_seqs * sizeof(int), 256);
        l.logits_off = l.draw_off + align_up(accept_draw_scratch_bytes(num_seqs, vocab), 256);
        l.total = l.logits_off + align_up((size_t)rows * (size_t)vocab * sizeof(float), 256);
    }
    return l;
}

template <bool GREEDY, int NP, int APS>
int ve_launch(const CUtensorMap& wmap, const VeParams& p, int grid, const DeviceInfo& dev, cudaStream_t stream) {
    static std::mutex cfg_mu;        // per instantiation (a template's own statics)
    static int configured[64] = {};
    const size_t smem = ve_smem_bytes<NP, APS>();
    if (dev.device >= 0 && dev.device < 64) {
        std::lock_guard<std::mutex> cfg_lock(cfg_mu);  // once per device, from any host thread
        if (!configured[dev.device]) {
            if (cudaFuncSetAttribute(verify_epilogue_kernel<GREEDY, NP, APS>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
                return BP_ERR_CUDA;
            int per_sm = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, verify_epilogue_kernel<GREEDY, NP, APS>,
                                                              kVeThreads, smem) != cudaSuccess ||
                per_sm < 1)
                return BP_ERR_UNSUPPORTED;
            configured[dev.device] = 1;
        }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kVeThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // every CTA co-resident: the grid barriers need it
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, verify_epilogue_kernel<GREEDY, NP, APS>, wmap, p) == cudaSuccess ? BP_OK
                                                                                               : BP_ERR_CUDA;
}

}  // namespace

size_t verify_epilogue_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    return ve_layout(num_seqs, total_draft, vocab).total;
}

int verify_epilogue_config(int rows, int vocab, int hidden, int sm_count, int* grid, int* np, int* tiles_per_cta) {
    if (hidden % kVeAtom != 0) return BP_ERR_UNSUPPORTED;
    const int tiles_total = (vocab + kVeM - 1) / kVeM;
    const int g = min(min(sm_count, kVeMaxGrid), tiles_total);
    if (g < 1 || rows < 1 || rows > kVerifyResidentRows) return BP_ERR_UNSUPPORTED;
    const int NP = rows <= 32 ? 32 : 64;
    const int per = (tiles_total + g - 1) / g;
    if (per > kVeMaxTiles || per * NP > 512) return BP_ERR_UNSUPPORTED;
    *grid = g;
    *np = NP;
    *tiles_per_cta = per;
    return BP_OK;
}

int launch_verify_epilogue(const VerifyEpilogueArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    const bool greedy = a.temperature == 0.f;
    const int rows_t = a.total_draft + a.num_seqs;
    const int rows = rows_t + (greedy ? 0 : a.total_draft);
    const VeLayout l = ve_layout(a.num_seqs, a.total_draft, a.vocab);
    uint8_t* ws = static_cast<uint8_t*>(a.scratch);
    if (rows > kVerifyResidentRows) {
        VerifyStreamScratch s;
        s.logits = reinterpret_cast<float*>(ws + l.logits_off);
        s.part = reinterpret_cast<float2*>(ws + l.part_off);
        s.row_stats = reinterpret_cast<float2*>(ws + l.rowst_off);
        s.tickets = reinterpret_cast<int*>(ws + l.tickets_off);
        s.draw = ws + l.draw_off;
        return launch_verify_stream(a, s, dev, stream);
    }
    int grid = 0, NP = 0, per = 0;
    int rc = verify_epilogue_config(rows, a.vocab, a.hidden, dev.sm_count, &grid, &NP, &per);
    if (rc != BP_OK) return rc;
    const int tiles_total = (a.vocab + kVeM - 1) / kVeM;
    uint32_t cols = 32;
    while (cols < (uint32_t)(per * NP)) cols <<= 1;

    CUtensorMap wmap;
    const cuuint64_t dims[2] = {(cuuint64_t)a.hidden, (cuuint64_t)a.vocab};
    const cuuint64_t strides[1] = {(cuuint64_t)a.hidden * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kVeAtom, (cuuint32_t)kVeM};
    if (encode_tensor_map(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a.lm_head), dims, strides, box,
                          CU_TENSOR_MAP_SWIZZLE_128B) != BP_OK)
        return BP_ERR_CUDA;

    VeParams p;
    p.h_target = static_cast<const __nv_bfloat16*>(a.h_target);
    p.h_draft = static_cast<const __nv_bfloat16*>(greedy ? a.h_target : a.h_draft);
    p.hidden = a.hidden;
    p.vocab = a.vocab;
    p.atoms = a.hidden / kVeAtom;
    p.num_seqs = a.num_seqs;
    p.total_draft = a.total_draft;
    p.rows_t = rows_t;
    p.rows = rows;
    p.tiles_base = tiles_total / grid;
    p.tiles_extra = tiles_total % grid;
    p.tmem_cols = cols;
    p.c2 = greedy ? 0.f : 1.4426950408889634f / a.temperature;
    p.tokens = a.tokens;
    p.cu_draft = a.cu_draft;
    p.u_accept = a.u_accept;
    p.u_sample = a.u_sample;
    p.n_accepted = a.n_accepted;
    p.out_tokens = a.out_tokens;
    p.accept_prob = a.accept_prob;
    p.logits_out = a.logits_out;
    p.part = reinterpret_cast<float2*>(ws + l.part_off);
    p.xg = reinterpret_cast<float2*>(ws + l.xg_off);
    p.tot = reinterpret_cast<ulonglong2*>(ws + l.tot_off);
    p.sync = reinterpret_cast<unsigned int*>(ws + l.sync_off);
    p.err = a.err_word;
    const bool two = p.atoms % 2 == 0;  // two atoms per stage where the hidden size allows
    if (greedy && NP == 32)
        return two ? ve_launch<true, 32, 2>(wmap, p, grid, dev, stream)
                   : ve_launch<true, 32, 1>(wmap, p, grid, dev, stream);
    if (greedy)
        return two ? ve_launch<true, 64, 2>(wmap, p, grid, dev, stream)
                   : ve_launch<true, 64, 1>(wmap, p, grid, dev, stream);
    if (NP == 32)
        return two ? ve_launch<false, 32, 2>(wmap, p, grid, dev, stream)
                   : ve_launch<false, 32, 1>(wmap, p, grid, dev, stream);
    return two ? ve_launch<false, 64, 2>(wmap, p, grid, dev, stream)
               : ve_launch<false, 64, 1>(wmap, p, grid, dev, stream);
}

}  // namespace bp
