// Block attention for the verify (causal-within-block) and drafter (bidirectional-
// within-block) passes of block-diffusion speculative decoding (Section 2.1,
// Figure 1 of the BlockPilot paper).
//
// bf16 tensor-core path (sm_103a):
//   * One work unit = (sequence, KV head, 128-row query tile).  The B_s block
//     queries of the g = Hq/Hkv query heads that share a KV head are packed as the
//     rows of one M=128 tile (row r = i*g + j: block position i, head j of the
//     group), so QK^T and PV are M=128 tcgen05 MMAs that read each K/V tile once.
//   * A thread-block cluster of CS CTAs splits the unit's keys; each CTA streams its
//     share of 128-key K/V tiles through a 3-stage TMA ring (SWIZZLE_128B), computes
//     S = Q K^T into tensor memory, runs an online softmax (fp32, exp2 domain, lazy
//     rescale of the TMEM accumulator when the row max grows by more than 2^8),
//     writes P (bf16) back into tensor memory and accumulates O += P V with P as the
//     TMEM A operand.  The CS partial results are merged through distributed shared
//     memory -- no global scratch, one launch.
//   * Units are issued longest-first so that ragged batches finish together.
//   Warp roles: warp 0 = TMA producer + TMEM allocator, warp 1 = MMA issuer,
//   warps 2..5 = softmax / epilogue (one query row per thread, TMEM lane = row).  Units of at
//   most 64 rows (a block of up to 64/g positions) use the spread layout instead: the rows fill
//   16 lanes of each TMEM sub-partition and each half-warp takes one 64-key half of a row, so
//   all four softmax warps share the exp2 work.
//
// fp32 path: a plain SIMT kernel (one warp per output row, online softmax).
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "ptx_sm103.cuh"

namespace cg = cooperative_groups;

namespace bp {
namespace {

constexpr int kD = 128;       // head_dim of the tensor-core path
constexpr int kTileN = 128;   // keys per K/V tile
constexpr int kM = 128;       // query rows per tile
constexpr int kStages = 3;    // K/V ring depth
constexpr int kHalf = kTileN * 64 * 2;          // one 64-column SW128 half of a 128-row tile: 16 KB
constexpr int kQBytes = kM * kD * 2;            // 32 KB
constexpr int kKVBytes = kTileN * kD * 2;       // 32 KB for K, 32 KB for V
constexpr int kStageBytes = 2 * kKVBytes;       // 64 KB
constexpr int kDynSmem = kQBytes + kStages * kStageBytes + 1024;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 256;
constexpr int kMaxOrderedSeqs = 256;  // longest-first ordering for batches up to this size
constexpr int kMaxCluster = 16;

struct AttnParams {
    const __nv_bfloat16* q;
    __nv_bfloat16* o;
    float* lse;
    const int32_t* cu_q;
    const int32_t* cu_kv;
    int num_seqs, num_q_heads, num_kv_heads, group, m_tiles;
    int total_q, total_kv;
    int causal;
    float scale_log2;  // softmax scale * log2(e)
    int q_tma;         // Q tile loaded by TMA (group divides 128)
    // paged KV cache: sequence s's key j lives in page block_table[s * pages_per_seq + (j >> page_shift)]
    // at row j & (page size - 1); NULL block_table = contiguous K/V rows from cu_kv[s]
    const int32_t* block_table;
    int pages_per_seq, page_shift;
    // flat split: partial (O, m, l) slots in the workspace, two per CTA, slot_rows rows each; and one
    // work entry (two int4) per CTA for the merge: (first tile, end tile, all tiles, rows) and (first
    // query row, query tile) of the cut unit whose first tile the CTA holds, or first tile -1
    float* part;
    int4* work;
    int slot_rows;
    int early_release;  // the grid runs in one wave: dependents may launch as soon as every CTA has started
    unsigned int* err;
};
constexpr int kMaxSub = kTileN / 16;  // sub-boxes per K/V tile at the smallest page size (16 keys)

__device__ __forceinline__ uint32_t col_s(int sb) { return sb ? 128u : 0u; }  // TMEM column of S buffer sb

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ int cdiv(int a, int b) { return (a + b - 1) / b; }

// One stretch of consecutive 128-key tiles of one work unit (sequence s, KV head h, 128-row query
// tile mt), processed by one CTA.
struct Seg {
    int s, h, mt;
    int q0, B, kv0, n;  // the sequence's first query row, block size, first key row, key count
    int jt0, nt;        // first tile of the stretch within the unit, tiles in it
    int whole;          // flat split: the stretch is the whole unit (the CTA writes the output)
    int slot;           // flat split, part of a unit: the CTA's partial slot (0 first stretch, 1 last)
};

// Flat split: key tiles of every sequence over its 128-row query tiles, counted once for all KV heads
// (a group of CTAs, one per KV head, streams the same tiles of every head at the same time); a
// sequence without block rows has none.
__device__ __forceinline__ int flat_seq_tiles(int B, int n, int G) {
    return B > 0 ? cdiv(B * G, kM) * cdiv(n, kTileN) : 0;
}

// Flat split: the prefix sums of the sequences' tile counts into pre[0..S] (S <= kMaxOrderedSeqs), by one
// warp: each lane sums 8 consecutive sequences, then an exclusive scan of the lane sums.
__device__ __forceinline__ void flat_prefix(const AttnParams& p, int32_t* pre, int lane) {
    constexpr int kPer = (kMaxOrderedSeqs + 31) / 32;
    int loc[kPer];
    int run = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        const int s = lane * kPer + k;
        if (s < p.num_seqs) {
            const int B = __ldg(p.cu_q + s + 1) - __ldg(p.cu_q + s);
            const int n = __ldg(p.cu_kv + s + 1) - __ldg(p.cu_kv + s);
            run += flat_seq_tiles(B, n, p.group);
        }
        loc[k] = run;
    }
    int incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    const int excl = incl - run;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        const int s = lane * kPer + k;
        if (s < p.num_seqs) pre[s + 1] = excl + loc[k];
    }
    if (lane == 0) pre[0] = 0;
}

// Flat split: the stretch that starts at global tile t of a CTA (KV head h) whose range ends at t_end
// (pre: the sequences' tile prefix sums; a single sequence needs none).  first: the CTA's first stretch.
__device__ __forceinline__ Seg flat_seg(const AttnParams& p, const int32_t* pre, int t, int t_end, int h, bool first) {
    Seg g;
    int s = 0;
    if (p.num_seqs > 1) {  // the last sequence whose tiles start at or before t
        int lo = 0, hi = p.num_seqs;
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (pre[mid] <= t) lo = mid; else hi = mid;
        }
        s = lo;
    }
    const int base = p.num_seqs > 1 ? pre[s] : 0;
    g.s = s;
    g.q0 = p.num_seqs == 1 ? 0 : __ldg(p.cu_q + s);
    g.B = p.num_seqs == 1 ? p.total_q : __ldg(p.cu_q + s + 1) - g.q0;
    g.kv0 = p.num_seqs == 1 ? 0 : __ldg(p.cu_kv + s);
    g.n = p.num_seqs == 1 ? p.total_kv : __ldg(p.cu_kv + s + 1) - g.kv0;
    const int ntu = cdiv(g.n, kTileN);
    const int local = t - base;
    g.mt = local / ntu;
    g.jt0 = local - g.mt * ntu;
    g.h = h;
    g.nt = min(ntu - g.jt0, t_end - t);
    g.whole = g.jt0 == 0 && g.nt == ntu;
    g.slot = first ? 0 : 1;
    return g;
}

// PAGED: K/V rows come from pages named by p.block_table (the contiguous instantiation carries no
// paging code at all).
// SPREAD (units of at most 64 query rows, group size dividing 16): logical row r sits at TMEM lane
// (r / 16) * 32 + r % 16, so the 64 rows fill 16 lanes of each of the four TMEM sub-partitions and
// all four softmax warps (and their SMSPs' exp2 units) work; the two half-warps take the two
// 64-column halves of a row (tcgen05 16x32bx2 accesses), combining row statistics by shuffle.
// FLAT: the flat split.  The key tiles of all units, in order, are cut into gridDim.x equal ranges,
// one per CTA (no clusters); a CTA works through the stretches of its range one after another with
// one pipeline (K/V ring, S double buffer, O accumulator) and writes a unit it covers whole straight
// to the output, a partial stretch to its workspace slot for attn_combine_kernel.  Otherwise the
// cluster split: a unit per cluster, its tiles cut into CS ranges, partials merged through
// distributed shared memory.
template <bool PAGED, bool SPREAD, bool FLAT>
__global__ void __launch_bounds__(kThreads, 1)
    attn_bf16_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                        const __grid_constant__ CUtensorMap vmap, const AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sQ = smem;
    uint8_t* sKV = smem + kQBytes;  // stage s: K at s*64KB, V at s*64KB + 32KB

    __shared__ uint64_t bar_kv_full[kStages], bar_kv_empty[kStages];
    __shared__ uint64_t bar_s_full[2], bar_p_full[2], bar_pv_done[2], bar_o_done, bar_q_full, bar_q_empty;
    __shared__ uint32_t tmem_base_sh;
    __shared__ int unit_seq_sh;
    // cluster split: the sequences' key offsets (longest-first order); flat split: their tile prefix sums
    __shared__ int32_t seq_sh[kMaxOrderedSeqs + 1];

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        if (p.q_tma) prefetch_tensormap(&qmap);
        prefetch_tensormap(&kmap);
        prefetch_tensormap(&vmap);
    }
    if (p.early_release) griddep_launch_dependents();
    if (p.num_seqs > 1) griddep_wait();  // the sequence offsets are read from global memory
    const int G = p.group;
    const uint32_t CS = FLAT ? 1u : cluster_size();
    const uint32_t crank = FLAT ? 0u : cluster_rank();

    // ---- work assignment.  Flat split: global tiles [t_lo, t_hi).  Cluster split: one stretch, `one`.
    int t_lo = 0, t_hi = 0, T = 0;
    Seg one{};
    if (FLAT) {
        if (p.num_seqs > 1) {
            if (warp == 0) flat_prefix(p, seq_sh, lane);
            __syncthreads();
            T = seq_sh[p.num_seqs];
        } else {
            T = flat_seq_tiles(p.total_q, p.total_kv, G);
        }
        // CTAs come in groups of one per KV head; group j has tiles [t_lo, t_hi) of every head
        const int ngroups = gridDim.x / p.num_kv_heads, grp = blockIdx.x / p.num_kv_heads;
        t_lo = (int)((long long)grp * T / ngroups);
        t_hi = (int)((long long)(grp + 1) * T / ngroups);
    } else {
        const int unit_rank = blockIdx.x / CS;
        const int units_per_seq = p.num_kv_heads * p.m_tiles;
        const int seq_rank = unit_rank / units_per_seq;
        one.h = (unit_rank / p.m_tiles) % p.num_kv_heads;
        one.mt = unit_rank % p.m_tiles;
        // which sequence: the seq_rank-th longest (ties by index) for small batches
        int s;
        if (p.num_seqs == 1) {
            s = 0;
        } else if (p.num_seqs <= kMaxOrderedSeqs) {
            for (int t = tid; t <= p.num_seqs; t += kThreads) seq_sh[t] = p.cu_kv[t];
            __syncthreads();
            for (int t = tid; t < p.num_seqs; t += kThreads) {
                const int len = seq_sh[t + 1] - seq_sh[t];
                int rank = 0;
                for (int u = 0; u < p.num_seqs; ++u) {
                    const int lu = seq_sh[u + 1] - seq_sh[u];
                    rank += (lu > len) || (lu == len && u < t);
                }
                if (rank == seq_rank) unit_seq_sh = t;
            }
            __syncthreads();
            s = unit_seq_sh;
        } else {
            s = seq_rank;
        }
        one.s = s;
        // a single sequence starts at offset 0 (cu_*[0] = 0) and spans the whole tensors: no loads
        one.q0 = p.num_seqs == 1 ? 0 : __ldg(p.cu_q + s);
        one.B = p.num_seqs == 1 ? p.total_q : __ldg(p.cu_q + s + 1) - one.q0;
        one.kv0 = p.num_seqs == 1 ? 0 : __ldg(p.cu_kv + s);
        one.n = p.num_seqs == 1 ? p.total_kv : __ldg(p.cu_kv + s + 1) - one.kv0;
        if (one.B * G - one.mt * kM <= 0) {  // uniform across the cluster: every CTA decodes the same unit
            griddep_wait();  // this grid must not complete before the one it depends on
            return;
        }
        const int tiles = cdiv(one.n, kTileN);
        one.jt0 = (int)((long long)crank * tiles / CS);
        one.nt = (int)((long long)(crank + 1) * tiles / CS) - one.jt0;
        one.whole = 0;
        one.slot = 0;
    }
    // The stretches of this CTA, in order: `first` is the CTA's first one; t advances past each.
    auto seg_at = [&](int t, bool first) -> Seg {
        return FLAT ? flat_seg(p, seq_sh, t, t_hi, (int)(blockIdx.x % p.num_kv_heads), first) : one;
    };
    const int t_begin = FLAT ? t_lo : 0;
    const int t_end = FLAT ? t_hi : 1;
    auto seg_len = [&](const Seg& g) { return FLAT ? g.nt : 1; };

    // ---- Q tile -> shared memory, SWIZZLE_128B K-major (two 64-column halves).  With a TMA map the
    // 128/G block positions x G heads box lands exactly as rows r = i*G + j; otherwise (cluster split
    // only) plain loads.
    if (!FLAT && !p.q_tma) {
        griddep_wait();
        const int row0 = one.mt * kM, m_valid = min(kM, one.B * G - row0);
        for (int idx = tid; idx < kM * 16; idx += kThreads) {
            const int r = idx >> 4, ch = idx & 15;
            uint4 val = make_uint4(0, 0, 0, 0);
            if (r < m_valid) {
                const int lr = row0 + r;
                const int i = lr / G, j = lr % G;
                val = *reinterpret_cast<const uint4*>(p.q + ((size_t)(one.q0 + i) * p.num_q_heads + one.h * G + j) *
                                                      kD + ch * 8);
            }
            const int half = ch >> 3, c8 = ch & 7;
            *reinterpret_cast<uint4*>(sQ + half * kHalf + r * 128 + ((c8 ^ (r & 7)) << 4)) = val;
        }
        fence_proxy_async_smem();
    }
    // paged cache: the pool rows of a tile's sub-boxes (sub_rows keys each); keys past the end of the
    // sequence read the rows of its last page (finite values the mask then drops)
    constexpr bool paged = PAGED;
    const int sub_rows = paged ? min(kTileN, 1 << p.page_shift) : kTileN;
    const int nsub = kTileN / sub_rows;
    auto tile_rows = [&](const Seg& g, int jl, int (&row)[kMaxSub]) {
        if (!paged) return;
        const int32_t* bt = p.block_table + (size_t)g.s * p.pages_per_seq;
        const int last_page = max(0, (g.n - 1) >> p.page_shift);
        const int key0 = (g.jt0 + jl) * kTileN;
#pragma unroll
        for (int sb = 0; sb < kMaxSub; ++sb)
            if (sb < nsub) {
                const int key = key0 + sb * sub_rows;
                const int pi = min(key >> p.page_shift, last_page);
                row[sb] = __ldg(bt + pi) * (1 << p.page_shift) + (key & ((1 << p.page_shift) - 1));
            }
    };
    // K/V tile jl of stretch g -> ring stage J % kStages (J counts the CTA's tiles; producer thread only)
    auto issue_kv = [&](int J, const Seg& g, int jl, const int (&row)[kMaxSub]) {
        const int st = J % kStages;
        uint8_t* sK = sKV + st * kStageBytes;
        uint8_t* sV = sK + kKVBytes;
        mbar_arrive_expect_tx(&bar_kv_full[st], kStageBytes);
        if (!paged) {
            const int key = g.kv0 + (g.jt0 + jl) * kTileN;
            tma_load_3d(sK, &kmap, &bar_kv_full[st], 0, g.h, key);
            tma_load_3d(sK + kHalf, &kmap, &bar_kv_full[st], 64, g.h, key);
            tma_load_3d(sV, &vmap, &bar_kv_full[st], 0, g.h, key);
            tma_load_3d(sV + kHalf, &vmap, &bar_kv_full[st], 64, g.h, key);
        } else {
#pragma unroll
            for (int sb = 0; sb < kMaxSub; ++sb) {  // sub-box sb lands at row sb * sub_rows of the tile
                if (sb < nsub) {
                    const int off = sb * sub_rows * 128;
                    tma_load_3d(sK + off, &kmap, &bar_kv_full[st], 0, g.h, row[sb]);
                    tma_load_3d(sK + kHalf + off, &kmap, &bar_kv_full[st], 64, g.h, row[sb]);
                    tma_load_3d(sV + off, &vmap, &bar_kv_full[st], 0, g.h, row[sb]);
                    tma_load_3d(sV + kHalf + off, &vmap, &bar_kv_full[st], 64, g.h, row[sb]);
                }
            }
        }
    };
    // the Q tile of stretch g (producer thread only)
    auto issue_q = [&](const Seg& g) {
        const int row0 = g.mt * kM;
        if (SPREAD) {  // four boxes of 16 rows, at shared-memory rows 0, 32, 64, 96
            mbar_arrive_expect_tx(&bar_q_full, kQBytes / 2);
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
                const int qrow = g.q0 + (row0 + 16 * qq) / G;
                tma_load_3d(sQ + qq * 32 * 128, &qmap, &bar_q_full, 0, g.h * G, qrow);
                tma_load_3d(sQ + kHalf + qq * 32 * 128, &qmap, &bar_q_full, 64, g.h * G, qrow);
            }
        } else {
            mbar_arrive_expect_tx(&bar_q_full, kQBytes);
            const int qrow = g.q0 + row0 / G;
            tma_load_3d(sQ, &qmap, &bar_q_full, 0, g.h * G, qrow);
            tma_load_3d(sQ + kHalf, &qmap, &bar_q_full, 64, g.h * G, qrow);
        }
    };
    if (tid == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&bar_kv_full[i], 1);
            mbar_init(&bar_kv_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bar_s_full[i], 1);
            mbar_init(&bar_p_full[i], 128);
            mbar_init(&bar_pv_done[i], 1);
        }
        mbar_init(&bar_o_done, 1);
        mbar_init(&bar_q_full, 1);
        mbar_init(&bar_q_empty, 1);
        fence_mbar_init();
    }
    if (warp == 1) {  // tensor memory is allocated (and released) by warp 1, in parallel
        tmem_alloc(&tmem_base_sh, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;
    // inputs may be produced by the previous kernel on the stream: wait for it before any global access
    griddep_wait();

    if (warp == 0) {
        // ================= TMA producer: the Q tile of each stretch, the K/V tiles through the ring
        if (lane == 0) {
            int J = 0, nq = 0;
            bool ok = true;
            for (int t = t_begin; t < t_end && ok;) {
                const Seg g = seg_at(t, t == t_begin);
                t += seg_len(g);
                if (g.nt == 0) continue;
                for (int jl = 0; jl < g.nt; ++jl, ++J) {
                    int rows[kMaxSub];
                    tile_rows(g, jl, rows);  // page lookups in flight while the stage drains
                    if (J >= kStages &&
                        !mbar_wait(&bar_kv_empty[J % kStages], ((J / kStages) - 1) & 1, kWaitBudget)) {
                        ok = false;
                        break;
                    }
                    issue_kv(J, g, jl, rows);
                    if (jl == 0 && p.q_tma) {
                        // the stretch's Q, once the MMAs of the previous stretch no longer read the buffer
                        if (nq > 0 && !mbar_wait(&bar_q_empty, (nq - 1) & 1, kWaitBudget)) {
                            ++J;
                            ok = false;
                            break;
                        }
                        issue_q(g);
                        ++nq;
                    }
                }
            }
            if (!ok) raise_error(p.err, kErrTimeout);
            // no copy may still be in flight when the CTA leaves
            for (int j = max(0, J - kStages); j < J; ++j)
                if (!mbar_wait(&bar_kv_full[j % kStages], (j / kStages) & 1, kDrainBudget)) raise_error(p.err, kErrTimeout);
            if (nq > 0 && !mbar_wait(&bar_q_full, (nq - 1) & 1, kDrainBudget)) raise_error(p.err, kErrTimeout);
        }
    } else if (warp == 1) {
        // ================= MMA issuer
        if (lane == 0) {
            const uint32_t id_s = idesc_bf16_f32(kM, kTileN, false, false);
            const uint32_t id_o = idesc_bf16_f32(kM, kD, false, true);
            const uint32_t q_addr = smem_addr(sQ);
            int J = 0, nq = 0;
            bool ok = true;
            auto issue_pv = [&](int Jx, bool first) {
                const int sb = Jx & 1, st = Jx % kStages;
                if (!mbar_wait(&bar_p_full[sb], (Jx >> 1) & 1, kWaitBudget)) return false;
                tc_fence_after();
                const uint32_t v_addr = smem_addr(sKV + st * kStageBytes + kKVBytes);
                for (int kk = 0; kk < kTileN / 16; ++kk) {
                    const uint64_t bdesc = smem_desc(v_addr + kk * 2048, kHalf, 1024, kSwizzle128B);
                    umma_ts(tmem + kColO, tmem + col_s(sb) + kk * 8, bdesc, id_o, (!first || kk > 0) ? 1u : 0u);
                }
                umma_commit(&bar_pv_done[sb]);
                umma_commit(&bar_kv_empty[st]);
                return true;
            };
            for (int t = t_begin; t < t_end && ok;) {
                const Seg g = seg_at(t, t == t_begin);
                t += seg_len(g);
                if (g.nt == 0) continue;
                if (p.q_tma && !mbar_wait(&bar_q_full, nq & 1, kWaitBudget)) {
                    ok = false;
                    break;
                }
                for (int jl = 0; jl < g.nt; ++jl, ++J) {
                    const int sb = J & 1, st = J % kStages;
                    if (!mbar_wait(&bar_kv_full[st], (J / kStages) & 1, kWaitBudget)) { ok = false; break; }
                    if (J >= 2 && !mbar_wait(&bar_pv_done[sb], ((J - 2) >> 1) & 1, kWaitBudget)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t k_addr = smem_addr(sKV + st * kStageBytes);
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kHalf + (kk & 3) * 32;
                        const uint64_t adesc = smem_desc(q_addr + off, 16, 1024, kSwizzle128B);
                        const uint64_t bdesc = smem_desc(k_addr + off, 16, 1024, kSwizzle128B);
                        umma_ss(tmem + col_s(sb), adesc, bdesc, id_s, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(&bar_s_full[sb]);
                    if (jl == g.nt - 1) umma_commit(&bar_q_empty);  // the last read of this stretch's Q
                    if (jl >= 1 && !issue_pv(J - 1, jl == 1)) { ++J; ok = false; break; }
                }
                if (!ok) break;
                if (!issue_pv(J - 1, g.nt == 1)) { ok = false; break; }
                umma_commit(&bar_o_done);
                ++nq;
            }
            if (!ok) raise_error(p.err, kErrTimeout);
            if (J > 0) {
                // no MMA may still be writing tensor memory when it is released
                umma_commit(&bar_o_done);
                if (!mbar_wait(&bar_o_done, nq & 1, kDrainBudget)) raise_error(p.err, kErrTimeout);
            }
        }
    }

    // ================= softmax / epilogue warps (2..5).  Dense: row r = TMEM lane quad*32 + lane, all
    // columns.  SPREAD: row r = quad*16 + lane%16 at TMEM lane quad*32 + lane%16, columns of half lane/16.
    constexpr int kCols = SPREAD ? kTileN / 2 : kTileN;  // S / P columns (keys) per thread
    constexpr int kOCols = SPREAD ? kD / 2 : kD;         // O columns per thread
    const int quad = warp & 3;
    const int half = SPREAD ? (lane >> 4) : 0;
    const int r = SPREAD ? quad * 16 + (lane & 15) : quad * 32 + lane;
    const bool is_softmax = warp >= 2;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    const float kLn2 = 0.6931471805599453f;
    float m_run = -INFINITY, l_run = 0.f;  // SPREAD: l_run is this half's share of the row sum
    float o_acc[kOCols];
    bool failed = false;
    bool row_active = false;  // the cluster split's merge below needs the (one) stretch's values
    int m_valid = 0;

    // normalised output row r of stretch g (and its log-sum-exp)
    auto write_row = [&](const Seg& g) {
        const int lr = g.mt * kM + r;
        const int i = lr / G, jh = lr % G;
        const size_t orow = (size_t)(g.q0 + i) * p.num_q_heads + g.h * G + jh;
        const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
        __nv_bfloat16* dst = p.o + orow * kD + half * kOCols;
#pragma unroll
        for (int c = 0; c < kOCols / 8; ++c) {
            uint4 w;
            w.x = pack_bf16x2(o_acc[c * 8 + 0] * inv, o_acc[c * 8 + 1] * inv);
            w.y = pack_bf16x2(o_acc[c * 8 + 2] * inv, o_acc[c * 8 + 3] * inv);
            w.z = pack_bf16x2(o_acc[c * 8 + 4] * inv, o_acc[c * 8 + 5] * inv);
            w.w = pack_bf16x2(o_acc[c * 8 + 6] * inv, o_acc[c * 8 + 7] * inv);
            *reinterpret_cast<uint4*>(dst + c * 8) = w;
        }
        if (p.lse && half == 0) p.lse[orow] = (m_run + __log2f(l_run)) * kLn2;
    };

    if (is_softmax) {
        int J = 0, nq = 0;
        int4 entry = make_int4(-1, 0, 0, 0), entry2 = make_int4(0, 0, 0, 0);  // flat split: the merge's work entry
        for (int t = t_begin; t < t_end && !failed;) {
            const Seg g = seg_at(t, t == t_begin);
            if (FLAT && !g.whole && g.jt0 == 0) {  // a cut unit that starts here
                entry = make_int4(t, t + cdiv(g.n, kTileN), T, min(min(kM, g.B * G - g.mt * kM), p.slot_rows));
                entry2 = make_int4(g.q0, g.mt, 0, 0);
            }
            t += seg_len(g);
            const int row0 = g.mt * kM;
            m_valid = min(kM, g.B * G - row0);
            row_active = r < m_valid;
            const bool warp_active = (SPREAD ? quad * 16 : quad * 32) < m_valid;
            const int L = g.n - g.B;
            const int limit = row_active ? (p.causal ? L + (row0 + r) / G + 1 : g.n) : 0;
            m_run = -INFINITY;
            l_run = 0.f;
            for (int jl = 0; jl < g.nt; ++jl, ++J) {
                const int sb = J & 1;
                if (!__all_sync(0xffffffffu, mbar_wait(&bar_s_full[sb], (J >> 1) & 1, kWaitBudget))) {
                    failed = true;
                    break;
                }
                tc_fence_after();
                if (warp_active) {
                    const int nvalid = limit - (g.jt0 + jl) * kTileN;
                    float x[kCols];
#pragma unroll
                    for (int c = 0; c < kCols / 32; ++c) {
                        uint32_t v[32];
                        if (SPREAD) tmem_ld16x2_32<kTileN / 2>(tmem + lane_base + col_s(sb) + c * 32, v);
                        else tmem_ld32(tmem + lane_base + col_s(sb) + c * 32, v);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const int kidx = half * (kTileN / 2) + c * 32 + e;
                            x[c * 32 + e] = (kidx < nvalid) ? __uint_as_float(v[e]) * p.scale_log2 : -INFINITY;
                        }
                    }
                    float mt_ = -INFINITY;
#pragma unroll
                    for (int e = 0; e < kCols; ++e) mt_ = fmaxf(mt_, x[e]);
                    if (SPREAD) mt_ = fmaxf(mt_, __shfl_xor_sync(0xffffffffu, mt_, 16));
                    const float m_new = fmaxf(m_run, mt_);
                    const bool need = m_new > m_run + 8.f;
                    const float alpha = need ? fast_exp2(m_run - m_new) : 1.f;
                    // rescale the TMEM accumulator of rows whose max grew (warp-uniform TMEM access)
                    if (__any_sync(0xffffffffu, need && jl > 0 && m_run != -INFINITY)) {
                        if (!__all_sync(0xffffffffu,
                                        mbar_wait(&bar_pv_done[(J - 1) & 1], ((J - 1) >> 1) & 1, kWaitBudget))) {
                            failed = true;
                        } else {
                            tc_fence_after();
#pragma unroll
                            for (int c = 0; c < kOCols / 32; ++c) {
                                uint32_t v[32];
                                if (SPREAD) tmem_ld16x2_32<kD / 2>(tmem + lane_base + kColO + c * 32, v);
                                else tmem_ld32(tmem + lane_base + kColO + c * 32, v);
                                tmem_ld_wait();
                                if (SPREAD) {
#pragma unroll
                                    for (int e = 0; e < 32; ++e)
                                        v[e] = __float_as_uint(__uint_as_float(v[e]) * alpha);
                                    tmem_st16x2_32<kD / 2>(tmem + lane_base + kColO + c * 32, v);
                                } else {
                                    uint32_t w0[16], w1[16];
#pragma unroll
                                    for (int e = 0; e < 16; ++e) {
                                        w0[e] = __float_as_uint(__uint_as_float(v[e]) * alpha);
                                        w1[e] = __float_as_uint(__uint_as_float(v[16 + e]) * alpha);
                                    }
                                    tmem_st16(tmem + lane_base + kColO + c * 32, w0);
                                    tmem_st16(tmem + lane_base + kColO + c * 32 + 16, w1);
                                }
                            }
                        }
                    }
                    if (need) {
                        l_run *= alpha;
                        m_run = m_new;
                    }
                    float lsum = 0.f;
                    const bool any = m_run != -INFINITY;
                    if (SPREAD) {  // this half's 64 keys -> 32 packed P columns (the other half 32 further)
                        uint32_t pk[32];
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const float a = any ? fast_exp2(x[2 * e] - m_run) : 0.f;
                            const float b = any ? fast_exp2(x[2 * e + 1] - m_run) : 0.f;
                            lsum += a + b;
                            pk[e] = pack_bf16x2(a, b);
                        }
                        tmem_st16x2_32<kTileN / 4>(tmem + lane_base + col_s(sb), pk);
                    } else {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            uint32_t pk[16];
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                const float a = any ? fast_exp2(x[c * 32 + 2 * e] - m_run) : 0.f;
                                const float b = any ? fast_exp2(x[c * 32 + 2 * e + 1] - m_run) : 0.f;
                                lsum += a + b;
                                pk[e] = pack_bf16x2(a, b);
                            }
                            tmem_st16(tmem + lane_base + col_s(sb) + c * 16, pk);
                        }
                    }
                    l_run += lsum;
                    tmem_st_wait();
                }
                tc_fence_before();
                mbar_arrive(&bar_p_full[sb]);
                if (failed) break;
            }
            // the stretch's accumulator
            if (g.nt > 0 && !failed && !__all_sync(0xffffffffu, mbar_wait(&bar_o_done, nq & 1, kWaitBudget)))
                failed = true;
            failed = __any_sync(0xffffffffu, failed);
            tc_fence_after();
            if (warp_active && g.nt > 0 && !failed) {
#pragma unroll
                for (int c = 0; c < kOCols / 32; ++c) {
                    uint32_t v[32];
                    if (SPREAD) tmem_ld16x2_32<kD / 2>(tmem + lane_base + kColO + c * 32, v);
                    else tmem_ld32(tmem + lane_base + kColO + c * 32, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; ++e) o_acc[c * 32 + e] = __uint_as_float(v[e]);
                }
            } else {
#pragma unroll
                for (int e = 0; e < kOCols; ++e) o_acc[e] = 0.f;
                if (g.nt == 0 || failed) {
                    m_run = -INFINITY;
                    l_run = 0.f;
                }
            }
            if (SPREAD) l_run += __shfl_xor_sync(0xffffffffu, l_run, 16);  // the whole row's sum
            if (g.nt > 0) ++nq;
            if (FLAT && !g.whole && m_valid > p.slot_rows) {  // a block longer than max_q_len: rows past the slot are dropped
                if (r == 0 && warp == 2) raise_error(p.err, kErrDeviceArg);
                row_active = row_active && r < p.slot_rows;
            }
            if (FLAT && !failed && row_active) {
                if (g.whole) {
                    write_row(g);
                } else {  // the partial (O, m, l) of this stretch's rows, for attn_combine_kernel
                    float* slot = p.part + (size_t)(2 * blockIdx.x + g.slot) * p.slot_rows * (kD + 2);
                    float* orow = slot + (size_t)r * kD + half * kOCols;
#pragma unroll
                    for (int c = 0; c < kOCols / 4; ++c)
                        *reinterpret_cast<float4*>(orow + c * 4) =
                            make_float4(o_acc[c * 4], o_acc[c * 4 + 1], o_acc[c * 4 + 2], o_acc[c * 4 + 3]);
                    if (half == 0)
                        *reinterpret_cast<float2*>(slot + (size_t)p.slot_rows * kD + 2 * r) = make_float2(m_run, l_run);
                }
            }
        }
        if (failed) raise_error(p.err, kErrTimeout);
        if (FLAT && tid == 64) {
            p.work[2 * blockIdx.x] = entry;
            p.work[2 * blockIdx.x + 1] = entry2;
        }
    }

    if (!FLAT) {
        if (CS == 1) {
            if (row_active) write_row(one);
        } else {
            // ---- merge of the CS partial (m, l, O) triples through distributed shared memory.  After the
            // first cluster barrier every K/V ring is idle (all of its TMA loads were consumed); each CTA
            // leaves its partial there and pulls the rows it owns from all peers:
            //   opart  [kM rows][kD] fp32 partial O (16-byte chunks swizzled by row)
            //   row_ml [kM] (m, l) of each row's partial
            //   ml_st, w_st, inv_st  the peers' (m, l) of the owned rows, their weights, 1/L
            m_valid = min(kM, one.B * G - one.mt * kM);
            const int row0 = one.mt * kM;
            cg::cluster_group cluster = cg::this_cluster();
            float* opart = reinterpret_cast<float*>(sKV);
            float2* row_ml = reinterpret_cast<float2*>(sKV + kM * kD * sizeof(float));
            __syncthreads();  // the producer has drained the ring (after an expired wait copies may still land)
            if (is_softmax) {
                if (row_active) {
#pragma unroll
                    for (int c = 0; c < kOCols / 4; ++c) {
                        const int pc = (half * (kOCols / 4) + c) ^ (r & 31);
                        *reinterpret_cast<float4*>(opart + r * kD + pc * 4) =
                            make_float4(o_acc[c * 4], o_acc[c * 4 + 1], o_acc[c * 4 + 2], o_acc[c * 4 + 3]);
                    }
                }
                if (half == 0) row_ml[r] = make_float2(m_run, l_run);
            }
            cluster.sync();
            const int per = (m_valid + (int)CS - 1) / (int)CS;
            const int rbeg = (int)crank * per;
            const int nmy = max(0, min(m_valid, rbeg + per) - rbeg);
            // one round of remote loads per owned row: a warp takes the row, lane c its 16-byte chunk c of
            // every peer's partial O and, for c below the cluster size, peer c's (m, l); the weights then
            // go round the warp by shuffles.  With more owned rows than warps a warp takes two rows per pass
            // (rows w and w + 6 of warp w), so up to twelve owned rows take one pass
            static_assert(kD / 4 == 32 && kThreads % 32 == 0, "a warp's 32 items are one row");
            const int nitems = nmy * (kD / 4);
            // one pass: the row of `item` and (PAIR, when present) the row six further, their loads in flight
            // together and their shuffle chains interleaved
            auto merge_pass = [&](auto pair_tag, int item) {
                constexpr bool PAIR = decltype(pair_tag)::value;
                const bool two = PAIR && item + kThreads < nitems;  // warp-uniform
                const int c = item % (kD / 4);
                const int rowa = rbeg + item / (kD / 4), rowb = rowa + kThreads / 32;
                float4 va[kMaxCluster], vb[kMaxCluster];
                const float* srca = opart + rowa * kD + ((c ^ (rowa & 31)) * 4);
                const float* srcb = opart + rowb * kD + ((c ^ (rowb & 31)) * 4);
#pragma unroll
                for (int pr = 0; pr < kMaxCluster; ++pr) {
                    if (pr < (int)CS) va[pr] = *cluster.map_shared_rank(reinterpret_cast<const float4*>(srca), pr);
                    if constexpr (PAIR) {
                        if (pr < (int)CS && two)
                            vb[pr] = *cluster.map_shared_rank(reinterpret_cast<const float4*>(srcb), pr);
                        else
                            vb[pr] = make_float4(0.f, 0.f, 0.f, 0.f);
                    }
                }
                const float2 mla = c < (int)CS ? *cluster.map_shared_rank(&row_ml[rowa], c) : make_float2(-INFINITY, 0.f);
                float2 mlb = make_float2(-INFINITY, 0.f);
                if constexpr (PAIR) {
                    if (c < (int)CS && two) mlb = *cluster.map_shared_rank(&row_ml[rowb], c);
                }
                float Ma = mla.x, Mb = mlb.x;
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) {
                    Ma = fmaxf(Ma, __shfl_xor_sync(0xffffffffu, Ma, o));
                    if constexpr (PAIR) Mb = fmaxf(Mb, __shfl_xor_sync(0xffffffffu, Mb, o));
                }
                const float wla = mla.x == -INFINITY ? 0.f : fast_exp2(mla.x - Ma);
                const float wlb = mlb.x == -INFINITY ? 0.f : fast_exp2(mlb.x - Mb);
                float La = wla * mla.y, Lb = wlb * mlb.y;
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) {
                    La += __shfl_xor_sync(0xffffffffu, La, o);
                    if constexpr (PAIR) Lb += __shfl_xor_sync(0xffffffffu, Lb, o);
                }
                float4 acca = make_float4(0.f, 0.f, 0.f, 0.f), accb = acca;
#pragma unroll
                for (int pr = 0; pr < kMaxCluster; ++pr) {
                    if (pr < (int)CS) {
                        const float wa = __shfl_sync(0xffffffffu, wla, pr);
                        acca.x += wa * va[pr].x;
                        acca.y += wa * va[pr].y;
                        acca.z += wa * va[pr].z;
                        acca.w += wa * va[pr].w;
                        if constexpr (PAIR) {
                            const float wb = __shfl_sync(0xffffffffu, wlb, pr);
                            accb.x += wb * vb[pr].x;
                            accb.y += wb * vb[pr].y;
                            accb.z += wb * vb[pr].z;
                            accb.w += wb * vb[pr].w;
                        }
                    }
                }
                auto store = [&](int row, float4 acc, float M, float Lsum) {
                    const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
                    const int lr = row0 + row;
                    const size_t orow = (size_t)(one.q0 + lr / G) * p.num_q_heads + one.h * G + lr % G;
                    uint2 w2;
                    w2.x = pack_bf16x2(acc.x * inv, acc.y * inv);
                    w2.y = pack_bf16x2(acc.z * inv, acc.w * inv);
                    *reinterpret_cast<uint2*>(p.o + orow * kD + c * 4) = w2;
                    if (p.lse && c == 0) p.lse[orow] = (M + __log2f(Lsum)) * kLn2;
                };
                store(rowa, acca, Ma, La);
                if (two) store(rowb, accb, Mb, Lb);
            };
            if (nmy > kThreads / 32) {  // more owned rows than warps: two rows per warp and pass
                for (int item = tid; item < nitems; item += 2 * kThreads) merge_pass(std::true_type{}, item);
            } else {
                for (int item = tid; item < nitems; item += kThreads) merge_pass(std::false_type{}, item);
            }
            cluster.sync();  // no CTA leaves while peers may still read its shared memory
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
    // A grid of one wave lets its dependents launch from its start (their prologues overlap it: batch-1
    // calls back to back, 9.25 against 9.87 us each); otherwise they launch once every CTA is here or has
    // left.  Released at the start, a grid of two waves followed by the acceptance's statistics (thousands
    // of CTAs, chained by programmatic launch) made a step of the ragged batch take 720-820 us instead of
    // 195, and the flat split's step took 206.8 us instead of 200.3.
    if (!p.early_release) griddep_launch_dependents();
}

// Flat split, second kernel: the units whose tiles were cut between CTA groups.  The CTA of the main
// kernel that holds a cut unit's first tile names it in its work entry; CTA (c, r) here takes work entry
// c and its rows [r * kCombRows, (r + 1) * kCombRows).  Thread (row, 16-byte chunk) merges the partial
// (O, m, l) of the unit's CTAs in order -- O = sum_j 2^(m_j - M) O_j / sum_j 2^(m_j - M) l_j, M the
// largest m_j, as a running merge over batches of kCombBatch partials whose loads are all in flight --
// and writes the bf16 output chunk (and the row's log-sum-exp).
constexpr int kCombRows = 8;
constexpr int kCombThreads = kCombRows * kD / 4;  // 256: one 16-byte chunk of a row each
constexpr int kCombBatch = 8;
__global__ void __launch_bounds__(kCombThreads) attn_combine_kernel(const AttnParams p, int grid_main) {
    __shared__ int32_t gstart[kAttnFlatMaxGrid + 1];  // the CTA groups' ranges: group j has [gstart[j], gstart[j+1])
    griddep_launch_dependents();
    griddep_wait();  // the partials and work entries of the main kernel
    const int tid = threadIdx.x;
    const int G = p.group;
    const int chunks = (p.slot_rows + kCombRows - 1) / kCombRows;
    const int c = blockIdx.x / chunks, r = blockIdx.x - c * chunks;
    const int4 wk = __ldcg(p.work + 2 * c), wk2 = __ldcg(p.work + 2 * c + 1);
    if (wk.x < 0) return;  // CTA c holds no cut unit's first tile (uniform per CTA)
    const int U0 = wk.x, U1 = wk.y, T = wk.z, rows = wk.w, q0 = wk2.x, mt = wk2.y;
    const int h = c % p.num_kv_heads;
    if (r * kCombRows >= rows) return;  // uniform per CTA
    const int ngroups = grid_main / p.num_kv_heads;
    for (int j = tid; j <= ngroups; j += kCombThreads) gstart[j] = (int)((long long)j * T / ngroups);
    __syncthreads();
    // the group whose range holds the unit's last tile: the last j with gstart[j] <= U1 - 1
    int lo = c / p.num_kv_heads, hi = ngroups;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (gstart[mid] <= U1 - 1) lo = mid; else hi = mid;
    }
    const int j0 = c / p.num_kv_heads, j1 = lo;
    const int rl = r * kCombRows + tid / (kD / 4);  // the row within the unit
    const int c4 = tid % (kD / 4);                  // its 16-byte chunk
    if (rl >= rows) return;
    const size_t slot_floats = (size_t)p.slot_rows * (kD + 2);
    const size_t ml_off = (size_t)p.slot_rows * kD + 2 * rl;
    float M = -INFINITY, Lsum = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int jb = j0; jb <= j1; jb += kCombBatch) {
        float2 ml[kCombBatch];
        float4 v[kCombBatch];
#pragma unroll
        for (int k = 0; k < kCombBatch; ++k) {
            const int j = jb + k;
            ml[k] = make_float2(-INFINITY, 0.f);
            v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (j <= j1 && gstart[j] < gstart[j + 1]) {
                // CTA (group j, head h): its first stretch (slot 0) unless its range began before the unit
                const float* sp =
                    p.part + (size_t)(2 * (j * p.num_kv_heads + h) + (gstart[j] >= U0 ? 0 : 1)) * slot_floats;
                ml[k] = __ldcg(reinterpret_cast<const float2*>(sp + ml_off));
                v[k] = __ldcg(reinterpret_cast<const float4*>(sp + (size_t)rl * kD + c4 * 4));
            }
        }
#pragma unroll
        for (int k = 0; k < kCombBatch; ++k) {
            if (ml[k].x == -INFINITY) continue;  // nothing (or no visible key) in this partial
            if (ml[k].x > M) {
                const float sc = M == -INFINITY ? 0.f : fast_exp2(M - ml[k].x);
                Lsum *= sc;
                acc.x *= sc;
                acc.y *= sc;
                acc.z *= sc;
                acc.w *= sc;
                M = ml[k].x;
            }
            const float w = fast_exp2(ml[k].x - M);
            Lsum += w * ml[k].y;
            acc.x += w * v[k].x;
            acc.y += w * v[k].y;
            acc.z += w * v[k].z;
            acc.w += w * v[k].w;
        }
    }
    const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
    const int lr = mt * kM + rl;
    const size_t orow = (size_t)(q0 + lr / G) * p.num_q_heads + h * G + lr % G;
    uint2 w2;
    w2.x = pack_bf16x2(acc.x * inv, acc.y * inv);
    w2.y = pack_bf16x2(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(p.o + orow * kD + c4 * 4) = w2;
    if (p.lse && c4 == 0) p.lse[orow] = (M + __log2f(Lsum)) * 0.6931471805599453f;
}

// --------------------------------------------------------------------------- fp32 SIMT path
// One warp per (query row, query head): online softmax over the row's visible keys in
// chunks of 32 (lane = key), lane d-slices of the output.
constexpr int kF32MaxD = 128;

__global__ void __launch_bounds__(128) attn_f32_simt_kernel(const float* __restrict__ q, const float* __restrict__ k,
                                                            const float* __restrict__ v, float* __restrict__ o,
                                                            float* __restrict__ lse, const int32_t* __restrict__ cu_q,
                                                            const int32_t* __restrict__ cu_kv, int num_seqs,
                                                            int total_q, int hq, int hkv, int D, int causal,
                                                            float scale) {
    __shared__ float qs[4][kF32MaxD];
    griddep_launch_dependents();
    griddep_wait();
    const int wib = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long row = (long long)blockIdx.x * 4 + wib;
    if (row >= (long long)total_q * hq) return;
    const int t = (int)(row / hq), h = (int)(row % hq);
    const int g = hq / hkv, kvh = h / g;
    int lo = 0, hi = num_seqs;  // sequence containing query t: cu_q[s] <= t < cu_q[s+1]
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (cu_q[mid] <= t) lo = mid; else hi = mid;
    }
    const int s = lo;
    const int B = cu_q[s + 1] - cu_q[s];
    const int i = t - cu_q[s];
    const int kv0 = cu_kv[s];
    const int n = cu_kv[s + 1] - kv0;
    const int L = n - B;
    const int nk = causal ? L + i + 1 : n;
    for (int d = lane; d < D; d += 32) qs[wib][d] = q[((size_t)t * hq + h) * D + d];
    __syncwarp();
    float m = -INFINITY, l = 0.f;
    float acc[kF32MaxD / 32];
#pragma unroll
    for (int e = 0; e < kF32MaxD / 32; ++e) acc[e] = 0.f;
    for (int j0 = 0; j0 < nk; j0 += 32) {
        const int j = j0 + lane;
        float sc = -INFINITY;
        if (j < nk) {
            const float* kr = k + ((size_t)(kv0 + j) * hkv + kvh) * D;
            float dot = 0.f;
            for (int d = 0; d < D; ++d) dot = fmaf(qs[wib][d], kr[d], dot);
            sc = dot * scale;
        }
        float cm = sc;
        for (int off = 16; off; off >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, off));
        const float m_new = fmaxf(m, cm);
        const float alpha = (m == -INFINITY) ? 0.f : expf(m - m_new);
        const float pj = (j < nk) ? expf(sc - m_new) : 0.f;
        float ps = pj;
        for (int off = 16; off; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
        l = l * alpha + ps;
#pragma unroll
        for (int e = 0; e < kF32MaxD / 32; ++e) acc[e] *= alpha;
        const int cnt = min(32, nk - j0);
        for (int jj = 0; jj < cnt; ++jj) {
            const float pjj = __shfl_sync(0xffffffffu, pj, jj);
            const float* vr = v + ((size_t)(kv0 + j0 + jj) * hkv + kvh) * D;
#pragma unroll
            for (int e = 0; e < kF32MaxD / 32; ++e) {
                const int d = lane + e * 32;
                if (d < D) acc[e] = fmaf(pjj, vr[d], acc[e]);
            }
        }
        m = m_new;
    }
#pragma unroll
    for (int e = 0; e < kF32MaxD / 32; ++e) {
        const int d = lane + e * 32;
        if (d < D) o[((size_t)t * hq + h) * D + d] = acc[e] / l;
    }
    if (lse && lane == 0) lse[(size_t)t * hq + h] = m + logf(l);
}

}  // namespace

namespace {
// Rows of one partial slot of the flat split: a unit's query rows (at most one 128-row tile), rounded
// up to 16 so that every slot starts on a 16-byte boundary.
int flat_slot_rows(int max_q_len, int group) {
    const long long rows = (long long)max_q_len * group;
    return (int)((std::min<long long>(kM, rows) + 15) / 16 * 16);
}
}  // namespace

size_t attention_flat_scratch_bytes(int max_q_len, int group) {
    if (max_q_len < 1 || group < 1) return 0;
    return (size_t)2 * kAttnFlatMaxGrid * flat_slot_rows(max_q_len, group) * (kD + 2) * sizeof(float) +
           (size_t)2 * kAttnFlatMaxGrid * sizeof(int4);
}

int launch_attention_bf16(const AttentionArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    if (a.head_dim != kD) return BP_ERR_UNSUPPORTED;
    const int G = a.num_q_heads / a.num_kv_heads;
    const int m_tiles = (a.max_q_len * G + kM - 1) / kM;
    const long long units = (long long)a.num_seqs * a.num_kv_heads * m_tiles;
    if (units == 0 || a.total_q == 0) return BP_OK;

    CUtensorMap qmap, kmap, vmap;
    // Q: box of (64 columns) x (G heads) x (128/G block positions) = the packed 128-row tile; for units
    // of at most 64 rows (spread layout) four boxes of 16 rows (16/G block positions) instead
    const bool q_tma = (kM % G == 0);
    const bool spread = q_tma && 16 % G == 0 && (long long)a.max_q_len * G <= 64;
    if (q_tma) {
        const cuuint64_t qdims[3] = {(cuuint64_t)kD, (cuuint64_t)a.num_q_heads, (cuuint64_t)a.total_q};
        const cuuint64_t qstrides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)a.num_q_heads * kD * 2};
        const cuuint32_t qbox[3] = {64, (cuuint32_t)G, (cuuint32_t)((spread ? 16 : kM) / G)};
        const int rq = encode_tensor_map(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), qdims,
                                         qstrides, qbox, CU_TENSOR_MAP_SWIZZLE_128B);
        if (rq != BP_OK) return rq;
    }
    // K/V: contiguous rows, or the page pool with boxes of one page (at most one 128-key tile)
    const bool paged = a.block_table != nullptr;
    const cuuint64_t kv_rows = paged ? (cuuint64_t)a.num_pages * a.page_size : (cuuint64_t)a.total_kv;
    const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)a.num_kv_heads, kv_rows};
    const cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)a.num_kv_heads * kD * 2};
    const cuuint32_t box[3] = {64, 1, (cuuint32_t)(paged && a.page_size < kTileN ? a.page_size : kTileN)};
    int rc = encode_tensor_map(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.k), dims, strides,
                               box, CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != BP_OK) return rc;
    rc = encode_tensor_map(&vmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.v), dims, strides, box,
                           CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != BP_OK) return rc;

    AttnParams p;
    p.q = static_cast<const __nv_bfloat16*>(a.q);
    p.o = static_cast<__nv_bfloat16*>(a.o);
    p.lse = a.lse;
    p.cu_q = a.cu_q;
    p.cu_kv = a.cu_kv;
    p.num_seqs = a.num_seqs;
    p.total_q = a.total_q;
    p.total_kv = a.total_kv;
    p.num_q_heads = a.num_q_heads;
    p.num_kv_heads = a.num_kv_heads;
    p.group = G;
    p.m_tiles = m_tiles;
    p.causal = a.mask == BP_MASK_CAUSAL_BLOCK;
    p.scale_log2 = a.scale * 1.4426950408889634f;
    p.q_tma = q_tma ? 1 : 0;
    p.block_table = a.block_table;
    p.pages_per_seq = paged ? a.pages_per_seq : 0;
    p.page_shift = 0;
    while (paged && (1 << p.page_shift) < a.page_size) ++p.page_shift;
    p.part = nullptr;
    p.work = nullptr;
    p.slot_rows = flat_slot_rows(a.max_q_len, G);
    p.early_release = 0;
    p.err = a.err_word;
    if (!q_tma) qmap = kmap;  // unused by the kernel

    // once per device (under a lock: calls may come from several host threads): opt in to the
    // shared-memory size and non-portable clusters, and record how many clusters of each size (1..16)
    // the GPU can keep resident at once (queried outside any graph capture; the answer reflects how
    // the SMs are grouped into GPCs)
    static std::mutex cfg_mu;
    static bool configured[64] = {};
    static int max_active_dev[64][kMaxCluster + 1];
    if (dev.device < 0 || dev.device >= 64) return BP_ERR_UNSUPPORTED;
    int max_active[kMaxCluster + 1];
    std::unique_lock<std::mutex> cfg_lock(cfg_mu);
    if (!configured[dev.device]) {
        for (auto kern : {attn_bf16_tc_kernel<false, false, false>, attn_bf16_tc_kernel<true, false, false>,
                          attn_bf16_tc_kernel<false, true, false>, attn_bf16_tc_kernel<true, true, false>,
                          attn_bf16_tc_kernel<false, false, true>, attn_bf16_tc_kernel<true, false, true>,
                          attn_bf16_tc_kernel<false, true, true>, attn_bf16_tc_kernel<true, true, true>})
            if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kDynSmem) != cudaSuccess ||
                cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
                cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared) != cudaSuccess)
                return BP_ERR_CUDA;
        for (int cs = 1; cs <= kMaxCluster; ++cs) {
            cudaLaunchConfig_t probe = {};
            cudaLaunchAttribute pa[1];
            probe.gridDim = dim3(cs, 1, 1);
            probe.blockDim = dim3(kThreads, 1, 1);
            probe.dynamicSmemBytes = kDynSmem;
            pa[0].id = cudaLaunchAttributeClusterDimension;
            pa[0].val.clusterDim.x = cs;
            pa[0].val.clusterDim.y = 1;
            pa[0].val.clusterDim.z = 1;
            probe.attrs = pa;
            probe.numAttrs = 1;
            int n_clusters = 0;
            if (cudaOccupancyMaxActiveClusters(&n_clusters, attn_bf16_tc_kernel<false, false, false>, &probe) !=
                cudaSuccess) {
                cudaGetLastError();
                n_clusters = 0;
            }
            max_active_dev[dev.device][cs] = n_clusters;
        }
        configured[dev.device] = true;
    }
    for (int c = 0; c <= kMaxCluster; ++c) max_active[c] = max_active_dev[dev.device][c];
    cfg_lock.unlock();

    const int max_tiles = (a.max_kv_len + kTileN - 1) / kTileN;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kDynSmem;
    cfg.stream = stream;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;

    // cluster split: a split of each unit's keys for which every unit's cluster is resident in the same
    // wave (a unit left for a second wave would double the time).  The tiles of the longest unit per CTA
    // set the time: minimise them; among equal counts take the smallest cluster whose merge needs the
    // fewest passes (a pass merges up to 12 owned rows per CTA).  A cluster's barriers and merge cost
    // about three tiles of one CTA's chain (batch 1, Qwen3-4B heads: 2 tiles 5.3 us alone against
    // 7.3-9.9 us in clusters; 4 tiles 7.6 us alone, 7.4 us in clusters of 6), so a split that saves
    // fewer than three tiles stays whole
    const int m_rows = std::min(kM, a.max_q_len * G);
    int cs = 1, best = max_tiles, best_pass = 0;
    for (int c = 2; c <= kMaxCluster; ++c) {
        if (c > max_tiles || units > max_active[c] || units * c > dev.sm_count) continue;
        const int per = (max_tiles + c - 1) / c;
        const int passes = ((m_rows + c - 1) / c + 11) / 12;
        if (per < best || (per == best && cs > 1 && passes < best_pass)) {
            best = per;
            cs = c;
            best_pass = passes;
        }
    }
    if (cs > 1 && max_tiles - best < 3) cs = 1;

    // flat split: the tiles of every sequence's query tiles cut evenly over groups of CTAs, one CTA per KV
    // head and per SM (at most kAttnFlatMaxGrid in all, and no more groups than one head has tiles); units
    // cut between groups are merged by a second kernel.  It needs the Q tile by TMA, the sequences'
    // offsets in shared memory and the workspace's partial slots and work entries.  Measured on this GPU,
    // it gains where the cluster split leaves SMs idle while every CTA of the flat split streams a long
    // run (8 x 32K keys: 170 vs 175 us), and where the cluster split needs three or more waves (64 x 528
    // keys: 46 vs 50 us); elsewhere the second kernel and the stretch boundaries cost more than the idle
    // SMs (1 x 2K keys: 13.8 vs 9.3 us; 16 x 4K: 60 vs 52 us; the ragged 32: 109 vs 100 us).
    // BP_ATTENTION_SPLIT=flat or =cluster overrides the choice, =cluster:N also the cluster size (for tests
    // and measurements).
    const long long tiles_bound = (long long)a.num_seqs * m_tiles * max_tiles;
    const int ngroups = (int)std::min<long long>(std::min(dev.sm_count, kAttnFlatMaxGrid) / a.num_kv_heads,
                                                 tiles_bound);
    const int flat_grid = ngroups * a.num_kv_heads;
    const bool flat_ok = q_tma && a.num_seqs <= kMaxOrderedSeqs && a.scratch != nullptr &&
                         a.scratch_bytes >= attention_flat_scratch_bytes(a.max_q_len, G) && ngroups >= 1;
    const long long cluster_ctas = units * cs;
    bool flat = flat_ok && ((cluster_ctas * 10 <= 9LL * dev.sm_count && tiles_bound >= 64LL * ngroups) ||
                            cluster_ctas >= 3LL * dev.sm_count);
    if (const char* force = getenv("BP_ATTENTION_SPLIT")) {
        if (strcmp(force, "flat") == 0) {
            flat = flat_ok;
        } else if (strncmp(force, "cluster", 7) == 0) {
            flat = false;
            // cluster:N forces clusters of N CTAs when every unit's cluster is then resident in one wave
            const int c = force[7] == ':' ? atoi(force + 8) : 0;
            if (c >= 2 && c <= kMaxCluster && units <= max_active[c] && units * c <= dev.sm_count) cs = c;
        }
    }
    cudaError_t e;
    if (flat) {
        p.part = static_cast<float*>(a.scratch);
        p.work = reinterpret_cast<int4*>(p.part + (size_t)2 * kAttnFlatMaxGrid * p.slot_rows * (kD + 2));
        cfg.gridDim = dim3((unsigned)flat_grid, 1, 1);
        cfg.attrs = &attr[1];
        cfg.numAttrs = 1;
        if (paged) e = spread ? cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<true, true, true>, qmap, kmap, vmap, p)
                              : cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<true, false, true>, qmap, kmap, vmap, p);
        else e = spread ? cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<false, true, true>, qmap, kmap, vmap, p)
                        : cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<false, false, true>, qmap, kmap, vmap, p);
        if (e != cudaSuccess) return BP_ERR_CUDA;
        if (max_tiles <= 1) return BP_OK;  // every unit is one tile: none is cut between CTAs
        cudaLaunchConfig_t cc = {};
        cc.gridDim = dim3((unsigned)(flat_grid * ((p.slot_rows + kCombRows - 1) / kCombRows)), 1, 1);
        cc.blockDim = dim3(kCombThreads, 1, 1);
        cc.stream = stream;
        cc.attrs = &attr[1];
        cc.numAttrs = 1;
        return cudaLaunchKernelEx(&cc, attn_combine_kernel, p, flat_grid) == cudaSuccess ? BP_OK : BP_ERR_CUDA;
    }

    cfg.gridDim = dim3((unsigned)(units * cs), 1, 1);
    p.early_release = units <= max_active[cs] && units * cs <= dev.sm_count;  // one wave
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    if (paged) e = spread ? cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<true, true, false>, qmap, kmap, vmap, p)
                          : cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<true, false, false>, qmap, kmap, vmap, p);
    else e = spread ? cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<false, true, false>, qmap, kmap, vmap, p)
                    : cudaLaunchKernelEx(&cfg, attn_bf16_tc_kernel<false, false, false>, qmap, kmap, vmap, p);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    return BP_OK;
}

int launch_attention_f32(const AttentionArgs& a, cudaStream_t stream) {
    if (a.head_dim > kF32MaxD) return BP_ERR_UNSUPPORTED;
    const long long rows = (long long)a.total_q * a.num_q_heads;
    if (rows == 0) return BP_OK;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)((rows + 3) / 4), 1, 1);
    cfg.blockDim = dim3(128, 1, 1);
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(
        &cfg, attn_f32_simt_kernel, static_cast<const float*>(a.q), static_cast<const float*>(a.k),
        static_cast<const float*>(a.v), static_cast<float*>(a.o), a.lse, a.cu_q, a.cu_kv, a.num_seqs, a.total_q,
        a.num_q_heads, a.num_kv_heads, a.head_dim, (int)(a.mask == BP_MASK_CAUSAL_BLOCK), a.scale);
    return e == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

// --------------------------------------------------------------------------- paged KV append
// Writes each sequence's new K/V rows (its block) into their slots of the paged cache: new row
// i of sequence s is key L_s + i, with L_s = (cu_kv[s+1] - cu_kv[s]) - (cu_new[s+1] - cu_new[s]).
// One warp per (new row, KV head): 16-byte copies of the K row and of the V row.
__global__ void __launch_bounds__(256) kv_append_kernel(uint8_t* __restrict__ kc, uint8_t* __restrict__ vc,
                                                        const uint8_t* __restrict__ kn,
                                                        const uint8_t* __restrict__ vn,
                                                        const int32_t* __restrict__ cu_new,
                                                        const int32_t* __restrict__ cu_kv,
                                                        const int32_t* __restrict__ bt, int pages_per_seq,
                                                        int page_shift, int num_seqs, int total_new, int hkv,
                                                        int row_bytes) {
    griddep_launch_dependents();
    griddep_wait();
    const int warp = (int)((blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (warp >= total_new * hkv) return;
    const int t = warp / hkv, hh = warp % hkv;
    int lo = 0, hi = num_seqs;  // largest s with cu_new[s] <= t
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(cu_new + mid) <= t) lo = mid; else hi = mid;
    }
    const int s = lo;
    const int nb = __ldg(cu_new + s + 1) - __ldg(cu_new + s);
    const int len = __ldg(cu_kv + s + 1) - __ldg(cu_kv + s);
    const int pos = len - nb + (t - __ldg(cu_new + s));
    const long long page = __ldg(bt + (size_t)s * pages_per_seq + (pos >> page_shift));
    const long long slot = (page << page_shift) + (pos & ((1 << page_shift) - 1));
    const size_t dst = ((size_t)slot * hkv + hh) * row_bytes;
    const size_t src = ((size_t)t * hkv + hh) * row_bytes;
    for (int b = lane * 16; b < row_bytes; b += 32 * 16) {
        *reinterpret_cast<uint4*>(kc + dst + b) = *reinterpret_cast<const uint4*>(kn + src + b);
        *reinterpret_cast<uint4*>(vc + dst + b) = *reinterpret_cast<const uint4*>(vn + src + b);
    }
}

int launch_kv_append(const KvAppendArgs& a, cudaStream_t stream) {
    if (a.total_new == 0) return BP_OK;
    int shift = 0;
    while ((1 << shift) < a.page_size) ++shift;
    const long long warps = (long long)a.total_new * a.num_kv_heads;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)((warps + 7) / 8), 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kv_append_kernel, static_cast<uint8_t*>(a.k_cache), static_cast<uint8_t*>(a.v_cache),
                              static_cast<const uint8_t*>(a.k_new), static_cast<const uint8_t*>(a.v_new), a.cu_new,
                              a.cu_kv, a.block_table, a.pages_per_seq, shift, a.num_seqs, a.total_new,
                              a.num_kv_heads, a.row_bytes) == cudaSuccess
               ? BP_OK
               : BP_ERR_CUDA;
}

}  // namespace bp
