// Lossless acceptance for many rows at once (a batch of sequences): the same rule as accept.cu --
// standard speculative sampling (accept x_i with probability min(1, p_i(x_i) / q_i(x_i)), redraw at
// the first rejection k from norm(max(0, p_k - q_k)), a bonus draw from p_gamma when every draft is
// accepted, greedy at T = 0; Section 2.1 / Figure 1) -- arranged for throughput instead of latency.
//
// The cluster kernel of accept.cu gives every target row a cluster, brings the row into shared memory
// once and computes every row's draw speculatively; with many rows its clusters run in waves, each
// paying the per-row chain of exchanges.  Here:
//   1. stats: one CTA per 16384-entry chunk of every target and drafter row streams the chunk once
//      (coalesced 16-byte loads) and writes the chunk's (scaled max, sum of 2^(l*log2e/T - max)) --
//      at T = 0 its (max, lowest index) -- so the whole batch is one HBM-bound pass;
//   2. T = 0: decide: one warp per sequence, one lane per block position, merges its row's chunk
//      statistics in a fixed order and compares the drafted token with the argmax; the first mismatch k
//      and the outputs (the emitted argmax too).  (Taking the decisions in the statistics kernel, in the
//      CTA that completes a sequence, costs every CTA a gpu-scope ticket behind its store: measured
//      slower for large batches);
//   2. T > 0: draw: one CTA per chunk of each sequence's draw row pair (or per part of a chunk, when the
//      chunks alone would leave SMs idle).  Its first warp derives the sequence's decisions the same
//      way (ratios a_i, the first rejection k -- the rejected row k and its drafter row, or the bonus
//      row -- one CTA writing the outputs); then every thread forms the part's segment masses of
//      max(0, p_k - q_k) and of p_k in exact 2^-52 fixed point; the last CTA of the sequence (ticket)
//      finds the part and the 128-entry segment where the inverse CDF crosses u_s * total from the
//      stored masses, then the entry from that segment's 128 logits, and writes the emitted token.
// Only the one draw row pair per sequence is read twice.  Every kernel of the chain launches with
// programmatic dependent launch.  The statistics kernel releases the decisions (or the draw) only once
// its own grid-dependency wait has returned, i.e. once every kernel before the chain is complete, so
// their decision warps load the inputs that the statistics kernel does not write (offsets, drafted
// tokens, uniforms, the drafted tokens' logits) before their own wait.
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "ptx_sm103.cuh"
#include "softmax_math.cuh"

namespace bp {
namespace {

constexpr int kBThreads = 256;
constexpr int kBChunk = 16384;                 // vocabulary entries per chunk
constexpr int kBVec = kBChunk / 4 / kBThreads;  // 16-byte groups per thread: 16 (64 entries)
constexpr int kBSegs = kBVec;                  // 128-entry segments per warp of a chunk
constexpr int kMaxDrawSplit = 4;               // parts a draw chunk may be cut into

struct BatchParams {
    const float* target;  // [rows_t][vocab]
    const float* draft;   // [total_draft][vocab] (T > 0)
    const int32_t* tokens;
    const int32_t* cu_draft;
    int num_seqs, total_draft, rows_t, vocab, chunks;
    int nparts;           // statistics per row in part: the chunks, or 1 for rows merged beforehand
    float c2;  // log2(e) / T; 0 at T = 0
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    float2* part;      // [rows][nparts] partial statistics (T = 0: value, index bits)
    ulonglong2* ctot;  // [num_seqs][chunks * parts] draw masses of r and p of the chunks' parts (fixed point)
    unsigned long long* segm;  // [num_seqs][chunks][2][128] their segment masses
    int* tickets;      // [num_seqs], zero between calls
    int inputs_early;  // every input was complete when the statistics kernel released this one (DecideIn)
    unsigned int* err;
};

__device__ __forceinline__ int ticket_acq_rel(int* addr) {
    int old;
    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], 1;" : "=r"(old) : "l"(addr) : "memory");
    return old;
}

// Row r of the stacked rows: target rows first, then the drafter's rows.
__device__ __forceinline__ const float* row_ptr(const BatchParams& p, int r) {
    return r < p.rows_t ? p.target + (size_t)r * p.vocab : p.draft + (size_t)(r - p.rows_t) * p.vocab;
}

// Entry e (16-byte group q, element k) of a chunk held by thread t: q = t + 256 j, so a warp's
// groups for one j are 128 consecutive entries (segment (j, warp)) and segments in (j, warp) order
// are in entry order.
template <bool VEC>
__device__ __forceinline__ float4 load4(const float* __restrict__ src, int e, int n) {
    if (VEC)
        return e < n ? __ldcs(reinterpret_cast<const float4*>(src + e))
                     : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    return make_float4(e < n ? __ldcs(src + e) : -INFINITY, e + 1 < n ? __ldcs(src + e + 1) : -INFINITY,
                       e + 2 < n ? __ldcs(src + e + 2) : -INFINITY, e + 3 < n ? __ldcs(src + e + 3) : -INFINITY);
}
template <bool VEC>
__device__ __forceinline__ void load_chunk(const float* __restrict__ src, int n, int tid,
                                           float4 (&v)[kBVec]) {
#pragma unroll
    for (int j = 0; j < kBVec; ++j) v[j] = load4<VEC>(src, 4 * (tid + j * kBThreads), n);
}

// The draw of a sequence: its row pair, the constants of its weights and the output slot.
struct DrawPair {
    int trow, drow;  // drow < 0: a bonus draw from p alone
    float Mt, izt, Md, izd;
    int out;         // the emitted token's slot in out_tokens
};

// ---- 1. chunk statistics of every row
template <bool GREEDY, bool VEC>
__global__ void __launch_bounds__(kBThreads) batch_stats_kernel(const BatchParams p) {
    __shared__ float2 red[kBThreads / 32];
    griddep_wait();
    griddep_launch_dependents();  // after the wait: the decisions kernel may read inputs early (DecideIn)
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int row = blockIdx.x / p.chunks, chunk = blockIdx.x - row * p.chunks;
    const int v0 = chunk * kBChunk, n = min(kBChunk, p.vocab - v0);
    float4 v[kBVec];
    load_chunk<VEC>(row_ptr(p, row) + v0, n, tid, v);
    float a0, a1;  // (scaled max, sum) or (value, index bits)
    if (GREEDY) {
        float best = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int j = 0; j < kBVec; ++j) {  // increasing entries: strict > keeps the lowest index
            const int e = v0 + 4 * (tid + j * kBThreads);
            if (v[j].x > best) { best = v[j].x; bi = e; }
            if (v[j].y > best) { best = v[j].y; bi = e + 1; }
            if (v[j].z > best) { best = v[j].z; bi = e + 2; }
            if (v[j].w > best) { best = v[j].w; bi = e + 3; }
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            amax_merge(best, bi, __shfl_xor_sync(0xffffffffu, best, o),
                       __shfl_xor_sync(0xffffffffu, bi, o));
        a0 = best;
        a1 = __int_as_float(bi);
    } else {
        float m = -INFINITY;
#pragma unroll
        for (int j = 0; j < kBVec; ++j)
            m = fmaxf(m, fmaxf(fmaxf(v[j].x, v[j].y), fmaxf(v[j].z, v[j].w)));
        float s = 0.f;
        if (m != -INFINITY) {  // 2^(l*c2 - m) of every entry, m the thread's scaled maximum
            m = __fmul_rn(m, p.c2);
#pragma unroll
            for (int j = 0; j < kBVec; ++j)
                s += (ex2(__fmaf_rn(v[j].x, p.c2, -m)) + ex2(__fmaf_rn(v[j].y, p.c2, -m))) +
                     (ex2(__fmaf_rn(v[j].z, p.c2, -m)) + ex2(__fmaf_rn(v[j].w, p.c2, -m)));
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            lse_merge(m, s, __shfl_xor_sync(0xffffffffu, m, o), __shfl_xor_sync(0xffffffffu, s, o));
        a0 = m;
        a1 = s;
    }
    if (lane == 0) red[warp] = make_float2(a0, a1);
    __syncthreads();
    if (tid == 0) {
        float2 r = red[0];
        for (int w = 1; w < kBThreads / 32; ++w) {
            if (GREEDY) {
                int ri = __float_as_int(r.y);
                amax_merge(r.x, ri, red[w].x, __float_as_int(red[w].y));
                r.y = __int_as_float(ri);
            } else {
                lse_merge(r.x, r.y, red[w].x, red[w].y);
            }
        }
        p.part[(size_t)row * p.chunks + chunk] = r;
    }
}


// Statistics of row r from its chunks', merged in chunk order by one lane (the order every path uses),
// all chunks' loads in flight at once (up to kMergeBatch chunks, i.e. vocabularies up to 262144, in
// one round trip).  GREEDY: (max, lowest index); else (scaled max, sum of 2^(l*c2 - max)).
constexpr int kMergeBatch = 16;
template <bool GREEDY>
__device__ __forceinline__ void load_row_parts(const BatchParams& p, int r, int c0, float2 (&x)[kMergeBatch]) {
    const float2 ident = make_float2(-INFINITY, GREEDY ? __int_as_float(INT_MAX) : 0.f);
#pragma unroll
    for (int q = 0; q < kMergeBatch; ++q)
        x[q] = r >= 0 && c0 + q < p.nparts ? __ldcg(&p.part[(size_t)r * p.nparts + c0 + q]) : ident;
}
template <bool GREEDY>
__device__ __forceinline__ void merge_parts(float2& acc, const float2 (&x)[kMergeBatch]) {
#pragma unroll
    for (int q = 0; q < kMergeBatch; ++q) {
        if (GREEDY) {
            int ai = __float_as_int(acc.y);
            amax_merge(acc.x, ai, x[q].x, __float_as_int(x[q].y));
            acc.y = __int_as_float(ai);
        } else {
            lse_merge(acc.x, acc.y, x[q].x, x[q].y);
        }
    }
}
// Both rows r1, r2 (r2 < 0: none) at once: every load of the first batch is issued before any merge.
template <bool GREEDY>
__device__ __forceinline__ void merge_rows(const BatchParams& p, int r1, int r2, float2& a1, float2& a2) {
    const float2 ident = make_float2(-INFINITY, GREEDY ? __int_as_float(INT_MAX) : 0.f);
    a1 = ident;
    a2 = ident;
    for (int c0 = 0; c0 < p.nparts; c0 += kMergeBatch) {
        float2 x1[kMergeBatch], x2[kMergeBatch];
        load_row_parts<GREEDY>(p, r1, c0, x1);
        load_row_parts<GREEDY>(p, r2, c0, x2);
        merge_parts<GREEDY>(a1, x1);
        merge_parts<GREEDY>(a2, x2);
    }
}

// A decision warp's inputs for block positions 0..31 of sequence s: the sequence's offsets, lane i's
// drafted token, its acceptance uniform and (T > 0) that token's target and drafter logits.  None of
// them is written by the statistics kernel, and the statistics kernel releases its dependents only
// after its own grid-dependency wait (every earlier kernel complete), so behind it (`inputs_early`)
// the warp loads them before its grid-dependency wait, while the statistics still stream; behind the
// streamed LM head, which writes the logits, right after it.  That takes two dependent round trips
// (offsets -> tokens -> logits) off the path behind the statistics.
struct DecideIn {
    int d0, g, x;
    float u, tx, dx;
};
template <bool GREEDY>
__device__ __forceinline__ DecideIn decide_inputs(const BatchParams& p, int s, int lane) {
    DecideIn q;
    q.d0 = p.cu_draft[s];
    q.g = p.cu_draft[s + 1] - q.d0;
    const bool draft = lane < q.g;
    q.x = draft ? p.tokens[q.d0 + lane] : -1;
    q.u = !GREEDY && draft ? p.u_accept[q.d0 + lane] : 1.f;
    q.tx = -INFINITY;
    q.dx = -INFINITY;
    if (!GREEDY && draft && q.x >= 0 && q.x < p.vocab) {
        q.tx = p.target[(size_t)(q.d0 + s + lane) * p.vocab + q.x];
        q.dx = p.draft[(size_t)(q.d0 + lane) * p.vocab + q.x];
    }
    return q;
}

// Greedy decisions (T = 0) of sequence s by one warp, one lane per block position (32 at a time): lane
// i <= gamma merges target row i's (max, lowest index) from its chunks' and compares drafted token i
// with it; the first mismatch k by ballot; the emitted token is row k's argmax (the bonus row's when
// every draft matches).
__device__ __forceinline__ void decide_greedy(const BatchParams& p, int s, int lane, const DecideIn& in) {
    const int d0 = in.d0, g = in.g, t0 = d0 + s;
    int k = g, emitted = 0, bonus = 0;
    for (int i0 = 0; i0 <= g; i0 += 32) {
        const int i = i0 + lane;
        const int x = i0 == 0 ? in.x : (i < g ? p.tokens[d0 + i] : -1);
        float2 st, none;
        merge_rows<true>(p, i <= g ? t0 + i : -1, -1, st, none);
        int am = __float_as_int(st.y);
        if (am >= p.vocab) am = 0;  // every entry -inf: index 0
        bool rej = false;
        if (i < g) {
            const bool valid = x >= 0 && x < p.vocab;
            if (!valid) raise_error(p.err, kErrDeviceArg);
            rej = !(valid && x == am);
            if (p.accept_prob) p.accept_prob[d0 + i] = rej ? 0.f : 1.f;
        }
        if (g - i0 < 32) bonus = __shfl_sync(0xffffffffu, am, g - i0);
        const unsigned b = __ballot_sync(0xffffffffu, rej);
        if (b && k == g) {
            const int l = __ffs(b) - 1;
            k = i0 + l;
            emitted = __shfl_sync(0xffffffffu, am, l);
        }
    }
    if (k == g) emitted = bonus;
    for (int j = lane; j <= g; j += 32) {
        if (j < k) p.out_tokens[t0 + j] = p.tokens[d0 + j];
        else if (j > k) p.out_tokens[t0 + j] = -1;
        else p.out_tokens[t0 + j] = emitted;
    }
    if (lane == 0) p.n_accepted[s] = k;
}

// The decisions of sequence s at T > 0 by one warp, one lane per block position (32 at a time): lane
// i < gamma takes drafted position i -- its target and drafter row statistics, a_i -- and lane i =
// gamma the bonus row's statistics; the first rejection k by ballot; then the draw's row pair and the
// constants of its weights into *d (lane 0).  Every CTA of the sequence's draw derives the same k; the
// writer CTA also writes n_accepted, accept_prob and the out_tokens slots other than the emitted
// token's, and reports draft tokens outside the vocabulary; the others stop at the first block of 32
// positions that holds a rejection.
__device__ __forceinline__ void decide_draw(const BatchParams& p, int s, int lane, bool writer, DrawPair* d,
                                            const DecideIn& in) {
    const int d0 = in.d0, g = in.g, t0 = d0 + s;
    int k = g;
    float2 stk = make_float2(-INFINITY, 0.f), sdk = stk, bonus = stk;
    for (int i0 = 0; i0 <= g; i0 += 32) {
        const int i = i0 + lane;
        const bool draft = i < g;
        // every load at once: the tokens (their logits follow), the uniforms, both rows' chunk statistics
        const int x = i0 == 0 ? in.x : (draft ? p.tokens[d0 + i] : -1);
        const float u = i0 == 0 ? in.u : (draft ? p.u_accept[d0 + i] : 1.f);
        float2 st, sd;
        merge_rows<false>(p, i <= g ? t0 + i : -1, draft ? p.rows_t + d0 + i : -1, st, sd);
        bool rej = false;
        if (draft) {
            const bool valid = x >= 0 && x < p.vocab;
            float tx = -INFINITY, dx = -INFINITY;
            if (i0 == 0) {
                tx = in.tx;
                dx = in.dx;
            } else if (valid) {
                tx = p.target[(size_t)(t0 + i) * p.vocab + x];
                dx = p.draft[(size_t)(d0 + i) * p.vocab + x];
            }
            // a = min(1, p(x)/q(x)) in the log domain (q(x) = 0 < p(x) gives 1, p(x) = 0 gives 0)
            float a;
            if (!valid || tx == -INFINITY) a = 0.f;
            else if (dx == -INFINITY) a = 1.f;
            else a = fminf(1.f, ex2(__fmaf_rn(tx, p.c2, -st.x) - __fmaf_rn(dx, p.c2, -sd.x)) * (sd.y / st.y));
            rej = !(u < a);
            if (writer) {
                if (!valid) raise_error(p.err, kErrDeviceArg);
                if (p.accept_prob) p.accept_prob[d0 + i] = a;
            }
        }
        if (g - i0 < 32) {  // this block holds the bonus row (lane g - i0)
            bonus.x = __shfl_sync(0xffffffffu, st.x, g - i0);
            bonus.y = __shfl_sync(0xffffffffu, st.y, g - i0);
        }
        const unsigned b = __ballot_sync(0xffffffffu, rej);
        if (b && k == g) {
            const int l = __ffs(b) - 1;
            k = i0 + l;
            stk = make_float2(__shfl_sync(0xffffffffu, st.x, l), __shfl_sync(0xffffffffu, st.y, l));
            sdk = make_float2(__shfl_sync(0xffffffffu, sd.x, l), __shfl_sync(0xffffffffu, sd.y, l));
            if (!writer) break;
        }
    }
    if (k == g) stk = bonus;  // every draft accepted: the bonus row
    if (writer) {
        for (int j = lane; j <= g; j += 32) {
            if (j < k) p.out_tokens[t0 + j] = p.tokens[d0 + j];
            else if (j > k) p.out_tokens[t0 + j] = -1;
        }
        if (lane == 0) p.n_accepted[s] = k;
    }
    if (lane == 0) {
        // a row whose entries are all -inf weighs every entry 0 (M = 0, 1/Z = 0 keep it free of NaN)
        const bool tz = stk.x == -INFINITY, dz = k == g || sdk.x == -INFINITY;
        d->trow = t0 + k;
        d->drow = k < g ? p.rows_t + d0 + k : -1;
        d->Mt = tz ? 0.f : stk.x;
        d->izt = tz ? 0.f : __fdiv_rn(1.f, stk.y);
        d->Md = dz ? 0.f : sdk.x;
        d->izd = dz ? 0.f : __fdiv_rn(1.f, sdk.y);
        d->out = t0 + k;
    }
}

// ---- 2. greedy decisions (T = 0): one warp per sequence.  (At T > 0 the draw kernel decides.)
__global__ void __launch_bounds__(kBThreads) batch_decide_kernel(const BatchParams p) {
    griddep_launch_dependents();
    const int s = blockIdx.x * (kBThreads / 32) + (threadIdx.x >> 5);
    DecideIn in = {};
    if (p.inputs_early && s < p.num_seqs) in = decide_inputs<true>(p, s, threadIdx.x & 31);
    griddep_wait();
    if (s >= p.num_seqs) return;
    if (!p.inputs_early) in = decide_inputs<true>(p, s, threadIdx.x & 31);
    decide_greedy(p, s, threadIdx.x & 31, in);
}

// Weights of four entries: (r = max(0, p - q), p) with p = 2^(l*c2 - Mt) / Zt (r = 0 without a draft row).
__device__ __forceinline__ void weights4(float4 lt, float4 ld, const DrawPair& d, float c2, float4& r, float4& pw) {
    const auto pt = [&](float l) { return __fmul_rn(ex2(__fmaf_rn(l, c2, -d.Mt)), d.izt); };
    pw = make_float4(pt(lt.x), pt(lt.y), pt(lt.z), pt(lt.w));
    r = make_float4(0.f, 0.f, 0.f, 0.f);
    if (d.drow >= 0) {
        const auto qt = [&](float l) { return __fmul_rn(ex2(__fmaf_rn(l, c2, -d.Md)), d.izd); };
        const float4 q = make_float4(qt(ld.x), qt(ld.y), qt(ld.z), qt(ld.w));
        r = make_float4(fmaxf(0.f, __fsub_rn(pw.x, q.x)), fmaxf(0.f, __fsub_rn(pw.y, q.y)),
                        fmaxf(0.f, __fsub_rn(pw.z, q.z)), fmaxf(0.f, __fsub_rn(pw.w, q.w)));
    }
}
__device__ __forceinline__ float sum4f(float4 v) { return (v.x + v.y) + (v.z + v.w); }

// Masses of the 128-entry segments (j, warp) of one chunk of the draw pair, 2^-52 fixed point, into
// segR / segP; returns the calling thread's one: segment (lane, warp)'s r mass for lanes below 16,
// segment (lane - 16, warp)'s p mass above.  With SPLIT > 1 the CTA takes part `sub` of the chunk only
// (groups j in [sub * 16 / SPLIT, (sub + 1) * 16 / SPLIT): 16384 / SPLIT consecutive entries); the other
// segments come out 0.  The part's 16-byte groups are loaded in PH phases: one keeps every load in
// flight, two fit 128 registers, i.e. two CTAs per SM (for grids larger than the SM count).
template <bool VEC, int PH, int SPLIT>
__device__ __forceinline__ unsigned long long chunk_masses(const BatchParams& p, const DrawPair& d, int chunk, int sub,
                                                           int tid, unsigned long long (*segR)[kBSegs],
                                                           unsigned long long (*segP)[kBSegs]) {
    const int lane = tid & 31, warp = tid >> 5;
    const int v0 = chunk * kBChunk, n = min(kBChunk, p.vocab - v0);
    const float* tp = row_ptr(p, d.trow) + v0;
    const float* dp = d.drow >= 0 ? row_ptr(p, d.drow) + v0 : tp;
    constexpr int JS = kBVec / SPLIT, JP = JS / PH;
    float vr[JS], vp[JS];  // the lane's r and p sums of its part's segments
#pragma unroll
    for (int h = 0; h < PH; ++h) {
        float4 lt[JP], ld[JP];
#pragma unroll
        for (int jj = 0; jj < JP; ++jj) {
            const int e = 4 * (tid + (sub * JS + h * JP + jj) * kBThreads);
            lt[jj] = load4<VEC>(tp, e, n);
            if (d.drow >= 0) ld[jj] = load4<VEC>(dp, e, n);
        }
#pragma unroll
        for (int jj = 0; jj < JP; ++jj) {
            float4 r, pw;
            weights4(lt[jj], d.drow >= 0 ? ld[jj] : lt[jj], d, p.c2, r, pw);
            vr[h * JP + jj] = sum4f(r);
            vp[h * JP + jj] = sum4f(pw);
        }
    }
    float v[32];  // segment j's r sum at v[j], its p sum at v[16 + j] (0 outside the part)
#pragma unroll
    for (int j = 0; j < kBVec; ++j) {
        v[j] = 0.f;
        v[kBVec + j] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < SPLIT; ++q)
        if (q == sub)
#pragma unroll
            for (int jj = 0; jj < JS; ++jj) {
                v[q * JS + jj] = vr[jj];
                v[kBVec + q * JS + jj] = vp[jj];
            }
    const unsigned long long f = to_fix(reduce_scatter32(v, lane));  // lane j: segment j's r; 16 + j: its p
    if (lane < kBSegs) segR[warp][lane] = f;
    else segP[warp][lane - kBSegs] = f;
    return f;
}

// ---- 3. the draw (T > 0): the sequence's decisions, chunk-part masses, then the last part of the
// sequence finds the entry.  One CTA per (sequence, chunk, part): SPLIT parts of 16384 / SPLIT entries
// per chunk when the sequences' chunks alone would leave SMs idle.
template <bool VEC, int PH, int SPLIT>
__global__ void __launch_bounds__(kBThreads, SPLIT > 1 ? 2 : PH) batch_draw_kernel(const BatchParams p) {
    __shared__ unsigned long long segR[kBThreads / 32][kBSegs], segP[kBThreads / 32][kBSegs];
    __shared__ int last_sh, cstar_sh, jstar_sh, wstar_sh, use_r_sh;
    __shared__ unsigned long long off_sh, base_sh;
    __shared__ DrawPair d_sh;
    griddep_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int units = p.chunks * SPLIT;  // parts of the sequence's draw, in entry order
    const int s = blockIdx.x / units, unit = blockIdx.x - s * units;
    const int chunk = unit / SPLIT, sub = unit - chunk * SPLIT;
    DecideIn in = {};
    if (p.inputs_early && warp == 0) in = decide_inputs<false>(p, s, lane);
    griddep_wait();
    if (warp == 0) {
        if (!p.inputs_early) in = decide_inputs<false>(p, s, lane);
        decide_draw(p, s, lane, unit == 0, &d_sh, in);
    }
    __syncthreads();
    const DrawPair d = d_sh;
    constexpr int kSeg = kBThreads / 32 * kBSegs;  // 128 segments per chunk
    constexpr int kJS = kBVec / SPLIT;             // segment rows j of one part
    static_assert(kBSegs == 16 && 2 * kSeg == kBThreads, "one segment mass per thread");
    const unsigned long long f = chunk_masses<VEC, PH, SPLIT>(p, d, chunk, sub, tid, segR, segP);
    if (p.chunks > 1 || SPLIT > 1) {  // this part's segment masses, for the last CTA should the crossing fall here
        unsigned long long* segm = p.segm + ((size_t)s * p.chunks + chunk) * 2 * kSeg;
        if ((lane & (kBSegs - 1)) / kJS == sub)
            segm[(lane < kBSegs ? 0 : kSeg) + warp * kBSegs + (lane & (kBSegs - 1))] = f;  // segR / segP layout
    }
    __syncthreads();
    if (warp == 0) {
        unsigned long long R = 0, P = 0;
#pragma unroll
        for (int e = 0; e < kSeg / 32; ++e) {
            R += (&segR[0][0])[lane + 32 * e];
            P += (&segP[0][0])[lane + 32 * e];
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) {
            R += __shfl_xor_sync(0xffffffffu, R, o);
            P += __shfl_xor_sync(0xffffffffu, P, o);
        }
        if (lane == 0) {
            p.ctot[(size_t)s * units + unit] = make_ulonglong2(R, P);
            // release (cumulative through the barrier): this part's total and every thread's segment
            // mass before the ticket; acquire: the last CTA sees every part's
            last_sh = ticket_acq_rel(p.tickets + s) == units - 1;
        }
    }
    __syncthreads();
    if (!last_sh) return;
    // ---- every part is in: the distribution, the threshold and the crossing part (exact sums)
    if (warp == 0) {
        unsigned long long R = 0, P = 0;
        for (int c = lane; c < units; c += 32) {
            const ulonglong2 x = __ldcg(&p.ctot[(size_t)s * units + c]);
            R += x.x;
            P += x.y;
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) {
            R += __shfl_xor_sync(0xffffffffu, R, o);
            P += __shfl_xor_sync(0xffffffffu, P, o);
        }
        const bool use_r = d.drow >= 0 && R > 0;  // a vanishing residual (p == q) draws from p
        const unsigned long long total = use_r ? R : P;
        float u = p.u_sample[s];
        if (!(u >= 0.f)) u = 0.f;
        u = fminf(u, 0.99999994f);  // u in [0, 1): the crossing always exists
        const unsigned long long thr = __umul64hi(__float2ull_rn(u * 18446744073709551616.f), total);
        int cstar = -1;
        unsigned long long below = 0;
        for (int c0 = 0; c0 < units && cstar < 0; c0 += 32) {  // parts in entry order, 32 at a time
            const int c = c0 + lane;
            unsigned long long x = 0;
            if (c < units) {
                const ulonglong2 t = __ldcg(&p.ctot[(size_t)s * units + c]);
                x = use_r ? t.x : t.y;
            }
            const unsigned long long incl = warp_incl_scan(x, lane) + below;
            const unsigned long long excl = incl - x;
            const unsigned hit = __ballot_sync(0xffffffffu, x > 0 && excl <= thr && thr < incl);
            if (hit) {
                const int l = __ffs(hit) - 1;
                cstar = c0 + l;
                below = __shfl_sync(0xffffffffu, excl, l);
            } else {
                below = __shfl_sync(0xffffffffu, incl, 31);
            }
        }
        if (lane == 0) {
            if (total == 0 || cstar < 0) {  // no positive mass (or unreachable with exact sums): report
                raise_error(p.err, kErrDeviceArg);
                p.out_tokens[d.out] = 0;
                cstar = -1;
            }
            cstar_sh = cstar;
            off_sh = thr - below;
            use_r_sh = use_r;
        }
    }
    __syncthreads();
    const int ustar = cstar_sh;                                  // the crossing part
    const int cstar = ustar < 0 ? -1 : ustar / SPLIT;            // its chunk
    if (cstar >= 0) {
        // ---- the crossing part's segment masses (stored by its CTA; this CTA's own are in shared memory,
        // the rest of its chunk's at 0), then the segment
        if (ustar != unit) {
            const unsigned long long* sm = p.segm + ((size_t)s * p.chunks + cstar) * 2 * kSeg;
            const int j = (tid & (kSeg - 1) & (kBSegs - 1));  // layout [r / p][warp][j]
            const unsigned long long x = j / kJS == ustar - cstar * SPLIT ? __ldcg(sm + tid) : 0ull;
            if (tid < kSeg) (&segR[0][0])[tid] = x;
            else (&segP[0][0])[tid - kSeg] = x;
            __syncthreads();
        }
        const bool use_r = use_r_sh != 0;
        if (warp == 0) {  // segments in entry order: key = j * 8 + warp; lane L holds keys 4L .. 4L + 3
            unsigned long long x[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = 4 * lane + e, j = key >> 3, w = key & 7;
                x[e] = use_r ? segR[w][j] : segP[w][j];
            }
            const unsigned long long lsum = (x[0] + x[1]) + (x[2] + x[3]);
            const unsigned long long off = off_sh;
            unsigned long long cum = warp_incl_scan(lsum, lane) - lsum;
            int hitkey = -1;
            unsigned long long hb = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                if (hitkey < 0 && x[e] > 0 && cum <= off && off < cum + x[e]) {
                    hitkey = 4 * lane + e;
                    hb = cum;
                }
                cum += x[e];
            }
            const unsigned hit = __ballot_sync(0xffffffffu, hitkey >= 0);
            if (hit == 0u) {
                if (lane == 0) {  // unreachable with exact sums: report, emit the chunk's first entry
                    raise_error(p.err, kErrDeviceArg);
                    p.out_tokens[d.out] = cstar * kBChunk;
                    jstar_sh = -1;
                }
            } else if (lane == __ffs(hit) - 1) {
                jstar_sh = hitkey >> 3;
                wstar_sh = hitkey & 7;
                base_sh = hb;
            }
        }
        __syncthreads();
        const int jstar = jstar_sh;
        if (jstar >= 0 && warp == wstar_sh) {
            // ---- the entry: this lane's four entries of the segment, weighed as above
            const int v0 = cstar * kBChunk, n = min(kBChunk, p.vocab - v0);
            const int e0 = 4 * (tid + jstar * kBThreads);
            const auto at = [&](const float* row, int e) { return e < n ? __ldcg(row + e) : -INFINITY; };
            const float* st = row_ptr(p, d.trow) + v0;
            const float4 lt = make_float4(at(st, e0), at(st, e0 + 1), at(st, e0 + 2), at(st, e0 + 3));
            float4 ld = lt;
            if (d.drow >= 0) {
                const float* sd = row_ptr(p, d.drow) + v0;
                ld = make_float4(at(sd, e0), at(sd, e0 + 1), at(sd, e0 + 2), at(sd, e0 + 3));
            }
            float4 r, pw;
            weights4(lt, ld, d, p.c2, r, pw);
            const float4 w4 = use_r ? r : pw;
            const float wa[4] = {w4.x, w4.y, w4.z, w4.w};
            // offset of the threshold inside the segment, back in probability units
            const float off = __ull2float_rn(off_sh - base_sh) * 2.220446049250313e-16f;
            const float lsum = (wa[0] + wa[1]) + (wa[2] + wa[3]);
            float run = warp_incl_scan_f(lsum, lane) - lsum;
            int hit = -1, lastpos = -1;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                run += wa[e];
                if (hit < 0 && wa[e] > 0.f && run > off) hit = v0 + e0 + e;
                if (wa[e] > 0.f) lastpos = v0 + e0 + e;
            }
            const unsigned any = __ballot_sync(0xffffffffu, hit >= 0);
            const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
            // fp32 rounding inside the segment can leave the crossing just past its end: then the
            // segment's last entry with positive weight
            const int tok = any ? __shfl_sync(0xffffffffu, hit, __ffs(any) - 1)
                                : (pos ? __shfl_sync(0xffffffffu, lastpos, 31 - __clz(pos)) : v0 + e0);
            if (lane == 0) p.out_tokens[d.out] = tok;
        }
    }
    if (tid == 0) p.tickets[s] = 0;  // ready for the next call
}

}  // namespace

size_t accept_draw_scratch_bytes(int num_seqs, int vocab) {
    const size_t chunks = ((size_t)vocab + kBChunk - 1) / kBChunk;
    const size_t segm = (size_t)num_seqs * chunks * 2 * 128 * sizeof(unsigned long long);
    return align_up((size_t)num_seqs * chunks * kMaxDrawSplit * sizeof(ulonglong2), 256) + align_up(segm, 256);
}

size_t accept_batch_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    const size_t chunks = ((size_t)vocab + kBChunk - 1) / kBChunk;
    const size_t rows = 2 * (size_t)total_draft + num_seqs;
    return align_up(rows * chunks * sizeof(float2), 256) + accept_draw_scratch_bytes(num_seqs, vocab);
}

namespace {
// pdl: the prologue may overlap the previous kernel's tail (programmatic stream serialization).  The
// statistics kernel too (at T > 0): its CTAs wait for the previous kernel at their start.  Behind a
// kernel of several waves that releases its dependents early, its thousands of CTAs would take the SMs
// those waves need; the attention kernels release theirs early only when they run in one wave
// (released early from two waves, a step of the ragged batch ran 720-820 us instead of 195).
template <typename Kernel>
int launch_pdl(Kernel kernel, unsigned blocks, const BatchParams& p, cudaStream_t stream, bool pdl = true) {
    if (blocks == 0) return BP_OK;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(kBThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, p) == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

// The decisions (and at T > 0 the draw) once p.part holds the rows' statistics.
template <bool GREEDY, bool VEC>
int run_decisions(const BatchParams& p, int sm_count, cudaStream_t stream) {
    if (GREEDY)
        return launch_pdl(batch_decide_kernel, (unsigned)((p.num_seqs + kBThreads / 32 - 1) / (kBThreads / 32)), p,
                          stream);
    // the draw (with the decisions): its chunks cut into 4 or 2 parts while every CTA stays in the first
    // wave (two CTAs per SM: the sequences' chunks alone would leave SMs idle), else whole chunks
    const long long draw = (long long)p.num_seqs * p.chunks;
    if (draw * 4 <= 2LL * sm_count) return launch_pdl(batch_draw_kernel<VEC, 1, 4>, (unsigned)(draw * 4), p, stream);
    if (draw * 2 <= 2LL * sm_count) return launch_pdl(batch_draw_kernel<VEC, 1, 2>, (unsigned)(draw * 2), p, stream);
    return draw > sm_count ? launch_pdl(batch_draw_kernel<VEC, 2, 1>, (unsigned)draw, p, stream)
                           : launch_pdl(batch_draw_kernel<VEC, 1, 1>, (unsigned)draw, p, stream);
}

template <bool GREEDY, bool VEC>
int run_batch(const BatchParams& p, int sm_count, cudaStream_t stream) {
    const int rows = p.rows_t + (GREEDY ? 0 : p.total_draft);
    // chained at T > 0 (long-context step 200.3 against 202.0 us in plain order, graphs of 32 steps); at
    // T = 0, where the statistics CTAs are small enough to sit eight to an SM, plain order (184.5 against
    // 187.1 us chained)
    const int rc = launch_pdl(batch_stats_kernel<GREEDY, VEC>, (unsigned)(rows * p.chunks), p, stream, !GREEDY);
    return rc != BP_OK ? rc : run_decisions<GREEDY, VEC>(p, sm_count, stream);
}

BatchParams batch_params(const AcceptArgs& a, int* tickets, void* draw_scratch) {
    BatchParams p;
    p.target = a.target;
    p.draft = a.draft;
    p.tokens = a.tokens;
    p.cu_draft = a.cu_draft;
    p.num_seqs = a.num_seqs;
    p.total_draft = a.total_draft;
    p.rows_t = a.total_draft + a.num_seqs;
    p.vocab = a.vocab;
    p.chunks = (a.vocab + kBChunk - 1) / kBChunk;
    p.nparts = p.chunks;
    p.c2 = a.temperature == 0.f ? 0.f : 1.4426950408889634f / a.temperature;
    p.u_accept = a.u_accept;
    p.u_sample = a.u_sample;
    p.n_accepted = a.n_accepted;
    p.out_tokens = a.out_tokens;
    p.accept_prob = a.accept_prob;
    p.part = nullptr;
    uint8_t* w = static_cast<uint8_t*>(draw_scratch);
    p.ctot = reinterpret_cast<ulonglong2*>(w);
    w += align_up((size_t)a.num_seqs * p.chunks * kMaxDrawSplit * sizeof(ulonglong2), 256);
    p.segm = reinterpret_cast<unsigned long long*>(w);
    p.tickets = tickets;
    p.inputs_early = 0;
    p.err = a.err_word;
    return p;
}
bool batch_vec(const AcceptArgs& a, bool greedy) {
    return (a.vocab % 4 == 0) && (reinterpret_cast<uintptr_t>(a.target) % 16 == 0) &&
           (greedy || reinterpret_cast<uintptr_t>(a.draft) % 16 == 0);
}
}  // namespace

int launch_accept_batch(const AcceptArgs& a, int sm_count, int* tickets, void* scratch, cudaStream_t stream) {
    const size_t chunks = ((size_t)a.vocab + kBChunk - 1) / kBChunk, rows = 2 * (size_t)a.total_draft + a.num_seqs;
    uint8_t* w = static_cast<uint8_t*>(scratch);
    BatchParams p = batch_params(a, tickets, w + align_up(rows * chunks * sizeof(float2), 256));
    p.part = reinterpret_cast<float2*>(w);
    p.inputs_early = 1;  // the statistics kernel releases the decisions after its own wait
    const bool greedy = a.temperature == 0.f, vec = batch_vec(a, greedy);
    if (greedy) return vec ? run_batch<true, true>(p, sm_count, stream) : run_batch<true, false>(p, sm_count, stream);
    return vec ? run_batch<false, true>(p, sm_count, stream) : run_batch<false, false>(p, sm_count, stream);
}

int launch_accept_rows(const AcceptArgs& a, const float2* row_stats, int sm_count, int* tickets, void* draw_scratch,
                       cudaStream_t stream) {
    BatchParams p = batch_params(a, tickets, draw_scratch);
    p.part = const_cast<float2*>(row_stats);
    p.nparts = 1;
    const bool greedy = a.temperature == 0.f, vec = batch_vec(a, greedy);
    if (greedy) return run_decisions<true, true>(p, sm_count, stream);  // reads no logits
    return vec ? run_decisions<false, true>(p, sm_count, stream) : run_decisions<false, false>(p, sm_count, stream);
}

}  // namespace bp
