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
//   2. decide: one warp per sequence merges its rows' chunk statistics in a fixed order, forms the
//      ratios a_i, the first rejection k and the outputs (at T = 0 the emitted argmax too).  (Taking
//      the decisions in the statistics kernel, in the CTA that completes a sequence, costs every CTA a
//      gpu-scope ticket behind its store: measured slower for large batches);
//   3. draw (T > 0): one CTA per chunk of each sequence's draw row pair (the rejected row, or the bonus
//      row) forms the chunk's segment masses of max(0, p_k - q_k) and of p_k in exact 2^-52 fixed
//      point; the last CTA of the sequence (ticket) finds the chunk and the 128-entry segment where the
//      inverse CDF crosses u_s * total from the stored masses, then the entry from that segment's 128
//      logits, and writes the emitted token.
// Only the one draw row pair per sequence is read twice.  The kernels chain with programmatic dependent
// launch.
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

struct BatchParams {
    const float* target;  // [rows_t][vocab]
    const float* draft;   // [total_draft][vocab] (T > 0)
    const int32_t* tokens;
    const int32_t* cu_draft;
    int num_seqs, total_draft, rows_t, vocab, chunks;
    float c2;  // log2(e) / T; 0 at T = 0
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    float2* part;      // [rows][chunks] chunk statistics (T = 0: value, index bits)
    float2* rowstat;   // [rows] row statistics
    float4* drawrec;   // [num_seqs][2] the draw's rows, weight constants and output slot (T > 0)
    ulonglong2* ctot;  // [num_seqs][chunks] draw masses of r and p (fixed point)
    unsigned long long* segm;  // [num_seqs][chunks][2][128] their segment masses (chunks > 1)
    int* tickets;      // [num_seqs], zero between calls
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

// The draw of a sequence: its row pair, the constants of its weights and the output slot, written by
// the decisions as two 16-byte words and read back by every draw CTA in one round trip.
struct DrawPair {
    int trow, drow;  // drow < 0: a bonus draw from p alone
    float Mt, izt, Md, izd;
    int out;         // the emitted token's slot in out_tokens
};
__device__ __forceinline__ void store_draw(float4* rec, int trow, int drow, float2 st, float2 sd, int out) {
    // a row whose entries are all -inf weighs every entry 0 (M = 0, 1/Z = 0 keep it free of NaN)
    const bool tz = st.x == -INFINITY, dz = drow < 0 || sd.x == -INFINITY;
    rec[0] = make_float4(__int_as_float(trow), __int_as_float(drow), tz ? 0.f : st.x, tz ? 0.f : __fdiv_rn(1.f, st.y));
    rec[1] = make_float4(dz ? 0.f : sd.x, dz ? 0.f : __fdiv_rn(1.f, sd.y), __int_as_float(out), 0.f);
}
__device__ __forceinline__ DrawPair load_draw(const float4* rec) {
    const float4 a = __ldcg(rec), b = __ldcg(rec + 1);
    DrawPair d;
    d.trow = __float_as_int(a.x);
    d.drow = __float_as_int(a.y);
    d.Mt = a.z;
    d.izt = a.w;
    d.Md = b.x;
    d.izd = b.y;
    d.out = __float_as_int(b.z);
    return d;
}

// Decisions of sequence s, by one warp: its rows' statistics from their chunks', the ratios a_i, the
// first rejection k and the outputs (at T = 0 the emitted argmax too).
template <bool GREEDY>
__device__ __forceinline__ void decide_seq(const BatchParams& p, int s, int lane) {
    const int d0 = p.cu_draft[s], g = p.cu_draft[s + 1] - d0, t0 = d0 + s;
    const int nrows = GREEDY ? g + 1 : 2 * g + 1;  // the target rows, then (T > 0) the drafter's
    // the drafted tokens, their two logits and uniforms do not depend on the statistics: the first 32
    // positions' loads are issued before the merges
    struct Pick {
        int x;
        bool valid;
        float tx, dx, u;
    };
    const auto pick = [&](int i) {
        Pick q{-1, false, -INFINITY, -INFINITY, 1.f};
        if (i < g) {
            q.x = p.tokens[d0 + i];
            q.valid = q.x >= 0 && q.x < p.vocab;
            if (!GREEDY && q.valid) {
                q.tx = p.target[(size_t)(t0 + i) * p.vocab + q.x];
                q.dx = p.draft[(size_t)(d0 + i) * p.vocab + q.x];
            }
            if (!GREEDY) q.u = p.u_accept[d0 + i];
        }
        return q;
    };
    const Pick first = pick(lane);
    // each lane merges whole rows (two at a time), chunks in order, eight chunks' loads in flight
    constexpr int RH = 2, CQ = 8;
    const float2 ident = make_float2(-INFINITY, GREEDY ? __int_as_float(INT_MAX) : 0.f);
    for (int rr0 = lane; rr0 < nrows; rr0 += 32 * RH) {
        int r[RH];
        float2 acc[RH];
#pragma unroll
        for (int h = 0; h < RH; ++h) {
            const int rr = rr0 + 32 * h;
            r[h] = rr >= nrows ? -1 : rr <= g ? t0 + rr : p.rows_t + d0 + (rr - g - 1);
            acc[h] = ident;
        }
        for (int c0 = 0; c0 < p.chunks; c0 += CQ) {
            float2 x[RH][CQ];
#pragma unroll
            for (int h = 0; h < RH; ++h)
#pragma unroll
                for (int q = 0; q < CQ; ++q)
                    x[h][q] = r[h] >= 0 && c0 + q < p.chunks ? __ldcg(&p.part[(size_t)r[h] * p.chunks + c0 + q])
                                                             : ident;
#pragma unroll
            for (int h = 0; h < RH; ++h)
#pragma unroll
                for (int q = 0; q < CQ; ++q) {
                    if (GREEDY) {
                        int ai = __float_as_int(acc[h].y);
                        amax_merge(acc[h].x, ai, x[h][q].x, __float_as_int(x[h][q].y));
                        acc[h].y = __int_as_float(ai);
                    } else {
                        lse_merge(acc[h].x, acc[h].y, x[h][q].x, x[h][q].y);
                    }
                }
        }
#pragma unroll
        for (int h = 0; h < RH; ++h) {
            if (r[h] < 0) continue;
            float2 a = acc[h];
            if (GREEDY && __float_as_int(a.y) >= p.vocab) a.y = __int_as_float(0);  // every entry -inf: index 0
            p.rowstat[r[h]] = a;
        }
    }
    __syncwarp();  // the warp's row statistics are written (and visible to its lanes)
    int k = g;
    for (int i0 = 0; i0 < g; i0 += 32) {
        const int i = i0 + lane;
        const Pick q = i0 == 0 ? first : pick(i);
        bool rej = false;
        if (i < g) {
            if (!q.valid) raise_error(p.err, kErrDeviceArg);
            const float2 st = p.rowstat[t0 + i];
            float a;
            if (GREEDY) {
                a = q.valid && q.x == __float_as_int(st.y) ? 1.f : 0.f;
                rej = a == 0.f;
            } else {
                const float2 sd = p.rowstat[p.rows_t + d0 + i];
                // a = min(1, p(x)/q(x)) in the log domain (q(x) = 0 < p(x) gives 1, p(x) = 0 gives 0)
                if (!q.valid || q.tx == -INFINITY) a = 0.f;
                else if (q.dx == -INFINITY) a = 1.f;
                else a = fminf(1.f, ex2(__fmaf_rn(q.tx, p.c2, -st.x) - __fmaf_rn(q.dx, p.c2, -sd.x)) * (sd.y / st.y));
                rej = !(q.u < a);
            }
            if (p.accept_prob) p.accept_prob[d0 + i] = a;
        }
        const unsigned b = __ballot_sync(0xffffffffu, rej);
        if (b && k == g) k = i0 + __ffs(b) - 1;
    }
    for (int j = lane; j <= g; j += 32) {
        if (j < k) p.out_tokens[t0 + j] = p.tokens[d0 + j];
        else if (j > k) p.out_tokens[t0 + j] = -1;
        else if (GREEDY) p.out_tokens[t0 + j] = __float_as_int(p.rowstat[t0 + k].y);
    }
    if (lane == 0) {
        p.n_accepted[s] = k;
        if (!GREEDY) {
            const int drow = k < g ? p.rows_t + d0 + k : -1;
            store_draw(p.drawrec + 2 * s, t0 + k, drow, p.rowstat[t0 + k],
                       drow >= 0 ? p.rowstat[drow] : make_float2(-INFINITY, 0.f), t0 + k);
        }
    }
}

// ---- 1. chunk statistics of every row
template <bool GREEDY, bool VEC>
__global__ void __launch_bounds__(kBThreads) batch_stats_kernel(const BatchParams p) {
    __shared__ float2 red[kBThreads / 32];
    griddep_launch_dependents();
    griddep_wait();
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

// ---- 2. decisions: one warp per sequence
template <bool GREEDY>
__global__ void __launch_bounds__(kBThreads) batch_decide_kernel(const BatchParams p) {
    griddep_launch_dependents();
    griddep_wait();
    const int s = blockIdx.x * (kBThreads / 32) + (threadIdx.x >> 5);
    if (s < p.num_seqs) decide_seq<GREEDY>(p, s, threadIdx.x & 31);
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
// segment (lane - 16, warp)'s p mass above.  The chunk's 16-byte groups are loaded in PH phases: one
// keeps every load in flight (for grids of at most one CTA per SM), two fit 128 registers, i.e. two
// CTAs per SM (for larger grids).
template <bool VEC, int PH>
__device__ __forceinline__ unsigned long long chunk_masses(const BatchParams& p, const DrawPair& d, int chunk, int tid,
                                                           unsigned long long (*segR)[kBSegs],
                                                           unsigned long long (*segP)[kBSegs]) {
    const int lane = tid & 31, warp = tid >> 5;
    const int v0 = chunk * kBChunk, n = min(kBChunk, p.vocab - v0);
    const float* tp = row_ptr(p, d.trow) + v0;
    const float* dp = d.drow >= 0 ? row_ptr(p, d.drow) + v0 : tp;
    constexpr int JP = kBVec / PH;
    float v[32];  // the lane's r sums of segments j = 0..15, then its p sums
#pragma unroll
    for (int h = 0; h < PH; ++h) {
        float4 lt[JP], ld[JP];
#pragma unroll
        for (int jj = 0; jj < JP; ++jj) {
            const int e = 4 * (tid + (h * JP + jj) * kBThreads);
            lt[jj] = load4<VEC>(tp, e, n);
            if (d.drow >= 0) ld[jj] = load4<VEC>(dp, e, n);
        }
#pragma unroll
        for (int jj = 0; jj < JP; ++jj) {
            const int j = h * JP + jj;
            float4 r, pw;
            weights4(lt[jj], d.drow >= 0 ? ld[jj] : lt[jj], d, p.c2, r, pw);
            v[j] = sum4f(r);
            v[kBVec + j] = sum4f(pw);
        }
    }
    const unsigned long long f = to_fix(reduce_scatter32(v, lane));  // lane j: segment j's r; 16 + j: its p
    if (lane < kBSegs) segR[warp][lane] = f;
    else segP[warp][lane - kBSegs] = f;
    return f;
}

// ---- 3. the draw (T > 0): chunk masses, then the last chunk of the sequence finds the entry
template <bool VEC, int PH>
__global__ void __launch_bounds__(kBThreads, PH) batch_draw_kernel(const BatchParams p) {
    __shared__ unsigned long long segR[kBThreads / 32][kBSegs], segP[kBThreads / 32][kBSegs];
    __shared__ int last_sh, cstar_sh, jstar_sh, wstar_sh, use_r_sh;
    __shared__ unsigned long long off_sh, base_sh;
    griddep_launch_dependents();
    griddep_wait();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int s = blockIdx.x / p.chunks, chunk = blockIdx.x - s * p.chunks;
    const DrawPair d = load_draw(p.drawrec + 2 * s);
    constexpr int kSeg = kBThreads / 32 * kBSegs;  // 128 segments per chunk
    static_assert(kBSegs == 16 && 2 * kSeg == kBThreads, "one segment mass per thread");
    const unsigned long long f = chunk_masses<VEC, PH>(p, d, chunk, tid, segR, segP);
    if (p.chunks > 1) {  // the segment masses, for the last CTA should the crossing fall in this chunk
        unsigned long long* segm = p.segm + ((size_t)s * p.chunks + chunk) * 2 * kSeg;
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
            p.ctot[(size_t)s * p.chunks + chunk] = make_ulonglong2(R, P);
            // release (cumulative through the barrier): this chunk's total and every thread's segment
            // mass before the ticket; acquire: the last CTA sees every chunk's
            last_sh = ticket_acq_rel(p.tickets + s) == p.chunks - 1;
        }
    }
    __syncthreads();
    if (!last_sh) return;
    // ---- every chunk is in: the distribution, the threshold and the crossing chunk (exact sums)
    if (warp == 0) {
        unsigned long long R = 0, P = 0;
        for (int c = lane; c < p.chunks; c += 32) {
            const ulonglong2 x = __ldcg(&p.ctot[(size_t)s * p.chunks + c]);
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
        for (int c0 = 0; c0 < p.chunks && cstar < 0; c0 += 32) {  // chunks in order, 32 at a time
            const int c = c0 + lane;
            unsigned long long x = 0;
            if (c < p.chunks) {
                const ulonglong2 t = __ldcg(&p.ctot[(size_t)s * p.chunks + c]);
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
    const int cstar = cstar_sh;
    if (cstar >= 0) {
        // ---- the crossing chunk's segment masses (stored by its CTA), then the segment
        if (cstar != chunk) {
            const unsigned long long* sm = p.segm + ((size_t)s * p.chunks + cstar) * 2 * kSeg;
            const unsigned long long x = __ldcg(sm + tid);
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

size_t accept_batch_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    const size_t chunks = ((size_t)vocab + kBChunk - 1) / kBChunk;
    const size_t rows = 2 * (size_t)total_draft + num_seqs;
    const size_t segm = chunks > 1 ? (size_t)num_seqs * chunks * 2 * 128 * sizeof(unsigned long long) : 0;
    return align_up(rows * chunks * sizeof(float2), 256) + align_up(rows * sizeof(float2), 256) +
           align_up((size_t)num_seqs * 2 * sizeof(float4), 256) +
           align_up((size_t)num_seqs * chunks * sizeof(ulonglong2), 256) + align_up(segm, 256);
}

namespace {
template <typename Kernel>
int launch_pdl(Kernel kernel, unsigned blocks, const BatchParams& p, cudaStream_t stream) {
    if (blocks == 0) return BP_OK;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(kBThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // the prologue may overlap the
    attr[0].val.programmaticStreamSerializationAllowed = 1;            // previous kernel's tail
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, p) == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

template <bool GREEDY, bool VEC>
int run_batch(const BatchParams& p, int sm_count, cudaStream_t stream) {
    const int rows = p.rows_t + (GREEDY ? 0 : p.total_draft);
    int rc = launch_pdl(batch_stats_kernel<GREEDY, VEC>, (unsigned)(rows * p.chunks), p, stream);
    if (rc != BP_OK) return rc;
    rc = launch_pdl(batch_decide_kernel<GREEDY>, (unsigned)((p.num_seqs + kBThreads / 32 - 1) / (kBThreads / 32)), p,
                    stream);
    if (rc != BP_OK || GREEDY) return rc;
    const unsigned draw_ctas = (unsigned)(p.num_seqs * p.chunks);
    return draw_ctas > (unsigned)sm_count ? launch_pdl(batch_draw_kernel<VEC, 2>, draw_ctas, p, stream)
                                          : launch_pdl(batch_draw_kernel<VEC, 1>, draw_ctas, p, stream);
}
}  // namespace

int launch_accept_batch(const AcceptArgs& a, int sm_count, int* tickets, void* scratch, cudaStream_t stream) {
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
    const bool greedy = a.temperature == 0.f;
    p.c2 = greedy ? 0.f : 1.4426950408889634f / a.temperature;
    p.u_accept = a.u_accept;
    p.u_sample = a.u_sample;
    p.n_accepted = a.n_accepted;
    p.out_tokens = a.out_tokens;
    p.accept_prob = a.accept_prob;
    const size_t chunks = (size_t)p.chunks, rows = 2 * (size_t)a.total_draft + a.num_seqs;
    uint8_t* w = static_cast<uint8_t*>(scratch);
    p.part = reinterpret_cast<float2*>(w);
    w += align_up(rows * chunks * sizeof(float2), 256);
    p.rowstat = reinterpret_cast<float2*>(w);
    w += align_up(rows * sizeof(float2), 256);
    p.drawrec = reinterpret_cast<float4*>(w);
    w += align_up((size_t)a.num_seqs * 2 * sizeof(float4), 256);
    p.ctot = reinterpret_cast<ulonglong2*>(w);
    w += align_up((size_t)a.num_seqs * chunks * sizeof(ulonglong2), 256);
    p.segm = reinterpret_cast<unsigned long long*>(w);
    p.tickets = tickets;
    p.err = a.err_word;
    const bool vec = (a.vocab % 4 == 0) && (reinterpret_cast<uintptr_t>(a.target) % 16 == 0) &&
                     (greedy || reinterpret_cast<uintptr_t>(a.draft) % 16 == 0);
    if (greedy) return vec ? run_batch<true, true>(p, sm_count, stream) : run_batch<true, false>(p, sm_count, stream);
    return vec ? run_batch<false, true>(p, sm_count, stream) : run_batch<false, false>(p, sm_count, stream);
}

}  // namespace bp
