// Lossless speculative acceptance over the full vocabulary (the verification step of
// Figure 1 of the BlockPilot paper; the rule is standard speculative sampling).
//
// One thread-block cluster of CS CTAs per target row; the CTA of cluster rank c owns the
// c-th slice of the vocabulary of that target row and of the matching draft row.
//   load    each warp owns a contiguous range of the slice and brings it into shared memory
//           with one bulk copy (cp.async.bulk) per row, so the logits are read from HBM once
//           and a warp starts on its range as soon as that range has landed;
//   pass 1  each lane finds a reference maximum m over its entries of the range, then the
//           weights 2^(l*log2e/T - m) replace the logits in place and are summed.  Warp and
//           CTA reductions, then every CTA pushes its slice statistics into every other CTA's
//           shared memory (one cluster barrier); one warp merges them into the row's
//           log-sum-exp, and the CTA holding x_i gives a_i = min(1, p(x_i)/q(x_i));
//   pass 2  one multiply per entry turns the stored weights into p and r = max(0, p - q);
//           128-entry segment sums go to exact 2^-52 fixed point, a second cluster exchange
//           of the slice totals locates the slice, then one warp finds the range, the segment
//           and the entry where the inverse CDF of this row's own distribution crosses u_s * Z
//           -- the token the sequence emits if its first rejection falls on this row (a
//           residual draw; a bonus draw from p on the last row), computed speculatively by
//           every row in parallel;
//   final   the thread that publishes the last row token of a sequence (atomic ticket, no
//           waiting) finds the first rejection k from the a_i and emits the tokens of row k.
// Temperature 0 (greedy): one pass reduces the argmax (lowest index on ties).
#include <cooperative_groups.h>

#include <mutex>

#include "common.cuh"
#include "ptx_sm103.cuh"
#include "softmax_math.cuh"

namespace cg = cooperative_groups;

namespace bp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxSmemSeqs = 512;  // sequence offsets cached in shared memory (else binary search in L2)
constexpr int kMaxCS = 16;
constexpr int kMaxSeg = 16;  // 128-entry segments per warp range (pass 2 keeps one sum per segment per lane)

struct AccParams {
    const float* target;
    const float* draft;
    const int32_t* tokens;
    const int32_t* cu_draft;
    int num_seqs, total_draft, vocab;
    float c2;  // log2(e) / T
    const float* u_accept;
    const float* u_sample;
    int32_t* n_accepted;
    int32_t* out_tokens;
    float* accept_prob;
    int* tickets;  // [num_seqs], zero between calls
    float* a_ws;   // [total_draft] ratio a_i
    int* tok_ws;   // [total_rows] token each row would emit (argmax when greedy)
    int chunk4;    // float4 slots per CTA slice
    int wr;        // float4 slots per warp range of a slice
    unsigned int* err;
};

__device__ __forceinline__ int atomic_add_acq_rel(int* addr, int v) {
    int old;
    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], %2;" : "=r"(old) : "l"(addr), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ float max4(float4 v) { return fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)); }
__device__ __forceinline__ float pick(float4 v, int e) { return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w; }
// 2^(l*c2 - m) of four logits (m finite)
__device__ __forceinline__ float4 ex2_4(float4 v, float c2, float m) {
    return make_float4(ex2(__fmaf_rn(v.x, c2, -m)), ex2(__fmaf_rn(v.y, c2, -m)), ex2(__fmaf_rn(v.z, c2, -m)),
                       ex2(__fmaf_rn(v.w, c2, -m)));
}
__device__ __forceinline__ float sum4(float4 v) { return (v.x + v.y) + (v.z + v.w); }
__device__ __forceinline__ float4 mul4(float4 v, float f) {
    return make_float4(__fmul_rn(v.x, f), __fmul_rn(v.y, f), __fmul_rn(v.z, f), __fmul_rn(v.w, f));
}
__device__ __forceinline__ float4 resid4(float4 p, float4 q) {
    return make_float4(fmaxf(0.f, __fsub_rn(p.x, q.x)), fmaxf(0.f, __fsub_rn(p.y, q.y)),
                       fmaxf(0.f, __fsub_rn(p.z, q.z)), fmaxf(0.f, __fsub_rn(p.w, q.w)));
}

// Shared memory of one CTA: the target slice sT and (sampling only) the draft slice sD, up to
// chunk4 float4 slots each.  Warp w owns the contiguous slot range [w*wr, w*wr + wr) of both
// slices and brings it in with its own bulk copies (one mbarrier per range and row), so every
// warp starts on its range as soon as that range has landed.  Lane l works on the slots
// w*wr + 32j + l: slot row j of a range is a segment of 128 consecutive vocabulary entries,
// the leaf of the inverse-CDF search (a range has at most kMaxSeg segments).
__host__ __device__ inline size_t smem_bytes(int chunk4, bool greedy) { return (size_t)chunk4 * (greedy ? 16 : 32); }
__host__ __device__ inline int warp_range(int chunk4) { return (chunk4 + kWarps - 1) / kWarps; }

// A warp's range of one row slice -> shared memory: one bulk copy (16-byte aligned rows, lane 0
// issues it) or plain loads by the warp (padding past the vocabulary reads -inf).
template <bool VEC>
__device__ __forceinline__ void fetch_range(float4* dst, const float* row, int first4, int nw, int V, uint64_t* bar,
                                            int lane) {
    if (nw <= 0) return;
    if (VEC) {
        if (lane == 0) {
            mbar_arrive_expect_tx(bar, (uint32_t)nw * 16u);
            bulk_load(dst, row + (size_t)first4 * 4, (uint32_t)nw * 16u, bar);
        }
    } else {
        float* d = reinterpret_cast<float*>(dst);
        for (int idx = lane; idx < nw * 4; idx += 32) {
            const int x = first4 * 4 + idx;
            d[idx] = x < V ? __ldg(row + x) : -INFINITY;
        }
        __syncwarp();
    }
}
// Waits for the warp's copy; if the wait expires, the error is recorded and the copy is still waited
// out (drain budget): no copy may land in shared memory after the CTA has moved on or left.
template <bool VEC>
__device__ __forceinline__ void wait_range(uint64_t* bar, int nw, unsigned int* err) {
    if (VEC && nw > 0 && !mbar_wait(bar, 0, kWaitBudget)) {
        raise_error(err, kErrTimeout);
        mbar_wait(bar, 0, kDrainBudget);
    }
}

// Scaled maximum l*c2 of a lane's entries of a range (-inf if none is finite), then the weights
// 2^(l*c2 - m) replace the logits in place (zeros when no entry is finite, so that pass 2 never
// multiplies a -inf logit); returns (m, sum of the weights).
__device__ __forceinline__ float2 weigh_range(float4* s, int w0, int nw, int Kw, int lane, float c2) {
    float m = -INFINITY;
    for (int j = 0; j < Kw; ++j) {
        const int f = j * 32 + lane;
        if (f < nw) m = fmaxf(m, max4(s[w0 + f]));
    }
    float sum = 0.f;
    if (m != -INFINITY) {
        m = __fmul_rn(m, c2);
        for (int j = 0; j < Kw; ++j) {
            const int f = j * 32 + lane;
            if (f < nw) {
                const float4 e = ex2_4(s[w0 + f], c2, m);
                sum += sum4(e);
                s[w0 + f] = e;
            }
        }
    } else {
        for (int j = 0; j < Kw; ++j) {
            const int f = j * 32 + lane;
            if (f < nw) s[w0 + f] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    return make_float2(m, sum);
}

template <bool GREEDY, bool VEC>
__global__ void __launch_bounds__(kThreads, 2) accept_kernel(const AccParams p) {
    cg::cluster_group cluster = cg::this_cluster();
    const int CS = (int)cluster.num_blocks();
    const int c = (int)cluster.block_rank();
    const int rt = blockIdx.x / CS;  // global target row
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int V = p.vocab;

    extern __shared__ __align__(128) uint8_t dyn_smem[];
    __shared__ uint64_t bar_t[kWarps], bar_d[kWarps];
    __shared__ int32_t cu_sh[kMaxSmemSeqs + 1];  // sequence offsets; the final step reuses it
    __shared__ float4 red4[kWarps];
    __shared__ int red_i[kWarps];
    __shared__ float4 peer_stat[kMaxCS];     // (scaled max t, sum t, scaled max d, sum d)
    __shared__ float4 peer_x[kMaxCS];        // (t[x_i], d[x_i], owns x_i, -); greedy: (max, index)
    __shared__ ulonglong2 peer_tot[kMaxCS];  // slice totals of r and p (fixed point)
    __shared__ unsigned long long segR[kWarps * kMaxSeg], segP[kWarps * kMaxSeg];
    __shared__ ulonglong2 wtot[kWarps];      // range totals of r and p (fixed point)
    __shared__ float4 own_sh;
    __shared__ float4 stat_sh;  // (scaled max t, sum t, scaled max d, sum d) of the row
    __shared__ int last_sh, k_sh;

    cluster_arrive_relaxed();  // peers must be running before any distributed shared memory write
    griddep_launch_dependents();
    float4* sT = reinterpret_cast<float4*>(dyn_smem);
    float4* sD = sT + p.chunk4;
    const int v4 = (V + 3) / 4;
    const int f0 = c * p.chunk4;
    const int n4 = max(0, min(v4, f0 + p.chunk4) - f0);
    const int w0 = warp * p.wr;  // this warp's range of the slice
    const int nw = max(0, min(n4, w0 + p.wr) - w0);
    const int Kw = (nw + 31) >> 5;
    const float* trow = p.target + (size_t)rt * V;

    if (lane == 0) {
        mbar_init(&bar_t[warp], 1);
        mbar_init(&bar_d[warp], 1);
        fence_mbar_init();
    }
    __syncwarp();
    // inputs may be produced by the previous kernel on the stream: wait for it before any global access
    griddep_wait();
    fetch_range<VEC>(sT + w0, trow, f0 + w0, nw, V, &bar_t[warp], lane);  // the target row needs no lookup
    int s, d_begin, d_end;
    if (p.num_seqs == 1) {
        s = 0;
        d_begin = 0;  // cu_draft[0] = 0
        d_end = p.total_draft;
    } else if (p.num_seqs <= kMaxSmemSeqs) {
        for (int t = tid; t <= p.num_seqs; t += kThreads) cu_sh[t] = p.cu_draft[t];
        __syncthreads();
        int lo = 0, hi = p.num_seqs;  // largest s with cu[s] + s <= rt
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (cu_sh[mid] + mid <= rt) lo = mid; else hi = mid;
        }
        s = lo;
        d_begin = cu_sh[s];
        d_end = cu_sh[s + 1];
    } else {
        int lo = 0, hi = p.num_seqs;
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(p.cu_draft + mid) + mid <= rt) lo = mid; else hi = mid;
        }
        s = lo;
        d_begin = __ldg(p.cu_draft + s);
        d_end = __ldg(p.cu_draft + s + 1);
    }
    const int gamma = d_end - d_begin;
    const int tstart = d_begin + s;
    const int i = rt - tstart;
    const bool has_draft = i < gamma;
    const bool use_draft = !GREEDY && has_draft;
    if (use_draft) fetch_range<VEC>(sD + w0, p.draft + (size_t)(d_begin + i) * V, f0 + w0, nw, V, &bar_d[warp], lane);
    int xi = has_draft ? __ldg(p.tokens + d_begin + i) : -1;
    if (has_draft && (xi < 0 || xi >= V)) {
        if (c == 0 && tid == 0) raise_error(p.err, kErrDeviceArg);
        xi = -1;
    }
    // inputs of the final step, read ahead of it (any CTA may turn out to run it)
    const int my_tok = tid < gamma ? __ldg(p.tokens + d_begin + tid) : -1;
    const float my_ua = (!GREEDY && tid < gamma) ? __ldg(p.u_accept + d_begin + tid) : 0.f;
    const float u_s = GREEDY ? 0.f : __ldg(p.u_sample + s);
    const float c2 = p.c2;
    bool writer = false;  // the thread that publishes this row's token and takes the ticket
    int tok_out = 0;

    if (GREEDY) {
        // ================= argmax of the target row (lowest index on ties)
        wait_range<VEC>(&bar_t[warp], nw, p.err);
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int j = 0; j < Kw; ++j) {
            const int f = j * 32 + lane;
            if (f < nw) {
                const float4 v = sT[w0 + f];
                const int x = (f0 + w0 + f) * 4;
                amax_merge(bv, bi, v.x, x + 0);
                amax_merge(bv, bi, v.y, x + 1);
                amax_merge(bv, bi, v.z, x + 2);
                amax_merge(bv, bi, v.w, x + 3);
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
            const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
            amax_merge(bv, bi, v2, i2);
        }
        if (lane == 0) {
            red4[warp].x = bv;
            red_i[warp] = bi;
        }
        __syncthreads();
        cluster_wait();
        if (tid < CS) {
            float v = red4[0].x;
            int ix = red_i[0];
            for (int w = 1; w < kWarps; ++w) amax_merge(v, ix, red4[w].x, red_i[w]);
            *cluster.map_shared_rank(&peer_x[c], tid) = make_float4(v, __int_as_float(ix), 0.f, 0.f);
        }
        cluster_sync_all();
        if (c != 0) return;
        if (tid == 0) {
            float v = -INFINITY;
            int ix = 0x7fffffff;
            for (int r = 0; r < CS; ++r) amax_merge(v, ix, peer_x[r].x, __float_as_int(peer_x[r].y));
            if (ix >= V) ix = 0;  // every entry -inf: lowest index
            writer = true;
            tok_out = ix;
            if (has_draft && p.accept_prob) p.accept_prob[d_begin + i] = (xi == ix) ? 1.f : 0.f;
        }
    } else {
        // ================= pass 1: per lane, a reference maximum and the sum of the weights
        const bool own_x = xi >= 0 && (xi >> 2) >= f0 && (xi >> 2) < f0 + n4;  // this CTA holds x_i
        const bool own_xw = own_x && (xi >> 2) - f0 >= w0 && (xi >> 2) - f0 < w0 + nw;  // this warp
        float own_t = 0.f, own_d = 0.f;
        wait_range<VEC>(&bar_t[warp], nw, p.err);
        if (own_xw && lane == 0) own_t = pick(sT[(xi >> 2) - f0], xi & 3);  // the raw logit, before weighing
        __syncwarp();
        const float2 wt = weigh_range(sT, w0, nw, Kw, lane, c2);
        float2 wd = make_float2(-INFINITY, 0.f);
        if (use_draft) {
            wait_range<VEC>(&bar_d[warp], nw, p.err);
            if (own_xw && lane == 0) own_d = pick(sD[(xi >> 2) - f0], xi & 3);
            __syncwarp();
            wd = weigh_range(sD, w0, nw, Kw, lane, c2);
        }
        if (own_xw && lane == 0) own_sh = make_float4(own_t, own_d, 1.f, 0.f);
        // warp statistics: the warp maximum, then every lane's sum rescaled to it
        float mt = wt.x, md = wd.x;
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
            md = fmaxf(md, __shfl_xor_sync(0xffffffffu, md, o));
        }
        float st = wt.y * ex2d(wt.x, mt), sd = wd.y * ex2d(wd.x, md);
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            st += __shfl_xor_sync(0xffffffffu, st, o);
            sd += __shfl_xor_sync(0xffffffffu, sd, o);
        }
        if (lane == 0) red4[warp] = make_float4(mt, st, md, sd);
        __syncthreads();
        cluster_wait();  // peers are running
        if (tid < CS) {
            float4 a = red4[0];
            for (int w = 1; w < kWarps; ++w) {
                lse_merge(a.x, a.y, red4[w].x, red4[w].y);
                lse_merge(a.z, a.w, red4[w].z, red4[w].w);
            }
            *cluster.map_shared_rank(&peer_stat[c], tid) = a;
            *cluster.map_shared_rank(&peer_x[c], tid) = own_x ? own_sh : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        cluster_sync_all();
        // ---- row statistics: warp 0 merges the CS slice statistics along a butterfly (the merge is
        // commutative bit for bit, so every lane and every CTA of the cluster gets the same values)
        if (warp == 0) {
            float4 a = lane < CS ? peer_stat[lane] : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float4 b = make_float4(__shfl_xor_sync(0xffffffffu, a.x, o), __shfl_xor_sync(0xffffffffu, a.y, o),
                                             __shfl_xor_sync(0xffffffffu, a.z, o), __shfl_xor_sync(0xffffffffu, a.w, o));
                lse_merge(a.x, a.y, b.x, b.y);
                lse_merge(a.z, a.w, b.z, b.w);
            }
            const unsigned holder = __ballot_sync(0xffffffffu, lane < CS && peer_x[lane].z != 0.f);
            if (lane == 0) {
                stat_sh = a;
                const float4 x = holder ? peer_x[__ffs(holder) - 1] : make_float4(-INFINITY, -INFINITY, 0.f, 0.f);
                own_sh = x;  // (t[x_i], d[x_i]) of the row, read below
            }
        }
        __syncthreads();
        const float Mt = stat_sh.x, Zt = stat_sh.y, Md = stat_sh.z, Zd = stat_sh.w;
        const float tx = own_sh.x, dx = own_sh.y;
        if (c == 0 && tid == 0 && has_draft) {
            // a = min(1, p(x)/q(x)) evaluated in the log domain
            float a;
            if (xi < 0 || tx == -INFINITY) a = 0.f;
            else if (dx == -INFINITY) a = 1.f;
            else a = fminf(1.f, ex2(__fmaf_rn(tx, c2, -Mt) - __fmaf_rn(dx, c2, -Md)) * (Zd / Zt));
            // reaches the last ticket holder through the cluster barriers below and the writer's
            // gpu-scope release at its ticket (both cumulative): no fence of its own
            p.a_ws[d_begin + i] = a;
            if (p.accept_prob) p.accept_prob[d_begin + i] = a;
        }

        // ================= pass 2: fixed-point segment sums of r and p, one multiply per entry
        const float izt = __fdiv_rn(1.f, Zt);
        const float izd = use_draft ? __fdiv_rn(1.f, Zd) : 0.f;
        const float ft = wt.x == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(wt.x, Mt)), izt);
        const float fd = (use_draft && wd.x != -INFINITY) ? __fmul_rn(ex2(__fsub_rn(wd.x, Md)), izd) : 0.f;
        float v[2 * kMaxSeg];  // r then p of the lane's entries of each segment
#pragma unroll
        for (int j = 0; j < kMaxSeg; ++j) {
            const int f = j * 32 + lane;
            float sr = 0.f, sp = 0.f;
            if (j < Kw && f < nw) {
                const float4 pv = mul4(sT[w0 + f], ft);
                sp = sum4(pv);
                if (use_draft) sr = sum4(resid4(pv, mul4(sD[w0 + f], fd)));
            }
            v[j] = sr;
            v[kMaxSeg + j] = sp;
        }
        // lane j < 16 gets the r-sum of segment j, lane 16 + j its p-sum; one conversion each
        const unsigned long long fx = to_fix(reduce_scatter32(v, lane));
        if (lane < kMaxSeg) segR[warp * kMaxSeg + lane] = fx;
        else segP[warp * kMaxSeg + lane - kMaxSeg] = fx;
        unsigned long long rtot = fx;
#pragma unroll
        for (int o = kMaxSeg / 2; o; o >>= 1) rtot += __shfl_xor_sync(0xffffffffu, rtot, o);
        if (lane == 0) wtot[warp].x = rtot;
        if (lane == kMaxSeg) wtot[warp].y = rtot;
        __syncthreads();
        if (tid < CS) {
            ulonglong2 t = wtot[0];
            for (int w = 1; w < kWarps; ++w) {
                t.x += wtot[w].x;
                t.y += wtot[w].y;
            }
            *cluster.map_shared_rank(&peer_tot[c], tid) = t;
        }
        cluster_sync_all();
        // ---- which distribution, the threshold, and the slice where the CDF crosses it
        unsigned long long R = 0, P = 0, Rb = 0, Pb = 0;
        for (int r = 0; r < CS; ++r) {
            if (r < c) {
                Rb += peer_tot[r].x;
                Pb += peer_tot[r].y;
            }
            R += peer_tot[r].x;
            P += peer_tot[r].y;
        }
        const bool use_r = use_draft && R > 0;  // a vanishing residual (p == q) draws from p
        const unsigned long long total = use_r ? R : P;
        const unsigned long long mine = use_r ? peer_tot[c].x : peer_tot[c].y;
        const unsigned long long below = use_r ? Rb : Pb;
        float u = u_s;
        if (!(u >= 0.f)) u = 0.f;
        u = fminf(u, 0.99999994f);  // u in [0, 1): the crossing always exists
        const unsigned long long thr = __umul64hi(__float2ull_rn(u * 18446744073709551616.f), total);
        if (total == 0) {
            // no positive mass at all (a row without a finite logit): report, emit 0
            if (c != 0) return;
            if (tid == 0) {
                raise_error(p.err, kErrDeviceArg);
                writer = true;
                tok_out = 0;
            }
        } else {
            if (!(below <= thr && thr < below + mine)) return;  // the crossing is in another slice
            // ---- the warp range, then the segment holding the threshold (exact integer sums:
            // exactly one of each holds it)
            unsigned long long cum = below, wbase = 0;
            int wsel = -1;
            for (int q = 0; q < kWarps; ++q) {
                const unsigned long long x = use_r ? wtot[q].x : wtot[q].y;
                if (wsel < 0 && x > 0 && cum <= thr && thr < cum + x) {
                    wsel = q;
                    wbase = cum;
                }
                cum += x;
            }
            if (wsel < 0) {  // unreachable with exact sums: report, emit the slice's first entry
                if (tid == 0) {
                    raise_error(p.err, kErrDeviceArg);
                    writer = true;
                    tok_out = f0 * 4;
                }
            } else if (warp == wsel) {
                const unsigned long long sg =
                    lane < kMaxSeg ? (use_r ? segR : segP)[warp * kMaxSeg + lane] : 0ull;
                const unsigned long long incl = warp_incl_scan(sg, lane);
                const unsigned long long sb = wbase + incl - sg;
                const unsigned hm = __ballot_sync(0xffffffffu, sg > 0 && sb <= thr && thr < sb + sg);
                if (hm == 0u) {  // unreachable with exact sums
                    if (lane == 0) {
                        raise_error(p.err, kErrDeviceArg);
                        writer = true;
                        tok_out = (f0 + w0) * 4;
                    }
                } else {
                    const int j = __ffs(hm) - 1;
                    const unsigned long long base = __shfl_sync(0xffffffffu, sb, j);
                    // ---- entry of segment j: this lane's slot, weighed exactly as in pass 2
                    const int f = j * 32 + lane;
                    float4 wv = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (f < nw) {
                        wv = mul4(sT[w0 + f], ft);
                        if (use_r) wv = resid4(wv, mul4(sD[w0 + f], fd));
                    }
                    const float wa[4] = {wv.x, wv.y, wv.z, wv.w};
                    // offset of the threshold inside the segment, back in probability units
                    const float off = __ull2float_rn(thr - base) * 2.220446049250313e-16f;
                    const float lsum = (wa[0] + wa[1]) + (wa[2] + wa[3]);
                    float run = warp_incl_scan_f(lsum, lane) - lsum;
                    const int x0 = (f0 + w0 + f) * 4;
                    int hit = -1, lastpos = -1;
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        run += wa[e];
                        if (hit < 0 && wa[e] > 0.f && run > off) hit = x0 + e;
                        if (wa[e] > 0.f) lastpos = x0 + e;
                    }
                    const unsigned any = __ballot_sync(0xffffffffu, hit >= 0);
                    const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
                    // fp32 rounding inside the segment can leave the crossing just past its end:
                    // then the segment's last entry with positive weight
                    const int first = any ? __shfl_sync(0xffffffffu, hit, __ffs(any) - 1)
                                          : (pos ? __shfl_sync(0xffffffffu, lastpos, 31 - __clz(pos)) : x0);
                    if (lane == 0) {
                        writer = true;
                        tok_out = first;
                    }
                }
            }
        }
    }

    // ---- publish the row's token and take a ticket; the last row of the sequence resolves it
    if (writer) {
        p.tok_ws[rt] = tok_out;
        // release: this row's token (and, through the cluster barriers, a_i) before the ticket;
        // acquire: the last ticket sees every other row's results
        const int old = atomic_add_acq_rel(p.tickets + s, 1);
        last_sh = (old == gamma);
        k_sh = gamma;
    }
    __syncthreads();
    if (!last_sh) return;
    if (tid == 0) p.tickets[s] = 0;  // ready for the next call
    // one round of loads: the rows' tokens and ratios, then the first rejection k
    for (int ii = tid; ii <= gamma; ii += kThreads) {
        const int tw = __ldcg(p.tok_ws + tstart + ii);
        bool rej = false;
        if (ii < gamma) {
            const int tok = ii == tid ? my_tok : __ldg(p.tokens + d_begin + ii);
            if (GREEDY) {
                rej = tok != tw;
            } else {
                const float ua = ii == tid ? my_ua : __ldg(p.u_accept + d_begin + ii);
                rej = !(ua < __ldcg(p.a_ws + d_begin + ii));
            }
        }
        if (rej) atomicMin(&k_sh, ii);
        if (ii <= kMaxSmemSeqs) cu_sh[ii] = tw;
    }
    __syncthreads();
    const int k = k_sh;
    const int token = k <= kMaxSmemSeqs ? cu_sh[k] : __ldcg(p.tok_ws + tstart + k);
    for (int ii = tid; ii <= gamma; ii += kThreads) {
        int v;
        if (ii < k) v = (ii == tid) ? my_tok : __ldg(p.tokens + d_begin + ii);
        else if (ii == k) v = token;
        else v = -1;
        p.out_tokens[tstart + ii] = v;
    }
    if (tid == 0) p.n_accepted[s] = k;
}

constexpr size_t kSmemBudget = 104 * 1024;  // dynamic shared memory per CTA: two CTAs per SM with the static part

struct Variant {
    int max_active[kMaxCS + 1];
    bool ready;
};

template <bool GREEDY, bool VEC>
Variant& variant(int dev) {
    static Variant v[64];
    Variant& x = v[dev];
    if (!x.ready) {
        auto kern = accept_kernel<GREEDY, VEC>;
        cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
        cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBudget);
        for (int cs = 1; cs <= kMaxCS; ++cs) {
            cudaLaunchConfig_t probe = {};
            cudaLaunchAttribute pa[1];
            probe.gridDim = dim3(cs, 1, 1);
            probe.blockDim = dim3(kThreads, 1, 1);
            probe.dynamicSmemBytes = kSmemBudget;
            pa[0].id = cudaLaunchAttributeClusterDimension;
            pa[0].val.clusterDim.x = cs;
            pa[0].val.clusterDim.y = 1;
            pa[0].val.clusterDim.z = 1;
            probe.attrs = pa;
            probe.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, kern, &probe) != cudaSuccess) {
                cudaGetLastError();
                n = 0;
            }
            x.max_active[cs] = n;
        }
        x.ready = true;
    }
    return x;
}

// Smallest cluster whose slices fit the shared-memory budget (0 if none).
int min_cluster(int vocab, bool greedy) {
    const int v4 = (vocab + 3) / 4;
    for (int cs = 1; cs <= kMaxCS; ++cs)
        if (smem_bytes((v4 + cs - 1) / cs, greedy) <= kSmemBudget) return cs;
    return 0;
}

template <bool GREEDY, bool VEC>
int launch_variant(const AccParams& prm0, int rows, const DeviceInfo& dev, cudaStream_t stream) {
    Variant& var = variant<GREEDY, VEC>(dev.device);
    const int v4 = (prm0.vocab + 3) / 4;
    const int cs_min = min_cluster(prm0.vocab, GREEDY);
    if (cs_min == 0) return BP_ERR_UNSUPPORTED;
    // cluster size: the widest split whose clusters are all resident in one wave (two CTAs per SM),
    // with at least one full slot per thread; otherwise the smallest split that fits
    int cs = cs_min;
    for (int c = kMaxCS; c >= cs_min; --c) {
        if (rows <= var.max_active[c] && (long long)rows * c <= 2LL * dev.sm_count &&
            (v4 + c - 1) / c >= kThreads) {
            cs = c;
            break;
        }
    }
    AccParams p = prm0;
    p.chunk4 = (v4 + cs - 1) / cs;
    p.wr = warp_range(p.chunk4);
    if (!GREEDY && p.wr > kMaxSeg * 32) return BP_ERR_UNSUPPORTED;  // excluded by the shared-memory budget
    const size_t smem = smem_bytes(p.chunk4, GREEDY);
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)(rows * cs), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    // No programmatic (early) launch here: clusters placed while the previous kernel still holds
    // SMs land in whatever is left of each GPC and a wide cluster then needs a second wave (a
    // measured 3 us loss after block attention).  The kernel still releases its own dependents early.
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, accept_kernel<GREEDY, VEC>, p) == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

}  // namespace

// Scratch of the cluster kernel (tickets first: the no-workspace path clears them before each call).
static size_t cluster_scratch_bytes(int num_seqs, int total_draft) {
    const size_t rows = (size_t)total_draft + num_seqs;
    return align_up(sizeof(int) * (size_t)num_seqs, 256) + align_up(sizeof(float) * (size_t)total_draft, 256) +
           align_up(sizeof(int) * rows, 256);
}

size_t accept_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    if (vocab < 1 || min_cluster(vocab, false) == 0) return 0;  // slices must fit in shared memory
    size_t b = cluster_scratch_bytes(num_seqs, total_draft);
    if (accept_may_batch(num_seqs, total_draft, vocab))  // the throughput kernels' regions follow
        b += accept_batch_scratch_bytes(num_seqs, total_draft, vocab);
    return b;
}

int launch_accept(const AcceptArgs& a, const DeviceInfo& dev, cudaStream_t stream, bool allow_batch) {
    if (accept_scratch_bytes(a.num_seqs, a.total_draft, a.vocab) == 0) return BP_ERR_UNSUPPORTED;
    if (a.num_seqs == 0) return BP_OK;
    const int rows = a.total_draft + a.num_seqs;
    uint8_t* w = static_cast<uint8_t*>(a.scratch);
    if (allow_batch && accept_use_batch(a.num_seqs, a.total_draft, a.vocab, a.temperature == 0.f))
        return launch_accept_batch(a, dev.sm_count, reinterpret_cast<int*>(w),
                                   w + cluster_scratch_bytes(a.num_seqs, a.total_draft), stream);
    AccParams p;
    p.tickets = reinterpret_cast<int*>(w);
    w += align_up(sizeof(int) * (size_t)a.num_seqs, 256);
    p.a_ws = reinterpret_cast<float*>(w);
    w += align_up(sizeof(float) * (size_t)a.total_draft, 256);
    p.tok_ws = reinterpret_cast<int*>(w);
    p.target = a.target;
    p.draft = a.draft;
    p.tokens = a.tokens;
    p.cu_draft = a.cu_draft;
    p.num_seqs = a.num_seqs;
    p.total_draft = a.total_draft;
    p.vocab = a.vocab;
    const bool greedy = a.temperature == 0.f;
    p.c2 = greedy ? 0.f : 1.4426950408889634f / a.temperature;
    p.u_accept = a.u_accept;
    p.u_sample = a.u_sample;
    p.n_accepted = a.n_accepted;
    p.out_tokens = a.out_tokens;
    p.accept_prob = a.accept_prob;
    p.chunk4 = 0;
    p.wr = 0;
    p.err = a.err_word;
    const bool vec = (a.vocab % 4 == 0) && (reinterpret_cast<uintptr_t>(a.target) % 16 == 0) &&
                     (greedy || reinterpret_cast<uintptr_t>(a.draft) % 16 == 0);
    if (greedy) return vec ? launch_variant<true, true>(p, rows, dev, stream) : launch_variant<true, false>(p, rows, dev, stream);
    return vec ? launch_variant<false, true>(p, rows, dev, stream) : launch_variant<false, false>(p, rows, dev, stream);
}

// ---------------------------------------------------------------------------------------
// Scratch of bp_spec_accept_noalloc.
//
// Some callers cannot allocate device memory for a workspace: for example a plugin that runs
// inside another inference engine and only receives its input and output buffers from it, or
// a serving loop that must not call cudaMalloc while requests are in flight (cudaMalloc can
// synchronize the device and stall every other stream).  For them the acceptance step can use
// this fixed array instead, which the CUDA runtime places in device memory when the library's
// module is loaded; every GPU that loads the library keeps these BP_NOALLOC_SCRATCH_BYTES
// until the process exits.
//
// All calls share the array and it keeps whatever the previous call left in it, so each call
// clears the part that must start at zero (the per-sequence tickets) on its own stream before
// the kernel runs.  Calls whose execution overlaps on the GPU (different streams without an
// ordering between them) race on this array and give undefined results.
static __device__ __align__(256) unsigned char g_noalloc_scratch[BP_NOALLOC_SCRATCH_BYTES];

namespace {
// Device address of g_noalloc_scratch for the current device.  In host code the symbol is only
// a host-side stand-in, so the address is looked up once per device (with that device current)
// and cached; the lookup happens on the first call of bp_spec_accept_noalloc on each device.
int noalloc_scratch_address(void** out) {
    static void* addr[64] = {};
    static std::mutex mu;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return BP_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(mu);
    if (addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return BP_ERR_CUDA;
        }
        addr[dev] = p;
    }
    *out = addr[dev];
    return BP_OK;
}
}  // namespace

int launch_accept_noalloc(const AcceptArgs& args, const DeviceInfo& dev, cudaStream_t stream) {
    const size_t need = accept_scratch_bytes(args.num_seqs, args.total_draft, args.vocab);
    if (need == 0) return BP_ERR_UNSUPPORTED;
    // the throughput kernels only when their regions fit too; else the cluster kernel alone
    const bool allow_batch = need <= (size_t)BP_NOALLOC_SCRATCH_BYTES;
    if (cluster_scratch_bytes(args.num_seqs, args.total_draft) > (size_t)BP_NOALLOC_SCRATCH_BYTES)
        return BP_ERR_WORKSPACE;  // problem too large for the array
    void* base = nullptr;
    int rc = noalloc_scratch_address(&base);
    if (rc != BP_OK) return rc;
    // the tickets (first region of the scratch layout) must be zero when the kernel starts
    if (cudaMemsetAsync(base, 0, align_up(sizeof(int) * (size_t)args.num_seqs, 256), stream) != cudaSuccess) {
        cudaGetLastError();
        return BP_ERR_CUDA;
    }
    AcceptArgs a = args;
    a.scratch = base;
    return launch_accept(a, dev, stream, allow_batch);
}

}  // namespace bp
