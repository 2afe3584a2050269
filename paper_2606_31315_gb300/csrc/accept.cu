// Lossless speculative acceptance over the full vocabulary (the verification step of
// Figure 1 of the BlockPilot paper; the rule is standard speculative sampling).
//
// Layout of the work.  One thread-block cluster of CS CTAs per target row; the CTA of
// cluster rank c owns the c-th slice of the vocabulary of that target row and of the
// matching draft row, and keeps both slices in registers (16-byte loads, issued
// up front, so every byte of the logits is read from HBM exactly once):
//   1. per-slice max and sum of 2^(l*log2e/T - max), block-reduced with warp shuffles;
//   2. the CS slice statistics are merged through distributed shared memory into the
//      row's log-sum-exp, which gives a_i = min(1, p(x_i)/q(x_i));
//   3. speculatively -- before the first rejection k is known -- every CTA computes the
//      sums of r = max(0, p - q) and of p over 128-entry vocabulary segments from the
//      values still in registers and stores them (a few KB per row);
//   4. an atomic ticket per sequence elects the CTA that finishes last; it finds k,
//      scans the segment sums of row k (fp64 prefix) to the segment where the inverse
//      CDF crosses u*Z, recomputes that segment's 128 weights bit-identically from the
//      logits and picks the token.  No CTA waits for another, no second launch.
// Temperature 0 (greedy): only target rows are read; each cluster reduces the argmax
// (lowest index on ties) and the last CTA of the sequence compares it with the drafts.
#include <cooperative_groups.h>

#include <mutex>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace bp {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxSmemSeqs = 2048;

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
    int* tickets;     // [num_seqs], zero between calls
    float* a_ws;      // [total_draft] ratio a_i
    int* g_ws;        // [total_rows] greedy argmax
    float4* rowinfo;  // [total_rows * CS] (slice max of t, slice max of d, p factor, q factor)
    float* seg_r;     // [total_rows * nseg] residual segment sums
    float* seg_p;     // [total_rows * nseg] target-probability segment sums
    int chunk4;       // float4 slots per CTA slice
    int nseg;         // segments per row = CS * NV4 * kWarps
    unsigned int* err;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Weight of one element in the speculative pass and in the final re-scan; the
// explicit _rn operations keep both evaluations bit-identical (no FMA contraction).
__device__ __forceinline__ float scaled(float l, float c2) { return __fmul_rn(l, c2); }
__device__ __forceinline__ float expo(float t2, float m) { return m == -INFINITY ? 0.f : ex2(__fsub_rn(t2, m)); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Block-wide reductions over 512 threads; the result is returned to every thread.
__device__ float block_max(float v, float* red) {
    v = warp_max(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = red[0];
    for (int w = 1; w < kWarps; ++w) r = fmaxf(r, red[w]);
    __syncthreads();
    return r;
}
__device__ float block_sum(float v, float* red) {
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = red[0];
    for (int w = 1; w < kWarps; ++w) r += red[w];
    __syncthreads();
    return r;
}
// argmax with the lowest index winning ties
__device__ __forceinline__ void amax_merge(float& v, int& i, float v2, int i2) {
    if (v2 > v || (v2 == v && i2 < i)) {
        v = v2;
        i = i2;
    }
}

template <int NV4, bool GREEDY, bool VEC>
__global__ void __launch_bounds__(kThreads, 1) accept_rows_kernel(const AccParams p) {
    cg::cluster_group cluster = cg::this_cluster();
    const int CS = (int)cluster.num_blocks();
    const int c = (int)cluster.block_rank();
    const int rt = blockIdx.x / CS;  // global target row
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int V = p.vocab;

    __shared__ int32_t cu_sh[kMaxSmemSeqs + 1];
    __shared__ float red[kWarps];
    __shared__ int redi[kWarps];
    __shared__ float st_m[2], st_s[2], st_x[2];  // slice stats of target [0] and draft [1]
    __shared__ int st_has, st_gi;
    __shared__ float st_gv;
    __shared__ int last_sh, k_sh, seg_sh, dist_sh;
    __shared__ double cum_sh, z_sh;
    __shared__ double scan_sh[kWarps];

    // ---- 1. stream the target slice (independent of the sequence lookup)
    const int f0 = c * p.chunk4;
    const float* trow = p.target + (size_t)rt * V;
    float4 tv[NV4], dv[NV4];
#pragma unroll
    for (int j = 0; j < NV4; ++j) {
        const int fl = j * kThreads + tid;
        const int x = (f0 + fl) * 4;
        if (VEC) {
            tv[j] = (fl < p.chunk4 && x < V) ? __ldg(reinterpret_cast<const float4*>(trow + x))
                                             : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        } else {
            const bool in = fl < p.chunk4;
            tv[j].x = (in && x + 0 < V) ? __ldg(trow + x + 0) : -INFINITY;
            tv[j].y = (in && x + 1 < V) ? __ldg(trow + x + 1) : -INFINITY;
            tv[j].z = (in && x + 2 < V) ? __ldg(trow + x + 2) : -INFINITY;
            tv[j].w = (in && x + 3 < V) ? __ldg(trow + x + 3) : -INFINITY;
        }
    }

    // ---- 2. which sequence / position this target row belongs to
    int s;
    if (tid == 0) st_has = 0;
    if (p.num_seqs <= kMaxSmemSeqs)
        for (int i = tid; i <= p.num_seqs; i += kThreads) cu_sh[i] = p.cu_draft[i];
    __syncthreads();
    if (p.num_seqs <= kMaxSmemSeqs) {
        int lo = 0, hi = p.num_seqs;  // largest s with cu[s] + s <= rt
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (cu_sh[mid] + mid <= rt) lo = mid; else hi = mid;
        }
        s = lo;
    } else {
        int lo = 0, hi = p.num_seqs;
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(p.cu_draft + mid) + mid <= rt) lo = mid; else hi = mid;
        }
        s = lo;
    }
    const int d_begin = (p.num_seqs <= kMaxSmemSeqs) ? cu_sh[s] : __ldg(p.cu_draft + s);
    const int d_end = (p.num_seqs <= kMaxSmemSeqs) ? cu_sh[s + 1] : __ldg(p.cu_draft + s + 1);
    const int gamma = d_end - d_begin;
    const int tstart = d_begin + s;
    const int i = rt - tstart;
    const bool has_draft = i < gamma;
    int xi = has_draft ? __ldg(p.tokens + d_begin + i) : -1;
    if (has_draft && (xi < 0 || xi >= V)) {
        if (c == 0 && tid == 0) raise_error(p.err, kErrDeviceArg);
        xi = -1;
    }
    const bool use_draft = !GREEDY && has_draft;
    const float* drow = p.draft + (size_t)(d_begin + i) * V;
    if (use_draft) {
#pragma unroll
        for (int j = 0; j < NV4; ++j) {
            const int fl = j * kThreads + tid;
            const int x = (f0 + fl) * 4;
            if (VEC) {
                dv[j] = (fl < p.chunk4 && x < V) ? __ldg(reinterpret_cast<const float4*>(drow + x))
                                                 : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            } else {
                const bool in = fl < p.chunk4;
                dv[j].x = (in && x + 0 < V) ? __ldg(drow + x + 0) : -INFINITY;
                dv[j].y = (in && x + 1 < V) ? __ldg(drow + x + 1) : -INFINITY;
                dv[j].z = (in && x + 2 < V) ? __ldg(drow + x + 2) : -INFINITY;
                dv[j].w = (in && x + 3 < V) ? __ldg(drow + x + 3) : -INFINITY;
            }
        }
    }

    // slot of the drafted token inside this CTA's slice (if any)
    int own_j = -1, own_e = 0;
    if (xi >= 0) {
        const int fl = xi / 4 - f0;
        if (fl >= 0 && fl < p.chunk4 && fl % kThreads == tid) {
            own_j = fl / kThreads;
            own_e = xi & 3;
        }
    }

    if (GREEDY) {
        // ================= argmax of the target row
        float bv = -INFINITY;
        int bi = 0x7fffffff;
#pragma unroll
        for (int j = 0; j < NV4; ++j) {
            const int x = (f0 + j * kThreads + tid) * 4;
            amax_merge(bv, bi, tv[j].x, x + 0);
            amax_merge(bv, bi, tv[j].y, x + 1);
            amax_merge(bv, bi, tv[j].z, x + 2);
            amax_merge(bv, bi, tv[j].w, x + 3);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
            const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
            amax_merge(bv, bi, v2, i2);
        }
        if (lane == 0) {
            red[warp] = bv;
            redi[warp] = bi;
        }
        __syncthreads();
        if (tid == 0) {
            float v = red[0];
            int ix = redi[0];
            for (int w = 1; w < kWarps; ++w) amax_merge(v, ix, red[w], redi[w]);
            st_gv = v;
            st_gi = ix;
        }
        cluster.sync();
        if (c == 0 && tid == 0) {
            float v = -INFINITY;
            int ix = 0x7fffffff;
            for (int r = 0; r < CS; ++r)
                amax_merge(v, ix, *cluster.map_shared_rank(&st_gv, r), *cluster.map_shared_rank(&st_gi, r));
            if (ix >= V) ix = 0;  // every entry -inf: lowest index
            p.g_ws[rt] = ix;
            if (has_draft && p.accept_prob) p.accept_prob[d_begin + i] = (xi == ix) ? 1.f : 0.f;
            __threadfence();
        }
        cluster.sync();
    } else {
        // ================= softmax statistics of the slice
        const float c2 = p.c2;
        float mloc_t = -INFINITY, mloc_d = -INFINITY;
#pragma unroll
        for (int j = 0; j < NV4; ++j) {
            tv[j].x = scaled(tv[j].x, c2);
            tv[j].y = scaled(tv[j].y, c2);
            tv[j].z = scaled(tv[j].z, c2);
            tv[j].w = scaled(tv[j].w, c2);
            mloc_t = fmaxf(mloc_t, fmaxf(fmaxf(tv[j].x, tv[j].y), fmaxf(tv[j].z, tv[j].w)));
            if (use_draft) {
                dv[j].x = scaled(dv[j].x, c2);
                dv[j].y = scaled(dv[j].y, c2);
                dv[j].z = scaled(dv[j].z, c2);
                dv[j].w = scaled(dv[j].w, c2);
                mloc_d = fmaxf(mloc_d, fmaxf(fmaxf(dv[j].x, dv[j].y), fmaxf(dv[j].z, dv[j].w)));
            }
        }
        if (own_j >= 0) {
            // register-resident arrays: select the slot with compile-time indices only
            float tx_ = 0.f, dx_ = 0.f;
#pragma unroll
            for (int j = 0; j < NV4; ++j) {
                if (j == own_j) {
                    tx_ = own_e == 0 ? tv[j].x : own_e == 1 ? tv[j].y : own_e == 2 ? tv[j].z : tv[j].w;
                    if (use_draft) dx_ = own_e == 0 ? dv[j].x : own_e == 1 ? dv[j].y : own_e == 2 ? dv[j].z : dv[j].w;
                }
            }
            st_x[0] = tx_;
            st_x[1] = dx_;
            st_has = 1;
        }
        mloc_t = block_max(mloc_t, red);
        if (use_draft) mloc_d = block_max(mloc_d, red);
        float st = 0.f, sd = 0.f;
#pragma unroll
        for (int j = 0; j < NV4; ++j) {
            tv[j].x = expo(tv[j].x, mloc_t);
            tv[j].y = expo(tv[j].y, mloc_t);
            tv[j].z = expo(tv[j].z, mloc_t);
            tv[j].w = expo(tv[j].w, mloc_t);
            st += ((tv[j].x + tv[j].y) + (tv[j].z + tv[j].w));
            if (use_draft) {
                dv[j].x = expo(dv[j].x, mloc_d);
                dv[j].y = expo(dv[j].y, mloc_d);
                dv[j].z = expo(dv[j].z, mloc_d);
                dv[j].w = expo(dv[j].w, mloc_d);
                sd += ((dv[j].x + dv[j].y) + (dv[j].z + dv[j].w));
            }
        }
        st = block_sum(st, red);
        if (use_draft) sd = block_sum(sd, red);
        if (tid == 0) {
            st_m[0] = mloc_t;
            st_s[0] = st;
            st_m[1] = mloc_d;
            st_s[1] = sd;
        }
        cluster.sync();
        // ---- merge the CS slices: row max and normaliser of p and q (same order in every CTA)
        float mt = -INFINITY, md = -INFINITY;
        for (int r = 0; r < CS; ++r) {
            mt = fmaxf(mt, *cluster.map_shared_rank(&st_m[0], r));
            if (use_draft) md = fmaxf(md, *cluster.map_shared_rank(&st_m[1], r));
        }
        float zt = 0.f, zd = 0.f, tx = -INFINITY, dx = -INFINITY;
        for (int r = 0; r < CS; ++r) {
            const float m_r = *cluster.map_shared_rank(&st_m[0], r);
            zt += m_r == -INFINITY ? 0.f : *cluster.map_shared_rank(&st_s[0], r) * ex2(__fsub_rn(m_r, mt));
            if (use_draft) {
                const float md_r = *cluster.map_shared_rank(&st_m[1], r);
                zd += md_r == -INFINITY ? 0.f : *cluster.map_shared_rank(&st_s[1], r) * ex2(__fsub_rn(md_r, md));
            }
            if (*cluster.map_shared_rank(&st_has, r)) {
                tx = *cluster.map_shared_rank(&st_x[0], r);
                if (use_draft) dx = *cluster.map_shared_rank(&st_x[1], r);
            }
        }
        cluster.sync();  // peers' shared memory is no longer read after this point

        const float ft = __fdiv_rn(expo(mloc_t, mt), zt);
        const float fd = use_draft ? __fdiv_rn(expo(mloc_d, md), zd) : 0.f;
        if (tid == 0) {
            p.rowinfo[(size_t)rt * CS + c] = make_float4(mloc_t, mloc_d, ft, fd);
            if (c == 0 && has_draft) {
                // a = min(1, p(x)/q(x)) evaluated in the log domain
                float a;
                if (xi < 0 || tx == -INFINITY) a = 0.f;
                else if (dx == -INFINITY) a = 1.f;
                else {
                    const float lr = (tx - mt) - (dx - md);
                    a = fminf(1.f, ex2(lr) * (zd / zt));
                }
                p.a_ws[d_begin + i] = a;
                if (p.accept_prob) p.accept_prob[d_begin + i] = a;
            }
        }
        // ---- speculative segment sums of r = max(0, p - q) and of p (128 entries per (j, warp))
        float* segr = p.seg_r + (size_t)rt * p.nseg;
        float* segp = p.seg_p + (size_t)rt * p.nseg;
#pragma unroll
        for (int j = 0; j < NV4; ++j) {
            const float p0 = __fmul_rn(tv[j].x, ft), p1 = __fmul_rn(tv[j].y, ft);
            const float p2 = __fmul_rn(tv[j].z, ft), p3 = __fmul_rn(tv[j].w, ft);
            float rs = 0.f;
            if (use_draft) {
                rs = fmaxf(0.f, __fsub_rn(p0, __fmul_rn(dv[j].x, fd))) + fmaxf(0.f, __fsub_rn(p1, __fmul_rn(dv[j].y, fd))) +
                     fmaxf(0.f, __fsub_rn(p2, __fmul_rn(dv[j].z, fd))) + fmaxf(0.f, __fsub_rn(p3, __fmul_rn(dv[j].w, fd)));
            }
            float ps = ((p0 + p1) + (p2 + p3));
            rs = warp_sum(rs);
            ps = warp_sum(ps);
            if (lane == 0) {
                const int seg = (c * NV4 + j) * kWarps + warp;
                segr[seg] = rs;
                segp[seg] = ps;
            }
        }
        __threadfence();
    }

    // ---- 4. the last CTA of the sequence resolves the prefix and the emitted token
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        const int old = atomicAdd(p.tickets + s, 1);
        last_sh = (old == (gamma + 1) * CS - 1);
    }
    __syncthreads();
    if (!last_sh) return;
    __threadfence();
    if (tid == 0) {
        p.tickets[s] = 0;  // ready for the next call
        int k = gamma;
        for (int ii = 0; ii < gamma; ++ii) {
            bool acc;
            if (GREEDY) {
                acc = __ldcg(p.tokens + d_begin + ii) == __ldcg(p.g_ws + tstart + ii);
            } else {
                acc = __ldg(p.u_accept + d_begin + ii) < __ldcg(p.a_ws + d_begin + ii);
            }
            if (!acc) {
                k = ii;
                break;
            }
        }
        k_sh = k;
    }
    __syncthreads();
    const int k = k_sh;
    int token;
    if (GREEDY) {
        token = __ldcg(p.g_ws + tstart + k);
    } else {
        const int rk = tstart + k;
        const int nseg = p.nseg;
        const int per = (nseg + kThreads - 1) / kThreads;
        const int sb = min(nseg, tid * per), se = min(nseg, sb + per);
        // u in [0, 1): clamp so that the inverse CDF always has a crossing
        float u = __ldg(p.u_sample + s);
        if (!(u >= 0.f)) u = 0.f;
        u = fminf(u, 0.99999994f);
        // distribution: residual of row k (k < gamma), unless it vanishes; else p of row k
        for (int pass = (k < gamma ? 0 : 1); pass < 2; ++pass) {
            const float* seg = (pass == 0 ? p.seg_r : p.seg_p) + (size_t)rk * nseg;
            double loc = 0.0;
            for (int q = sb; q < se; ++q) loc += (double)__ldcg(seg + q);
            // exclusive block scan of the per-thread totals (fp64)
            double incl = loc;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const double y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            if (lane == 31) scan_sh[warp] = incl;
            if (tid == 0) seg_sh = 0x7fffffff;
            __syncthreads();
            double wbase = 0.0, total = 0.0;
            for (int w = 0; w < kWarps; ++w) {
                if (w < warp) wbase += scan_sh[w];
                total += scan_sh[w];
            }
            const double excl = wbase + incl - loc;
            if (pass == 0 && !(total > 0.0)) {
                __syncthreads();
                continue;  // p_k == q_k: draw from p_k instead
            }
            const double thr = (double)u * total;
            double cum = excl;
            for (int q = sb; q < se; ++q) {
                const double sq = (double)__ldcg(seg + q);
                if (sq > 0.0 && cum + sq > thr) {
                    atomicMin(&seg_sh, q);
                    break;
                }
                cum += sq;
            }
            __syncthreads();
            const int sel = seg_sh;
            if (sel >= sb && sel < se) {
                double cb = excl;
                for (int q = sb; q < sel; ++q) cb += (double)__ldcg(seg + q);
                cum_sh = cb;
                dist_sh = pass;
                z_sh = thr;
            }
            __syncthreads();
            break;
        }
        // re-scan the crossing segment (warp 0): bit-identical weights, fp64 running sum
        if (warp == 0 && seg_sh >= nseg) {
            // no positive mass at all (a row without a finite logit): report and emit 0
            if (lane == 0) {
                raise_error(p.err, kErrDeviceArg);
                k_sh = 0;
            }
        } else if (warp == 0) {
            const int sel = seg_sh;
            const int NW = NV4 * kWarps;
            const int cc = sel / NW, jj = (sel / kWarps) % NV4, ww = sel % kWarps;
            const float4 info = __ldcg(p.rowinfo + (size_t)rk * CS + cc);
            const int xbase = (cc * p.chunk4 + jj * kThreads + ww * 32 + lane) * 4;
            const bool fl_in = (jj * kThreads + ww * 32 + lane) < p.chunk4;
            float w4[4];
            const bool resid = dist_sh == 0;
            const float* tr = p.target + (size_t)rk * V;
            const float* dr = p.draft + (size_t)(d_begin + k) * V;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int x = xbase + e;
                float wv = 0.f;
                if (fl_in && x < V) {
                    const float pe = __fmul_rn(expo(scaled(__ldg(tr + x), p.c2), info.x), info.z);
                    if (resid) {
                        const float qe = __fmul_rn(expo(scaled(__ldg(dr + x), p.c2), info.y), info.w);
                        wv = fmaxf(0.f, __fsub_rn(pe, qe));
                    } else {
                        wv = pe;
                    }
                }
                w4[e] = wv;
            }
            const double lsum = (double)w4[0] + (double)w4[1] + (double)w4[2] + (double)w4[3];
            double incl = lsum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const double y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            double run = cum_sh + incl - lsum;
            const double thr = z_sh;
            int hit = -1;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                if (hit < 0 && w4[e] > 0.f && run + (double)w4[e] > thr) hit = xbase + e;
                run += (double)w4[e];
            }
            const unsigned any = __ballot_sync(0xffffffffu, hit >= 0);
            int chosen;
            if (any) {
                chosen = __shfl_sync(0xffffffffu, hit, __ffs(any) - 1);
            } else {
                // rounding left the crossing past the segment end: its last positive entry
                int lastpos = -1;
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (w4[e] > 0.f) lastpos = xbase + e;
                const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
                chosen = pos ? __shfl_sync(0xffffffffu, lastpos, 31 - __clz(pos)) : xbase - lane * 4;
            }
            if (lane == 0) k_sh = chosen;  // reuse: token
        }
        __syncthreads();
        token = k_sh;
    }
    // outputs of the sequence
    for (int ii = tid; ii <= gamma; ii += kThreads) {
        int v;
        if (ii < k) v = __ldg(p.tokens + d_begin + ii);
        else if (ii == k) v = token;
        else v = -1;
        p.out_tokens[tstart + ii] = v;
    }
    if (tid == 0) p.n_accepted[s] = k;
}

struct Config {
    int cs, nv4;
};

Config choose_config(int vocab) {
    const long long v4 = (vocab + 3) / 4;
    static const int nv4s[] = {1, 2, 4, 8, 10, 16};
    for (int cs = 1; cs <= 16; cs *= 2) {
        const long long per = (v4 + cs - 1) / cs;
        const long long need = (per + kThreads - 1) / kThreads;
        for (int n : nv4s)
            if (need <= n && (n <= 10 || cs == 16)) return Config{cs, n};
    }
    return Config{0, 0};
}

template <int NV4>
int launch_cfg(const AccParams& prm, int cs, bool greedy, bool vec, int total_rows, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)(total_rows * cs), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e;
    auto go = [&](auto kern) {
        if (cs > 8) cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        return cudaLaunchKernelEx(&cfg, kern, prm);
    };
    if (greedy) {
        e = vec ? go(accept_rows_kernel<NV4, true, true>) : go(accept_rows_kernel<NV4, true, false>);
    } else {
        e = vec ? go(accept_rows_kernel<NV4, false, true>) : go(accept_rows_kernel<NV4, false, false>);
    }
    return e == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

}  // namespace

size_t accept_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    const Config cfg = choose_config(vocab);
    if (cfg.cs == 0) return 0;
    const size_t rows = (size_t)total_draft + num_seqs;
    const size_t nseg = (size_t)cfg.cs * cfg.nv4 * kWarps;
    size_t b = 0;
    b += align_up(sizeof(int) * (size_t)num_seqs, 256);
    b += align_up(sizeof(float) * (size_t)total_draft, 256);
    b += align_up(sizeof(int) * rows, 256);
    b += align_up(sizeof(float4) * rows * cfg.cs, 256);
    b += 2 * align_up(sizeof(float) * rows * nseg, 256);
    return b;
}

int launch_accept(const AcceptArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    (void)dev;
    const Config cfg = choose_config(a.vocab);
    if (cfg.cs == 0) return BP_ERR_UNSUPPORTED;
    if (a.num_seqs == 0) return BP_OK;
    const size_t rows = (size_t)a.total_draft + a.num_seqs;
    const size_t nseg = (size_t)cfg.cs * cfg.nv4 * kWarps;
    uint8_t* w = static_cast<uint8_t*>(a.scratch);
    AccParams p;
    p.tickets = reinterpret_cast<int*>(w);
    w += align_up(sizeof(int) * (size_t)a.num_seqs, 256);
    p.a_ws = reinterpret_cast<float*>(w);
    w += align_up(sizeof(float) * (size_t)a.total_draft, 256);
    p.g_ws = reinterpret_cast<int*>(w);
    w += align_up(sizeof(int) * rows, 256);
    p.rowinfo = reinterpret_cast<float4*>(w);
    w += align_up(sizeof(float4) * rows * cfg.cs, 256);
    p.seg_r = reinterpret_cast<float*>(w);
    w += align_up(sizeof(float) * rows * nseg, 256);
    p.seg_p = reinterpret_cast<float*>(w);
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
    const long long v4 = (a.vocab + 3) / 4;
    p.chunk4 = (int)((v4 + cfg.cs - 1) / cfg.cs);
    p.nseg = (int)nseg;
    p.err = a.err_word;
    const bool vec = (a.vocab % 4 == 0) && (reinterpret_cast<uintptr_t>(a.target) % 16 == 0) &&
                     (greedy || reinterpret_cast<uintptr_t>(a.draft) % 16 == 0);
    switch (cfg.nv4) {
        case 1: return launch_cfg<1>(p, cfg.cs, greedy, vec, (int)rows, stream);
        case 2: return launch_cfg<2>(p, cfg.cs, greedy, vec, (int)rows, stream);
        case 4: return launch_cfg<4>(p, cfg.cs, greedy, vec, (int)rows, stream);
        case 8: return launch_cfg<8>(p, cfg.cs, greedy, vec, (int)rows, stream);
        case 10: return launch_cfg<10>(p, cfg.cs, greedy, vec, (int)rows, stream);
        case 16: return launch_cfg<16>(p, cfg.cs, greedy, vec, (int)rows, stream);
        default: return BP_ERR_UNSUPPORTED;
    }
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
    if (need > (size_t)BP_NOALLOC_SCRATCH_BYTES) return BP_ERR_WORKSPACE;  // problem too large for the array
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
    return launch_accept(a, dev, stream);
}

}  // namespace bp
