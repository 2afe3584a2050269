// Lossless speculative acceptance over the full vocabulary (the verification step of
// Figure 1 of the BlockPilot paper; the rule is standard speculative sampling).
//
// One thread-block cluster of CS CTAs per target row; the CTA of cluster rank c owns the
// c-th slice of the vocabulary of that target row and of the matching draft row.
//   load    one thread issues a single bulk copy (cp.async.bulk) per row slice into shared
//           memory, so each slice is one transfer in flight and the logits are read from HBM
//           exactly once;
//   pass 1  each thread walks its slots in batches of 16 entries keeping an online maximum
//           and sum of 2^(l*log2e/T - max); the weights replace the logits in place and each
//           batch records the maximum they are relative to.  Warp shuffles, then every CTA
//           pushes its slice statistics into every other CTA's shared memory (one cluster
//           barrier) and each derives the row's log-sum-exp and a_i = min(1, p(x_i)/q(x_i));
//   pass 2  one multiply per entry turns the stored weights into p and r = max(0, p - q);
//           128-entry segment sums go to exact 2^-52 fixed point, a second cluster exchange
//           of the slice totals locates the slice, then the segment, then the entry where the
//           inverse CDF of this row's own distribution crosses u_s * Z -- the token the
//           sequence emits if its first rejection falls on this row (a residual draw; a bonus
//           draw from p on the last row), computed speculatively by every row in parallel;
//   final   the CTA that wrote the last row token of a sequence (atomic ticket, no waiting)
//           finds the first rejection k from the a_i and emits the tokens of row k.
// Temperature 0 (greedy): one pass reduces the argmax (lowest index on ties).
#include <cooperative_groups.h>

#include <mutex>

#include "common.cuh"
#include "ptx_sm103.cuh"

namespace cg = cooperative_groups;

namespace bp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxSmemSeqs = 512;  // sequence offsets cached in shared memory (else binary search in L2)
constexpr int kMaxCS = 16;

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
    unsigned int* err;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// 2^(a - b) for scaled log-values, 0 when a is -inf
__device__ __forceinline__ float ex2d(float a, float b) { return a == -INFINITY ? 0.f : ex2(__fsub_rn(a, b)); }

// Probability mass in 2^-52 units: segment, slice and row sums are exact integer additions
// (a row's masses add up to about 1, i.e. about 2^52 units, far from the 2^64 limit).  Built
// from the float's fields with integer shifts (truncating below 2^-52): the float -> 64-bit
// integer conversion instruction runs on the slow FP64 pipe of this GPU.
__device__ __forceinline__ unsigned long long to_fix(float x) {
    const unsigned bits = __float_as_uint(x);
    const int e = (int)((bits >> 23) & 0xffu);  // x = mant * 2^(e - 150) for normal x >= 0
    if (e == 0 || (bits >> 31)) return 0ull;      // zero, denormal (< 2^-126) or negative
    const unsigned long long mant = (unsigned long long)((bits & 0x7fffffu) | 0x800000u);
    const int sh = e - 98;                         // x * 2^52 = mant * 2^(e - 98)
    if (sh >= 0) return sh < 40 ? mant << sh : ~0ull;  // x >= 2^12 is out of range: saturate
    return sh > -24 ? mant >> (-sh) : 0ull;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_incl_scan_f(float v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}
__device__ __forceinline__ unsigned long long warp_incl_scan(unsigned long long v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}
// merge two (scaled max, sum) pairs of a log-sum-exp
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
    const float M = fmaxf(m, m2);
    s = s * ex2d(m, M) + s2 * ex2d(m2, M);
    m = M;
}
// argmax with the lowest index winning ties
__device__ __forceinline__ void amax_merge(float& v, int& i, float v2, int i2) {
    if (v2 > v || (v2 == v && i2 < i)) {
        v = v2;
        i = i2;
    }
}

__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_sync_all() {
    cluster_arrive_release();
    cluster_wait();
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

// Shared-memory layout of one CTA (dynamic part), for a slice of up to chunk4 float4 slots:
//   sT [chunk4] float4   target slice: raw logits, then (pass 1) the weights 2^(l*c2 - m_batch)
//   sD [chunk4] float4   draft slice, likewise
//   bmT, bmD [nb*256]    m_batch of every (batch, thread): the reference of the stored weights
//   segR, segP [nseg]    fixed-point segment sums of r and p
// Thread tid owns slots k*256 + tid; batch b is slots 4b..4b+3 of a thread; segment k*8 + w is
// the 128 entries of slot k held by warp w (in vocabulary order).
struct Smem {
    float4 *sT, *sD;
    float *bmT, *bmD;
    unsigned long long *segR, *segP;
};
__host__ __device__ inline size_t smem_bytes(int chunk4, bool greedy) {
    const int K = (chunk4 + kThreads - 1) / kThreads;
    const int nb = (K + 3) / 4;
    if (greedy) return (size_t)chunk4 * 16;
    return (size_t)chunk4 * 32 + (size_t)nb * kThreads * 8 + (size_t)K * kWarps * 16;
}
__device__ inline Smem carve(uint8_t* base, int chunk4) {
    const int K = (chunk4 + kThreads - 1) / kThreads;
    const int nb = (K + 3) / 4;
    Smem m;
    m.sT = reinterpret_cast<float4*>(base);
    m.sD = m.sT + chunk4;
    m.bmT = reinterpret_cast<float*>(m.sD + chunk4);
    m.bmD = m.bmT + nb * kThreads;
    m.segR = reinterpret_cast<unsigned long long*>(m.bmD + nb * kThreads);
    m.segP = m.segR + K * kWarps;
    return m;
}

// Brings a slice into shared memory: one bulk copy (16-byte aligned rows) or scalar loads.
template <bool VEC>
__device__ __forceinline__ void fetch_slice(float4* dst, const float* row, int f0, int n4, int V, uint64_t* bar,
                                            int tid) {
    if (VEC) {
        if (tid == 0 && n4 > 0) {
            mbar_arrive_expect_tx(bar, (uint32_t)n4 * 16u);
            bulk_load(dst, row + (size_t)f0 * 4, (uint32_t)n4 * 16u, bar);
        }
    } else {
        float* d = reinterpret_cast<float*>(dst);
        for (int idx = tid; idx < n4 * 4; idx += kThreads) {
            const int x = f0 * 4 + idx;
            d[idx] = x < V ? __ldg(row + x) : -INFINITY;
        }
    }
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
    __shared__ uint64_t bar_t, bar_d;
    __shared__ int32_t cu_sh[kMaxSmemSeqs + 1];
    __shared__ float4 red4[kWarps];
    __shared__ int red_i[kWarps];
    __shared__ float4 peer_stat[kMaxCS];     // (scaled max t, sum t, scaled max d, sum d)
    __shared__ float4 peer_x[kMaxCS];        // (t[x_i], d[x_i], owns x_i, -); greedy: (max, index)
    __shared__ ulonglong2 peer_tot[kMaxCS];  // slice totals of r and p (fixed point)
    __shared__ float4 own_sh;
    __shared__ ulonglong2 tot_sh[kWarps];
    __shared__ int sel_sh, last_sh, k_sh;
    __shared__ unsigned long long base_sh;

    cluster_arrive_relaxed();  // peers must be running before any distributed shared memory write
    const Smem sm = carve(dyn_smem, p.chunk4);
    const int v4 = (V + 3) / 4;
    const int f0 = c * p.chunk4;
    const int n4 = max(0, min(v4, f0 + p.chunk4) - f0);
    const float* trow = p.target + (size_t)rt * V;

    // ---- start the target slice's copy at once; the draft row needs the sequence lookup
    if (tid == 0) {
        mbar_init(&bar_t, 1);
        mbar_init(&bar_d, 1);
        fence_mbar_init();
        own_sh = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (VEC) fetch_slice<VEC>(sm.sT, trow, f0, n4, V, &bar_t, tid);
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
    const float* drow = p.draft + (size_t)(d_begin + i) * V;
    if (use_draft) fetch_slice<VEC>(sm.sD, drow, f0, n4, V, &bar_d, tid);
    if (!VEC) fetch_slice<VEC>(sm.sT, trow, f0, n4, V, &bar_t, tid);
    int xi = has_draft ? __ldg(p.tokens + d_begin + i) : -1;
    __syncthreads();  // barriers initialised, scalar fills complete
    if (has_draft && (xi < 0 || xi >= V)) {
        if (c == 0 && tid == 0) raise_error(p.err, kErrDeviceArg);
        xi = -1;
    }
    if (VEC && n4 > 0) {
        bool ok = mbar_wait(&bar_t, 0, kWaitBudget);
        if (use_draft) ok = mbar_wait(&bar_d, 0, kWaitBudget) && ok;
        if (!ok) raise_error(p.err, kErrTimeout);
    }
    const int K = (n4 + kThreads - 1) / kThreads;  // slots per thread (the last may be partial)
    const int nb = (K + 3) / 4;
    const float c2 = p.c2;

    if (GREEDY) {
        // ================= argmax of the target row
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int k = 0; k < K; ++k) {
            const int f = k * kThreads + tid;
            if (f < n4) {
                const float4 v = sm.sT[f];
                const int x = (f0 + f) * 4;
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
            p.tok_ws[rt] = ix;
            if (has_draft && p.accept_prob) p.accept_prob[d_begin + i] = (xi == ix) ? 1.f : 0.f;
        }
    } else {
        // the drafted token's raw logits, read before pass 1 overwrites the slice
        if (tid == 0 && xi >= 0 && xi / 4 >= f0 && xi / 4 < f0 + n4) {
            const int f = xi / 4 - f0;
            own_sh = make_float4(pick(sm.sT[f], xi & 3), use_draft ? pick(sm.sD[f], xi & 3) : 0.f, 1.f, 0.f);
        }
        __syncthreads();
        // ================= pass 1: online (scaled max, sum) per thread; weights stored in place
        float mt = -INFINITY, st = 0.f, md = -INFINITY, sd = 0.f;
        for (int b = 0; b < nb; ++b) {
            float4 tv[4], dv[4];
            float bt = -INFINITY, bd = -INFINITY;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int f = (4 * b + q) * kThreads + tid;
                tv[q] = f < n4 ? sm.sT[f] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
                bt = fmaxf(bt, max4(tv[q]));
                if (use_draft) {
                    dv[q] = f < n4 ? sm.sD[f] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
                    bd = fmaxf(bd, max4(dv[q]));
                }
            }
            if (bt != -INFINITY) {
                const float nm = fmaxf(mt, __fmul_rn(bt, c2));
                st *= ex2d(mt, nm);
                mt = nm;
            }
            sm.bmT[b * kThreads + tid] = mt;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int f = (4 * b + q) * kThreads + tid;
                if (f < n4) {
                    const float4 e = mt == -INFINITY ? make_float4(0.f, 0.f, 0.f, 0.f) : ex2_4(tv[q], c2, mt);
                    st += sum4(e);
                    sm.sT[f] = e;
                }
            }
            if (use_draft) {
                if (bd != -INFINITY) {
                    const float nm = fmaxf(md, __fmul_rn(bd, c2));
                    sd *= ex2d(md, nm);
                    md = nm;
                }
                sm.bmD[b * kThreads + tid] = md;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int f = (4 * b + q) * kThreads + tid;
                    if (f < n4) {
                        const float4 e = md == -INFINITY ? make_float4(0.f, 0.f, 0.f, 0.f) : ex2_4(dv[q], c2, md);
                        sd += sum4(e);
                        sm.sD[f] = e;
                    }
                }
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            lse_merge(mt, st, __shfl_xor_sync(0xffffffffu, mt, o), __shfl_xor_sync(0xffffffffu, st, o));
            lse_merge(md, sd, __shfl_xor_sync(0xffffffffu, md, o), __shfl_xor_sync(0xffffffffu, sd, o));
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
            *cluster.map_shared_rank(&peer_x[c], tid) = own_sh;
        }
        cluster_sync_all();
        // ---- row statistics (same order in every CTA of the cluster)
        float Mt = -INFINITY, Zt = 0.f, Md = -INFINITY, Zd = 0.f, tx = -INFINITY, dx = -INFINITY;
        for (int r = 0; r < CS; ++r) {
            lse_merge(Mt, Zt, peer_stat[r].x, peer_stat[r].y);
            lse_merge(Md, Zd, peer_stat[r].z, peer_stat[r].w);
            if (peer_x[r].z != 0.f) {
                tx = peer_x[r].x;
                dx = peer_x[r].y;
            }
        }
        if (c == 0 && tid == 0 && has_draft) {
            // a = min(1, p(x)/q(x)) evaluated in the log domain
            float a;
            if (xi < 0 || tx == -INFINITY) a = 0.f;
            else if (dx == -INFINITY) a = 1.f;
            else a = fminf(1.f, ex2(__fmaf_rn(tx, c2, -Mt) - __fmaf_rn(dx, c2, -Md)) * (Zd / Zt));
            p.a_ws[d_begin + i] = a;
            if (p.accept_prob) p.accept_prob[d_begin + i] = a;
            __threadfence();
        }

        // ================= pass 2: fixed-point segment sums of r and p, one multiply per entry
        const float izt = __fdiv_rn(1.f, Zt);
        const float izd = use_draft ? __fdiv_rn(1.f, Zd) : 0.f;
        unsigned long long totr = 0, totp = 0;
        for (int b = 0; b < nb; ++b) {
            const float bmt = sm.bmT[b * kThreads + tid];
            const float ft = bmt == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(bmt, Mt)), izt);
            float fd = 0.f;
            if (use_draft) {
                const float bmd = sm.bmD[b * kThreads + tid];
                fd = bmd == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(bmd, Md)), izd);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int k = 4 * b + q;
                if (k < K) {  // warp-uniform
                    const int f = k * kThreads + tid;
                    float sp = 0.f, sr = 0.f;
                    if (f < n4) {
                        const float4 pv = mul4(sm.sT[f], ft);
                        sp = sum4(pv);
                        if (use_draft) sr = sum4(resid4(pv, mul4(sm.sD[f], fd)));
                    }
                    sp = warp_sum(sp);
                    sr = warp_sum(sr);
                    if (lane == 0) {  // one fixed-point conversion per 128-entry segment
                        const unsigned long long fr = to_fix(sr), fp = to_fix(sp);
                        sm.segR[k * kWarps + warp] = fr;
                        sm.segP[k * kWarps + warp] = fp;
                        totr += fr;
                        totp += fp;
                    }
                }
            }
        }
        if (lane == 0) tot_sh[warp] = make_ulonglong2(totr, totp);
        __syncthreads();
        if (tid < CS) {
            ulonglong2 t = tot_sh[0];
            for (int w = 1; w < kWarps; ++w) {
                t.x += tot_sh[w].x;
                t.y += tot_sh[w].y;
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
        float u = __ldg(p.u_sample + s);
        if (!(u >= 0.f)) u = 0.f;
        u = fminf(u, 0.99999994f);  // u in [0, 1): the crossing always exists
        const unsigned long long thr = __umul64hi(__float2ull_rn(u * 18446744073709551616.f), total);
        if (total == 0) {
            // no positive mass at all (a row without a finite logit): report, emit 0
            if (c != 0) return;
            if (tid == 0) {
                raise_error(p.err, kErrDeviceArg);
                p.tok_ws[rt] = 0;
            }
        } else {
            if (!(below <= thr && thr < below + mine)) return;  // the crossing is in another slice
            // ---- segment of this slice (block scan of the segment sums, exact)
            const unsigned long long* seg = use_r ? sm.segR : sm.segP;
            const int nseg = K * kWarps;
            const int per = (nseg + kThreads - 1) / kThreads;
            const int sb = min(nseg, tid * per), se = min(nseg, sb + per);
            unsigned long long loc = 0;
            for (int q = sb; q < se; ++q) loc += seg[q];
            const unsigned long long incl = warp_incl_scan(loc, lane);
            if (lane == 31) tot_sh[warp].x = incl;
            if (tid == 0) sel_sh = 0x7fffffff;
            __syncthreads();
            unsigned long long cum = below + incl - loc;
            for (int w = 0; w < warp; ++w) cum += tot_sh[w].x;
            for (int q = sb; q < se; ++q) {
                if (seg[q] > 0 && cum <= thr && thr < cum + seg[q]) {
                    sel_sh = q;  // exact integer sums: exactly one segment holds the threshold
                    base_sh = cum;
                    break;
                }
                cum += seg[q];
            }
            __syncthreads();
            const int sel = sel_sh;
            // ---- entry of the segment (warp 0): the stored weights of its owner thread
            if (warp == 0) {
                if (sel >= nseg) {  // unreachable with exact sums: report, emit the slice's first entry
                    if (lane == 0) {
                        raise_error(p.err, kErrDeviceArg);
                        p.tok_ws[rt] = f0 * 4;
                    }
                } else {
                    const int k = sel / kWarps, w = sel % kWarps;
                    const int owner = w * 32 + lane;  // thread whose slot k holds this lane's entries
                    const int f = k * kThreads + owner;
                    const int b = k / 4;
                    float4 wv = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (f < n4) {
                        const float bmt = sm.bmT[b * kThreads + owner];
                        const float ft = bmt == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(bmt, Mt)), izt);
                        wv = mul4(sm.sT[f], ft);
                        if (use_r) {
                            const float bmd = sm.bmD[b * kThreads + owner];
                            const float fd = bmd == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(bmd, Md)), izd);
                            wv = resid4(wv, mul4(sm.sD[f], fd));
                        }
                    }
                    const float wa[4] = {wv.x, wv.y, wv.z, wv.w};
                    // offset of the threshold inside the segment, back in probability units
                    const float off = __ull2float_rn(thr - base_sh) * 2.220446049250313e-16f;
                    const float lsum = (wa[0] + wa[1]) + (wa[2] + wa[3]);
                    float run = warp_incl_scan_f(lsum, lane) - lsum;
                    const int x0 = (f0 + f) * 4;
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
                    if (lane == 0) p.tok_ws[rt] = first;
                }
            }
        }
    }

    // ---- this CTA wrote the row's token: take a ticket; the last row of the sequence resolves it
    if (tid == 0) {
        __threadfence();
        const int old = atomicAdd(p.tickets + s, 1);
        last_sh = (old == gamma);
        k_sh = gamma;
    }
    __syncthreads();
    if (!last_sh) return;
    __threadfence();
    if (tid == 0) p.tickets[s] = 0;  // ready for the next call
    int my_tok = -1;  // drafted token of position tid (first iteration)
    for (int ii = tid; ii <= gamma; ii += kThreads) {
        const int tok = ii < gamma ? __ldg(p.tokens + d_begin + ii) : -1;
        bool rej = false;
        if (ii < gamma) {
            rej = GREEDY ? (tok != __ldcg(p.tok_ws + tstart + ii))
                         : !(__ldg(p.u_accept + d_begin + ii) < __ldcg(p.a_ws + d_begin + ii));
        }
        if (rej) atomicMin(&k_sh, ii);
        if (ii == tid) my_tok = tok;
    }
    __syncthreads();
    const int k = k_sh;
    const int token = __ldcg(p.tok_ws + tstart + k);
    for (int ii = tid; ii <= gamma; ii += kThreads) {
        int v;
        if (ii < k) v = (ii < kThreads) ? my_tok : __ldg(p.tokens + d_begin + ii);
        else if (ii == k) v = token;
        else v = -1;
        p.out_tokens[tstart + ii] = v;
    }
    if (tid == 0) p.n_accepted[s] = k;
}

constexpr size_t kSmemBudget = 108 * 1024;  // dynamic shared memory per CTA: two CTAs per SM

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
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, accept_kernel<GREEDY, VEC>, p) == cudaSuccess ? BP_OK : BP_ERR_CUDA;
}

}  // namespace

size_t accept_scratch_bytes(int num_seqs, int total_draft, int vocab) {
    if (vocab < 1 || min_cluster(vocab, false) == 0) return 0;  // slices must fit in shared memory
    const size_t rows = (size_t)total_draft + num_seqs;
    size_t b = 0;
    b += align_up(sizeof(int) * (size_t)num_seqs, 256);    // tickets (first: cleared by the no-workspace path)
    b += align_up(sizeof(float) * (size_t)total_draft, 256);
    b += align_up(sizeof(int) * rows, 256);
    return b;
}

int launch_accept(const AcceptArgs& a, const DeviceInfo& dev, cudaStream_t stream) {
    if (accept_scratch_bytes(a.num_seqs, a.total_draft, a.vocab) == 0) return BP_ERR_UNSUPPORTED;
    if (a.num_seqs == 0) return BP_OK;
    const int rows = a.total_draft + a.num_seqs;
    uint8_t* w = static_cast<uint8_t*>(a.scratch);
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
