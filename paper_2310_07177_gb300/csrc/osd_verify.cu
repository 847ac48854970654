// osd_verify.cu -- speculative-sampling verification (Section 3 and
// Appendix A.1 of the paper; the verify step of Algorithm 1) on sm_103a.
//
// Two launches on the caller's stream:
//
//   row_stats_kernel    one CTA per (row, vocabulary slice) over all B*k draft
//                       rows and B*(k+1) target rows: a single streaming pass of
//                       16-byte loads computing the online max and sum of
//                       exp((x - max)/T) of the slice (or the argmax for T = 0).
//                       This pass reads every logit once and carries almost all
//                       of the operation's HBM traffic.
//   verify_finalize     (T > 0) one thread-block cluster per sequence: merges the slice
//                       statistics, runs the k accept tests u_i < p_i(y_i)/q_i(y_i),
//                       all at once (a is the first failure), then draws the extra token from
//                       norm(max(0, p_a - q_a)) (or p_k when all k pass) by inverse
//                       CDF.  Each CTA of the cluster sums the residual weights of
//                       its part of the vocabulary per tile; the partial sums meet
//                       through distributed shared memory as exact 64-bit fixed
//                       point, and the CTA whose part holds u*W rescans that one
//                       tile with an exact warp scan.
//
//   verify_greedy       (T = 0) one warp per sequence: the argmax of every target
//                       row from its slices, the matches in order, the target
//                       argmax at the first mismatch.
//
// The log-ratio of the accept test is formed from differences of raw logits and
// maxima, (t_y - m_t) - (z_y - m_z), and the ratio of the two sums, so no
// log-sum-exp is rounded on its own.
#include <cuda.h>

#include <atomic>
#include <climits>
#include <cstdint>
#include <mutex>
#include <type_traits>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"
#include "osd_rowstats.cuh"

namespace osd {

constexpr int kFinThreads = 128;
constexpr int kFinMaxCluster = 8;
constexpr uint64_t kDrawWaitNs = 3000000000ull;  // bound on the wait for the pushed span totals
constexpr int kFinMaxSub = 8192;  // sub-tiles of one CTA's vocabulary span (>= span / 32)
constexpr int kFinUnroll = 4;     // sub-tiles of loads in flight per warp

// ------------------------------------------------------------------ pass 2
struct FinParams {
    const void* draft;
    const void* target;
    int B, k, V;
    const int32_t* tokens;
    const float* uniforms;
    float T, c_hi, c_lo;
    const RowStat* stats;
    int n_slices;
    long long n_draft_rows;  // B*k when draft rows have statistics, 0 for greedy
    int32_t* accepted;
    int32_t* out_tokens;
    uint8_t* mask;
    float* diag_margin;
    float* diag_gap;
    int csize;  // CTAs per sequence (cluster size)
    int span;   // vocabulary entries per CTA of the cluster
};


// T = 0: the accept tests are argmax matches, and the extra token is the target
// argmax at the first mismatch.  One warp per sequence, a small kernel of its
// own: at serving batch sizes this pass is latency-bound, and a compact kernel
// starts faster than the sampling kernel with its greedy branch would.
constexpr int kGreedyWarps = 4;
__global__ void __launch_bounds__(kGreedyWarps * 32) verify_greedy_kernel(FinParams p) {
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.x * kGreedyWarps + (threadIdx.x >> 5);
    if (b >= p.B) return;
    const int k = p.k, V = p.V;
    const int32_t* y = p.tokens + size_t(b) * k;
    // the draft tokens before the statistics are needed (one round of loads)
    constexpr int kC = (OSD_VERIFY_MAX_K + 1 + 31) / 32;
    int yv[kC];
    bool bad = false;
#pragma unroll
    for (int c = 0; c < kC; ++c) {
        const int i = c * 32 + lane;
        yv[c] = (i < k) ? y[i] : 0;
        bad |= (i < k) && (yv[c] < 0 || yv[c] >= V);
    }
    grid_dependency_wait();  // the row statistics are complete from here on
    // row i <= k of the sequence: its target argmax, lowest index on ties, merged
    // from the slices by the lane that owns the row
    int idx[kC];
    unsigned fail = 0;
    int a = k;
#pragma unroll
    for (int c = 0; c < kC; ++c) {
        const int i = c * 32 + lane;
        idx[c] = 0;
        if (i <= k) {
            const RowStat* st = p.stats + ((long long)b * (k + 1) + i) * p.n_slices;
            MaxIdx acc{kNegInf, INT_MAX};
            for (int sl = 0; sl < p.n_slices; ++sl) acc = merge_mi(acc, MaxIdx{st[sl].m, st[sl].idx});
            idx[c] = (acc.i == INT_MAX) ? 0 : acc.i;
        }
        fail = __ballot_sync(0xffffffffu, i < k && yv[c] != idx[c]);
        if (fail && a == k) a = c * 32 + __ffs(fail) - 1;
    }
    bad = __any_sync(0xffffffffu, bad);
    int32_t* out = p.out_tokens + size_t(b) * (k + 1);
    if (lane == 0) {
        p.accepted[b] = bad ? -1 : a;
        if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000);
    }
    // the token at a is the target argmax there, held by lane a % 32 in slot a / 32
    int at = 0;
#pragma unroll
    for (int c = 0; c < kC; ++c) {
        const int v = __shfl_sync(0xffffffffu, idx[c], a & 31);
        if (c == a / 32) at = v;
    }
#pragma unroll
    for (int c = 0; c < kC; ++c) {
        const int i = c * 32 + lane;
        if (i <= k) out[i] = bad ? -1 : (i < a ? yv[c] : (i == a ? at : -1));
        if (i < k) {
            p.mask[size_t(b) * k + i] = (!bad && i == a) ? 1 : 0;
            if (p.diag_margin) p.diag_margin[size_t(b) * k + i] = __int_as_float(0x7fc00000);
        }
    }
}

// Shared memory of one sequence's decision: the merged statistics of its 2k+1
// rows (local row r <= k is target row r, r > k is draft row r-k-1), the draft
// tokens, the two logits each accept test needs, the uniforms, and a.
struct SeqSmem {
    float m[2 * OSD_VERIFY_MAX_K + 1];
    float s[2 * OSD_VERIFY_MAX_K + 1];
    float zy[OSD_VERIFY_MAX_K], ty[OSD_VERIFY_MAX_K];
    int y[OSD_VERIFY_MAX_K];
    float u[OSD_VERIFY_MAX_K + 1];
    int a;
};

// Prologue of sequence b's decision, run by every thread of a CTA of kThreads:
// every independent global load goes out in one round (the last warp fetches
// the draft tokens and gathers the two logits each accept test needs, the warp
// before it the uniforms); then, once the row statistics are complete, the
// warps merge each row's slice statistics, loading up to four rows per lane
// before reducing.  Returns non-zero, for every thread, when a draft token
// lies outside [0, V).
template <typename In, int kThreads>
__device__ __forceinline__ int seq_prologue(const FinParams& p, int b, SeqSmem& sh) {
    using E = Elem<In>;
    constexpr int kWarps = kThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int k = p.k, V = p.V;
    const int32_t* y = p.tokens + size_t(b) * k;
    const In* draft = static_cast<const In*>(p.draft);
    const In* target = static_cast<const In*>(p.target);
    int bad = 0;
    if (warp == kWarps - 1) {
        for (int i = lane; i < k; i += 32) {
            const int t = y[i];
            sh.y[i] = t;
            if (t < 0 || t >= V) {
                bad = 1;
            } else {
                sh.zy[i] = E::load(draft + (size_t(b) * k + i) * V + t);
                sh.ty[i] = E::load(target + (size_t(b) * (k + 1) + i) * V + t);
            }
        }
    }
    if (warp == kWarps - 2)
        for (int i = lane; i <= k; i += 32) sh.u[i] = p.uniforms[size_t(b) * (k + 1) + i];
    grid_dependency_wait();  // the row statistics are complete from here on
    const int nrows = 2 * k + 1;
    const float ch0 = p.c_hi, cl0 = p.c_lo;
    auto srow_of = [&](int r) -> long long {
        return (r <= k) ? (p.n_draft_rows + (long long)b * (k + 1) + r) : ((long long)b * k + (r - k - 1));
    };
    for (int r0 = warp; r0 < nrows; r0 += 4 * kWarps) {
        RowStat part[4][1];
        bool have[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int r = r0 + q * kWarps;
            have[q] = r < nrows && lane < p.n_slices;
            if (have[q]) part[q][0] = p.stats[srow_of(r) * p.n_slices + lane];
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int r = r0 + q * kWarps;
            if (r >= nrows) break;  // uniform across the warp
            const RowStat* st = p.stats + srow_of(r) * p.n_slices;
            auto merge = [ch0, cl0](MaxSum x, MaxSum z) { return merge_ms(x, z, ch0, cl0); };
            MaxSum acc{kNegInf, 0.f};
            if (have[q]) acc = MaxSum{part[q][0].m, part[q][0].s};
            for (int sl = lane + 32; sl < p.n_slices; sl += 32) acc = merge(acc, MaxSum{st[sl].m, st[sl].s});
            acc = warp_reduce(acc, merge);
            if (lane == 0) { sh.m[r] = acc.m; sh.s[r] = acc.s; }
        }
    }
    return __syncthreads_or(bad);
}

// Outputs of a sequence with a bad draft token (one CTA of kThreads writes them).
template <int kThreads>
__device__ __forceinline__ void seq_write_bad(const FinParams& p, int b) {
    const int tid = threadIdx.x, k = p.k;
    int32_t* out = p.out_tokens + size_t(b) * (k + 1);
    if (tid == 0) { p.accepted[b] = -1; if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000); }
    for (int i = tid; i <= k; i += kThreads) out[i] = -1;
    for (int i = tid; i < k; i += kThreads) {
        p.mask[size_t(b) * k + i] = 0;
        if (p.diag_margin) p.diag_margin[size_t(b) * k + i] = __int_as_float(0x7fc00000);
    }
}

// The k accept tests: warp 0 runs them all at once, one position per lane, and
// the first failing position is a (the tests after it are not decided).  Sets
// sh.a, writes the margins of the decided positions when `margins` is set, and
// ends on a block barrier.
__device__ __forceinline__ void seq_accept(const FinParams& p, int b, SeqSmem& sh, bool margins) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, k = p.k;
    if (warp == 0) {
        int a = k;
        float r_all[(OSD_VERIFY_MAX_K + 31) / 32];
#pragma unroll
        for (int c = 0; c < (OSD_VERIFY_MAX_K + 31) / 32; ++c) {
            const int i = c * 32 + lane;
            bool fail = false;
            r_all[c] = 0.f;
            if (i < k) {
                const float mt = sh.m[i], st = sh.s[i];
                const float mz = sh.m[k + 1 + i], sz = sh.s[k + 1 + i];
                const float D = (sh.ty[i] - mt) - (sh.zy[i] - mz);
                r_all[c] = expf(__fdiv_rn(D, p.T)) * __fdiv_rn(sz, st);
                fail = !(sh.u[i] < r_all[c]);
            }
            const unsigned f = __ballot_sync(0xffffffffu, fail);
            if (f && a == k) a = c * 32 + __ffs(f) - 1;
        }
        if (margins) {
#pragma unroll
            for (int c = 0; c < (OSD_VERIFY_MAX_K + 31) / 32; ++c) {
                const int i = c * 32 + lane;
                if (i < k && i <= a) p.diag_margin[size_t(b) * k + i] = fabsf(sh.u[i] - r_all[c]);
            }
        }
        if (lane == 0) sh.a = a;
    }
    __syncthreads();
}

// accepted, the accepted tokens and the -1 padding after a, the mask, and the
// margins past the decision (one CTA of kThreads); the token at a is the draw's.
template <int kThreads>
__device__ __forceinline__ void seq_write_outputs(const FinParams& p, int b, const SeqSmem& sh, int a) {
    const int tid = threadIdx.x, k = p.k;
    int32_t* out = p.out_tokens + size_t(b) * (k + 1);
    if (tid == 0) p.accepted[b] = a;
    for (int i = tid; i <= k; i += kThreads)
        if (i < a) out[i] = sh.y[i];
        else if (i > a) out[i] = -1;
    for (int i = tid; i < k; i += kThreads) {
        p.mask[size_t(b) * k + i] = (i == a) ? 1 : 0;
        if (p.diag_margin && i > a) p.diag_margin[size_t(b) * k + i] = __int_as_float(0x7fc00000);
    }
}

// Shared memory of the extra token's draw (span_total is read by the other CTAs
// of the cluster).
struct DrawSmem {
    unsigned long long span_total;
    unsigned long long tau, W, base;
    int owner, mode, tile;
    // pushed span totals (the one-launch kernel): slot r from CTA r, completing on tbar
    unsigned long long totals[kFinMaxCluster];
    uint64_t tbar;
};

// The extra token of sequence b (Appendix A.1; reading 4 and 4b for the
// convention and the arithmetic): inverse CDF of w = max(0, p_a - q_a) when
// a < k, of p_k when a = k.  This CTA, rank `rank` of a cluster of p.csize,
// owns entries [e0, e0 + n) of the vocabulary: it sums their weights per
// sub-tile (fp32 in a warp, exact 64-bit fixed point beyond), the CTAs' span
// totals meet through distributed shared memory, and the CTA whose span holds
// tau = floor(u W) rescans that one sub-tile exactly.  Entry j of the target and
// draft rows at position a is trow[j - off], zrow[j - off], in shared memory when
// kSmem (a staged span) and global memory otherwise; trow_g is the whole target
// row in global memory, for the case W = 0 (argmax of p_a).  s_sub holds at least
// n / (32 kW) floats.  Every thread calls it.  Without kPush the totals are read
// from the peers' shared memory after a cluster barrier, and the draw ends
// having arrived (relaxed) at the cluster barrier, where the caller waits before
// it exits.  With kPush (ds.tbar initialised with count 1 and visible to the
// cluster) each CTA pushes its total by st.async into slot `rank` of every CTA's
// ds.totals and waits on its own ds.tbar: no cluster barrier, nothing read from
// a peer.  Returns false if that wait gave up (the draw is then not made).
template <typename In, bool kVecPath, int kThreads, bool kSmem, bool kPush = false>
__device__ __forceinline__ bool residual_draw(const FinParams& p, int b, int a, const SeqSmem& sh, int rank,
                                              int e0, int n, const In* trow, const In* zrow, int off,
                                              const In* trow_g, float* s_sub, DrawSmem& ds) {
    using E = Elem<In>;
    constexpr int kW = kVecPath ? E::kVec : 1;  // entries per lane per sub-tile
    constexpr int kSub = 32 * kW;
    constexpr int kWarps = kThreads / 32;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int k = p.k, V = p.V;
    const bool bonus = (a == k);
    int32_t* out = p.out_tokens + size_t(b) * (k + 1);
    // entry j of the two rows: trow[j - off], zrow[j - off], from shared memory when kSmem
    auto ldv = [&](const In* q) { return kSmem ? lds_v4(q) : ldg_stream(q); };
    auto ld1 = [&](const In* q) { return kSmem ? E::lds(q) : E::load(q); };
    const float mt = sh.m[a], inv_st = 1.0f / sh.s[a];
    const float mz = bonus ? 0.f : sh.m[k + 1 + a];
    const float inv_sz = bonus ? 0.f : 1.0f / sh.s[k + 1 + a];
    const float ch = p.c_hi, cl = p.c_lo;
    auto weight = [&](float t, float z) -> float {
        const float pj = ex2(mul_c(t - mt, ch, cl)) * inv_st;
        if (bonus) return pj;
        const float qj = ex2(mul_c(z - mz, ch, cl)) * inv_sz;
        return fmaxf(pj - qj, 0.f);
    };
    const int nsub = (n + kSub - 1) / kSub;  // sub-tiles: one warp step of 32 x kW entries
    // raw entries of this lane in sub-tile s (slots past the span read as -inf: weight 0)
    struct Raw {
        uint4 t, z;
    };
    auto load_sub = [&](int s, Raw& r) {
        const int j0 = e0 + s * kSub + lane * kW;
        const int cnt = min(kW, e0 + n - j0);
        if (kVecPath && cnt == kW) {
            r.t = ldv(trow + (j0 - off));
            r.z = bonus ? r.t : ldv(zrow + (j0 - off));
        } else {
            float tv[kW], zv[kW];
#pragma unroll
            for (int e = 0; e < kW; ++e) {
                tv[e] = (e < cnt) ? ld1(trow + (j0 - off) + e) : kNegInf;
                zv[e] = (e < cnt && !bonus) ? ld1(zrow + (j0 - off) + e) : kNegInf;
            }
            r.t = pack_raw<In, kW>(tv);
            r.z = pack_raw<In, kW>(zv);
        }
    };
    // residual weights of one sub-tile slot, two entries per packed f32x2 step
    // (the same operations as `weight`, so both passes round identically)
    auto sub_weights = [&](const Raw& r, float* w) {
        float tv[kW], zv[kW];
        unpack_raw<In, kW>(r.t, tv);
        unpack_raw<In, kW>(r.z, zv);
        if constexpr (kW == 1) {
            w[0] = weight(tv[0], zv[0]);
        } else {
#pragma unroll
            for (int e = 0; e < kW; e += 2) {
                const float2 dt = sub2(make_float2(tv[e], tv[e + 1]), f2(mt));
                const float2 at = fma2(dt, f2(ch), mul2(dt, f2(cl)));
                const float2 pj = mul2(make_float2(ex2(at.x), ex2(at.y)), f2(inv_st));
                if (bonus) {
                    w[e] = pj.x;
                    w[e + 1] = pj.y;
                } else {
                    const float2 dz = sub2(make_float2(zv[e], zv[e + 1]), f2(mz));
                    const float2 az = fma2(dz, f2(ch), mul2(dz, f2(cl)));
                    const float2 qj = mul2(make_float2(ex2(az.x), ex2(az.y)), f2(inv_sz));
                    const float2 df = sub2(pj, qj);
                    w[e] = fmaxf(df.x, 0.f);
                    w[e + 1] = fmaxf(df.y, 0.f);
                }
            }
        }
    };

    // pass 1: one fp32 sum per sub-tile, reduced inside the warp, no block barrier
    for (int s0 = warp; s0 < nsub; s0 += kWarps * kFinUnroll) {
        Raw r[kFinUnroll];
#pragma unroll
        for (int u = 0; u < kFinUnroll; ++u)
            if (s0 + u * kWarps < nsub) load_sub(s0 + u * kWarps, r[u]);
#pragma unroll
        for (int u = 0; u < kFinUnroll; ++u) {
            const int s = s0 + u * kWarps;
            if (s < nsub) {
                float w[kW];
                sub_weights(r[u], w);
                float sum = 0.f;
#pragma unroll
                for (int e = 0; e < kW; ++e) sum += w[e];
                for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
                if (lane == 0) s_sub[s] = sum;
            }
        }
    }
    __syncthreads();
    // span total, exact, reduced across warp 0
    bool got = true;
    if (warp == 0) {
        unsigned long long part = 0ull;
        for (int s2 = lane; s2 < nsub; s2 += 32) part += fix_of(s_sub[s2]);
        part = warp_sum_u64(part);
        if (lane == 0) ds.span_total = part;
        if (kPush && p.csize > 1) {
            if (lane < p.csize)
                st_async_u64(map_rank(&ds.totals[rank], static_cast<uint32_t>(lane)), part,
                             map_rank(&ds.tbar, static_cast<uint32_t>(lane)));
            if (lane == 0) mbar_arrive_expect_tx(&ds.tbar, static_cast<uint32_t>(p.csize) * 8u);
            got = __all_sync(0xffffffffu, mbar_wait_cluster_bounded(&ds.tbar, 0, kDrawWaitNs));
        }
    }
    if (!kPush && p.csize > 1) cluster_sync_publish(tid == 0); else __syncthreads();

    // warp 0 of every CTA derives W, tau = floor(u W) and the owning CTA identically:
    // lane r holds CTA r's total, a warp scan gives the prefix in rank order
    if (warp == 0 && got) {
        const float u = sh.u[k];
        unsigned long long tot = 0ull;
        if (lane < p.csize) {
            if (kPush) tot = (p.csize > 1) ? ds.totals[lane] : ds.span_total;
            else tot = (lane == rank) ? ds.span_total : ld_dsmem_u64(map_rank(&ds.span_total, lane));
        }
        const unsigned long long incl = warp_incl_scan_u64(tot);
        const unsigned long long W = __shfl_sync(0xffffffffu, incl, 31);
        const unsigned long long tau = fix_scale(u, W);
        int owner, mode = 0;  // mode 0: inverse CDF, 1: largest positive entry, 2: argmax p
        unsigned long long base = 0ull;
        if (W > 0ull) {
            const unsigned hit = __ballot_sync(0xffffffffu, lane < p.csize && incl > tau);
            if (hit) {
                owner = __ffs(hit) - 1;
                base = __shfl_sync(0xffffffffu, incl - tot, owner);
            } else {  // tau >= W (u >= 1 or rounding): largest j with w_j > 0
                mode = 1;
                const unsigned pos = __ballot_sync(0xffffffffu, lane < p.csize && tot > 0ull);
                owner = 31 - __clz(pos);
            }
        } else {
            mode = 2;
            owner = 0;
        }
        int tile = -1;
        if (rank == owner) {
            // sub-tile holding tau: each lane owns a run of consecutive sub-tiles
            const int per = (nsub + 31) / 32;
            const int s_lo = min(nsub, lane * per), s_hi = min(nsub, s_lo + per);
            unsigned long long mine = 0ull;
            for (int s2 = s_lo; s2 < s_hi; ++s2) mine += fix_of(s_sub[s2]);
            const unsigned long long excl = base + warp_incl_scan_u64(mine) - mine;
            if (mode == 0) {
                const unsigned hit = __ballot_sync(0xffffffffu, excl <= tau && excl + mine > tau);
                if (hit) {
                    const int l = __ffs(hit) - 1;
                    if (lane == l) {  // the sums are exact: the run holds tau in one sub-tile
                        unsigned long long c = excl;
                        for (int s2 = s_lo; s2 < s_hi; ++s2) {
                            const unsigned long long v = fix_of(s_sub[s2]);
                            if (c + v > tau) { tile = s2; break; }
                            c += v;
                        }
                        base = c;
                    }
                    tile = __shfl_sync(0xffffffffu, tile, l);
                    base = __shfl_sync(0xffffffffu, base, l);
                } else {
                    mode = 1;
                }
            }
            if (mode == 1) {  // the last sub-tile with positive mass
                int last = -1;
                for (int s2 = s_lo; s2 < s_hi; ++s2)
                    if (s_sub[s2] > 0.f) last = s2;
                for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
                tile = last;
            }
        }
        if (lane == 0) { ds.owner = owner; ds.mode = mode; ds.tau = tau; ds.W = W; ds.base = base; ds.tile = tile; }
    }
    if (warp == 0 && lane == 0 && !got) ds.owner = -1;
    __syncthreads();
    if (!kPush && p.csize > 1) cluster_arrive_relaxed();  // done reading the other CTAs' shared memory
    if (ds.owner < 0) return false;

    if (rank == ds.owner && warp == 0) {
        const unsigned long long tau = ds.tau, W = ds.W;
        const int mode = ds.mode, s = ds.tile;
        if (mode == 0 || mode == 1) {
            float w[kW];
            {
                Raw r;
                if (s >= 0) load_sub(s, r);
                else { r.t = ninf_raw<In>(); r.z = r.t; }
                sub_weights(r, w);
            }
            const int j0 = e0 + max(s, 0) * kSub + lane * kW;
            bool done = false;
            if (mode == 0) {
                // exact scan of the sub-tile across the warp, then within the lane
                unsigned long long mine = 0ull;
#pragma unroll
                for (int e = 0; e < kW; ++e) mine += fix_of(w[e]);
                const unsigned long long excl = ds.base + warp_incl_scan_u64(mine) - mine;
                const bool hit = excl <= tau && excl + mine > tau;
                if (hit) {
                    unsigned long long C = excl;
                    for (int e = 0; e < kW; ++e) {
                        const unsigned long long Cprev = C;
                        C += fix_of(w[e]);
                        if (C > tau) {
                            out[a] = j0 + e;
                            if (p.diag_gap)
                                p.diag_gap[b] = fminf(fix_to_float(C - tau), fix_to_float(tau - Cprev)) / fix_to_float(W);
                            break;
                        }
                    }
                }
                done = __any_sync(0xffffffffu, hit);
            }
            if (!done) {
                // largest j of the sub-tile with w_j > 0 (rounding fallback)
                int best = -1;
                float wbest = 0.f;
#pragma unroll
                for (int e = 0; e < kW; ++e)
                    if (w[e] > 0.f) { best = j0 + e; wbest = w[e]; }
                int jb = best;
                for (int o = 16; o > 0; o >>= 1) jb = max(jb, __shfl_xor_sync(0xffffffffu, jb, o));
                if (jb >= 0 && best == jb) {
                    out[a] = jb;
                    if (p.diag_gap) {
                        const float Wf = fix_to_float(W), tf = fix_to_float(tau);
                        p.diag_gap[b] = fminf(Wf - tf, tf - (Wf - wbest)) / Wf;
                    }
                } else if (jb < 0 && lane == 0) {
                    out[a] = e0;  // no positive entry found: cannot happen when W > 0
                }
            }
        } else {
            // no residual mass at all: argmax of p_a over the whole row
            MaxIdx acc{kNegInf, INT_MAX};
            for (int j = lane; j < V; j += 32) {
                const float t = E::load(trow_g + j);
                if (t > acc.m) { acc.m = t; acc.i = j; }
            }
            acc = warp_reduce(acc, [](MaxIdx x, MaxIdx y) { return merge_mi(x, y); });
            if (lane == 0) {
                out[a] = (acc.i == INT_MAX) ? 0 : acc.i;
                if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000);
            }
        }
    }
    return true;
}

template <typename In, bool kVecPath>
__global__ void __launch_bounds__(kFinThreads) verify_finalize_kernel(FinParams p) {
    __shared__ SeqSmem sh;
    extern __shared__ float s_sub[];  // one residual sum per sub-tile of this CTA's span
    // residual masses in exact 64-bit fixed point (fix_of): a dependent fp64 add is slow here
    __shared__ DrawSmem ds;

    const int rank = (p.csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const int b = blockIdx.x / p.csize;
    const int k = p.k, V = p.V;
    const In* draft = static_cast<const In*>(p.draft);
    const In* target = static_cast<const In*>(p.target);

    const int bad = seq_prologue<In, kFinThreads>(p, b, sh);
    if (bad) {  // uniform over the cluster, before any distributed shared memory access
        if (rank == 0) seq_write_bad<kFinThreads>(p, b);
        return;
    }
    seq_accept(p, b, sh, rank == 0 && p.diag_margin);
    const int a = sh.a;
    if (rank == 0) seq_write_outputs<kFinThreads>(p, b, sh, a);

    // ---- extra token: inverse CDF of w = max(0, p_a - q_a) (a < k) or p_k (a == k)
    {
        const bool bonus = (a == k);
        const In* trow = target + (size_t(b) * (k + 1) + a) * V;
        const In* zrow = draft + (size_t(b) * k + (bonus ? 0 : a)) * V;
        const int e0 = rank * p.span;
        const int n = max(0, min(p.span, V - e0));
        residual_draw<In, kVecPath, kFinThreads, false>(p, b, a, sh, rank, e0, n, trow, zrow, 0, trow, s_sub, ds);
    }
    if (p.csize > 1) cluster_wait();  // keep this CTA's shared memory alive for its peers
}

// ------------------------------------------------------------------ one launch for small batches
// At serving batch sizes the two launches above cost more in latency than in
// bytes.  One thread-block cluster per sequence does both passes (T > 0): each
// CTA bulk-copies its vocabulary span of all 2k+1 rows into shared memory,
// computes the span's statistics of every row from there, merges them across
// the cluster, runs the accept tests, and draws the extra token from the staged
// rows (residual_draw) without reading them again.  The CTAs exchange the span
// statistics and the residual totals by pushing them with st.async into every
// peer's shared memory, each CTA waiting on its own barrier: no cluster barrier
// after the start, no fence, and nothing read from a peer.  It runs only when
// its grid fits in one wave (fused_shape).  At B = 32, k = 5, V = 32000 it measured 23.9 us
// in the bench step against 27.1 us for the two launches (512 threads; 256 threads
// 26.7 us; 16-CTA clusters 38 us).  The greedy pass (T = 0) keeps its two
// launches: one launch over the k+1 target rows measured 11.2 against 10.3 us.
constexpr int kFuseThreads = 512;
constexpr int kFuseCluster = 8;          // CTAs per sequence (above 8 needs the non-portable opt-in)
constexpr int kFuseParts = 4;           // warp items per row for the span statistics
constexpr int kFuseMaxB = 64;           // at most this many sequences, and the grid in one wave
constexpr size_t kFuseMaxSmem = 200 * 1024;  // staged rows + sub-tile sums per CTA
constexpr uint64_t kFuseWaitNs = 1000000000ull;  // bound on the wait for the staged rows

// Byte offset of the one-launch kernel's receive slots in its dynamic shared
// memory: after the staged rows and the sub-tile sums, 16-byte aligned.
__host__ __device__ inline size_t fused_recv_offset(int nrows, int span, size_t es) {
    return (size_t(nrows) * span * es + size_t(span / 128 + 1) * sizeof(float) + 15) / 16 * 16;
}

// Rows of sequence b staged by this CTA: local row r <= k is target row r, r > k
// draft row r-k-1; each holds entries [e0, e0 + n) at r * span.
template <typename In>
__device__ __forceinline__ const In* fused_src(const FinParams& p, int b, int r, int e0) {
    const In* draft = static_cast<const In*>(p.draft);
    const In* target = static_cast<const In*>(p.target);
    return (r <= p.k) ? target + (size_t(b) * (p.k + 1) + r) * p.V + e0
                      : draft + (size_t(b) * p.k + (r - p.k - 1)) * p.V + e0;
}

template <typename In>
__global__ void __launch_bounds__(kFuseThreads) verify_fused_kernel(FinParams p) {
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    constexpr int kWarps = kFuseThreads / 32;
    constexpr int kMaxRows = 2 * OSD_VERIFY_MAX_K + 1;
    extern __shared__ __align__(128) unsigned char fsm[];
    __shared__ __align__(8) uint64_t rbar[kMaxRows];  // one staging barrier per row
    __shared__ SeqSmem sh;
    __shared__ DrawSmem ds;
    __shared__ MaxSum part_ms[kMaxRows * kFuseParts];
    __shared__ __align__(8) uint64_t sbar;  // the cluster's span statistics have arrived
    __shared__ int s_any_tmo;  // a staging copy (or a wait for the peers) gave up in the cluster

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int csize = p.csize;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const int b = blockIdx.x / csize;
    const int k = p.k, V = p.V;
    const int nrows = 2 * k + 1;
    const int e0 = rank * p.span;
    const int n = min(p.span, V - e0);
    In* rows = reinterpret_cast<In*>(fsm);
    float* s_sub = reinterpret_cast<float*>(fsm + size_t(nrows) * p.span * sizeof(In));
    // [csize][nrows]: CTA c's span statistics of every row, pushed by CTA c
    MaxSum* recv_ms = reinterpret_cast<MaxSum*>(fsm + fused_recv_offset(nrows, p.span, sizeof(In)));
    const uint32_t bytes = static_cast<uint32_t>(n * sizeof(In));  // a multiple of 16 on this path

    // ---- stage every row's span (all the copies in flight at once, a barrier per row,
    // so that a row's statistics start as soon as it has landed)
    if (tid == 0) {
        for (int r = 0; r < nrows; ++r) mbar_init_only(&rbar[r], 1);
        mbar_init_only(&sbar, 1);
        mbar_init_only(&ds.tbar, 1);
        fence_mbarrier_init();
        for (int r = 0; r < nrows; ++r) {
            mbar_arrive_expect_tx(&rbar[r], bytes);
            bulk_g2s(rows + size_t(r) * p.span, fused_src<In>(p, b, r, e0), bytes, &rbar[r]);
        }
    }
    // meanwhile the draft tokens, the two logits each accept test needs, and the uniforms
    int bad = 0;
    const int32_t* y = p.tokens + size_t(b) * k;
    if (warp == kWarps - 1) {
        for (int i = lane; i < k; i += 32) {
            const int t = y[i];
            sh.y[i] = t;
            if (t < 0 || t >= V) {
                bad = 1;
            } else {
                sh.zy[i] = E::load(static_cast<const In*>(p.draft) + (size_t(b) * k + i) * V + t);
                sh.ty[i] = E::load(static_cast<const In*>(p.target) + (size_t(b) * (k + 1) + i) * V + t);
            }
        }
    }
    if (warp == kWarps - 2)
        for (int i = lane; i <= k; i += 32) sh.u[i] = p.uniforms[size_t(b) * (k + 1) + i];
    __syncthreads();  // the barriers are initialised before anyone waits on them
    // ... and before any peer pushes to them: arrive now, wait before the first push
    if (csize > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    bad = __syncthreads_or(bad);
    // every row's copy has landed (or its wait gave up) before this CTA leaves
    auto wait_all = [&]() {
        int t = 0;
        for (int r = 0; r < nrows; ++r) t |= mbar_wait_bounded(&rbar[r], 0, kFuseWaitNs) ? 0 : 1;
        return t;
    };
    if (bad) {  // uniform over the cluster, before any push to a peer
        wait_all();
        if (rank == 0) seq_write_bad<kFuseThreads>(p, b);
        return;
    }

    // ---- span statistics of every row: warp items (row, part), each its row's
    // maximum first, then the sum of 2^((x - m) c) against it; then per row over the parts
    const int nch = n / kVec;
    const float ch = p.c_hi, cl = p.c_lo;
    int timed_out = 0;
    for (int it = warp; it < nrows * kFuseParts; it += kWarps) {
        const int r = it / kFuseParts, part = it - r * kFuseParts;
        if (!mbar_wait_bounded(&rbar[r], 0, kFuseWaitNs)) timed_out = 1;
        const In* row = rows + size_t(r) * p.span;
        const int c0 = nch * part / kFuseParts, c1 = nch * (part + 1) / kFuseParts;
        float m = kNegInf;
        for (int c = c0 + lane; c < c1; c += 32) m = fmaxf(m, E::max_raw(lds_v4(row + c * kVec)));
        for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
        float2 s2 = f2(0.f);
        if (m != kNegInf) {
            for (int c = c0 + lane; c < c1; c += 32) {
                float x[kVec];
                E::unpack(lds_v4(row + c * kVec), x);
#pragma unroll
                for (int e = 0; e < kVec; e += 2) {
                    const float2 d = sub2(make_float2(x[e], x[e + 1]), f2(m));
                    const float2 g = fma2(d, f2(ch), mul2(d, f2(cl)));
                    s2 = add2(s2, make_float2(ex2(g.x), ex2(g.y)));
                }
            }
        }
        float s = s2.x + s2.y;
        for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
        if (lane == 0) part_ms[it] = MaxSum{m, s};
    }
    const int tmo = __syncthreads_or(timed_out);
    if (tmo) wait_all();  // a copy that gave up gets a last chance to land
    // ---- the cluster's spans: thread r < nrows merges its row's parts and pushes the
    // result (a negative sum flags a copy that gave up) into slot `rank` of every CTA;
    // every CTA then merges the csize slots of each row in rank order (lane c <- CTA c)
    if (tid < nrows) {
        MaxSum acc = part_ms[tid * kFuseParts];
        for (int q = 1; q < kFuseParts; ++q) acc = merge_ms(acc, part_ms[tid * kFuseParts + q], ch, cl);
        if (tmo) acc.s = -1.f;
        if (csize > 1) {
            asm volatile("barrier.cluster.wait.acquire;" ::: "memory");  // the peers' barriers are ready
            for (int d = 0; d < csize; ++d)
                st_async_v2(map_rank(&recv_ms[rank * nrows + tid], static_cast<uint32_t>(d)), make_float2(acc.m, acc.s),
                            map_rank(&sbar, static_cast<uint32_t>(d)));
        } else {
            recv_ms[tid] = acc;
        }
    }
    if (csize > 1) {
        if (tid >= nrows) asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
        if (tid == 0) mbar_arrive_expect_tx(&sbar, static_cast<uint32_t>(csize * nrows) * 8u);
    }
    bool got = true;
    if (csize > 1) got = mbar_wait_cluster_bounded(&sbar, 0, kFuseWaitNs); else __syncthreads();
    got = __syncthreads_and(got);
    int any_tmo = got ? 0 : 1;
    for (int r = warp; r < nrows; r += kWarps) {
        MaxSum o{kNegInf, 0.f};
        if (lane < csize && got) o = recv_ms[lane * nrows + r];
        if (__any_sync(0xffffffffu, o.s < 0.f)) any_tmo = 1;
        o.s = fmaxf(o.s, 0.f);
        o = warp_reduce(o, [ch, cl](MaxSum x, MaxSum z) { return merge_ms(x, z, ch, cl); });
        if (lane == 0) { sh.m[r] = o.m; sh.s[r] = o.s; }
    }
    any_tmo = __syncthreads_or(any_tmo);
    if (any_tmo) {  // the GPU did not deliver a row in time: the sequence is reported as bad
        if (rank == 0) seq_write_bad<kFuseThreads>(p, b);
        return;
    }

    seq_accept(p, b, sh, rank == 0 && p.diag_margin);
    const int a = sh.a;
    if (rank == 0) seq_write_outputs<kFuseThreads>(p, b, sh, a);
    // ---- extra token from the staged rows at position a
    const bool bonus = (a == k);
    const In* trow_s = rows + size_t(a) * p.span;
    const In* zrow_s = bonus ? trow_s : rows + size_t(k + 1 + a) * p.span;
    const In* trow_g = static_cast<const In*>(p.target) + (size_t(b) * (k + 1) + a) * V;
    // (a peer whose pushed total did not arrive in time reports the sequence as bad)
    if (!residual_draw<In, true, kFuseThreads, true, true>(p, b, a, sh, rank, e0, n, trow_s, zrow_s, e0, trow_g,
                                                        s_sub, ds))
        seq_write_bad<kFuseThreads>(p, b);
}

// ------------------------------------------------------------------ host
static int verify_slice_len(int B, int k) { return stats_slice_len((long long)B * (2 * k + 1)); }

static int verify_slices(int B, int k, int V) {
    const int len = verify_slice_len(B, k);
    return (V + len - 1) / len;
}

static size_t round256(size_t x) { return (x + 255) / 256 * 256; }

// CTAs per sequence: up to 8 for few sequences (short spans, low latency); 4 past
// 128 sequences, where 8 would leave more clusters than fit on the GPU at once and
// the second wave would wait out the first one's latency phases.  A span must fit
// in kFinMaxSub sub-tiles of `sub` entries: the element-wise path (32-entry
// sub-tiles) takes 8 CTAs at any B once V passes 4 * 8192 * 32 = 2^20.
static void finalize_shape(int B, int V, int sub, int* csize, int* span) {
    int cmax = (B > 128) ? kFinMaxCluster / 2 : kFinMaxCluster;
    const long long per_cta = (long long)kFinMaxSub * sub;
    if ((long long)cmax * per_cta < V) cmax = kFinMaxCluster;
    int c = (V + 4095) / 4096;
    c = c < 1 ? 1 : (c > cmax ? cmax : c);
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    *csize = c;
    *span = s;
}

// Resident CTAs an SM of the one-launch kernel with `smem` bytes of dynamic shared
// memory, or 0 when a query fails.  The opt-in for that much shared memory is set
// here first; both are kept per device for the last size asked, so repeated calls
// (and calls under stream capture) make no runtime query.
template <typename In>
static int fused_ctas_per_sm(size_t smem) {
    auto kern = verify_fused_kernel<In>;
    static std::mutex mu;
    static size_t allowed[64] = {};
    static size_t last_smem[64] = {};
    static int last_occ[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (last_smem[dev] == smem && last_occ[dev] > 0) return last_occ[dev];
    if (allowed[dev] < smem) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
            cudaSuccess)
            return 0;
        allowed[dev] = smem;
    }
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kFuseThreads, smem) != cudaSuccess) return 0;
    last_smem[dev] = smem;
    last_occ[dev] = occ;
    return occ;
}

// One launch for small batches: the cluster shape and shared memory, or false
// when the rows are not 16-byte aligned, the staged rows do not fit, or the
// grid would not fit in one wave (the two-launch path then runs).
template <typename In>
static bool fused_shape(int B, int k, int V, bool greedy, const void* draft, const void* target, int* csize,
                        int* span, size_t* smem) {
    if (greedy || B > kFuseMaxB) return false;
    if (!aligned_to(target, 16) || !aligned_to(draft, 16) || ((size_t)V * sizeof(In)) % 16 != 0) return false;
    int c = kFuseCluster;
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    const int nrows = 2 * k + 1;
    const size_t bytes = fused_recv_offset(nrows, s, sizeof(In)) + size_t(c) * nrows * sizeof(MaxSum);
    if (bytes > kFuseMaxSmem) return false;
    // only in one wave: at B = 32, k = 5, V = 32000 (two CTAs an SM) one launch took
    // 22.2 us against 23.2 us for two; from B = 48 on, past one wave, 34 against 26 us
    const long long ctas = (long long)B * c;
    if (ctas > (long long)device_sms() * fused_ctas_per_sm<In>(bytes)) return false;
    *csize = c;
    *span = s;
    *smem = bytes;
    return true;
}
// The one-launch kernel (fused_shape has set its shared-memory opt-in).
template <typename In>
static cudaError_t launch_fused(const FinParams& fp, size_t smem, cudaStream_t stream) {
    auto kern = verify_fused_kernel<In>;
    if (kFuseCluster > 8) {
        static std::atomic<int> nonportable[64];
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= 64) return cudaErrorInvalidValue;
        if (!nonportable[dev].load(std::memory_order_relaxed)) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess) return e;
            nonportable[dev].store(1, std::memory_order_relaxed);
        }
    }
    return launch(kern, dim3(unsigned(fp.B) * unsigned(fp.csize)), dim3(kFuseThreads), smem, stream, fp.csize, fp);
}

template <typename In>
static osd_status launch_verify(const void* draft, const void* target, int B, int k, int V,
                                const int32_t* tokens, const float* uniforms, float T,
                                int32_t* accepted, int32_t* out_tokens, uint8_t* mask,
                                float* diag_margin, float* diag_gap, RowStat* stats,
                                cudaStream_t stream) {
    const bool greedy = (T == 0.f);
    {
        int fc = 1, fspan = V;
        size_t fsmem = 0;
        if (fused_shape<In>(B, k, V, greedy, draft, target, &fc, &fspan, &fsmem)) {
            FinParams fp = {};
            fp.draft = draft; fp.target = target; fp.B = B; fp.k = k; fp.V = V;
            fp.tokens = tokens; fp.uniforms = uniforms; fp.T = T;
            split_scale(T, &fp.c_hi, &fp.c_lo);
            fp.accepted = accepted; fp.out_tokens = out_tokens; fp.mask = mask;
            fp.diag_margin = diag_margin; fp.diag_gap = diag_gap;
            fp.csize = fc;
            fp.span = fspan;
            return from_cuda(launch_fused<In>(fp, fsmem, stream));
        }
    }
    const int slice_len = verify_slice_len(B, k);
    const int n_slices = verify_slices(B, k, V);
    const long long n_draft_rows = greedy ? 0 : (long long)B * k;
    const long long rows = n_draft_rows + (long long)B * (k + 1);
    float c_hi = 0.f, c_lo = 0.f;
    if (!greedy) split_scale(T, &c_hi, &c_lo);

    const long long grid1 = rows * n_slices;
    if (grid1 > INT_MAX) return OSD_ERR_UNSUPPORTED;
    cudaError_t e;
    if (greedy)
        e = launch(row_stats_kernel<In, true>, dim3(unsigned(grid1)), dim3(kStatThreads), 0, stream, 1,
                   static_cast<const In*>(draft), static_cast<const In*>(target), n_draft_rows, V,
                   slice_len, n_slices, c_hi, c_lo, stats);
    else
        e = launch(row_stats_kernel<In, false>, dim3(unsigned(grid1)), dim3(kStatThreads), 0, stream, 1,
                   static_cast<const In*>(draft), static_cast<const In*>(target), n_draft_rows, V,
                   slice_len, n_slices, c_hi, c_lo, stats);
    if (e != cudaSuccess) return OSD_ERR_CUDA;

    FinParams fp;
    fp.draft = draft; fp.target = target; fp.B = B; fp.k = k; fp.V = V;
    fp.tokens = tokens; fp.uniforms = uniforms; fp.T = T; fp.c_hi = c_hi; fp.c_lo = c_lo;
    fp.stats = stats; fp.n_slices = n_slices; fp.n_draft_rows = n_draft_rows;
    fp.accepted = accepted; fp.out_tokens = out_tokens; fp.mask = mask;
    fp.diag_margin = diag_margin; fp.diag_gap = diag_gap;
    if (greedy) {
        fp.csize = 1;
        fp.span = V;
        const dim3 grid_g(unsigned((B + kGreedyWarps - 1) / kGreedyWarps));
        return from_cuda(launch_ex(true, verify_greedy_kernel, grid_g, dim3(kGreedyWarps * 32), 0, stream, 1, fp));
    }
    const bool vec = aligned_to(draft, 16) && aligned_to(target, 16) && ((size_t)V * sizeof(In)) % 16 == 0;
    const int sub = 32 * (vec ? Elem<In>::kVec : 1);
    int csize = 1, span = V;
    finalize_shape(B, V, sub, &csize, &span);
    fp.csize = csize;
    fp.span = span;
    const dim3 grid2(unsigned(B) * unsigned(csize));
    const size_t smem2 = size_t((span + sub - 1) / sub) * sizeof(float);
    if (smem2 > size_t(kFinMaxSub) * sizeof(float)) return OSD_ERR_UNSUPPORTED;
    if (vec)
        e = launch_ex(true, verify_finalize_kernel<In, true>, grid2, dim3(kFinThreads), smem2, stream, csize, fp);
    else
        e = launch_ex(true, verify_finalize_kernel<In, false>, grid2, dim3(kFinThreads), smem2, stream, csize, fp);
    return from_cuda(e);
}

}  // namespace osd

using osd::RowStat;

extern "C" osd_status osd_verify_workspace_size(int B, int k, int V, size_t* bytes) {
    if (!bytes || B < 0 || k < 1 || V < 1) return OSD_ERR_INVALID_ARG;
    if (k > OSD_VERIFY_MAX_K || V > OSD_VERIFY_MAX_V) return OSD_ERR_UNSUPPORTED;
    const size_t rows = size_t(B) * size_t(2 * k + 1);
    const size_t need = osd::round256(rows * size_t(osd::verify_slices(B, k, V)) * sizeof(RowStat));
    *bytes = need < 256 ? 256 : need;
    return OSD_OK;
}

extern "C" osd_status osd_verify(const void* draft_logits, const void* target_logits, osd_dtype dtype,
                                 int B, int k, int V, const int32_t* draft_tokens, const float* uniforms,
                                 float temperature, int32_t* accepted, int32_t* out_tokens,
                                 uint8_t* mismatch_mask, float* diag_margin, float* diag_cdf_gap,
                                 void* workspace, size_t workspace_bytes, void* stream) {
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    size_t need = 0;
    const osd_status st = osd_verify_workspace_size(B, k, V, &need);
    if (st != OSD_OK) return st;
    if (!(temperature >= 0.f) || !std::isfinite(temperature)) return OSD_ERR_INVALID_ARG;
    if (B == 0) return OSD_OK;
    const bool greedy = (temperature == 0.f);
    const size_t es = osd::dtype_size(dtype);
    if (!target_logits || !draft_tokens || !accepted || !out_tokens || !mismatch_mask || !workspace)
        return OSD_ERR_INVALID_ARG;
    if (!greedy && (!draft_logits || !uniforms)) return OSD_ERR_INVALID_ARG;
    if (!osd::aligned_to(target_logits, es) || (draft_logits && !osd::aligned_to(draft_logits, es)) ||
        !osd::aligned_to(draft_tokens, 4) || (uniforms && !osd::aligned_to(uniforms, 4)) ||
        !osd::aligned_to(accepted, 4) || !osd::aligned_to(out_tokens, 4) ||
        (diag_margin && !osd::aligned_to(diag_margin, 4)) ||
        (diag_cdf_gap && !osd::aligned_to(diag_cdf_gap, 4)) || !osd::aligned_to(workspace, 16))
        return OSD_ERR_INVALID_ARG;
    if (workspace_bytes < need) return OSD_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == OSD_BF16)
        return osd::launch_verify<__nv_bfloat16>(draft_logits, target_logits, B, k, V, draft_tokens, uniforms,
                                                 temperature, accepted, out_tokens, mismatch_mask, diag_margin,
                                                 diag_cdf_gap, static_cast<RowStat*>(workspace), s);
    return osd::launch_verify<float>(draft_logits, target_logits, B, k, V, draft_tokens, uniforms, temperature,
                                     accepted, out_tokens, mismatch_mask, diag_margin, diag_cdf_gap,
                                     static_cast<RowStat*>(workspace), s);
}

// ------------------------------------------------------------------ no-allocation variant
// Some callers cannot call cudaMalloc while they serve: engines that reserve all
// free device memory for their KV cache at start-up and hand out nothing
// afterwards, plugins that run inside such an engine without an allocator of
// their own, and latency-critical loops where cudaMalloc (which may synchronise
// the device) would stall every other stream.  osd_verify_noalloc serves them
// with a fixed workspace that lives in the library itself: a file-scope device
// array, one copy per GPU that loads the library, held until the process exits.
namespace {
constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB
constexpr int kNoAllocMaxDevices = 64;
__device__ __align__(256) unsigned char g_verify_scratch[kNoAllocScratchBytes];

// The device address of the array, per device, with the ID of the context it
// was looked up in: a new context (cudaDeviceReset, or a context the caller
// made current) loads the module again, possibly elsewhere, so the address is
// looked up again whenever the current context's ID differs.
struct ScratchSlot {
    unsigned long long ctx_id;
    void* addr;
};
std::mutex g_scratch_mu;
ScratchSlot g_scratch[kNoAllocMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// ID of the context current on the calling thread; false when there is none yet
// (the runtime makes the primary context current on its first device call) or
// the driver does not provide the query.
bool current_context_id(unsigned long long* id) {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<CtxGetCurrentFn>(f);
        f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<CtxGetIdFn>(f);
    });
    if (!get_current || !get_id) return false;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
    return get_id(ctx, id) == CUDA_SUCCESS;
}
}  // namespace

extern "C" osd_status osd_verify_noalloc(const void* draft_logits, const void* target_logits,
                                         osd_dtype dtype, int B, int k, int V,
                                         const int32_t* draft_tokens, const float* uniforms,
                                         float temperature, int32_t* accepted, int32_t* out_tokens,
                                         uint8_t* mismatch_mask, float* diag_margin, float* diag_cdf_gap,
                                         void* stream) {
    size_t need = 0;
    const osd_status st = osd_verify_workspace_size(B, k, V, &need);
    if (st != OSD_OK) return st;
    if (need > kNoAllocScratchBytes) return OSD_ERR_UNSUPPORTED;  // beyond the static scratch
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return OSD_ERR_CUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return OSD_ERR_UNSUPPORTED;
    void* scratch = nullptr;
    {
        // Set-up once per device and context, with that device current: the
        // host-side name of the array is not a device address, so ask the runtime.
        std::lock_guard<std::mutex> lock(g_scratch_mu);
        unsigned long long id = 0;
        const bool have_id = current_context_id(&id);
        ScratchSlot& slot = g_scratch[dev];
        if (!have_id || !slot.addr || slot.ctx_id != id) {
            void* addr = nullptr;
            if (cudaGetSymbolAddress(&addr, g_verify_scratch) != cudaSuccess || !addr) return OSD_ERR_CUDA;
            // the lookup made a context current if none was: key the address on it;
            // without a context ID the address is not cached and is looked up every call
            const bool keyed = have_id || current_context_id(&id);
            slot.addr = keyed ? addr : nullptr;
            slot.ctx_id = keyed ? id : 0ull;
            scratch = addr;
        } else {
            scratch = slot.addr;
        }
    }
    // The statistics pass writes every workspace entry before the finalize pass
    // reads it, so nothing in the shared array needs clearing between calls.
    return osd_verify(draft_logits, target_logits, dtype, B, k, V, draft_tokens, uniforms, temperature,
                      accepted, out_tokens, mismatch_mask, diag_margin, diag_cdf_gap, scratch,
                      kNoAllocScratchBytes, stream);
}
