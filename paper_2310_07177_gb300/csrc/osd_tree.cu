// osd_tree.cu -- multi-candidate verification over a token tree (the tree-style
// speculative decoding the paper runs OSD on with Medusa heads: several
// candidates per position) on sm_103a.
//
// Two launches on the caller's stream:
//
//   row_stats_kernel   (osd_rowstats.cuh) the max and sum of 2^((x - max) c) of
//                      every vocabulary slice of every node's draft and target
//                      row (the argmax at T = 0): the one pass over all logits.
//   tree_walk_kernel   one thread-block cluster per sequence walks the tree from
//                      the root.  It merges every node's slice statistics up
//                      front; at a node it tests the children in index order
//                      with the accept rule of Appendix A.1 against the current
//                      residual.  After j rejections the residual is
//                      norm(max(0, p - s_j q)) with s_0 = 0 and s_{j+1} = s_j + N_j,
//                      N_j = sum max(0, p - s_j q), so child y passes iff
//                      u < max(0, p(y)/q(y) - s_j) / N_j.  Every rejection costs one
//                      cluster-wide pass that recomputes N_{j+1}; an acceptance
//                      moves the walk to the child.  When no child passes, the
//                      extra token is drawn from max(0, p - s q) by inverse CDF
//                      from the sub-tile sums of the last pass, as the verifier's
//                      finalize kernel draws its residual token (masses summed in
//                      exact 64-bit fixed point).
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdint>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"
#include "osd_rowstats.cuh"

namespace osd {

constexpr int kTreeThreads = 128;
constexpr int kTreeWarps = kTreeThreads / 32;
constexpr int kTreeMaxCluster = 8;
constexpr int kTreeMaxSub = 8192;  // sub-tiles of one CTA's vocabulary span
constexpr int kTreeUnroll = 4;     // sub-tiles of loads in flight per warp in a mass pass

// Children lists of the static tree: first child and next sibling, increasing
// index; and each node's parent (-1 at the root).
struct TreeTopo {
    int8_t first_child[OSD_TREE_MAX_NODES];
    int8_t next_sibling[OSD_TREE_MAX_NODES];
    int8_t parent[OSD_TREE_MAX_NODES];
};

struct TreeParams {
    const void* draft;
    const void* target;
    int n, V;  // nodes per tree, vocabulary
    const int32_t* tokens;
    const float* uniforms;
    float T, c_hi, c_lo;
    const RowStat* stats;
    int n_slices;
    long long n_draft_rows;  // rows of draft statistics ahead of the target rows (0 at T = 0)
    int32_t* accepted;
    int32_t* path;
    int32_t* out_tokens;
    int32_t* last_node;
    float* diag_margin;
    float* diag_gap;
    int csize, span;
    TreeTopo topo;
};

template <typename In, bool kVecPath>
__global__ void __launch_bounds__(kTreeThreads) tree_walk_kernel(TreeParams p) {
    using E = Elem<In>;
    constexpr int kW = kVecPath ? E::kVec : 1;  // entries per lane per sub-tile
    constexpr int kSub = 32 * kW;
    extern __shared__ float s_sub[];           // mass of every sub-tile of this CTA's span (last pass)
    // masses in exact 64-bit fixed point (fix_of): a dependent fp64 add is slow here
    __shared__ unsigned long long s_span_total;            // read by the other CTAs of the cluster
    __shared__ unsigned long long s_cta_incl[kTreeMaxCluster];  // inclusive prefix of the CTA masses, rank order
    __shared__ unsigned long long s_W;
    __shared__ int s_next, s_extra;
    // per node: merged statistics of its target (0) and draft (1) rows, or the target argmax at T = 0
    __shared__ float s_nm[2][OSD_TREE_MAX_NODES], s_ns[2][OSD_TREE_MAX_NODES];
    __shared__ int s_nidx[OSD_TREE_MAX_NODES];
    // per child c: its token's logits in the draft and target rows of its parent, and its uniform
    __shared__ float s_zy[OSD_TREE_MAX_NODES], s_ty[OSD_TREE_MAX_NODES], s_u[OSD_TREE_MAX_NODES];
    __shared__ double s_nratio[OSD_TREE_MAX_NODES];  // per node with children: E_z / E_t

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int csize = p.csize;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const int b = blockIdx.x / csize;
    const int n = p.n, V = p.V;
    const bool greedy = (p.T == 0.f);
    const int32_t* y = p.tokens + size_t(b) * n;
    const float* u = p.uniforms ? p.uniforms + size_t(b) * n : nullptr;
    int32_t* pth = p.path + size_t(b) * n;
    int32_t* out = p.out_tokens + size_t(b) * n;
    const float ch = p.c_hi, cl = p.c_lo;

    // Prologue, before the statistics are ready: check the tokens and gather the two
    // logits every child's accept test needs, all in one round of loads.
    int bad = 0;
    if (!greedy)
        for (int i = tid; i < n; i += kTreeThreads) s_u[i] = u[i];
    for (int i = 1 + tid; i < n; i += kTreeThreads) {
        const int yi = y[i];
        if (yi < 0 || yi >= V) {
            bad = 1;
        } else if (!greedy) {
            const size_t prow = size_t(b) * n + p.topo.parent[i];
            s_zy[i] = E::load(static_cast<const In*>(p.draft) + prow * V + yi);
            s_ty[i] = E::load(static_cast<const In*>(p.target) + prow * V + yi);
        }
    }
    bad = __syncthreads_or(bad);
    if (rank == 0) {
        for (int i = tid; i < n; i += kTreeThreads) {
            pth[i] = -1;
            out[i] = -1;
            if (p.diag_margin) p.diag_margin[size_t(b) * n + i] = __int_as_float(0x7fc00000);
        }
        if (tid == 0 && p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000);
        if (tid == 0 && bad) {
            p.accepted[b] = -1;
            p.last_node[b] = -1;
        }
    }
    if (bad) return;  // uniform over the cluster, before any shared-memory exchange
    __syncthreads();  // the initialisation above lands before the walk writes its entries
    grid_dependency_wait();  // the row statistics are complete from here on

    // Every node's row statistics, merged from their slices up front (one thread per
    // node and row, all loads in one round) instead of one dependent round per node
    // on the walk.  Draft rows matter only where children are tested.
    for (int t = tid; t < 2 * n; t += kTreeThreads) {
        const int nd = t >> 1, which = t & 1;
        if (greedy) {
            if (which == 0) {
                const RowStat* st = p.stats + (size_t(b) * n + nd) * p.n_slices;
                MaxIdx acc{kNegInf, INT_MAX};
#pragma unroll 4
                for (int sl = 0; sl < p.n_slices; ++sl) acc = merge_mi(acc, MaxIdx{st[sl].m, st[sl].idx});
                s_nidx[nd] = (acc.i == INT_MAX) ? 0 : acc.i;
            }
        } else if (which == 0 || p.topo.first_child[nd] >= 0) {
            const RowStat* st = p.stats + ((which == 0 ? p.n_draft_rows : 0) + size_t(b) * n + nd) * p.n_slices;
            MaxSum acc{kNegInf, 0.f};
#pragma unroll 4
            for (int sl = 0; sl < p.n_slices; ++sl) acc = merge_ms(acc, MaxSum{st[sl].m, st[sl].s}, ch, cl);
            s_nm[which][nd] = acc.m;
            s_ns[which][nd] = acc.s;
        }
    }
    __syncthreads();
    // the sum ratio of each accept test's p/q, once per node (fp64 divisions are slow here)
    if (!greedy) {
        for (int nd = tid; nd < n; nd += kTreeThreads)
            if (p.topo.first_child[nd] >= 0) s_nratio[nd] = double(s_ns[1][nd]) / double(s_ns[0][nd]);
        __syncthreads();
    }
    float cur_mt = 0.f, cur_st = 1.f, cur_mz = 0.f, cur_sz = 1.f;  // the current node's statistics

    const int e0 = rank * p.span;
    const int cnt = max(0, min(p.span, V - e0));
    const int nsub = (cnt + kSub - 1) / kSub;
    bool pending = false;  // a cluster barrier phase is open: peers may still read s_span_total

    // weights w = max(0, p - s q) of kW entries of one lane (q only when s > 0)
    struct Raw {
        uint4 t, z;
    };
    auto load_sub = [&](const In* trow, const In* zrow, bool use_q, int sb, Raw& r) {
        const int j0 = e0 + sb * kSub + lane * kW;
        const int m = min(kW, e0 + cnt - j0);
        if (kVecPath && m == kW) {
            r.t = ldg_stream(trow + j0);
            r.z = use_q ? ldg_stream(zrow + j0) : r.t;
        } else {
            float tv[kW], zv[kW];
#pragma unroll
            for (int e = 0; e < kW; ++e) {
                tv[e] = (e < m) ? E::load(trow + j0 + e) : kNegInf;
                zv[e] = (e < m && use_q) ? E::load(zrow + j0 + e) : kNegInf;
            }
            r.t = pack_raw<In, kW>(tv);
            r.z = pack_raw<In, kW>(zv);
        }
    };
    auto weights = [&](const Raw& r, bool use_q, float s, float* w) {
        const float mt = cur_mt, inv_st = 1.0f / cur_st;
        float tv[kW], zv[kW];
        unpack_raw<In, kW>(r.t, tv);
        unpack_raw<In, kW>(r.z, zv);
        const float mz = cur_mz, inv_sz = use_q ? 1.0f / cur_sz : 0.f;
#pragma unroll
        for (int e = 0; e < kW; ++e) {
            const float pj = ex2(mul_c(tv[e] - mt, ch, cl)) * inv_st;
            if (use_q) {
                const float qj = ex2(mul_c(zv[e] - mz, ch, cl)) * inv_sz;
                w[e] = fmaxf(fmaf(-s, qj, pj), 0.f);
            } else {
                w[e] = pj;
            }
        }
    };
    // One cluster-wide pass: the mass of every sub-tile of w = max(0, p - s q) into s_sub,
    // the CTA masses' inclusive prefix into s_cta_incl, and the row's mass W (returned,
    // fixed point).
    auto mass_pass = [&](const In* trow, const In* zrow, bool use_q, float s) -> unsigned long long {
        if (pending) cluster_wait();  // every peer has read the previous pass's total
        for (int sb0 = warp; sb0 < nsub; sb0 += kTreeWarps * kTreeUnroll) {
            Raw r[kTreeUnroll];  // the loads of kTreeUnroll sub-tiles go out together
#pragma unroll
            for (int u2 = 0; u2 < kTreeUnroll; ++u2)
                if (sb0 + u2 * kTreeWarps < nsub) load_sub(trow, zrow, use_q, sb0 + u2 * kTreeWarps, r[u2]);
#pragma unroll
            for (int u2 = 0; u2 < kTreeUnroll; ++u2) {
                const int sb = sb0 + u2 * kTreeWarps;
                if (sb < nsub) {
                    float w[kW];
                    weights(r[u2], use_q, s, w);
                    float sum = 0.f;
#pragma unroll
                    for (int e = 0; e < kW; ++e) sum += w[e];
                    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
                    if (lane == 0) s_sub[sb] = sum;
                }
            }
        }
        __syncthreads();
        if (warp == 0) {
            unsigned long long part = 0ull;
            for (int sb = lane; sb < nsub; sb += 32) part += fix_of(s_sub[sb]);
            part = warp_sum_u64(part);
            if (lane == 0) s_span_total = part;
        }
        if (csize > 1) cluster_sync_publish(tid == 0); else __syncthreads();
        if (warp == 0) {
            unsigned long long tot = 0ull;
            if (lane < csize) tot = (lane == rank) ? s_span_total : ld_dsmem_u64(map_rank(&s_span_total, lane));
            const unsigned long long incl = warp_incl_scan_u64(tot);
            if (lane < csize) s_cta_incl[lane] = incl;
            if (lane == 31) s_W = incl;
        }
        __syncthreads();
        if (csize > 1) {
            cluster_arrive_relaxed();  // done reading the peers' totals
            pending = true;
        }
        return s_W;
    };

    int node = 0, depth = 0;
    for (;;) {
        const In* trow = static_cast<const In*>(p.target) + (size_t(b) * n + node) * V;
        const In* zrow = static_cast<const In*>(p.draft) + (size_t(b) * n + node) * V;
        const bool has_child = p.topo.first_child[node] >= 0;
        const bool need_q = !greedy && has_child;
        cur_mt = s_nm[0][node];
        cur_st = s_ns[0][node];
        if (need_q) {
            cur_mz = s_nm[1][node];
            cur_sz = s_ns[1][node];
        }

        int next = -1;
        if (greedy) {
            const int best = s_nidx[node];
            for (int c = p.topo.first_child[node]; c >= 0; c = p.topo.next_sibling[c])
                if (y[c] == best) { next = c; break; }
            if (next < 0) {
                if (tid == 0) s_extra = best;
                break;
            }
        } else {
            float s = 0.f;  // residual shift s_j
            double N = 1.0;  // residual mass N_j (p itself has mass 1)
            unsigned long long Nfix = 0ull;  // the same, in fixed point, after a mass pass
            bool passed = false;  // a mass pass of the current residual has run
            for (int c = p.topo.first_child[node]; c >= 0; c = p.topo.next_sibling[c]) {
                if (tid == 0) {
                    // p(y)/q(y) from the logit differences and the two sums, as the verifier
                    // forms it; the test u < max(0, p/q - s) / N is taken as u N < max(0, p/q - s)
                    const float zt = s_zy[c], tt = s_ty[c];
                    double rn;  // max(0, p(y)/q(y) - s_j)
                    if (zt == kNegInf) {
                        rn = (tt > kNegInf) ? INFINITY : 0.0;
                    } else {
                        const float D = (tt - cur_mt) - (zt - cur_mz);
                        const double rho = double(ex2(mul_c(D, ch, cl))) * s_nratio[node];
                        rn = fmax(rho - double(s), 0.0);
                    }
                    const float uc = s_u[c];
                    if (rank == 0 && p.diag_margin)  // |u - r|, a diagnostic: fp32 is enough
                        p.diag_margin[size_t(b) * n + c] = fabsf(uc - float(rn) / float(N));
                    s_next = (double(uc) * N < rn) ? c : -1;
                }
                __syncthreads();
                next = s_next;
                __syncthreads();  // s_next is rewritten by the next test
                if (next >= 0) break;
                s = static_cast<float>(double(s) + N);  // rejected: s_{j+1} = s_j + N_j
                Nfix = mass_pass(trow, zrow, true, s);
                N = __ull2double_rn(Nfix) * (1.0 / static_cast<double>(1ull << kFixBits));
                passed = true;
            }
            if (next < 0) {
                // ---- the extra token from w = max(0, p - s q) (p itself when nothing was rejected)
                const bool use_q = passed;
                const unsigned long long W = passed ? Nfix : mass_pass(trow, zrow, false, 0.f);
                const unsigned long long tau = fix_scale(s_u[0], W);  // floor(u W)
                int owner = -1, mode = 0;  // mode 0: inverse CDF, 1: largest positive entry, 2: argmax p
                unsigned long long base = 0ull;
                if (W > 0ull) {
                    for (int r = 0; r < csize; ++r)
                        if (s_cta_incl[r] > tau) { owner = r; break; }
                    if (owner >= 0) {
                        base = owner > 0 ? s_cta_incl[owner - 1] : 0ull;
                    } else {
                        mode = 1;
                        for (int r = csize - 1; r >= 0 && owner < 0; --r)
                            if (s_cta_incl[r] > (r > 0 ? s_cta_incl[r - 1] : 0ull)) owner = r;
                        if (owner < 0) owner = csize - 1;
                    }
                } else {
                    mode = 2;
                    owner = 0;
                }
                if (rank == owner && warp == 0) {
                    int pick = -1;
                    float gap = __int_as_float(0x7fc00000);
                    if (mode == 2) {  // no residual mass: argmax of p over the row, lowest index
                        MaxIdx acc{kNegInf, INT_MAX};
                        for (int j = lane; j < V; j += 32) {
                            const float t = E::load(trow + j);
                            if (t > acc.m) { acc.m = t; acc.i = j; }
                        }
                        acc = warp_reduce(acc, [](MaxIdx x, MaxIdx z) { return merge_mi(x, z); });
                        pick = (acc.i == INT_MAX) ? 0 : acc.i;
                    } else {
                        // the sub-tile: lane l owns the run [s_lo, s_hi) of sub-tiles
                        const int per = (nsub + 31) / 32;
                        const int s_lo = min(nsub, lane * per), s_hi = min(nsub, s_lo + per);
                        unsigned long long mine = 0ull;
                        for (int sb = s_lo; sb < s_hi; ++sb) mine += fix_of(s_sub[sb]);
                        const unsigned long long excl = base + warp_incl_scan_u64(mine) - mine;
                        int tile = -1;
                        unsigned long long tbase = 0ull;
                        if (mode == 0) {
                            const unsigned h = __ballot_sync(0xffffffffu, excl <= tau && excl + mine > tau);
                            if (h) {
                                const int l = __ffs(h) - 1;
                                if (lane == l) {  // the sums are exact: the run holds tau in one sub-tile
                                    unsigned long long c2 = excl;
                                    for (int sb = s_lo; sb < s_hi; ++sb) {
                                        const unsigned long long v = fix_of(s_sub[sb]);
                                        if (c2 + v > tau) { tile = sb; break; }
                                        c2 += v;
                                    }
                                    tbase = c2;
                                }
                                tile = __shfl_sync(0xffffffffu, tile, l);
                                tbase = __shfl_sync(0xffffffffu, tbase, l);
                            } else {
                                mode = 1;
                            }
                        }
                        if (mode == 1) {
                            int last = -1;
                            for (int sb = s_lo; sb < s_hi; ++sb)
                                if (s_sub[sb] > 0.f) last = sb;
                            for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
                            tile = max(last, 0);
                        }
                        Raw r;
                        load_sub(trow, zrow, use_q, tile, r);
                        float w[kW];
                        weights(r, use_q, s, w);
                        const int j0 = e0 + tile * kSub + lane * kW;
                        bool done = false;
                        if (mode == 0) {
                            unsigned long long wsum = 0ull;
#pragma unroll
                            for (int e = 0; e < kW; ++e) wsum += fix_of(w[e]);
                            const unsigned long long wex = tbase + warp_incl_scan_u64(wsum) - wsum;
                            const bool hit = wex <= tau && wex + wsum > tau;
                            if (hit) {
                                unsigned long long C = wex;
                                for (int e = 0; e < kW; ++e) {
                                    const unsigned long long Cprev = C;
                                    C += fix_of(w[e]);
                                    if (C > tau) {
                                        pick = j0 + e;
                                        gap = fminf(fix_to_float(C - tau), fix_to_float(tau - Cprev)) / fix_to_float(W);
                                        break;
                                    }
                                }
                            }
                            done = __any_sync(0xffffffffu, hit);
                        }
                        if (!done) {  // the largest j of the sub-tile with w_j > 0 (rounding fallback)
                            int best = -1;
                            float wbest = 0.f;
#pragma unroll
                            for (int e = 0; e < kW; ++e)
                                if (w[e] > 0.f) { best = j0 + e; wbest = w[e]; }
                            int jb = best;
                            for (int o = 16; o > 0; o >>= 1) jb = max(jb, __shfl_xor_sync(0xffffffffu, jb, o));
                            pick = -1;
                            if (jb >= 0 && best == jb) {
                                pick = jb;
                                const float Wf = fix_to_float(W), tf = fix_to_float(tau);
                                gap = fminf(Wf - tf, tf - (Wf - wbest)) / Wf;
                            } else if (jb < 0 && lane == 0) {
                                pick = j0;  // no positive entry: cannot happen when W > 0
                            }
                        }
                    }
                    if (pick >= 0 && (mode != 2 || lane == 0)) {
                        out[depth] = pick;
                        if (p.diag_gap && mode != 2) p.diag_gap[b] = gap;
                    }
                }
                if (tid == 0) s_extra = -1;  // written by the owner
                break;
            }
        }
        if (rank == 0 && tid == 0) {
            pth[depth] = next;
            out[depth] = y[next];
        }
        ++depth;
        node = next;
    }
    if (rank == 0 && tid == 0) {
        if (greedy) out[depth] = s_extra;
        p.accepted[b] = depth;
        p.last_node[b] = node;
    }
    if (pending) cluster_wait();  // keep this CTA's total readable until every peer is done
}

// ------------------------------------------------------------------ host
static void tree_shape(int V, int* csize, int* span) {
    int c = (V + 4095) / 4096;
    c = c < 1 ? 1 : (c > kTreeMaxCluster ? kTreeMaxCluster : c);
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    *csize = c;
    *span = s;
}

static bool tree_topology(const int32_t* parent, int n, TreeTopo* topo) {
    if (!parent || parent[0] != -1) return false;
    for (int i = 0; i < OSD_TREE_MAX_NODES; ++i) {
        topo->first_child[i] = -1;
        topo->next_sibling[i] = -1;
    }
    int8_t last_child[OSD_TREE_MAX_NODES];
    for (int i = 0; i < OSD_TREE_MAX_NODES; ++i) last_child[i] = -1;
    for (int i = 0; i < OSD_TREE_MAX_NODES; ++i) topo->parent[i] = -1;
    for (int i = 1; i < n; ++i) {
        const int par = parent[i];
        if (par < 0 || par >= i) return false;
        topo->parent[i] = static_cast<int8_t>(par);
        if (last_child[par] < 0) topo->first_child[par] = static_cast<int8_t>(i);
        else topo->next_sibling[last_child[par]] = static_cast<int8_t>(i);
        last_child[par] = static_cast<int8_t>(i);
    }
    return true;
}

static long long tree_stat_rows(int B, int n, bool greedy) { return (greedy ? 1LL : 2LL) * B * n; }

template <typename In>
static osd_status launch_tree(const TreeParams& base, int B, const void* draft, const void* target,
                              RowStat* stats, cudaStream_t stream) {
    TreeParams tp = base;
    const bool greedy = (tp.T == 0.f);
    const int n = tp.n, V = tp.V;
    const long long rows = tree_stat_rows(B, n, greedy);
    const int slice_len = stats_slice_len(rows);
    const int n_slices = (V + slice_len - 1) / slice_len;
    const long long n_draft_rows = greedy ? 0 : (long long)B * n;
    const long long grid1 = rows * n_slices;
    if (grid1 > INT_MAX) return OSD_ERR_UNSUPPORTED;
    cudaError_t e;
    if (greedy)
        e = launch(row_stats_kernel<In, true>, dim3(unsigned(grid1)), dim3(kStatThreads), 0, stream, 1,
                   static_cast<const In*>(draft), static_cast<const In*>(target), n_draft_rows, V, slice_len,
                   n_slices, tp.c_hi, tp.c_lo, stats);
    else
        e = launch(row_stats_kernel<In, false>, dim3(unsigned(grid1)), dim3(kStatThreads), 0, stream, 1,
                   static_cast<const In*>(draft), static_cast<const In*>(target), n_draft_rows, V, slice_len,
                   n_slices, tp.c_hi, tp.c_lo, stats);
    if (e != cudaSuccess) return OSD_ERR_CUDA;

    tp.stats = stats;
    tp.n_slices = n_slices;
    tp.n_draft_rows = n_draft_rows;
    int csize = 1, span = V;
    if (!greedy) tree_shape(V, &csize, &span);
    tp.csize = csize;
    tp.span = span;
    const bool vec = !greedy && aligned_to(draft, 16) && aligned_to(target, 16) && ((size_t)V * sizeof(In)) % 16 == 0;
    const int sub = 32 * (vec ? Elem<In>::kVec : 1);
    const size_t smem = greedy ? 0 : size_t((span + sub - 1) / sub) * sizeof(float);
    if (smem > size_t(kTreeMaxSub) * sizeof(float)) return OSD_ERR_UNSUPPORTED;
    const dim3 grid2(unsigned(B) * unsigned(csize));
    if (vec)
        e = launch_ex(true, tree_walk_kernel<In, true>, grid2, dim3(kTreeThreads), smem, stream, csize, tp);
    else
        e = launch_ex(true, tree_walk_kernel<In, false>, grid2, dim3(kTreeThreads), smem, stream, csize, tp);
    return from_cuda(e);
}

}  // namespace osd

extern "C" osd_status osd_verify_tree_workspace_size(int B, int n_nodes, int V, size_t* bytes) {
    using namespace osd;
    if (!bytes || B < 0 || n_nodes < 1 || V < 1) return OSD_ERR_INVALID_ARG;
    if (n_nodes > OSD_TREE_MAX_NODES || V > OSD_VERIFY_MAX_V) return OSD_ERR_UNSUPPORTED;
    const long long rows = tree_stat_rows(B, n_nodes, false);
    const int len = stats_slice_len(rows);
    // the greedy pass has half the rows but may take shorter slices: size for the larger
    const int len0 = stats_slice_len(tree_stat_rows(B, n_nodes, true));
    const size_t need = std::max(size_t(rows) * size_t((V + len - 1) / len),
                                 size_t(tree_stat_rows(B, n_nodes, true)) * size_t((V + len0 - 1) / len0)) *
                        sizeof(RowStat);
    *bytes = (need + 255) / 256 * 256;
    return OSD_OK;
}

extern "C" osd_status osd_verify_tree(const void* draft_logits, const void* target_logits, osd_dtype dtype, int B,
                                      int n_nodes, int V, const int32_t* parent, const int32_t* tokens,
                                      const float* uniforms, float temperature, int32_t* accepted, int32_t* path,
                                      int32_t* out_tokens, int32_t* last_node, float* diag_margin,
                                      float* diag_cdf_gap, void* workspace, size_t workspace_bytes, void* stream) {
    using namespace osd;
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    if (B < 0 || n_nodes < 1 || V < 1) return OSD_ERR_INVALID_ARG;
    if (!(temperature >= 0.f) || !std::isfinite(temperature)) return OSD_ERR_INVALID_ARG;
    if (n_nodes > OSD_TREE_MAX_NODES || V > OSD_VERIFY_MAX_V) return OSD_ERR_UNSUPPORTED;
    TreeParams tp = {};
    if (!tree_topology(parent, n_nodes, &tp.topo)) return OSD_ERR_INVALID_ARG;
    if (B == 0) return OSD_OK;
    const bool greedy = (temperature == 0.f);
    const size_t es = dtype_size(dtype);
    if (!target_logits || !tokens || !accepted || !path || !out_tokens || !last_node || !workspace)
        return OSD_ERR_INVALID_ARG;
    if (!greedy && (!draft_logits || !uniforms)) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(target_logits, es) || (draft_logits && !aligned_to(draft_logits, es)) ||
        !aligned_to(workspace, 16))
        return OSD_ERR_INVALID_ARG;
    size_t need = 0;
    osd_verify_tree_workspace_size(B, n_nodes, V, &need);
    if (workspace_bytes < need) return OSD_ERR_INVALID_ARG;
    tp.draft = draft_logits;
    tp.target = target_logits;
    tp.n = n_nodes;
    tp.V = V;
    tp.tokens = tokens;
    tp.uniforms = uniforms;
    tp.T = temperature;
    if (!greedy) split_scale(temperature, &tp.c_hi, &tp.c_lo);
    tp.accepted = accepted;
    tp.path = path;
    tp.out_tokens = out_tokens;
    tp.last_node = last_node;
    tp.diag_margin = diag_margin;
    tp.diag_gap = diag_cdf_gap;
    RowStat* stats = static_cast<RowStat*>(workspace);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the draft rows are not read at T = 0; any aligned pointer stands in
    const void* draft = greedy ? target_logits : draft_logits;
    return dtype == OSD_BF16 ? launch_tree<__nv_bfloat16>(tp, B, draft, target_logits, stats, s)
                             : launch_tree<float>(tp, B, draft, target_logits, stats, s);
}
