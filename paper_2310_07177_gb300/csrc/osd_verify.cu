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
//   verify_finalize     one thread-block cluster per sequence: merges the slice
//                       statistics, runs the k accept tests u_i < p_i(y_i)/q_i(y_i)
//                       in order, then draws the extra token from
//                       norm(max(0, p_a - q_a)) (or p_k when all k pass) by inverse
//                       CDF.  Each CTA of the cluster sums the residual weights of
//                       its part of the vocabulary per tile; the partial sums meet
//                       through distributed shared memory and the CTA whose part
//                       holds u*W rescans that one tile with an fp64 block scan.
//
// The log-ratio of the accept test is formed from differences of raw logits and
// maxima, (t_y - m_t) - (z_y - m_z), and the ratio of the two sums, so no
// log-sum-exp is rounded on its own.
#include <climits>
#include <cstdint>
#include <mutex>
#include <type_traits>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"

namespace osd {

struct RowStat {
    float m;   // max raw logit of the slice
    float s;   // sum of 2^((x - m) c) over the slice (T > 0)
    int idx;   // first index of the max (T == 0)
    int pad;
};

constexpr int kStatThreads = 256;
constexpr int kStatUnroll = 4;
constexpr int kStatSlice = 8192;  // vocabulary entries per row_stats CTA

constexpr int kFinThreads = 256;
constexpr int kFinMaxCluster = 8;
constexpr int kFinMaxTiles = 1024;  // tiles of one CTA's vocabulary span

// ------------------------------------------------------------------ pass 1
template <typename In, bool kGreedy>
__global__ void __launch_bounds__(kStatThreads)
row_stats_kernel(const In* __restrict__ draft, const In* __restrict__ target,
                 long long n_draft_rows, int V, int n_slices, float c_hi, float c_lo,
                 RowStat* __restrict__ stats) {
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    __shared__ MaxSum red_ms[kStatThreads / 32];
    __shared__ MaxIdx red_mi[kStatThreads / 32];

    const long long item = blockIdx.x;
    const long long row = item / n_slices;
    const int slice = static_cast<int>(item - row * n_slices);
    const In* rowp = (row < n_draft_rows) ? draft + row * V : target + (row - n_draft_rows) * V;
    const int s0 = slice * kStatSlice;
    const int n = min(V - s0, kStatSlice);
    const In* p = rowp + s0;

    // head (scalar up to the first 16-byte boundary), body (vectors), tail
    const uintptr_t addr = reinterpret_cast<uintptr_t>(p);
    int head = static_cast<int>(((16u - (addr & 15u)) & 15u) / sizeof(In));
    if (head > n) head = n;
    const int nvec = (n - head) / kVec;
    const int tail0 = head + nvec * kVec;
    const In* body = p + head;
    const int tid = threadIdx.x;

    if constexpr (kGreedy) {
        MaxIdx acc{kNegInf, INT_MAX};
        auto take = [&](float x, int j) {
            if (x > acc.m) { acc.m = x; acc.i = j; }
        };
        if (tid < head) take(E::load(p + tid), s0 + tid);
        int v = tid;
        for (; v + (kStatUnroll - 1) * kStatThreads < nvec; v += kStatUnroll * kStatThreads) {
            uint4 r[kStatUnroll];
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) r[u] = ldg_stream(body + size_t(v + u * kStatThreads) * kVec);
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) {
                float x[kVec];
                E::unpack(r[u], x);
                const int j0 = s0 + head + (v + u * kStatThreads) * kVec;
#pragma unroll
                for (int e = 0; e < kVec; ++e) take(x[e], j0 + e);
            }
        }
        for (; v < nvec; v += kStatThreads) {
            float x[kVec];
            E::unpack(ldg_stream(body + size_t(v) * kVec), x);
            const int j0 = s0 + head + v * kVec;
#pragma unroll
            for (int e = 0; e < kVec; ++e) take(x[e], j0 + e);
        }
        if (tid < n - tail0) take(E::load(p + tail0 + tid), s0 + tail0 + tid);
        acc = block_reduce<kStatThreads>(acc, merge_mi, red_mi);
        if (tid == 0) stats[item] = RowStat{acc.m, 0.f, acc.i, 0};
    } else {
        MaxSum acc{kNegInf, 0.f};
        // Fold a chunk of values: one max (and at most one rescale) per chunk.
        auto fold = [&](const float* x, auto cnt_tag) {
            constexpr int kCnt = decltype(cnt_tag)::value;
            float cm = x[0];
#pragma unroll
            for (int e = 1; e < kCnt; ++e) cm = fmaxf(cm, x[e]);
            if (cm > acc.m) {
                acc.s = (acc.m == kNegInf) ? 0.f : acc.s * ex2(mul2(acc.m - cm, c_hi, c_lo));
                acc.m = cm;
            }
            if (acc.m != kNegInf) {
                float s0v = 0.f, s1v = 0.f;
#pragma unroll
                for (int e = 0; e < kCnt; e += 2) {
                    s0v += ex2(mul2(x[e] - acc.m, c_hi, c_lo));
                    if (e + 1 < kCnt) s1v += ex2(mul2(x[e + 1] - acc.m, c_hi, c_lo));
                }
                acc.s += s0v + s1v;
            }
        };
        using One = std::integral_constant<int, 1>;
        if (tid < head) { const float x = E::load(p + tid); fold(&x, One{}); }
        int v = tid;
        for (; v + (kStatUnroll - 1) * kStatThreads < nvec; v += kStatUnroll * kStatThreads) {
            uint4 r[kStatUnroll];
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) r[u] = ldg_stream(body + size_t(v + u * kStatThreads) * kVec);
            float x[kStatUnroll * kVec];
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) E::unpack(r[u], x + u * kVec);
            fold(x, std::integral_constant<int, kStatUnroll * kVec>{});
        }
        for (; v < nvec; v += kStatThreads) {
            float x[kVec];
            E::unpack(ldg_stream(body + size_t(v) * kVec), x);
            fold(x, std::integral_constant<int, kVec>{});
        }
        if (tid < n - tail0) { const float x = E::load(p + tail0 + tid); fold(&x, One{}); }
        auto merge = [c_hi, c_lo](MaxSum a, MaxSum b) { return merge_ms(a, b, c_hi, c_lo); };
        acc = block_reduce<kStatThreads>(acc, merge, red_ms);
        if (tid == 0) stats[item] = RowStat{acc.m, acc.s, 0, 0};
    }
}

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

// Inclusive block scan of doubles; returns the exclusive prefix, `total` gets the sum.
template <int kThreads>
__device__ __forceinline__ double block_exclusive_scan(double v, double* warp_tot, double* total) {
    constexpr int kWarps = kThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    double x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    double before = 0.0, all = 0.0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
        if (w < warp) before += warp_tot[w];
        all += warp_tot[w];
    }
    *total = all;
    return before + x - v;
}

template <typename In, bool kVecPath>
__global__ void __launch_bounds__(kFinThreads) verify_finalize_kernel(FinParams p) {
    using E = Elem<In>;
    constexpr int kW = kVecPath ? E::kVec : 1;  // entries per thread per tile
    constexpr int kTile = kFinThreads * kW;
    constexpr int kWarps = kFinThreads / 32;

    __shared__ float s_m[2 * OSD_VERIFY_MAX_K + 1];
    __shared__ float s_s[2 * OSD_VERIFY_MAX_K + 1];
    __shared__ int s_idx[OSD_VERIFY_MAX_K + 1];
    __shared__ float s_zy[OSD_VERIFY_MAX_K], s_ty[OSD_VERIFY_MAX_K];
    __shared__ int s_bad, s_a, s_owner, s_mode, s_tile, s_found;
    __shared__ double s_tiles[kFinMaxTiles];
    __shared__ double s_span_total;  // read by the other CTAs of the cluster
    __shared__ double s_tau, s_W, s_base;
    __shared__ double red_d[kWarps];
    __shared__ MaxIdx red_mi[kWarps];
    __shared__ int red_i[kWarps];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int rank = (p.csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const int b = blockIdx.x / p.csize;
    const int k = p.k, V = p.V;
    const bool greedy = (p.T == 0.f);
    const int32_t* y = p.tokens + size_t(b) * k;
    const In* draft = static_cast<const In*>(p.draft);
    const In* target = static_cast<const In*>(p.target);

    if (tid == 0) s_bad = 0;
    __syncthreads();
    if (tid < k) {
        const int t = y[tid];
        if (t < 0 || t >= V) atomicOr(&s_bad, 1);
    }
    // Merge slice statistics: local row r <= k is target row r, r > k is draft row r-k-1.
    const int nrows = greedy ? (k + 1) : (2 * k + 1);
    for (int r = warp; r < nrows; r += kWarps) {
        const long long srow = (r <= k) ? (p.n_draft_rows + (long long)b * (k + 1) + r)
                                        : ((long long)b * k + (r - k - 1));
        const RowStat* st = p.stats + srow * p.n_slices;
        if (greedy) {
            MaxIdx acc{kNegInf, INT_MAX};
            for (int sl = lane; sl < p.n_slices; sl += 32) acc = merge_mi(acc, MaxIdx{st[sl].m, st[sl].idx});
            acc = warp_reduce(acc, merge_mi);
            if (lane == 0) { s_m[r] = acc.m; s_idx[r] = (acc.i == INT_MAX) ? 0 : acc.i; }
        } else {
            const float ch = p.c_hi, cl = p.c_lo;
            auto merge = [ch, cl](MaxSum a, MaxSum c) { return merge_ms(a, c, ch, cl); };
            MaxSum acc{kNegInf, 0.f};
            for (int sl = lane; sl < p.n_slices; sl += 32) acc = merge(acc, MaxSum{st[sl].m, st[sl].s});
            acc = warp_reduce(acc, merge);
            if (lane == 0) { s_m[r] = acc.m; s_s[r] = acc.s; }
        }
    }
    if (!greedy && tid < k) {
        const int t = y[tid];
        if (t >= 0 && t < V) {
            s_zy[tid] = E::load(draft + (size_t(b) * k + tid) * V + t);
            s_ty[tid] = E::load(target + (size_t(b) * (k + 1) + tid) * V + t);
        }
    }
    __syncthreads();

    int32_t* out = p.out_tokens + size_t(b) * (k + 1);
    if (s_bad) {  // uniform over the cluster, before any distributed shared memory access
        if (rank == 0) {
            if (tid == 0) { p.accepted[b] = -1; if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000); }
            for (int i = tid; i <= k; i += kFinThreads) out[i] = -1;
            for (int i = tid; i < k; i += kFinThreads) {
                p.mask[size_t(b) * k + i] = 0;
                if (p.diag_margin) p.diag_margin[size_t(b) * k + i] = __int_as_float(0x7fc00000);
            }
        }
        return;
    }

    // ---- accept tests, in order, stopping at the first rejection
    if (tid == 0) {
        int a = 0;
        if (greedy) {
            while (a < k && y[a] == s_idx[a]) ++a;
        } else {
            for (; a < k; ++a) {
                const float mt = s_m[a], st = s_s[a];
                const float mz = s_m[k + 1 + a], sz = s_s[k + 1 + a];
                const float D = (s_ty[a] - mt) - (s_zy[a] - mz);
                const float r = expf(__fdiv_rn(D, p.T)) * __fdiv_rn(sz, st);
                const float u = p.uniforms[size_t(b) * (k + 1) + a];
                if (rank == 0 && p.diag_margin) p.diag_margin[size_t(b) * k + a] = fabsf(u - r);
                if (!(u < r)) break;
            }
        }
        s_a = a;
    }
    __syncthreads();
    const int a = s_a;
    if (rank == 0) {
        if (tid == 0) p.accepted[b] = a;
        for (int i = tid; i <= k; i += kFinThreads)
            if (i < a) out[i] = y[i];
            else if (i > a) out[i] = -1;
        for (int i = tid; i < k; i += kFinThreads) {
            p.mask[size_t(b) * k + i] = (i == a) ? 1 : 0;
            if (p.diag_margin && (greedy || i > a)) p.diag_margin[size_t(b) * k + i] = __int_as_float(0x7fc00000);
        }
    }
    if (greedy) {  // launched with one CTA per sequence
        if (tid == 0) {
            out[a] = s_idx[a];
            if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000);
        }
        return;
    }

    // ---- extra token: inverse CDF of w = max(0, p_a - q_a) (a < k) or p_k (a == k)
    const bool bonus = (a == k);
    const In* trow = target + (size_t(b) * (k + 1) + a) * V;
    const In* zrow = draft + (size_t(b) * k + (bonus ? 0 : a)) * V;
    const float mt = s_m[a], inv_st = 1.0f / s_s[a];
    const float mz = bonus ? 0.f : s_m[k + 1 + a];
    const float inv_sz = bonus ? 0.f : 1.0f / s_s[k + 1 + a];
    const float ch = p.c_hi, cl = p.c_lo;
    auto weight = [&](float t, float z) -> float {
        const float pj = ex2(mul2(t - mt, ch, cl)) * inv_st;
        if (bonus) return pj;
        const float qj = ex2(mul2(z - mz, ch, cl)) * inv_sz;
        return fmaxf(pj - qj, 0.f);
    };
    const int e0 = rank * p.span;
    const int n = max(0, min(p.span, V - e0));
    const int ntiles = (n + kTile - 1) / kTile;
    // weights of this thread's entries of tile `tile` (entries past the span get 0)
    auto tile_weights = [&](int tile, float* w) {
        const int j0 = e0 + tile * kTile + tid * kW;
        const int cnt = min(kW, e0 + n - j0);
        if (kVecPath && cnt == kW) {
            float t[kW], z[kW];
            E::unpack(ldg_stream(trow + j0), t);
            if (!bonus) E::unpack(ldg_stream(zrow + j0), z);
#pragma unroll
            for (int e = 0; e < kW; ++e) w[e] = weight(t[e], bonus ? 0.f : z[e]);
        } else {
#pragma unroll
            for (int e = 0; e < kW; ++e)
                w[e] = (e < cnt) ? weight(E::load(trow + j0 + e), bonus ? 0.f : E::load(zrow + j0 + e)) : 0.f;
        }
    };

    // pass 1: per-tile sums of this CTA's span
    double span_total = 0.0;
    for (int tile = 0; tile < ntiles; ++tile) {
        float w[kW];
        tile_weights(tile, w);
        float sum = 0.f;
#pragma unroll
        for (int e = 0; e < kW; ++e) sum += w[e];
        const double ts = block_reduce<kFinThreads>(double(sum), [](double x, double z) { return x + z; }, red_d);
        if (tid == 0) s_tiles[tile] = ts;
        span_total += ts;
    }
    if (tid == 0) s_span_total = span_total;
    if (p.csize > 1) cluster_sync(); else __syncthreads();

    // every CTA derives W, tau and the owning CTA identically (rank order)
    if (tid == 0) {
        const float u = p.uniforms[size_t(b) * (k + 1) + k];
        double tot[kFinMaxCluster];
        for (int r = 0; r < p.csize; ++r)
            tot[r] = (r == rank) ? s_span_total : ld_dsmem_f64(map_rank(&s_span_total, r));
        double W = 0.0;
        for (int r = 0; r < p.csize; ++r) W += tot[r];
        const double tau = double(u) * W;
        int owner = -1, mode = 0;  // mode 0: inverse CDF, 1: largest positive entry, 2: argmax p
        double cum = 0.0, base = 0.0;
        if (W > 0.0) {
            for (int r = 0; r < p.csize; ++r) {
                if (cum + tot[r] > tau) { owner = r; base = cum; break; }
                cum += tot[r];
            }
            if (owner < 0) {  // tau >= W (u >= 1 or rounding): largest j with w_j > 0
                mode = 1;
                for (int r = p.csize - 1; r >= 0; --r)
                    if (tot[r] > 0.0) { owner = r; break; }
            }
        } else {
            mode = 2;
            owner = 0;
        }
        s_owner = owner; s_mode = mode; s_tau = tau; s_W = W; s_base = base;
    }
    __syncthreads();
    if (p.csize > 1) cluster_arrive();  // done reading the other CTAs' shared memory

    if (rank == s_owner) {
        const double tau = s_tau, W = s_W;
        int mode = s_mode;
        if (mode == 0 && tid == 0) {  // tile holding tau inside this span
            double cum = s_base;
            int tsel = -1;
            for (int t = 0; t < ntiles; ++t) {
                if (cum + s_tiles[t] > tau) { tsel = t; break; }
                cum += s_tiles[t];
            }
            s_tile = tsel;
            s_base = cum;
            if (tsel < 0) s_mode = 1;
        }
        __syncthreads();
        mode = s_mode;
        if (mode == 0) {
            // pass 2: fp64 scan of the selected tile
            const int tile = s_tile;
            float w[kW];
            tile_weights(tile, w);
            double mine = 0.0;
#pragma unroll
            for (int e = 0; e < kW; ++e) mine += double(w[e]);
            double tile_total;
            const double excl = s_base + block_exclusive_scan<kFinThreads>(mine, red_d, &tile_total);
            if (tid == 0) s_found = 0;
            __syncthreads();
            if (excl <= tau && excl + mine > tau) {
                double C = excl;
                const int j0 = e0 + tile * kTile + tid * kW;
                for (int e = 0; e < kW; ++e) {
                    const double Cprev = C;
                    C += double(w[e]);
                    if (C > tau) {
                        out[a] = j0 + e;
                        if (p.diag_gap) p.diag_gap[b] = float(fmin(C - tau, tau - Cprev) / W);
                        atomicExch(&s_found, 1);
                        break;
                    }
                }
            }
            __syncthreads();
            if (!s_found) mode = 1;  // rounding between the two passes: fall through
        }
        if (mode == 1) {
            // largest j of this span with w_j > 0
            int best = -1;
            float wbest = 0.f;
            for (int tile = 0; tile < ntiles; ++tile) {
                float w[kW];
                tile_weights(tile, w);
                const int j0 = e0 + tile * kTile + tid * kW;
#pragma unroll
                for (int e = 0; e < kW; ++e)
                    if (w[e] > 0.f && j0 + e > best) { best = j0 + e; wbest = w[e]; }
            }
            const int jb = block_reduce<kFinThreads>(best, [](int x, int z) { return max(x, z); }, red_i);
            if (jb >= 0 && best == jb) {
                out[a] = jb;
                if (p.diag_gap) {
                    const double g1 = W - tau, g0 = tau - (W - double(wbest));
                    p.diag_gap[b] = float(fmin(g1, g0) / W);
                }
            }
        } else if (mode == 2) {
            // no residual mass at all: argmax of p_a over the whole row
            MaxIdx acc{kNegInf, INT_MAX};
            for (int j = tid; j < V; j += kFinThreads) {
                const float t = E::load(trow + j);
                if (t > acc.m) { acc.m = t; acc.i = j; }
            }
            acc = block_reduce<kFinThreads>(acc, merge_mi, red_mi);
            if (tid == 0) {
                out[a] = (acc.i == INT_MAX) ? 0 : acc.i;
                if (p.diag_gap) p.diag_gap[b] = __int_as_float(0x7fc00000);
            }
        }
    }
    if (p.csize > 1) cluster_wait();  // keep this CTA's shared memory alive for its peers
}

// ------------------------------------------------------------------ host
static int verify_slices(int V) { return (V + kStatSlice - 1) / kStatSlice; }

static void finalize_shape(int V, int* csize, int* span) {
    int c = (V + 4095) / 4096;
    c = c < 1 ? 1 : (c > kFinMaxCluster ? kFinMaxCluster : c);
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    *csize = c;
    *span = s;
}

template <typename In>
static osd_status launch_verify(const void* draft, const void* target, int B, int k, int V,
                                const int32_t* tokens, const float* uniforms, float T,
                                int32_t* accepted, int32_t* out_tokens, uint8_t* mask,
                                float* diag_margin, float* diag_gap, RowStat* stats,
                                cudaStream_t stream) {
    const bool greedy = (T == 0.f);
    const int n_slices = verify_slices(V);
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
                   n_slices, c_hi, c_lo, stats);
    else
        e = launch(row_stats_kernel<In, false>, dim3(unsigned(grid1)), dim3(kStatThreads), 0, stream, 1,
                   static_cast<const In*>(draft), static_cast<const In*>(target), n_draft_rows, V,
                   n_slices, c_hi, c_lo, stats);
    if (e != cudaSuccess) return OSD_ERR_CUDA;

    FinParams fp;
    fp.draft = draft; fp.target = target; fp.B = B; fp.k = k; fp.V = V;
    fp.tokens = tokens; fp.uniforms = uniforms; fp.T = T; fp.c_hi = c_hi; fp.c_lo = c_lo;
    fp.stats = stats; fp.n_slices = n_slices; fp.n_draft_rows = n_draft_rows;
    fp.accepted = accepted; fp.out_tokens = out_tokens; fp.mask = mask;
    fp.diag_margin = diag_margin; fp.diag_gap = diag_gap;
    int csize = 1, span = V;
    if (!greedy) finalize_shape(V, &csize, &span);
    fp.csize = csize;
    fp.span = span;
    const bool vec = !greedy && aligned_to(draft, 16) && aligned_to(target, 16) &&
                     ((size_t)V * sizeof(In)) % 16 == 0;
    const dim3 grid2(unsigned(B) * unsigned(csize));
    if (vec)
        e = launch(verify_finalize_kernel<In, true>, grid2, dim3(kFinThreads), 0, stream, csize, fp);
    else
        e = launch(verify_finalize_kernel<In, false>, grid2, dim3(kFinThreads), 0, stream, csize, fp);
    return from_cuda(e);
}

}  // namespace osd

using osd::RowStat;

extern "C" osd_status osd_verify_workspace_size(int B, int k, int V, size_t* bytes) {
    if (!bytes || B < 0 || k < 1 || V < 1) return OSD_ERR_INVALID_ARG;
    if (k > OSD_VERIFY_MAX_K || V > OSD_VERIFY_MAX_V) return OSD_ERR_UNSUPPORTED;
    const size_t rows = size_t(B) * size_t(2 * k + 1);
    size_t need = rows * size_t(osd::verify_slices(V)) * sizeof(RowStat);
    need = (need + 255) / 256 * 256;
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
    RowStat* stats = static_cast<RowStat*>(workspace);
    if (dtype == OSD_BF16)
        return osd::launch_verify<__nv_bfloat16>(draft_logits, target_logits, B, k, V, draft_tokens, uniforms,
                                                 temperature, accepted, out_tokens, mismatch_mask, diag_margin,
                                                 diag_cdf_gap, stats, s);
    return osd::launch_verify<float>(draft_logits, target_logits, B, k, V, draft_tokens, uniforms, temperature,
                                     accepted, out_tokens, mismatch_mask, diag_margin, diag_cdf_gap, stats, s);
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
std::mutex g_scratch_mu;
void* g_scratch_addr[kNoAllocMaxDevices] = {};
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
        // One-time set-up per device, with that device current: the host-side name
        // of the array is not a device address, so ask the runtime for it.
        std::lock_guard<std::mutex> lock(g_scratch_mu);
        if (!g_scratch_addr[dev]) {
            void* addr = nullptr;
            if (cudaGetSymbolAddress(&addr, g_verify_scratch) != cudaSuccess || !addr) return OSD_ERR_CUDA;
            g_scratch_addr[dev] = addr;
        }
        scratch = g_scratch_addr[dev];
    }
    // The statistics pass writes every workspace entry before the finalize pass
    // reads it, so nothing in the shared array needs clearing between calls.
    return osd_verify(draft_logits, target_logits, dtype, B, k, V, draft_tokens, uniforms, temperature,
                      accepted, out_tokens, mismatch_mask, diag_margin, diag_cdf_gap, scratch,
                      kNoAllocScratchBytes, stream);
}
