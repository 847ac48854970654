// osd_rowstats.cuh -- the row-statistics pass shared by the verifiers
// (osd_verify.cu, osd_tree.cu): one CTA per (row, vocabulary slice) over a
// batch of draft rows followed by target rows, a single streaming pass of
// 16-byte loads computing the max and the sum of 2^((x - max) c) of the slice
// (or its first argmax at T = 0).  This pass reads every logit once and
// carries almost all of a verification's HBM traffic.
#pragma once

#include <climits>
#include <cstdint>

#include "osd_device.cuh"

namespace osd {

struct RowStat {
    float m;   // max raw logit of the slice
    float s;   // sum of 2^((x - m) c) over the slice (T > 0)
    int idx;   // first index of the max (T == 0)
    int pad;
};

constexpr int kStatThreads = 256;
constexpr int kStatUnroll = 2;  // 16-byte vectors per thread per group (one group in flight ahead)

// Vocabulary entries per row_stats CTA: long slices amortise the per-CTA merge,
// short ones keep enough CTAs in flight when there are few rows.
inline int stats_slice_len(long long rows) {
    return rows >= 2048 ? 32768 : (rows >= 512 ? 16384 : 8192);
}

// ------------------------------------------------------------------ pass 1
template <typename In, bool kGreedy>
__global__ void __launch_bounds__(kStatThreads)
row_stats_kernel(const In* __restrict__ draft, const In* __restrict__ target,
                 long long n_draft_rows, int V, int slice_len, int n_slices, float c_hi, float c_lo,
                 RowStat* __restrict__ stats) {
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    constexpr int kGroup = kStatUnroll * kVec;
    __shared__ float2 red_m[kStatThreads / 32];
    __shared__ float red_s[kStatThreads / 32];
    __shared__ MaxIdx red_mi[kStatThreads / 32];

    allow_dependent_launch();  // the consumer of the statistics waits for them in-kernel
    const long long item = blockIdx.x;
    const long long row = item / n_slices;
    const int slice = static_cast<int>(item - row * n_slices);
    const In* rowp = (row < n_draft_rows) ? draft + row * V : target + (row - n_draft_rows) * V;
    const int s0 = slice * slice_len;
    const int n = min(V - s0, slice_len);
    const In* p = rowp + s0;

    // head (scalar up to the first 16-byte boundary), body (vectors), tail
    const uintptr_t addr = reinterpret_cast<uintptr_t>(p);
    int head = static_cast<int>(((16u - (addr & 15u)) & 15u) / sizeof(In));
    if (head > n) head = n;
    const int nvec = (n - head) / kVec;
    const int tail0 = head + nvec * kVec;
    const In* body = p + head;
    const int tid = threadIdx.x;
    const uint4 ninf = make_uint4(NegInfRaw<In>::bits, NegInfRaw<In>::bits, NegInfRaw<In>::bits,
                                  NegInfRaw<In>::bits);
    auto load_group = [&](int v, uint4* r) {
#pragma unroll
        for (int u = 0; u < kStatUnroll; ++u) {
            const int vv = v + u * kStatThreads;
            r[u] = (vv < nvec) ? ldg_stream(body + size_t(vv) * kVec) : ninf;
        }
    };

    if constexpr (kGreedy) {
        MaxIdx acc{kNegInf, INT_MAX};
        auto take = [&](float x, int j) {
            if (x > acc.m) { acc.m = x; acc.i = j; }
        };
        if (tid < head) take(E::load(p + tid), s0 + tid);
        uint4 cur[kStatUnroll], nxt[kStatUnroll];
        int v = tid;
        if (v < nvec) load_group(v, cur);
        for (; v < nvec; v += kStatUnroll * kStatThreads) {
            const int vn = v + kStatUnroll * kStatThreads;
            if (vn < nvec) load_group(vn, nxt);
            float cm = E::max_raw(cur[0]);
#pragma unroll
            for (int u = 1; u < kStatUnroll; ++u) cm = fmaxf(cm, E::max_raw(cur[u]));
            if (cm > acc.m) {  // rare: find the first entry equal to the group maximum
#pragma unroll
                for (int u = 0; u < kStatUnroll; ++u) {
                    float x[kVec];
                    E::unpack(cur[u], x);
                    const int j0 = s0 + head + (v + u * kStatThreads) * kVec;
#pragma unroll
                    for (int e = 0; e < kVec; ++e) take(x[e], j0 + e);
                }
            }
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) cur[u] = nxt[u];
        }
        if (tid < n - tail0) take(E::load(p + tail0 + tid), s0 + tail0 + tid);
        acc = block_reduce<kStatThreads>(acc, [](MaxIdx a, MaxIdx b) { return merge_mi(a, b); }, red_mi);
        if (tid == 0) stats[item] = RowStat{acc.m, 0.f, acc.i, 0};
    } else {
        float m = kNegInf;
        float2 s2 = f2(0.f);
        // 2^((x - m) c) with x - m exact and c = c_hi + c_lo carried as a float pair
        auto exp_pair = [&](float a, float b) {
            const float2 d = sub2(make_float2(a, b), f2(m));
            const float2 g = fma2(d, f2(c_hi), mul2(d, f2(c_lo)));
            return make_float2(ex2(g.x), ex2(g.y));
        };
        auto raise_max = [&](float cm) {
            if (cm > m) {
                s2 = (m == kNegInf) ? f2(0.f) : mul2(s2, f2(ex2(mul_c(m - cm, c_hi, c_lo))));
                m = cm;
            }
        };
        auto one = [&](float x) {
            raise_max(x);
            if (m != kNegInf) s2.x += ex2(mul_c(x - m, c_hi, c_lo));
        };
        if (tid < head) one(E::load(p + tid));
        uint4 cur[kStatUnroll], nxt[kStatUnroll];
        int v = tid;
        if (v < nvec) load_group(v, cur);
        for (; v < nvec; v += kStatUnroll * kStatThreads) {
            const int vn = v + kStatUnroll * kStatThreads;
            if (vn < nvec) load_group(vn, nxt);
            float cm = E::max_raw(cur[0]);
#pragma unroll
            for (int u = 1; u < kStatUnroll; ++u) cm = fmaxf(cm, E::max_raw(cur[u]));
            raise_max(cm);
            if (m != kNegInf) {
                float x[kGroup];
#pragma unroll
                for (int u = 0; u < kStatUnroll; ++u) E::unpack(cur[u], x + u * kVec);
#pragma unroll
                for (int e = 0; e < kGroup; e += 2) s2 = add2(s2, exp_pair(x[e], x[e + 1]));
            }
#pragma unroll
            for (int u = 0; u < kStatUnroll; ++u) cur[u] = nxt[u];
        }
        if (tid < n - tail0) one(E::load(p + tail0 + tid));
        // block merge: maximum first, then one rescale per thread and a plain sum
        float bm = m;
        for (int o = 16; o > 0; o >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, o));
        const int lane = tid & 31, warp = tid >> 5;
        if (lane == 0) red_m[warp].x = bm;
        __syncthreads();
        bm = red_m[0].x;
#pragma unroll
        for (int w = 1; w < kStatThreads / 32; ++w) bm = fmaxf(bm, red_m[w].x);
        float s = (m == kNegInf) ? 0.f : (s2.x + s2.y) * ex2(mul_c(m - bm, c_hi, c_lo));
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) red_s[warp] = s;
        __syncthreads();
        if (tid == 0) {
            float tot = red_s[0];
#pragma unroll
            for (int w = 1; w < kStatThreads / 32; ++w) tot += red_s[w];
            stats[item] = RowStat{bm, tot, 0, 0};
        }
    }
}

}  // namespace osd
