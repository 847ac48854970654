// osd_mixed.cu -- mixed-token sampling (Section 4.1 of the paper): one draw
// per position from beta p + (1 - beta) q_theta, p = softmax(t / tau),
// q = softmax(z / tau), by inverse CDF in ascending vocabulary order,
// j* = min{ j : C_j > u W } (the convention of the verifier's extra token).
//
// One CTA of kMixThreads threads per row, streaming both rows straight from
// HBM with 16-byte loads (one step of loads in flight ahead), no staging:
//
//   pass    every warp owns a contiguous quarter of the row and splits
//           its steps into kPieces runs; each lane keeps, per run, the
//           online max and sum of 2^((x - max) c) of both rows, and the warp
//           merges them at the end of the run: 32 pieces of the CDF per row;
//   pick    one warp merges the pieces into both normalisers, scans the 32
//           piece masses in fp64 for the piece that holds u W, and re-reads
//           that one piece to find the entry.
//
// Each logit is read once (plus one piece per row).  Small CTAs capped at 32
// registers a thread keep 16 rows (64 warps) in flight on every SM, and the
// single-warp pick of one row overlaps the streaming of the others.
#include <climits>
#include <cmath>
#include <cstdint>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"

namespace osd {

constexpr int kMixThreads = 128;
constexpr int kMixWarps = kMixThreads / 32;
constexpr int kPieces = 8;  // runs per warp: kMixWarps * kPieces = 32 pieces, one per lane of the picker
static_assert(kMixWarps * kPieces == 32, "one CDF piece per lane of the picking warp");

struct MixParams {
    const void* draft;
    const void* target;
    int V;
    long long dstride, tstride;  // elements between consecutive rows
    const float* uniforms;
    float beta;
    float c;  // log2(e) / tau, rounded to fp32
    int32_t* tokens;
    float* cdf_gap;
};

// Online sums of both rows over one piece, each as (M, s) with M = rn(max c)
// and s = sum 2^(x c - M).
struct Piece {
    float Mt, st, Mz, sz;
};

template <typename In, bool kVecPath>
__global__ void __launch_bounds__(kMixThreads, 16) mixed_sample_kernel(MixParams p) {
    using E = Elem<In>;
    constexpr int kW = kVecPath ? E::kVec : 1;  // entries per chunk
    __shared__ Piece s_piece[32];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long row = blockIdx.x;
    const In* zrow = static_cast<const In*>(p.draft) + row * p.dstride;
    const In* trow = static_cast<const In*>(p.target) + row * p.tstride;
    const int V = p.V;
    const float c = p.c;
    // chunks of the row, the warp ranges and the runs (pieces) of steps in them
    const int nch = (V + kW - 1) / kW;
    const int rch = (nch + kMixWarps - 1) / kMixWarps;  // chunks per warp range
    const int steps = (rch + 31) / 32;                   // steps of 32 chunks per range
    const int per_piece = (steps + kPieces - 1) / kPieces;
    auto range_lo = [&](int w) { return min(nch, w * rch); };

    // the kW raw entries of chunk c (past the row end they read as -inf)
    auto load_chunk = [&](const In* rp, int ci) -> uint4 {
        if constexpr (kVecPath) {
            if ((ci + 1) * kW <= V) return ldg_stream(rp + size_t(ci) * kW);
            float v[kW];  // the ragged last chunk of the row
#pragma unroll
            for (int e = 0; e < kW; ++e) v[e] = (ci * kW + e < V) ? E::load(rp + ci * kW + e) : kNegInf;
            return pack_raw<In, kW>(v);
        } else {
            float v[1] = {ci < V ? E::load(rp + ci) : kNegInf};
            return pack_raw<In, 1>(v);
        }
    };
    // a chunk of -inf, in the chunk's own layout (single entries are held as fp32)
    const uint4 none = kVecPath ? ninf_raw<In>() : ninf_raw<float>();
    auto chunk_max = [](const uint4& r) {
        if constexpr (kVecPath) return E::max_raw(r);
        else return __uint_as_float(r.x);
    };
    // Exponent arguments are x c - M as one FMA, M = rn(m c): the FMA rounds
    // once, after the cancellation, so the terms that carry the mass come out
    // as exact as from the difference (x - m) c, and the rounding of M is a
    // factor common to all the sums it scales.  Rescaling between two
    // references is 2^(M - M'), a difference of two floats.
    auto chunk_sum = [&](const uint4& r, float M) {
        float x[kW];
        unpack_raw<In, kW>(r, x);
        if constexpr (kW == 1) {
            return ex2(fmaf(x[0], c, -M));
        } else {
            float2 s2 = f2(0.f);
#pragma unroll
            for (int e = 0; e < kW; e += 2) {
                const float2 g = fma2(make_float2(x[e], x[e + 1]), f2(c), f2(-M));
                s2 = add2(s2, make_float2(ex2(g.x), ex2(g.y)));
            }
            return s2.x + s2.y;
        }
    };
    // one lane's running (reference M, sum s) absorbs a chunk: rescale when the
    // reference rises (rarely, once the first chunks are in), then add; a lane
    // that has seen only -inf keeps s = 0 and skips the sum
    auto absorb = [&](float& M, float& s, const uint4& r) {
        const float cM = __fmul_rn(chunk_max(r), c);
        if (cM > M) {
            s = (M == kNegInf) ? 0.f : s * ex2(M - cM);
            M = cM;
        }
        if (M != kNegInf) s += chunk_sum(r, M);
    };
    // the warp's merge of every lane's (M, s); M = -inf marks a lane without mass
    auto warp_merge = [&](float& M, float& s) {
        float gM = M;
        for (int o = 16; o > 0; o >>= 1) gM = fmaxf(gM, __shfl_xor_sync(0xffffffffu, gM, o));
        s = (M == kNegInf) ? 0.f : s * ex2(M - gM);
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        M = gM;
    };

    // ---- pass: the warp's steps, one step of loads in flight ahead
    {
        const int c0 = range_lo(warp), c1 = range_lo(warp + 1);
        auto chunk_of = [&](int st) { return c0 + st * 32 + lane; };
        uint4 zc = none, tc = none;
        if (steps > 0 && chunk_of(0) < c1) {
            zc = load_chunk(zrow, chunk_of(0));
            tc = load_chunk(trow, chunk_of(0));
        }
        for (int g = 0; g < kPieces; ++g) {
            float Mt = kNegInf, st_ = 0.f, Mz = kNegInf, sz = 0.f;
            const int s_end = min((g + 1) * per_piece, steps);
            for (int st = g * per_piece; st < s_end; ++st) {
                uint4 zn = none, tn = none;
                if (st + 1 < steps && chunk_of(st + 1) < c1) {
                    zn = load_chunk(zrow, chunk_of(st + 1));
                    tn = load_chunk(trow, chunk_of(st + 1));
                }
                absorb(Mt, st_, tc);
                absorb(Mz, sz, zc);
                zc = zn;
                tc = tn;
            }
            warp_merge(Mt, st_);
            warp_merge(Mz, sz);
            if (lane == 0) s_piece[warp * kPieces + g] = Piece{Mt, st_, Mz, sz};
        }
    }
    __syncthreads();
    if (warp != 0) return;

    // ---- pick: lane l holds piece l (in vocabulary order)
    const Piece pc = s_piece[lane];
    float Gt = pc.Mt, Gz = pc.Mz;  // rn(row max c): rounding is monotone, so the max of the M
    for (int o = 16; o > 0; o >>= 1) {
        Gt = fmaxf(Gt, __shfl_xor_sync(0xffffffffu, Gt, o));
        Gz = fmaxf(Gz, __shfl_xor_sync(0xffffffffu, Gz, o));
    }
    // each piece's sums against the row references (a piece of -inf only has none)
    const float rt = (pc.Mt == kNegInf) ? 0.f : pc.st * ex2(pc.Mt - Gt);
    const float rz = (pc.Mz == kNegInf) ? 0.f : pc.sz * ex2(pc.Mz - Gz);
    float Et = rt, Ez = rz;
    for (int o = 16; o > 0; o >>= 1) {
        Et += __shfl_xor_sync(0xffffffffu, Et, o);
        Ez += __shfl_xor_sync(0xffffffffu, Ez, o);
    }
    // weights w_j = a 2^(t_j c - G_t) + b 2^(z_j c - G_z) against the row references
    const float a = (Et > 0.f) ? p.beta / Et : 0.f;
    const float b = (Ez > 0.f) ? (1.f - p.beta) / Ez : 0.f;
    const double mass = double(a) * double(rt) + double(b) * double(rz);
    const double incl = warp_incl_scan_f64(mass);
    const double W = __shfl_sync(0xffffffffu, incl, 31);
    const double tau = double(p.uniforms[row]) * W;
    int mode = 0, piece;  // mode 0: inverse CDF; 1: the largest j with w_j > 0
    double run = 0.0;
    const unsigned h = __ballot_sync(0xffffffffu, incl - mass <= tau && incl > tau);
    if (h) {
        piece = __ffs(h) - 1;
        run = __shfl_sync(0xffffffffu, incl - mass, piece);
    } else {
        mode = 1;
        const unsigned pos = __ballot_sync(0xffffffffu, mass > 0.0);
        piece = pos ? 31 - __clz(pos) : 0;
    }
    // a row without mass: its logits are -inf, and so are x c - 0
    const float Gt_ref = (Gt == kNegInf) ? 0.f : Gt, Gz_ref = (Gz == kNegInf) ? 0.f : Gz;
    const int pw = piece / kPieces, pg = piece % kPieces;
    const int c0 = range_lo(pw), c1 = range_lo(pw + 1);
    const int s_end = min((pg + 1) * per_piece, steps);
    int pick = -1, last_pos = -1;
    double gap = 0.0;
    bool found = false;
    for (int st = pg * per_piece; st < s_end; ++st) {  // warp-uniform trip count
        const int ci = c0 + st * 32 + lane;
        float z[kW], t[kW], w[kW];
        unpack_raw<In, kW>(ci < c1 ? load_chunk(zrow, ci) : none, z);
        unpack_raw<In, kW>(ci < c1 ? load_chunk(trow, ci) : none, t);
#pragma unroll
        for (int e = 0; e < kW; ++e) {
            const float pt = ex2(fmaf(t[e], c, -Gt_ref));
            const float qz = ex2(fmaf(z[e], c, -Gz_ref));
            w[e] = fmaf(a, pt, b * qz);
            if (w[e] > 0.f) last_pos = ci * kW + e;
        }
        double mine = 0.0;
#pragma unroll
        for (int e = 0; e < kW; ++e) mine += double(w[e]);
        const double wincl = warp_incl_scan_f64(mine);
        if (mode == 0) {
            const double excl = run + wincl - mine;
            const unsigned hh = __ballot_sync(0xffffffffu, excl <= tau && excl + mine > tau);
            if (hh) {
                if (lane == __ffs(hh) - 1) {
                    double C = excl;
                    for (int e = 0; e < kW; ++e) {
                        const double Cprev = C;
                        C += double(w[e]);
                        if (C > tau) {
                            pick = ci * kW + e;
                            gap = fmin(C - tau, tau - Cprev) / W;
                            break;
                        }
                    }
                    if (pick < 0) {  // the lane's entries pass tau only after rounding
                        pick = last_pos;
                        gap = 0.0;
                    }
                }
                found = true;
            }
        }
        if (found) break;
        run += __shfl_sync(0xffffffffu, wincl, 31);
    }
    if (!found) {  // mode 1, or rounding left tau past the piece: the largest j with w_j > 0
        int lp = last_pos;
        for (int o = 16; o > 0; o >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
        if (lane == 0) {
            pick = (lp >= 0) ? lp : c0 * kW;
            gap = (mode == 1) ? (W - tau) / W : 0.0;
        }
    }
    if (pick >= 0) {
        p.tokens[row] = pick;
        if (p.cdf_gap) p.cdf_gap[row] = float(gap);
    }
}

}  // namespace osd

extern "C" osd_status osd_mixed_sample(const void* draft_logits, const void* target_logits, osd_dtype dtype, int N,
                                       int V, int64_t d_stride, int64_t t_stride, const float* uniforms, float beta,
                                       float temperature, int32_t* tokens, float* cdf_gap, int32_t* status,
                                       void* stream) {
    using namespace osd;
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    if (N < 0 || V < 1 || d_stride < 0 || t_stride < 0) return OSD_ERR_INVALID_ARG;
    if (!(beta >= 0.f && beta <= 1.f)) return OSD_ERR_INVALID_ARG;
    if (!(temperature > 0.f) || !std::isfinite(temperature)) return OSD_ERR_INVALID_ARG;
    if (V > OSD_VERIFY_MAX_V) return OSD_ERR_UNSUPPORTED;
    const size_t es = dtype_size(dtype);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (status && !aligned_to(status, 4)) return OSD_ERR_INVALID_ARG;
    if (status) {  // no wait in this kernel can run out: the status is OSD_OK once the launch is queued
        const cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
        if (e != cudaSuccess) return OSD_ERR_CUDA;
    }
    if (N == 0) return OSD_OK;
    if (!draft_logits || !target_logits || !uniforms || !tokens) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(draft_logits, es) || !aligned_to(target_logits, es) || !aligned_to(uniforms, 4) ||
        !aligned_to(tokens, 4) || (cdf_gap && !aligned_to(cdf_gap, 4)))
        return OSD_ERR_INVALID_ARG;
    auto row_ok = [&](int64_t stride) { return N <= 1 || (stride * int64_t(es)) % 16 == 0; };
    const bool vec = aligned_to(draft_logits, 16) && aligned_to(target_logits, 16) && row_ok(d_stride) &&
                     row_ok(t_stride);
    MixParams mp;
    mp.draft = draft_logits;
    mp.target = target_logits;
    mp.V = V;
    mp.dstride = d_stride;
    mp.tstride = t_stride;
    mp.uniforms = uniforms;
    mp.beta = beta;
    mp.c = static_cast<float>(1.4426950408889634074 / static_cast<double>(temperature));
    mp.tokens = tokens;
    mp.cdf_gap = cdf_gap;
    const dim3 grid(static_cast<unsigned>(N)), block(kMixThreads);
    cudaError_t e;
    if (dtype == OSD_BF16)
        e = vec ? launch(mixed_sample_kernel<__nv_bfloat16, true>, grid, block, 0, s, 1, mp)
                : launch(mixed_sample_kernel<__nv_bfloat16, false>, grid, block, 0, s, 1, mp);
    else
        e = vec ? launch(mixed_sample_kernel<float, true>, grid, block, 0, s, 1, mp)
                : launch(mixed_sample_kernel<float, false>, grid, block, 0, s, 1, mp);
    return from_cuda(e);
}
