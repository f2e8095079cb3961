// stream_blocks.cuh -- the HBM-bound stages of the MALT / MALTER step as
// block-level device functions of 256 threads (tid 0..255).  The kernels of
// stream_kernels.cu run one call per CUDA block; malt_stats_noalloc
// (noalloc.cu) runs the statistics and finalize blocks of one matrix on its
// own scratch.  Every multiply-add that decides a rounding is an explicit
// fmaf / fma, so each block computes bitwise the same result in every
// translation unit it is compiled into.
//
//   stats     Algorithm 1, M_t / l_t / r_t lines: one pass over G and M that
//             updates the momentum and writes per-tile partial sums of G^2 for
//             every row and every column (eq. dp_preconditioner).
//   finalize  l, r EMAs from the partials and L = (l+eps)^(-1/8),
//             R = (r+eps)^(-1/8) (Algorithm 1, L_t / R_t line).
//   prescale  Mt = L M R (Algorithm 1, Mt line), written as bf16 in the
//             Newton-Schulz frame (transposed when m > n), with partial sums
//             of Mt^2 (and of (L G R)^2 for MALTER, Algorithm 2 nu_t line).
//   norms     ||Mt||_F and ||L G R||_F^2 per matrix from those partials.
//   scalars   ||O||_F, ||D||_F, MALTER's nu and alpha (Section 3.5) and the
//             grafted scale lr * alpha * ||O|| / (||D|| + eps) per matrix.
//   apply     W <- (1 - lr wd) W - scale * L O R (Algorithm 1, W_t line), with
//             O in W's layout, streamed contiguously; for fp32 master weights
//             also their bf16 copy, when the caller registered one.
#pragma once
#include <cuda_bf16.h>
#include <cstdint>

#include "common.cuh"

namespace malt {
namespace blk {

constexpr int kThreads = 256;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Compensated (Kahan) summation in fp32: the error of the total stays near
// one rounding however many terms are added (no reassociation: the library
// is compiled without fast-math).
struct CompensatedSum {
    float s = 0.f, c = 0.f;
    __device__ __forceinline__ void add(float x) {
        const float y = x - c;
        const float t = s + y;
        c = (t - s) - y;
        s = t;
    }
};

// Sum of v over the first nthreads threads (a multiple of 32) in a fixed
// order; every thread of the block calls it, the result is valid in tid 0.
__device__ __forceinline__ float block_sum(float v, float* sh /* >= 32 */, int tid, int nthreads) {
    v = warp_sum(v);
    const int w = tid >> 5, lane = tid & 31;
    if (lane == 0 && tid < nthreads) sh[w] = v;
    __syncthreads();
    float s = 0.f;
    if (tid == 0) {
        const int nw = nthreads >> 5;
        for (int i = 0; i < nw; ++i) s += sh[i];
    }
    __syncthreads();
    return s;
}

// Load paths: read-only cache, plain (L1 and L2), L2 only.
enum LoadPath { kLdRO = 0, kLdPlain = 1, kLdL2 = 2 };

template <int kPath>
__device__ __forceinline__ uint4 ld_u4(const void* p) {
    const uint4* q = reinterpret_cast<const uint4*>(p);
    return kPath == kLdRO ? __ldg(q) : kPath == kLdL2 ? __ldcg(q) : *q;
}

template <int kPath>
__device__ __forceinline__ float4 ld_f4(const float* p) {
    const float4* q = reinterpret_cast<const float4*>(p);
    return kPath == kLdRO ? __ldg(q) : kPath == kLdL2 ? __ldcg(q) : *q;
}

template <int kPath>
__device__ __forceinline__ float ld_f(const float* p) {
    return kPath == kLdRO ? __ldg(p) : kPath == kLdL2 ? __ldcg(p) : *p;
}

// 8 consecutive elements (bf16 or fp32) at element offset off, as floats.
template <int kPath = kLdRO>
__device__ __forceinline__ void load8(const void* base, bool bf16, size_t off, float (&v)[8]) {
    if (bf16) {
        const uint4 u = ld_u4<kPath>(static_cast<const __nv_bfloat16*>(base) + off);
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 f = __bfloat1622float2(h[k]);
            v[2 * k] = f.x;
            v[2 * k + 1] = f.y;
        }
    } else {
        const float* p = static_cast<const float*>(base) + off;
        const float4 a = ld_f4<kPath>(p), b = ld_f4<kPath>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
}

__device__ __forceinline__ uint4 pack8_bf16(const float (&v)[8]) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) h[k] = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
    return u;
}

// ------------------------------------------------------------------ stats
// Block `local` = kStatRows x kStatCols of W: warp w owns 8 rows, lane owns 8
// consecutive columns.  Row sums reduce across the warp; column sums
// accumulate in registers over the warp's rows, then across the 8 warps in
// shared memory (colsh: 8 x kStatCols floats).  kStats = false (Muon through
// the same engine): momentum only.  G is never written by the library, so it
// is read through the read-only path.
constexpr int kStatRowsPerWarp = kStatRows / 8;
constexpr int kStatBatch = 4;

template <bool kStats>
__device__ __forceinline__ void stats_block(const MatDesc& d, const UserPtrs& up, int local,
                                            float mu1, int tid, float* colsh) {
    const int m = d.m, n = d.n;
    const int rb = local / d.stat_cb, cb = local - rb * d.stat_cb;
    const int warp = tid >> 5, lane = tid & 31;
    const int col = cb * kStatCols + lane * 8;
    const bool colok = col < n;
    const int row0 = rb * kStatRows + warp * kStatRowsPerWarp;
    const bool gbf = d.g_bf16 != 0;
    float* __restrict__ Mp = up.m;
    const float om = 1.f - mu1;

    float csum[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) csum[j] = 0.f;
    float myrow = 0.f;

#pragma unroll
    for (int rb4 = 0; rb4 < kStatRowsPerWarp; rb4 += kStatBatch) {
        float gv[kStatBatch][8], mv[kStatBatch][8];
        bool ok[kStatBatch];
#pragma unroll
        for (int u = 0; u < kStatBatch; ++u) {
            const int row = row0 + rb4 + u;
            ok[u] = colok && row < m;
            if (ok[u]) {
                const size_t off = static_cast<size_t>(row) * n + col;
                load8<kLdRO>(up.g, gbf, off, gv[u]);
                const float4* mp = reinterpret_cast<const float4*>(Mp + off);
                const float4 a = mp[0], b = mp[1];
                mv[u][0] = a.x; mv[u][1] = a.y; mv[u][2] = a.z; mv[u][3] = a.w;
                mv[u][4] = b.x; mv[u][5] = b.y; mv[u][6] = b.z; mv[u][7] = b.w;
            } else {
#pragma unroll
                for (int j = 0; j < 8; ++j) { gv[u][j] = 0.f; mv[u][j] = 0.f; }
            }
        }
#pragma unroll
        for (int u = 0; u < kStatBatch; ++u) {
            float rs = 0.f;
            float nm[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float gj = gv[u][j];
                nm[j] = fmaf(mu1, mv[u][j], om * gj);
                // explicit fused multiply-adds: the same rounding in every
                // compilation of this block
                rs = fmaf(gj, gj, rs);
                csum[j] = fmaf(gj, gj, csum[j]);
            }
            if (ok[u]) {
                const size_t off = static_cast<size_t>(row0 + rb4 + u) * n + col;
                float4* mp = reinterpret_cast<float4*>(Mp + off);
                mp[0] = make_float4(nm[0], nm[1], nm[2], nm[3]);
                mp[1] = make_float4(nm[4], nm[5], nm[6], nm[7]);
            }
            if (kStats) {
                rs = warp_sum(rs);
                if (lane == rb4 + u) myrow = rs;
            }
        }
    }
    if (!kStats) return;
    if (lane < kStatRowsPerWarp && row0 + lane < m)
        d.rowpart[static_cast<size_t>(cb) * m + row0 + lane] = myrow;

    float4* cs = reinterpret_cast<float4*>(colsh + warp * kStatCols + lane * 8);
    cs[0] = make_float4(csum[0], csum[1], csum[2], csum[3]);
    cs[1] = make_float4(csum[4], csum[5], csum[6], csum[7]);
    __syncthreads();
    const int c = tid;
    const int gc = cb * kStatCols + c;
    if (gc < n) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) s += colsh[w * kStatCols + c];
        d.colpart[static_cast<size_t>(rb) * n + gc] = s;
    }
}

// --------------------------------------------------------------- finalize
// Entry `local` of the matrix's m + n statistics: row i = local (< m) or
// column j = local - m.  identity (Muon): L = R = 1, statistics untouched.
// The per-block partial sums are added with compensation: a row of a matrix
// near the size limit has 8192 of them (a column up to 262144), which a plain
// fp32 sum in sequence would carry to a relative error near 1e-5.
__device__ __forceinline__ void finalize_entry(const MatDesc& d, const UserPtrs& up, int local,
                                               float mu2, float eps, int identity) {
    constexpr int P = kLdPlain;
    if (identity) {
        if (local < d.m) d.L[local] = 1.f; else d.R[local - d.m] = 1.f;
        return;
    }
    if (local < d.m) {
        const int i = local;
        CompensatedSum s;
        for (int cb = 0; cb < d.stat_cb; ++cb) s.add(ld_f<P>(d.rowpart + static_cast<size_t>(cb) * d.m + i));
        const float l = fmaf(mu2, up.l[i], (1.f - mu2) * s.s);
        up.l[i] = l;
        d.L[i] = powf(l + eps, -0.125f);
    } else {
        const int j = local - d.m;
        CompensatedSum s;
        for (int rb = 0; rb < d.stat_rb; ++rb) s.add(ld_f<P>(d.colpart + static_cast<size_t>(rb) * d.n + j));
        const float r = fmaf(mu2, up.r[j], (1.f - mu2) * s.s);
        up.r[j] = r;
        d.R[j] = powf(r + eps, -0.125f);
    }
}

// --------------------------------------------------------------- prescale
// Block `local` = kPreRows x kPreCols of Mt.  A wide matrix is streamed like
// the statistics pass (warp w owns 8 rows, lane 8 consecutive columns,
// kPreBatch rows of loads in flight) and written as bf16 in place of its NS
// frame; a
// tall matrix's NS frame is Mt^T, so its block walks four 64 x 64 sub-tiles
// through shared memory and writes each transposed.
// tile: two 64 x 64 float buffers (kPreTileFloats, 16-byte aligned), used in
// turn.  Row r of a buffer holds its 16 float4 chunks XOR-permuted by
// (r / 8) mod 8, so that both the row-wise float4 writes and the column-wise
// reads (eight rows 8 apart per warp) hit 32 distinct banks.
// red: 8 float2.
constexpr int kPreTileFloats = 2 * 64 * 64;
// Loads in flight per thread: rows of a wide block loaded together, and
// sub-tiles of a tall block loaded ahead.  Small, so that the wide blocks fit
// 5 per SM in 48 registers and the tall ones 4 per SM in 64 registers without
// spilling: resident warps keep more of HBM busy than loads in flight per
// thread (four rows and two sub-tiles spilled at 4 blocks per SM and streamed
// 7 % slower on GPT-2 Large, 14 % on a 16384 x 4096 matrix; one row at 6
// blocks per SM was 2 % slower on GPT-2 Large and 5-10 % on wide stress
// matrices).
constexpr int kPreBatch = 2;
constexpr int kPreAhead = 1;
template <bool kTall>
__device__ __forceinline__ void prescale_block(const MatDesc& d, const UserPtrs& up, int local,
                                               int malter, int tid, float* tile,
                                               float2* red) {
    constexpr int P = kLdPlain;
    const int m = d.m, n = d.n;
    // A tall matrix's blocks walk down a column band first, so the blocks
    // resident at once write neighbouring pieces of the same X0 rows.
    const int tr = kTall ? local % d.pre_tr : local / d.pre_tc;
    const int tc = kTall ? local / d.pre_tr : local - tr * d.pre_tc;
    const int r0 = tr * kPreRows, c0 = tc * kPreCols;
    const int t = tid, warp = t >> 5, lane = t & 31;
    const float* __restrict__ Lv = d.L;
    const float* __restrict__ Rv = d.R;
    const float* __restrict__ Mp = up.m;
    const bool gbf = d.g_bf16 != 0;
    float s_mt = 0.f, s_lgr = 0.f;

    if constexpr (!kTall) {
        const int col = c0 + lane * 8;
        const bool colok = col < n;
        float rj[8];
        if (colok) {
            const float4 a = ld_f4<P>(Rv + col);
            const float4 b = ld_f4<P>(Rv + col + 4);
            rj[0] = a.x; rj[1] = a.y; rj[2] = a.z; rj[3] = a.w;
            rj[4] = b.x; rj[5] = b.y; rj[6] = b.z; rj[7] = b.w;
        }
        const int row0 = r0 + warp * 8;
#pragma unroll
        for (int rb = 0; rb < 8; rb += kPreBatch) {
            float mv[kPreBatch][8], li[kPreBatch];
            bool ok[kPreBatch];
#pragma unroll
            for (int u = 0; u < kPreBatch; ++u) {
                const int row = row0 + rb + u;
                ok[u] = colok && row < m;
                li[u] = 0.f;
                if (ok[u]) {
                    const size_t off = static_cast<size_t>(row) * n + col;
                    const float4 a = ld_f4<P>(Mp + off);
                    const float4 b = ld_f4<P>(Mp + off + 4);
                    mv[u][0] = a.x; mv[u][1] = a.y; mv[u][2] = a.z; mv[u][3] = a.w;
                    mv[u][4] = b.x; mv[u][5] = b.y; mv[u][6] = b.z; mv[u][7] = b.w;
                    li[u] = ld_f<P>(Lv + row);
                }
            }
#pragma unroll
            for (int u = 0; u < kPreBatch; ++u) {
                if (!ok[u]) continue;
                const int row = row0 + rb + u;
                const size_t off = static_cast<size_t>(row) * n + col;
                float v[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    v[j] = li[u] * mv[u][j] * rj[j];
                    s_mt = fmaf(v[j], v[j], s_mt);
                }
                *reinterpret_cast<uint4*>(d.X0 + off) = pack8_bf16(v);
                if (malter) {
                    float gv[8];
                    load8<kLdRO>(up.g, gbf, off, gv);
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const float a = li[u] * gv[j] * rj[j];
                        s_lgr = fmaf(a, a, s_lgr);
                    }
                }
            }
        }
    } else {
        // Keep the M loads of the next sub-tile in flight while this one goes
        // through shared memory: each 64 x 64 sub-tile is four rows of one
        // float4 per thread, loaded kPreAhead sub-tiles ahead.
        const int cc = (t & 15) * 4;
        constexpr int kSubs = kPreCols / 64;
        float li[4];
#pragma unroll
        for (int pass = 0; pass < 4; ++pass) {
            const int row = r0 + pass * 16 + (t >> 4);
            li[pass] = row < m ? ld_f<P>(Lv + row) : 0.f;
        }
        auto load_sub = [&](int sub, float4 (&dst)[4]) {
            const int col = c0 + sub * 64 + cc;
#pragma unroll
            for (int pass = 0; pass < 4; ++pass) {
                const int row = r0 + pass * 16 + (t >> 4);
                dst[pass] = (row < m && col < n)
                                ? ld_f4<P>(Mp + static_cast<size_t>(row) * n + col)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
            }
        };
        float4 mq[kPreAhead][4];
#pragma unroll
        for (int a = 0; a < kPreAhead; ++a) load_sub(a, mq[a]);
#pragma unroll
        for (int sub = 0; sub < kSubs; ++sub) {
            const int cs = c0 + sub * 64;
            if (cs >= n) break;                          // uniform across the block
            const int col = cs + cc;
            float* __restrict__ tb = tile + (sub & 1) * (64 * 64);
            float4 R4 = make_float4(0.f, 0.f, 0.f, 0.f);
            if (col < n) R4 = ld_f4<P>(Rv + col);
#pragma unroll
            for (int pass = 0; pass < 4; ++pass) {
                const int rr = pass * 16 + (t >> 4);
                const int row = r0 + rr;
                float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f;
                if (row < m && col < n) {
                    const size_t off = static_cast<size_t>(row) * n + col;
                    const float Li = li[pass];
                    const float4 q = mq[sub % kPreAhead][pass];
                    v0 = Li * q.x * R4.x; v1 = Li * q.y * R4.y;
                    v2 = Li * q.z * R4.z; v3 = Li * q.w * R4.w;
                    // explicit fused multiply-adds: the same rounding wherever
                    // this block is compiled
                    s_mt = fmaf(v3, v3, fmaf(v2, v2, fmaf(v1, v1, fmaf(v0, v0, s_mt))));
                    if (malter) {
                        float gq[4];
                        if (gbf) {
                            const uint2 u = *reinterpret_cast<const uint2*>(
                                static_cast<const __nv_bfloat16*>(up.g) + off);
                            const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
                            const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
                            gq[0] = a.x; gq[1] = a.y; gq[2] = b.x; gq[3] = b.y;
                        } else {
                            const float4 gf = *reinterpret_cast<const float4*>(
                                static_cast<const float*>(up.g) + off);
                            gq[0] = gf.x; gq[1] = gf.y; gq[2] = gf.z; gq[3] = gf.w;
                        }
                        const float a0 = Li * gq[0] * R4.x, a1 = Li * gq[1] * R4.y;
                        const float a2 = Li * gq[2] * R4.z, a3 = Li * gq[3] * R4.w;
                        s_lgr = fmaf(a3, a3, fmaf(a2, a2, fmaf(a1, a1, fmaf(a0, a0, s_lgr))));
                    }
                }
                *reinterpret_cast<float4*>(tb + rr * 64 + (((t & 15) ^ ((rr >> 3) & 7)) << 2)) =
                    make_float4(v0, v1, v2, v3);
            }
            if (sub + kPreAhead < kSubs) load_sub(sub + kPreAhead, mq[sub % kPreAhead]);
            // One barrier per sub-tile: the buffer written next was last read
            // two sub-tiles ago, before every thread passed the previous barrier.
            __syncthreads();
            // Output row = column of Mt, 8 consecutive rows of Mt per thread;
            // those rows share one chunk permutation, t mod 8.
            const int seg = (t & 7) * 8, sw = t & 7;
#pragma unroll
            for (int pass = 0; pass < 2; ++pass) {
                const int oc = pass * 32 + (t >> 3);
                const int gcol = cs + oc, grow = r0 + seg;
                if (gcol < n && grow < m) {
                    const int pc = ((((oc >> 2) ^ sw) << 2) | (oc & 3));
                    float v[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) v[j] = tb[(seg + j) * 64 + pc];
                    *reinterpret_cast<uint4*>(d.X0 + static_cast<size_t>(gcol) * m + grow) =
                        pack8_bf16(v);
                }
            }
        }
    }
    // One fixed-order reduction of both partial sums.
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        s_mt += __shfl_xor_sync(0xffffffffu, s_mt, o);
        s_lgr += __shfl_xor_sync(0xffffffffu, s_lgr, o);
    }
    if (lane == 0) red[warp] = make_float2(s_mt, s_lgr);
    __syncthreads();
    if (t == 0) {
        float a = 0.f, b = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            a += red[w].x;
            b += red[w].y;
        }
        d.prepart[2 * local + 0] = a;
        d.prepart[2 * local + 1] = b;
    }
}

// ------------------------------------------------------------------ norms
// ||Mt||_F, 1 / (||Mt||_F + ns_eps) and ||L G R||_F^2 of one matrix (256 threads).
__device__ __forceinline__ void norms_matrix(const MatDesc& d, MatScalars* sc, float ns_eps,
                                             int malter, int tid, float* red) {
    constexpr int P = kLdPlain;
    const int tiles = d.pre_tr * d.pre_tc;
    // each thread's share of the block partials with compensation (512 of
    // them per thread for a matrix near the size limit), then one fp32 tree
    CompensatedSum as, bs;
    for (int i = tid; i < tiles; i += kThreads) {
        as.add(ld_f<P>(d.prepart + 2 * i));
        bs.add(ld_f<P>(d.prepart + 2 * i + 1));
    }
    const float a = block_sum(as.s, red, tid, kThreads);
    const float b = block_sum(bs.s, red, tid, kThreads);
    if (tid == 0) {
        const float nrm = sqrtf(a);
        sc->norm_mt = nrm;
        sc->k = 1.f / (nrm + ns_eps);
        sc->lgr_sq = malter ? b : 0.f;
    }
}

// ---------------------------------------------------------------- scalars
// Graft norms, MALTER's nu and alpha, and the applied scale of one matrix.
// The sums run over the first kScalarThreads threads (the standalone kernel's
// block size), so the result does not depend on who runs it.
constexpr int kScalarThreads = 128;

__device__ __forceinline__ void scalars_matrix(const MatDesc& d, MatScalars* sc,
                                               const long long* tcount, const StepHyper& hp,
                                               int tid, float* red) {
    constexpr int P = kLdPlain;
    CompensatedSum as, bs;
    // One partial per epilogue warp per GEMM tile of the last iteration, each
    // thread's share added with compensation (thousands per thread near the
    // size limit).
    if (tid < kScalarThreads) {
        for (int i = tid; i < kNsPartsPerTile * d.ns_tiles; i += kScalarThreads) {
            as.add(ld_f<P>(d.nspart + 2 * i));
            bs.add(ld_f<P>(d.nspart + 2 * i + 1));
        }
    }
    const float a = block_sum(as.s, red, tid, kScalarThreads);
    const float b = block_sum(bs.s, red, tid, kScalarThreads);
    if (tid == 0) {
        MatScalars s;
        {
            const float4 lo = ld_f4<P>(reinterpret_cast<const float*>(sc));
            const float4 hi = ld_f4<P>(reinterpret_cast<const float*>(sc) + 4);
            s.k = lo.x; s.norm_mt = lo.y; s.lgr_sq = lo.z; s.scale = lo.w;
            s.norm_o = hi.x; s.norm_d = hi.y; s.alpha = hi.z; s.nu = hi.w;
        }
        const double norm_o = sqrt(static_cast<double>(a));
        const double norm_d = sqrt(static_cast<double>(b));
        double alpha = 1.0;
        if (hp.malter) {
            // Algorithm 2, nu_t line; alpha_t as displayed in Section 3.5.
            const double t = static_cast<double>(*tcount);
            // One explicit fma, so that no compilation of this block
            // contracts the two products differently.
            const double nu = fma(static_cast<double>(hp.mu2), static_cast<double>(s.nu),
                                  (1.0 - static_cast<double>(hp.mu2)) * s.lgr_sq);
            const double bc = sqrt(1.0 - pow(static_cast<double>(hp.mu2), t)) /
                              (1.0 - pow(static_cast<double>(hp.mu1), t) + hp.eps);
            alpha = bc * s.norm_mt / (sqrt(nu) + hp.eps);
            s.nu = static_cast<float>(nu);
        }
        s.norm_o = static_cast<float>(norm_o);
        s.norm_d = static_cast<float>(norm_d);
        s.alpha = static_cast<float>(alpha);
        s.scale = static_cast<float>(hp.lr * alpha * norm_o / (norm_d + hp.eps));
        *sc = s;
    }
}

// ------------------------------------------------------------------ apply
template <int P>
__device__ __forceinline__ void apply8(const MatDesc& d, const UserPtrs& up, bool wbf, float s,
                                       float decay, int i, int j, const float (&o)[8]) {
    const size_t e = static_cast<size_t>(i) * d.n + j;
    const float Li = ld_f<P>(d.L + i);
    const float4 r0 = ld_f4<P>(d.R + j);
    const float4 r1 = ld_f4<P>(d.R + j + 4);
    const float rj[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
    float w[8];
    if (wbf) {
        const uint4 u = *reinterpret_cast<const uint4*>(static_cast<__nv_bfloat16*>(up.w) + e);
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 f = __bfloat1622float2(h[k]);
            w[2 * k] = f.x;
            w[2 * k + 1] = f.y;
        }
    } else {
        const float4* wp = reinterpret_cast<const float4*>(static_cast<float*>(up.w) + e);
        const float4 a = wp[0], b = wp[1];
        w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
        w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
    }
    const float sl = s * Li;
#pragma unroll
    for (int k = 0; k < 8; ++k) w[k] = fmaf(-sl * o[k], rj[k], decay * w[k]);
    if (wbf) {
        *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(up.w) + e) = pack8_bf16(w);
    } else {
        float4* wp = reinterpret_cast<float4*>(static_cast<float*>(up.w) + e);
        wp[0] = make_float4(w[0], w[1], w[2], w[3]);
        wp[1] = make_float4(w[4], w[5], w[6], w[7]);
        // fp32 master weights: the bf16 copy the model computes with
        if (up.wcopy != nullptr)
            *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(up.wcopy) + e) = pack8_bf16(w);
    }
}

// Block `local` of the apply pass: kApplyElems contiguous elements (O is in
// W's layout).  s = the grafted scale.
__device__ __forceinline__ void apply_block(const MatDesc& d, const UserPtrs& up, int local,
                                            float s, float decay, int tid) {
    constexpr int P = kLdPlain;
    constexpr int PO = kLdRO;                     // O: written by an earlier launch
    const int m = d.m, n = d.n;
    const bool wbf = d.w_bf16 != 0;
    const int32_t total = m * n;
    const int32_t e0 = local * kApplyElems;
#pragma unroll 4
    for (int v = 0; v < kApplyElems / (kThreads * 8); ++v) {
        const int32_t e = e0 + (v * kThreads + tid) * 8;
        if (e >= total) break;
        const int i = e / n, j = e - i * n;
        float o[8];
        load8<PO>(d.O, true, static_cast<size_t>(e), o);
        apply8<P>(d, up, wbf, s, decay, i, j, o);
    }
}

}  // namespace blk
}  // namespace malt
