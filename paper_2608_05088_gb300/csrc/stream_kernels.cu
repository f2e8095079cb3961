// stream_kernels.cu -- standalone launches of the HBM-bound stages of the
// MALT / MALTER step (stats, finalize, prescale, norms, scalars, apply; the
// block bodies and their paper references are in stream_blocks.cuh), plus
// pointer binding and the bounded-wait probe.
//
// All reductions run in a fixed order (no atomics), so a step is bitwise
// reproducible.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"
#include "stream_blocks.cuh"

namespace malt {

namespace {

__device__ __forceinline__ int find_mat(const int32_t* __restrict__ pref, int nmat, int32_t x) {
    int lo = 0, hi = nmat - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(pref + mid) <= x) lo = mid; else hi = mid - 1;
    }
    return lo;
}

}  // namespace

// ---------------------------------------------------------------- binding
__global__ void bind_kernel(const __grid_constant__ BindParams P, UserPtrs* __restrict__ table) {
    const int i = threadIdx.x;
    if (i < P.count) table[P.offset + i] = P.p[i];
}

// ------------------------------------------------------------ pad / unpad
// One block copies kPadRows rows of one matrix (one warp per row, lanes along
// the row); the matrix's first block also copies l and r.
template <typename T>
__device__ __forceinline__ void copy_row(const T* __restrict__ src, T* __restrict__ dst, int n,
                                         int lane) {
    for (int j = lane; j < n; j += 32) dst[j] = src[j];
}

template <bool kIn>
__global__ void __launch_bounds__(256) pad_kernel(const __grid_constant__ PadParams P) {
    int k = 0;
    while (k + 1 < P.count && P.e[k + 1].block_begin <= static_cast<int32_t>(blockIdx.x)) ++k;
    const PadEntry& e = P.e[k];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = (static_cast<int>(blockIdx.x) - e.block_begin) * kPadRows + warp;
    if (row < e.m) {
        const size_t u = static_cast<size_t>(row) * e.n;      // caller layout, ld = n
        const size_t q = static_cast<size_t>(row) * e.n8;     // padded layout, ld = n8
        if (kIn) {
            if (e.w_bf16)
                copy_row(static_cast<const uint16_t*>(e.w_user) + u, static_cast<uint16_t*>(e.w_pad) + q, e.n, lane);
            else
                copy_row(static_cast<const float*>(e.w_user) + u, static_cast<float*>(e.w_pad) + q, e.n, lane);
            if (e.g_bf16)
                copy_row(static_cast<const uint16_t*>(e.g_user) + u, static_cast<uint16_t*>(e.g_pad) + q, e.n, lane);
            else
                copy_row(static_cast<const float*>(e.g_user) + u, static_cast<float*>(e.g_pad) + q, e.n, lane);
            copy_row<float>(e.m_user + u, e.m_pad + q, e.n, lane);
        } else {
            if (e.w_bf16) {
                copy_row(static_cast<const uint16_t*>(e.w_pad) + q, static_cast<uint16_t*>(e.w_user) + u, e.n, lane);
            } else {
                const float* src = static_cast<const float*>(e.w_pad) + q;
                copy_row(src, static_cast<float*>(e.w_user) + u, e.n, lane);
                if (e.wcopy_user != nullptr) {
                    __nv_bfloat16* c = static_cast<__nv_bfloat16*>(e.wcopy_user) + u;
                    for (int j = lane; j < e.n; j += 32) c[j] = __float2bfloat16_rn(src[j]);
                }
            }
            copy_row<float>(e.m_pad + q, e.m_user + u, e.n, lane);
        }
    }
    if (static_cast<int>(blockIdx.x) == e.block_begin) {
        for (int i = threadIdx.x; i < e.m; i += blockDim.x) {
            if (kIn) e.l_pad[i] = e.l_user[i]; else e.l_user[i] = e.l_pad[i];
        }
        for (int j = threadIdx.x; j < e.n; j += blockDim.x) {
            if (kIn) e.r_pad[j] = e.r_user[j]; else e.r_user[j] = e.r_pad[j];
        }
    }
}

// ------------------------------------------------------------------ stats
// The streaming kernels' minimum resident blocks per SM (statistics 3,
// prescale 5 for wide matrices and 4 for tall ones, apply 8) trade registers
// for resident warps: more warps per SM kept more of HBM busy than more loads
// in flight per thread did.
template <bool kStats>
__global__ void __launch_bounds__(256, 3)
stats_kernel(const MatDesc* __restrict__ mats, const UserPtrs* __restrict__ ptrs,
             const int32_t* __restrict__ pref, int nmat, float mu1) {
    __shared__ __align__(16) float colsh[8 * kStatCols];
    const int g = find_mat(pref, nmat, blockIdx.x);
    blk::stats_block<kStats>(mats[g], ptrs[g], blockIdx.x - __ldg(pref + g), mu1, threadIdx.x,
                             colsh);
}

// --------------------------------------------------------------- finalize
__global__ void __launch_bounds__(256)
finalize_kernel(const MatDesc* __restrict__ mats, const UserPtrs* __restrict__ ptrs,
                const int32_t* __restrict__ pref, int nmat, int32_t total,
                float mu2, float eps, long long* tcount, int identity) {
    const int32_t x = blockIdx.x * blockDim.x + threadIdx.x;
    if (x == 0) *tcount += 1;                 // 1-based step count
    if (x >= total) return;
    const int g = find_mat(pref, nmat, x);
    blk::finalize_entry(mats[g], ptrs[g], x - __ldg(pref + g), mu2, eps, identity);
}

// --------------------------------------------------------------- prescale
// One launch for the wide matrices, one for the tall ones (their NS frame is
// Mt^T, written through shared-memory transposes): ids lists the launch's
// matrices and pref its block prefix.
__global__ void __launch_bounds__(256, 5)
prescale_wide_kernel(const MatDesc* __restrict__ mats, const UserPtrs* __restrict__ ptrs,
                     const int32_t* __restrict__ ids, const int32_t* __restrict__ pref, int count,
                     int malter) {
    __shared__ float2 red[8];
    const int32_t x = blockIdx.x;
    const int k = find_mat(pref, count, x);
    const int g = __ldg(ids + k);
    blk::prescale_block<false>(mats[g], ptrs[g], x - __ldg(pref + k), malter, threadIdx.x, nullptr,
                               red);
}

__global__ void __launch_bounds__(256, 4)
prescale_tall_kernel(const MatDesc* __restrict__ mats, const UserPtrs* __restrict__ ptrs,
                     const int32_t* __restrict__ ids, const int32_t* __restrict__ pref, int count,
                     int32_t base, int malter) {
    __shared__ __align__(16) float tile[blk::kPreTileFloats];
    __shared__ float2 red[8];
    const int32_t x = base + static_cast<int32_t>(blockIdx.x);   // pref continues the wide launch's
    const int k = find_mat(pref, count, x);
    const int g = __ldg(ids + k);
    blk::prescale_block<true>(mats[g], ptrs[g], x - __ldg(pref + k), malter, threadIdx.x, tile,
                              red);
}

// ------------------------------------------------------------------ norms
__global__ void __launch_bounds__(256)
norms_kernel(const MatDesc* __restrict__ mats, MatScalars* __restrict__ scal, float ns_eps,
             int malter) {
    __shared__ float red[32];
    const int g = blockIdx.x;
    blk::norms_matrix(mats[g], scal + g, ns_eps, malter, threadIdx.x, red);
}

// ---------------------------------------------------------------- scalars
__global__ void __launch_bounds__(blk::kScalarThreads)
scalars_kernel(const MatDesc* __restrict__ mats, MatScalars* __restrict__ scal,
               const long long* __restrict__ tcount, StepHyper hp) {
    __shared__ float red[32];
    const int g = blockIdx.x;
    blk::scalars_matrix(mats[g], scal + g, tcount, hp, threadIdx.x, red);
}

// ------------------------------------------------------------------ apply
__global__ void __launch_bounds__(256, 8)
apply_kernel(const MatDesc* __restrict__ mats, const UserPtrs* __restrict__ ptrs,
             const MatScalars* __restrict__ scal, const int32_t* __restrict__ pref, int nmat,
             float decay) {
    const int g = find_mat(pref, nmat, blockIdx.x);
    blk::apply_block(mats[g], ptrs[g], blockIdx.x - __ldg(pref + g), scal[g].scale, decay,
                     threadIdx.x);
}

// ------------------------------------------------------------- wait probe
// One thread waits on an mbarrier that nothing ever arrives on, for at most
// budget_ns, and records whether the wait gave up.
__global__ void wait_probe_kernel(int32_t* status, uint64_t budget_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const bool ok = mbar_wait_bounded(&bar, 0, budget_ns, nullptr);
        *status = ok ? 0 : kStatusTimeout;
    }
}

// ----------------------------------------------------------------- guards
constexpr uint32_t kGuardWord = 0xA5C3E10Fu;

// One block per guard region, one thread per 32-bit word.
__global__ void guard_kernel(uint8_t* base, const uint64_t* __restrict__ offsets, bool check,
                             unsigned long long* bad) {
    uint32_t* g = reinterpret_cast<uint32_t*>(base + offsets[blockIdx.x]);
    const int i = threadIdx.x;
    if (!check) {
        g[i] = kGuardWord;
        return;
    }
    const uint32_t diff = g[i] ^ kGuardWord;
    int nbytes = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) nbytes += ((diff >> (8 * k)) & 0xffu) != 0;
    if (nbytes != 0) atomicAdd(bad, static_cast<unsigned long long>(nbytes));
}

// ------------------------------------------------------------------ launch
cudaError_t launch_bind(const BindParams& P, UserPtrs* table, cudaStream_t s) {
    bind_kernel<<<1, kBindChunk, 0, s>>>(P, table);
    return cudaGetLastError();
}

cudaError_t launch_pad(const PadParams& P, int32_t blocks, bool in, cudaStream_t s) {
    if (in)
        pad_kernel<true><<<blocks, 256, 0, s>>>(P);
    else
        pad_kernel<false><<<blocks, 256, 0, s>>>(P);
    return cudaGetLastError();
}

cudaError_t launch_stats(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                         int nmat, int32_t blocks, float mu1, int with_stats, cudaStream_t s) {
    if (with_stats)
        stats_kernel<true><<<blocks, 256, 0, s>>>(mats, ptrs, pref, nmat, mu1);
    else
        stats_kernel<false><<<blocks, 256, 0, s>>>(mats, ptrs, pref, nmat, mu1);
    return cudaGetLastError();
}

cudaError_t launch_finalize(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                            int nmat, int32_t total, float mu2, float eps, long long* tcount,
                            int identity, cudaStream_t s) {
    const int blocks = (total + 255) / 256 > 0 ? (total + 255) / 256 : 1;
    finalize_kernel<<<blocks, 256, 0, s>>>(mats, ptrs, pref, nmat, total, mu2, eps, tcount,
                                          identity);
    return cudaGetLastError();
}

cudaError_t launch_prescale(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* ids,
                            const int32_t* pref, int wide, int32_t wide_blocks, int tall,
                            int32_t tall_blocks, int malter, cudaStream_t s) {
    if (wide > 0 && wide_blocks > 0) {
        prescale_wide_kernel<<<wide_blocks, 256, 0, s>>>(mats, ptrs, ids, pref, wide, malter);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (tall > 0 && tall_blocks > 0) {
        prescale_tall_kernel<<<tall_blocks, 256, 0, s>>>(mats, ptrs, ids + wide, pref + wide, tall,
                                                         wide_blocks, malter);
        return cudaGetLastError();
    }
    return cudaSuccess;
}

cudaError_t launch_norms(const MatDesc* mats, MatScalars* scal, int nmat, float ns_eps,
                         int malter, cudaStream_t s) {
    norms_kernel<<<nmat, 256, 0, s>>>(mats, scal, ns_eps, malter);
    return cudaGetLastError();
}

cudaError_t launch_scalars(const MatDesc* mats, MatScalars* scal, const long long* tcount,
                           int nmat, const StepHyper& hp, cudaStream_t s) {
    scalars_kernel<<<nmat, blk::kScalarThreads, 0, s>>>(mats, scal, tcount, hp);
    return cudaGetLastError();
}

cudaError_t launch_apply(const MatDesc* mats, const UserPtrs* ptrs, const MatScalars* scal,
                         const int32_t* pref, int nmat, int32_t blocks, float decay,
                         cudaStream_t s) {
    apply_kernel<<<blocks, 256, 0, s>>>(mats, ptrs, scal, pref, nmat, decay);
    return cudaGetLastError();
}


cudaError_t launch_guards(void* base, const uint64_t* offsets, int32_t n, bool check,
                          unsigned long long* bad, cudaStream_t s) {
    guard_kernel<<<n, static_cast<int>(kGuardBytes / 4), 0, s>>>(static_cast<uint8_t*>(base), offsets,
                                                                 check, bad);
    return cudaGetLastError();
}

cudaError_t launch_wait_probe(int32_t* status, uint64_t budget_ns, cudaStream_t s) {
    wait_probe_kernel<<<1, 32, 0, s>>>(status, budget_ns);
    return cudaGetLastError();
}

}  // namespace malt
