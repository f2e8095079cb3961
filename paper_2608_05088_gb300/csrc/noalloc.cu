// noalloc.cu -- malt_stats_noalloc: the statistics stage of one matrix
// (momentum, row/column statistics and the two diagonal preconditioners)
// without any device allocation.
//
// Some callers cannot allocate device memory at the moment they need this
// work done: code under a framework allocator that owns all device memory and
// forbids allocations behind its back, code in a latency-critical loop that
// must not risk the implicit device synchronisation an allocation may cause,
// and services that reserve all their memory at start-up and may not
// allocate afterwards.  The regular entry points need a workspace from
// malt_init_state; this one keeps its only scratch -- the per-tile partial
// sums of G^2 -- in a fixed array that lives in the library image itself.
// It runs the step's own statistics and finalize blocks, so its results are
// bitwise those of a MALT step on the same matrix.
//
// The array is a file-scope __device__ variable, so every GPU that loads the
// library holds MALT_NOALLOC_SCRATCH_FLOATS floats (4 MiB) of it until the
// process exits.
// Host code never uses the array's name as a pointer (on the host that name
// is only a stand-in): the first call on each device looks up the array's
// device address with cudaGetSymbolAddress, with that device current, and
// later calls reuse it.  That first call should therefore happen before any
// stream capture begins.  All calls share the one array: calls whose kernels
// overlap on the GPU (different streams, or different host threads) race on
// it and must be serialised by the caller.  Every partial sum is written
// before it is read in the same call, so nothing in the array has to start at
// zero and no clearing is needed between calls.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "../../include/malt.h"
#include "common.cuh"
#include "stream_blocks.cuh"

namespace {

using malt::MatDesc;
using malt::UserPtrs;
constexpr int kMaxDevices = 64;

static_assert(MALT_NOALLOC_SCRATCH_FLOATS % 64 == 0, "scratch size must keep 256-byte alignment");

// The scratch array: [col_chunks][m] row partials, then [row_bands][n] column
// partials -- the layout the step keeps in its workspace.
static __device__ __align__(256) float g_noalloc_scratch[MALT_NOALLOC_SCRATCH_FLOATS];

std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};

// Momentum update and per-tile partial sums of G^2 (Algorithm 1, M_t / l_t /
// r_t lines): the statistics block of the step, one kStatRows x kStatCols
// tile of G per CUDA block.
__global__ void __launch_bounds__(256)
noalloc_stats_kernel(const __grid_constant__ MatDesc d, const __grid_constant__ UserPtrs up,
                     float mu1) {
    __shared__ __align__(16) float colsh[8 * malt::kStatCols];
    malt::blk::stats_block<true>(d, up, blockIdx.x, mu1, threadIdx.x, colsh);
}

// EMAs of the statistics and the diagonal preconditioners (Algorithm 1, l_t,
// r_t and L_t / R_t lines): the finalize entry of the step, one thread per
// row or column.
__global__ void __launch_bounds__(256)
noalloc_finalize_kernel(const __grid_constant__ MatDesc d, const __grid_constant__ UserPtrs up,
                        float mu2, float eps) {
    const int x = blockIdx.x * blockDim.x + threadIdx.x;
    if (x < d.m + d.n) malt::blk::finalize_entry(d, up, x, mu2, eps, 0);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Device address of the scratch array on the current device, looked up once.
int scratch_for_current_device(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        std::fprintf(stderr, "malt_stats_noalloc: cudaGetDevice failed: %s\n", cudaGetErrorString(e));
        return MALT_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return MALT_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_ptr[dev] == nullptr) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) {
            std::fprintf(stderr, "malt_stats_noalloc: cudaGetSymbolAddress failed: %s\n",
                         cudaGetErrorString(e));
            return MALT_ERR_CUDA;
        }
        g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_ptr[dev];
    return MALT_OK;
}

}  // namespace

extern "C" int malt_stats_noalloc(const void* g, int32_t g_dtype, float* m, float* l, float* r,
                                  float* L_out, float* R_out, int64_t rows, int64_t cols,
                                  float mu1, float mu2, float eps, void* stream) {
    if (g == nullptr || m == nullptr || l == nullptr || r == nullptr || L_out == nullptr ||
        R_out == nullptr)
        return MALT_ERR_INVALID_ARG;
    if (!(mu1 >= 0.f && mu1 < 1.f) || !(mu2 >= 0.f && mu2 < 1.f) || !(eps >= 0.f))
        return MALT_ERR_INVALID_ARG;
    if (g_dtype != MALT_F32 && g_dtype != MALT_BF16) return MALT_ERR_UNSUPPORTED;
    if (rows <= 0 || cols <= 0 || rows % 8 != 0 || cols % 8 != 0 ||
        rows * cols >= (static_cast<int64_t>(1) << 31))
        return MALT_ERR_UNSUPPORTED;
    if (!aligned16(g) || !aligned16(m) || !aligned16(l) || !aligned16(r) || !aligned16(L_out) ||
        !aligned16(R_out))
        return MALT_ERR_MISALIGNED;
    const int64_t cb_count = (cols + malt::kStatCols - 1) / malt::kStatCols;
    const int64_t rb_count = (rows + malt::kStatRows - 1) / malt::kStatRows;
    const int64_t row_floats = ((cb_count * rows + 63) / 64) * 64;   // keeps colpart 256-B aligned
    const int64_t need = row_floats + rb_count * cols;
    if (need > MALT_NOALLOC_SCRATCH_FLOATS) {
        std::fprintf(stderr,
                     "malt_stats_noalloc: a %lld x %lld matrix needs %lld floats of scratch; "
                     "the fixed limit is %d\n",
                     static_cast<long long>(rows), static_cast<long long>(cols),
                     static_cast<long long>(need), MALT_NOALLOC_SCRATCH_FLOATS);
        return MALT_ERR_UNSUPPORTED;
    }
    float* scratch = nullptr;
    const int rc = scratch_for_current_device(&scratch);
    if (rc != MALT_OK) return rc;
    // The step's description of this one matrix, with its partial sums in
    // the fixed scratch and its preconditioners in the caller's buffers.
    MatDesc d;
    std::memset(&d, 0, sizeof(d));
    d.m = static_cast<int32_t>(rows);
    d.n = static_cast<int32_t>(cols);
    d.g_bf16 = g_dtype == MALT_BF16 ? 1 : 0;
    d.stat_rb = static_cast<int32_t>(rb_count);
    d.stat_cb = static_cast<int32_t>(cb_count);
    d.rowpart = scratch;
    d.colpart = scratch + row_floats;
    d.L = L_out;
    d.R = R_out;
    const UserPtrs up{nullptr, g, m, l, r, nullptr};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    noalloc_stats_kernel<<<static_cast<unsigned>(cb_count * rb_count), 256, 0, s>>>(d, up, mu1);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) {
        noalloc_finalize_kernel<<<static_cast<unsigned>((rows + cols + 255) / 256), 256, 0, s>>>(
            d, up, mu2, eps);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        std::fprintf(stderr, "malt_stats_noalloc: launch failed: %s\n", cudaGetErrorString(e));
        return MALT_ERR_CUDA;
    }
    return MALT_OK;
}
