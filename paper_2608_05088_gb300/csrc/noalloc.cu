// noalloc.cu -- malt_stats_noalloc: the statistics stage of one matrix
// (momentum, row/column statistics and the two diagonal preconditioners)
// without any device allocation.
//
// Some callers cannot allocate device memory at the moment they need this
// work done: code running while a stream is being captured into a CUDA graph
// (an allocation there is either illegal or ends up baked into the graph),
// code that must not trigger the implicit device synchronisation an
// allocation may cause, and code that lives under a framework allocator which
// owns all device memory and forbids allocations behind its back.  The
// regular entry points need a workspace from malt_init_state; this one keeps
// its only scratch -- the per-tile partial sums of G^2 -- in a fixed array
// that lives in the library image itself.
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
#include <mutex>

#include "../../include/malt.h"

namespace {

constexpr int kRows = 64;         // rows of G per block
constexpr int kCols = 256;        // columns of G per block
constexpr int kRowsPerWarp = kRows / 8;
constexpr int kMaxDevices = 64;

static_assert(MALT_NOALLOC_SCRATCH_FLOATS % 64 == 0, "scratch size must keep 256-byte alignment");

// The scratch array: [col_chunks][m] row partials, then [row_bands][n] column partials.
static __device__ __align__(256) float g_noalloc_scratch[MALT_NOALLOC_SCRATCH_FLOATS];

std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Momentum update and per-tile partial sums of G^2 (Algorithm 1, M_t / l_t /
// r_t lines): one block covers kRows x kCols of G; each warp owns 8 rows and
// each lane 8 consecutive columns.
__global__ void __launch_bounds__(256)
noalloc_stats_kernel(const void* __restrict__ g, int g_bf16, float* __restrict__ mom, int m, int n,
                     float mu1, float* __restrict__ rowpart, float* __restrict__ colpart) {
    __shared__ __align__(16) float colsh[8][kCols];
    const int cb_count = (n + kCols - 1) / kCols;
    const int rb = blockIdx.x / cb_count, cb = blockIdx.x - rb * cb_count;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int col = cb * kCols + lane * 8;
    const bool colok = col < n;
    const int row0 = rb * kRows + warp * kRowsPerWarp;
    float csum[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) csum[j] = 0.f;
    float myrow = 0.f;
    for (int rr = 0; rr < kRowsPerWarp; ++rr) {
        const int row = row0 + rr;
        float rs = 0.f;
        if (colok && row < m) {
            const size_t off = static_cast<size_t>(row) * n + col;
            float gv[8];
            if (g_bf16) {
                const uint4 u = *reinterpret_cast<const uint4*>(
                    static_cast<const __nv_bfloat16*>(g) + off);
                const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float2 f = __bfloat1622float2(h[k]);
                    gv[2 * k] = f.x;
                    gv[2 * k + 1] = f.y;
                }
            } else {
                const float4* p = reinterpret_cast<const float4*>(static_cast<const float*>(g) + off);
                const float4 a = p[0], b = p[1];
                gv[0] = a.x; gv[1] = a.y; gv[2] = a.z; gv[3] = a.w;
                gv[4] = b.x; gv[5] = b.y; gv[6] = b.z; gv[7] = b.w;
            }
            float4* mp = reinterpret_cast<float4*>(mom + off);
            const float4 a = mp[0], b = mp[1];
            const float mv[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
            float nm[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                nm[j] = fmaf(mu1, mv[j], (1.f - mu1) * gv[j]);
                const float sq = gv[j] * gv[j];
                rs += sq;
                csum[j] += sq;
            }
            mp[0] = make_float4(nm[0], nm[1], nm[2], nm[3]);
            mp[1] = make_float4(nm[4], nm[5], nm[6], nm[7]);
        }
        rs = warp_sum(rs);
        if (lane == rr) myrow = rs;
    }
    if (lane < kRowsPerWarp && row0 + lane < m)
        rowpart[static_cast<size_t>(cb) * m + row0 + lane] = myrow;
#pragma unroll
    for (int j = 0; j < 8; ++j) colsh[warp][lane * 8 + j] = csum[j];
    __syncthreads();
    const int gc = cb * kCols + threadIdx.x;
    if (gc < n) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) s += colsh[w][threadIdx.x];
        colpart[static_cast<size_t>(rb) * n + gc] = s;
    }
}

// EMAs of the statistics and the diagonal preconditioners (Algorithm 1, l_t,
// r_t and L_t / R_t lines), one thread per row or column.
__global__ void __launch_bounds__(256)
noalloc_finalize_kernel(int m, int n, const float* __restrict__ rowpart,
                        const float* __restrict__ colpart, float* __restrict__ l,
                        float* __restrict__ r, float* __restrict__ Lout, float* __restrict__ Rout,
                        float mu2, float eps) {
    const int x = blockIdx.x * blockDim.x + threadIdx.x;
    const int cb_count = (n + kCols - 1) / kCols;
    const int rb_count = (m + kRows - 1) / kRows;
    if (x < m) {
        float s = 0.f;
        for (int cb = 0; cb < cb_count; ++cb) s += rowpart[static_cast<size_t>(cb) * m + x];
        const float v = fmaf(mu2, l[x], (1.f - mu2) * s);
        l[x] = v;
        Lout[x] = powf(v + eps, -0.125f);
    } else if (x < m + n) {
        const int j = x - m;
        float s = 0.f;
        for (int rb = 0; rb < rb_count; ++rb) s += colpart[static_cast<size_t>(rb) * n + j];
        const float v = fmaf(mu2, r[j], (1.f - mu2) * s);
        r[j] = v;
        Rout[j] = powf(v + eps, -0.125f);
    }
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
    const int64_t cb_count = (cols + kCols - 1) / kCols;
    const int64_t rb_count = (rows + kRows - 1) / kRows;
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
    float* rowpart = scratch;
    float* colpart = scratch + row_floats;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int mi = static_cast<int>(rows), ni = static_cast<int>(cols);
    noalloc_stats_kernel<<<static_cast<unsigned>(cb_count * rb_count), 256, 0, s>>>(
        g, g_dtype == MALT_BF16, m, mi, ni, mu1, rowpart, colpart);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) {
        noalloc_finalize_kernel<<<(mi + ni + 255) / 256, 256, 0, s>>>(mi, ni, rowpart, colpart, l, r,
                                                                       L_out, R_out, mu2, eps);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        std::fprintf(stderr, "malt_stats_noalloc: launch failed: %s\n", cudaGetErrorString(e));
        return MALT_ERR_CUDA;
    }
    return MALT_OK;
}
