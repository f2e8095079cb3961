// adamw.cu -- the AdamW update of the parameters the paper does not give to
// MALT: vectors, scalars, embeddings and the output head (Section 5.1,
// parameter grouping), with the decoupled weight decay of the appendix
// hyperparameter table.  Together with malt_step on the 2-D weight matrices
// it makes the whole optimizer step of a GPT-2 model.
//
// Per tensor, at step t (1-based; the step counter lives on the device):
//   m <- b1 m + (1 - b1) g,   v <- b2 v + (1 - b2) g^2
//   w <- (1 - lr wd) w - (lr / (1 - b1^t)) m / (sqrt(v) / sqrt(1 - b2^t) + eps)
// with fp32 master weights w and an optional bf16 copy written from the
// updated w (round to nearest even).
//
// One grouped launch covers every tensor of a step: block b takes a
// contiguous run of kAdamChunk elements of one tensor (a block-prefix table
// maps blocks to tensors).  Each thread streams 4 elements per 128-bit load
// of w, m, v and g (64-bit for a bf16 gradient), two such groups in flight.
// The update is 30 B/elem of HBM traffic with an fp32 gradient and a bf16
// copy (g 4, w 4+4, m 4+4, v 4+4, copy 2).  A tiny bind launch before it
// copies the caller's pointers to the device and advances t, so the step
// needs no host synchronisation and can be replayed from a CUDA graph.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/malt.h"

namespace {

constexpr int kAdamThreads = 256;
constexpr int kAdamVec = 4;                                     // elements per 128-bit group
// One group per thread per pass at 6 blocks per SM (39 registers) measured
// faster than two groups in flight at 4 blocks (63 registers): resident warps
// keep more of HBM busy.
constexpr int kAdamInFlight = 1;                                // groups per thread per pass
constexpr int kAdamChunk = kAdamThreads * kAdamVec * kAdamInFlight * 4;   // 4096 elements
constexpr int kAdamBindChunk = 96;                              // tensors per bind launch

struct AdamPtrs {
    float* w;
    void* wcopy;
    const void* g;
    float* m;
    float* v;
    float decay;        // 1 - lr * weight_decay of this tensor, for this step
    int32_t pad_;
};

struct AdamDesc {
    int64_t numel;
    int32_t g_bf16;
    int32_t pad_;
};

struct AdamHyper {
    float lr, beta1, beta2, eps;
};

struct AdamBind {
    AdamPtrs p[kAdamBindChunk];
    int32_t count, offset;
    long long* tcount;      // advanced by the first chunk's launch
    float* factors;         // [2]: lr / (1 - beta1^t), 1 / sqrt(1 - beta2^t)
    AdamHyper h;
};

// Copies the caller's pointers; the first chunk's launch also advances the
// step count t and computes the step's two bias-correction factors once (in
// double: the update kernel itself does no fp64 arithmetic).
__global__ void adamw_bind_kernel(const __grid_constant__ AdamBind B, AdamPtrs* __restrict__ table) {
    const int i = threadIdx.x;
    if (i < B.count) table[B.offset + i] = B.p[i];
    if (i == 0 && B.tcount != nullptr) {
        const long long tc = *B.tcount + 1;                      // 1-based step count
        *B.tcount = tc;
        const double t = static_cast<double>(tc);
        B.factors[0] = static_cast<float>(static_cast<double>(B.h.lr) /
                                          (1.0 - pow(static_cast<double>(B.h.beta1), t)));
        B.factors[1] = static_cast<float>(1.0 / sqrt(1.0 - pow(static_cast<double>(B.h.beta2), t)));
    }
}

__device__ __forceinline__ int find_tensor(const int32_t* __restrict__ pref, int n, int32_t x) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(pref + mid) <= x) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// Four consecutive gradient elements (fp32 or bf16) as floats.
__device__ __forceinline__ float4 load_g4(const void* g, bool bf16, int64_t e) {
    if (bf16) {
        const uint2 u = __ldg(reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(g) + e));
        const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
        const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
        return make_float4(a.x, a.y, b.x, b.y);
    }
    return __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(g) + e));
}

// One element of the update (explicit fused multiply-adds: one rounding
// order wherever it is compiled).
__device__ __forceinline__ void adam1(float& w, float& m, float& v, float g, const AdamHyper& h,
                                      float step, float inv_sqrt_bc2, float decay) {
    m = fmaf(h.beta1, m, (1.f - h.beta1) * g);
    v = fmaf(h.beta2, v, ((1.f - h.beta2) * g) * g);
    const float denom = fmaf(sqrtf(v), inv_sqrt_bc2, h.eps);
    w = fmaf(-step, m / denom, decay * w);
}

__global__ void __launch_bounds__(kAdamThreads, 6)
adamw_kernel(const AdamDesc* __restrict__ desc, const AdamPtrs* __restrict__ ptrs,
             const int32_t* __restrict__ pref, int n, const float* __restrict__ factors,
             AdamHyper h) {
    const int k = find_tensor(pref, n, blockIdx.x);
    const AdamDesc d = desc[k];
    const AdamPtrs p = ptrs[k];
    const int64_t begin = static_cast<int64_t>(blockIdx.x - __ldg(pref + k)) * kAdamChunk;
    const int64_t end = d.numel < begin + kAdamChunk ? d.numel : begin + kAdamChunk;
    // Bias corrections of this step t, computed by the bind launch.
    const float step = factors[0];
    const float inv_sqrt_bc2 = factors[1];
    const bool gbf = d.g_bf16 != 0;
    const int64_t vec_end = begin + ((end - begin) / kAdamVec) * kAdamVec;
    constexpr int64_t kPass = static_cast<int64_t>(kAdamThreads) * kAdamVec * kAdamInFlight;
    for (int64_t base = begin; base < vec_end; base += kPass) {
        float4 w4[kAdamInFlight], m4[kAdamInFlight], v4[kAdamInFlight], g4[kAdamInFlight];
        int64_t e[kAdamInFlight];
        bool ok[kAdamInFlight];
#pragma unroll
        for (int u = 0; u < kAdamInFlight; ++u) {
            e[u] = base + (static_cast<int64_t>(u) * kAdamThreads + threadIdx.x) * kAdamVec;
            ok[u] = e[u] < vec_end;
            if (ok[u]) {
                w4[u] = *reinterpret_cast<const float4*>(p.w + e[u]);
                m4[u] = *reinterpret_cast<const float4*>(p.m + e[u]);
                v4[u] = *reinterpret_cast<const float4*>(p.v + e[u]);
                g4[u] = load_g4(p.g, gbf, e[u]);
            }
        }
#pragma unroll
        for (int u = 0; u < kAdamInFlight; ++u) {
            if (!ok[u]) continue;
            adam1(w4[u].x, m4[u].x, v4[u].x, g4[u].x, h, step, inv_sqrt_bc2, p.decay);
            adam1(w4[u].y, m4[u].y, v4[u].y, g4[u].y, h, step, inv_sqrt_bc2, p.decay);
            adam1(w4[u].z, m4[u].z, v4[u].z, g4[u].z, h, step, inv_sqrt_bc2, p.decay);
            adam1(w4[u].w, m4[u].w, v4[u].w, g4[u].w, h, step, inv_sqrt_bc2, p.decay);
            *reinterpret_cast<float4*>(p.w + e[u]) = w4[u];
            *reinterpret_cast<float4*>(p.m + e[u]) = m4[u];
            *reinterpret_cast<float4*>(p.v + e[u]) = v4[u];
            if (p.wcopy != nullptr) {
                uint2 c;
                *reinterpret_cast<__nv_bfloat162*>(&c.x) = __floats2bfloat162_rn(w4[u].x, w4[u].y);
                *reinterpret_cast<__nv_bfloat162*>(&c.y) = __floats2bfloat162_rn(w4[u].z, w4[u].w);
                *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.wcopy) + e[u]) = c;
            }
        }
    }
    // The last 1-3 elements of a tensor whose size is not a multiple of 4.
    const int64_t i = vec_end + threadIdx.x;
    if (i < end) {
        float w = p.w[i], m = p.m[i], v = p.v[i];
        const float g = gbf ? __bfloat162float(static_cast<const __nv_bfloat16*>(p.g)[i])
                            : static_cast<const float*>(p.g)[i];
        adam1(w, m, v, g, h, step, inv_sqrt_bc2, p.decay);
        p.w[i] = w;
        p.m[i] = m;
        p.v[i] = v;
        if (p.wcopy != nullptr) static_cast<__nv_bfloat16*>(p.wcopy)[i] = __float2bfloat16_rn(w);
    }
}

int cuda_fail(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return MALT_OK;
    std::fprintf(stderr, "malt_adamw: %s failed: %s\n", what, cudaGetErrorString(e));
    return MALT_ERR_CUDA;
}

#define ADAM_CUDA(call, what)                              \
    do {                                                   \
        const int rc_ = cuda_fail((call), (what));         \
        if (rc_ != MALT_OK) return rc_;                    \
    } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int validate(const malt_adamw_param_t& p) {
    if (p.w == nullptr || p.g == nullptr || p.m == nullptr || p.v == nullptr)
        return MALT_ERR_INVALID_ARG;
    if (p.numel <= 0 || (p.g_dtype != MALT_F32 && p.g_dtype != MALT_BF16))
        return MALT_ERR_UNSUPPORTED;
    if (!(p.weight_decay == p.weight_decay)) return MALT_ERR_INVALID_ARG;
    if (!aligned16(p.w) || !aligned16(p.g) || !aligned16(p.m) || !aligned16(p.v) ||
        (p.w_copy != nullptr && !aligned16(p.w_copy)))
        return MALT_ERR_MISALIGNED;
    return MALT_OK;
}

}  // namespace

struct malt_adamw_state {
    int device = 0;
    int n = 0;
    std::vector<malt_adamw_param_t> shape0;     // sizes and gradient types fixed at init
    void* ws = nullptr;
    AdamDesc* d_desc = nullptr;
    AdamPtrs* d_ptrs = nullptr;
    int32_t* d_pref = nullptr;
    long long* d_t = nullptr;
    float* d_factors = nullptr;
    int32_t blocks = 0;
    cudaStream_t last_stream = nullptr;
};

namespace {
// Bind launches and the update launch of one step (after validation).
int enqueue_adamw(malt_adamw_state* st, const malt_adamw_param_t* params, int32_t n,
                  const malt_adamw_hparams_t* hp, cudaStream_t s);
}  // namespace

extern "C" {

int malt_adamw_init_state(malt_adamw_state_t** out, const malt_adamw_param_t* params, int32_t n,
                          void* stream) {
    if (out == nullptr) return MALT_ERR_INVALID_ARG;
    *out = nullptr;
    if (n < 0 || (n > 0 && params == nullptr)) return MALT_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i) {
        const int rc = validate(params[i]);
        if (rc != MALT_OK) return rc;
    }
    std::vector<int32_t> pref(n + 1, 0);
    std::vector<AdamDesc> desc(n);
    for (int i = 0; i < n; ++i) {
        const int64_t blocks = (params[i].numel + kAdamChunk - 1) / kAdamChunk;
        if (pref[i] + blocks >= (int64_t{1} << 31)) return MALT_ERR_UNSUPPORTED;
        pref[i + 1] = static_cast<int32_t>(pref[i] + blocks);
        desc[i] = AdamDesc{params[i].numel, params[i].g_dtype == MALT_BF16 ? 1 : 0, 0};
    }
    malt_adamw_state* st = new malt_adamw_state();
    st->n = n;
    st->shape0.assign(params, params + n);
    st->blocks = pref[n];
    auto fail = [&](int rc) {
        if (st->ws != nullptr) cudaFree(st->ws);
        delete st;
        return rc;
    };
    if (cudaGetDevice(&st->device) != cudaSuccess) return fail(MALT_ERR_CUDA);
    const size_t nn = static_cast<size_t>(std::max(n, 1));
    const size_t o_desc = 0;
    const size_t o_ptrs = (o_desc + sizeof(AdamDesc) * nn + 255) & ~size_t(255);
    const size_t o_pref = (o_ptrs + sizeof(AdamPtrs) * nn + 255) & ~size_t(255);
    const size_t o_t = (o_pref + sizeof(int32_t) * (nn + 1) + 255) & ~size_t(255);
    const size_t bytes = o_t + 256;
    if (cudaMalloc(&st->ws, bytes) != cudaSuccess) {
        st->ws = nullptr;
        cudaGetLastError();
        return fail(MALT_ERR_OUT_OF_MEMORY);
    }
    uint8_t* base = static_cast<uint8_t*>(st->ws);
    st->d_desc = reinterpret_cast<AdamDesc*>(base + o_desc);
    st->d_ptrs = reinterpret_cast<AdamPtrs*>(base + o_ptrs);
    st->d_pref = reinterpret_cast<int32_t*>(base + o_pref);
    st->d_t = reinterpret_cast<long long*>(base + o_t);
    st->d_factors = reinterpret_cast<float*>(base + o_t + 64);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int rc = cuda_fail(cudaMemset(st->ws, 0, bytes), "cudaMemset(state)");
    if (rc == MALT_OK && n > 0)
        rc = cuda_fail(cudaMemcpy(st->d_desc, desc.data(), sizeof(AdamDesc) * n,
                                  cudaMemcpyHostToDevice), "cudaMemcpy(desc)");
    if (rc == MALT_OK)
        rc = cuda_fail(cudaMemcpy(st->d_pref, pref.data(), sizeof(int32_t) * (n + 1),
                                  cudaMemcpyHostToDevice), "cudaMemcpy(prefix)");
    // Zero moments (the algorithm's initial m_0 = v_0 = 0).
    for (int i = 0; rc == MALT_OK && i < n; ++i) {
        const size_t b = sizeof(float) * static_cast<size_t>(params[i].numel);
        rc = cuda_fail(cudaMemsetAsync(params[i].m, 0, b, s), "cudaMemsetAsync(m)");
        if (rc == MALT_OK) rc = cuda_fail(cudaMemsetAsync(params[i].v, 0, b, s), "cudaMemsetAsync(v)");
    }
    if (rc != MALT_OK) return fail(rc);
    st->last_stream = s;
    *out = st;
    return MALT_OK;
}

int malt_adamw_step(malt_adamw_state_t* st, const malt_adamw_param_t* params, int32_t n,
                    const malt_adamw_hparams_t* hp, void* stream) {
    if (st == nullptr || hp == nullptr || (n > 0 && params == nullptr)) return MALT_ERR_INVALID_ARG;
    if (!(hp->beta1 >= 0.f && hp->beta1 < 1.f) || !(hp->beta2 >= 0.f && hp->beta2 < 1.f) ||
        !(hp->eps >= 0.f) || !(hp->lr == hp->lr))
        return MALT_ERR_INVALID_ARG;
    if (n != st->n) return MALT_ERR_SHAPE_CHANGED;
    for (int i = 0; i < n; ++i) {
        const int rc = validate(params[i]);
        if (rc != MALT_OK) return rc;
        if (params[i].numel != st->shape0[i].numel || params[i].g_dtype != st->shape0[i].g_dtype)
            return MALT_ERR_SHAPE_CHANGED;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    st->last_stream = s;
    ADAM_CUDA(cudaSetDevice(st->device), "cudaSetDevice");
    nvtxRangePushA("malt_adamw_step");
    const int rc = enqueue_adamw(st, params, n, hp, s);
    nvtxRangePop();
    return rc;
}

}  // extern "C"

namespace {

int enqueue_adamw(malt_adamw_state* st, const malt_adamw_param_t* params, int32_t n,
                  const malt_adamw_hparams_t* hp, cudaStream_t s) {
    AdamBind B;
    for (int off = 0; off == 0 || off < n; off += kAdamBindChunk) {
        const int cnt = std::min(kAdamBindChunk, n - off);
        std::memset(&B, 0, sizeof(B));
        B.count = cnt;
        B.offset = off;
        B.tcount = off == 0 ? st->d_t : nullptr;
        B.factors = st->d_factors;
        B.h = AdamHyper{hp->lr, hp->beta1, hp->beta2, hp->eps};
        for (int i = 0; i < cnt; ++i) {
            const malt_adamw_param_t& p = params[off + i];
            B.p[i] = AdamPtrs{p.w, p.w_copy, p.g, p.m, p.v, 1.f - hp->lr * p.weight_decay, 0};
        }
        adamw_bind_kernel<<<1, kAdamBindChunk, 0, s>>>(B, st->d_ptrs);
        ADAM_CUDA(cudaGetLastError(), "adamw_bind_kernel");
    }
    if (st->blocks == 0) return MALT_OK;
    const AdamHyper h{hp->lr, hp->beta1, hp->beta2, hp->eps};
    adamw_kernel<<<st->blocks, kAdamThreads, 0, s>>>(st->d_desc, st->d_ptrs, st->d_pref, n,
                                                     st->d_factors, h);
    ADAM_CUDA(cudaGetLastError(), "adamw_kernel");
    return MALT_OK;
}

}  // namespace

extern "C" {

int malt_adamw_get_step(malt_adamw_state_t* st, int64_t* t_host) {
    if (st == nullptr || t_host == nullptr) return MALT_ERR_INVALID_ARG;
    ADAM_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    long long t = 0;
    ADAM_CUDA(cudaMemcpy(&t, st->d_t, sizeof(t), cudaMemcpyDeviceToHost), "cudaMemcpy(t)");
    *t_host = t;
    return MALT_OK;
}

int malt_adamw_set_step(malt_adamw_state_t* st, int64_t t_host) {
    if (st == nullptr || t_host < 0) return MALT_ERR_INVALID_ARG;
    ADAM_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    const long long t = t_host;
    ADAM_CUDA(cudaMemcpy(st->d_t, &t, sizeof(t), cudaMemcpyHostToDevice), "cudaMemcpy(t)");
    return MALT_OK;
}

void malt_adamw_destroy_state(malt_adamw_state_t* st) {
    if (st == nullptr) return;
    cudaStreamSynchronize(st->last_stream);
    if (st->ws != nullptr) cudaFree(st->ws);
    delete st;
}

}  // extern "C"
