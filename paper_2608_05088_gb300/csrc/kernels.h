// kernels.h -- launchers of the library's kernels (internal to the library).
#pragma once
#include <cuda_runtime.h>
#include <cstdint>

#include "common.cuh"

namespace malt {

struct BindParams {
    UserPtrs p[kBindChunk];
    int32_t count;
    int32_t offset;
};

// Matrices whose rows or cols are not multiples of 8 run on zero-padded
// copies in the workspace (rows and cols rounded up to 8).  Before a step the
// pad launch copies the caller's W, G, M, l, r in; after it the unpad launch
// copies W, M, l, r back (and writes the bf16 copy of an fp32 W, if one is
// registered).  The padding is zero at init and every stage keeps it zero.
constexpr int kPadChunk = 48;      // matrices per pad / unpad launch
constexpr int kPadRows = 8;        // rows per block (one warp per row)
struct PadEntry {
    void* w_user;  void* w_pad;    // W (bf16 when w_bf16, else fp32)
    const void* g_user; void* g_pad;   // G (bf16 when g_bf16, else fp32)
    float* m_user; float* m_pad;
    float* l_user; float* l_pad;
    float* r_user; float* r_pad;
    void* wcopy_user;              // bf16 copy of an fp32 W (rows x cols), or null
    int32_t m, n, n8;              // caller rows and cols; padded leading dimension
    int32_t w_bf16, g_bf16;
    int32_t block_begin;           // first block of this matrix in the launch
};
struct PadParams {
    PadEntry e[kPadChunk];
    int32_t count;
};

cudaError_t launch_bind(const BindParams& P, UserPtrs* table, cudaStream_t s);
// in = true: caller -> padded copies; false: padded -> caller.
cudaError_t launch_pad(const PadParams& P, int32_t blocks, bool in, cudaStream_t s);
cudaError_t launch_stats(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                         int nmat, int32_t blocks, float mu1, int with_stats, cudaStream_t s);
cudaError_t launch_finalize(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                            int nmat, int32_t total, float mu2, float eps, long long* tcount,
                            int identity, cudaStream_t s);
// Prescale: `wide` wide matrices (ids[0 .. wide), wide_blocks blocks) in one
// launch, then `tall` tall ones (ids[wide ..), tall_blocks blocks) in another;
// pref is the block prefix over ids.
cudaError_t launch_prescale(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* ids,
                            const int32_t* pref, int wide, int32_t wide_blocks, int tall,
                            int32_t tall_blocks, int malter, cudaStream_t s);
cudaError_t launch_norms(const MatDesc* mats, MatScalars* scal, int nmat, float ns_eps,
                         int malter, cudaStream_t s);
cudaError_t launch_scalars(const MatDesc* mats, MatScalars* scal, const long long* tcount,
                           int nmat, const StepHyper& hp, cudaStream_t s);
cudaError_t launch_apply(const MatDesc* mats, const UserPtrs* ptrs, const MatScalars* scal,
                         const int32_t* pref, int nmat, int32_t blocks, float decay,
                         cudaStream_t s);
cudaError_t launch_wait_probe(int32_t* status, uint64_t budget_ns, cudaStream_t s);
// Guard regions after the workspace buffers: kGuardBytes each at the listed
// byte offsets of base.  check = false fills them with the pattern; check =
// true adds the number of bytes that differ from it to *bad.
constexpr size_t kGuardBytes = 256;
cudaError_t launch_guards(void* base, const uint64_t* offsets, int32_t n, bool check,
                          unsigned long long* bad, cudaStream_t s);

// Newton-Schulz products over up to kMaxClasses shape classes on grid_pairs
// CTA pairs (clusters of two).  mode kNsPhased: the items
// [P.item_begin, P.item_end) of one product, static round-robin.
// kNsPersistent: the work table P.table, claimed dynamically, each item
// waiting for its matrix's previous product (P.queue and P.done zeroed before
// the launch).
cudaError_t launch_ns_gemm(const NsParams& P, int mode, int grid_pairs, cudaStream_t s);
size_t ns_gemm_smem_bytes();
int ns_gemm_max_pairs();
// Opt the GEMM kernel into its shared memory and count the resident CTA pairs,
// once per device (on the current device; later calls only look it up).
cudaError_t ns_gemm_configure();

}  // namespace malt
