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

cudaError_t launch_bind(const BindParams& P, UserPtrs* table, cudaStream_t s);
cudaError_t launch_stats(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                         int nmat, int32_t blocks, float mu1, int with_stats, cudaStream_t s);
cudaError_t launch_finalize(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                            int nmat, int32_t total, float mu2, float eps, long long* tcount,
                            int identity, cudaStream_t s);
cudaError_t launch_prescale(const MatDesc* mats, const UserPtrs* ptrs, const int32_t* pref,
                            int nmat, int32_t blocks, int malter, cudaStream_t s);
cudaError_t launch_norms(const MatDesc* mats, MatScalars* scal, int nmat, float ns_eps,
                         int malter, cudaStream_t s);
cudaError_t launch_scalars(const MatDesc* mats, MatScalars* scal, const long long* tcount,
                           int nmat, const StepHyper& hp, cudaStream_t s);
cudaError_t launch_apply(const MatDesc* mats, const UserPtrs* ptrs, const MatScalars* scal,
                         const int32_t* pref, int nmat, int32_t blocks, float decay,
                         cudaStream_t s);
cudaError_t launch_wait_probe(int32_t* status, uint64_t budget_ns, cudaStream_t s);

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
