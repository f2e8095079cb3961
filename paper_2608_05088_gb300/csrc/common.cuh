// common.cuh -- data structures shared by the host runtime and the kernels.
//
// Naming follows the paper: W weights, G gradient, M momentum, l / r row and
// column statistics, L / R their diagonal preconditioners, Mt = L M R, O the
// orthogonalised direction, D = L O R the back-mapped direction, nu the MALTER
// scalar.  "NS frame": Newton-Schulz runs on the wide orientation of Mt,
// p x q with p = min(m, n), q = max(m, n); a matrix with m > n is transposed.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>

namespace malt {

// Statistics kernel tile (rows x cols of W per block).
constexpr int kStatRows = 64;
constexpr int kStatCols = 256;
// Prescale block (rows x cols of Mt); the apply pass of a tall matrix uses
// the same block shape.
constexpr int kPreRows = 64;
constexpr int kPreCols = 256;
// Apply kernel (wide matrices): contiguous elements per block.
constexpr int kApplyElems = 16384;
// Newton-Schulz GEMM: a CTA pair computes a kTileM x kBN output tile; each CTA
// owns kBM rows of it, loads kBM rows of A and kBN/2 rows (N) of B per kBK
// reduction slice (one 128-byte swizzle row of bf16).
constexpr int kBM = 128;
constexpr int kTileM = 2 * kBM;
constexpr int kBN = 256;
constexpr int kBK = 64;
constexpr int kStages = 6;
constexpr int kBMN = 64;            // MN extent of one 128-byte swizzle atom (bf16)
constexpr int kEpiWarpsPerCta = 8;  // two per TMEM lane quarter
constexpr int kNsPartsPerTile = 2 * kEpiWarpsPerCta;  // graft partial pairs per tile
constexpr int kMaxClasses = 8;     // shape classes per GEMM launch
constexpr int kBindChunk = 128;    // parameters per pointer-binding launch
constexpr int kScalarsPerMat = 8;  // debug scalars per matrix

// Status bits set by kernels (OR-ed into the device status word).
constexpr int kStatusTimeout = 1;

// Caller pointers of one parameter for the current step (bound each step).
struct UserPtrs {
    void* w;
    const void* g;
    float* m;
    float* l;
    float* r;
};

// Static per-matrix description, built at init and kept on the device.
struct MatDesc {
    int32_t m, n;            // W is m x n
    int32_t trans;           // 1 when the NS frame is the transpose (m > n)
    int32_t p, q;            // NS frame shape
    int32_t w_bf16, g_bf16;  // element types of W and G
    int32_t cls, bidx;       // shape class and index within its batch
    int32_t stat_rb, stat_cb;       // statistics row bands / column chunks
    int32_t pre_tr, pre_tc;         // prescale blocks (kPreRows x kPreCols), rows and cols
    int32_t ns_tiles;               // GEMM tiles of one p x q product
    int32_t pad_;
    float* rowpart;          // [stat_cb][m] partial row sums of G^2
    float* colpart;          // [stat_rb][n] partial column sums of G^2
    float* L;                // [m]  (l + eps)^(-1/8)
    float* R;                // [n]  (r + eps)^(-1/8)
    float* prepart;          // [pre_tiles][2]  sum Mt^2, sum (L G R)^2
    float* nspart;           // [ns_tiles][kNsPartsPerTile][2]: sum O^2, sum D^2
    __nv_bfloat16* X0;       // NS-frame Mt (p x q, bf16): Mt, or Mt^T when trans
    __nv_bfloat16* O;        // [p][q] orthogonalised direction in the NS frame
};

// Per-matrix scalars kept on the device (index = matrix).
struct MatScalars {
    float k;        // 1 / (||Mt||_F + ns_eps)
    float norm_mt;  // ||Mt||_F
    float lgr_sq;   // ||L G R||_F^2 (MALTER)
    float scale;    // lr * alpha * ||O|| / (||D|| + eps)
    float norm_o, norm_d, alpha, nu;
};

struct StepHyper {
    float lr, mu1, mu2, eps, weight_decay;
    float ns_a, ns_b, ns_c, ns_eps;
    int32_t malter;
};

// --------------------------------------------------------------- GEMM launch
enum GemmPhase : int32_t { kGram = 0, kPoly = 1, kBX = 2 };

struct GemmClass {  // 64-byte aligned through its CUtensorMap members
    CUtensorMap tmA;              // operand A: rows of a K-major matrix (box kBK x kBM)
    CUtensorMap tmB;              // operand B: K-major rows (box kBK x kBM), or for kBX
                                  // an MN-major [K][N] matrix (box kBMN x kBK)
    CUtensorMap tmOut;            // output [batch][M][N], store box 32 x 32, 64-byte swizzle
                                  // (the last kBX stores O)
    int32_t M, N, K;              // per-matrix product shape
    int32_t batch;
    int32_t tiles_m, tiles_n;
    int32_t tile_begin;           // first global tile of this class in the launch
    int32_t pad_;
    const int32_t* mat_of;        // [batch] -> matrix index
    const __nv_bfloat16* ein;     // epilogue input (A for kPoly), [batch][M][N]

};

struct GemmParams {
    GemmClass cls[kMaxClasses];
    int32_t nclasses;
    int32_t total_tiles;
    int32_t phase;
    int32_t first;                // first NS iteration: apply the 1/||Mt|| scale
    int32_t last;                 // last NS iteration: write O and norm partials
    float a, b, c;
    const MatDesc* mats;
    const MatScalars* scal;
    int32_t* status;
    uint64_t budget_ns;
};

}  // namespace malt
