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
// Prescale block (rows x cols of Mt).
constexpr int kPreRows = 64;
constexpr int kPreCols = 256;
// Apply kernel: contiguous elements per block (O is stored in W's layout, so
// wide and tall matrices stream alike).
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
    void* wcopy;    // bf16 copy of an fp32 W written by the apply pass, or null
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
    __nv_bfloat16* O;        // orthogonalised direction in W's layout (m x n)
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

// ------------------------------------------------------ Newton-Schulz engine
enum GemmPhase : int32_t { kGram = 0, kPoly = 1, kBX = 2 };

// Launch modes of the Newton-Schulz kernel: one product with a static tile
// split, or a persistent work table of all products of the k iterations.
enum NsMode : int32_t { kNsPhased = 0, kNsPersistent = 1 };

// Epilogue warps of a CTA pair; each one signals a finished item once.
constexpr uint32_t kNsSignalsPerTile = 2 * kEpiWarpsPerCta;

// Stages of a persistent work table: the products of Newton-Schulz
// iteration i are stages 3 i + {kGram, kPoly, kBX}.  The table of k
// iterations is the first k iterations' entries of any longer table.
constexpr int kMaxNsSteps = 64;

// One item of a persistent work table.
struct __align__(16) NsEntry {
    int32_t code;     // stage (bits 0-11) | class slot (bits 12-15) | batch slot (bits 16-31)
    int32_t g;        // matrix; -1 marks the end of the table
    int32_t local;    // tile of the product
    uint32_t target;  // signals the previous stage of matrix g must reach (0: none)
};

__host__ __device__ __forceinline__ int32_t entry_stage(const NsEntry& e) { return e.code & 0xfff; }
__host__ __device__ __forceinline__ int32_t entry_cls(const NsEntry& e) { return (e.code >> 12) & 0xf; }
__host__ __device__ __forceinline__ int32_t entry_b(const NsEntry& e) {
    return static_cast<int32_t>(static_cast<uint32_t>(e.code) >> 16);
}

// One shape class (every matrix whose NS frame is p x q, stored batched) with
// all the tensor maps of the three products of an NS iteration.
struct NsClass {  // 64-byte aligned through its CUtensorMap members
    CUtensorMap tmX[2];           // the ping-pong iterates X as K-major rows (box kBK x kBM)
    CUtensorMap tmXmn[2];         // the same buffers as an MN-major [K][N] operand (box kBMN x kBK)
    CUtensorMap tmA, tmB;         // A = X X^T and B' = aI + bA + cA^2, K-major rows
    CUtensorMap stX[2], stA, stB, stO;   // epilogue stores: box 32 x 32, 64-byte swizzle
    CUtensorMap stOt;             // the O buffer as [q][p]: a tall W's O, stored in W's layout
    int32_t p, q, batch;
    int32_t tiles_p, tiles_q;     // 256-wide tiles along p and along q
    int32_t sym_begin;            // first item of this class within a Gram or Poly phase
    int32_t full_begin;           // first item of this class within a BX phase
    int32_t bx_col_major;         // list B*X tiles column by column (X larger than kBxColBytes)
    const int32_t* mat_of;        // [batch] -> matrix index
    const __nv_bfloat16* A;       // the A buffer [batch][p][p] (read by the Poly epilogue)
};

// Work list of one launch: for each NS iteration i, the Gram tiles of every
// class (sym_items), then the Poly tiles (sym_items), then the BX tiles
// (full_items); item s-phase index = 3 i + kind.  A launch runs the items
// [item_begin, item_end): one phase (phased schedule, static round-robin) or
// the whole list (persistent schedule, claimed through *queue, each tile
// waiting for its matrix's previous phase in done[]).
struct NsParams {
    NsClass cls[kMaxClasses];
    int32_t nclasses;
    int32_t nmat;                 // size of one row of done[]
    int32_t ns_steps;
    int32_t sym_items, full_items;
    int32_t item_begin, item_end;
    float a, b, c;
    const MatDesc* mats;
    MatScalars* scal;
    int32_t* status;
    uint32_t* queue;              // next unclaimed item (persistent schedule)
    uint32_t* done;               // [stages][nmat] finished-item signals (persistent)
    uint64_t budget_ns;
    // Persistent launches: the work table (item_end entries) and its stages.
    const NsEntry* table;
    int32_t nstages;              // 3 ns_steps
};
static_assert(sizeof(NsParams) <= 32764, "NsParams is passed by value as the kernel parameter");

// One decoded work item: a 256 x 256 output tile of one product.
struct NsWork {
    int32_t s;                    // 3 * iter + kind
    int32_t iter, kind;
    int32_t cls, b;               // class and batch slot (matrix = cls.mat_of[b])
    int32_t mt, nt;               // tile row / column
    int32_t local;                // tile index within the matrix's product
};

// Tiles of one matrix in a product of this kind: all of them for B X, the
// upper triangle (nt >= mt) for the symmetric Gram and polynomial products.
__host__ __device__ __forceinline__ int32_t ns_phase_tiles(const NsClass& C, int32_t kind) {
    return kind == kBX ? C.tiles_p * C.tiles_q : C.tiles_p * (C.tiles_p + 1) / 2;
}

// B*X tile order.  Row by row, the tiles that run at once read every column
// block of X; column by column, they read a few column blocks and all of B'
// (p x p).  Once one matrix's X is large against L2 (a 4096 x 16384 frame is
// 134 MB), row order reads X from DRAM once per wave of tiles: column order
// then cuts its DRAM reads five-fold and its time by 13 %.  Where X fits in
// L2 row order measured about 1.5 % faster (GPT-2 Large), so it stays there.
constexpr int64_t kBxColBytes = 32ll << 20;

// Tile row / column of the rem-th tile of one matrix's product of this kind:
// B*X row by row or column by column (bx_col_major), the upper triangle of
// the symmetric products row by row.
__host__ __device__ __forceinline__ void ns_tile_coords(const NsClass& C, int32_t kind, int32_t rem,
                                                        int32_t* mt, int32_t* nt) {
    if (kind == kBX) {
        if (C.bx_col_major) {
            *nt = rem / C.tiles_p;
            *mt = rem - *nt * C.tiles_p;
        } else {
            *mt = rem / C.tiles_q;
            *nt = rem - *mt * C.tiles_q;
        }
        return;
    }
    int32_t r = 0, u = rem;
    while (u >= C.tiles_p - r) {
        u -= C.tiles_p - r;
        ++r;
    }
    *mt = r;
    *nt = r + u;
}

// Blocks of the apply pass of one matrix: kApplyElems contiguous elements
// (O is stored in W's layout for every matrix).
__host__ __device__ __forceinline__ int32_t mat_apply_blocks(const MatDesc& d) {
    return static_cast<int32_t>((static_cast<int64_t>(d.m) * d.n + kApplyElems - 1) / kApplyElems);
}

__host__ __device__ __forceinline__ NsWork ns_decode(const NsParams& P, int32_t item) {
    NsWork w;
    const int32_t per_iter = 2 * P.sym_items + P.full_items;
    w.iter = item / per_iter;
    int32_t r = item - w.iter * per_iter;
    if (r < P.sym_items) {
        w.kind = kGram;
    } else if (r < 2 * P.sym_items) {
        w.kind = kPoly;
        r -= P.sym_items;
    } else {
        w.kind = kBX;
        r -= 2 * P.sym_items;
    }
    w.s = 3 * w.iter + w.kind;
    const bool sym = w.kind != kBX;
    int32_t c = 0;
    while (c + 1 < P.nclasses && r >= (sym ? P.cls[c + 1].sym_begin : P.cls[c + 1].full_begin)) ++c;
    const NsClass& C = P.cls[c];
    const int32_t local = r - (sym ? C.sym_begin : C.full_begin);
    const int32_t per = ns_phase_tiles(C, w.kind);
    w.cls = c;
    w.b = local / per;
    const int32_t rem = local - w.b * per;
    w.local = rem;
    ns_tile_coords(C, w.kind, rem, &w.mt, &w.nt);
    return w;
}

}  // namespace malt
