// malt_api.cu -- host runtime behind include/malt.h.
//
// At init the parameters are planned once: each matrix gets its Newton-Schulz
// frame (transposed when m > n), matrices with the same frame shape p x q form
// a shape class whose NS buffers are stored batched ([batch][p][q] etc.) so one
// 3-D TMA descriptor serves the whole class, and every grouped element-wise
// launch gets a block-prefix table.  A step then enqueues, on the caller's
// stream and without any host synchronisation:
//   bind (caller pointers) -> stats -> finalize -> prescale (wide matrices,
//   then tall ones) -> norms -> Newton-Schulz -> scalars -> apply,
// where Newton-Schulz runs, per group of up to kMaxClasses classes, either as
// one persistent launch over all k x (Gram, Poly, BX) products or as one
// launch per product (the phased schedule); by default a group whose Gram
// product is shallow (few tile waves) takes the persistent launch and a deep
// one the phased launches.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <map>
#include <utility>
#include <vector>

#include "../../include/malt.h"
#include "common.cuh"
#include "kernels.h"

using namespace malt;

namespace {

// Time budget of every device-side wait: 1 s, plus the time one 256 x 256
// output tile of the launch's longest reduction could take at a tenth of a
// CTA pair's share of the bf16 peak (2 x 256 x 256 flops per unit of K at
// 2 TFLOP/s), so that the budget still flags a hang, never an elongated
// matrix whose Gram product reduces over hundreds of millions of columns.
constexpr uint64_t kWaitBudgetNs = 1000000000ull;
constexpr uint64_t kWaitNsPerK = 66;

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

bool get_encoder() {
    if (g_encode != nullptr) return true;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
        return false;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return true;
}

// 3-D bf16 tensor [batch][rows][cols], box box_cols x box_rows x 1, zero fill
// outside the tensor on loads (stores skip the outside).
bool encode_3d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint64_t batch,
               uint32_t box_rows, uint32_t box_cols = kBK,
               CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
    const cuuint64_t dims[3] = {cols, rows, batch};
    const cuuint64_t strides[2] = {cols * 2, rows * cols * 2};
    const cuuint32_t box[3] = {box_cols, box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base),
                                dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Store map of an epilogue output: 32 x 32 boxes with 64-byte swizzle.
bool encode_store(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint64_t batch) {
    return encode_3d(map, base, cols, rows, batch, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
}

struct ShapeClass {
    int p = 0, q = 0, batch = 0;
    std::vector<int> mats;
    int32_t* d_mat_of = nullptr;
    __nv_bfloat16* X[2] = {nullptr, nullptr};   // ping-pong NS iterates [batch][p][q]
    __nv_bfloat16* A = nullptr;                  // X X^T        [batch][p][p]
    __nv_bfloat16* B = nullptr;                  // aI + bA + cA^2 [batch][p][p]
    __nv_bfloat16* O = nullptr;                  // last iterate, per matrix in W's layout:
                                                 // [p][q] (wide) or [q][p] (tall)
    CUtensorMap tmX[2], tmXmn[2], tmA, tmB;    // 128-row K-major boxes; 64x64 MN boxes
    CUtensorMap stX[2], stA, stB, stO, stOt;   // epilogue store maps (stOt: O as [q][p])
};

// Workspace carving: 256-byte aligned buffers, each followed by a guard
// region that init fills with a pattern; malt_debug_check_guards counts
// guard bytes a kernel has overwritten (an out-of-bounds write detector for
// the tests, where no memory checker runs).
struct Carver {
    size_t off = 0;
    std::vector<size_t> guards;
    size_t take(size_t bytes) {
        const size_t o = off;
        off += (bytes + 255) & ~static_cast<size_t>(255);
        guards.push_back(off);
        off += kGuardBytes;
        return o;
    }
};

int cuda_fail(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return MALT_OK;
    std::fprintf(stderr, "malt: %s failed: %s\n", what, cudaGetErrorString(e));
    return MALT_ERR_CUDA;
}

#define MALT_CUDA(call, what)                              \
    do {                                                   \
        const int rc_ = cuda_fail((call), (what));         \
        if (rc_ != MALT_OK) return rc_;                    \
    } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Rows and cols as the kernels see them: rounded up to a multiple of 8 (a
// matrix with other dimensions runs on zero-padded copies in the workspace).
int64_t round8(int64_t x) { return (x + 7) / 8 * 8; }

// Workspace copies of a matrix whose rows or cols are not multiples of 8.
struct PadBuf {
    void* w = nullptr;
    void* g = nullptr;
    float* m = nullptr;
    float* l = nullptr;
    float* r = nullptr;
};

}  // namespace

struct malt_state {
    int device = 0;
    int nmat = 0;
    int num_sms = 0;
    std::vector<malt_param_t> shape0;      // shapes / dtypes fixed at init
    std::vector<void*> wcopy;              // bf16 copies of fp32 weights (malt_set_weight_copies)
    std::vector<int> padded;               // matrices whose rows or cols are not multiples of 8
    std::vector<PadBuf> padbuf;            // their zero-padded workspace copies (index = matrix)
    std::vector<MatDesc> hmats;
    std::vector<ShapeClass> classes;
    void* ws = nullptr;
    size_t ws_bytes = 0;
    MatDesc* d_mats = nullptr;
    UserPtrs* d_ptrs = nullptr;
    MatScalars* d_scal = nullptr;
    long long* d_t = nullptr;
    int32_t* d_status = nullptr;
    int32_t* d_pref[4] = {nullptr, nullptr, nullptr, nullptr};  // stats, fin, pre, apply
    int32_t blocks_stats = 0, total_fin = 0, blocks_pre = 0, blocks_apply = 0;
    // The prescale pass runs wide and tall matrices in two launches (their
    // blocks differ): d_pre_ids lists the wide matrices, then the tall ones,
    // and d_pref[2] is the block prefix in that order.
    int32_t* d_pre_ids = nullptr;
    int32_t pre_wide = 0, blocks_pre_wide = 0;
    // Newton-Schulz work lists, one per group of up to kMaxClasses classes,
    // and the persistent schedule's counters: [groups_pad] claim counters,
    // then [3 * kMaxNsSteps][nmat] finished-tile signals.
    std::vector<NsParams> ns_groups;
    std::vector<std::vector<int>> ns_slot_class;   // class index of each slot of each group
    uint32_t* d_sched = nullptr;
    int sched_groups_pad = 0;
    int ns_schedule = MALT_NS_AUTO;
    // Work table of the persistent launches, one per launch group, for
    // kMaxNsSteps iterations (in the workspace, uploaded at init); a launch of
    // k iterations claims its first k * table_per_iter[group] entries.
    std::vector<NsEntry*> table_dev;
    std::vector<int32_t> table_per_iter;
    int32_t last_timeout[5] = {};   // site record of the last timeout malt_check reported
    uint64_t* d_guard_off = nullptr;   // byte offsets of the guard regions
    unsigned long long* d_guard_bad = nullptr;   // corrupted guard bytes found by the check
    int32_t nguards = 0;
    cudaStream_t last_stream = nullptr;
    // Profiling: event pairs recorded around launches, folded in on read.
    bool profiling = false;
    std::vector<cudaEvent_t> ev_pool;
    std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> ev_pending;
    double prof_ms[MALT_NUM_KINDS] = {};
    int64_t prof_launches[MALT_NUM_KINDS] = {};
    // Host-buffer steps: copy streams and the events that order them against
    // the compute stream (created on first use).
    cudaStream_t h2d = nullptr, d2h = nullptr;
    cudaEvent_t ev_h2d = nullptr, ev_applied = nullptr, ev_d2h = nullptr;
    // "G consumed" events per device gradient buffer set (keyed by the first
    // parameter's G pointer), so callers that alternate two sets let the next
    // copy-in run while the current step still reads the other set.
    static constexpr int kGSlots = 2;
    const void* g_key[kGSlots] = {nullptr, nullptr};
    cudaEvent_t ev_g_consumed[kGSlots] = {nullptr, nullptr};
    bool g_recorded[kGSlots] = {false, false};
    int g_next_slot = 0;
    bool pipe_primed = false;
};

// Ordering hooks of a host-buffer step inside run_step.
struct PipeHooks {
    cudaEvent_t record_g_consumed;   // after the last kernel that reads G
    cudaEvent_t wait_before_apply;   // the previous step's weight read-back (or null)
    cudaEvent_t record_applied;      // after the apply kernel
};

namespace {

int validate_param(const malt_param_t& p) {
    if (p.w == nullptr || p.g == nullptr || p.m == nullptr || p.l == nullptr || p.r == nullptr)
        return MALT_ERR_INVALID_ARG;
    if (p.rows <= 0 || p.cols <= 0) return MALT_ERR_UNSUPPORTED;
    if (round8(p.rows) * round8(p.cols) >= (static_cast<int64_t>(1) << 31)) return MALT_ERR_UNSUPPORTED;
    if ((p.w_dtype != MALT_F32 && p.w_dtype != MALT_BF16) ||
        (p.g_dtype != MALT_F32 && p.g_dtype != MALT_BF16))
        return MALT_ERR_UNSUPPORTED;
    if (!aligned16(p.w) || !aligned16(p.g) || !aligned16(p.m) || !aligned16(p.l) ||
        !aligned16(p.r))
        return MALT_ERR_MISALIGNED;
    return MALT_OK;
}

int validate_hparams(const malt_hparams_t* hp) {
    if (hp == nullptr) return MALT_ERR_INVALID_ARG;
    if (!(hp->mu1 >= 0.f && hp->mu1 < 1.f) || !(hp->mu2 >= 0.f && hp->mu2 < 1.f))
        return MALT_ERR_INVALID_ARG;
    if (!(hp->eps >= 0.f) || !(hp->ns_eps >= 0.f) || hp->ns_steps < 1 || hp->ns_steps > 64)
        return MALT_ERR_INVALID_ARG;
    if (!(hp->lr == hp->lr) || !(hp->weight_decay == hp->weight_decay)) return MALT_ERR_INVALID_ARG;
    return MALT_OK;
}

void free_state(malt_state* st) {
    if (st == nullptr) return;
    for (cudaEvent_t e : {st->ev_g_consumed[0], st->ev_g_consumed[1], st->ev_h2d, st->ev_applied,
                          st->ev_d2h})
        if (e != nullptr) cudaEventDestroy(e);
    for (cudaStream_t q : {st->h2d, st->d2h})
        if (q != nullptr) cudaStreamDestroy(q);
    for (auto& p : st->ev_pending) {
        cudaEventDestroy(p.second.first);
        cudaEventDestroy(p.second.second);
    }
    for (cudaEvent_t e : st->ev_pool) cudaEventDestroy(e);
    if (st->ws != nullptr) cudaFree(st->ws);
    delete st;
}

cudaEvent_t take_event(malt_state* st) {
    if (!st->ev_pool.empty()) {
        cudaEvent_t e = st->ev_pool.back();
        st->ev_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

// NVTX range names of the kernel kinds (MALT_KIND_*), for timeline tools.
const char* const kKindRange[MALT_NUM_KINDS] = {
    "malt:bind", "malt:stats", "malt:finalize", "malt:prescale", "malt:norms", "malt:ns_gram",
    "malt:ns_poly", "malt:ns_bx", "malt:scalars", "malt:apply", "malt:ns_persistent", "malt:pad"};

// An NVTX range over a scope (host-side enqueue; a timeline tool maps it to
// the GPU work it launches).  Costs a pointer check when no tool is attached.
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

// Bracket one launch (or launch group) of a kernel kind with events when
// profiling is on, and with an NVTX range; always counts the launches.
struct LaunchScope {
    malt_state* st;
    int kind;
    cudaStream_t s;
    cudaEvent_t a = nullptr;
    NvtxRange range;
    LaunchScope(malt_state* st_, int kind_, cudaStream_t s_, int launches = 1)
        : st(st_), kind(kind_), s(s_), range(kKindRange[kind_]) {
        st->prof_launches[kind] += launches;
        if (st->profiling) {
            a = take_event(st);
            if (a != nullptr) cudaEventRecord(a, s);
        }
    }
    ~LaunchScope() {
        if (a == nullptr) return;
        cudaEvent_t b = take_event(st);
        if (b == nullptr) return;
        cudaEventRecord(b, s);
        st->ev_pending.push_back({kind, {a, b}});
    }
};

constexpr int kMaxStages = 3 * kMaxNsSteps;
// Auto schedule: persistent when a symmetric product has fewer tiles than
// this many waves of the resident CTA pairs.
constexpr int kAutoPersistentWaves = 16;
constexpr int kStatusWords = 8;

// Per-matrix descriptions and shape classes (one per NS frame p x q, in order
// of first appearance).  Host only.
void build_classes(const malt_param_t* params, int n, std::vector<MatDesc>& hmats,
                   std::vector<ShapeClass>& classes) {
    hmats.resize(n);
    std::map<std::pair<int, int>, int> cls_of;
    for (int i = 0; i < n; ++i) {
        // the kernels' view: rows and cols rounded up to multiples of 8
        const int m = static_cast<int>(round8(params[i].rows));
        const int c = static_cast<int>(round8(params[i].cols));
        const int p = std::min(m, c), q = std::max(m, c);
        auto it = cls_of.find({p, q});
        int k;
        if (it == cls_of.end()) {
            k = static_cast<int>(classes.size());
            cls_of[{p, q}] = k;
            classes.emplace_back();
            classes.back().p = p;
            classes.back().q = q;
        } else {
            k = it->second;
        }
        MatDesc& d = hmats[i];
        std::memset(&d, 0, sizeof(d));
        d.m = m;
        d.n = c;
        d.trans = m > c ? 1 : 0;
        d.p = p;
        d.q = q;
        d.w_bf16 = params[i].w_dtype == MALT_BF16;
        d.g_bf16 = params[i].g_dtype == MALT_BF16;
        d.cls = k;
        d.bidx = classes[k].batch++;
        classes[k].mats.push_back(i);
        d.stat_rb = (m + kStatRows - 1) / kStatRows;
        d.stat_cb = (c + kStatCols - 1) / kStatCols;
        d.pre_tr = (m + kPreRows - 1) / kPreRows;
        d.pre_tc = (c + kPreCols - 1) / kPreCols;
        d.ns_tiles = ((p + kTileM - 1) / kTileM) * ((q + kBN - 1) / kBN);
    }
}

// Newton-Schulz work lists: classes ordered by Gram reduction length (q, then
// p; the heaviest tiles are claimed first), in groups of up to kMaxClasses
// per launch.  Tensor maps and device pointers are copied from the classes
// as they stand (host-only callers leave them empty).  Host only.
void plan_ns_groups(const std::vector<ShapeClass>& classes, int nmat, std::vector<NsParams>& groups,
                    std::vector<std::vector<int>>* slot_class = nullptr) {
    std::vector<int> order(classes.size());
    for (size_t k = 0; k < order.size(); ++k) order[k] = static_cast<int>(k);
    std::stable_sort(order.begin(), order.end(), [&](int x, int y) {
        const ShapeClass& a = classes[x];
        const ShapeClass& b = classes[y];
        return a.q != b.q ? a.q > b.q : a.p > b.p;
    });
    groups.clear();
    if (slot_class != nullptr) slot_class->clear();
    for (size_t start = 0; start < order.size(); start += kMaxClasses) {
        groups.emplace_back();
        if (slot_class != nullptr) slot_class->emplace_back();
        NsParams& P = groups.back();
        std::memset(&P, 0, sizeof(P));
        const size_t cnt = std::min(order.size() - start, static_cast<size_t>(kMaxClasses));
        int32_t sym = 0, full = 0;
        for (size_t j = 0; j < cnt; ++j) {
            const ShapeClass& S = classes[order[start + j]];
            if (slot_class != nullptr) slot_class->back().push_back(order[start + j]);
            NsClass& C = P.cls[j];
            for (int b = 0; b < 2; ++b) {
                C.tmX[b] = S.tmX[b];
                C.tmXmn[b] = S.tmXmn[b];
                C.stX[b] = S.stX[b];
            }
            C.tmA = S.tmA;
            C.tmB = S.tmB;
            C.stA = S.stA;
            C.stB = S.stB;
            C.stO = S.stO;
            C.stOt = S.stOt;
            C.p = S.p;
            C.q = S.q;
            C.batch = S.batch;
            C.tiles_p = (S.p + kTileM - 1) / kTileM;
            C.tiles_q = (S.q + kBN - 1) / kBN;
            C.sym_begin = sym;
            C.full_begin = full;
            C.bx_col_major = static_cast<int64_t>(S.p) * S.q * 2 > kBxColBytes ? 1 : 0;
            C.mat_of = S.d_mat_of;
            C.A = S.A;
            sym += ns_phase_tiles(C, kGram) * S.batch;
            full += ns_phase_tiles(C, kBX) * S.batch;
        }
        P.nclasses = static_cast<int32_t>(cnt);
        P.nmat = nmat;
        P.sym_items = sym;
        P.full_items = full;
    }
}

// ------------------------------------------------------------- work tables
// Tiles of one matrix in one product of this kind.
int32_t stage_items(int kind, const NsClass& C) { return ns_phase_tiles(C, kind); }

// The work table of one launch group for k iterations: for each product of
// each iteration, every tile of every class (slot order), batch slot by
// batch slot.  Every item depends on the previous product of its own matrix,
// listed earlier: claiming in table order never waits on an item that has
// not been claimed.  The table of k iterations is the prefix of any longer
// one (an iteration adds entries at the end and changes none before it).
void build_table(const NsParams& G, const std::vector<int>& slot_class,
                 const std::vector<ShapeClass>& classes, int k, std::vector<NsEntry>& out) {
    out.clear();
    for (int st = 0; st < 3 * k; ++st) {
        const int kind = st % 3;
        for (int c = 0; c < G.nclasses; ++c) {
            const ShapeClass& S = classes[slot_class[c]];
            const int32_t items = stage_items(kind, G.cls[c]);
            const int32_t prev = st == 0 ? 0 : stage_items((st - 1) % 3, G.cls[c]);
            for (int b = 0; b < S.batch; ++b) {
                for (int t = 0; t < items; ++t) {
                    NsEntry e;
                    e.code = st | (c << 12) | (b << 16);
                    e.g = S.mats[b];
                    e.local = t;
                    e.target = kNsSignalsPerTile * static_cast<uint32_t>(prev);
                    out.push_back(e);
                }
            }
        }
    }
}

// Entries per iteration of a launch group's table.
int32_t table_per_iter(const NsParams& G) { return 2 * G.sym_items + G.full_items; }

int plan_and_allocate(malt_state* st, const malt_param_t* params, int n) {
    st->nmat = n;
    st->shape0.assign(params, params + n);
    st->wcopy.assign(n, nullptr);
    build_classes(params, n, st->hmats, st->classes);

    // Workspace layout.
    Carver cv;
    std::vector<size_t> o_row(n), o_col(n), o_L(n), o_R(n), o_pre(n), o_ns(n);
    for (int i = 0; i < n; ++i) {
        const MatDesc& d = st->hmats[i];
        o_row[i] = cv.take(sizeof(float) * static_cast<size_t>(d.stat_cb) * d.m);
        o_col[i] = cv.take(sizeof(float) * static_cast<size_t>(d.stat_rb) * d.n);
        o_L[i] = cv.take(sizeof(float) * d.m);
        o_R[i] = cv.take(sizeof(float) * d.n);
        o_pre[i] = cv.take(sizeof(float) * 2 * static_cast<size_t>(d.pre_tr) * d.pre_tc);
        o_ns[i] = cv.take(sizeof(float) * 2 * kNsPartsPerTile * static_cast<size_t>(d.ns_tiles));
    }
    const int nc = static_cast<int>(st->classes.size());
    std::vector<size_t> o_X0(nc), o_X1(nc), o_A(nc), o_B(nc), o_O(nc), o_matof(nc);
    for (int k = 0; k < nc; ++k) {
        const ShapeClass& C = st->classes[k];
        const size_t pq = static_cast<size_t>(C.batch) * C.p * C.q * 2;
        const size_t pp = static_cast<size_t>(C.batch) * C.p * C.p * 2;
        o_X0[k] = cv.take(pq);
        o_X1[k] = cv.take(pq);
        o_A[k] = cv.take(pp);
        o_B[k] = cv.take(pp);
        o_O[k] = cv.take(pq);
        o_matof[k] = cv.take(sizeof(int32_t) * C.batch);
    }
    const size_t o_mats = cv.take(sizeof(MatDesc) * std::max(n, 1));
    const size_t o_ptrs = cv.take(sizeof(UserPtrs) * std::max(n, 1));
    const size_t o_scal = cv.take(sizeof(MatScalars) * std::max(n, 1));
    const size_t o_t = cv.take(sizeof(long long));
    // status word, then the first timeout's site record (site, item, seq, block, thread)
    const size_t o_status = cv.take(sizeof(int32_t) * kStatusWords);
    size_t o_pref[4];
    for (int j = 0; j < 4; ++j) o_pref[j] = cv.take(sizeof(int32_t) * (n + 1));
    const size_t o_pre_ids = cv.take(sizeof(int32_t) * std::max(n, 1));
    const int ngroups = (nc + kMaxClasses - 1) / kMaxClasses;
    st->sched_groups_pad = ((ngroups + 63) / 64) * 64;
    const size_t o_sched = cv.take(sizeof(uint32_t) * (st->sched_groups_pad +
                                                       static_cast<size_t>(kMaxStages) * n));
    // Persistent work tables for kMaxNsSteps iterations, one per launch group
    // (planned here without tensor maps, which only the launches need).
    std::vector<std::vector<NsEntry>> tables;
    {
        std::vector<NsParams> groups;
        std::vector<std::vector<int>> slot_class;
        plan_ns_groups(st->classes, n, groups, &slot_class);
        tables.resize(groups.size());
        for (size_t gi = 0; gi < groups.size(); ++gi) {
            build_table(groups[gi], slot_class[gi], st->classes, kMaxNsSteps, tables[gi]);
            st->table_per_iter.push_back(table_per_iter(groups[gi]));
        }
    }
    // Zero-padded copies of matrices whose rows or cols are not multiples of 8.
    st->padbuf.assign(n, PadBuf{});
    std::vector<size_t> o_pw(n), o_pg(n), o_pm(n), o_pl(n), o_pr(n);
    for (int i = 0; i < n; ++i) {
        if (params[i].rows % 8 == 0 && params[i].cols % 8 == 0) continue;
        st->padded.push_back(i);
        const MatDesc& d = st->hmats[i];
        const size_t e = static_cast<size_t>(d.m) * d.n;
        o_pw[i] = cv.take(e * (params[i].w_dtype == MALT_BF16 ? 2 : 4));
        o_pg[i] = cv.take(e * (params[i].g_dtype == MALT_BF16 ? 2 : 4));
        o_pm[i] = cv.take(e * sizeof(float));
        o_pl[i] = cv.take(sizeof(float) * d.m);
        o_pr[i] = cv.take(sizeof(float) * d.n);
    }
    std::vector<size_t> o_table(tables.size());
    for (size_t gi = 0; gi < tables.size(); ++gi)
        o_table[gi] = cv.take(sizeof(NsEntry) * std::max<size_t>(tables[gi].size(), 1));

    // The guard list itself and the check's counter (not guarded).
    const size_t nguards = cv.guards.size();
    const size_t o_guard_off = cv.off;
    cv.off += (sizeof(uint64_t) * std::max<size_t>(nguards, 1) + 255) & ~static_cast<size_t>(255);
    const size_t o_guard_bad = cv.off;
    cv.off += 256;
    st->ws_bytes = cv.off;
    if (cudaMalloc(&st->ws, st->ws_bytes) != cudaSuccess) {
        st->ws = nullptr;
        cudaGetLastError();
        return MALT_ERR_OUT_OF_MEMORY;
    }
    uint8_t* base = static_cast<uint8_t*>(st->ws);
    auto F = [&](size_t o) { return reinterpret_cast<float*>(base + o); };
    auto H = [&](size_t o) { return reinterpret_cast<__nv_bfloat16*>(base + o); };
    for (int k = 0; k < nc; ++k) {
        ShapeClass& C = st->classes[k];
        C.X[0] = H(o_X0[k]);
        C.X[1] = H(o_X1[k]);
        C.A = H(o_A[k]);
        C.B = H(o_B[k]);
        C.O = H(o_O[k]);
        C.d_mat_of = reinterpret_cast<int32_t*>(base + o_matof[k]);
    }
    for (int i = 0; i < n; ++i) {
        MatDesc& d = st->hmats[i];
        const ShapeClass& C = st->classes[d.cls];
        d.rowpart = F(o_row[i]);
        d.colpart = F(o_col[i]);
        d.L = F(o_L[i]);
        d.R = F(o_R[i]);
        d.prepart = F(o_pre[i]);
        d.nspart = F(o_ns[i]);
        const size_t slot = static_cast<size_t>(d.bidx) * C.p * C.q;
        d.X0 = C.X[0] + slot;
        d.O = C.O + slot;
    }
    st->d_mats = reinterpret_cast<MatDesc*>(base + o_mats);
    st->d_ptrs = reinterpret_cast<UserPtrs*>(base + o_ptrs);
    st->d_scal = reinterpret_cast<MatScalars*>(base + o_scal);
    st->d_t = reinterpret_cast<long long*>(base + o_t);
    st->d_status = reinterpret_cast<int32_t*>(base + o_status);
    for (int j = 0; j < 4; ++j) st->d_pref[j] = reinterpret_cast<int32_t*>(base + o_pref[j]);
    st->d_pre_ids = reinterpret_cast<int32_t*>(base + o_pre_ids);
    st->d_sched = reinterpret_cast<uint32_t*>(base + o_sched);
    for (size_t gi = 0; gi < tables.size(); ++gi)
        st->table_dev.push_back(reinterpret_cast<NsEntry*>(base + o_table[gi]));
    for (int i : st->padded) {
        PadBuf& b = st->padbuf[i];
        b.w = base + o_pw[i];
        b.g = base + o_pg[i];
        b.m = F(o_pm[i]);
        b.l = F(o_pl[i]);
        b.r = F(o_pr[i]);
    }

    // Block-prefix tables.
    std::vector<int32_t> pref[4];
    for (int j = 0; j < 4; ++j) pref[j].assign(n + 1, 0);
    std::vector<int32_t> pre_ids;
    for (int tall = 0; tall < 2; ++tall)
        for (int i = 0; i < n; ++i)
            if (st->hmats[i].trans == tall) pre_ids.push_back(i);
    for (int i = 0; i < n; ++i) {
        const MatDesc& d = st->hmats[i];
        pref[0][i + 1] = pref[0][i] + d.stat_rb * d.stat_cb;
        pref[1][i + 1] = pref[1][i] + d.m + d.n;
        const MatDesc& e = st->hmats[pre_ids[i]];        // prescale order: wide, then tall
        pref[2][i + 1] = pref[2][i] + e.pre_tr * e.pre_tc;
        if (e.trans == 0) st->pre_wide = i + 1;
        // apply: contiguous runs of kApplyElems (O is in W's layout)
        pref[3][i + 1] = pref[3][i] + mat_apply_blocks(d);
    }
    st->blocks_stats = pref[0][n];
    st->total_fin = pref[1][n];
    st->blocks_pre = pref[2][n];
    st->blocks_pre_wide = pref[2][st->pre_wide];
    st->blocks_apply = pref[3][n];

    // Tensor maps of every class buffer.
    if (nc > 0 && !get_encoder()) return MALT_ERR_CUDA;
    for (int k = 0; k < nc; ++k) {
        ShapeClass& C = st->classes[k];
        bool ok = true;
        for (int b = 0; b < 2; ++b) {
            ok &= encode_3d(&C.tmX[b], C.X[b], C.q, C.p, C.batch, kBM);
            ok &= encode_3d(&C.tmXmn[b], C.X[b], C.q, C.p, C.batch, kBK);
        }
        ok &= encode_3d(&C.tmA, C.A, C.p, C.p, C.batch, kBM);
        ok &= encode_3d(&C.tmB, C.B, C.p, C.p, C.batch, kBM);
        for (int b = 0; b < 2; ++b) ok &= encode_store(&C.stX[b], C.X[b], C.q, C.p, C.batch);
        ok &= encode_store(&C.stA, C.A, C.p, C.p, C.batch);
        ok &= encode_store(&C.stB, C.B, C.p, C.p, C.batch);
        ok &= encode_store(&C.stO, C.O, C.q, C.p, C.batch);
        ok &= encode_store(&C.stOt, C.O, C.p, C.q, C.batch);
        if (!ok) {
            std::fprintf(stderr, "malt: cuTensorMapEncodeTiled failed for class %d x %d\n", C.p, C.q);
            return MALT_ERR_CUDA;
        }
    }
    plan_ns_groups(st->classes, n, st->ns_groups, &st->ns_slot_class);
    for (size_t gi = 0; gi < st->ns_groups.size(); ++gi) {
        NsParams& P = st->ns_groups[gi];
        P.mats = st->d_mats;
        P.scal = st->d_scal;
        P.status = st->d_status;
        P.queue = st->d_sched + gi;
        P.done = st->d_sched + st->sched_groups_pad;
        uint64_t kmax = 0;                // the Gram's K = q is the longest reduction
        for (int j = 0; j < P.nclasses; ++j) kmax = std::max<uint64_t>(kmax, P.cls[j].q);
        P.budget_ns = kWaitBudgetNs + kmax * kWaitNsPerK;
    }

    // Upload the static tables (init is allowed to synchronise).
    MALT_CUDA(cudaMemset(st->ws, 0, st->ws_bytes), "cudaMemset(workspace)");
    st->d_guard_off = reinterpret_cast<uint64_t*>(base + o_guard_off);
    st->d_guard_bad = reinterpret_cast<unsigned long long*>(base + o_guard_bad);
    st->nguards = static_cast<int32_t>(nguards);
    if (nguards > 0) {
        std::vector<uint64_t> goff(cv.guards.begin(), cv.guards.end());
        MALT_CUDA(cudaMemcpy(st->d_guard_off, goff.data(), sizeof(uint64_t) * nguards,
                             cudaMemcpyHostToDevice), "cudaMemcpy(guards)");
        MALT_CUDA(launch_guards(base, st->d_guard_off, st->nguards, false, st->d_guard_bad, nullptr),
                  "guard_kernel (fill)");
        MALT_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize(guards)");
    }
    if (n > 0) {
        MALT_CUDA(cudaMemcpy(st->d_mats, st->hmats.data(), sizeof(MatDesc) * n,
                             cudaMemcpyHostToDevice), "cudaMemcpy(mats)");
        for (int j = 0; j < 4; ++j)
            MALT_CUDA(cudaMemcpy(st->d_pref[j], pref[j].data(), sizeof(int32_t) * (n + 1),
                                 cudaMemcpyHostToDevice), "cudaMemcpy(prefix)");
        MALT_CUDA(cudaMemcpy(st->d_pre_ids, pre_ids.data(), sizeof(int32_t) * n,
                             cudaMemcpyHostToDevice), "cudaMemcpy(prescale order)");
        for (int k = 0; k < nc; ++k) {
            const ShapeClass& C = st->classes[k];
            MALT_CUDA(cudaMemcpy(C.d_mat_of, C.mats.data(), sizeof(int32_t) * C.batch,
                                 cudaMemcpyHostToDevice), "cudaMemcpy(mat_of)");
        }
        for (size_t gi = 0; gi < tables.size(); ++gi)
            MALT_CUDA(cudaMemcpy(st->table_dev[gi], tables[gi].data(),
                                 sizeof(NsEntry) * tables[gi].size(), cudaMemcpyHostToDevice),
                      "cudaMemcpy(work table)");
    }
    return MALT_OK;
}

int bind_pointers(malt_state* st, const malt_param_t* params, cudaStream_t s) {
    BindParams bp;
    for (int off = 0; off < st->nmat; off += kBindChunk) {
        const int cnt = std::min(kBindChunk, st->nmat - off);
        std::memset(&bp, 0, sizeof(bp));
        bp.count = cnt;
        bp.offset = off;
        for (int i = 0; i < cnt; ++i) {
            const malt_param_t& p = params[off + i];
            const PadBuf& b = st->padbuf[off + i];
            // A padded matrix's kernels work on its workspace copies; its
            // bf16 copy is written by the unpad launch, in the caller's layout.
            bp.p[i] = b.w != nullptr ? UserPtrs{b.w, b.g, b.m, b.l, b.r, nullptr}
                                     : UserPtrs{p.w, p.g, p.m, p.l, p.r, st->wcopy[off + i]};
        }
        LaunchScope ls(st, MALT_KIND_BIND, s);
        MALT_CUDA(launch_bind(bp, st->d_ptrs, s), "bind_kernel");
    }
    return MALT_OK;
}

// Copy the padded matrices' caller buffers into their workspace copies (in)
// or back (out), kPadChunk matrices per launch.
int run_padding(malt_state* st, const malt_param_t* params, bool in, cudaStream_t s) {
    thread_local PadParams P;
    for (size_t off = 0; off < st->padded.size(); off += kPadChunk) {
        const int cnt = static_cast<int>(std::min<size_t>(kPadChunk, st->padded.size() - off));
        std::memset(&P, 0, sizeof(P));
        P.count = cnt;
        int32_t blocks = 0;
        for (int k = 0; k < cnt; ++k) {
            const int i = st->padded[off + k];
            const malt_param_t& p = params[i];
            const PadBuf& b = st->padbuf[i];
            PadEntry& e = P.e[k];
            e.w_user = p.w;
            e.w_pad = b.w;
            e.g_user = p.g;
            e.g_pad = b.g;
            e.m_user = p.m;
            e.m_pad = b.m;
            e.l_user = p.l;
            e.l_pad = b.l;
            e.r_user = p.r;
            e.r_pad = b.r;
            e.wcopy_user = st->wcopy[i];
            e.m = static_cast<int32_t>(p.rows);
            e.n = static_cast<int32_t>(p.cols);
            e.n8 = st->hmats[i].n;
            e.w_bf16 = p.w_dtype == MALT_BF16;
            e.g_bf16 = p.g_dtype == MALT_BF16;
            e.block_begin = blocks;
            blocks += static_cast<int32_t>((p.rows + kPadRows - 1) / kPadRows);
        }
        LaunchScope ls(st, MALT_KIND_PAD, s);
        MALT_CUDA(launch_pad(P, blocks, in, s), in ? "pad_kernel (in)" : "pad_kernel (out)");
    }
    return MALT_OK;
}

// The k Newton-Schulz iterations over every class (after the norms kernel
// has set 1 / (||Mt|| + ns_eps)).
int run_newton_schulz(malt_state* st, const malt_hparams_t* hp, cudaStream_t s) {
    thread_local NsParams P;  // ~12 KB of tensor maps: keep off the stack
    const int k = hp->ns_steps;
    const int max_pairs = ns_gemm_max_pairs();
    auto prepare = [&](const NsParams& G) {
        P = G;
        P.ns_steps = k;
        P.a = hp->ns_a;
        P.b = hp->ns_b;
        P.c = hp->ns_c;
    };
    // Auto: the persistent schedule where a product is only a few waves of
    // CTA pairs deep (there the tails and launch gaps between products are a
    // large share of the time), the phased one where products are deep.
    auto persistent = [&](const NsParams& G) {
        if (st->ns_schedule != MALT_NS_AUTO) return st->ns_schedule == MALT_NS_PERSISTENT;
        return G.sym_items < kAutoPersistentWaves * max_pairs;
    };
    bool any_persistent = false;
    for (const NsParams& G : st->ns_groups) any_persistent |= persistent(G);
    if (any_persistent) {
        LaunchScope ls(st, MALT_KIND_NS_PERSISTENT, s, 0);   // launches counted below
        const size_t counters = st->sched_groups_pad + static_cast<size_t>(3 * k) * st->nmat;
        MALT_CUDA(cudaMemsetAsync(st->d_sched, 0, counters * sizeof(uint32_t), s),
                  "cudaMemsetAsync(schedule counters)");
        for (size_t gi = 0; gi < st->ns_groups.size(); ++gi) {
            const NsParams& G = st->ns_groups[gi];
            if (!persistent(G)) continue;
            prepare(G);
            const int items = k * st->table_per_iter[gi];
            P.table = st->table_dev[gi];
            P.nstages = 3 * k;
            P.item_begin = 0;
            P.item_end = items;
            const int pairs = std::max(1, std::min(items, max_pairs));
            ++st->prof_launches[MALT_KIND_NS_PERSISTENT];
            MALT_CUDA(launch_ns_gemm(P, kNsPersistent, pairs, s), "ns_gemm_kernel (persistent)");
        }
    }
    for (int it = 0; it < k; ++it) {
        for (int phase = kGram; phase <= kBX; ++phase) {
            for (const NsParams& G : st->ns_groups) {
                if (persistent(G)) continue;
                prepare(G);
                const int per_iter = 2 * G.sym_items + G.full_items;
                const int begin = it * per_iter + (phase == kGram ? 0
                                                   : phase == kPoly ? G.sym_items
                                                                    : 2 * G.sym_items);
                const int items = phase == kBX ? G.full_items : G.sym_items;
                P.item_begin = begin;
                P.item_end = begin + items;
                const int pairs = std::max(1, std::min(items, max_pairs));
                LaunchScope ls(st, MALT_KIND_NS_GRAM + phase, s);
                MALT_CUDA(launch_ns_gemm(P, kNsPhased, pairs, s), "ns_gemm_kernel");
            }
        }
    }
    return MALT_OK;
}

int validate_step(malt_state* st, const malt_param_t* params, int32_t n,
                  const malt_hparams_t* hp) {
    if (st == nullptr || (n > 0 && params == nullptr)) return MALT_ERR_INVALID_ARG;
    int rc = validate_hparams(hp);
    if (rc != MALT_OK) return rc;
    if (n != st->nmat) return MALT_ERR_SHAPE_CHANGED;
    for (int i = 0; i < n; ++i) {
        rc = validate_param(params[i]);
        if (rc != MALT_OK) return rc;
        const malt_param_t& a = st->shape0[i];
        if (a.rows != params[i].rows || a.cols != params[i].cols ||
            a.w_dtype != params[i].w_dtype || a.g_dtype != params[i].g_dtype)
            return MALT_ERR_SHAPE_CHANGED;
    }
    return MALT_OK;
}

// Update flavours sharing the engine: MALT (Algorithm 1), MALTER (Algorithm 2),
// and Muon with the same EMA momentum (identity preconditioners, no statistics).
enum Flavour { kMalt = 0, kMalter = 1, kMuon = 2 };

StepHyper step_hyper(const malt_hparams_t* hp, int malter) {
    StepHyper sh;
    sh.lr = hp->lr;
    sh.mu1 = hp->mu1;
    sh.mu2 = hp->mu2;
    sh.eps = hp->eps;
    sh.weight_decay = hp->weight_decay;
    sh.ns_a = hp->ns_a;
    sh.ns_b = hp->ns_b;
    sh.ns_c = hp->ns_c;
    sh.ns_eps = hp->ns_eps;
    sh.malter = malter;
    return sh;
}

int run_step(malt_state* st, const malt_param_t* params, int32_t n, const malt_hparams_t* hp,
             void* stream, int flavour, const PipeHooks* hooks = nullptr) {
    const NvtxRange range(flavour == kMalter ? "malter_step" : flavour == kMuon ? "muon_step" : "malt_step");
    const int malter = flavour == kMalter ? 1 : 0;
    const int muon = flavour == kMuon ? 1 : 0;
    int rc = validate_step(st, params, n, hp);
    if (rc != MALT_OK) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    st->last_stream = s;
    if (n == 0) return MALT_OK;
    MALT_CUDA(cudaSetDevice(st->device), "cudaSetDevice");
    rc = bind_pointers(st, params, s);
    if (rc != MALT_OK) return rc;
    if (!st->padded.empty()) {
        // The padded copies are overwritten: the previous host step's weight
        // read-back must be done (the read-back reads the caller's W).
        rc = run_padding(st, params, true, s);
        if (rc != MALT_OK) return rc;
    }
    const int nm = st->nmat;
    {
        LaunchScope ls(st, MALT_KIND_STATS, s);
        MALT_CUDA(launch_stats(st->d_mats, st->d_ptrs, st->d_pref[0], nm, st->blocks_stats,
                               hp->mu1, !muon, s), "stats_kernel");
    }
    {
        LaunchScope ls(st, MALT_KIND_FINALIZE, s);
        MALT_CUDA(launch_finalize(st->d_mats, st->d_ptrs, st->d_pref[1], nm, st->total_fin,
                                  hp->mu2, hp->eps, st->d_t, muon, s), "finalize_kernel");
    }
    {
        const int wide = st->pre_wide, tall = nm - st->pre_wide;
        LaunchScope ls(st, MALT_KIND_PRESCALE, s, (wide > 0) + (tall > 0));
        MALT_CUDA(launch_prescale(st->d_mats, st->d_ptrs, st->d_pre_ids, st->d_pref[2], wide,
                                  st->blocks_pre_wide, tall, st->blocks_pre - st->blocks_pre_wide,
                                  malter, s), "prescale kernels");
    }
    if (hooks != nullptr)   // stats and prescale are the only readers of G
        MALT_CUDA(cudaEventRecord(hooks->record_g_consumed, s), "cudaEventRecord(G consumed)");
    {
        LaunchScope ls(st, MALT_KIND_NORMS, s);
        MALT_CUDA(launch_norms(st->d_mats, st->d_scal, nm, hp->ns_eps, malter, s), "norms_kernel");
    }
    rc = run_newton_schulz(st, hp, s);
    if (rc != MALT_OK) return rc;
    const StepHyper sh = step_hyper(hp, malter);
    {
        LaunchScope ls(st, MALT_KIND_SCALARS, s);
        MALT_CUDA(launch_scalars(st->d_mats, st->d_scal, st->d_t, nm, sh, s), "scalars_kernel");
    }
    if (hooks != nullptr && hooks->wait_before_apply != nullptr)
        MALT_CUDA(cudaStreamWaitEvent(s, hooks->wait_before_apply, 0), "cudaStreamWaitEvent(W read)");
    {
        LaunchScope ls(st, MALT_KIND_APPLY, s);
        MALT_CUDA(launch_apply(st->d_mats, st->d_ptrs, st->d_scal, st->d_pref[3], nm,
                               st->blocks_apply, 1.f - hp->lr * hp->weight_decay, s),
                  "apply_kernel");
    }
    if (!st->padded.empty()) {
        rc = run_padding(st, params, false, s);
        if (rc != MALT_OK) return rc;
    }
    if (hooks != nullptr)
        MALT_CUDA(cudaEventRecord(hooks->record_applied, s), "cudaEventRecord(applied)");
    return MALT_OK;
}

size_t elem_bytes(int32_t dtype) { return dtype == MALT_BF16 ? 2 : 4; }

int ensure_pipe(malt_state* st) {
    if (st->h2d != nullptr) return MALT_OK;
    MALT_CUDA(cudaStreamCreateWithFlags(&st->h2d, cudaStreamNonBlocking), "cudaStreamCreate(h2d)");
    MALT_CUDA(cudaStreamCreateWithFlags(&st->d2h, cudaStreamNonBlocking), "cudaStreamCreate(d2h)");
    for (cudaEvent_t* e : {&st->ev_g_consumed[0], &st->ev_g_consumed[1], &st->ev_h2d,
                           &st->ev_applied, &st->ev_d2h})
        MALT_CUDA(cudaEventCreateWithFlags(e, cudaEventDisableTiming), "cudaEventCreate");
    return MALT_OK;
}

// Slot of the "G consumed" event for this device gradient buffer set, and
// the copy stream's wait before gradients are copied into the set: for a set
// among the last two used, the last step that read it; for any other set
// (new, or last used further back), the latest consumption recorded in either
// slot, which on one compute stream follows every earlier step's.
int g_slot_wait(malt_state* st, const void* key, int* slot) {
    for (int k = 0; k < malt_state::kGSlots; ++k) {
        if (st->g_key[k] != key) continue;
        if (st->g_recorded[k])
            MALT_CUDA(cudaStreamWaitEvent(st->h2d, st->ev_g_consumed[k], 0), "cudaStreamWaitEvent(G)");
        *slot = k;
        return MALT_OK;
    }
    for (int k = 0; k < malt_state::kGSlots; ++k)
        if (st->g_recorded[k])
            MALT_CUDA(cudaStreamWaitEvent(st->h2d, st->ev_g_consumed[k], 0), "cudaStreamWaitEvent(G)");
    const int k = st->g_next_slot;
    st->g_next_slot = (k + 1) % malt_state::kGSlots;
    st->g_key[k] = key;
    st->g_recorded[k] = false;
    *slot = k;
    return MALT_OK;
}

int run_host_step(malt_state* st, const malt_param_t* params, int32_t n, const malt_hparams_t* hp,
                  int flavour, const void* const* g_host, void* const* w_host, void* stream) {
    int rc = validate_step(st, params, n, hp);
    if (rc != MALT_OK) return rc;
    if (n > 0 && (g_host == nullptr || w_host == nullptr)) return MALT_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i)
        if (g_host[i] == nullptr || w_host[i] == nullptr) return MALT_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (n == 0) {
        st->last_stream = s;
        return MALT_OK;
    }
    MALT_CUDA(cudaSetDevice(st->device), "cudaSetDevice");
    rc = ensure_pipe(st);
    if (rc != MALT_OK) return rc;
    // Gradients in: wait until the steps that read this device G set have
    // consumed it.  (A step whose set differs may still be running.)
    int slot = 0;
    rc = g_slot_wait(st, params[0].g, &slot);
    if (rc != MALT_OK) return rc;
    for (int i = 0; i < n; ++i) {
        const size_t bytes = static_cast<size_t>(params[i].rows) * params[i].cols *
                             elem_bytes(params[i].g_dtype);
        MALT_CUDA(cudaMemcpyAsync(const_cast<void*>(params[i].g), g_host[i], bytes,
                                  cudaMemcpyHostToDevice, st->h2d), "cudaMemcpyAsync(G in)");
    }
    MALT_CUDA(cudaEventRecord(st->ev_h2d, st->h2d), "cudaEventRecord(h2d)");
    MALT_CUDA(cudaStreamWaitEvent(s, st->ev_h2d, 0), "cudaStreamWaitEvent(h2d)");
    const PipeHooks hooks{st->ev_g_consumed[slot], st->pipe_primed ? st->ev_d2h : nullptr,
                          st->ev_applied};
    rc = run_step(st, params, n, hp, stream, flavour, &hooks);
    if (rc != MALT_OK) return rc;
    st->g_recorded[slot] = true;
    // Weights out, overlapping the next step's statistics and Newton-Schulz work.
    MALT_CUDA(cudaStreamWaitEvent(st->d2h, st->ev_applied, 0), "cudaStreamWaitEvent(applied)");
    for (int i = 0; i < n; ++i) {
        const size_t bytes = static_cast<size_t>(params[i].rows) * params[i].cols *
                             elem_bytes(params[i].w_dtype);
        MALT_CUDA(cudaMemcpyAsync(w_host[i], params[i].w, bytes, cudaMemcpyDeviceToHost, st->d2h),
                  "cudaMemcpyAsync(W out)");
    }
    MALT_CUDA(cudaEventRecord(st->ev_d2h, st->d2h), "cudaEventRecord(d2h)");
    st->pipe_primed = true;
    return MALT_OK;
}

}  // namespace

extern "C" {

int malt_init_state(malt_state_t** out, const malt_param_t* params, int32_t n, void* stream) {
    if (out == nullptr) return MALT_ERR_INVALID_ARG;
    *out = nullptr;
    if (n < 0 || (n > 0 && params == nullptr)) return MALT_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i) {
        const int rc = validate_param(params[i]);
        if (rc != MALT_OK) return rc;
    }
    malt_state* st = new malt_state();
    int rc = cuda_fail(cudaGetDevice(&st->device), "cudaGetDevice");
    if (rc == MALT_OK)
        rc = cuda_fail(cudaDeviceGetAttribute(&st->num_sms, cudaDevAttrMultiProcessorCount, st->device),
                       "cudaDeviceGetAttribute");
    if (rc == MALT_OK) rc = plan_and_allocate(st, params, n);
    // One-time kernel configuration (shared-memory opt-in, resident CTA pairs)
    // happens here, so a first step taken inside a stream capture makes no
    // such calls.
    if (rc == MALT_OK && n > 0) rc = cuda_fail(ns_gemm_configure(), "ns_gemm_configure");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    for (int i = 0; rc == MALT_OK && i < n; ++i) {
        const malt_param_t& p = params[i];
        const size_t e = static_cast<size_t>(p.rows) * p.cols;
        rc = cuda_fail(cudaMemsetAsync(p.m, 0, e * sizeof(float), s), "cudaMemsetAsync(M)");
        if (rc == MALT_OK) rc = cuda_fail(cudaMemsetAsync(p.l, 0, p.rows * sizeof(float), s), "memset(l)");
        if (rc == MALT_OK) rc = cuda_fail(cudaMemsetAsync(p.r, 0, p.cols * sizeof(float), s), "memset(r)");
    }
    if (rc != MALT_OK) {
        free_state(st);
        return rc;
    }
    st->last_stream = s;
    *out = st;
    return MALT_OK;
}

int malt_step(malt_state_t* st, const malt_param_t* params, int32_t n, const malt_hparams_t* hp,
              void* stream) {
    return run_step(st, params, n, hp, stream, kMalt);
}

int malter_step(malt_state_t* st, const malt_param_t* params, int32_t n, const malt_hparams_t* hp,
                void* stream) {
    return run_step(st, params, n, hp, stream, kMalter);
}

int muon_step(malt_state_t* st, const malt_param_t* params, int32_t n, const malt_hparams_t* hp,
              void* stream) {
    return run_step(st, params, n, hp, stream, kMuon);
}

int malt_step_host(malt_state_t* st, const malt_param_t* params, int32_t n,
                   const malt_hparams_t* hp, int32_t malter, const void* const* g_host,
                   void* const* w_host, void* stream) {
    return run_host_step(st, params, n, hp, malter != 0 ? kMalter : kMalt, g_host, w_host, stream);
}

int malt_check(malt_state_t* st) {
    if (st == nullptr) return MALT_ERR_INVALID_ARG;
    MALT_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    if (st->d2h != nullptr) {
        MALT_CUDA(cudaStreamSynchronize(st->h2d), "cudaStreamSynchronize(h2d)");
        MALT_CUDA(cudaStreamSynchronize(st->d2h), "cudaStreamSynchronize(d2h)");
    }
    if (st->ws == nullptr) return MALT_OK;
    int32_t status[kStatusWords] = {};
    MALT_CUDA(cudaMemcpy(status, st->d_status, sizeof(status), cudaMemcpyDeviceToHost),
              "cudaMemcpy(status)");
    if (status[0] != 0) {
        std::memcpy(st->last_timeout, status + 1, sizeof(st->last_timeout));
        MALT_CUDA(cudaMemset(st->d_status, 0, sizeof(status)), "cudaMemset(status)");
        return MALT_ERR_TIMEOUT;
    }
    return MALT_OK;
}

int malt_get_scalars(malt_state_t* st, float* nu_host, int32_t n, int64_t* t_host) {
    if (st == nullptr || n != st->nmat || (n > 0 && nu_host == nullptr) || t_host == nullptr)
        return MALT_ERR_INVALID_ARG;
    MALT_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    long long t = 0;
    MALT_CUDA(cudaMemcpy(&t, st->d_t, sizeof(t), cudaMemcpyDeviceToHost), "cudaMemcpy(t)");
    *t_host = t;
    if (n > 0) {
        std::vector<MatScalars> s(n);
        MALT_CUDA(cudaMemcpy(s.data(), st->d_scal, sizeof(MatScalars) * n, cudaMemcpyDeviceToHost),
                  "cudaMemcpy(scalars)");
        for (int i = 0; i < n; ++i) nu_host[i] = s[i].nu;
    }
    return MALT_OK;
}

int malt_set_scalars(malt_state_t* st, const float* nu_host, int32_t n, int64_t t_host) {
    if (st == nullptr || n != st->nmat || (n > 0 && nu_host == nullptr) || t_host < 0)
        return MALT_ERR_INVALID_ARG;
    MALT_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    const long long t = t_host;
    MALT_CUDA(cudaMemcpy(st->d_t, &t, sizeof(t), cudaMemcpyHostToDevice), "cudaMemcpy(t)");
    if (n > 0) {
        std::vector<MatScalars> s(n);
        MALT_CUDA(cudaMemcpy(s.data(), st->d_scal, sizeof(MatScalars) * n, cudaMemcpyDeviceToHost),
                  "cudaMemcpy(scalars)");
        for (int i = 0; i < n; ++i) s[i].nu = nu_host[i];
        MALT_CUDA(cudaMemcpy(st->d_scal, s.data(), sizeof(MatScalars) * n, cudaMemcpyHostToDevice),
                  "cudaMemcpy(scalars)");
    }
    return MALT_OK;
}

int malt_debug_direction(malt_state_t* st, int32_t idx, void* out, void* stream) {
    if (st == nullptr || idx < 0 || idx >= st->nmat || out == nullptr) return MALT_ERR_INVALID_ARG;
    const MatDesc& d = st->hmats[idx];
    const malt_param_t& p = st->shape0[idx];
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // O is stored in W's layout for every matrix (the last B*X epilogue
    // writes a tall matrix's tiles transposed), with leading dimension d.n
    // (cols rounded up to 8); the caller's copy is rows x cols, dense.
    MALT_CUDA(cudaMemcpy2DAsync(out, static_cast<size_t>(p.cols) * 2, d.O, static_cast<size_t>(d.n) * 2,
                                static_cast<size_t>(p.cols) * 2, static_cast<size_t>(p.rows),
                                cudaMemcpyDeviceToDevice, s), "cudaMemcpy2DAsync(O)");
    return MALT_OK;
}

int malt_debug_precond(malt_state_t* st, int32_t idx, float* L_out, float* R_out, void* stream) {
    if (st == nullptr || idx < 0 || idx >= st->nmat || L_out == nullptr || R_out == nullptr)
        return MALT_ERR_INVALID_ARG;
    const MatDesc& d = st->hmats[idx];
    const malt_param_t& p = st->shape0[idx];
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    MALT_CUDA(cudaMemcpyAsync(L_out, d.L, sizeof(float) * p.rows, cudaMemcpyDeviceToDevice, s),
              "cudaMemcpyAsync(L)");
    MALT_CUDA(cudaMemcpyAsync(R_out, d.R, sizeof(float) * p.cols, cudaMemcpyDeviceToDevice, s),
              "cudaMemcpyAsync(R)");
    return MALT_OK;
}

int malt_debug_check_guards(malt_state_t* st, int64_t* bad_bytes) {
    if (st == nullptr || bad_bytes == nullptr) return MALT_ERR_INVALID_ARG;
    *bad_bytes = 0;
    if (st->nguards == 0) return MALT_OK;
    cudaStream_t s = st->last_stream;
    MALT_CUDA(cudaMemsetAsync(st->d_guard_bad, 0, sizeof(unsigned long long), s), "cudaMemsetAsync(guard count)");
    MALT_CUDA(launch_guards(st->ws, st->d_guard_off, st->nguards, true, st->d_guard_bad, s),
              "guard_kernel (check)");
    unsigned long long bad = 0;
    MALT_CUDA(cudaMemcpyAsync(&bad, st->d_guard_bad, sizeof(bad), cudaMemcpyDeviceToHost, s),
              "cudaMemcpyAsync(guard count)");
    MALT_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    *bad_bytes = static_cast<int64_t>(bad);
    return MALT_OK;
}

int malt_debug_scalars(malt_state_t* st, float* out_host, int32_t n) {
    if (st == nullptr || n != st->nmat || (n > 0 && out_host == nullptr)) return MALT_ERR_INVALID_ARG;
    MALT_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    if (n == 0) return MALT_OK;
    std::vector<MatScalars> s(n);
    MALT_CUDA(cudaMemcpy(s.data(), st->d_scal, sizeof(MatScalars) * n, cudaMemcpyDeviceToHost),
              "cudaMemcpy(scalars)");
    for (int i = 0; i < n; ++i) {
        float* o = out_host + static_cast<size_t>(i) * kScalarsPerMat;
        o[0] = s[i].norm_o;
        o[1] = s[i].norm_d;
        o[2] = s[i].norm_mt;
        o[3] = s[i].lgr_sq;
        o[4] = s[i].nu;
        o[5] = s[i].alpha;
        o[6] = s[i].scale;
        o[7] = s[i].k;
    }
    return MALT_OK;
}

int malt_debug_wait_timeout(int64_t budget_ns, void* stream) {
    if (budget_ns <= 0) return MALT_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t* d = nullptr;
    MALT_CUDA(cudaMalloc(&d, sizeof(int32_t)), "cudaMalloc(probe)");
    int rc = cuda_fail(cudaMemsetAsync(d, 0, sizeof(int32_t), s), "cudaMemsetAsync(probe)");
    if (rc == MALT_OK) rc = cuda_fail(launch_wait_probe(d, static_cast<uint64_t>(budget_ns), s), "wait_probe");
    if (rc == MALT_OK) rc = cuda_fail(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    int32_t h = 0;
    if (rc == MALT_OK) rc = cuda_fail(cudaMemcpy(&h, d, sizeof(h), cudaMemcpyDeviceToHost), "cudaMemcpy(probe)");
    cudaFree(d);
    if (rc != MALT_OK) return rc;
    return h != 0 ? MALT_ERR_TIMEOUT : MALT_OK;
}

int malt_profile_enable(malt_state_t* st, int32_t enable) {
    if (st == nullptr) return MALT_ERR_INVALID_ARG;
    st->profiling = enable != 0;
    return MALT_OK;
}

int malt_profile_read(malt_state_t* st, double* ms_out, int64_t* launches_out, int32_t nkinds) {
    if (st == nullptr || nkinds < 0 || nkinds > MALT_NUM_KINDS ||
        (nkinds > 0 && (ms_out == nullptr || launches_out == nullptr)))
        return MALT_ERR_INVALID_ARG;
    MALT_CUDA(cudaStreamSynchronize(st->last_stream), "cudaStreamSynchronize");
    for (auto& p : st->ev_pending) {
        float ms = 0.f;
        MALT_CUDA(cudaEventElapsedTime(&ms, p.second.first, p.second.second), "cudaEventElapsedTime");
        st->prof_ms[p.first] += ms;
        st->ev_pool.push_back(p.second.first);
        st->ev_pool.push_back(p.second.second);
    }
    st->ev_pending.clear();
    for (int k = 0; k < nkinds; ++k) {
        ms_out[k] = st->prof_ms[k];
        launches_out[k] = st->prof_launches[k];
    }
    for (int k = 0; k < MALT_NUM_KINDS; ++k) {
        st->prof_ms[k] = 0.0;
        st->prof_launches[k] = 0;
    }
    return MALT_OK;
}

size_t malt_workspace_bytes(const malt_state_t* st) { return st == nullptr ? 0 : st->ws_bytes; }

int malt_debug_timeout_site(const malt_state_t* st, int32_t* out5) {
    if (st == nullptr || out5 == nullptr) return MALT_ERR_INVALID_ARG;
    std::memcpy(out5, st->last_timeout, sizeof(st->last_timeout));
    return MALT_OK;
}

int malt_set_weight_copies(malt_state_t* st, void* const* copies, int32_t n) {
    if (st == nullptr || n != st->nmat) return MALT_ERR_INVALID_ARG;
    for (int i = 0; copies != nullptr && i < n; ++i) {
        if (copies[i] == nullptr) continue;
        if (st->shape0[i].w_dtype != MALT_F32) return MALT_ERR_UNSUPPORTED;
        if (!aligned16(copies[i])) return MALT_ERR_MISALIGNED;
    }
    for (int i = 0; i < n; ++i) st->wcopy[i] = copies != nullptr ? copies[i] : nullptr;
    return MALT_OK;
}

int malt_set_ns_schedule(malt_state_t* st, int32_t schedule) {
    if (st == nullptr || (schedule != MALT_NS_PHASED && schedule != MALT_NS_PERSISTENT &&
                          schedule != MALT_NS_AUTO))
        return MALT_ERR_INVALID_ARG;
    st->ns_schedule = schedule;
    return MALT_OK;
}

int malt_ns_schedule(const malt_param_t* params, int32_t n, int32_t ns_steps, int32_t* out,
                     int64_t capacity, int64_t* count) {
    if (count == nullptr || n < 0 || (n > 0 && params == nullptr) || ns_steps < 1 ||
        ns_steps > kMaxNsSteps || capacity < 0 || (capacity > 0 && out == nullptr))
        return MALT_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i)
        if (params[i].rows <= 0 || params[i].cols <= 0 ||
            round8(params[i].rows) * round8(params[i].cols) >= (int64_t{1} << 31))
            return MALT_ERR_UNSUPPORTED;
    std::vector<MatDesc> hmats;
    std::vector<ShapeClass> classes;
    build_classes(params, n, hmats, classes);
    std::vector<NsParams> groups;
    std::vector<std::vector<int>> slot_class;
    plan_ns_groups(classes, n, groups, &slot_class);
    int64_t total = 0;
    std::vector<NsEntry> table;
    for (size_t gi = 0; gi < groups.size(); ++gi) {
        const NsParams& G = groups[gi];
        build_table(G, slot_class[gi], classes, ns_steps, table);
        for (const NsEntry& e : table) {
            if (total < capacity) {
                const int st = entry_stage(e);
                const int kind = st % 3;
                int32_t* o = out + total * 8;
                o[0] = static_cast<int32_t>(gi);
                o[1] = st;
                o[2] = kind;
                o[3] = e.g;
                o[4] = e.local;
                o[5] = e.target > 0 ? (st - 1) * n + e.g : -1;
                o[6] = static_cast<int32_t>(e.target);
                o[7] = stage_items(kind, G.cls[entry_cls(e)]);
            }
            ++total;
        }
    }
    *count = total;
    return MALT_OK;
}

const char* malt_status_string(int code) {
    switch (code) {
        case MALT_OK: return "ok";
        case MALT_ERR_INVALID_ARG: return "invalid argument";
        case MALT_ERR_UNSUPPORTED: return "unsupported shape or dtype (rows and cols must be positive, with rows*cols < 2^31 after rounding each up to a multiple of 8)";
        case MALT_ERR_MISALIGNED: return "device pointer not 16-byte aligned";
        case MALT_ERR_SHAPE_CHANGED: return "parameter shapes or dtypes differ from init";
        case MALT_ERR_CUDA: return "CUDA runtime error";
        case MALT_ERR_TIMEOUT: return "device-side wait timed out";
        case MALT_ERR_OUT_OF_MEMORY: return "workspace allocation failed";
        default: return "unknown status";
    }
}

void malt_destroy_state(malt_state_t* st) {
    if (st == nullptr) return;
    cudaStreamSynchronize(st->last_stream);
    if (st->d2h != nullptr) {
        cudaStreamSynchronize(st->h2d);
        cudaStreamSynchronize(st->d2h);
    }
    free_state(st);
}

}  // extern "C"
