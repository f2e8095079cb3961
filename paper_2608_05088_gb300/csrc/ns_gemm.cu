// ns_gemm.cu -- the Newton-Schulz engine: batched same-shape bf16 GEMMs on the
// sm_103a tensor cores, two SMs per tile (tcgen05.mma.cta_group::2, fp32
// accumulators in TMEM, operands staged into shared memory by TMA with
// 128-byte swizzle).
//
// One Newton-Schulz iteration (the Orth step of Algorithm 1, run on the wide
// orientation X of Mt, p x q) is three launches of this kernel:
//   kGram  A  = X X^T               (M = N = p, K = q)    operands: rows of X, rows of X
//   kPoly  B' = a I + b A + c A A   (M = N = p, K = p)    operands: rows of A, rows of A (A = A^T)
// A and B' are symmetric, so those two phases compute only the tiles on and
// above the diagonal and store each off-diagonal tile twice (as is and
// transposed); the products are then exactly symmetric.
//   kBX    X' = B' X                (M = p, N = q, K = p) operands: rows of B', X read MN-major
// so a X + (b A + c A A) X = B' X with the a X term folded into B' (its error
// is that of the bf16 B it rides on).  The kBX B operand is X itself, read as
// an MN-major [K][N] matrix, so no transposed copy of X is ever written.  The
// 1/(||Mt||_F + ns_eps) normalisation is folded into the first iteration's
// epilogues (A scaled by k^2, X' by k).  The last iteration's epilogue writes O
// in W's orientation and per-warp partial sums of O^2 and of D^2 with
// D = L O R (Algorithm 1, D_t line) for the graft.  O is stored in W's layout:
// a tall matrix's tiles go out transposed (the staging used for the mirror
// of a symmetric tile), so the apply pass streams every matrix the same way.
//
// Work split.  A cluster of two CTAs (a CTA pair on two SMs) computes one
// 256 x 256 output tile per turn: CTA r owns rows [128 r, 128 r + 128) of the
// tile in its own TMEM.  Per 64-wide reduction slice each CTA loads its 128
// rows of A and its half (128 N-rows or N-columns) of B, 32 KB, into one of
// kStages slice slots; the MMA, issued by one thread of the even CTA, reads
// both CTAs' shared memory.  Each SM therefore pulls 32 KB from L2 per
// 128 x 256 x 64 of MMA work instead of 48 KB (16 KB on a diagonal tile of
// a symmetric product, whose B half is the CTA's own A rows).  The slots are filled,
// awaited and released in groups of kGroup slices (a 3-stage ring of 128-wide
// reductions): every barrier wait and commit on the MMA thread's path stalls
// the tensor pipe a little, and one per 8 MMAs measured 4 % faster on B*X
// than one per 4.
//
// Roles per CTA: warp 0 issues TMA loads (the peer's loads complete on the
// even CTA's full barrier, and both producers arrive on it), warp 1 owns
// TMEM (allocated for the pair) and, in the even CTA, issues tcgen05.mma into
// one of two TMEM accumulators; warps 2-9 drain the other accumulator
// (tcgen05.ld, pipelined per 32-column chunk) and run the epilogue, so the
// epilogue of tile i overlaps the MMAs of tile i+1.  Each epilogue warp
// converts its 32 x 32 chunk to bf16 in a double-buffered shared-memory box
// (64-byte swizzle, bank-conflict free) and writes it with one TMA bulk
// tensor store.  MMA completion is multicast to both CTAs' barriers; both
// CTAs' epilogue warps release an accumulator on the even CTA's barrier.
// Every wait is bounded; a timeout sets the status word (and records where,
// for malt_debug_timeout_site) and the CTA winds down.
//
// Schedules.  A launch runs a range of the work list (NsParams): every tile
// of every product of every NS iteration, product by product.
//  * Phased: one launch per product (Gram, Poly, BX of one iteration); pair
//    j takes items j, j + npairs, ...  The stream orders the products.
//  * Persistent: one launch for all k iterations.  A scheduler thread per
//    pair (the odd CTA's otherwise idle MMA-warp thread) claims the next
//    item with an atomic on a global counter, waits (bounded, acquire) until
//    the previous product of the item's matrix is complete -- every epilogue
//    warp of every tile of that product has signalled done[] after its TMA
//    stores completed -- and publishes the item to a 4-slot ring in both
//    CTAs' shared memory (st.async messages on mbarriers), a few items ahead
//    of the producers, MMA and epilogues that read it.  Each product of a
//    matrix depends only on the previous product of the same matrix, so
//    tiles of the next product of one matrix start while the current
//    product of another matrix is still running: no grid-wide barrier
//    between products, no launch gaps, no wave tails except the last.
//    Items are claimed in list order by running CTAs only, so every item a
//    tile waits for is held by a CTA that is running and whose own
//    dependencies come earlier still: the schedule cannot deadlock, whatever
//    number of CTA pairs is resident.
//  Both schedules run the same per-tile arithmetic, so their results are
//  bitwise identical.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace malt {

namespace {

constexpr int kEpiWarps = kEpiWarpsPerCta;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kEpiCols = kBN / (kEpiWarps / 4);        // accumulator columns per warp
constexpr int kEpiChunks = kEpiCols / 32;
constexpr int kHalfN = kBN / 2;                        // B rows (or columns) per CTA
constexpr uint32_t kABytes = kBM * kBK * 2;            // 16 KB
constexpr uint32_t kBBytes = kHalfN * kBK * 2;         // 16 KB
constexpr uint32_t kStageBytes = kABytes + kBBytes;     // one 64-wide reduction slice
// Ring granularity: the producer fills, and the MMA thread waits for and
// releases, kGroup slices at a time.  A barrier wait and a commit sit on the
// MMA issue path once per kGroup slices (8 MMAs) instead of once per 4 MMAs.
constexpr int kGroup = 2;
constexpr int kRing = kStages / kGroup;
static_assert(kStages % kGroup == 0, "the slice slots form whole ring stages");
constexpr uint32_t kTmemCols = 2 * kBN;
constexpr uint32_t kIdesc = idesc_bf16_f32(kTileM, kBN);
constexpr uint32_t kIdescBmn = idesc_bf16_f32(kTileM, kBN, true);
constexpr uint32_t kMnBoxBytes = kBMN * kBK * 2;       // one 64 x 64 MN-major box
constexpr uint32_t kMnLbo = kMnBoxBytes;               // next 64 MN-elements
constexpr uint32_t kStoreBoxBytes = 32 * 32 * 2;      // one 32 x 32 bf16 output box
constexpr uint32_t kStageOutBytes = 2 * kStoreBoxBytes * kEpiWarps;  // double-buffered per warp
constexpr size_t kSmemBytes =
    static_cast<size_t>(kStages) * kStageBytes + kStageOutBytes + 1024;
constexpr uint16_t kPairMask = 0x3;
// Persistent schedule: slots of the item ring (how far the scheduler may run
// ahead of the slowest reader, the epilogue), and the readers of each slot:
// both producers, the even CTA's MMA thread, every epilogue warp of both CTAs.
constexpr int kItemSlots = 4;
constexpr int kNoItem = -0x7fffffff;   // never stored in the ring
constexpr uint32_t kItemReaders = 3 + 2 * kEpiWarps;
static_assert(2 * kEpiWarps == static_cast<int>(kNsSignalsPerTile),
              "every epilogue warp of the pair signals a finished tile once");

static_assert(kBK * 2 == 128, "one K slice must be one 128-byte swizzle row");
static_assert(kTmemCols <= 512, "two accumulators must fit in TMEM");
static_assert(kHalfN % kBMN == 0, "B half must be whole MN-major boxes");
static_assert(kEpiWarps == 8, "epilogue layout assumes two warps per lane quarter");
static_assert(kTileM == kBN, "symmetric products need square tiles");

// Operands and output of one work item.
struct Ops {
    const CUtensorMap* a;
    const CUtensorMap* b;
    const CUtensorMap* out;
    int M, N, K;
};

__device__ __forceinline__ Ops item_operands(const NsParams& P, const NsWork& w) {
    const NsClass& C = P.cls[w.cls];
    const int cur = w.iter & 1;
    if (w.kind == kGram) return Ops{&C.tmX[cur], &C.tmX[cur], &C.stA, C.p, C.p, C.q};
    if (w.kind == kPoly) return Ops{&C.tmA, &C.tmA, &C.stB, C.p, C.p, C.p};
    const bool last = w.iter == P.ns_steps - 1;
    return Ops{&C.tmB, &C.tmXmn[cur], last ? &C.stO : &C.stX[cur ^ 1], C.p, C.q, C.p};
}

// Bytes CTA `rank` loads for one reduction slice of a tile.  Boxes that lie
// wholly past M or N are skipped: they only feed accumulator rows / columns
// that are never stored.
__device__ __forceinline__ uint32_t slice_bytes(const Ops& op, const NsWork& w, int rank,
                                                bool b_mn, int* nbox_b) {
    uint32_t bytes = 0;
    if (w.mt * kTileM + rank * kBM < op.M) bytes += kABytes;
    const int n0 = w.nt * kBN + rank * kHalfN;
    int nb = 0;
    if (b_mn) {
        for (int j = 0; j < kHalfN / kBMN; ++j)
            if (n0 + j * kBMN < op.N) ++nb;
        bytes += nb * kMnBoxBytes;
    } else if (n0 < op.N) {
        nb = 1;
        bytes += kBBytes;
    }
    *nbox_b = nb;
    return bytes;
}

__device__ __forceinline__ void unpack8(const uint4& u, float* v) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(h[k]);
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float* v) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) h[k] = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
    return u;
}

// Where a wait gave up (recorded once per status word, for malt_debug_timeout_site).
enum WaitSite : int32_t {
    kSiteClaim = 1,      // scheduler: a ring slot to become free
    kSiteDepLoad = 2,    // scheduler: the previous product of the item's matrix
    kSiteStage = 3,      // producer: a free operand stage
    kSiteItem = 4,       // ring reader: the next item (+ 16 * role)
    kSiteAccFree = 5,    // MMA: a free accumulator
    kSiteStageFull = 6,  // MMA: operands of a stage
    kSiteAccFull = 7,    // epilogue: a finished accumulator
    kSiteDrain = 9,      // MMA: the last MMAs before TMEM is freed
};

__device__ __forceinline__ void raise_timeout(const NsParams& P, volatile int* abort_flag,
                                              int site = 0, int item = -1, int seq = -1) {
    if (atomicCAS(P.status + 1, 0, site == 0 ? -1 : site) == 0) {
        P.status[2] = item;
        P.status[3] = seq;
        P.status[4] = static_cast<int32_t>(blockIdx.x);
        P.status[5] = static_cast<int32_t>(threadIdx.x);
    }
    atomicOr(P.status, kStatusTimeout);
    *abort_flag = 1;
}

// One unit of work as a role of the pair sees it.
enum JobState : int32_t { kJobWork = 0, kJobEnd = -1, kJobTimeout = -2 };
struct Job {
    int32_t state;
    int32_t stage;    // stage of the work table (persistent) or product index (phased)
    int32_t g;        // matrix (-1 when not known yet: phased)
    int32_t local;
    NsWork w;
};

__device__ __forceinline__ Job job_of_entry(const NsParams& P, const NsEntry& e) {
    Job j;
    if (e.g < 0) {
        j.state = kJobEnd;
        return j;
    }
    j.state = kJobWork;
    j.stage = entry_stage(e);
    j.g = e.g;
    j.local = e.local;
    j.w.s = j.stage;
    j.w.iter = j.stage / 3;
    j.w.kind = j.stage - 3 * j.w.iter;
    j.w.cls = entry_cls(e);
    j.w.b = entry_b(e);
    j.w.local = e.local;
    ns_tile_coords(P.cls[j.w.cls], j.w.kind, e.local, &j.w.mt, &j.w.nt);
    return j;
}

}  // namespace

template <int kMode>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
ns_gemm_kernel(const __grid_constant__ NsParams P) {
    constexpr bool kPersistent = kMode == kNsPersistent;   // table-driven, claimed dynamically
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[kRing];
    __shared__ __align__(8) uint64_t empty_bar[kRing];
    __shared__ __align__(8) uint64_t tfull_bar[2];
    __shared__ __align__(8) uint64_t tempty_bar[2];
    __shared__ __align__(8) uint64_t drain_bar;
    __shared__ __align__(8) uint64_t item_full[kItemSlots];
    __shared__ __align__(8) uint64_t item_empty[kItemSlots];
    __shared__ NsEntry item_ring[kItemSlots];
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_sh;
    volatile int* abort_flag = &abort_sh;

    // Same offset in both CTAs: the MMA addresses the peer's tiles through
    // the even CTA's descriptors.
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint64_t budget = P.budget_ns;
    const int rank = static_cast<int>(cluster_ctarank());
    const bool leader = (rank == 0);
    const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kRing; ++s) {
            // Both producers arrive on the even CTA's full barrier for every
            // ring stage (the even one with the pair's transaction bytes), so the
            // MMA never consumes a slice the odd producer has not reached --
            // even when the odd CTA loads nothing (M or N within its partner's
            // half) -- and the odd producer can never fall a whole parity
            // cycle behind the empty barriers it waits on.
            mbar_init(&full_bar[s], 2);
            mbar_init(&empty_bar[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull_bar[a], 1);
            mbar_init(&tempty_bar[a], 2 * kEpiWarps);
        }
        mbar_init(&drain_bar, 1);
        if (kPersistent) {
            for (int s = 0; s < kItemSlots; ++s) {
                mbar_init(&item_full[s], 1);
                mbar_init(&item_empty[s], kItemReaders);
            }
        }
        abort_sh = 0;
        fence_barrier_init();
        fence_proxy_async_smem();
    }
    if (warp == 0 && lane == 0) {
        for (int c = 0; c < P.nclasses; ++c) {
            const NsClass& C = P.cls[c];
            for (int j = 0; j < 2; ++j) {
                tma_prefetch_desc(&C.tmX[j]);
                tma_prefetch_desc(&C.tmXmn[j]);
            }
            tma_prefetch_desc(&C.tmA);
            tma_prefetch_desc(&C.tmB);
        }
    }
    if (warp == 1) {
        tmem_alloc_pair(&tmem_slot, kTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();          // both CTAs' barriers initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem_base = tmem_slot;

    // Work number `seq` of this pair.  Phased: static round-robin over the
    // product's item range.  Persistent: the next entry of the ring, which
    // the scheduler thread of the odd CTA fills from the work table.
    auto static_job = [&](int seq) -> Job {
        Job j;
        const long long it = static_cast<long long>(P.item_begin) + pair +
                             static_cast<long long>(seq) * npairs;
        if (it >= P.item_end) {
            j.state = kJobEnd;
            return j;
        }
        j.state = kJobWork;
        j.w = ns_decode(P, static_cast<int>(it));
        j.stage = j.w.s;
        j.g = -1;
        j.local = j.w.local;
        return j;
    };
    // The ring entry of sequence number seq (false when the wait gave up).
    auto ring_entry = [&](int seq, NsEntry& e) -> bool {
        const int slot = seq % kItemSlots;
        const uint32_t par = static_cast<uint32_t>(seq / kItemSlots) & 1u;
        if (!mbar_wait_cluster_bounded(&item_full[slot], par, budget, abort_flag)) return false;
        const volatile int32_t* v = reinterpret_cast<const volatile int32_t*>(&item_ring[slot]);
        e.code = v[0];
        e.g = v[1];
        e.local = v[2];
        e.target = static_cast<uint32_t>(v[3]);
        // Free the slot (its barrier lives in the odd CTA, with the
        // scheduler).  The arrive carries no data, so it is relaxed; it is
        // issued only once the slot's value is in hand (the branch depends on
        // it), so the scheduler cannot overwrite the slot before this read.
        if (e.code != kNoItem)
            mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(&item_empty[slot]), 1));
        return true;
    };
    auto ring_job = [&](int seq) -> Job {
        NsEntry e;
        if (!ring_entry(seq, e)) {
            Job j;
            j.state = kJobTimeout;
            return j;
        }
        return job_of_entry(P, e);
    };
    auto next_job = [&](int seq) -> Job { return kPersistent ? ring_job(seq) : static_job(seq); };
    // Scheduler (odd CTA): the table entry of the next claimed item (an end
    // marker past the end), and its publication to the ring slot of sequence
    // number seq in both CTAs (false when the slot did not come free in time).
    auto claim_next = [&]() -> NsEntry {
        const uint32_t claimed = atomicAdd(P.queue, 1u);
        if (claimed >= static_cast<uint32_t>(P.item_end - P.item_begin)) {
            NsEntry e;
            e.code = 0;
            e.g = -1;
            e.local = 0;
            e.target = 0;
            return e;
        }
        const int4 v = __ldg(reinterpret_cast<const int4*>(P.table + P.item_begin + claimed));
        NsEntry e;
        e.code = v.x;
        e.g = v.y;
        e.local = v.z;
        e.target = static_cast<uint32_t>(v.w);
        return e;
    };
    auto publish_item = [&](int seq, const NsEntry& e) -> bool {
        const int slot = seq % kItemSlots;
        const uint32_t par = static_cast<uint32_t>(seq / kItemSlots) & 1u;
        if (!mbar_wait_cluster_bounded(&item_empty[slot], par ^ 1u, budget, abort_flag)) return false;
        // The entry travels as an asynchronous store that completes on the
        // slot's full barrier in each CTA.  The arrive releases at cluster
        // scope what this thread acquired from the dependency counter, so a
        // reader that sees the item also sees the data the item reads.
        for (uint32_t r = 0; r < 2; ++r) {
            const uint32_t bar = mapa_shared(smem_u32(&item_full[slot]), r);
            mbar_arrive_expect_tx_cluster(bar, 16u);
            st_async_v4(mapa_shared(smem_u32(&item_ring[slot]), r), e.code, e.g, e.local,
                        static_cast<int32_t>(e.target), bar);
        }
        return true;
    };

    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            uint32_t stage = 0, phase = 0;
            for (int seq = 0;; ++seq) {
                const Job job = next_job(seq);
                if (job.state == kJobTimeout) {
                    raise_timeout(P, abort_flag, kSiteItem, -2, seq);
                    break;
                }
                if (job.state == kJobEnd) break;
                const int item = job.local;
                // The loads below read what other CTAs stored in this launch.
                if (kPersistent) fence_proxy_async_global();
                const NsWork& w = job.w;
                const Ops op = item_operands(P, w);
                const bool b_mn = w.kind == kBX;
                // A diagonal tile of a symmetric product: each CTA's half of B is
                // its own rows of A, so B is not loaded and the MMA reads A twice.
                const bool same_ab = !b_mn && w.mt == w.nt;
                const int nkb = (op.K + kBK - 1) / kBK;
                int nb_self = 0, nb_peer = 0;
                uint32_t bytes_pair = slice_bytes(op, w, rank, b_mn, &nb_self) +
                                      slice_bytes(op, w, rank ^ 1, b_mn, &nb_peer);
                if (same_ab) {
                    nb_self = 0;
                    bytes_pair = (w.mt * kTileM < op.M ? kABytes : 0u) +
                                 (w.mt * kTileM + kBM < op.M ? kABytes : 0u);
                }
                const bool load_a = w.mt * kTileM + rank * kBM < op.M;
                const int a_row = w.mt * kTileM + rank * kBM;
                const int n0 = w.nt * kBN + rank * kHalfN;
                bool ok = true;
                for (int k0 = 0; k0 < nkb; k0 += kGroup) {
                    if (!mbar_wait_cluster_bounded(&empty_bar[stage], phase ^ 1u, budget, abort_flag)) {
                        raise_timeout(P, abort_flag, kSiteStage, item, k0);
                        ok = false;
                        break;
                    }
                    const int nsub = min(kGroup, nkb - k0);
                    const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
                    if (leader) mbar_arrive_expect_tx(&full_bar[stage], nsub * bytes_pair);
                    for (int j = 0; j < nsub; ++j) {
                        const int kb = k0 + j;
                        uint8_t* sa = smem + (stage * kGroup + j) * kStageBytes;
                        if (load_a) tma_load_3d_pair(sa, op.a, kb * kBK, a_row, w.b, fb);
                        if (b_mn) {
                            for (int jb = 0; jb < nb_self; ++jb)
                                tma_load_3d_pair(sa + kABytes + jb * kMnBoxBytes, op.b,
                                                 n0 + jb * kBMN, kb * kBK, w.b, fb);
                        } else if (nb_self > 0) {
                            tma_load_3d_pair(sa + kABytes, op.b, kb * kBK, n0, w.b, fb);
                        }
                    }
                    if (!leader) mbar_arrive_cluster_relaxed(fb);
                    if (++stage == kRing) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
            }
        }
    } else if (warp == 1) {
        if (kPersistent && lane == 0 && !leader) {
            // ------------------------------------------ scheduler (odd CTA)
            // Claim items in table order, one ahead; publish each once the
            // previous stage of its matrix is complete, up to kItemSlots
            // ahead of the slowest reader.  Waiting here keeps the acquire
            // round trip off the producers' path.
            NsEntry next = claim_next();
            for (int seq = 0;; ++seq) {
                const NsEntry e = next;
                if (e.g >= 0 && e.target > 0 &&
                    !counter_wait_bounded(P.done + (entry_stage(e) - 1) * P.nmat + e.g, e.target,
                                          P.budget_ns, P.status, kStatusTimeout, abort_flag)) {
                    raise_timeout(P, abort_flag, kSiteDepLoad, e.local, seq);
                    break;
                }
                if (!publish_item(seq, e)) {
                    raise_timeout(P, abort_flag, kSiteClaim, e.local, seq);
                    break;
                }
                if (e.g < 0) break;
                next = claim_next();
            }
        }
        // ------------------------------------------- MMA issuer (even CTA)
        if (lane == 0 && leader) {
            uint32_t stage = 0, phase = 0;
            int gi = 0;                                  // product tiles so far (accumulator)
            for (int seq = 0;; ++seq) {
                const Job job = next_job(seq);
                if (job.state == kJobTimeout) {
                    raise_timeout(P, abort_flag, kSiteItem + 16, -2, seq);
                    break;
                }
                if (job.state == kJobEnd) break;
                const int item = job.local;
                const NsWork& w = job.w;
                const bool b_mn = w.kind == kBX;
                const int K = w.kind == kGram ? P.cls[w.cls].q : P.cls[w.cls].p;
                const int nkb = (K + kBK - 1) / kBK;
                const uint32_t acc = gi & 1, acc_phase = (gi >> 1) & 1;
                ++gi;
                if (!mbar_wait_cluster_bounded(&tempty_bar[acc], acc_phase ^ 1u, budget, abort_flag)) {
                    raise_timeout(P, abort_flag, kSiteAccFree, item, seq);
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + acc * kBN;
                bool ok = true;
                for (int k0 = 0; k0 < nkb; k0 += kGroup) {
                    if (!mbar_wait_cluster_bounded(&full_bar[stage], phase, budget, abort_flag)) {
                        raise_timeout(P, abort_flag, kSiteStageFull, item, k0);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const int nsub = min(kGroup, nkb - k0);
                    for (int j = 0; j < nsub; ++j) {
                        const int kb = k0 + j;
                        const uint32_t sa = smem_u32(smem + (stage * kGroup + j) * kStageBytes);
                        const uint64_t da = smem_desc_k_sw128(sa);
                        if (b_mn) {
                            const uint64_t db = smem_desc_mn_sw128(sa + kABytes, kMnLbo);
#pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk) {
                                // A: +32 bytes along K; B: +16 K-rows = two 1024-byte atoms.
                                tc_mma_bf16_pair(d_tmem, da + 2 * kk, db + (2048u >> 4) * kk,
                                                 kIdescBmn, (kb | kk) != 0 ? 1u : 0u);
                            }
                        } else {
                            // (a diagonal tile of a symmetric product reads B from A's rows)
                            const uint64_t db = smem_desc_k_sw128(w.mt == w.nt ? sa : sa + kABytes);
#pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk) {
                                // +32 bytes along K per 16-element MMA slice (encoded >> 4).
                                tc_mma_bf16_pair(d_tmem, da + 2 * kk, db + 2 * kk, kIdesc,
                                                 (kb | kk) != 0 ? 1u : 0u);
                            }
                        }
                    }
                    tc_commit_pair_multicast(&empty_bar[stage], kPairMask);
                    if (++stage == kRing) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                tc_commit_pair_multicast(&tfull_bar[acc], kPairMask);
            }
            // Do not release TMEM while MMAs may still be in flight.
            tc_commit_pair_multicast(&drain_bar, 0x1);
            if (!mbar_wait_cluster_bounded(&drain_bar, 0, budget, nullptr)) raise_timeout(P, abort_flag, kSiteDrain);
        }
    } else {
        // -------------------------------------------------------- epilogue
        uint8_t* stage_out = smem + kStages * kStageBytes;   // 1024-byte aligned
        int obuf = 0;
        const int ew = warp - 2;                  // epilogue warp 0..kEpiWarps-1
        const int quarter = warp & 3;             // TMEM lanes this warp may read
        const int colw = (ew >> 2) * kEpiCols;    // first accumulator column of this warp
        const uint32_t tempty_leader0 = mapa_shared(smem_u32(&tempty_bar[0]), 0);
        const uint32_t tempty_leader1 = mapa_shared(smem_u32(&tempty_bar[1]), 0);
        int gi = 0;                               // product tiles so far (accumulator)
        for (int seq = 0;; ++seq) {
            Job job;
            if (kPersistent) {
                // One lane waits on the ring; the warp shares the entry.
                NsEntry e;
                e.code = 0;
                e.g = -1;
                e.local = 0;
                e.target = 0;
                int ok = 1;
                if (lane == 0) ok = ring_entry(seq, e) ? 1 : 0;
                ok = __shfl_sync(0xffffffffu, ok, 0);
                e.code = __shfl_sync(0xffffffffu, e.code, 0);
                e.g = __shfl_sync(0xffffffffu, e.g, 0);
                e.local = __shfl_sync(0xffffffffu, e.local, 0);
                if (!ok) {
                    job.state = kJobTimeout;
                } else {
                    job = job_of_entry(P, e);
                }
            } else {
                job = static_job(seq);
            }
            if (job.state == kJobTimeout) {
                if (lane == 0) raise_timeout(P, abort_flag, kSiteItem + 32, -2, seq);
                break;
            }
            if (job.state == kJobEnd) break;
            const int item = job.local;
            const NsWork& w = job.w;
            const NsClass& C = P.cls[w.cls];
            const uint32_t acc = gi & 1, acc_phase = (gi >> 1) & 1;
            ++gi;
            const int M = C.p, N = w.kind == kBX ? C.q : C.p;
            const CUtensorMap* out_map0 = item_operands(P, w).out;
            const bool sym = w.kind != kBX;
            const int row = w.mt * kTileM + rank * kBM + quarter * 32 + lane;
            const bool rok = row < M;
            const int g = job.g >= 0 ? job.g : C.mat_of[w.b];
            const MatDesc& md = P.mats[g];
            // Persistent launches read what the launch itself wrote (1/||Mt||,
            // L, R, A) through L2 only.
            const float kx = w.iter == 0 ? (kPersistent ? __ldcg(&P.scal[g].k) : P.scal[g].k) : 1.f;
            const bool need_ein = (w.kind == kPoly);
            const __nv_bfloat16* ein =
                need_ein ? C.A + static_cast<size_t>(w.b) * C.p * C.p : nullptr;
            const bool last_bx = (w.kind == kBX) && (w.iter == P.ns_steps - 1);
            // O of a tall W (NS frame = W^T) goes out transposed, in W's layout.
            const bool store_t = last_bx && md.trans;
            const CUtensorMap* out_map = store_t ? &C.stOt : out_map0;
            // NS frame row / column scalings of D = L O R (swapped when transposed).
            const float* uvec = md.trans ? md.R : md.L;
            const float* vvec = md.trans ? md.L : md.R;
            const float urow = (last_bx && rok) ? (kPersistent ? __ldcg(uvec + row) : uvec[row]) : 0.f;
            float sum_o = 0.f, sum_d = 0.f;

            const int col_base = w.nt * kBN + colw;     // first output column of this warp
            const int nch = max(0, min(kEpiChunks, (N - col_base + 31) / 32));
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                   acc * kBN + colw;
            auto load_ein = [&](int ch, uint4 (&dst)[4]) {
                const int col0 = col_base + ch * 32;
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) {
                    if (rok && col0 + q8 * 8 < N) {
                        const uint4* src = reinterpret_cast<const uint4*>(
                            ein + static_cast<size_t>(row) * N + col0 + q8 * 8);
                        // Phased: A was written by an earlier launch, so the
                        // read-only path is safe.  Persistent: A is rewritten
                        // each iteration inside this launch; read through L2
                        // (ordered by the ring's acquire).
                        dst[q8] = kPersistent ? __ldcg(src) : __ldg(src);
                    }
                    else
                        dst[q8] = make_uint4(0u, 0u, 0u, 0u);
                }
            };
            uint4 xin[4];
            uint32_t rv[32];
            const int row0 = w.mt * kTileM + rank * kBM + quarter * 32;   // warp's first row
            // The first chunk's A values (and the scalars above) are in flight
            // while the accumulator is still being computed.
            if (need_ein && nch > 0) load_ein(0, xin);
            // The epilogue warps poll with a short sleep: sixteen warps spinning
            // on this barrier cost issue slots and power the MMA and load
            // warps need (measured 0.5-1 % on every product).
            if (!mbar_wait_cluster_bounded_sleep(&tfull_bar[acc], acc_phase, budget, abort_flag, 128)) {
                raise_timeout(P, abort_flag, kSiteAccFull, item, seq);
                break;
            }
            tc_fence_after();
            if (nch > 0) {
                tmem_ld_issue(tbase, rv);
                tmem_ld_wait(rv);
            }
#pragma unroll
            for (int ch = 0; ch < kEpiChunks; ++ch) {
                if (ch >= nch) break;
                uint4 xcur[4];
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) xcur[q8] = xin[q8];
                if (need_ein && ch + 1 < nch) load_ein(ch + 1, xin);   // next chunk's A, one ahead

                const int col0 = col_base + ch * 32;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(rv[j]);
                // The next chunk's TMEM load is in flight during this chunk's work.
                if (ch + 1 < nch) tmem_ld_issue(tbase + (ch + 1) * 32, rv);
                if (w.kind == kGram) {
                    const float sc = kx * kx;
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] *= sc;
                } else if (w.kind == kPoly) {
                    float x[32];
#pragma unroll
                    for (int q8 = 0; q8 < 4; ++q8) unpack8(xcur[q8], x + 8 * q8);
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        v[j] = fmaf(P.b, x[j], P.c * v[j]) + (col0 + j == row ? P.a : 0.f);
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] *= kx;
                }
                if (!store_t) {
                    // Stage the 32 x 32 chunk (row = lane, 64 bytes) with the 64-byte
                    // swizzle the store map expects, then one TMA store writes it
                    // (A, B', the next X, or a wide matrix's O on the last iteration).
                    uint8_t* box = stage_out + (ew * 2 + obuf) * kStoreBoxBytes;
                    if (lane == 0) bulk_wait_group_read<1>();   // this buffer's last store read it
                    __syncwarp();
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        *reinterpret_cast<uint4*>(box + lane * 64 + ((c ^ ((lane >> 1) & 3)) << 4)) =
                            pack8(v + 8 * c);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_3d(out_map, box, col0, row0, w.b);
                        bulk_commit_group();
                    }
                    obuf ^= 1;
                }
                if (store_t || (sym && w.nt != w.mt)) {
                    // Mirror an off-diagonal tile of the symmetric product, or
                    // store a tall matrix's O in W's layout: the transposed chunk
                    // (box row = column j, 32 rows of this warp) goes to rows
                    // [col0, col0+32) x columns [row0, row0+32) of the map.
                    // Lane pairs swap one value per column pair so each lane
                    // writes a 32-bit (two-row) word.
                    uint8_t* box = stage_out + (ew * 2 + obuf) * kStoreBoxBytes;
                    if (lane == 0) bulk_wait_group_read<1>();
                    __syncwarp();
                    const bool odd = lane & 1;
                    const int r2 = lane & ~1;                 // first of the two rows
#pragma unroll
                    for (int j = 0; j < 32; j += 2) {
                        // even lane keeps column j, odd lane keeps column j + 1
                        const float send = odd ? v[j] : v[j + 1];
                        const float recv = __shfl_xor_sync(0xffffffffu, send, 1);
                        const float lo = odd ? recv : v[j];        // row r2
                        const float hi = odd ? v[j + 1] : recv;    // row r2 + 1
                        const int jc = j + (odd ? 1 : 0);          // box row
                        const int off = jc * 64 + (((r2 >> 3) ^ ((jc >> 1) & 3)) << 4) + (r2 & 7) * 2;
                        *reinterpret_cast<__nv_bfloat162*>(box + off) = __floats2bfloat162_rn(lo, hi);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_3d(out_map, box, row0, col0, w.b);
                        bulk_commit_group();
                    }
                    obuf ^= 1;
                }
                if (last_bx) {
                    // Partial sums of O^2 and (O v)^2 over the stored (bf16) O of this
                    // row; D^2 = u_row^2 (O v)^2 is formed once per tile.  Lane j holds
                    // v[col0 + j] and broadcasts it (columns past N contribute 0).
                    const float vl = (col0 + lane < N)
                                         ? (kPersistent ? __ldcg(vvec + col0 + lane) : vvec[col0 + lane])
                                         : 0.f;
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const float vj = __shfl_sync(0xffffffffu, vl, j);
                        const float o = __bfloat162float(__float2bfloat16_rn(v[j]));
                        const float ov = o * vj;
                        sum_o = fmaf(o, (col0 + j < N) ? o : 0.f, sum_o);
                        sum_d = fmaf(ov, ov, sum_d);
                    }
                }
                if (ch + 1 < nch) tmem_ld_wait(rv);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acc ? tempty_leader1 : tempty_leader0);
            if (last_bx) {
                if (!rok) sum_o = 0.f;
                sum_d = rok ? urow * urow * sum_d : 0.f;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    sum_o += __shfl_xor_sync(0xffffffffu, sum_o, o);
                    sum_d += __shfl_xor_sync(0xffffffffu, sum_d, o);
                }
                if (lane == 0) {
                    float* dst = md.nspart + (static_cast<size_t>(w.local) * kNsPartsPerTile +
                                              rank * kEpiWarps + ew) * 2;
                    dst[0] = sum_o;
                    dst[1] = sum_d;
                }
            }
            if (kPersistent && job.stage + 1 < P.nstages && lane == 0) {
                // This warp's part of the tile is in global memory: signal it
                // (the last stage has no reader inside the launch).
                bulk_wait_group_all();
                fence_proxy_async_global();
                red_release_gpu_add(P.done + job.stage * P.nmat + g, 1u);
            }
        }
        if (lane == 0) bulk_wait_group_all();     // every output store has landed
    }

    // Neither CTA may leave (or free TMEM) while its pair partner can still
    // signal its barriers or read its shared memory.
    tc_fence_before();
    cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, kTmemCols);
    }
}

size_t ns_gemm_smem_bytes() { return kSmemBytes; }

namespace {

template <int kMode>
cudaError_t set_smem_attr() {
    return cudaFuncSetAttribute(ns_gemm_kernel<kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(kSmemBytes));
}

cudaError_t set_all_smem_attrs() {
    cudaError_t e = set_smem_attr<kNsPhased>();
    if (e == cudaSuccess) e = set_smem_attr<kNsPersistent>();
    return e;
}

// Per-device one-time set-up: the shared-memory opt-in of every
// instantiation (a function attribute holds for the device that was current
// when it was set) and the number of CTA pairs resident at once.  0 = not
// yet done on that device.
constexpr int kMaxDevices = 64;
std::mutex g_cfg_mu;
int g_pairs[kMaxDevices] = {};

cudaError_t configure_current_device(int* pairs) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_cfg_mu);
    if (g_pairs[dev] == 0) {
        e = set_all_smem_attrs();
        if (e != cudaSuccess) return e;
        // All instantiations have the same block shape and shared memory.
        int n = 0;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2, 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = kSmemBytes;
        if (cudaOccupancyMaxActiveClusters(&n, ns_gemm_kernel<kNsPersistent>, &cfg) != cudaSuccess ||
            n <= 0) {
            cudaGetLastError();
            int sms = 0;
            e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (e != cudaSuccess) return e;
            n = std::max(1, sms / 2);
        }
        g_pairs[dev] = n;
    }
    *pairs = g_pairs[dev];
    return cudaSuccess;
}

}  // namespace

// Number of CTA pairs that can be resident at once on the current device (the
// persistent grid); 1 if the device cannot be configured (the next launch
// then reports the error).
int ns_gemm_max_pairs() {
    int pairs = 0;
    if (configure_current_device(&pairs) != cudaSuccess) {
        cudaGetLastError();
        return 1;
    }
    return pairs;
}

cudaError_t ns_gemm_configure() {
    int pairs = 0;
    return configure_current_device(&pairs);
}

cudaError_t launch_ns_gemm(const NsParams& P, int mode, int grid_pairs, cudaStream_t s) {
    const cudaError_t ce = ns_gemm_configure();
    if (ce != cudaSuccess) return ce;
    if (mode == kNsPersistent)
        ns_gemm_kernel<kNsPersistent><<<2 * grid_pairs, kThreads, kSmemBytes, s>>>(P);
    else
        ns_gemm_kernel<kNsPhased><<<2 * grid_pairs, kThreads, kSmemBytes, s>>>(P);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        cudaFuncAttributes fa{};
        if (mode == kNsPersistent)
            cudaFuncGetAttributes(&fa, ns_gemm_kernel<kNsPersistent>);
        else
            cudaFuncGetAttributes(&fa, ns_gemm_kernel<kNsPhased>);
        std::fprintf(stderr,
                     "malt: ns_gemm_kernel<%d> launch (%d CTAs x %d threads, %zu B dynamic smem, "
                     "%zu B parameters) refused: %s; kernel uses %d registers, %zu B static "
                     "smem, allows %d threads and %d B dynamic smem per block\n",
                     mode, 2 * grid_pairs, kThreads, kSmemBytes, sizeof(NsParams),
                     cudaGetErrorString(e), fa.numRegs, fa.sharedSizeBytes,
                     fa.maxThreadsPerBlock, fa.maxDynamicSharedSizeBytes);
        cudaGetLastError();
    }
    return e;
}

}  // namespace malt
