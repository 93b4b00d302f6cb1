// heddle_internal.cuh -- definitions shared by the library's translation
// units (never installed, never included by the oracle).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "heddle.h"

namespace hd {

constexpr int kMaxTypes = HEDDLE_MAX_TYPES;
constexpr int kMaxStages = HEDDLE_MAX_STAGES;
static_assert(kMaxStages == 32, "the searches hold one stage (or one depth) per lane");
constexpr int kMaxLayers = HEDDLE_MAX_LAYERS;
constexpr int kMaxTopK = HEDDLE_MAX_TOPK;
constexpr int64_t kInf = INT64_MAX;

typedef unsigned __int128 u128;

// Device error flags (heddle_device_errors).
constexpr uint32_t kErrStageWait = 1u;
constexpr uint32_t kErrSearchBound = 2u;
constexpr uint32_t kErrInternal = 4u;
constexpr uint32_t kErrBounds = 8u;  // a bounds check of the checked build failed

// The bounds-checked build (HEDDLE_CHECKED) tests the data-dependent
// indices -- worklist entries, candidate indices, table rows -- before it
// uses them; a failed test raises kErrBounds and the access is skipped (no
// trap, no out-of-range access).  The product build compiles the tests away.
#ifdef HEDDLE_CHECKED
constexpr bool kChecked = true;
#else
constexpr bool kChecked = false;
#endif
__device__ __forceinline__ bool in_range(int64_t i, int64_t n, uint32_t* err) {
    if (!kChecked) return true;
    if (i >= 0 && i < n) return true;
    atomicOr(err, kErrBounds);
    return false;
}
// Table-build flags (checked by the host at load time).
constexpr uint32_t kTabBadValue = 1u;   // non-finite or negative per-layer cost
constexpr uint32_t kTabTooLarge = 2u;   // a table total or P2P term above its limit

// Byte layout of the cost-table image.  The pricing kernel copies the whole
// image into shared memory with one bulk (TMA) copy per CTA, so every
// section starts on a 16-byte boundary and the total is a multiple of 16.
struct Layout {
    int32_t L, NT;
    uint32_t offP;      // int64 [NT][4][L+1]   prefix of per-layer ns per (type, degree)
    uint32_t offSA;     // int64x2 [L+1]         prefix of (state bytes, activation bytes)
    uint32_t offPB;     // int64 [L+1]           prefix of gradient bytes
    uint32_t offP2P;    // int64 [8][8][2]       P2P ns (from, to, same-node)
    uint32_t offMem;    // int64 [8]             memory per GPU
    uint32_t offInter;  // int64 [8]             slowest NIC of the type
    uint32_t offMinQ;   // int64 [NT][4]         cheapest single layer per (type, degree)
    uint32_t offMaxN;   // int32 [8]             largest node of the type
    uint32_t offPow2;   // int32 [8]             largest power of two <= largest node (<= 8)
    uint32_t offGpus;   // int32 [8]             GPUs of the type
    uint32_t offCap;    // int32 [8][4]          sum over nodes of floor(gpus / 2^e) * 2^e
    uint32_t offWin;    // uint8 [8][4][33]      longest run of layers that fits memory per
                        //                       (type, degree, in-flight microbatches f)
    uint32_t offModel;  // int32 [4]             [0] every layer has the same state and
                        //                       activation bytes; [1] every layer has the
                        //                       same quantised cost per (type, degree)
    uint32_t bytes;
};

inline uint32_t align16(uint32_t x) { return (x + 15u) & ~15u; }

inline Layout make_layout(int L, int NT) {
    Layout y{};
    y.L = L;
    y.NT = NT;
    uint32_t o = 0;
    y.offP = o;     o = align16(o + 8u * NT * 4 * (L + 1));
    y.offSA = o;    o = align16(o + 16u * (L + 1));
    y.offPB = o;    o = align16(o + 8u * (L + 1));
    y.offP2P = o;   o = align16(o + 8u * 8 * 8 * 2);
    y.offMem = o;   o = align16(o + 8u * 8);
    y.offInter = o; o = align16(o + 8u * 8);
    y.offMinQ = o;  o = align16(o + 8u * NT * 4);
    y.offMaxN = o;  o = align16(o + 4u * 8);
    y.offPow2 = o;  o = align16(o + 4u * 8);
    y.offGpus = o;  o = align16(o + 4u * 8);
    y.offCap = o;   o = align16(o + 4u * 8 * 4);
    y.offWin = o;   o = align16(o + 8u * 4 * 33);
    y.offModel = o; o = align16(o + 4u * 4);
    y.bytes = o;
    return y;
}

struct TopkEntry {
    int64_t idx;
    int64_t T;
    uint32_t nM;
    uint32_t pad;
};

struct TableArgs {
    Layout lay;
    const heddle_gpu_type* types;
    const heddle_node* nodes;
    int32_t n_nodes;
    const heddle_layer* layers;
    const double* profile;   // nullable
    int64_t boundary_bytes;
    int32_t moe;
    unsigned char* img;      // out
    int64_t* q;              // out [NT][4][L]
    uint32_t* flags;         // out
};
cudaError_t launch_tables(const TableArgs& a, cudaStream_t st);

// Blocks of `func` (a kernel) resident per SM at `block` threads and `smem`
// bytes of dynamic shared memory, after raising the kernel's dynamic
// shared-memory limit to smem.  The answer is cached per (kernel, block,
// smem, device): the two runtime queries cost microseconds of host time,
// which a small pricing call would otherwise pay on every launch.
cudaError_t resident_blocks(const void* func, int block, size_t smem, int* per_sm);

struct PriceArgs {
    Layout lay;
    const unsigned char* img;
    int32_t moe;
    const uint8_t* S;
    const uint16_t* M;
    const uint8_t* code;
    const uint8_t* skip;  // nullable: nonzero prices the candidate SKIPPED (a template its plan does not reach)
    int64_t n;
    int64_t stride;
    int32_t s_max;
    int64_t* T;
    int64_t* B;
    uint16_t* ndp;
    uint8_t* status;
    uint8_t* bounds;
    int64_t bstride;  // plane stride of bounds (>= n)
    uint32_t* err;
    unsigned long long* counters;  // non-null selects the counting variant
    // worklist of the candidates that need the threshold search (device
    // scratch owned by the context, capacity wl_cap candidates)
    int32_t* wl_count;   // [kWlMeta]: entries, the general list, per depth S the entries
                         // of that depth, two take counters, survivors (cleared per chunk)
    int32_t* wl_idx;
    uint16_t* wl_n;
    uint16_t* wl_M;
    uint8_t* wl_S;
    uint8_t* wl_memok;   // 1: memory feasibility already decided by the screen
    uint8_t* wl_code;    // [wl_cap][kMaxStages] stage bytes, a 32-byte row per entry (zero past S)
    int32_t* wl_bucket;  // [kMaxStages][wl_cap]: per depth S (row S - 1) the entries of
                         // that depth, in any order (equal-layer search)
    int32_t wl_cap;
    int32_t uniform;     // search with the equal-layer closed form (model flags [0] and [1])
    int32_t mbs_shift;   // micro-batch size 2^shift: M >> shift micro-batches (invalid unless 2^shift | M)
    int32_t split_mode;  // 1: the paper's own split rule (distribute_kernel) instead of PartitionLayers
    int32_t thread_min;  // general search: the bucketed entries below which only the warp search runs
    // per worklist entry, written by the search: T (-1 unless OK) and n * M,
    // so a top-k can run over the searched candidates only
    int64_t* wl_T;
    uint32_t* wl_nM;
    // survivors of the top-k threshold (equal-layer search inside a top-k
    // pricing; sv_count null otherwise): OK entries whose n*M / T, in
    // float, is at least the float threshold *thr are appended as (chunk
    // index, T, n*M).  *thr never exceeds the running top-k's k-th key
    // (see TopkArgs::thr), so no entry that can enter the top-k is left out.
    int32_t* sv_count;
    int32_t* sv_idx;
    int64_t* sv_T;
    uint32_t* sv_nM;
    uint32_t* thr;
    const int32_t* topk_k;  // the state's k (device)
};
// Prices candidates [0, a.n) with a.n <= a.wl_cap: screen, then search.
// `mid` (nullable) is recorded on st between the two; `launches` (nullable)
// gains the kernels launched: [0] screen, [1] search.
cudaError_t launch_price(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid = nullptr,
                         int64_t* launches = nullptr);
// The equal-layer search over the worklist the screen produced.
cudaError_t launch_eq_search(const PriceArgs& a, int num_sms, cudaStream_t st);
// Multi-template plans (Algorithm 1): per template slot the plans' arrays,
// already priced standalone (bounds required), overwritten with the plan's
// prices; per plan the templates placed and the summed throughput.
constexpr int kMaxTemplates = HEDDLE_MAX_TEMPLATES;
constexpr int kPlanMaxNode = HEDDLE_PLAN_MAX_NODE;
struct PlanSlot {
    const uint8_t* S;
    const uint16_t* M;
    const uint8_t* code;  // [s][stride]
    int64_t stride;
    int64_t* T;
    int64_t* B;
    uint16_t* ndp;
    uint8_t* status;
    uint8_t* bounds;  // [33][bstride]
    int64_t bstride;
};
struct PlanArgs {
    Layout lay;
    const unsigned char* img;
    int64_t n;
    int32_t slots;
    const uint8_t* n_tmpl;
    PlanSlot slot[kMaxTemplates];
    const int32_t* node_type;
    const int32_t* node_gpus;
    int32_t n_nodes;
    int32_t vmax;  // largest node (GPUs), <= kPlanMaxNode
    uint8_t* placed;
    double* thr;
    uint32_t* err;
};
cudaError_t launch_plans(const PlanArgs& a, int num_sms, cudaStream_t st);
// The SKIPPED mask of slot t of a plan batch (see plan_mask_kernel).
cudaError_t launch_plan_mask(const uint8_t* n_tmpl, int slots, int t, const uint8_t* prev_status, uint8_t* skip,
                             int64_t n, int num_sms, cudaStream_t st);

// The paper's own layer split over the worklist (comparison mode).
cudaError_t launch_distribute(const PriceArgs& a, int num_sms, cudaStream_t st);
constexpr int32_t kWorklistCap = 1 << 20;
constexpr int kWlMeta = 1 + kMaxStages + 1 + 2 + 1;  // ints of a.wl_count
constexpr int kWlGeneral = 1;  // entries the thread-per-entry general search left to the warp search
// the next entries the general searches take (each warp of the thread
// search takes 32 at a time, each warp of the warp search one)
constexpr int kWlTakeThread = kWlMeta - 3;
constexpr int kWlTakeWarp = kWlMeta - 2;
// The thread-per-entry general search runs when the depth buckets hold at
// least one warp of entries per SM; with fewer it would run one warp or less
// per SM, its time the latency of its longest serial chain, and the warp
// search (whose probes spread over 32 lanes) prices every entry instead.
inline int thread_search_min(int num_sms) { return num_sms * 32; }
constexpr int kWlSurv = kWlMeta - 1;             // the survivor count (see PriceArgs::sv_count)


struct TopkArgs {
    // results of a batch (heddle_topk) ...
    const uint16_t* M;
    const int64_t* T;
    const uint16_t* ndp;
    const uint8_t* status;
    int64_t n;
    int64_t base_index;
    heddle_topk_state* state;  // device, in/out
    TopkEntry* scratch;        // [grid][kMaxTopK]
    int32_t* scratch_count;    // [grid]
    int32_t max_blocks;
    // ... or the worklist of a priced chunk (heddle_price_topk)
    const int32_t* wl_count;
    const int32_t* wl_idx;
    const int64_t* wl_T;
    const uint32_t* wl_nM;
    int32_t wl_cap;
    // second-level lists of the two-level merge (group lists of the
    // one-launch worklist top-k), and that kernel's tickets: [16] per group,
    // then one for the final merge; zero between launches
    TopkEntry* scratch2;
    int32_t* scratch2_count;
    int32_t* tickets;
    // nullable: raised (atomicMax on the bits of a positive float) to the
    // new state's k-th key n*M / T in float times (1 - 2^-16) once the state
    // holds k entries.  Float conversions and the division are each within
    // 2^-24 relative, so the stored value stays below every key at least
    // the k-th's, exactly compared, by more than the rounding of a key
    // computed the same way.
    uint32_t* thr;
};
// `launches` (nullable) gains the number of kernels launched.
cudaError_t launch_topk(const TopkArgs& a, int num_sms, cudaStream_t st, int64_t* launches = nullptr);
// Top-k of the searched candidates of a priced chunk (a.wl_*), merged into
// *a.state; `n` bounds the worklist length (the chunk size).
cudaError_t launch_topk_worklist(const TopkArgs& a, int64_t n, int num_sms, cudaStream_t st,
                                 int64_t* launches = nullptr);
cudaError_t launch_topk_reset(heddle_topk_state* state, int32_t k, cudaStream_t st);

// Micro-batch-size fill: fold the results of one size (level) into the
// running best (smaller T wins, ties keep the earlier, smaller size).
struct MbsMergeArgs {
    int64_t n;
    const int64_t* T_l;
    const int64_t* B_l;
    const uint16_t* n_l;
    const uint8_t* status_l;
    const uint8_t* bounds_l;  // nullable, plane stride bstride_l
    int64_t bstride_l;
    int64_t* T;
    int64_t* B;
    uint16_t* ndp;
    uint8_t* status;
    uint8_t* bounds;  // nullable, plane stride bstride
    int64_t bstride;
    uint8_t* mbs;     // nullable
    int32_t level;
};
cudaError_t launch_mbs_merge(const MbsMergeArgs& a, int num_sms, cudaStream_t st);

// Conversions between non-negative 64-bit integers and float through their
// 32-bit halves: the 32-bit conversions run on the fast pipes, while a
// 64-bit conversion instruction runs on the (narrow) FP64 pipe.
// u64_to_float: relative error below 2^-23.
__device__ __forceinline__ float u64_to_float(uint64_t x) {
    return __fmaf_rn((float)(uint32_t)(x >> 32), 4294967296.0f, (float)(uint32_t)x);
}

// Truncation of a float in [0, 2^63) to an integer (exact: the low part
// f - hi 2^32 is representable).
__device__ __forceinline__ uint64_t float_to_u64(float f) {
    const float hi = floorf(f * 2.3283064365386963e-10f);
    const float lo = __fmaf_rn(-hi, 4294967296.0f, f);
    return ((uint64_t)(uint32_t)hi << 32) + (uint64_t)(uint32_t)fmaxf(lo, 0.f);
}

// ceil(A / C) for a 128-bit A and 1 <= C < 2^64 whose quotient is below
// 2^62: a float estimate of the quotient refined with exact 128-bit
// remainders (each refinement leaves about 2^-22 of the error), then exact
// unit steps.  *ok is cleared if the steps did not settle (never expected).
__device__ __forceinline__ float u128_to_float(u128 v) {
    return __fmaf_rn(u64_to_float((uint64_t)(v >> 64)), 18446744073709551616.0f, u64_to_float((uint64_t)v));
}

__device__ inline uint64_t ceil_div_u128(u128 A, uint64_t C, bool* ok) {
    const float rc = 1.0f / u64_to_float(C);
    const float e = u128_to_float(A) * rc;
    uint64_t q = e < 4.0e18f ? float_to_u64(e) : 4000000000000000000ull;
    for (int it = 0; it < 6; ++it) {
        const u128 qc = (u128)q * C;
        if (qc > A) {
            const uint64_t d = float_to_u64(u128_to_float(qc - A) * rc);
            q -= d == 0 ? 1 : (d < q ? d : q);
        } else {
            const u128 r = A - qc;
            if (r < C) break;
            const uint64_t d = float_to_u64(u128_to_float(r) * rc);
            q += d == 0 ? 1 : d;
        }
    }
    const u128 qc = (u128)q * C;
    if (qc > A || A - qc >= C) *ok = false;
    return q + (qc != A ? 1 : 0);
}

}  // namespace hd
