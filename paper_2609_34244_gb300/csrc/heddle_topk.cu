// heddle_topk.cu -- rank and top-k of priced candidates.
//
// The rank order and the warp-level lists are in heddle_rank.cuh.
//
// Launch 1: every CTA scans a slice of the batch (or, after a pricing call,
// of the worklist of searched candidates only); an entry that does not beat
// the incoming state's k-th is dropped at once, the others are offered to
// the warp's sorted list in shared memory (inserted only if they beat its
// current k-th), the CTA merges its warps' lists (a tree of parallel
// two-list merges) and writes one list to scratch.  While the state is not
// yet full, a first pass over the same slice finds each warp's k-th largest
// float key (a running top-32 per warp, merged by a bitonic network); the
// CTA's largest, lowered by a margin, drops the entries that k others beat
// before any is offered, so a warp inserts a handful of entries instead of
// every new best of an unsorted slice.  Then the per-CTA lists are folded
// into the state by merge levels of 16 lists per CTA: one level for up to
// 16 lists, else two.  No CTA waits on another.

#include <algorithm>

#include "heddle_rank.cuh"

namespace hd {
namespace {

constexpr int kTopkBlock = 256;
constexpr int kMergeBlock = 1024;  // warps 0-15 stage lists, warp 16 the state
constexpr int kMergeWarps = kMergeBlock / 32;

// One candidate entry: from a batch's results, or from the worklist of a
// priced chunk (only the searched candidates, T = -1 unless OK).  Every
// field is loaded whether or not the entry turns out valid, so the loads of
// several entries are independent and can be in flight together.
template <bool kWorklist>
__device__ __forceinline__ bool fetch(const TopkArgs& a, int64_t i, TopkEntry& e) {
    e.pad = 0;
    if (kWorklist) {
        e.T = a.wl_T[i];
        e.idx = a.base_index + a.wl_idx[i];
        e.nM = a.wl_nM[i];
        return e.T >= 0;
    }
    const bool ok = a.status[i] == HEDDLE_CAND_OK;
    e.idx = a.base_index + i;
    e.T = a.T[i];
    e.nM = (uint32_t)a.ndp[i] * (uint32_t)a.M[i];
    return ok;
}

// Entries that do not beat the incoming state's k-th entry (when it holds
// k) cannot enter the merged top-k, so they are not offered: after the
// first batches almost every entry stops at this one comparison.
template <bool kWorklist, int kBlock>
__global__ void __launch_bounds__(kBlock) topk_block_kernel(TopkArgs a) {
    constexpr int W = kBlock / 32;
    const int k = state_k(a.state);
    __shared__ TopkEntry lists[W * kMaxTopK];
    __shared__ TopkEntry tmp[(W / 2) * kMaxTopK];
    __shared__ int counts[W], tmp_counts[W / 2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool full = a.state->count >= k;
    TopkEntry bar;
    bar.idx = full ? a.state->idx[k - 1] : 0;
    bar.T = full ? a.state->T[k - 1] : 0;
    bar.nM = full ? a.state->nM[k - 1] : 0;
    bar.pad = 0;
    int cnt = 0;
    TopkEntry* list = lists + warp * kMaxTopK;
    const int64_t n = kWorklist ? min((int64_t)*a.wl_count, (int64_t)a.wl_cap) : a.n;
    const int64_t nwarps = (int64_t)gridDim.x * W;
    const int64_t gw = (int64_t)blockIdx.x * W + warp;
    // four rounds of 32 entries per warp are loaded before any is offered
    constexpr int U = 4;
    const int64_t step = nwarps * 32;
    // first pass (k <= 32, while the state is not full): the k-th largest
    // float key n*M / T among the entries each warp visits; k of them reach
    // it, so the CTA's largest such key, lowered by 2^-16 (more than the
    // rounding of two keys computed the same way), is a floor below which
    // no entry can enter the top-k
    __shared__ unsigned floor_bits;
    float floor_cta = 0.0f;
    if (k <= 32 && !full) {
        if (threadIdx.x == 0) floor_bits = 0;
        __syncthreads();
        float run = -1.0f;
        for (int64_t base = gw * 32; base < n; base += step) {
            const int64_t i = base + lane;
            float key = -1.0f;
            TopkEntry e;
            if (i < n && fetch<kWorklist>(a, i, e) && e.T > 0) key = (float)e.nM / (float)e.T;
            run = warp_keep_top32(run, key);
        }
        const float kth = __shfl_sync(0xffffffffu, run, k - 1);
        if (lane == 0 && kth > 0.0f) atomicMax(&floor_bits, __float_as_uint(kth * (1.0f - 1.0f / 65536.0f)));
        __syncthreads();
        floor_cta = __uint_as_float(floor_bits);
    }
    for (int64_t base = gw * 32; base < n; base += step * U) {
        TopkEntry e[U];
        bool valid[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t i = base + u * step + lane;
            valid[u] = false;
            e[u].idx = 0;
            e[u].T = 0;
            e[u].nM = 0;
            e[u].pad = 0;
            if (i < n) valid[u] = fetch<kWorklist>(a, i, e[u]);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const bool above = valid[u] && (floor_cta <= 0.0f || (float)e[u].nM / (float)e[u].T >= floor_cta);
            warp_offer(list, cnt, k, above && (!full || better(e[u], bar)), e[u]);
        }
    }
    if (lane == 0) counts[warp] = cnt;
    cta_tree_merge(lists, counts, tmp, tmp_counts, W, k);
    for (int p = threadIdx.x; p < counts[0]; p += blockDim.x)
        a.scratch[(size_t)blockIdx.x * kMaxTopK + p] = lists[p];
    if (threadIdx.x == 0) a.scratch_count[blockIdx.x] = counts[0];
}

// One merge level: CTA b folds lists [kFan b, kFan b + kFan) of src into
// dst[b]; with `final` (one CTA) the incoming state joins as one more list
// and the result is written to the state.
constexpr int kFan = 16;
__global__ void __launch_bounds__(kMergeBlock) topk_level_kernel(TopkArgs a, const TopkEntry* src,
                                                                 const int32_t* src_count, int nsrc,
                                                                 TopkEntry* dst, int32_t* dst_count,
                                                                 int final_level) {
    static_assert(kMergeWarps > kFan, "one warp per list plus one for the state");
    __shared__ TopkEntry lists[(kFan + 1) * kMaxTopK];
    __shared__ TopkEntry tmp[((kFan + 2) / 2) * kMaxTopK];
    __shared__ int counts[kFan + 1], tmp_counts[(kFan + 2) / 2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = state_k(a.state);
    // warp w stages list kFan b + w (and warp kFan the state, on the last level)
    if (warp < kFan) {
        const int l = blockIdx.x * kFan + warp;
        const int c = l < nsrc ? min(src_count[l], k) : 0;
        for (int i = lane; i < c; i += 32) lists[warp * kMaxTopK + i] = src[(size_t)l * kMaxTopK + i];
        if (lane == 0) counts[warp] = c;
    } else if (warp == kFan) {
        const int c = final_level ? min(max(a.state->count, 0), k) : 0;
        for (int i = lane; i < c; i += 32) {
            TopkEntry e;
            e.idx = a.state->idx[i];
            e.T = a.state->T[i];
            e.nM = a.state->nM[i];
            e.pad = 0;
            lists[kFan * kMaxTopK + i] = e;
        }
        if (lane == 0) counts[kFan] = c;
    }
    cta_tree_merge(lists, counts, tmp, tmp_counts, kFan + 1, k);
    const int cnt = counts[0];
    if (final_level) {
        for (int p = threadIdx.x; p < kMaxTopK; p += blockDim.x) {
            const bool live = p < cnt;
            a.state->idx[p] = live ? lists[p].idx : -1;
            a.state->T[p] = live ? lists[p].T : -1;
            a.state->nM[p] = live ? lists[p].nM : 0;
        }
        if (threadIdx.x == 0) a.state->count = cnt;
    } else {
        for (int p = threadIdx.x; p < cnt; p += blockDim.x) dst[(size_t)blockIdx.x * kMaxTopK + p] = lists[p];
        if (threadIdx.x == 0) dst_count[blockIdx.x] = cnt;
    }
}

// Fold `blocks` per-CTA lists of a.scratch (at most kFan * kFan) into
// *a.state: directly when there are few, else through one level into
// a.scratch2 first.
cudaError_t merge_lists(const TopkArgs& a, int blocks, cudaStream_t st, int64_t* launches) {
    if (blocks > kFan * kFan) return cudaErrorInvalidValue;
    if (launches) *launches += blocks > kFan ? 2 : 1;
    if (blocks > kFan) {
        const int m1 = (blocks + kFan - 1) / kFan;
        topk_level_kernel<<<m1, kMergeBlock, 0, st>>>(a, a.scratch, a.scratch_count, blocks, a.scratch2,
                                                      a.scratch2_count, 0);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        topk_level_kernel<<<1, kMergeBlock, 0, st>>>(a, a.scratch2, a.scratch2_count, m1, nullptr, nullptr, 1);
        return cudaGetLastError();
    }
    topk_level_kernel<<<1, kMergeBlock, 0, st>>>(a, a.scratch, a.scratch_count, blocks, nullptr, nullptr, 1);
    return cudaGetLastError();
}

// ---- one-launch top-k of a priced chunk's worklist.  Up to 64 CTAs scan
// the worklist as topk_block_kernel does; CTAs form groups of kFan: the last
// CTA of a group to finish (a ticket counter after a memory fence, no
// waiting) merges the group's lists, and the last group to finish folds
// the group lists and the incoming state into the state, then clears the
// tickets for the next launch.  Shorter worklists take fewer CTAs: up to
// kOneGroupEntries one group (its last CTA folds the state at once), up to
// kFewEntries CTA 0 alone.
constexpr int kFusedBlock = 256;
constexpr int kFusedGroups = 4;
// at most this many entries (typically the survivors of the threshold once
// a pricing's first chunks have filled the state): CTA 0 alone merges them
// with the state and the other CTAs leave at once
constexpr int kFewEntries = 4096;
// at most this many (and more than kFewEntries): the first kFan CTAs scan
// them as one group, whose last CTA folds the group's lists and the state
// directly -- one ticket level instead of two
constexpr int kOneGroupEntries = 32768;

// Stage lists [first, first + nl) of src into lists[0 ..), one warp per
// list; the entries were written by other CTAs, so they are read past L1.
template <int W>
__device__ void stage_lists(TopkEntry* lists, int* counts, const TopkEntry* src, const int32_t* src_count,
                            int first, int nl, int k) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int w = warp; w < nl; w += W) {
        const int l = first + w;
        const int c = min(__ldcg(src_count + l), k);
        const TopkEntry* from = src + (size_t)l * kMaxTopK;
        for (int i = lane; i < c; i += 32) {
            TopkEntry e;
            e.idx = __ldcg(&from[i].idx);
            e.T = __ldcg(&from[i].T);
            e.nM = __ldcg(&from[i].nM);
            e.pad = 0;
            lists[w * kMaxTopK + i] = e;
        }
        if (lane == 0) counts[w] = c;
    }
}

// Write list 0 (counts[0] entries) to dst / dst_count and draw a ticket:
// the barrier gathers the CTA's stores, thread 0 fences them (fences are
// cumulative) before its atomic, and the CTA that draws the last of
// `expected` tickets fences again before it reads the others' lists.
__device__ bool publish(const TopkEntry* list, const int* counts, TopkEntry* dst, int32_t* dst_count,
                        int32_t* ticket, int expected, int* last_flag) {
    for (int p = threadIdx.x; p < counts[0]; p += blockDim.x) dst[p] = list[p];
    if (threadIdx.x == 0) *dst_count = counts[0];
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const bool last = atomicAdd(ticket, 1) == expected - 1;
        if (last) __threadfence();
        *last_flag = last;
    }
    __syncthreads();
    return *last_flag != 0;
}

__global__ void __launch_bounds__(kFusedBlock) topk_fused_kernel(TopkArgs a) {
    constexpr int W = kFusedBlock / 32;
    static_assert(W >= (kFan + 1) / 2, "a tree merge of W lists runs W / 2 warps at once");
    static_assert(kFusedGroups + 1 <= kFan + 1, "the final merge holds the group lists and the state");
    const int k = state_k(a.state);
    __shared__ TopkEntry lists[(kFan + 1) * kMaxTopK];
    __shared__ TopkEntry tmp[((kFan + 2) / 2) * kMaxTopK];
    __shared__ int counts[kFan + 1], tmp_counts[(kFan + 2) / 2];
    __shared__ int last_flag;
    __shared__ unsigned floor_bits;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool full = a.state->count >= k;
    TopkEntry bar;
    bar.idx = full ? a.state->idx[k - 1] : 0;
    bar.T = full ? a.state->T[k - 1] : 0;
    bar.nM = full ? a.state->nM[k - 1] : 0;
    bar.pad = 0;
    // the running threshold of the call (a float lower bound, lowered by a
    // margin that covers the rounding, on the k-th key of the candidates
    // priced so far): an entry whose key n*M / T, computed the same way,
    // falls below it has k entries of the call that rank before it
    const float floor_key = a.thr ? __uint_as_float(__ldcg(a.thr)) : 0.0f;
    // ---- this CTA's share of the worklist (all of it when it is short)
    int cnt = 0;
    TopkEntry* list = lists + warp * kMaxTopK;
    const int64_t n = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const bool few = n <= kFewEntries;
    const bool one_group = !few && n <= kOneGroupEntries;
    if (few && blockIdx.x != 0) return;
    if (one_group && blockIdx.x >= kFan) return;
    const int ncta = one_group ? min((int)gridDim.x, kFan) : (int)gridDim.x;  // CTAs that scan
    if (n <= 32) {
        // at most one entry per lane: warp 0 ranks them against each other
        // (the order is strict, so the ranks are distinct), places them,
        // and merges them with the state -- no CTA barrier
        if (warp != 0) return;
        TopkEntry e;
        e.idx = 0;
        e.T = 0;
        e.nM = 0;
        e.pad = 0;
        bool valid = lane < n && fetch<true>(a, lane, e);
        if (valid && full) valid = better(e, bar);
        int rank = 0;
        for (int j = 0; j < 32; ++j) {
            TopkEntry o;
            o.idx = __shfl_sync(0xffffffffu, e.idx, j);
            o.T = __shfl_sync(0xffffffffu, e.T, j);
            o.nM = __shfl_sync(0xffffffffu, e.nM, j);
            o.pad = 0;
            const bool ov = __shfl_sync(0xffffffffu, valid, j);
            rank += (valid && ov && better(o, e)) ? 1 : 0;
        }
        const int nv = min(__popc(__ballot_sync(0xffffffffu, valid)), k);
        TopkEntry* mine = lists + kMaxTopK;
        if (valid && rank < k) mine[rank] = e;
        const int c = min(max(a.state->count, 0), k);
        for (int i = lane; i < c; i += 32) {
            TopkEntry x;
            x.idx = a.state->idx[i];
            x.T = a.state->T[i];
            x.nM = a.state->nM[i];
            x.pad = 0;
            lists[i] = x;
        }
        __syncwarp();
        const int total = warp_merge(lists, c, mine, nv, tmp, k);
        for (int i = lane; i < kMaxTopK; i += 32) {
            const bool live = i < total;
            a.state->idx[i] = live ? tmp[i].idx : -1;
            a.state->T[i] = live ? tmp[i].T : -1;
            a.state->nM[i] = live ? tmp[i].nM : 0;
        }
        if (lane == 0) {
            a.state->count = total;
            if (a.thr && total >= k) {
                // the new k-th key, rounded and lowered by 2^-16 (see TopkArgs::thr)
                const TopkEntry x = tmp[k - 1];
                const float r = (float)x.nM / (float)x.T * (1.0f - 1.0f / 65536.0f);
                atomicMax(a.thr, __float_as_uint(r));
            }
        }
        return;
    }
    const int64_t step = few ? (int64_t)W * 32 : (int64_t)ncta * W * 32;
    const int64_t start = few ? (int64_t)warp * 32 : ((int64_t)blockIdx.x * W + warp) * 32;
    // ---- first pass (k <= 32, while the state is not full: once it is,
    //      its k-th entry stops almost every entry): the k-th largest float
    //      key among the entries each warp visits; k of them reach it, so
    //      the CTA's largest such key, lowered by the margin, is a floor for
    //      every entry that can enter the top-k, and it raises the call's
    //      threshold for the other CTAs
    float floor_cta = floor_key;
    if (k <= 32 && !full) {
        if (threadIdx.x == 0) floor_bits = 0;
        __syncthreads();
        float run = -1.0f;
        for (int64_t base = start; base < n; base += step) {
            const int64_t i = base + lane;
            float key = -1.0f;
            if (i < n) {
                const int64_t T = a.wl_T[i];
                if (T > 0) key = (float)a.wl_nM[i] / (float)T;
            }
            run = warp_keep_top32(run, key);
        }
        const float kth = __shfl_sync(0xffffffffu, run, k - 1);
        if (lane == 0 && kth > 0.0f) atomicMax(&floor_bits, __float_as_uint(kth * (1.0f - 1.0f / 65536.0f)));
        __syncthreads();
        floor_cta = fmaxf(floor_cta, __uint_as_float(floor_bits));
        if (threadIdx.x == 0 && a.thr && floor_cta > floor_key) atomicMax(a.thr, __float_as_uint(floor_cta));
        if (a.thr) floor_cta = fmaxf(floor_cta, __uint_as_float(__ldcg(a.thr)));
    }
    constexpr int U = 4;
    for (int64_t base = start; base < n; base += step * U) {
        TopkEntry e[U];
        bool valid[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t i = base + u * step + lane;
            valid[u] = false;
            e[u].idx = 0;
            e[u].T = 0;
            e[u].nM = 0;
            e[u].pad = 0;
            if (i < n) valid[u] = fetch<true>(a, i, e[u]);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const bool above = valid[u] && (floor_cta <= 0.0f || (float)e[u].nM / (float)e[u].T >= floor_cta);
            warp_offer(list, cnt, k, above && (!full || better(e[u], bar)), e[u]);
        }
    }
    if (lane == 0) counts[warp] = cnt;
    cta_tree_merge(lists, counts, tmp, tmp_counts, W, k);
    int nl = 1;  // lists to fold with the incoming state
    if (!few) {
        // ---- the last CTA of its group merges the group's lists
        const int group = blockIdx.x / kFan, ngroups = (ncta + kFan - 1) / kFan;
        const int first = group * kFan, gsize = min(kFan, ncta - first);
        if (!publish(lists, counts, a.scratch + (size_t)blockIdx.x * kMaxTopK, a.scratch_count + blockIdx.x,
                     a.tickets + group, gsize, &last_flag))
            return;
        stage_lists<W>(lists, counts, a.scratch, a.scratch_count, first, gsize, k);
        cta_tree_merge(lists, counts, tmp, tmp_counts, gsize, k);
        // ---- the last group folds the group lists and the incoming state
        //      (a single group's list is already in lists[0])
        if (ngroups > 1) {
            if (!publish(lists, counts, a.scratch2 + (size_t)group * kMaxTopK, a.scratch2_count + group,
                         a.tickets + kFan, ngroups, &last_flag))
                return;
            stage_lists<W>(lists, counts, a.scratch2, a.scratch2_count, 0, ngroups, k);
        }
        nl = ngroups;
    }
    const int ngroups = nl;
    if (warp == W - 1) {
        const int c = min(max(a.state->count, 0), k);
        for (int i = lane; i < c; i += 32) {
            TopkEntry e;
            e.idx = a.state->idx[i];
            e.T = a.state->T[i];
            e.nM = a.state->nM[i];
            e.pad = 0;
            lists[ngroups * kMaxTopK + i] = e;
        }
        if (lane == 0) counts[ngroups] = c;
    }
    cta_tree_merge(lists, counts, tmp, tmp_counts, ngroups + 1, k);
    const int total = counts[0];
    for (int p = threadIdx.x; p < kMaxTopK; p += blockDim.x) {
        const bool live = p < total;
        a.state->idx[p] = live ? lists[p].idx : -1;
        a.state->T[p] = live ? lists[p].T : -1;
        a.state->nM[p] = live ? lists[p].nM : 0;
    }
    if (threadIdx.x == 0) {
        a.state->count = total;
        if (a.thr && total >= k) {
            // the new k-th key, rounded and lowered by 2^-16 (see TopkArgs::thr)
            const TopkEntry e = lists[k - 1];
            const float r = (float)e.nM / (float)e.T * (1.0f - 1.0f / 65536.0f);
            atomicMax(a.thr, __float_as_uint(r));
        }
    }
    // every other CTA has drawn its tickets (none did on the short path):
    // clear them for the next launch
    if (!few)
        for (int i = threadIdx.x; i <= kFan; i += blockDim.x) a.tickets[i] = 0;
}

__global__ void topk_reset_kernel(heddle_topk_state* s, int k) {
    for (int p = threadIdx.x; p < kMaxTopK; p += blockDim.x) {
        s->idx[p] = -1;
        s->T[p] = -1;
        s->nM[p] = 0;
    }
    if (threadIdx.x == 0) {
        s->k = k;
        s->count = 0;
    }
}

}  // namespace

cudaError_t launch_topk(const TopkArgs& a, int num_sms, cudaStream_t st, int64_t* launches) {
    if (a.n <= 0) return cudaSuccess;
    const int64_t per_block = (int64_t)kTopkBlock * 16;  // at least 16 candidates per thread
    int grid = (int)std::min<int64_t>((a.n + per_block - 1) / per_block, (int64_t)kFan * kFan);
    grid = std::max(1, std::min(grid, a.max_blocks));
    (void)num_sms;
    topk_block_kernel<false, kTopkBlock><<<grid, kTopkBlock, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (launches) *launches += 1;
    return merge_lists(a, grid, st, launches);
}

cudaError_t launch_topk_worklist(const TopkArgs& a, int64_t n, int num_sms, cudaStream_t st,
                                 int64_t* launches) {
    if (n <= 0) return cudaSuccess;
    // one launch: the worklist holds only the searched candidates, most of
    // them rejected by the state's k-th
    const int64_t per_block = (int64_t)kFusedBlock * 16;
    int grid = (int)std::min<int64_t>((n + per_block - 1) / per_block, (int64_t)kFan * kFusedGroups);
    grid = std::max(1, std::min(grid, a.max_blocks));
    (void)num_sms;
    topk_fused_kernel<<<grid, kFusedBlock, 0, st>>>(a);
    if (launches) *launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_topk_reset(heddle_topk_state* state, int32_t k, cudaStream_t st) {
    topk_reset_kernel<<<1, 64, 0, st>>>(state, k);
    return cudaGetLastError();
}

}  // namespace hd
