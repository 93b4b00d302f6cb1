// heddle_topk.cu -- rank and top-k of priced candidates.
//
// The rank order and the warp-level lists are in heddle_rank.cuh.
//
// Launch 1: every CTA scans a slice of the batch (or, after a pricing call,
// of the worklist of searched candidates only); each warp keeps its own
// sorted list in shared memory (an entry is inserted only if it beats the
// current k-th, which after warm-up is rare), the CTA merges its warps'
// lists and writes one list to scratch.  Then the per-CTA lists are folded
// into the state: one CTA directly for up to 32 lists, else a reduction
// launch of 32 lists per CTA first.  No CTA waits on another.

#include <algorithm>

#include "heddle_rank.cuh"

namespace hd {
namespace {

constexpr int kTopkBlock = 256;
constexpr int kWarps = kTopkBlock / 32;
constexpr int kMergeBlock = 512;
constexpr int kMergeWarps = kMergeBlock / 32;

// One candidate entry: from a batch's results, or from the worklist of a
// priced chunk (only the searched candidates, T = -1 unless OK).
template <bool kWorklist>
__device__ __forceinline__ bool fetch(const TopkArgs& a, int64_t i, TopkEntry& e) {
    e.pad = 0;
    if (kWorklist) {
        const int64_t T = a.wl_T[i];
        if (T < 0) return false;
        e.idx = a.base_index + a.wl_idx[i];
        e.T = T;
        e.nM = a.wl_nM[i];
        return true;
    }
    if (a.status[i] != HEDDLE_CAND_OK) return false;
    e.idx = a.base_index + i;
    e.T = a.T[i];
    e.nM = (uint32_t)a.ndp[i] * (uint32_t)a.M[i];
    return true;
}

template <bool kWorklist>
__global__ void __launch_bounds__(kTopkBlock) topk_block_kernel(TopkArgs a) {
    const int k = state_k(a.state);
    __shared__ TopkEntry lists[kWarps][kMaxTopK];
    __shared__ int counts[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int cnt = 0;
    TopkEntry* list = lists[warp];
    const int64_t n = kWorklist ? min((int64_t)*a.wl_count, (int64_t)a.wl_cap) : a.n;
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
    for (int64_t base = gw * 32; base < n; base += nwarps * 32) {
        const int64_t i = base + lane;
        TopkEntry e;
        const bool valid = i < n && fetch<kWorklist>(a, i, e);
        warp_offer(list, cnt, k, valid, e);
    }
    if (lane == 0) counts[warp] = cnt;
    cta_merge_lists(&lists[0][0], counts, k, kWarps, cnt, a.scratch + (size_t)blockIdx.x * kMaxTopK,
                    a.scratch_count + blockIdx.x);
}

// Offer the entries of list `l` (count `c`) to this warp's list.
__device__ __forceinline__ void offer_list(const TopkEntry* l, int c, TopkEntry* list, int& cnt, int k) {
    const int lane = threadIdx.x & 31;
    for (int b = 0; b < c; b += 32) {
        const bool valid = b + lane < c;
        TopkEntry e;
        if (valid) e = l[b + lane];
        warp_offer(list, cnt, k, valid, e);
    }
}

// First merge level: CTA b folds lists [32 b, 32 b + 32) into out[b]; each
// warp takes two lists, whose counts it loads together.
__global__ void __launch_bounds__(kMergeBlock) topk_reduce_kernel(TopkArgs a, int blocks) {
    __shared__ TopkEntry lists[kMergeWarps * kMaxTopK];
    __shared__ int counts[kMergeWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = state_k(a.state);
    int cnt = 0;
    TopkEntry* list = lists + warp * kMaxTopK;
    const int l0 = blockIdx.x * 32 + warp, l1 = l0 + kMergeWarps;
    const int c0 = l0 < blocks ? a.scratch_count[l0] : 0;
    const int c1 = l1 < blocks ? a.scratch_count[l1] : 0;
    offer_list(a.scratch + (size_t)l0 * kMaxTopK, c0, list, cnt, k);
    offer_list(a.scratch + (size_t)l1 * kMaxTopK, c1, list, cnt, k);
    if (lane == 0) counts[warp] = cnt;
    cta_merge_lists(lists, counts, k, kMergeWarps, cnt, a.scratch2 + (size_t)blockIdx.x * kMaxTopK,
                    a.scratch2_count + blockIdx.x);
}

// Last merge level: one CTA folds `blocks` lists and the incoming state.
__global__ void __launch_bounds__(kMergeBlock) topk_merge_kernel(TopkArgs a, const TopkEntry* src,
                                                                 const int32_t* src_count, int blocks) {
    __shared__ TopkEntry lists[kMergeWarps * kMaxTopK];
    __shared__ int counts[kMergeWarps];
    __shared__ TopkEntry merged[kMaxTopK];
    __shared__ int32_t merged_count;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = state_k(a.state);
    int cnt = 0;
    TopkEntry* list = lists + warp * kMaxTopK;
    if (warp == 0) {
        // the incoming state
        const int c0 = min(max(a.state->count, 0), k);
        for (int b = 0; b < c0; b += 32) {
            const bool valid = b + lane < c0;
            TopkEntry e;
            if (valid) {
                e.idx = a.state->idx[b + lane];
                e.T = a.state->T[b + lane];
                e.nM = a.state->nM[b + lane];
                e.pad = 0;
            }
            warp_offer(list, cnt, k, valid, e);
        }
    }
    for (int l = warp; l < blocks; l += kMergeWarps) offer_list(src + (size_t)l * kMaxTopK, src_count[l], list, cnt, k);
    if (lane == 0) counts[warp] = cnt;
    cta_merge_lists(lists, counts, k, kMergeWarps, cnt, merged, &merged_count);
    __syncthreads();
    for (int p = threadIdx.x; p < kMaxTopK; p += blockDim.x) {
        const bool live = p < merged_count;
        a.state->idx[p] = live ? merged[p].idx : -1;
        a.state->T[p] = live ? merged[p].T : -1;
        a.state->nM[p] = live ? merged[p].nM : 0;
    }
    if (threadIdx.x == 0) a.state->count = merged_count;
}

// Merge `blocks` per-CTA lists of a.scratch into *a.state: directly, or
// through one reduction level of 32 lists per CTA when there are many.
cudaError_t merge_lists(const TopkArgs& a, int blocks, cudaStream_t st) {
    if (blocks <= 2 * kMergeWarps) {
        topk_merge_kernel<<<1, kMergeBlock, 0, st>>>(a, a.scratch, a.scratch_count, blocks);
        return cudaGetLastError();
    }
    const int m1 = (blocks + 31) / 32;
    topk_reduce_kernel<<<m1, kMergeBlock, 0, st>>>(a, blocks);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    topk_merge_kernel<<<1, kMergeBlock, 0, st>>>(a, a.scratch2, a.scratch2_count, m1);
    return cudaGetLastError();
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

cudaError_t launch_topk(const TopkArgs& a, int num_sms, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    const int64_t per_block = (int64_t)kTopkBlock * 8;  // at least 8 candidates per thread
    int grid = (int)std::min<int64_t>((a.n + per_block - 1) / per_block, (int64_t)2 * num_sms);
    grid = std::max(1, std::min(grid, a.max_blocks));
    topk_block_kernel<false><<<grid, kTopkBlock, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return merge_lists(a, grid, st);
}

cudaError_t launch_topk_worklist(const TopkArgs& a, int64_t n, int num_sms, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int64_t per_block = (int64_t)kTopkBlock * 8;
    int grid = (int)std::min<int64_t>((n + per_block - 1) / per_block, (int64_t)2 * num_sms);
    grid = std::max(1, std::min(grid, a.max_blocks));
    topk_block_kernel<true><<<grid, kTopkBlock, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return merge_lists(a, grid, st);
}

cudaError_t launch_topk_reset(heddle_topk_state* state, int32_t k, cudaStream_t st) {
    topk_reset_kernel<<<1, 64, 0, st>>>(state, k);
    return cudaGetLastError();
}

}  // namespace hd
