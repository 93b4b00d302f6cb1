// heddle_topk.cu -- rank and top-k of priced candidates.
//
// Plans are ranked by predicted throughput (§5 overview); with n replicas of
// M microbatches per iteration time T a plan processes n*M microbatches per
// T, so a ranks before b iff nM_a * T_b > nM_b * T_a (exact, 128-bit), and
// equal throughput goes to the smaller global index.  The order is strict, so
// the top-k is unique and the result does not depend on the launch shape.
//
// Launch 1: every CTA scans a slice of the batch; each warp keeps its own
// sorted list in shared memory (an entry is inserted only if it beats the
// current k-th, which after warm-up is rare), the CTA merges its warps'
// lists and writes one list to scratch.  Launch 2: one CTA merges the
// per-CTA lists with the incoming state.  No CTA waits on another.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

typedef unsigned __int128 u128;

constexpr int kTopkBlock = 256;
constexpr int kWarps = kTopkBlock / 32;

__device__ __forceinline__ bool better(const TopkEntry& a, const TopkEntry& b) {
    const u128 l = (u128)a.nM * (u128)(uint64_t)b.T;
    const u128 r = (u128)b.nM * (u128)(uint64_t)a.T;
    if (l != r) return l > r;
    return a.idx < b.idx;
}

// Warp-cooperative insertion into a sorted list of `cnt` entries (capacity
// k <= 64; lane l owns slots l and l + 32).  All lanes pass the same e.
__device__ void warp_insert(TopkEntry* list, int& cnt, int k, const TopkEntry& e) {
    const int lane = threadIdx.x & 31;
    const int p0 = lane, p1 = lane + 32;
    const bool b0 = p0 < cnt && better(list[p0], e);
    const bool b1 = p1 < cnt && better(list[p1], e);
    const int pos = __popc(__ballot_sync(0xffffffffu, b0)) + __popc(__ballot_sync(0xffffffffu, b1));
    if (pos >= k) return;
    const int ncnt = min(cnt + 1, k);
    TopkEntry v0, v1;
    if (p0 < ncnt) v0 = p0 == pos ? e : (p0 > pos ? list[p0 - 1] : list[p0]);
    if (p1 < ncnt) v1 = p1 == pos ? e : (p1 > pos ? list[p1 - 1] : list[p1]);
    __syncwarp();
    if (p0 < ncnt) list[p0] = v0;
    if (p1 < ncnt) list[p1] = v1;
    __syncwarp();
    cnt = ncnt;
}

// Offer one entry per lane (valid lanes only) to the warp's list.
__device__ void warp_offer(TopkEntry* list, int& cnt, int k, bool valid, const TopkEntry& e) {
    const bool full = cnt >= k;
    bool want = valid;
    if (valid && full) want = better(e, list[k - 1]);
    unsigned m = __ballot_sync(0xffffffffu, want);
    while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        TopkEntry x;
        x.idx = __shfl_sync(0xffffffffu, e.idx, src);
        x.T = __shfl_sync(0xffffffffu, e.T, src);
        x.nM = __shfl_sync(0xffffffffu, e.nM, src);
        x.pad = 0;
        // re-check against the list as it is now (earlier lanes may have raised the bar)
        if (cnt < k || better(x, list[k - 1])) warp_insert(list, cnt, k, x);
    }
}

// capacity of the state, clamped to the list size
__device__ __forceinline__ int state_k(const heddle_topk_state* s) {
    return min(max(s->k, 1), kMaxTopK);
}

__global__ void __launch_bounds__(kTopkBlock) topk_block_kernel(TopkArgs a) {
    const int k = state_k(a.state);
    __shared__ TopkEntry lists[kWarps][kMaxTopK];
    __shared__ int counts[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int cnt = 0;
    TopkEntry* list = lists[warp];
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
    for (int64_t base = gw * 32; base < a.n; base += nwarps * 32) {
        const int64_t c = base + lane;
        TopkEntry e;
        bool valid = false;
        if (c < a.n && a.status[c] == HEDDLE_CAND_OK) {
            e.idx = a.base_index + c;
            e.T = a.T[c];
            e.nM = (uint32_t)a.ndp[c] * (uint32_t)a.M[c];
            e.pad = 0;
            valid = true;
        }
        warp_offer(list, cnt, k, valid, e);
    }
    if (lane == 0) counts[warp] = cnt;
    __syncthreads();
    if (warp == 0) {
        for (int w2 = 1; w2 < kWarps; ++w2) {
            const int c2 = counts[w2];
            for (int b = 0; b < c2; b += 32) {
                const bool valid = b + lane < c2;
                TopkEntry e;
                if (valid) e = lists[w2][b + lane];
                warp_offer(list, cnt, k, valid, e);
            }
        }
        for (int p = lane; p < cnt; p += 32) a.scratch[(size_t)blockIdx.x * kMaxTopK + p] = list[p];
        if (lane == 0) a.scratch_count[blockIdx.x] = cnt;
    }
}

__global__ void __launch_bounds__(kTopkBlock) topk_merge_kernel(TopkArgs a, int blocks) {
    __shared__ TopkEntry lists[kWarps][kMaxTopK];
    __shared__ int counts[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = state_k(a.state);
    int cnt = 0;
    TopkEntry* list = lists[warp];
    // warp 0 starts from the incoming state; every warp takes a share of the CTA lists
    if (warp == 0) {
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
    for (int blk = warp; blk < blocks; blk += kWarps) {
        const int cb = a.scratch_count[blk];
        for (int b = 0; b < cb; b += 32) {
            const bool valid = b + lane < cb;
            TopkEntry e;
            if (valid) e = a.scratch[(size_t)blk * kMaxTopK + b + lane];
            warp_offer(list, cnt, k, valid, e);
        }
    }
    if (lane == 0) counts[warp] = cnt;
    __syncthreads();
    if (warp == 0) {
        for (int w2 = 1; w2 < kWarps; ++w2) {
            const int c2 = counts[w2];
            for (int b = 0; b < c2; b += 32) {
                const bool valid = b + lane < c2;
                TopkEntry e;
                if (valid) e = lists[w2][b + lane];
                warp_offer(list, cnt, k, valid, e);
            }
        }
        for (int p = lane; p < kMaxTopK; p += 32) {
            if (p < cnt) {
                a.state->idx[p] = list[p].idx;
                a.state->T[p] = list[p].T;
                a.state->nM[p] = list[p].nM;
            } else {
                a.state->idx[p] = -1;
                a.state->T[p] = -1;
                a.state->nM[p] = 0;
            }
        }
        if (lane == 0) a.state->count = cnt;
    }
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
    topk_block_kernel<<<grid, kTopkBlock, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    topk_merge_kernel<<<1, kTopkBlock, 0, st>>>(a, grid);
    return cudaGetLastError();
}

cudaError_t launch_topk_reset(heddle_topk_state* state, int32_t k, cudaStream_t st) {
    topk_reset_kernel<<<1, 64, 0, st>>>(state, k);
    return cudaGetLastError();
}

}  // namespace hd
