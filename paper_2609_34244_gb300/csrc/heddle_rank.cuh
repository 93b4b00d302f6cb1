// heddle_rank.cuh -- the rank order of priced plans and warp-level top-k
// lists, shared by the top-k kernels and the search kernels that fuse the
// block-level top-k.
//
// Plans are ranked by predicted throughput (§5 overview); with n replicas of
// M microbatches per iteration time T a plan processes n*M microbatches per
// T, so a ranks before b iff nM_a * T_b > nM_b * T_a (exact, 128-bit), and
// equal throughput goes to the smaller global index.  The order is strict, so
// the top-k is unique and does not depend on the launch shape.
#pragma once

#include "heddle_internal.cuh"

namespace hd {

typedef unsigned __int128 u128;

__device__ __forceinline__ bool better(const TopkEntry& a, const TopkEntry& b) {
    const u128 l = (u128)a.nM * (u128)(uint64_t)b.T;
    const u128 r = (u128)b.nM * (u128)(uint64_t)a.T;
    if (l != r) return l > r;
    return a.idx < b.idx;
}

// Warp-cooperative insertion into a sorted list of `cnt` entries (capacity
// k <= 64; lane l owns slots l and l + 32).  All lanes pass the same e.
__device__ inline void warp_insert(TopkEntry* list, int& cnt, int k, const TopkEntry& e) {
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
__device__ inline void warp_offer(TopkEntry* list, int& cnt, int k, bool valid, const TopkEntry& e) {
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

// One round of a warp's running top-32 of float keys: lane l holds the
// (l+1)-th largest key so far (run); the round's 32 keys (one per lane) are
// sorted by a bitonic network, reversed against run (the larger of each
// pair is a bitonic sequence holding the 32 largest of both) and merged.
__device__ __forceinline__ float warp_keep_top32(float run, float key) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const float o = __shfl_xor_sync(0xffffffffu, key, stride);
            const bool desc = (lane & size) == 0 || size == 32;
            key = (((lane & stride) == 0) == desc) ? fmaxf(key, o) : fminf(key, o);
        }
    float c = fmaxf(run, __shfl_sync(0xffffffffu, key, 31 - lane));
#pragma unroll
    for (int stride = 16; stride > 0; stride >>= 1) {
        const float o = __shfl_xor_sync(0xffffffffu, c, stride);
        c = (lane & stride) == 0 ? fmaxf(c, o) : fminf(c, o);
    }
    return c;
}

// Merge the sorted lists of the CTA's warps (lists[w], counts[w]) into
// lists[0] with warp 0, then write it and its length to out / out_count.
// Every thread of the CTA must call it (it synchronises the CTA).
__device__ inline void cta_merge_lists(TopkEntry* lists, int* counts, int k, int warps, int cnt0,
                                       TopkEntry* out, int32_t* out_count) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (warp == 0) {
        int cnt = cnt0;
        for (int w2 = 1; w2 < warps; ++w2) {
            const int c2 = counts[w2];
            for (int b = 0; b < c2; b += 32) {
                const bool valid = b + lane < c2;
                TopkEntry e;
                if (valid) e = lists[w2 * kMaxTopK + b + lane];
                warp_offer(lists, cnt, k, valid, e);
            }
        }
        for (int p = lane; p < cnt; p += 32) out[p] = lists[p];
        if (lane == 0) *out_count = cnt;
    }
}

// Merge two sorted lists A (na) and B (nb) into out (the first min(na + nb,
// k) entries), one warp, all lanes in parallel: an entry's place in the
// merged list is its place in its own list plus the number of entries of
// the other list that rank before it (a binary search); the order is strict,
// so the places are distinct.  out must not overlap A or B.
__device__ inline int warp_merge(const TopkEntry* A, int na, const TopkEntry* B, int nb, TopkEntry* out,
                                 int k) {
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < na && i < k; i += 32) {
        const TopkEntry x = A[i];
        int lo = 0, hi = nb;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (better(B[mid], x)) lo = mid + 1; else hi = mid;
        }
        if (i + lo < k) out[i + lo] = x;
    }
    for (int i = lane; i < nb && i < k; i += 32) {
        const TopkEntry x = B[i];
        int lo = 0, hi = na;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (better(A[mid], x)) lo = mid + 1; else hi = mid;
        }
        if (i + lo < k) out[i + lo] = x;
    }
    __syncwarp();
    return min(na + nb, k);
}

// Tree merge of W sorted lists (lists[w * kMaxTopK], counts[w]) held in
// shared memory, using tmp (ceil(W / 2) lists); the result ends in lists[0]
// with length counts[0].  Every thread of the CTA must call it, with at
// least W / 2 warps.
__device__ inline void cta_tree_merge(TopkEntry* lists, int* counts, TopkEntry* tmp, int* tmp_counts, int W,
                                      int k) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int width = W; width > 1; width = (width + 1) / 2) {
        const int half = (width + 1) / 2;
        __syncthreads();
        if (warp < width - half) {
            const int c = warp_merge(lists + warp * kMaxTopK, counts[warp], lists + (warp + half) * kMaxTopK,
                                     counts[warp + half], tmp + warp * kMaxTopK, k);
            if (lane == 0) tmp_counts[warp] = c;
        }
        __syncthreads();
        if (warp < width - half) {
            for (int i = lane; i < tmp_counts[warp]; i += 32) lists[warp * kMaxTopK + i] = tmp[warp * kMaxTopK + i];
            if (lane == 0) counts[warp] = tmp_counts[warp];
        }
    }
    __syncthreads();
}

// capacity of a top-k state, clamped to the list size
__device__ __forceinline__ int state_k(const heddle_topk_state* s) {
    return min(max(s->k, 1), kMaxTopK);
}

}  // namespace hd
