// heddle_noalloc.cu -- heddle_topk_noalloc: the top-k merge of a priced batch
// for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code that runs inside another
// framework's memory pool, where every device allocation must go through
// that pool, or code that must not allocate after start-up.  They also
// cannot create a heddle context, which allocates its scratch.  This entry
// point needs neither: its scratch -- one top-k list per CTA -- lives in a
// file-scope __device__ array that the CUDA runtime sets up when the library
// is loaded, and each CTA scans a fixed slice of the batch, so the array
// bounds the batch size instead of the call allocating for it.
//
// The array's name is only a host-side stand-in: host code passes the
// device address obtained from cudaGetSymbolAddress on the current device,
// looked up again on every call (a device reset reloads the module and can
// move the array, so an address kept from an earlier call could be stale).

#include "heddle_rank.cuh"

namespace hd {
namespace {

constexpr int kNaBlock = 256;
constexpr int kNaWarps = kNaBlock / 32;
constexpr int kNaMergeBlock = 512;
constexpr int kNaMergeWarps = kNaMergeBlock / 32;
constexpr int64_t kNaSlice = 65536;  // candidates per CTA
constexpr int kNaLists = HEDDLE_TOPK_NOALLOC_MAX_N / kNaSlice;
static_assert(kNaLists * kNaSlice == HEDDLE_TOPK_NOALLOC_MAX_N, "slices must tile the maximum batch");

// kNaLists lists of kMaxTopK entries, then kNaLists int32 counts
constexpr size_t kListBytes = sizeof(TopkEntry) * kMaxTopK * kNaLists;
constexpr size_t kScratchBytes = kListBytes + sizeof(int32_t) * kNaLists;
static __device__ __align__(256) unsigned char g_topk_scratch[kScratchBytes];

struct NaArgs {
    const uint16_t* M;
    const int64_t* T;
    const uint16_t* ndp;
    const uint8_t* status;
    int64_t n;
    int64_t base_index;
    heddle_topk_state* state;
    TopkEntry* lists;  // device address of g_topk_scratch
    int32_t* counts;   // device address of its count section
};

// CTA b scans candidates [b * kNaSlice, (b + 1) * kNaSlice) and writes one
// list and its length (every CTA writes its count, so nothing has to be
// cleared between calls).  A candidate that does not beat the incoming
// state's k-th entry (when the state is full) cannot enter the result and
// is not offered.
__global__ void __launch_bounds__(kNaBlock) noalloc_block_kernel(NaArgs a) {
    const int k = state_k(a.state);
    __shared__ TopkEntry lists[kNaWarps][kMaxTopK];
    __shared__ int counts[kNaWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool full = a.state->count >= k;
    TopkEntry bar;
    bar.idx = full ? a.state->idx[k - 1] : 0;
    bar.T = full ? a.state->T[k - 1] : 0;
    bar.nM = full ? a.state->nM[k - 1] : 0;
    bar.pad = 0;
    int cnt = 0;
    const int64_t lo = (int64_t)blockIdx.x * kNaSlice;
    const int64_t hi = min(a.n, lo + kNaSlice);
    for (int64_t base = lo + warp * 32; base < hi; base += kNaWarps * 32) {
        const int64_t c = base + lane;
        TopkEntry e;
        bool valid = false;
        if (c < hi && a.status[c] == HEDDLE_CAND_OK) {
            e.idx = a.base_index + c;
            e.T = a.T[c];
            e.nM = (uint32_t)a.ndp[c] * (uint32_t)a.M[c];
            e.pad = 0;
            valid = !full || better(e, bar);
        }
        warp_offer(&lists[warp][0], cnt, k, valid, e);
    }
    if (lane == 0) counts[warp] = cnt;
    cta_merge_lists(&lists[0][0], counts, k, kNaWarps, cnt, a.lists + (size_t)blockIdx.x * kMaxTopK,
                    a.counts + blockIdx.x);
}

// One CTA folds the `blocks` lists and the incoming state into the state.
__global__ void __launch_bounds__(kNaMergeBlock) noalloc_merge_kernel(NaArgs a, int blocks) {
    __shared__ TopkEntry lists[kNaMergeWarps * kMaxTopK];
    __shared__ int counts[kNaMergeWarps];
    __shared__ TopkEntry merged[kMaxTopK];
    __shared__ int32_t merged_count;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = state_k(a.state);
    int cnt = 0;
    TopkEntry* list = lists + warp * kMaxTopK;
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
    for (int l = warp; l < blocks; l += kNaMergeWarps) {
        const int cl = a.counts[l];
        for (int b = 0; b < cl; b += 32) {
            const bool valid = b + lane < cl;
            TopkEntry e;
            if (valid) e = a.lists[(size_t)l * kMaxTopK + b + lane];
            warp_offer(list, cnt, k, valid, e);
        }
    }
    if (lane == 0) counts[warp] = cnt;
    cta_merge_lists(lists, counts, k, kNaMergeWarps, cnt, merged, &merged_count);
    __syncthreads();
    for (int p = threadIdx.x; p < kMaxTopK; p += blockDim.x) {
        const bool live = p < merged_count;
        a.state->idx[p] = live ? merged[p].idx : -1;
        a.state->T[p] = live ? merged[p].T : -1;
        a.state->nM[p] = live ? merged[p].nM : 0;
    }
    if (threadIdx.x == 0) a.state->count = merged_count;
}

// Device address of g_topk_scratch on the current device, looked up on
// every call: cheap once the module is loaded, and never stale after a
// device reset.
cudaError_t scratch_for_current_device(unsigned char** out) {
    unsigned char* ptr = nullptr;
    const cudaError_t e = cudaGetSymbolAddress((void**)&ptr, g_topk_scratch);
    if (e != cudaSuccess) return e;
    *out = ptr;
    return cudaSuccess;
}

}  // namespace
}  // namespace hd

extern "C" heddle_status heddle_topk_noalloc(const heddle_candidates* cands, const heddle_results* results,
                                             heddle_topk_state* state, void* stream) {
    if (!cands || !results || !state) return HEDDLE_E_ARG;
    if (cands->n < 0) return HEDDLE_E_ARG;
    if (cands->n > HEDDLE_TOPK_NOALLOC_MAX_N) return HEDDLE_E_LIMIT;
    if (cands->n == 0) return HEDDLE_OK;
    if (!cands->M || !results->T || !results->n_dp || !results->status) return HEDDLE_E_ARG;
    unsigned char* scratch = nullptr;
    if (hd::scratch_for_current_device(&scratch) != cudaSuccess) return HEDDLE_E_CUDA;
    hd::NaArgs a;
    a.M = cands->M;
    a.T = results->T;
    a.ndp = results->n_dp;
    a.status = results->status;
    a.n = cands->n;
    a.base_index = cands->base_index;
    a.state = state;
    a.lists = reinterpret_cast<hd::TopkEntry*>(scratch);
    a.counts = reinterpret_cast<int32_t*>(scratch + hd::kListBytes);
    const int blocks = (int)((cands->n + hd::kNaSlice - 1) / hd::kNaSlice);
    cudaStream_t st = (cudaStream_t)stream;
    hd::noalloc_block_kernel<<<blocks, hd::kNaBlock, 0, st>>>(a);
    if (cudaGetLastError() != cudaSuccess) return HEDDLE_E_CUDA;
    hd::noalloc_merge_kernel<<<1, hd::kNaMergeBlock, 0, st>>>(a, blocks);
    if (cudaGetLastError() != cudaSuccess) return HEDDLE_E_CUDA;
    return HEDDLE_OK;
}
