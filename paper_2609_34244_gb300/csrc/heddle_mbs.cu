// heddle_mbs.cu -- the micro-batch-size fill (§5.3 "Micro-batch size"):
// the library prices a batch once per power-of-two micro-batch size (the
// same screen and search kernels, with that size's cost tables and M / 2^i
// micro-batches), and this kernel folds each size's results into the best
// so far: a size replaces the current choice when it is OK and its
// iteration time is strictly shorter (or the current choice is not OK), so
// equal times keep the smaller size.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

__global__ void __launch_bounds__(256) mbs_merge_kernel(MbsMergeArgs a) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < a.n; c += stride) {
        if (a.status_l[c] != HEDDLE_CAND_OK) continue;
        const int64_t T = a.T_l[c];
        if (a.status[c] == HEDDLE_CAND_OK && !(T < a.T[c])) continue;
        a.T[c] = T;
        a.B[c] = a.B_l[c];
        a.ndp[c] = a.n_l[c];
        a.status[c] = HEDDLE_CAND_OK;
        if (a.mbs) a.mbs[c] = (uint8_t)a.level;
        if (a.bounds && a.bounds_l)
            for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = a.bounds_l[(int64_t)s * a.bstride_l + c];
    }
}

}  // namespace

cudaError_t launch_mbs_merge(const MbsMergeArgs& a, int num_sms, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((a.n + 255) / 256, (int64_t)num_sms * 8);
    mbs_merge_kernel<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
