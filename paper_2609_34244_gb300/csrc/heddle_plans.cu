// heddle_plans.cu -- multi-template plan pricing (Algorithm 1: a plan is a
// sequence of structural templates, each holding its own GPUs; the reward
// of a step is the throughput the new template adds).
//
// The library first prices every template slot of every plan as a
// standalone candidate (screen + search, unchanged): PartitionLayers and
// the memory decision do not depend on the DP degree n, so the split, the
// bottleneck and OOM carry over.  This kernel then walks each plan in
// order against the GPUs the earlier templates left: the template's n
// comes from the free GPUs per node -- n = min over (type, size class e) of
// floor(cap / demand), cap = sum over nodes of floor(free / 2^e) 2^e, exact
// for power-of-two groups placed largest first -- then T is re-evaluated
// with that n (only the gradient term depends on it), and the template's
// groups are placed largest first on a node of its type whose free GPUs
// equal the group size, else on the node with the fewest free GPUs above
// it (§5.1).  Decisions depend on nodes only through their free counts, so
// each thread keeps, per GPU type, a histogram of nodes by free GPUs.  The
// first template that is not OK ends the plan; the plan's throughput is the
// sum over placed templates of n M 1e9 / T, each term rounded in IEEE
// double, in template order.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kPlanBlock = 128;

__global__ void __launch_bounds__(kPlanBlock) plan_kernel(PlanArgs a) {
    const Layout& y = a.lay;
    const int L = y.L;
    const int64_t* P = reinterpret_cast<const int64_t*>(a.img + y.offP);
    const int64_t* PB = reinterpret_cast<const int64_t*>(a.img + y.offPB);
    const int64_t* p2p = reinterpret_cast<const int64_t*>(a.img + y.offP2P);
    const int64_t* inter = reinterpret_cast<const int64_t*>(a.img + y.offInter);
    const int32_t* maxn = reinterpret_cast<const int32_t*>(a.img + y.offMaxN);
    const int32_t* pow2 = reinterpret_cast<const int32_t*>(a.img + y.offPow2);
    // the cluster's nodes per type and GPU count, shared by the CTA
    __shared__ uint32_t init[kMaxTypes][kPlanMaxNode + 1];
    for (int i = threadIdx.x; i < kMaxTypes * (kPlanMaxNode + 1); i += blockDim.x) (&init[0][0])[i] = 0;
    __syncthreads();
    for (int b = threadIdx.x; b < a.n_nodes; b += blockDim.x) atomicAdd(&init[a.node_type[b]][a.node_gpus[b]], 1u);
    __syncthreads();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < a.n; c += stride) {
        // nodes per type by free GPUs, and per (type, class e) the GPUs
        // groups of size >= 2^e can use: sum of floor(free / 2^e) 2^e
        uint16_t hist[kMaxTypes][kPlanMaxNode + 1];
        int64_t cap[kMaxTypes][4];
        for (int g = 0; g < kMaxTypes; ++g) {
            for (int e = 0; e < 4; ++e) cap[g][e] = 0;
            for (int v = 0; v <= kPlanMaxNode; ++v) {
                hist[g][v] = (uint16_t)init[g][v];
                for (int e = 0; e < 4; ++e) cap[g][e] += (int64_t)init[g][v] * ((v >> e) << e);
            }
        }
        const int nt = min((int)a.n_tmpl[c], a.slots);
        bool ended = false;
        int placed = 0;
        double thr = 0.0;
        for (int t = 0; t < a.slots; ++t) {
            const PlanSlot& sl = a.slot[t];
            uint8_t st = HEDDLE_CAND_SKIPPED;
            int64_t T = -1, B = -1;
            int64_t n = 0;
            const int S = sl.S[c];
            const int M = sl.M[c];
            if (!ended && t < nt) {
                const uint8_t st0 = sl.status[c];
                if (st0 == HEDDLE_CAND_INVALID) {
                    st = HEDDLE_CAND_INVALID;
                } else {
                    // demand per (type, size class) in GPUs of groups of that class
                    uint32_t dem[kMaxTypes][4];
                    for (int g = 0; g < kMaxTypes; ++g)
                        for (int e = 0; e < 4; ++e) dem[g][e] = 0;
                    for (int s = 0; s < S; ++s) {
                        const int b = sl.code[(int64_t)s * sl.stride + c];
                        const int g = b & 7, j = (b >> 3) & 3;
                        const int unit = (1 << j) <= maxn[g] ? (1 << j) : pow2[g];
                        dem[g][31 - __clz(unit)] += 1u << j;
                    }
                    int64_t best = -1;
                    for (int g = 0; g < kMaxTypes; ++g) {
                        uint32_t d = 0;
                        for (int e = 3; e >= 0; --e) {
                            d += dem[g][e];
                            if (dem[g][e] == 0) continue;  // dominated by the class above
                            const int64_t q = cap[g][e] / d;
                            if (best < 0 || q < best) best = q;
                        }
                    }
                    n = best < 0 ? 0 : best;
                    if (n == 0) {
                        st = HEDDLE_CAND_NO_FIT;
                    } else if (st0 == HEDDLE_CAND_OOM) {
                        st = HEDDLE_CAND_OOM;
                    } else {
                        // Evaluate with this n: T = (M-1) max t_s + sum t_s + max g_s
                        int64_t tmax = 0, tsum = 0;
                        uint64_t bestG = 0, bestD = 1;
                        int sg = -1;
                        for (int s = 0; s < S; ++s) {
                            const int b = sl.code[(int64_t)s * sl.stride + c];
                            const int g = b & 7, j = (b >> 3) & 3;
                            const int lo = sl.bounds[(int64_t)s * sl.bstride + c];
                            const int hi = sl.bounds[(int64_t)(s + 1) * sl.bstride + c];
                            int64_t cs = 0;
                            if (s + 1 < S) {
                                const int bn = sl.code[(int64_t)(s + 1) * sl.stride + c];
                                const int h = bn & 7, jn = (bn >> 3) & 3;
                                const int same = (g == h) && ((1 << j) + (1 << jn) <= maxn[g]);
                                cs = p2p[(g * 8 + h) * 2 + same];
                            }
                            const int64_t* row = P + (g * 4 + j) * (L + 1);
                            const int64_t ts = row[hi] - row[lo] + cs;
                            tmax = max(tmax, ts);
                            tsum += ts;
                            const uint64_t G = (uint64_t)(PB[hi] - PB[lo]);
                            const uint64_t D = (uint64_t)inter[g] << j;
                            if (sg < 0 || (u128)G * bestD > (u128)bestG * D) {
                                sg = s;
                                bestG = G;
                                bestD = D;
                            }
                        }
                        int64_t gmax = 0;
                        if (n > 1) {
                            const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * bestG;
                            bool ok = true;
                            gmax = (int64_t)ceil_div_u128(num, (uint64_t)n * bestD, &ok);
                            if (!ok) atomicOr(a.err, kErrInternal);
                        }
                        T = (int64_t)(M - 1) * tmax + tsum + gmax;
                        B = tmax;
                        st = HEDDLE_CAND_OK;
                        thr = __dadd_rn(thr, __ddiv_rn(__dmul_rn((double)(n * (int64_t)M), 1e9), (double)T));
                        placed = t + 1;
                        // place n copies of the groups, largest first
                        for (int e = 3; e >= 0; --e) {
                            const uint32_t w = 1u << e;
                            for (int g = 0; g < kMaxTypes; ++g) {
                                int64_t left = (int64_t)(dem[g][e] >> e) * n;
                                while (left > 0) {
                                    if (hist[g][w] > 0) {
                                        // nodes with exactly w free: m of them filled
                                        const int64_t m = min(left, (int64_t)hist[g][w]);
                                        hist[g][w] -= (uint16_t)m;
                                        hist[g][0] += (uint16_t)m;
                                        for (int e2 = 0; e2 < 4; ++e2) cap[g][e2] -= m * (((int64_t)w >> e2) << e2);
                                        left -= m;
                                        continue;
                                    }
                                    int v = w + 1;
                                    while (v <= kPlanMaxNode && hist[g][v] == 0) ++v;
                                    if (v > kPlanMaxNode) {
                                        atomicOr(a.err, kErrInternal);  // n came from these nodes
                                        break;
                                    }
                                    hist[g][v] -= 1;
                                    hist[g][v - w] += 1;
                                    for (int e2 = 0; e2 < 4; ++e2)
                                        cap[g][e2] -= (int64_t)(((v >> e2) << e2) - (((v - (int)w) >> e2) << e2));
                                    left -= 1;
                                }
                            }
                        }
                    }
                }
                if (st != HEDDLE_CAND_OK) ended = true;
            }
            sl.T[c] = T;
            sl.B[c] = B;
            sl.ndp[c] = (uint16_t)(st == HEDDLE_CAND_OK || st == HEDDLE_CAND_OOM ? n : 0);
            sl.status[c] = st;
            if (st != HEDDLE_CAND_OK)
                for (int s = 0; s <= kMaxStages; ++s) sl.bounds[(int64_t)s * sl.bstride + c] = 0;
        }
        a.placed[c] = (uint8_t)placed;
        a.thr[c] = thr;
    }
}

}  // namespace

cudaError_t launch_plans(const PlanArgs& a, int num_sms, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((a.n + kPlanBlock - 1) / kPlanBlock, (int64_t)num_sms * 16);
    plan_kernel<<<grid, kPlanBlock, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
