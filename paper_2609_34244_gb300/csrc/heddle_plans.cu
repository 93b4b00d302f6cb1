// heddle_plans.cu -- multi-template plan pricing (Algorithm 1: a plan is a
// sequence of structural templates, each holding its own GPUs; the reward
// of a step is the throughput the new template adds).
//
// The library first prices the template slots as standalone candidates
// (screen + search, unchanged): PartitionLayers and the memory decision do
// not depend on the DP degree n, so the split, the bottleneck and OOM carry
// over.  Slot t is priced only for the plans whose templates 0 .. t-1 are
// each OK alone (a walk ends at its first template that is not OK, and a
// template is OK in the walk only if it is OK alone); for the others the
// screen writes SKIPPED.  The first template, on the whole free cluster,
// keeps its standalone price.  This kernel then walks each plan in
// order against the GPUs the earlier templates left: the template's n
// comes from the free GPUs per node -- n = min over (type, size class e) of
// floor(cap / demand), cap = sum over nodes of floor(free / 2^e) 2^e, exact
// for power-of-two groups placed largest first -- then T is re-evaluated
// with that n (only the gradient term depends on it), and the template's
// groups are placed largest first on a node of its type whose free GPUs
// equal the group size, else on the node with the fewest free GPUs above
// it (§5.1).  Decisions depend on nodes only through their free counts, so
// each thread keeps, per GPU type, a histogram of nodes by free GPUs (in
// shared memory, sized to the cluster's types and largest node, capacities
// recomputed from it when a template's degree is needed).  The
// first template that is not OK ends the plan; the plan's throughput is the
// sum over placed templates of n M 1e9 / T, each term rounded in IEEE
// double, in template order.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kPlanBlock = 128;

// Per-thread arrays in shared memory, interleaved by thread (element e of
// thread t at [e * kPlanBlock + t]): the node histogram hist[g][v] (nodes of
// type g with v free GPUs, v <= vmax) and the demand word dem[g] (GPUs of
// groups per size class e in 16-bit field e).
__host__ __device__ inline size_t plan_smem(int NT, int vmax) {
    return (size_t)kPlanBlock * (2 * (size_t)NT * (vmax + 1) + 8 * kMaxTypes);
}

__global__ void __launch_bounds__(kPlanBlock, 8) plan_kernel(PlanArgs a) {
    const Layout& y = a.lay;
    const int L = y.L, NT = y.NT, V = a.vmax;
    const int64_t* P = reinterpret_cast<const int64_t*>(a.img + y.offP);
    const int64_t* PB = reinterpret_cast<const int64_t*>(a.img + y.offPB);
    const int64_t* p2p = reinterpret_cast<const int64_t*>(a.img + y.offP2P);
    const int64_t* inter = reinterpret_cast<const int64_t*>(a.img + y.offInter);
    const int32_t* maxn = reinterpret_cast<const int32_t*>(a.img + y.offMaxN);
    const int32_t* pow2 = reinterpret_cast<const int32_t*>(a.img + y.offPow2);
    extern __shared__ __align__(16) unsigned char psm[];
    uint64_t* dem = reinterpret_cast<uint64_t*>(psm) + threadIdx.x;  // [g * kPlanBlock]
    uint16_t* hist = reinterpret_cast<uint16_t*>(psm + (size_t)8 * kMaxTypes * kPlanBlock) + threadIdx.x;
    // the cluster's nodes per type and GPU count, shared by the CTA
    __shared__ __align__(4) uint16_t init[kMaxTypes][kPlanMaxNode + 1];
    for (int i = threadIdx.x; i < kMaxTypes * (kPlanMaxNode + 1); i += blockDim.x) (&init[0][0])[i] = 0;
    __syncthreads();
    for (int b = threadIdx.x; b < a.n_nodes; b += blockDim.x) {
        // 16-bit counts: at most 65535 nodes (the library's GPU limit)
        unsigned int* w = reinterpret_cast<unsigned int*>(&init[0][0]) +
                          ((a.node_type[b] * (kPlanMaxNode + 1) + a.node_gpus[b]) >> 1);
        atomicAdd(w, ((a.node_type[b] * (kPlanMaxNode + 1) + a.node_gpus[b]) & 1) ? 0x10000u : 1u);
    }
    __syncthreads();
    auto H = [&](int g, int v) -> uint16_t& { return hist[(size_t)(g * (V + 1) + v) * kPlanBlock]; };
    // Most plans end at their first template, whose standalone price is
    // already what the walk would give it (the whole cluster is free, so
    // its degree, split and T are the standalone ones): a quick pass writes
    // such plans' later slots as SKIPPED, and the others are queued in
    // shared memory and walked 128 at a time, one per thread, so the lanes
    // that walk are dense.
    __shared__ int32_t queue[2 * kPlanBlock];
    __shared__ int queued;
    if (threadIdx.x == 0) queued = 0;
    __syncthreads();
    auto walk = [&](int64_t c) {
        for (int g = 0; g < NT; ++g)
            for (int v = 0; v <= V; ++v) H(g, v) = init[g][v];
        const int nt = min((int)a.n_tmpl[c], a.slots);
        bool ended = false;
        int placed = 0;
        double thr = 0.0;
        // (the slots past the plan's templates were priced SKIPPED)
        for (int t = 0; t < nt; ++t) {
            const PlanSlot& sl = a.slot[t];
            uint8_t st = HEDDLE_CAND_SKIPPED;
            int64_t T = -1, B = -1;
            int64_t n = 0;
            const int S = sl.S[c];
            const int M = sl.M[c];
            if (!ended) {
                const uint8_t st0 = sl.status[c];
                if (st0 == HEDDLE_CAND_INVALID) {
                    st = HEDDLE_CAND_INVALID;
                } else {
                    // demand per (type, size class) in GPUs of groups of that class
                    for (int g = 0; g < NT; ++g) dem[g * kPlanBlock] = 0;
                    uint32_t present = 0;
                    for (int s = 0; s < S; ++s) {
                        const int b = sl.code[(int64_t)s * sl.stride + c];
                        const int g = b & 7, j = (b >> 3) & 3;
                        const int unit = (1 << j) <= maxn[g] ? (1 << j) : pow2[g];
                        dem[g * kPlanBlock] += (uint64_t)(1u << j) << (16 * (31 - __clz(unit)));
                        present |= 1u << g;
                    }
                    // n = min over (type, class e) of floor(cap / demand),
                    // cap = sum over nodes of floor(free / 2^e) 2^e
                    int64_t best = -1;
                    for (uint32_t pm = present; pm; pm &= pm - 1) {
                        const int g = __ffs(pm) - 1;
                        int64_t cap[4] = {0, 0, 0, 0};
                        for (int v = 1; v <= V; ++v) {
                            const int64_t h = H(g, v);
                            if (!h) continue;
                            cap[0] += h * v;
                            cap[1] += h * ((v >> 1) << 1);
                            cap[2] += h * ((v >> 2) << 2);
                            cap[3] += h * ((v >> 3) << 3);
                        }
                        const uint64_t dw = dem[g * kPlanBlock];
                        uint32_t d = 0;
#pragma unroll
                        for (int e = 3; e >= 0; --e) {
                            const uint32_t f = (uint32_t)(dw >> (16 * e)) & 0xffffu;
                            d += f;
                            if (f == 0) continue;  // dominated by the class above
                            const int64_t q = cap[e] / d;
                            if (best < 0 || q < best) best = q;
                        }
                    }
                    n = best < 0 ? 0 : best;
                    if (n == 0) {
                        st = HEDDLE_CAND_NO_FIT;
                    } else if (st0 == HEDDLE_CAND_OOM) {
                        st = HEDDLE_CAND_OOM;
                    } else if (t == 0) {
                        // the whole cluster is free: n, T and B are the standalone ones
                        T = sl.T[c];
                        B = sl.B[c];
                        st = HEDDLE_CAND_OK;
                        if (n != (int64_t)sl.ndp[c]) atomicOr(a.err, kErrInternal);
                    } else {
                        // Evaluate with this n: T = (M-1) max t_s + sum t_s + max g_s
                        int64_t tmax = 0, tsum = 0;
                        uint64_t bestG = 0, bestD = 1;
                        int sg = -1;
                        int hi = sl.bounds[c];
                        for (int s = 0; s < S; ++s) {
                            const int b = sl.code[(int64_t)s * sl.stride + c];
                            const int g = b & 7, j = (b >> 3) & 3;
                            const int lo = hi;
                            hi = sl.bounds[(int64_t)(s + 1) * sl.bstride + c];
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
                    }
                    if (st == HEDDLE_CAND_OK) {
                        thr = __dadd_rn(thr, __ddiv_rn(__dmul_rn((double)(n * (int64_t)M), 1e9), (double)T));
                        placed = t + 1;
                        // place n copies of the groups, largest first
                        for (int e = 3; e >= 0; --e) {
                            const int w = 1 << e;
                            for (uint32_t pm = present; pm; pm &= pm - 1) {
                                const int g = __ffs(pm) - 1;
                                int64_t left = (int64_t)(((dem[g * kPlanBlock] >> (16 * e)) & 0xffffu) >> e) * n;
                                while (left > 0) {
                                    if (w <= V && H(g, w) > 0) {
                                        // nodes with exactly w free: m of them filled
                                        const int64_t m = min(left, (int64_t)H(g, w));
                                        H(g, w) -= (uint16_t)m;
                                        H(g, 0) += (uint16_t)m;
                                        left -= m;
                                        continue;
                                    }
                                    int v = w + 1;
                                    while (v <= V && H(g, v) == 0) ++v;
                                    if (v > V) {
                                        atomicOr(a.err, kErrInternal);  // n came from these nodes
                                        break;
                                    }
                                    H(g, v) -= 1;
                                    H(g, v - w) += 1;
                                    left -= 1;
                                }
                            }
                        }
                    }
                }
                if (st != HEDDLE_CAND_OK) ended = true;
            }
            if (t > 0) {  // the first template keeps its standalone results
                sl.T[c] = T;
                sl.B[c] = B;
                sl.ndp[c] = (uint16_t)(st == HEDDLE_CAND_OK || st == HEDDLE_CAND_OOM ? n : 0);
                sl.status[c] = st;
                // an OK template keeps its standalone split; any other
                // status clears the planes
                if (st != HEDDLE_CAND_OK)
                    for (int s = 0; s <= kMaxStages; ++s) sl.bounds[(int64_t)s * sl.bstride + c] = 0;
            }
        }
        a.placed[c] = (uint8_t)placed;
        a.thr[c] = thr;
    };
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t c0 = (int64_t)blockIdx.x * blockDim.x;
    while (true) {
        const bool more = c0 < a.n;  // uniform over the CTA
        if (more) {
            const int64_t c = c0 + threadIdx.x;
            bool walks = false;
            if (c < a.n) {
                // a plan walks from its second template on; the others keep
                // their slots as priced (templates past the first OK-alone
                // prefix were priced SKIPPED) and take the first template's
                // throughput if it is OK
                const int nt = min((int)a.n_tmpl[c], a.slots);
                const bool ok0 = nt >= 1 && a.slot[0].status[c] == HEDDLE_CAND_OK;
                walks = ok0 && nt >= 2;
                if (!walks) {
                    double thr = 0.0;
                    if (ok0) {
                        const PlanSlot& s0 = a.slot[0];
                        const int64_t n0 = s0.ndp[c];
                        thr = __ddiv_rn(__dmul_rn((double)(n0 * (int64_t)s0.M[c]), 1e9), (double)s0.T[c]);
                    }
                    a.placed[c] = ok0 ? 1 : 0;
                    a.thr[c] = thr;
                }
            }
            const unsigned wm = __ballot_sync(0xffffffffu, walks);
            if (wm) {
                int q0 = 0;
                if (lane == __ffs(wm) - 1) q0 = atomicAdd(&queued, __popc(wm));
                q0 = __shfl_sync(0xffffffffu, q0, __ffs(wm) - 1);
                if (walks) queue[q0 + __popc(wm & ((1u << lane) - 1))] = (int32_t)(c0 + threadIdx.x);
            }
        }
        __syncthreads();
        const int have = queued;
        const int take = more ? (have >= kPlanBlock ? kPlanBlock : 0) : min(have, kPlanBlock);
        const int64_t mine = threadIdx.x < take ? (int64_t)queue[have - take + threadIdx.x] : -1;
        __syncthreads();
        if (threadIdx.x == 0) queued = have - take;
        if (mine >= 0) walk(mine);
        __syncthreads();
        if (!more && have - take == 0) break;
        if (more) c0 += stride;
    }
}

// skip[i] = plan i does not reach template t on its templates' own prices:
// it has at most t templates, or template t - 1 is not OK alone (a
// template priced SKIPPED is not OK either, so the mask of t covers every
// earlier template).
__global__ void plan_mask_kernel(const uint8_t* n_tmpl, int slots, int t, const uint8_t* prev_status,
                                 uint8_t* skip, int64_t n) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int nt = min((int)n_tmpl[i], slots);
        const bool reach = nt > t && (t == 0 || prev_status[i] == HEDDLE_CAND_OK);
        skip[i] = reach ? 0 : 1;
    }
}

}  // namespace

cudaError_t launch_plan_mask(const uint8_t* n_tmpl, int slots, int t, const uint8_t* prev_status, uint8_t* skip,
                             int64_t n, int num_sms, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((n + 255) / 256, (int64_t)num_sms * 8);
    plan_mask_kernel<<<grid, 256, 0, st>>>(n_tmpl, slots, t, prev_status, skip, n);
    return cudaGetLastError();
}

cudaError_t launch_plans(const PlanArgs& a, int num_sms, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    if (a.vmax < 1 || a.vmax > kPlanMaxNode) return cudaErrorInvalidValue;
    const size_t smem = plan_smem(a.lay.NT, a.vmax);
    int per_sm = 0;
    const cudaError_t e = resident_blocks(reinterpret_cast<const void*>(&plan_kernel), kPlanBlock, smem, &per_sm);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const int grid = (int)std::min<int64_t>((a.n + kPlanBlock - 1) / kPlanBlock, (int64_t)num_sms * per_sm);
    plan_kernel<<<grid, kPlanBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
