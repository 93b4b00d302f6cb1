// heddle_price.cu -- pricing kernel: decode + validate (§5.1 masks), DP
// degree (§5.3 packing), PartitionLayers (min-max split, §3.1 listing, with
// the memory validation of §5.2) and Evaluate (1F1B iteration time, §5.3).
//
// One thread prices one candidate; a persistent grid strides over the batch.
// Each CTA first copies the cost-table image into shared memory with one
// bulk TMA copy (cp.async.bulk, completion on an mbarrier).
//
// PartitionLayers is solved exactly by a threshold search on the bottleneck
// value B.  probe(B) decides whether some split has every stage time <= B
// and every stage within memory:
//   forward:  U_0 = 0, U_{s+1} = furthest end stage s can reach from U_s
//             (an upper bound on every feasible boundary a_{s+1});
//   backward: C_S = {L}; C_s = { i in [s, U_s] : the smallest j in C_{s+1}
//             above i gives a stage [i, j) that fits };  feasible iff stage 0
//             fits [0, min C_1).
// Stage costs grow with the interval, so the smallest successor dominates
// and every C_s is exactly the set of feasible stage-s starts below U_s.
// Each probe also returns the largest stage cost it accepted (hi) and the
// smallest it rejected (lo): every B' in [hi, B] (feasible probe) or
// [B, lo) (infeasible probe) takes the same decisions, so the search moves
// its bracket to those values and ends on B* = the smallest feasible B,
// itself a stage cost.  The C sets of that last probe give the canonical
// split directly: a_{s+1} = min { j in C_{s+1} : j > a_s }, the smallest
// boundary vector attaining B* (the feasible splits form a lattice under
// componentwise min).

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

typedef unsigned __int128 u128;

constexpr int kBlock = 128;
constexpr int kWords = 8;  // 256-bit position sets (L <= 255)
constexpr int kMaxIters = 256;
constexpr long long kStageWaitSpins = 1 << 22;

enum { CHK_OK = 0, CHK_FAIL = 1, CHK_MEM = 2 };

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Copy the table image into shared memory: one thread arms an mbarrier with
// the byte count and issues bulk copies; everyone waits on phase 0 with a
// bounded spin.  Returns false (and flags the error) if the wait gave up.
__device__ bool stage_tables(unsigned char* dst, const unsigned char* src, uint32_t bytes,
                             uint64_t* bar, uint32_t* err) {
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                     "r"(bytes)
                     : "memory");
        const uint32_t chunk = 32768;
        for (uint32_t o = 0; o < bytes; o += chunk) {
            const uint32_t nb = bytes - o < chunk ? bytes - o : chunk;
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, "
                "[%3];" ::"r"(smem_addr(dst + o)),
                "l"(src + o), "r"(nb), "r"(smem_addr(bar))
                : "memory");
        }
    }
    __syncthreads();
    uint32_t done = 0;
    for (long long spin = 0; spin < kStageWaitSpins; ++spin) {
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0; selp.u32 %0, 1, 0, p; }"
            : "=r"(done)
            : "r"(smem_addr(bar))
            : "memory");
        if (done) break;
    }
    const int all = __syncthreads_and(done != 0);
    if (!all && threadIdx.x == 0) atomicOr(err, kErrStageWait);
    return all != 0;
}

struct Tabs {
    const int64_t* P;
    const longlong2* SA;
    const int64_t* PB;
    const int64_t* p2p;
    const int64_t* mem;
    const int64_t* inter;
    const int64_t* minq;
    const int32_t* maxn;
    const int32_t* pow2;
    const int32_t* gpus;
    const int32_t* cap;
    int L, NT;
};

// One candidate's per-stage view plus the position sets of the probes.
struct Work {
    int S, L;
    uint16_t row[kMaxStages];      // offset of the stage's prefix row in P
    int64_t c[kMaxStages];         // P2P to the next stage
    int64_t capk[kMaxStages];      // memory per GPU x group size
    int32_t f[kMaxStages];         // in-flight microbatches
    uint8_t U[kMaxStages + 1];
    int16_t cmin[kMaxStages + 1], cmax[kMaxStages + 1];
    uint32_t C[kMaxStages + 1][kWords];
    int64_t hi_c, lo_c;            // snapping values of the current probe
    unsigned long long checks;
};

__device__ __forceinline__ int check(const Tabs& t, Work& w, int s, int i, int j, int64_t B) {
    const int64_t* P = t.P + w.row[s];
    const longlong2 a = t.SA[i], b = t.SA[j];
    const int64_t mem = (b.x - a.x) + (int64_t)w.f[s] * (b.y - a.y);
    ++w.checks;
    if (mem > w.capk[s]) return CHK_MEM;
    const int64_t cost = P[j] - P[i] + w.c[s];
    if (cost <= B) {
        if (cost > w.hi_c) w.hi_c = cost;
        return CHK_OK;
    }
    if (cost < w.lo_c) w.lo_c = cost;
    return CHK_FAIL;
}

__device__ __forceinline__ bool bit_test(const uint32_t* C, int i) { return (C[i >> 5] >> (i & 31)) & 1u; }

// largest set position in [lo, i], -1 if none
__device__ __forceinline__ int prev_set(const uint32_t* C, int i, int lo) {
    if (i < lo) return -1;
    int wd = i >> 5;
    uint32_t m = C[wd] & (0xffffffffu >> (31 - (i & 31)));
    while (m == 0) {
        if (--wd < (lo >> 5)) return -1;
        m = C[wd];
    }
    const int x = (wd << 5) + 31 - __clz(m);
    return x >= lo ? x : -1;
}

// smallest set position in [i, hi], -1 if none
__device__ __forceinline__ int next_set(const uint32_t* C, int i, int hi) {
    if (i > hi) return -1;
    int wd = i >> 5;
    uint32_t m = C[wd] & (0xffffffffu << (i & 31));
    while (m == 0) {
        if (++wd > (hi >> 5)) return -1;
        m = C[wd];
    }
    const int x = (wd << 5) + __ffs(m) - 1;
    return x <= hi ? x : -1;
}

__device__ bool probe(const Tabs& t, Work& w, int64_t B) {
    const int S = w.S, L = w.L;
    w.hi_c = -1;
    w.lo_c = kInf;
    // forward upper bounds on the boundaries
    w.U[0] = 0;
    for (int s = 0; s + 1 < S; ++s) {
        const int i = w.U[s];
        const int lim = L - (S - 1 - s);
        int j = i;
        while (j + 1 <= lim && check(t, w, s, i, j + 1, B) == CHK_OK) ++j;
        if (j < s + 1) return false;
        w.U[s + 1] = (uint8_t)j;
    }
    // backward feasible-start sets
    {
        // C_S = {L}; clear every word a successor search of stage S-1 can
        // read (positions S..L)
        uint32_t* CS = w.C[S];
        for (int wd = S >> 5; wd < (L >> 5); ++wd) CS[wd] = 0;
        CS[L >> 5] = 1u << (L & 31);
        w.cmin[S] = w.cmax[S] = (int16_t)L;
    }
    for (int s = S - 1; s >= 1; --s) {
        const uint32_t* Cn = w.C[s + 1];
        const int nmin = w.cmin[s + 1], nmax = w.cmax[s + 1];
        const int top = min((int)w.U[s], nmax - 1);
        if (top < s) return false;
        uint32_t* Cs = w.C[s];
        for (int wd = s >> 5; wd <= (top >> 5); ++wd) Cs[wd] = 0;
        int succ = next_set(Cn, top + 1, nmax);
        int i = top, hi = -1, lo = -1;
        while (i >= s) {
            const int r = check(t, w, s, i, succ, B);
            if (r == CHK_OK) {
                Cs[i >> 5] |= 1u << (i & 31);
                if (hi < 0) hi = i;
                lo = i;
                if (i >= nmin && bit_test(Cn, i)) succ = i;
                --i;
            } else {
                const int j2 = prev_set(Cn, i, nmin);
                if (j2 < 0) break;
                i = j2 - 1;
                succ = j2;
            }
        }
        if (hi < 0) return false;
        w.cmin[s] = (int16_t)lo;
        w.cmax[s] = (int16_t)hi;
    }
    return check(t, w, 0, 0, w.cmin[1], B) == CHK_OK;
}

template <bool kCount>
__global__ void __launch_bounds__(kBlock) price_kernel(PriceArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    if (!stage_tables(smem, a.img, a.lay.bytes, &bar, a.err)) return;

    const Layout& y = a.lay;
    Tabs t;
    t.P = reinterpret_cast<const int64_t*>(smem + y.offP);
    t.SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
    t.PB = reinterpret_cast<const int64_t*>(smem + y.offPB);
    t.p2p = reinterpret_cast<const int64_t*>(smem + y.offP2P);
    t.mem = reinterpret_cast<const int64_t*>(smem + y.offMem);
    t.inter = reinterpret_cast<const int64_t*>(smem + y.offInter);
    t.minq = reinterpret_cast<const int64_t*>(smem + y.offMinQ);
    t.maxn = reinterpret_cast<const int32_t*>(smem + y.offMaxN);
    t.pow2 = reinterpret_cast<const int32_t*>(smem + y.offPow2);
    t.gpus = reinterpret_cast<const int32_t*>(smem + y.offGpus);
    t.cap = reinterpret_cast<const int32_t*>(smem + y.offCap);
    t.L = y.L;
    t.NT = y.NT;
    const int L = y.L;

    Work w;
    w.L = L;
    unsigned long long probes = 0, priced = 0;
    w.checks = 0;

    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < a.n; c += stride) {
        const int S = a.S[c];
        const int M = a.M[c];
        int status = HEDDLE_CAND_OK;
        int64_t n = 0;
        uint8_t codes[kMaxStages];
        // ---- decode + validate (§5.1 depth / device / TP masks)
        if (S < 1 || S > kMaxStages || S > a.s_max || S > L || M < 1) {
            status = HEDDLE_CAND_INVALID;
        } else {
            for (int s = 0; s < S; ++s) {
                const int b = a.code[(int64_t)s * a.stride + c];
                codes[s] = (uint8_t)b;
                const int g = b & 7, j = (b >> 3) & 3;
                if ((b >> 5) != 0 || g >= t.NT || t.gpus[g] == 0 ||
                    (!a.moe && (1 << j) > t.maxn[g]))
                    status = HEDDLE_CAND_INVALID;
            }
        }
        // ---- DP degree: n = min over (type, size class) of capacity / demand
        if (status == HEDDLE_CAND_OK) {
            uint16_t dem[kMaxTypes][4];
            for (int g = 0; g < kMaxTypes; ++g)
                for (int e = 0; e < 4; ++e) dem[g][e] = 0;
            for (int s = 0; s < S; ++s) {
                const int g = codes[s] & 7, j = (codes[s] >> 3) & 3;
                const int k = 1 << j;
                const int unit = k <= t.maxn[g] ? k : t.pow2[g];
                for (int e = 0; (1 << e) <= unit; ++e) dem[g][e] += (uint16_t)k;
            }
            n = kInf;
            for (int g = 0; g < t.NT; ++g)
                for (int e = 0; e < 4; ++e)
                    if (dem[g][e]) n = min(n, (int64_t)(t.cap[g * 4 + e] / dem[g][e]));
            if (n == 0) status = HEDDLE_CAND_NO_FIT;
        }
        int64_t Bstar = -1, T = -1;
        if (status == HEDDLE_CAND_OK) {
            if (kCount) ++priced;
            // ---- stage views
            w.S = S;
            for (int s = 0; s < S; ++s) {
                const int g = codes[s] & 7, j = (codes[s] >> 3) & 3;
                w.row[s] = (uint16_t)((g * 4 + j) * (L + 1));
                if (s + 1 < S) {
                    const int h = codes[s + 1] & 7, jn = (codes[s + 1] >> 3) & 3;
                    const int same = (g == h) && ((1 << j) + (1 << jn) <= t.maxn[g]);
                    w.c[s] = t.p2p[(g * 8 + h) * 2 + same];
                } else {
                    w.c[s] = 0;
                }
                w.capk[s] = t.mem[g] << j;
                w.f[s] = min(S - s, M);
            }
            // ---- PartitionLayers: memory-only probe, then the threshold search
            if (kCount) ++probes;
            if (!probe(t, w, kInf)) {
                status = HEDDLE_CAND_OOM;
            } else {
                int64_t hi = w.hi_c, lo = 0;
                bool lo_known = false;
                // first guess: the balanced bottleneck of a proportional split
                float inv = 0.f, cw = 0.f;
                for (int s = 0; s < S; ++s) {
                    const float tot = (float)t.P[w.row[s] + L] + 1.0f;
                    inv += 1.0f / tot;
                    cw += (float)w.c[s] / tot;
                }
                int64_t B = (int64_t)((1.0f + cw) / inv);
                int64_t step = max((int64_t)1, (int64_t)((float)B * (float)S / (2.0f * (float)L)));
                int it = 0;
                while (lo < hi) {
                    if (B < lo) B = lo;
                    if (B > hi - 1) B = hi - 1;
                    if (kCount) ++probes;
                    if (probe(t, w, B)) {
                        hi = w.hi_c;
                    } else {
                        lo = w.lo_c;
                        lo_known = true;
                    }
                    if (lo >= hi) break;
                    if (!lo_known) {
                        B = hi - step;
                        step *= 2;
                    } else {
                        B = lo + (hi - lo) / 2;
                    }
                    if (++it > kMaxIters) {
                        atomicOr(a.err, kErrSearchBound);
                        break;
                    }
                }
                Bstar = hi;
                // sets of the optimum for the canonical split
                if (kCount) ++probes;
                if (!probe(t, w, Bstar)) atomicOr(a.err, kErrInternal);
                uint8_t bnd[kMaxStages + 1];
                bnd[0] = 0;
                for (int s = 0; s + 1 < S; ++s) {
                    const int x = next_set(w.C[s + 1], bnd[s] + 1, w.cmax[s + 1]);
                    bnd[s + 1] = (uint8_t)(x < 0 ? 0 : x);
                }
                bnd[S] = (uint8_t)L;
                // ---- Evaluate: T = (M-1) max t_s + sum t_s + max g_s
                int64_t tmax = 0, tsum = 0;
                int sg = -1;
                u128 bestG = 0, bestD = 1;
                for (int s = 0; s < S; ++s) {
                    const int64_t* P = t.P + w.row[s];
                    const int64_t ts = P[bnd[s + 1]] - P[bnd[s]] + w.c[s];
                    tmax = max(tmax, ts);
                    tsum += ts;
                    if (n > 1) {
                        // stage with the largest G_s / (k_s bw_s), compared exactly
                        const int g = codes[s] & 7, j = (codes[s] >> 3) & 3;
                        const u128 G = (u128)(t.PB[bnd[s + 1]] - t.PB[bnd[s]]);
                        const u128 D = (u128)t.inter[g] << j;
                        if (sg < 0 || G * bestD > bestG * D) {
                            sg = s;
                            bestG = G;
                            bestD = D;
                        }
                    }
                }
                if (tmax != Bstar) atomicOr(a.err, kErrInternal);
                int64_t gmax = 0;
                if (n > 1) {
                    // ring all-reduce over n replicas: ceil(2(n-1) G 1e9 / (n k bw))
                    const u128 num = (u128)2 * (u128)(n - 1) * bestG * 1000000000u;
                    const u128 den = (u128)n * bestD;
                    gmax = (int64_t)((num + den - 1) / den);
                }
                T = (int64_t)(M - 1) * Bstar + tsum + gmax;
                if (a.bounds) {
                    for (int s = 0; s <= kMaxStages; ++s)
                        a.bounds[(int64_t)s * a.n + c] = s <= S ? bnd[s] : 0;
                }
            }
        }
        a.T[c] = status == HEDDLE_CAND_OK ? T : -1;
        a.B[c] = status == HEDDLE_CAND_OK ? Bstar : -1;
        a.ndp[c] = (uint16_t)((status == HEDDLE_CAND_OK || status == HEDDLE_CAND_OOM) ? n : 0);
        a.status[c] = (uint8_t)status;
        if (a.bounds && status != HEDDLE_CAND_OK) {
            for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.n + c] = 0;
        }
    }
    if (kCount) {
        unsigned long long v0 = w.checks, v1 = probes, v2 = priced;
        for (int o = 16; o > 0; o >>= 1) {
            v0 += __shfl_down_sync(0xffffffffu, v0, o);
            v1 += __shfl_down_sync(0xffffffffu, v1, o);
            v2 += __shfl_down_sync(0xffffffffu, v2, o);
        }
        if ((threadIdx.x & 31) == 0) {
            atomicAdd(&a.counters[0], v0);
            atomicAdd(&a.counters[1], v1);
            atomicAdd(&a.counters[2], v2);
        }
    }
}

}  // namespace

cudaError_t launch_price(const PriceArgs& a, int num_sms, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    const size_t smem = a.lay.bytes;
    cudaError_t e;
    int per_sm = 0;
    if (a.counters) {
        e = cudaFuncSetAttribute(price_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, price_kernel<true>, kBlock, smem);
    } else {
        e = cudaFuncSetAttribute(price_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, price_kernel<false>, kBlock, smem);
    }
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t need = (a.n + kBlock - 1) / kBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    if (a.counters)
        price_kernel<true><<<grid, kBlock, smem, st>>>(a);
    else
        price_kernel<false><<<grid, kBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
