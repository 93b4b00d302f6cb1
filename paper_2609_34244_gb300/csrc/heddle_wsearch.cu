// heddle_wsearch.cu -- general PartitionLayers + Evaluate (§3.1 listing,
// §5.2 memory validation, §5.3 iteration time) for models whose layers
// differ, one warp per worklist entry.
//
// The search is the exact threshold search of the thread-per-entry kernel:
// probe(B) decides whether a split with every stage time <= B and every
// stage within memory exists,
//   forward:  U_0 = 0, U_{s+1} = the furthest end stage s reaches from U_s
//             (an upper bound on every feasible boundary a_{s+1});
//   backward: C_S = {L}; C_s = { i in [s, U_s] : the smallest j in C_{s+1}
//             above i gives a stage [i, j) that fits }; feasible iff stage 0
//             fits [0, min C_1);
// the probe also returns the largest accepted and the smallest rejected
// stage time, the bracket snaps to them, and the sets at B* give the
// canonical (lexicographically smallest) split.
//
// Here the 32 lanes of a warp judge 32 positions at once: the forward reach
// of a stage is the first rejection among 32 consecutive ends (stage time
// and memory grow with the end), and a backward set is built one 32-bit
// word per round -- lane l judges start 32 w + l against its smallest
// successor (a bit scan in the successor set) and the ballot is the word.
// Stage parameters come from the lane that holds the stage; the snap values
// are warp reductions; Evaluate runs with one lane per stage.  The table
// image is staged into shared memory with bulk asynchronous copies
// (cp.async.bulk, completion on an mbarrier, bounded wait); each warp keeps
// its sets and split in shared memory.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kWBlock = 256;
constexpr int kWarps = kWBlock / 32;
constexpr int kSetWords = 8;  // 256-bit position sets (L <= 255)
constexpr int kMaxIters = 256;
constexpr long long kWaitSpins = 1 << 22;
constexpr unsigned kFull = 0xffffffffu;

// per-warp shared state: sets C[0..32], forward bounds U, the split A
struct WarpArea {
    uint32_t C[kMaxStages + 1][kSetWords];
    uint8_t U[kMaxStages + 1];
    uint8_t A[kMaxStages + 1];
    uint8_t pad[30];
};

__device__ __forceinline__ uint32_t saddr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// The table image into shared memory: one thread arms an mbarrier with the
// byte count and issues the bulk copies; all wait on phase 0 with a bounded
// spin.  False (and the error flag) if the wait gave up.
__device__ bool load_image(unsigned char* dst, const unsigned char* src, uint32_t bytes, uint64_t* bar,
                           uint32_t* err) {
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(saddr(bar)));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(bar)), "r"(bytes)
                     : "memory");
        for (uint32_t o = 0; o < bytes; o += 32768) {
            const uint32_t nb = bytes - o < 32768 ? bytes - o : 32768;
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    saddr(dst + o)),
                "l"(src + o), "r"(nb), "r"(saddr(bar))
                : "memory");
        }
    }
    __syncthreads();
    uint32_t done = 0;
    for (long long spin = 0; spin < kWaitSpins; ++spin) {
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0; selp.u32 %0, 1, 0, p; }"
            : "=r"(done)
            : "r"(saddr(bar))
            : "memory");
        if (done) break;
    }
    const int all = __syncthreads_and(done != 0);
    if (!all && threadIdx.x == 0) atomicOr(err, kErrStageWait);
    return all != 0;
}

struct WTabs {
    const int64_t* P;
    const longlong2* SA;
    const int64_t* PB;
    const int64_t* p2p;
    const int64_t* mem;
    const int64_t* inter;
    const int32_t* maxn;
    int L;
};

// One stage's parameters, broadcast from the lane that holds them.
struct WStage {
    int row;       // offset of the (type, degree) prefix row
    int64_t c;     // P2P to the next stage
    int64_t capk;  // memory per GPU x devices
    int64_t f;     // in-flight micro-batches
};

__device__ __forceinline__ WStage bcast(const WStage& mine, int s) {
    WStage r;
    r.row = __shfl_sync(kFull, mine.row, s);
    r.c = __shfl_sync(kFull, mine.c, s);
    r.capk = __shfl_sync(kFull, mine.capk, s);
    r.f = __shfl_sync(kFull, mine.f, s);
    return r;
}

// Interval [i, j) on stage st: 0 fits (cost <= B), 1 too slow, 2 out of
// memory; the cost in *cost.
__device__ __forceinline__ int wjudge(const WTabs& t, const WStage& st, int i, int j, int64_t B, int64_t* cost) {
    const longlong2 si = t.SA[i], sj = t.SA[j];
    if ((sj.x - si.x) + st.f * (sj.y - si.y) > st.capk) return 2;
    const int64_t v = t.P[st.row + j] - t.P[st.row + i] + st.c;
    *cost = v;
    return v <= B ? 0 : 1;
}

__device__ __forceinline__ int64_t wmax64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, (int64_t)__shfl_xor_sync(kFull, v, o));
    return v;
}
__device__ __forceinline__ int64_t wmin64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = min(v, (int64_t)__shfl_xor_sync(kFull, v, o));
    return v;
}

// smallest set position of C in (i, L], -1 if none (warp-uniform inputs)
__device__ __forceinline__ int next_above(const uint32_t* C, int i, int L) {
    int w = (i + 1) >> 5;
    if (w > (L >> 5)) return -1;
    uint32_t m = C[w] & (0xffffffffu << ((i + 1) & 31));
    while (m == 0) {
        if (++w > (L >> 5)) return -1;
        m = C[w];
    }
    return (w << 5) + __ffs(m) - 1;
}

// Exact probe of bound B by one warp (all lanes, uniform result).  mine:
// the stage this lane holds (lane < S).  The sets land in wa.
__device__ bool wprobe(const WTabs& t, const WStage& mine, int S, int64_t B, WarpArea& wa, int64_t& hi_out,
                       int64_t& lo_out, unsigned long long& checks) {
    const int L = t.L;
    const int lane = threadIdx.x & 31;
    int64_t hi = -1, lo = kInf;
    bool ok = true;
    // forward upper bounds on the boundaries
    int u = 0;
    if (lane == 0) wa.U[0] = 0;
    for (int s = 0; s + 1 < S && ok; ++s) {
        const WStage st = bcast(mine, s);
        const int lim = L - (S - 1 - s);
        int reach = u;  // furthest accepted end (u: none yet)
        for (int base = u + 1; base <= lim; base += 32) {
            const int j = base + lane;
            int r = 1;  // beyond lim: treated as a rejection
            int64_t v = 0;
            if (j <= lim) {
                r = wjudge(t, st, u, j, B, &v);
                ++checks;
                if (r == 0) hi = max(hi, v);
                else if (r == 1) lo = min(lo, v);
            }
            const unsigned rej = __ballot_sync(kFull, r != 0);
            if (rej) {
                reach = base + __ffs(rej) - 2;
                break;
            }
            reach = base + 31;
        }
        if (reach < s + 1) ok = false;
        u = reach;
        if (lane == 0) wa.U[s + 1] = (uint8_t)reach;
    }
    __syncwarp();
    // backward feasible-start sets: C_S = {L}, then stages S-1 .. 1
    if (ok) {
        if (lane < kSetWords) wa.C[S][lane] = lane == (L >> 5) ? 1u << (L & 31) : 0u;
        __syncwarp();
        int nmax = L;
        for (int s = S - 1; s >= 1 && ok; --s) {
            const uint32_t* Cn = wa.C[s + 1];
            if (lane < kSetWords) wa.C[s][lane] = 0;
            __syncwarp();
            const int top = min((int)wa.U[s], nmax - 1);
            if (top < s) {
                ok = false;
                break;
            }
            const WStage st = bcast(mine, s);
            int any = 0, newmax = -1;
            for (int w = top >> 5; w >= (s >> 5); --w) {
                const int i = (w << 5) + lane;
                // smallest successor above i: in this word, else beyond it
                const uint32_t cw = Cn[w];
                const uint32_t above = lane == 31 ? 0u : (cw >> (lane + 1)) << (lane + 1);
                int beyond = -1;
                for (int w2 = w + 1; w2 <= (L >> 5); ++w2)
                    if (Cn[w2]) {
                        beyond = (w2 << 5) + __ffs(Cn[w2]) - 1;
                        break;
                    }
                const int succ = above ? (w << 5) + __ffs(above) - 1 : beyond;
                int r = 3;
                int64_t v = 0;
                if (i >= s && i <= top && succ >= 0) {
                    r = wjudge(t, st, i, succ, B, &v);
                    ++checks;
                    if (r == 0) hi = max(hi, v);
                    else if (r == 1) lo = min(lo, v);
                }
                const unsigned acc = __ballot_sync(kFull, r == 0);
                if (lane == 0) wa.C[s][w] = acc;
                if (acc) {
                    any = 1;
                    if (newmax < 0) newmax = (w << 5) + 31 - __clz(acc);
                }
            }
            __syncwarp();
            if (!any) ok = false;
            nmax = newmax;
        }
    }
    bool feasible = false;
    if (ok) {
        const int succ0 = S == 1 ? L : next_above(wa.C[1], 0, L);
        const WStage st0 = bcast(mine, 0);
        if (succ0 >= 0 && lane == 0) {
            int64_t v = 0;
            const int r = wjudge(t, st0, 0, succ0, B, &v);
            ++checks;
            if (r == 0) {
                hi = max(hi, v);
                feasible = true;
            } else if (r == 1) {
                lo = min(lo, v);
            }
        }
        feasible = __shfl_sync(kFull, feasible, 0);
    }
    hi_out = wmax64(hi);
    lo_out = wmin64(lo);
    return feasible;
}

template <bool kCount>
__global__ void __launch_bounds__(kWBlock) wsearch_kernel(PriceArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    if (!load_image(smem, a.img, a.lay.bytes, &bar, a.err)) return;
    const Layout& y = a.lay;
    WTabs t;
    t.P = reinterpret_cast<const int64_t*>(smem + y.offP);
    t.SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
    t.PB = reinterpret_cast<const int64_t*>(smem + y.offPB);
    t.p2p = reinterpret_cast<const int64_t*>(smem + y.offP2P);
    t.mem = reinterpret_cast<const int64_t*>(smem + y.offMem);
    t.inter = reinterpret_cast<const int64_t*>(smem + y.offInter);
    t.maxn = reinterpret_cast<const int32_t*>(smem + y.offMaxN);
    t.L = y.L;
    const int L = y.L;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    WarpArea& wa = reinterpret_cast<WarpArea*>(smem + ((y.bytes + 127u) & ~127u))[warp];

    unsigned long long checks = 0, probes = 0, priced = 0;
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    for (int64_t p = (int64_t)blockIdx.x * kWarps + warp; p < count; p += nwarps) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        const bool memok = a.wl_memok[p] != 0;
        if (kCount && lane == 0) ++priced;
        // this lane's stage (lane < S)
        const bool live = lane < S;
        const int code = a.wl_code[p * kMaxStages + lane];
        const int nxt = __shfl_down_sync(kFull, code, 1);
        const int g = code & 7, j = (code >> 3) & 3;
        WStage mine;
        mine.row = (g * 4 + j) * (L + 1);
        mine.capk = t.mem[g] << j;
        mine.f = live ? min(S - lane, M) : 0;
        mine.c = 0;
        if (lane + 1 < S) {
            const int h = nxt & 7, jn = (nxt >> 3) & 3;
            const int same = (g == h) && ((1 << j) + (1 << jn) <= t.maxn[g]);
            mine.c = t.p2p[(g * 8 + h) * 2 + same];
        }
        // a bound feasible whenever memory is, and the balanced guess
        int64_t hi = 0;
        float inv = 0.f, cw = 0.f;
        if (live) {
            const int64_t all = t.P[mine.row + L];
            hi = all + mine.c;
            const float tot = u64_to_float((uint64_t)all) + 1.0f;
            inv = 1.0f / tot;
            cw = u64_to_float((uint64_t)mine.c) / tot;
        }
        hi = wmax64(hi);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            inv += __shfl_xor_sync(kFull, inv, o);
            cw += __shfl_xor_sync(kFull, cw, o);
        }
        int64_t shi, slo;
        if (!memok) {
            // memory-only probe decides OOM and gives a tighter upper bound
            if (kCount && lane == 0) ++probes;
            if (!wprobe(t, mine, S, kInf, wa, shi, slo, checks)) {
                if (lane == 0) {
                    a.T[c] = -1;
                    a.B[c] = -1;
                    a.ndp[c] = (uint16_t)n;
                    a.status[c] = HEDDLE_CAND_OOM;
                    a.wl_T[p] = -1;
                }
                if (a.bounds) {
                    a.bounds[(int64_t)(lane + 1) * a.bstride + c] = 0;
                    if (lane == 0) a.bounds[c] = 0;
                }
                continue;
            }
            hi = shi;
        }
        // ---- PartitionLayers: threshold search from the balanced guess
        int64_t lo = 0;
        bool lo_known = false, hi_known = false;
        int64_t B = (int64_t)float_to_u64((1.0f + cw) / inv);
        int64_t step = max((int64_t)1, (int64_t)float_to_u64(u64_to_float(B) * (float)S / (2.0f * (float)L)));
        int it = 0;
        while (lo < hi) {
            B = min(max(B, lo), hi - 1);
            if (kCount && lane == 0) ++probes;
            if (wprobe(t, mine, S, B, wa, shi, slo, checks)) {
                hi = shi;
                hi_known = true;
            } else {
                lo = slo;
                lo_known = true;
            }
            if (lo >= hi) break;
            if (!lo_known) {
                B = hi - step;
                step *= 2;
            } else if (!hi_known) {
                B = lo + step;
                step *= 2;
            } else {
                B = lo + (hi - lo) / 2;
            }
            if (++it > kMaxIters) {
                if (lane == 0) atomicOr(a.err, kErrSearchBound);
                break;
            }
        }
        const int64_t Bstar = hi;
        // the sets of the optimum give the canonical split
        if (kCount && lane == 0) ++probes;
        if (!wprobe(t, mine, S, Bstar, wa, shi, slo, checks) && lane == 0) atomicOr(a.err, kErrInternal);
        if (lane == 0) {
            int at = 0;
            wa.A[0] = 0;
            for (int s = 0; s + 1 < S; ++s) {
                const int x = next_above(wa.C[s + 1], at, L);
                if (x < 0) atomicOr(a.err, kErrInternal);
                at = max(x, at + 1);
                wa.A[s + 1] = (uint8_t)at;
            }
            wa.A[S] = (uint8_t)L;
        }
        __syncwarp();
        // ---- Evaluate: T = (M-1) max t_s + sum t_s + max g_s, lane per stage
        int64_t ts = 0;
        uint64_t G = 0, D = 1;
        int a0 = 0, a1 = 0;
        if (live) {
            a0 = wa.A[lane];
            a1 = wa.A[lane + 1];
            ts = t.P[mine.row + a1] - t.P[mine.row + a0] + mine.c;
            G = (uint64_t)(t.PB[a1] - t.PB[a0]);
            D = (uint64_t)t.inter[g] << j;
        }
        const int64_t tmax = wmax64(ts);
        int64_t tsum = ts;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) tsum += __shfl_xor_sync(kFull, tsum, o);
        // the stage with the largest G / (k bw), compared exactly
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const uint64_t G2 = __shfl_xor_sync(kFull, G, o), D2 = __shfl_xor_sync(kFull, D, o);
            if ((u128)G2 * D > (u128)G * D2) {
                G = G2;
                D = D2;
            }
        }
        if (lane == 0) {
            if (tmax != Bstar) atomicOr(a.err, kErrInternal);
            int64_t gmax = 0;
            if (n > 1) {
                // ring all-reduce over n replicas: ceil(2(n-1) G 1e9 / (n k bw))
                const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * G;
                bool okd = true;
                gmax = (int64_t)ceil_div_u128(num, (uint64_t)n * D, &okd);
                if (!okd) atomicOr(a.err, kErrInternal);
            }
            const int64_t T = (int64_t)(M - 1) * Bstar + tsum + gmax;
            a.T[c] = T;
            a.wl_T[p] = T;
            a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
            a.B[c] = Bstar;
            a.ndp[c] = (uint16_t)n;
            a.status[c] = HEDDLE_CAND_OK;
        }
        if (a.bounds) {
            a.bounds[(int64_t)(lane + 1) * a.bstride + c] = live ? (uint8_t)a1 : 0;
            if (lane == 0) a.bounds[c] = 0;
        }
        __syncwarp();  // wa is reused by the next entry
    }
    if (kCount) {
        unsigned long long v0 = checks, v1 = probes, v2 = priced;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            v0 += __shfl_down_sync(kFull, v0, o);
            v1 += __shfl_down_sync(kFull, v1, o);
            v2 += __shfl_down_sync(kFull, v2, o);
        }
        if (lane == 0) {
            atomicAdd(&a.counters[0], v0);
            atomicAdd(&a.counters[1], v1);
            atomicAdd(&a.counters[2], v2);
        }
    }
}

template <bool kCount>
cudaError_t launch(const PriceArgs& a, int num_sms, cudaStream_t st) {
    const size_t smem = ((a.lay.bytes + 127u) & ~127u) + sizeof(WarpArea) * kWarps;
    cudaError_t e = cudaFuncSetAttribute(wsearch_kernel<kCount>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, wsearch_kernel<kCount>, kWBlock, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: one warp per entry,
    // at most one wave
    const int64_t need = (a.n + kWarps - 1) / kWarps;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    wsearch_kernel<kCount><<<grid, kWBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_warp_search(const PriceArgs& a, int num_sms, cudaStream_t st) {
    return a.counters ? launch<true>(a, num_sms, st) : launch<false>(a, num_sms, st);
}

}  // namespace hd
