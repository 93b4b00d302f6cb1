// heddle_wsearch.cu -- general PartitionLayers + Evaluate (§3.1 listing,
// §5.2 memory validation, §5.3 iteration time) for models whose layers
// differ, one warp per worklist entry.
//
// The exact threshold search: a memory-only probe decides OOM (unless the
// screen already knows a split fits) and bounds B*; the first guess solves
// the saturating continuous balance of the equal-layer search with each
// stage's average layer cost and its memory run from layer 0 (a few Newton
// steps), then each probe snaps the bracket to the largest accepted or the
// smallest rejected stage time and the next bound gallops from that value
// (1, 2, 4, ... away) until both sides are known, then bisects.  The sets
// of the probe at B* give the canonical split; a feasible probe that closes
// the bracket already holds them (every bound in [hi, B] takes the same
// decisions), so only a bracket closed from below costs a final probe.
// The probe (heddle_wprobe.cuh) checks 32 positions per round with the
// interval test of this file: stage time
// P[j] - P[i] + c and memory against k times the GPU memory.  Evaluate runs
// one lane per stage: the stage times' maximum and sum, the stage with the
// largest G / (k bw) by exact cross-multiplication, and one 128/64-bit
// ceiling division for the gradient term.  The table image is staged into
// shared memory with bulk asynchronous copies.  The kernel prices the
// entries the thread-per-entry search (heddle_gsearch.cu) left, or every
// worklist entry when that search had too few to run; each warp takes its
// own first entry, then the next untaken one from a counter.

#include <climits>

#include "heddle_wprobe.cuh"

namespace hd {
namespace {

using wp::kFull;
using wp::WarpArea;

constexpr int kWBlock = 256;
constexpr int kWarps = kWBlock / 32;
constexpr int kMaxIters = 256;

struct WTabs {
    const int64_t* qmax;  // [NT * 4] the most expensive single layer per (type, degree)
    int64_t smax, amax;   // the largest single-layer state and activation bytes
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

// The interval test of the general search: stage time P[j] - P[i] + c and
// memory (S[j] - S[i]) + f (A[j] - A[i]) against k times the GPU memory.
struct PlainCheck {
    typedef WStage Stage;
    const WTabs& t;
    WStage mine;  // the stage this lane holds
    __device__ WStage stage(int s) const {
        WStage r;
        r.row = __shfl_sync(kFull, mine.row, s);
        r.c = __shfl_sync(kFull, mine.c, s);
        r.capk = __shfl_sync(kFull, mine.capk, s);
        r.f = __shfl_sync(kFull, mine.f, s);
        return r;
    }
    __device__ __forceinline__ int eval(const WStage& st, int i, int j, int64_t B, int64_t* cost) const {
        const longlong2 si = t.SA[i], sj = t.SA[j];
        if ((sj.x - si.x) + st.f * (sj.y - si.y) > st.capk) return 2;
        const int64_t v = t.P[st.row + j] - t.P[st.row + i] + st.c;
        *cost = v;
        return v <= B ? 0 : 1;
    }
};

// The first guess of B* (warp-collective): each stage's average layer cost,
// P2P and memory run from layer 0 into the saturating balance; not
// inlined, so the probe loop around it keeps its registers.
__device__ __noinline__ int64_t plain_guess(const int64_t* P, const longlong2* SA, int row, int64_t c, int64_t capk,
                                            int64_t f, bool live, int S, int L, int64_t hi) {
    float rq = 0.f, cf = 0.f, mr = 0.f;
    if (live) {
        const int64_t all = P[row + L];
        rq = all > 0 ? (float)L / u64_to_float((uint64_t)all) : 0.f;
        cf = u64_to_float((uint64_t)c);
        int r0 = 0, r1 = L;  // the largest run [0, r) within memory
        while (r0 < r1) {
            const int mid = (r0 + r1 + 1) >> 1;
            const longlong2 sm = SA[mid];
            if ((sm.x - SA[0].x) + f * (sm.y - SA[0].y) <= capk) r0 = mid;
            else r1 = mid - 1;
        }
        mr = (float)r0;
    }
    return wp::first_guess(rq, cf, mr, S, L, hi);
}

// The entries of the list the thread-per-entry search left (a.sv_idx,
// count at wl_count[kWlGeneral]) -- or every worklist entry when the depth
// buckets hold fewer than thread_min entries (that search then ran none;
// thread_min is a.thread_min, or INT_MAX for the whole worklist).
template <bool kCount>
__global__ void __launch_bounds__(kWBlock, 3) wsearch_kernel(PriceArgs a, int thread_min) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ int64_t qmax[4 * kMaxTypes], single[2];
    if (!wp::load_image(smem, a.img, a.lay.bytes, &bar, a.err)) return;
    const Layout& y = a.lay;
    {
        // the most expensive single layer per (type, degree), and the
        // largest single-layer state and activation, for the forward-only
        // probe's condition
        const int64_t* P = reinterpret_cast<const int64_t*>(smem + y.offP);
        const longlong2* SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        for (int r = warp; r <= 4 * y.NT; r += kWarps) {
            int64_t m0 = 0, m1 = 0;
            for (int l = lane; l < y.L; l += 32) {
                if (r < 4 * y.NT) {
                    m0 = max(m0, P[r * (y.L + 1) + l + 1] - P[r * (y.L + 1) + l]);
                } else {
                    m0 = max(m0, (int64_t)(SA[l + 1].x - SA[l].x));
                    m1 = max(m1, (int64_t)(SA[l + 1].y - SA[l].y));
                }
            }
            m0 = wp::wmax64(m0);
            m1 = wp::wmax64(m1);
            if (lane == 0) {
                if (r < 4 * y.NT) {
                    qmax[r] = m0;
                } else {
                    single[0] = m0;
                    single[1] = m1;
                }
            }
        }
        __syncthreads();
    }
    WTabs t;
    t.qmax = qmax;
    t.smax = single[0];
    t.amax = single[1];
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
    int bucketed = a.wl_count[1 + 1 + lane];  // depth 1 + lane
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) bucketed += __shfl_xor_sync(kFull, bucketed, o);
    const bool listed = bucketed >= thread_min;
    const int64_t count = min((int64_t)(listed ? a.wl_count[kWlGeneral] : *a.wl_count), (int64_t)a.wl_cap);
    // each warp prices its own first entry, then the next untaken one
    // whenever it is free
    const int64_t first = (int64_t)gridDim.x * kWarps;
    auto take = [&]() {
        int e = 0;
        if (lane == 0) e = atomicAdd(a.wl_count + kWlTakeWarp, 1);
        return first + __shfl_sync(kFull, e, 0);
    };
    for (int64_t e = (int64_t)blockIdx.x * kWarps + warp; e < count; e = take()) {
        const int64_t p = listed ? a.sv_idx[e] : e;
        if (!in_range(p, a.wl_cap, a.err)) continue;
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        if (!in_range(c, a.n, a.err) || !in_range(S - 1, kMaxStages, a.err)) continue;
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
        // the forward-only probe is exact at bounds where every stage could
        // hold any single layer (time and memory)
        const int64_t qmc = live ? t.qmax[g * 4 + j] + mine.c : -1;
        const bool memfit = !live || t.smax + mine.f * t.amax <= mine.capk;
        // a bound feasible whenever memory is
        int64_t hi = live ? t.P[mine.row + L] + mine.c : 0;
        hi = wp::wmax64(hi);
        const PlainCheck check{t, mine};
        // one probe call site (the probe is large): phase 0 the memory-only
        // probe (OOM, else a tighter upper bound; skipped when the screen
        // knows a split fits), phase 1 the threshold search galloping from
        // the balanced guess, phase 2 the probe at B* whose sets give the
        // split
        int64_t lo = 0, B = kInf, step = 1;
        bool lo_known = false, hi_known = false, oom = false;
        int phase = memok ? 1 : 0, it = 0;
        if (memok) {
            B = min(max(plain_guess(t.P, t.SA, mine.row, mine.c, mine.capk, mine.f, live, S, L, hi), lo), hi - 1);
            if (lo >= hi) {
                phase = 2;
                B = hi;
            }
        }
        while (true) {
            int64_t shi, slo;
            if (kCount && lane == 0) ++probes;
            const bool fast = phase != 2 && __all_sync(kFull, qmc <= B && memfit);
            const bool feas = fast ? wp::forward_probe(check, S, L, B, shi, slo, checks)
                                   : wp::probe(check, S, L, B, wa, shi, slo, checks);
            if (phase == 0) {
                if (!feas) {
                    oom = true;
                    break;
                }
                hi = shi;
                B = plain_guess(t.P, t.SA, mine.row, mine.c, mine.capk, mine.f, live, S, L, hi);
                phase = 1;
            } else if (phase == 1) {
                if (feas) {
                    hi = shi;
                    hi_known = true;
                } else {
                    lo = slo;
                    lo_known = true;
                }
                if (!lo_known) {
                    B = hi - step;
                    step *= 2;
                } else if (!hi_known) {
                    B = lo + step - 1;
                    step *= 2;
                } else {
                    B = lo + (hi - lo) / 2;
                }
                if (++it > kMaxIters) {
                    if (lane == 0) atomicOr(a.err, kErrSearchBound);
                    lo = hi;
                }
                // closed by a feasible full probe: its sets are those of B* = hi
                if (lo >= hi && feas && !fast && it <= kMaxIters) break;
            } else {
                if (!feas && lane == 0) atomicOr(a.err, kErrInternal);
                break;
            }
            if (phase == 1 && lo >= hi) {
                phase = 2;
                B = hi;
            } else if (phase == 1) {
                B = min(max(B, lo), hi - 1);
            }
        }
        if (oom) {
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
        const int64_t Bstar = hi;
        if (!wp::walk(wa, S, L) && lane == 0) atomicOr(a.err, kErrInternal);
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
        const int64_t tmax = wp::wmax64(ts);
        const int64_t tsum = wp::wsum64(ts);
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
cudaError_t launch(const PriceArgs& a, int num_sms, cudaStream_t st, bool listed) {
    const size_t smem = ((a.lay.bytes + 127u) & ~127u) + sizeof(WarpArea) * kWarps;
    int per_sm = 0;
    const cudaError_t e = resident_blocks(reinterpret_cast<const void*>(&wsearch_kernel<kCount>), kWBlock, smem, &per_sm);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: one warp per entry,
    // at most one wave
    const int64_t need = (a.n + kWarps - 1) / kWarps;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    wsearch_kernel<kCount><<<grid, kWBlock, smem, st>>>(a, listed ? a.thread_min : INT_MAX);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_warp_search(const PriceArgs& a, int num_sms, cudaStream_t st, bool listed) {
    return a.counters ? launch<true>(a, num_sms, st, listed) : launch<false>(a, num_sms, st, listed);
}

}  // namespace hd
