// heddle_gsearch.cu -- general PartitionLayers + Evaluate (§3.1 listing,
// §5.2 memory validation, §5.3 iteration time) for models whose layers
// differ, one thread per worklist entry, wherever every stage could hold any
// single layer of the model.
//
// Call a bound B "single-fit" when every stage could hold any one layer
// within B (its most expensive layer's time plus its P2P at most B) and
// within its memory (the largest single-layer state plus its in-flight
// count times the largest single-layer activation).  At a single-fit bound:
//   * the feasible ends after stage s form an interval [s, U_s]: an end up
//     to U_{s-1} + 1 is reached one layer after its predecessor, one beyond
//     only from U_{s-1} (the largest predecessor dominates); so a probe is
//     the forward chain U_{s+1} = the furthest end stage s reaches from U_s
//     (a binary search: stage time and memory grow with the end), feasible
//     iff the last stage fits [U_{S-1}, L);
//   * symmetrically the feasible starts of stages s .. S-1 form an interval
//     [V_s, L - (S - s)], with V_s = the smallest start from which stage s
//     reaches V_{s+1}; the lexicographically smallest optimal split is then
//     a_{s+1} = max(a_s + 1, V_{s+1}) (a_s >= V_s, so [a_s, V_{s+1}) costs
//     no more than [V_s, V_{s+1}), and a single layer always fits).
// The search itself is that of the warp kernel (heddle_wsearch.cu): a
// memory-only probe where the screen could not decide memory, the
// saturating balance as first guess, each probe snapping the bracket to its
// largest accepted or smallest rejected stage time (every bound in [hi, B]
// or [B, lo) decides alike), galloping, then bisecting.  An entry that meets
// a bound that is not single-fit is left to the warp kernel, which runs the
// general set-based probe; it gets the list of those entries.  The kernel
// runs only when the depth buckets hold at least PriceArgs::thread_min
// entries (a few entries would leave it as long as its longest serial
// chain); each warp takes 32 entries at a time, deepest first.

#include <algorithm>

#include "heddle_wprobe.cuh"

namespace hd {
namespace {

constexpr int kGBlock = 128;
constexpr int kGWarps = kGBlock / 32;
constexpr int kGMaxIters = 256;
constexpr int kGZeroP2P = 128;  // index of a zero after the 8 x 8 x 2 P2P table

struct GTabs {
    const int64_t* P;      // [NT][4][L+1] prefix ns per (type, degree)
    const longlong2* SA;   // [L+1] prefix of (state bytes, activation bytes)
    const int64_t* PB;     // [L+1] prefix of gradient bytes
    const int64_t* p2p;    // [8][8][2] (index 128: no next stage, P2P 0)
    const int64_t* mem;    // [8]
    const int64_t* inter;  // [8]
    const int64_t* qmax;   // [NT * 4] the most expensive single layer
    const float* rqavg;    // [NT * 4] 1 / the average layer time
    int64_t smax, amax;    // the largest single-layer state and activation
    float avs, ava;        // the average layer state and activation bytes
    int L;
};

// Stage word (per thread, in shared memory): bits 0-4 the stage byte's type
// and degree, bits 5-12 the P2P index, bits 13-18 the in-flight count f,
// bits 19-26 V_s during the split.
constexpr int kVShift = 19;
constexpr uint32_t kNoV = (1u << kVShift) - 1;

struct GStage {
    int row;       // offset of the prefix row
    int64_t c;     // P2P to the next stage
    int64_t capk;  // memory per GPU x devices
    int64_t f;     // in-flight micro-batches
};

__device__ __forceinline__ GStage unpack(uint32_t w, const GTabs& t) {
    GStage st;
    const int g = w & 7, j = (w >> 3) & 3;
    st.row = (g * 4 + j) * (t.L + 1);
    const int pidx = (w >> 5) & 255;
    st.c = pidx < kGZeroP2P ? t.p2p[pidx] : 0;  // the image's table has 128 entries
    st.capk = t.mem[g] << j;
    st.f = (w >> 13) & 63;
    return st;
}

// Stage s holding layers [i, j): fits memory?  Its time in *cost.
__device__ __forceinline__ bool fits_mem(const GTabs& t, const GStage& st, int i, int j) {
    const longlong2 si = t.SA[i], sj = t.SA[j];
    return (int64_t)(sj.x - si.x) + st.f * (int64_t)(sj.y - si.y) <= st.capk;
}
__device__ __forceinline__ int64_t cost(const GTabs& t, const GStage& st, int i, int j) {
    return t.P[st.row + j] - t.P[st.row + i] + st.c;
}

// The largest x in [lo, hi] with ok(x), for a test that holds up to some
// point and fails beyond it (ok(lo) taken as true), searched from an
// estimate x0: gallop away from x0 (1, 2, 4, ... positions) until the
// boundary is bracketed, then bisect.  With a good estimate -- the prefix
// sums are nearly linear, exactly so for equal layers -- that is two tests
// instead of a bisection's eight.
template <class F>
__device__ __forceinline__ int last_ok(int lo, int hi, int x0, F ok) {
    x0 = min(max(x0, lo), hi);
    int a, b;
    if (x0 == lo || ok(x0)) {
        int good = x0, step = 1;
        b = hi;
        while (true) {
            const int k = good + step;
            if (k > hi) break;
            if (!ok(k)) {
                b = k - 1;
                break;
            }
            good = k;
            step <<= 1;
        }
        a = good;
    } else {
        int fail = x0, step = 1;
        a = lo;
        while (true) {
            const int k = fail - step;
            if (k <= lo) break;
            if (ok(k)) {
                a = k;
                break;
            }
            fail = k;
            step <<= 1;
        }
        b = fail - 1;
    }
    while (a < b) {
        const int mid = (a + b + 1) >> 1;
        if (ok(mid)) a = mid;
        else b = mid - 1;
    }
    return a;
}

// Layers of stage st that a bound B and its memory admit, estimated from
// the average layer time and footprint (for the searches' first guesses).
__device__ __forceinline__ float layers_est(const GTabs& t, const GStage& st, int row_idx, int64_t room) {
    const float by_time = room > 0 ? u64_to_float((uint64_t)room) * t.rqavg[row_idx] : 0.f;
    const float by_mem = u64_to_float((uint64_t)st.capk) / fmaxf(t.avs + (float)st.f * t.ava, 1.f);
    return fminf(fminf(by_time, by_mem), (float)t.L);
}

// The furthest end j in (u, lim] of a stage starting at u within B and its
// memory (u if none).  acc: the stage time at that end (-1 if none); rej:
// the stage time at the next end if memory admits it there and its time is
// above B (kInf otherwise).  checks counts the interval tests.
__device__ __forceinline__ int reach_of(const GTabs& t, const GStage& st, int row_idx, int u, int lim, int64_t B,
                                        int64_t& acc, int64_t& rej, unsigned long long& checks) {
    const int x0 = u + (int)layers_est(t, st, row_idx, B - st.c);
    const int lo = last_ok(u, lim, x0, [&](int j) {
        ++checks;
        return cost(t, st, u, j) <= B && fits_mem(t, st, u, j);
    });
    acc = lo > u ? cost(t, st, u, lo) : -1;
    rej = kInf;
    if (lo < lim && fits_mem(t, st, u, lo + 1)) {
        const int64_t v = cost(t, st, u, lo + 1);
        if (v > B) rej = v;
    }
    return lo;
}

// Exact probe of a single-fit bound B: the forward chain.  hi / lo: the
// snap values (the largest stage time of the chain; the smallest stage time
// that rejected an end).
__device__ bool gprobe(const GTabs& t, const uint32_t* sw, int S, int64_t B, int64_t& hi, int64_t& lo,
                       unsigned long long& checks) {
    const int L = t.L;
    hi = -1;
    lo = kInf;
    int u = 0;
    for (int s = 0; s + 1 < S; ++s) {
        const uint32_t w = sw[s * kGBlock];
        const GStage st = unpack(w, t);
        int64_t acc, rej;
        const int r = reach_of(t, st, (w & 7) * 4 + ((w >> 3) & 3), u, L - (S - 1 - s), B, acc, rej, checks);
        lo = min(lo, rej);
        if (r < s + 1) return false;
        hi = max(hi, acc);
        u = r;
    }
    const GStage st = unpack(sw[(S - 1) * kGBlock], t);
    ++checks;
    if (!fits_mem(t, st, u, L)) return false;
    const int64_t v = cost(t, st, u, L);
    if (v > B) {
        lo = min(lo, v);
        return false;
    }
    hi = max(hi, v);
    return true;
}

// Appends entry p to the list the warp kernel finishes.
__device__ __forceinline__ void defer(const PriceArgs& a, int64_t p) {
    const int pos = atomicAdd(a.wl_count + kWlGeneral, 1);
    if (in_range(pos, a.wl_cap, a.err)) a.sv_idx[pos] = (int32_t)p;
}

// Below a.thread_min bucketed entries the kernel returns at once and the
// warp kernel prices the whole worklist.  Four CTAs per SM (the table
// image and the stage words fill shared memory there), so up to 128
// registers a thread.
template <bool kCount>
__global__ void __launch_bounds__(kGBlock, 4) gsearch_kernel(PriceArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ int64_t qmax[4 * kMaxTypes], single[2];
    __shared__ float rqavg[4 * kMaxTypes], cfl[129];
    __shared__ int end_of[kMaxStages + 2];
    const Layout& y = a.lay;
    const int L = y.L;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x < 32) {
        // end_of[S] = entries of depths >= S (see eq_search_kernel)
        int x = a.wl_count[1 + (kMaxStages - lane)];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y2 = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y2;
        }
        end_of[kMaxStages - lane] = x;
        if (lane == 0) end_of[kMaxStages + 1] = 0;
    }
    __syncthreads();
    if (end_of[1] < a.thread_min) return;
    if (!wp::load_image(smem, a.img, y.bytes, &bar, a.err)) return;
    {
        const int64_t* P = reinterpret_cast<const int64_t*>(smem + y.offP);
        const longlong2* SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
        // per (type, degree) the most expensive single layer and 1 / the
        // average layer time; the largest single-layer state and activation
        for (int r = warp; r <= 4 * y.NT; r += kGWarps) {
            int64_t m0 = 0, m1 = 0;
            for (int l = lane; l < L; l += 32) {
                if (r < 4 * y.NT) {
                    m0 = max(m0, P[r * (L + 1) + l + 1] - P[r * (L + 1) + l]);
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
                    const int64_t all = P[r * (L + 1) + L];
                    rqavg[r] = all > 0 ? (float)L / u64_to_float((uint64_t)all) : 0.f;
                } else {
                    single[0] = m0;
                    single[1] = m1;
                }
            }
        }
        const int64_t* p2p = reinterpret_cast<const int64_t*>(smem + y.offP2P);
        for (int i = threadIdx.x; i < 129; i += blockDim.x) cfl[i] = i < 128 ? u64_to_float((uint64_t)p2p[i]) : 0.f;
        __syncthreads();
    }
    GTabs t;
    t.P = reinterpret_cast<const int64_t*>(smem + y.offP);
    t.SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
    t.PB = reinterpret_cast<const int64_t*>(smem + y.offPB);
    t.p2p = reinterpret_cast<const int64_t*>(smem + y.offP2P);
    t.mem = reinterpret_cast<const int64_t*>(smem + y.offMem);
    t.inter = reinterpret_cast<const int64_t*>(smem + y.offInter);
    t.qmax = qmax;
    t.rqavg = rqavg;
    t.smax = single[0];
    t.amax = single[1];
    {
        const longlong2 all = t.SA[L];
        t.avs = u64_to_float((uint64_t)all.x) / (float)L;
        t.ava = u64_to_float((uint64_t)all.y) / (float)L;
    }
    t.L = L;
    const int32_t* maxn = reinterpret_cast<const int32_t*>(smem + y.offMaxN);
    const int64_t* minq = reinterpret_cast<const int64_t*>(smem + y.offMinQ);
    uint32_t* sw = reinterpret_cast<uint32_t*>(smem + ((y.bytes + 127u) & ~127u)) + threadIdx.x;

    unsigned long long checks = 0, probes = 0, priced = 0;
    // the entries filed in the depth buckets (the screen lists the others
    // for the warp kernel directly)
    const int64_t entries = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t count = min((int64_t)end_of[1], entries);
    // each warp prices 32 entries (deepest first): its own first, then the
    // next untaken ones whenever it is free
    const int64_t first = (int64_t)gridDim.x * kGBlock;
    auto take = [&]() {
        int b = 0;
        if (lane == 0) b = atomicAdd(a.wl_count + kWlTakeThread, 32);
        return first + __shfl_sync(0xffffffffu, b, 0);
    };
    for (int64_t base = ((int64_t)blockIdx.x * kGWarps + warp) * 32; base < count; base = take()) {
        const int64_t g = base + lane;
        if (g >= count) continue;
        int lo_d = 1, hi_d = kMaxStages;
        while (lo_d < hi_d) {
            const int mid = (lo_d + hi_d + 1) >> 1;
            if (end_of[mid] > g) lo_d = mid; else hi_d = mid - 1;
        }
        const int64_t off = g - end_of[lo_d + 1];
        if (!in_range(off, end_of[lo_d] - end_of[lo_d + 1], a.err)) continue;
        const int64_t p = a.wl_bucket[(int64_t)(lo_d - 1) * a.wl_cap + off];
        if (!in_range(p, entries, a.err)) continue;
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p], M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        const bool memok = a.wl_memok[p] != 0;
        if (!in_range(c, a.n, a.err) || !in_range(S - 1, kMaxStages, a.err)) continue;
        if (kCount) ++priced;
        // pack the stages; the single-fit threshold QC (no bound below it
        // is single-fit), the memory test, a bound feasible whenever
        // memory is, and each stage's memory run from layer 0 for the guess
        // (the entry's 32-byte row of stage bytes, read a byte per stage:
        // an array indexed by the stage would live in local memory)
        const uint8_t* row = a.wl_code + p * kMaxStages;
        int64_t QC = 0, hiB = 0, LB = 0;
        bool memall = true;
        int next = __ldg(row);
        for (int s = 0; s < S; ++s) {
            const int code = next;
            next = s + 1 < S ? __ldg(row + s + 1) : 0;
            const int gg = code & 7, jj = (code >> 3) & 3;
            int pidx = kGZeroP2P;
            if (s + 1 < S) {
                const int h = next & 7, jn = (next >> 3) & 3;
                pidx = (gg * 8 + h) * 2 + ((gg == h) && ((1 << jj) + (1 << jn) <= maxn[gg]));
            }
            const int f = min(S - s, M);
            uint32_t w = (uint32_t)(code & 31) | ((uint32_t)pidx << 5) | ((uint32_t)f << 13);
            const GStage st = unpack(w, t);
            QC = max(QC, t.qmax[gg * 4 + jj] + st.c);
            LB = max(LB, minq[gg * 4 + jj] + st.c);
            hiB = max(hiB, t.P[st.row + L] + st.c);
            memall &= t.smax + st.f * t.amax <= st.capk;
            // the run of layers memory admits, estimated from the average
            // layer footprint (for the guess only)
            const int r0 = min(L, (int)layers_est(t, st, gg * 4 + jj, kInf));
            w |= (uint32_t)r0 << kVShift;
            sw[s * kGBlock] = w;
        }
        if (!memall) {
            defer(a, p);
            continue;
        }
        int64_t shi, slo;
        if (!memok) {
            // memory only: OOM, else a tighter feasible bound
            ++probes;
            if (!gprobe(t, sw, S, kInf, shi, slo, checks)) {
                a.T[c] = -1;
                a.B[c] = -1;
                a.ndp[c] = (uint16_t)n;
                a.status[c] = HEDDLE_CAND_OOM;
                a.wl_T[p] = -1;
                if (a.bounds)
                    for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = 0;
                continue;
            }
            hiB = shi;
        }
        // first guess: the saturating continuous balance with each stage's
        // average layer time and memory run from layer 0
        int64_t B;
        {
            float inv = 0.f, cw = 0.f, flo = 0.f;
            for (int s = 0; s < S; ++s) {
                const uint32_t w = sw[s * kGBlock];
                const float rq = rqavg[(w & 7) * 4 + ((w >> 3) & 3)], cf = cfl[(w >> 5) & 255];
                inv += rq;
                cw += cf * rq;
                if (rq > 0.f) flo = fmaxf(flo, cf + 1.0f / rq);
            }
            const float fhi = u64_to_float((uint64_t)hiB);
            float Bf = fmaxf(flo, inv > 0.f ? ((float)L + 0.5f * (float)S + cw) / inv : flo);
            for (int it = 0; it < 3; ++it) {
                Bf = fminf(Bf, fhi);
                float cnt = 0.f, sl = 0.f, nb = 0.f;
                for (int s = 0; s < S; ++s) {
                    const uint32_t w = sw[s * kGBlock];
                    const float rq = rqavg[(w & 7) * 4 + ((w >> 3) & 3)], cf = cfl[(w >> 5) & 255];
                    const float mr = (float)((w >> kVShift) & 255);
                    const float x = (Bf - cf) * rq;
                    if (rq <= 0.f || x >= mr) {
                        cnt += mr;
                    } else {
                        cnt += x;
                        sl += rq;
                        nb += 1.f;
                    }
                }
                const float tgt = (float)L + 0.5f * nb;
                if (cnt >= tgt - 0.25f || sl <= 0.f) break;
                Bf += (tgt - cnt) / sl;
            }
            B = (int64_t)float_to_u64(fmaxf(fminf(Bf, fhi), 0.f));
        }
        // the threshold search on single-fit bounds (heddle_wsearch.cu's
        // bracketing) from the lower bound LB (every stage holds at least
        // its cheapest layer); a bracket entirely below QC goes to the warp
        // kernel (with equal layers LB = QC, so that never happens)
        int64_t lo = LB, hi = hiB, step = 1;
        bool lo_known = false, hi_known = false, deferred = false;
        int it = 0;
        B = min(max(B, lo), hi - 1);
        while (lo < hi) {
            if (B < QC) {
                // the bracket reaches below the single-fit threshold: probe
                // QC itself while it is inside, else leave the entry
                if (QC >= hi) {
                    deferred = true;
                    break;
                }
                B = QC;
            }
            ++probes;
            if (gprobe(t, sw, S, B, shi, slo, checks)) {
                hi = shi;
                hi_known = true;
            } else {
                lo = min(slo, hi);
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
            if (++it > kGMaxIters) {
                atomicOr(a.err, kErrSearchBound);
                lo = hi;
            }
            B = min(max(B, lo), hi - 1);
        }
        const int64_t Bstar = hi;
        if (deferred || Bstar < QC) {
            defer(a, p);
            continue;
        }
        // the split: V_s, the smallest start from which stage s reaches
        // V_{s+1} (V_S = L), into bits 19-26 of the stage words; then
        // a_{s+1} = max(a_s + 1, V_{s+1})
        {
            int v = L;
            for (int s = S - 1; s >= 1; --s) {
                const uint32_t w = sw[s * kGBlock];
                const GStage st = unpack(w, t);
                // the most layers y + 1 ending at v that stage s holds
                // within B* (v - 1 holds a single layer), from the estimate
                const int vv = v;
                const int y0 = (int)layers_est(t, st, (w & 7) * 4 + ((w >> 3) & 3), Bstar - st.c) - 1;
                const int y = last_ok(0, vv - 1 - s, y0, [&](int yy) {
                    ++checks;
                    return cost(t, st, vv - 1 - yy, vv) <= Bstar && fits_mem(t, st, vv - 1 - yy, vv);
                });
                v = vv - 1 - y;
                sw[s * kGBlock] = (w & kNoV) | ((uint32_t)v << kVShift);
            }
        }
        // Evaluate: T = (M-1) max t_s + sum t_s + max g_s
        int64_t tmax = 0, tsum = 0;
        uint64_t bestG = 0, bestD = 1;
        int at = 0;
        bool bad = false;
        for (int s = 0; s < S; ++s) {
            const uint32_t w = sw[s * kGBlock];
            const GStage st = unpack(w, t);
            const int nxt = s + 1 == S ? L : max(at + 1, (int)((sw[(s + 1) * kGBlock] >> kVShift) & 255));
            bad |= !fits_mem(t, st, at, nxt);
            if (a.bounds) a.bounds[(int64_t)(s + 1) * a.bstride + c] = (uint8_t)nxt;
            const int64_t ts = cost(t, st, at, nxt);
            tmax = max(tmax, ts);
            tsum += ts;
            if (n > 1) {
                const uint64_t G = (uint64_t)(t.PB[nxt] - t.PB[at]);
                const uint64_t D = (uint64_t)t.inter[w & 7] << ((w >> 3) & 3);
                if (s == 0 || (u128)G * bestD > (u128)bestG * D) {
                    bestG = G;
                    bestD = D;
                }
            }
            at = nxt;
        }
        if (a.bounds) {
            a.bounds[c] = 0;
            for (int s = S + 1; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = 0;
        }
        if (bad || tmax != Bstar) atomicOr(a.err, kErrInternal);
        int64_t gmax = 0;
        if (n > 1) {
            // ring all-reduce over n replicas: ceil(2(n-1) G 1e9 / (n k bw))
            const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * bestG;
            bool ok = true;
            gmax = (int64_t)ceil_div_u128(num, (uint64_t)n * bestD, &ok);
            if (!ok) atomicOr(a.err, kErrInternal);
        }
        const int64_t T = (int64_t)(M - 1) * Bstar + tsum + gmax;
        a.T[c] = T;
        a.wl_T[p] = T;
        a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
        a.B[c] = Bstar;
        a.ndp[c] = (uint16_t)n;
        a.status[c] = HEDDLE_CAND_OK;
    }
    if (kCount) {
        unsigned long long v0 = checks, v1 = probes, v2 = priced;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            v0 += __shfl_down_sync(0xffffffffu, v0, o);
            v1 += __shfl_down_sync(0xffffffffu, v1, o);
            v2 += __shfl_down_sync(0xffffffffu, v2, o);
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
    const size_t smem = ((a.lay.bytes + 127u) & ~127u) + sizeof(uint32_t) * kMaxStages * kGBlock;
    int per_sm = 0;
    const cudaError_t e = resident_blocks(reinterpret_cast<const void*>(&gsearch_kernel<kCount>), kGBlock, smem, &per_sm);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: one wave at most
    const int64_t need = (a.n + kGBlock - 1) / kGBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    gsearch_kernel<kCount><<<grid, kGBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_thread_search(const PriceArgs& a, int num_sms, cudaStream_t st) {
    return a.counters ? launch<true>(a, num_sms, st) : launch<false>(a, num_sms, st);
}

}  // namespace hd
