// heddle_eqsearch.cu -- PartitionLayers + Evaluate for models whose layers
// all cost the same (§3.1 listing, §5.2 memory validation, §5.3 iteration
// time), over the worklist the screen kernel produced.
//
// When every layer has the same quantised cost q_s on a stage's (type,
// degree) and the same state and activation bytes, stage s holds exactly
//     cap_s(B) = min(m_s, floor((B - c_s) / q_s))
// layers within bound B (m_s: the longest run of layers that fits the
// stage's memory, c_s: its P2P).  A split with every stage time <= B exists
// iff every cap_s >= 1 and sum_s cap_s >= L, so a probe costs O(S).
// B* >= max_s (c_s + q_s) (every stage holds a layer), which starts the
// bracket; the first probe is the continuous balance
// sum_s (B - c_s) / q_s = L, later ones interpolate the cap count between
// the bracket's probes (a Newton step on the count while one side is
// missing), falling back to bisection.  Every probe snaps the bracket to
// exact breakpoints: a feasible probe keeps the same caps down to
// max_s (c_s + cap_s q_s), an infeasible one up to the smallest
// c_s + (cap_s + 1) q_s of a stage that can still grow, so the search ends
// on B* itself with the caps of its last feasible probe, which hold at B*.
// The componentwise smallest split -- hence the lexicographically smallest
// -- is then a_{s+1} = max(a_s + 1, L - sum_{t > s} cap_t).
//
// Layout: a few small tables (per-layer cost and its reciprocal per (type,
// degree), P2P, gradient-byte prefix, NIC, memory runs) are copied to shared
// memory once per CTA; every candidate's stages are packed once into 32-bit
// words (cost index | P2P index | memory run) held in shared memory
// interleaved by thread, so probes read one conflict-free word per stage.
// Each CTA takes 256 worklist entries at a time and sorts them by S
// (counting sort) so that the lanes of a warp run stage loops of equal
// length.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

typedef unsigned __int128 u128;

constexpr int kEqBlock = 256;
constexpr int kZeroP2P = 128;  // a zero entry after the 8 x 8 x 2 P2P table
constexpr int kMaxIters = 256;

struct EqLayout {
    uint32_t q, rq, p2p, inter, maxn, PB, win, sw, caps, bytes;
};

__host__ __device__ inline uint32_t al16(uint32_t x) { return (x + 15u) & ~15u; }

__host__ __device__ inline EqLayout eq_layout(int L) {
    EqLayout e;
    uint32_t o = 0;
    e.q = o;     o = al16(o + 8 * 32);             // int64 [j * 8 + g]
    e.rq = o;    o = al16(o + 4 * 32);             // float 1 / q
    e.p2p = o;   o = al16(o + 8 * 129);            // int64 [(g * 8 + h) * 2 + same], [128] = 0
    e.inter = o; o = al16(o + 8 * 8);              // int64 [g]
    e.maxn = o;  o = al16(o + 4 * 8);              // int32 [g]
    e.PB = o;    o = al16(o + 8 * (L + 1));        // int64 gradient-byte prefix
    e.win = o;   o = al16(o + 8 * 4 * 33);         // uint8 [(g * 4 + j) * 33 + f]
    e.sw = o;    o = al16(o + 4 * kMaxStages * kEqBlock);  // uint32 [s][thread]
    e.caps = o;  o = al16(o + 2 * (kMaxStages + 1) * kEqBlock);  // uint8 [2][s][thread]
    e.bytes = o;
    return e;
}

struct EqTabs {
    const int64_t* q;
    const float* rq;
    const int64_t* p2p;
    const int64_t* inter;
    const int32_t* maxn;
    const int64_t* PB;
    const uint8_t* win;
    uint32_t* sw;   // this thread's stage words, element s at [s * kEqBlock]
    uint8_t* caps;  // this thread's caps, two sets, set b element s at [(b * 33 + s) * kEqBlock]
    int L;
};

// Stage word: bits 0-4 cost index (the stage byte's type | degree bits),
// bits 5-12 P2P index, bits 13-20 memory run m.
__device__ __forceinline__ uint32_t stage_word(int code, int next, bool last, int f, const EqTabs& t) {
    const int g = code & 7, j = (code >> 3) & 3;
    int pidx = kZeroP2P;
    if (!last) {
        const int h = next & 7, jn = (next >> 3) & 3;
        const int same = (g == h) && ((1 << j) + (1 << jn) <= t.maxn[g]);
        pidx = (g * 8 + h) * 2 + same;
    }
    const int m = t.win[(g * 4 + j) * 33 + f];
    return (uint32_t)(code & 31) | ((uint32_t)pidx << 5) | ((uint32_t)m << 13);
}

struct Cap {
    int k;          // layers held within B (-1: not even one)
    int64_t q, c;
    int m;
};

__device__ __forceinline__ Cap stage_cap(const EqTabs& t, uint32_t w, int64_t B) {
    Cap r;
    r.q = t.q[w & 31];
    r.c = t.p2p[(w >> 5) & 255];
    r.m = (int)(w >> 13) & 255;
    if (B < r.c + r.q || r.m < 1) {
        r.k = -1;
        return r;
    }
    const int64_t x = B - r.c;
    if (r.q == 0 || x >= (int64_t)r.m * r.q) {
        r.k = r.m;
        return r;
    }
    // x < m q with m <= 255: the float estimate is off by at most one
    int k = (int)((float)x * t.rq[w & 31]);
    if ((int64_t)k * r.q > x) --k;
    if ((int64_t)(k + 1) * r.q <= x) ++k;
    r.k = k;
    return r;
}

struct Snap {
    int64_t hi, lo;  // snapping values
    int tot;         // layers the stages hold (stages holding one or more)
    float slope;     // growth of tot per unit of B: sum of 1/q over stages below their run
    unsigned long long units;
};

// Probe bound B; the caps go to cap set `set`.
__device__ bool eq_probe(const EqTabs& t, int S, int64_t B, int set, Snap& sn) {
    sn.hi = -1;
    sn.lo = kInf;
    sn.slope = 0.f;
    int sum = 0;
    bool ok = true;
    uint8_t* caps = t.caps + set * (kMaxStages + 1) * kEqBlock;
    for (int s = 0; s < S; ++s) {
        const uint32_t w = t.sw[s * kEqBlock];
        const Cap r = stage_cap(t, w, B);
        caps[s * kEqBlock] = (uint8_t)max(r.k, 0);
        if (r.k < r.m) sn.slope += t.rq[w & 31];
        if (r.k < 1) {
            ok = false;
            if (r.m >= 1) sn.lo = min(sn.lo, r.c + r.q);
            continue;
        }
        sum += r.k;
        sn.hi = max(sn.hi, r.c + (int64_t)r.k * r.q);
        if (r.k < r.m) sn.lo = min(sn.lo, r.c + (int64_t)(r.k + 1) * r.q);
    }
    sn.units += S;
    sn.tot = sum;
    return ok && sum >= t.L;
}

template <bool kCount>
__global__ void __launch_bounds__(kEqBlock) eq_search_kernel(PriceArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int bins[kMaxStages + 2];
    __shared__ uint16_t order[kEqBlock];
    const Layout& y = a.lay;
    const int L = y.L;
    const EqLayout el = eq_layout(L);
    // small tables, copied once per CTA
    {
        int64_t* q = reinterpret_cast<int64_t*>(smem + el.q);
        float* rq = reinterpret_cast<float*>(smem + el.rq);
        int64_t* p2p = reinterpret_cast<int64_t*>(smem + el.p2p);
        int64_t* inter = reinterpret_cast<int64_t*>(smem + el.inter);
        int32_t* maxn = reinterpret_cast<int32_t*>(smem + el.maxn);
        int64_t* PB = reinterpret_cast<int64_t*>(smem + el.PB);
        uint8_t* win = smem + el.win;
        const int64_t* gP = reinterpret_cast<const int64_t*>(a.img + y.offP);
        for (int i = threadIdx.x; i < 32; i += blockDim.x) {
            const int g = i & 7, j = i >> 3;
            const int64_t v = g < y.NT ? gP[(g * 4 + j) * (L + 1) + 1] - gP[(g * 4 + j) * (L + 1)] : 0;
            q[i] = v;
            rq[i] = v > 0 ? 1.0f / (float)v : 0.0f;
        }
        for (int i = threadIdx.x; i < 129; i += blockDim.x)
            p2p[i] = i < 128 ? reinterpret_cast<const int64_t*>(a.img + y.offP2P)[i] : 0;
        for (int i = threadIdx.x; i < 8; i += blockDim.x) {
            inter[i] = reinterpret_cast<const int64_t*>(a.img + y.offInter)[i];
            maxn[i] = reinterpret_cast<const int32_t*>(a.img + y.offMaxN)[i];
        }
        for (int i = threadIdx.x; i <= L; i += blockDim.x)
            PB[i] = reinterpret_cast<const int64_t*>(a.img + y.offPB)[i];
        for (int i = threadIdx.x; i < 8 * 4 * 33; i += blockDim.x) win[i] = a.img[y.offWin + i];
    }
    __syncthreads();
    EqTabs t;
    t.q = reinterpret_cast<const int64_t*>(smem + el.q);
    t.rq = reinterpret_cast<const float*>(smem + el.rq);
    t.p2p = reinterpret_cast<const int64_t*>(smem + el.p2p);
    t.inter = reinterpret_cast<const int64_t*>(smem + el.inter);
    t.maxn = reinterpret_cast<const int32_t*>(smem + el.maxn);
    t.PB = reinterpret_cast<const int64_t*>(smem + el.PB);
    t.win = smem + el.win;
    t.sw = reinterpret_cast<uint32_t*>(smem + el.sw) + threadIdx.x;
    t.caps = smem + el.caps + threadIdx.x;
    t.L = L;

    Snap sn;
    sn.units = 0;
    unsigned long long probes = 0, searched = 0;
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t count_r = (count + kEqBlock - 1) / kEqBlock * kEqBlock;
    const int64_t stride = (int64_t)gridDim.x * kEqBlock;
    for (int64_t base = (int64_t)blockIdx.x * kEqBlock; base < count_r; base += stride) {
        // ---- this CTA's 256 entries, counting-sorted by S (0: no entry)
        const int64_t p0 = base + threadIdx.x;
        const int s0 = p0 < count ? a.wl_S[p0] : 0;
        if (threadIdx.x < kMaxStages + 2) bins[threadIdx.x] = 0;
        __syncthreads();
        atomicAdd(&bins[s0], 1);
        __syncthreads();
        if (threadIdx.x == 0) {
            int run = 0;
            for (int b = 0; b <= kMaxStages; ++b) {
                const int v = bins[b];
                bins[b] = run;
                run += v;
            }
        }
        __syncthreads();
        order[atomicAdd(&bins[s0], 1)] = (uint16_t)threadIdx.x;
        __syncthreads();
        const int64_t p = base + order[threadIdx.x];
        __syncthreads();  // bins and order are reused by the next slice
        if (p >= count) continue;

        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        if (kCount) ++searched;
        // pack the stages; feasible upper bound (every stage at its memory
        // run, which the screen guarantees covers L), lower bound (every
        // stage holds one layer) and the continuous balance as first probe
        int64_t hi = 0, lo = 0;
        float inv = 0.f, cw = 0.f;
        int code = a.wl_code[p];
        for (int s = 0; s < S; ++s) {
            const bool last = s + 1 == S;
            const int next = last ? 0 : a.wl_code[(int64_t)(s + 1) * a.wl_cap + p];
            const uint32_t w = stage_word(code, next, last, min(S - s, M), t);
            t.sw[s * kEqBlock] = w;
            const int64_t q = t.q[w & 31], cc = t.p2p[(w >> 5) & 255];
            const int m = (int)(w >> 13) & 255;
            hi = max(hi, cc + (int64_t)m * q);
            lo = max(lo, cc + q);
            const float qf = (float)q + 0.5f;
            inv += 1.0f / qf;
            cw += (float)cc / qf;
            code = next;
        }
        int64_t B = (int64_t)(((float)L + cw) / inv);
        // bracket probes (bound, cap count) for the interpolation
        int64_t Blo = -1, Bhi = -1;
        int clo = 0, chi = 0;
        int wset = 0, fset = -1;  // cap set written next / of the last feasible probe
        int it = 0;
        while (lo < hi) {
            B = min(max(B, lo), hi - 1);
            if (kCount) ++probes;
            const bool feas = eq_probe(t, S, B, wset, sn);
            if (feas) {
                hi = sn.hi;
                Bhi = B;
                chi = sn.tot;
                fset = wset;
                wset ^= 1;
            } else {
                lo = max(lo, sn.lo);
                Blo = B;
                clo = sn.tot;
            }
            if (lo >= hi) break;
            // next bound: interpolate the cap count between the bracket's
            // probes, else a Newton step, else bisect
            float target;
            if (Blo >= 0 && Bhi >= 0 && chi > clo) {
                target = (float)Blo + ((float)L - 0.5f - (float)clo) / (float)(chi - clo) * (float)(Bhi - Blo);
            } else if (sn.slope > 0.f) {
                target = feas ? (float)B - ceilf(((float)sn.tot - (float)L + 0.5f) / sn.slope)
                              : (float)B + ceilf(((float)L - (float)sn.tot) / sn.slope);
            } else {
                target = -1.f;
            }
            B = (target >= (float)lo && target <= (float)(hi - 1)) ? (int64_t)target : lo + (hi - lo) / 2;
            if (++it > kMaxIters) {
                atomicOr(a.err, kErrSearchBound);
                break;
            }
        }
        const int64_t Bstar = hi;
        if (fset < 0) {
            // B* is the initial bound, never probed: its caps
            if (kCount) ++probes;
            if (!eq_probe(t, S, Bstar, 0, sn)) atomicOr(a.err, kErrInternal);
            fset = 0;
        }
        const uint8_t* caps = t.caps + fset * (kMaxStages + 1) * kEqBlock;
        int total = 0;
        for (int s = 0; s < S; ++s) total += caps[s * kEqBlock];
        // ---- the smallest boundaries, then Evaluate:
        //      T = (M-1) max t_s + sum t_s + max g_s, stage by stage
        int64_t tmax = 0, tsum = 0;
        int sg = -1;
        u128 bestG = 0, bestD = 1;
        int pre = 0, at = 0;
        uint8_t bnd[kMaxStages + 1];
        bnd[0] = 0;
        for (int s = 0; s < S; ++s) {
            const uint32_t w = t.sw[s * kEqBlock];
            const int k = caps[s * kEqBlock];
            if (k < 1) atomicOr(a.err, kErrInternal);
            pre += k;
            const int nxt = s + 1 == S ? L : max(at + 1, L - (total - pre));
            bnd[s + 1] = (uint8_t)nxt;
            const int64_t ts = (int64_t)(nxt - at) * t.q[w & 31] + t.p2p[(w >> 5) & 255];
            tmax = max(tmax, ts);
            tsum += ts;
            if (n > 1) {
                // stage with the largest G_s / (k_s bw_s), compared exactly
                const int g = w & 7, j = (w >> 3) & 3;
                const u128 G = (u128)(t.PB[nxt] - t.PB[at]);
                const u128 D = (u128)t.inter[g] << j;
                if (sg < 0 || G * bestD > bestG * D) {
                    sg = s;
                    bestG = G;
                    bestD = D;
                }
            }
            at = nxt;
        }
        if (tmax != Bstar) atomicOr(a.err, kErrInternal);
        int64_t gmax = 0;
        if (n > 1) {
            // ring all-reduce over n replicas: ceil(2(n-1) G 1e9 / (n k bw))
            const u128 num = (u128)2 * (u128)(n - 1) * bestG * 1000000000u;
            const u128 den = (u128)n * bestD;
            gmax = (int64_t)((num + den - 1) / den);
        }
        a.T[c] = (int64_t)(M - 1) * Bstar + tsum + gmax;
        a.wl_T[p] = a.T[c];
        a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
        a.B[c] = Bstar;
        a.ndp[c] = (uint16_t)n;
        a.status[c] = HEDDLE_CAND_OK;
        if (a.bounds) {
            for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = s <= S ? bnd[s] : 0;
        }
    }
    if (kCount) {
        unsigned long long v0 = sn.units, v1 = probes, v2 = searched;
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

template <bool kCount>
cudaError_t launch(const PriceArgs& a, int num_sms, cudaStream_t st) {
    const size_t smem = eq_layout(a.lay.L).bytes;
    cudaError_t e = cudaFuncSetAttribute(eq_search_kernel<kCount>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, eq_search_kernel<kCount>, kEqBlock, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: size for the batch
    const int64_t need = (a.n + kEqBlock - 1) / kEqBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    eq_search_kernel<kCount><<<grid, kEqBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_eq_search(const PriceArgs& a, int num_sms, cudaStream_t st) {
    return a.counters ? launch<true>(a, num_sms, st) : launch<false>(a, num_sms, st);
}

}  // namespace hd
