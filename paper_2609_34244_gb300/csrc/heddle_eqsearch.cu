// heddle_eqsearch.cu -- PartitionLayers + Evaluate for models whose layers
// all cost the same (§3.1 listing, §5.2 memory validation, §5.3 iteration
// time), over the worklist the screen kernel produced.
//
// When every layer has the same quantised cost q_s on a stage's (type,
// degree) and the same state and activation bytes, stage s holds exactly
//     cap_s(B) = min(m_s, floor((B - c_s) / q_s))
// layers within bound B (m_s: the longest run of layers that fits the
// stage's memory, c_s: its P2P).  A split with every stage time <= B exists
// iff every cap_s >= 1 and sum_s cap_s >= L, so a probe costs O(S).  The
// search snaps to exact breakpoints: a feasible probe keeps the same caps
// down to max_s (c_s + cap_s q_s), an infeasible one up to the smallest
// c_s + (cap_s + 1) q_s of a stage that can still grow; it starts from the
// continuous balance sum_s (B - c_s) / q_s = L and brackets by the largest q.
// At B* the componentwise smallest split -- hence the lexicographically
// smallest -- is a_{s+1} = max(a_s + 1, L - sum_{t > s} cap_t).
//
// Layout: a few small tables (per-layer cost per (type, degree), P2P,
// gradient-byte prefix, NIC, memory runs) are copied to shared memory once
// per CTA; every candidate's stages are packed once into 32-bit words
// (cost index | P2P index | memory run) held in shared memory interleaved by
// thread, so probes read one conflict-free word per stage.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

typedef unsigned __int128 u128;

constexpr int kEqBlock = 256;
constexpr int kZeroP2P = 128;  // a zero entry after the 8 x 8 x 2 P2P table
constexpr int kMaxIters = 256;

struct EqLayout {
    uint32_t q, p2p, inter, maxn, PB, win, sw, caps, bytes;
};

__host__ __device__ inline uint32_t al16(uint32_t x) { return (x + 15u) & ~15u; }

__host__ __device__ inline EqLayout eq_layout(int L) {
    EqLayout e;
    uint32_t o = 0;
    e.q = o;     o = al16(o + 8 * 32);             // int64 [j * 8 + g]
    e.p2p = o;   o = al16(o + 8 * 129);            // int64 [(g * 8 + h) * 2 + same], [128] = 0
    e.inter = o; o = al16(o + 8 * 8);              // int64 [g]
    e.maxn = o;  o = al16(o + 4 * 8);              // int32 [g]
    e.PB = o;    o = al16(o + 8 * (L + 1));        // int64 gradient-byte prefix
    e.win = o;   o = al16(o + 8 * 4 * 33);         // uint8 [(g * 4 + j) * 33 + f]
    e.sw = o;    o = al16(o + 4 * kMaxStages * kEqBlock);  // uint32 [s][thread]
    e.caps = o;  o = al16(o + (kMaxStages + 1) * kEqBlock); // uint8 [s][thread]
    e.bytes = o;
    return e;
}

struct EqTabs {
    const int64_t* q;
    const int64_t* p2p;
    const int64_t* inter;
    const int32_t* maxn;
    const int64_t* PB;
    const uint8_t* win;
    uint32_t* sw;   // this thread's stage words, element s at [s * kEqBlock]
    uint8_t* caps;  // this thread's caps, element s at [s * kEqBlock]
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
    int k = (int)((float)x / (float)r.q);
    if ((int64_t)k * r.q > x) --k;
    if ((int64_t)(k + 1) * r.q <= x) ++k;
    r.k = k;
    return r;
}

struct Snap {
    int64_t hi, lo;
    unsigned long long units;
};

__device__ bool eq_probe(const EqTabs& t, int S, int64_t B, Snap& sn) {
    sn.hi = -1;
    sn.lo = kInf;
    int sum = 0;
    bool ok = true;
    for (int s = 0; s < S; ++s) {
        const Cap r = stage_cap(t, t.sw[s * kEqBlock], B);
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
    return ok && sum >= t.L;
}

template <bool kCount>
__global__ void __launch_bounds__(kEqBlock) eq_search_kernel(PriceArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const Layout& y = a.lay;
    const int L = y.L;
    const EqLayout el = eq_layout(L);
    // small tables, copied once per CTA
    {
        int64_t* q = reinterpret_cast<int64_t*>(smem + el.q);
        int64_t* p2p = reinterpret_cast<int64_t*>(smem + el.p2p);
        int64_t* inter = reinterpret_cast<int64_t*>(smem + el.inter);
        int32_t* maxn = reinterpret_cast<int32_t*>(smem + el.maxn);
        int64_t* PB = reinterpret_cast<int64_t*>(smem + el.PB);
        uint8_t* win = smem + el.win;
        const int64_t* gP = reinterpret_cast<const int64_t*>(a.img + y.offP);
        for (int i = threadIdx.x; i < 32; i += blockDim.x) {
            const int g = i & 7, j = i >> 3;
            q[i] = g < y.NT ? gP[(g * 4 + j) * (L + 1) + 1] - gP[(g * 4 + j) * (L + 1)] : 0;
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
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < count; p += stride) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        if (kCount) ++searched;
        // pack the stages; feasible upper bound (every stage at its memory
        // run, which the screen guarantees covers L) and the continuous
        // balance sum_s (B - c_s) / q_s = L as the first probe
        int64_t hi = 0, qmax = 1;
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
            qmax = max(qmax, q);
            const float qf = (float)q + 0.5f;
            inv += 1.0f / qf;
            cw += (float)cc / qf;
            code = next;
        }
        int64_t lo = 0;
        bool lo_known = false, hi_known = false;
        int64_t B = (int64_t)(((float)L + cw) / inv);
        int64_t step = qmax;
        int it = 0;
        while (lo < hi) {
            B = min(max(B, lo), hi - 1);
            if (kCount) ++probes;
            if (eq_probe(t, S, B, sn)) {
                hi = sn.hi;
                hi_known = true;
            } else {
                lo = sn.lo;
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
                atomicOr(a.err, kErrSearchBound);
                break;
            }
        }
        const int64_t Bstar = hi;
        // caps at B*, then the smallest boundaries from suffix sums
        int total = 0;
        for (int s = 0; s < S; ++s) {
            const Cap r = stage_cap(t, t.sw[s * kEqBlock], Bstar);
            if (r.k < 1) atomicOr(a.err, kErrInternal);
            t.caps[s * kEqBlock] = (uint8_t)max(r.k, 0);
            total += r.k;
        }
        // ---- Evaluate: T = (M-1) max t_s + sum t_s + max g_s, stage by stage
        int64_t tmax = 0, tsum = 0;
        int sg = -1;
        u128 bestG = 0, bestD = 1;
        int pre = 0, at = 0;
        uint8_t bnd[kMaxStages + 1];
        bnd[0] = 0;
        for (int s = 0; s < S; ++s) {
            const uint32_t w = t.sw[s * kEqBlock];
            pre += t.caps[s * kEqBlock];
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
