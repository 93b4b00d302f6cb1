// heddle_eqsearch.cu -- PartitionLayers + Evaluate for models whose layers
// all cost the same (§3.1 listing, §5.2 memory validation, §5.3 iteration
// time), over the worklist the screen kernel produced.
//
// When every layer has the same quantised cost q_s on a stage's (type,
// degree) and the same state and activation bytes, stage s holds exactly
//     cap_s(B) = min(m_s, floor((B - c_s) / q_s))
// layers within bound B (m_s: the longest run of layers that fits the
// stage's memory, c_s: its P2P).  A split with every stage time <= B exists
// iff every cap_s >= 1 and sum_s cap_s >= L, so a probe costs O(S), and
// B* is the smallest such B -- a breakpoint c_s + k q_s of some stage.
//
// First guess, in float only: the continuous balance
// sum_s min(m_s, (B - c_s) / q_s) = L + (stages below their run) / 2 (the
// floors lose half a layer per such stage on average), solved by at most
// three Newton steps from the unsaturated balance.  One exact probe then
// decides the bracket, and exact stop rules name B* from that probe alone
// in almost every case:
//   feasible, and the stages at the largest stage time hi cannot all lose
//   a layer (one of them holds a single layer, or the count would drop
//   below L) -> B* = hi;
//   feasible, and the same holds one level down, at hi2 = the largest stage
//   time once the stages at hi have lost their top layer -> B* = hi2;
//   infeasible, and at the next breakpoint lo every stage holds a layer and
//   the stages that gain one there bring the total to L -> B* = lo.
// Every probe leaves each stage's cap in that stage's word, so the caps at
// B* follow from the last probe (the same, one fewer for the stages at hi,
// or one more for the stages gaining at lo) and Evaluate needs no division.
// A search still open after the first probe continues in its own thread:
// the next bound interpolates the cap count between the bracket's probes (a
// Newton step while one side is missing), else bisects.  The caps at B*
// give the componentwise smallest split -- hence the lexicographically
// smallest -- a_{s+1} = max(a_s + 1, L - sum_{t > s} cap_t).
//
// Scheduling: the screen files every entry in a bucket per depth S; warp w
// takes entries [32 w, 32 w + 32) of the buckets read in order of
// decreasing S, so its lanes run stage loops of equal length, and then the
// next 32 untaken entries from a counter whenever it is free.  Warps work
// independently (no CTA barrier after the tables are staged): every thread
// packs its candidate's stages once into 32-bit words (cost index | P2P
// index | memory run | cap) held in shared memory interleaved by thread,
// runs the float guess, the exact probe and Evaluate.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kEqBlock = 128;
constexpr int kEqWarps = kEqBlock / 32;
constexpr int kZeroP2P = 128;  // a zero entry after the 8 x 8 x 2 P2P table
constexpr int kMaxIters = 256;

// How the caps at B* follow from the caps the last probe stored.
enum CapMode : int { kCapsAsStored = 0, kCapsLessAtHi = 1, kCapsMoreAtLo = 2 };

// State of one threshold search (registers of the thread that owns it).
struct Search {
    int64_t lo, hi, B;  // B* lies in [lo, hi]; B is the next bound to probe
    int64_t Blo, Bhi;   // last infeasible / feasible bound probed (-1: none)
    int64_t anchor;     // hi (kCapsLessAtHi) or lo (kCapsMoreAtLo) of the last probe
    int32_t clo, chi;   // layer counts of those probes; chi is the count at hi
    int32_t probes;
    int32_t mode;       // CapMode of the stored caps relative to q.hi, -1: not at B* (yet)
};

struct EqLayout {
    uint32_t q, rq, p2p, cf, inter, maxn, PB, win, sw, bytes;
};

__host__ __device__ inline uint32_t al16(uint32_t x) { return (x + 15u) & ~15u; }

__host__ __device__ inline EqLayout eq_layout(int L) {
    EqLayout e;
    uint32_t o = 0;
    e.q = o;     o = al16(o + 8 * 32);             // int64 [j * 8 + g]
    e.rq = o;    o = al16(o + 4 * 32);             // float 1 / q
    e.p2p = o;   o = al16(o + 8 * 129);            // int64 [(g * 8 + h) * 2 + same], [128] = 0
    e.cf = o;    o = al16(o + 4 * 129);            // float P2P
    e.inter = o; o = al16(o + 8 * 8);              // int64 [g]
    e.maxn = o;  o = al16(o + 4 * 8);              // int32 [g]
    e.PB = o;    o = al16(o + 8 * (L + 1));        // int64 gradient-byte prefix
    e.win = o;   o = al16(o + 8 * 4 * 33);         // uint8 [(g * 4 + j) * 33 + f]
    e.sw = o;    o = al16(o + 4 * kMaxStages * kEqBlock);  // uint32 [s][thread]
    e.bytes = o;
    return e;
}

struct EqTabs {
    const int64_t* q;
    const float* rq;
    const int64_t* p2p;
    const float* cf;
    const int64_t* inter;
    const int32_t* maxn;
    const int64_t* PB;
    const uint8_t* win;
    int64_t pbytes;  // gradient bytes of every layer when they are all equal, else -1
    int L;
};

// Stage word: bits 0-4 cost index (the stage byte's type | degree bits),
// bits 5-12 P2P index, bits 13-20 memory run m, bits 21-28 the cap the last
// probe found.
constexpr int kCapShift = 21;
constexpr uint32_t kNoCap = 0x1fffffu;

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

// Continuous count at Bf (float): sum_s min(m_s, (Bf - c_s) / q_s), with
// the slope sum 1/q_s and the number of stages below their run.
__device__ float eq_count(const EqTabs& t, const uint32_t* sw, int S, float Bf, float& slope, int& below) {
    float cnt = 0.f, sl = 0.f;
    int nb = 0;
    for (int s = 0; s < S; ++s) {
        const uint32_t w = sw[s * kEqBlock];
        const float rq = t.rq[w & 31];
        const float m = (float)((w >> 13) & 255);
        const float x = (Bf - t.cf[(w >> 5) & 255]) * rq;
        if (rq == 0.f || x >= m) {
            cnt += m;
        } else {
            cnt += x;
            sl += rq;
            ++nb;
        }
    }
    slope = sl;
    below = nb;
    return cnt;
}

// Result of an exact probe at bound B.
struct Probe {
    int64_t hi;    // largest stage time c + k q over stages holding a layer
    int64_t lo;    // next breakpoint above B: min c + (k + 1) q over stages below their run
    int64_t zmax;  // largest c + q over stages holding no layer (-1: none)
    int64_t P;     // largest c + (k - 1) q over the stages at hi
    int64_t R;     // largest stage time below hi
    int tot;       // layers the stages hold
    int nhi, nlo;  // stages attaining hi / lo
    int nP, nR;    // stages attaining P / R
    bool hi1;      // a stage attaining hi holds a single layer
    bool P1, R1;   // a stage attaining P / R would hold a single layer there
    float slope;   // sum of 1/q over stages below their run
};

// Exact probe of bound B for the stages in column sw; stores each stage's
// cap in its word.
__device__ bool eq_probe(const EqTabs& t, uint32_t* sw, int S, int64_t B, Probe& p) {
    p.hi = -1;
    p.lo = kInf;
    p.zmax = -1;
    p.P = -1;
    p.R = -1;
    p.tot = 0;
    p.nhi = p.nlo = p.nP = p.nR = 0;
    p.hi1 = p.P1 = p.R1 = false;
    p.slope = 0.f;
    for (int s = 0; s < S; ++s) {
        const uint32_t w = sw[s * kEqBlock];
        const int64_t q = t.q[w & 31];
        const int64_t c = t.p2p[(w >> 5) & 255];
        const int m = (int)(w >> 13) & 255;
        int k;
        const int64_t x = B - c;
        if (m < 1 || x < q) {
            k = 0;
        } else if (q == 0 || x >= (int64_t)m * q) {
            k = m;
        } else {
            // x < m q with m <= 255: the float estimate is off by at most one
            k = (int)(u64_to_float((uint64_t)x) * t.rq[w & 31]);
            if ((int64_t)k * q > x) --k;
            if ((int64_t)(k + 1) * q <= x) ++k;
        }
        sw[s * kEqBlock] = (w & kNoCap) | ((uint32_t)k << kCapShift);
        if (m < 1) {
            p.zmax = kInf;  // never holds a layer
            continue;
        }
        if (k < m) {
            p.slope += t.rq[w & 31];
            const int64_t nb = c + (int64_t)(k + 1) * q;
            if (nb < p.lo) {
                p.lo = nb;
                p.nlo = 1;
            } else if (nb == p.lo) {
                ++p.nlo;
            }
        }
        if (k < 1) {
            p.zmax = max(p.zmax, c + q);
            continue;
        }
        p.tot += k;
        const int64_t v = c + (int64_t)k * q;
        if (v > p.hi) {
            // the stages at the old hi drop to the level below
            if (p.hi > p.R) {
                p.R = p.hi;
                p.nR = p.nhi;
                p.R1 = p.hi1;
            } else if (p.hi == p.R) {
                p.nR += p.nhi;
                p.R1 |= p.hi1;
            }
            p.hi = v;
            p.nhi = 1;
            p.hi1 = k == 1;
            p.P = v - q;
            p.nP = 1;
            p.P1 = k == 2;
        } else if (v == p.hi) {
            ++p.nhi;
            p.hi1 |= k == 1;
            const int64_t u = v - q;
            if (u > p.P) {
                p.P = u;
                p.nP = 1;
                p.P1 = k == 2;
            } else if (u == p.P) {
                ++p.nP;
                p.P1 |= k == 2;
            }
        } else if (v > p.R) {
            p.R = v;
            p.nR = 1;
            p.R1 = k == 1;
        } else if (v == p.R) {
            ++p.nR;
            p.R1 |= k == 1;
        }
    }
    return p.zmax < 0 && p.tot >= t.L;
}

// One exact probe of search q at q.B and the bracket update; returns true
// when B* = q.hi is known (q.mode then says how the stored caps give the
// caps at B*, or -1 if they do not).
__device__ bool eq_step(const EqTabs& t, uint32_t* sw, int S, Search& q, uint32_t* err) {
    q.B = min(max(q.B, q.lo), q.hi - 1);
    ++q.probes;
    Probe p;
    const bool feas = eq_probe(t, sw, S, q.B, p);
    q.mode = -1;
    if (feas) {
        q.hi = p.hi;
        q.Bhi = q.B;
        q.chi = p.tot;
        q.mode = kCapsAsStored;
        // just below hi every stage attaining hi loses a layer
        if (p.tot - p.nhi < t.L || p.hi1) {
            q.lo = q.hi;
        } else {
            // the next level down, hi2, is feasible with tot - nhi layers
            const int64_t hi2 = max(p.P, p.R);
            const int n2 = (p.P == hi2 ? p.nP : 0) + (p.R == hi2 ? p.nR : 0);
            const bool one2 = (p.P == hi2 && p.P1) || (p.R == hi2 && p.R1);
            q.anchor = p.hi;
            q.hi = hi2;
            q.chi = p.tot - p.nhi;
            q.mode = kCapsLessAtHi;
            if (p.tot - p.nhi - n2 < t.L || one2) q.lo = hi2;
        }
    } else {
        q.lo = min(max(q.lo, p.lo), q.hi);
        q.Blo = q.B;
        q.clo = p.tot;
        // at lo every stage attaining lo gains exactly one layer
        if (p.zmax <= p.lo && p.tot + p.nlo >= t.L && p.lo < kInf) {
            q.hi = q.lo;
            q.chi = p.tot + p.nlo;
            q.anchor = p.lo;
            q.mode = kCapsMoreAtLo;
        }
    }
    if (q.lo >= q.hi) return true;
    // next bound: interpolate the cap count between the bracket's probes,
    // else a Newton step, else bisect
    float target;
    if (q.Blo >= 0 && q.Bhi >= 0 && q.chi > q.clo) {
        target = u64_to_float(q.Blo) +
                 ((float)t.L - 0.5f - (float)q.clo) / (float)(q.chi - q.clo) * u64_to_float(q.Bhi - q.Blo);
    } else if (p.slope > 0.f) {
        const float Bf = u64_to_float(q.B);
        target = feas ? Bf - ceilf(((float)p.tot - (float)t.L + 0.5f) / p.slope)
                      : Bf + ceilf(((float)t.L - (float)p.tot) / p.slope);
    } else {
        target = -1.f;
    }
    q.B = (target >= u64_to_float(q.lo) && target <= u64_to_float(q.hi - 1)) ? (int64_t)float_to_u64(target)
                                                                                : q.lo + (q.hi - q.lo) / 2;
    if (q.probes > kMaxIters) {
        atomicOr(err, kErrSearchBound);
        q.lo = q.hi;
        q.mode = -1;
        return true;
    }
    return false;
}

// The smallest boundaries from the caps at B* (the stored caps, adjusted by
// q.mode), then Evaluate: T = (M-1) max t_s + sum t_s + max g_s; writes
// entry p and returns T.
__device__ int64_t eq_evaluate(const PriceArgs& a, const EqTabs& t, const uint32_t* sw, int64_t p, int S, int M,
                               int64_t n, const Search& q) {
    const int L = t.L;
    const int64_t Bstar = q.hi;
    const int total = q.chi;
    const int64_t c = a.wl_idx[p];
    if (!in_range(c, a.n, a.err)) return -1;
    int64_t tmax = 0, tsum = 0;
    int sg = -1;
    // the stage with the largest G_s / (k_s bw_s), compared exactly: with
    // equal gradient bytes per layer G_s = layers * bytes, and layers
    // (< 2^8) times bandwidth (< 2^43) fits 64 bits
    uint64_t bestG = 0, bestD = 1;
    int pre = 0, at = 0;
    int64_t pb_at = t.PB[0];
    for (int s = 0; s < S; ++s) {
        const uint32_t w = sw[s * kEqBlock];
        const int64_t qq = t.q[w & 31];
        const int64_t cc = t.p2p[(w >> 5) & 255];
        int k = (int)(w >> kCapShift) & 255;
        if (q.mode == kCapsLessAtHi) {
            if (cc + (int64_t)k * qq == q.anchor) --k;
        } else if (q.mode == kCapsMoreAtLo) {
            if (k < (int)((w >> 13) & 255) && cc + (int64_t)(k + 1) * qq == q.anchor) ++k;
        }
        if (k < 1) atomicOr(a.err, kErrInternal);
        pre += k;
        const int nxt = s + 1 == S ? L : max(at + 1, L - (total - pre));
        if (a.bounds) a.bounds[(int64_t)(s + 1) * a.bstride + c] = (uint8_t)nxt;
        const int64_t ts = (int64_t)(nxt - at) * qq + cc;
        tmax = max(tmax, ts);
        tsum += ts;
        if (n > 1) {
            const int g = w & 7, j = (w >> 3) & 3;
            const uint64_t D = (uint64_t)t.inter[g] << j;
            if (t.pbytes >= 0) {
                const uint64_t len = (uint64_t)(nxt - at);
                if (sg < 0 || len * bestD > bestG * D) {
                    sg = s;
                    bestG = len;
                    bestD = D;
                }
            } else {
                const int64_t pb_nxt = in_range(nxt, L + 1, a.err) ? t.PB[nxt] : pb_at;
                const uint64_t G = (uint64_t)(pb_nxt - pb_at);
                pb_at = pb_nxt;
                if (sg < 0 || (u128)G * bestD > (u128)bestG * D) {
                    sg = s;
                    bestG = G;
                    bestD = D;
                }
            }
        }
        at = nxt;
    }
    if (t.pbytes >= 0) bestG *= (uint64_t)t.pbytes;
    if (a.bounds) {
        a.bounds[c] = 0;
        for (int s = S + 1; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = 0;
    }
    if (tmax != Bstar || pre != total) atomicOr(a.err, kErrInternal);
    int64_t gmax = 0;
    if (n > 1) {
        // ring all-reduce over n replicas: ceil(2(n-1) G 1e9 / (n k bw))
        // (G < 2^50 and bandwidths < 2^40 keep n k bw below 2^64)
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
    return T;
}

template <bool kCount>
__global__ void __launch_bounds__(kEqBlock, 1024 / kEqBlock) eq_search_kernel(PriceArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int end_of[kMaxStages + 2];  // entries of depths >= S, [S]
    const Layout& y = a.lay;
    const int L = y.L;
    const EqLayout el = eq_layout(L);
    // small tables, copied once per CTA
    {
        int64_t* q = reinterpret_cast<int64_t*>(smem + el.q);
        float* rq = reinterpret_cast<float*>(smem + el.rq);
        int64_t* p2p = reinterpret_cast<int64_t*>(smem + el.p2p);
        float* cf = reinterpret_cast<float*>(smem + el.cf);
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
        for (int i = threadIdx.x; i < 129; i += blockDim.x) {
            const int64_t v = i < 128 ? reinterpret_cast<const int64_t*>(a.img + y.offP2P)[i] : 0;
            p2p[i] = v;
            cf[i] = (float)v;
        }
        for (int i = threadIdx.x; i < 8; i += blockDim.x) {
            inter[i] = reinterpret_cast<const int64_t*>(a.img + y.offInter)[i];
            maxn[i] = reinterpret_cast<const int32_t*>(a.img + y.offMaxN)[i];
        }
        for (int i = threadIdx.x; i < 8 * 4 * 33; i += blockDim.x) win[i] = a.img[y.offWin + i];
        for (int i = threadIdx.x; i <= L; i += blockDim.x)
            PB[i] = reinterpret_cast<const int64_t*>(a.img + y.offPB)[i];
    }
    if (threadIdx.x < 32) {
        // end_of[S] = entries of depths >= S: an inclusive scan of depths
        // 32 .. 1 in lanes 0 .. 31
        const int lane = threadIdx.x;
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
    EqTabs t;
    t.q = reinterpret_cast<const int64_t*>(smem + el.q);
    t.rq = reinterpret_cast<const float*>(smem + el.rq);
    t.p2p = reinterpret_cast<const int64_t*>(smem + el.p2p);
    t.cf = reinterpret_cast<const float*>(smem + el.cf);
    t.inter = reinterpret_cast<const int64_t*>(smem + el.inter);
    t.maxn = reinterpret_cast<const int32_t*>(smem + el.maxn);
    t.PB = reinterpret_cast<const int64_t*>(smem + el.PB);
    t.win = smem + el.win;
    t.pbytes = reinterpret_cast<const int32_t*>(a.img + y.offModel)[2]
                   ? t.PB[1] - t.PB[0]
                   : -1;
    t.L = L;
    uint32_t* mysw = reinterpret_cast<uint32_t*>(smem + el.sw) + threadIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    unsigned long long units = 0, probes = 0, searched = 0;
    // the entries filed in the depth buckets (every worklist entry here)
    const int64_t entries = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t count = min((int64_t)end_of[1], entries);
    // warp w of CTA b takes entries [32 (4 b + w), +32) of the order by
    // decreasing S, so its lanes have nearly equal S, then the next 32
    // untaken ones whenever it is free; warps never wait on one another
    const int64_t first = (int64_t)gridDim.x * kEqBlock;
    auto take = [&]() {
        int b = 0;
        if (lane == 0) b = atomicAdd(a.wl_count + kWlTakeThread, 32);
        return first + __shfl_sync(0xffffffffu, b, 0);
    };
    for (int64_t base = ((int64_t)blockIdx.x * kEqWarps + warp) * 32; base < count; base = take()) {
        const int64_t g = base + lane;
        bool have = g < count;
        int64_t p = 0;
        int S = 0, M = 0;
        int64_t n = 0;
        int64_t T = -1;
        if (have) {
            // its depth: the largest S with end_of[S] > g (end_of falls with S)
            int lo = 1, hi = kMaxStages;
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (end_of[mid] > g) lo = mid; else hi = mid - 1;
            }
            const int64_t off = g - end_of[lo + 1];
            if (!in_range(off, end_of[lo] - end_of[lo + 1], a.err)) have = false;
            else p = a.wl_bucket[(int64_t)(lo - 1) * a.wl_cap + off];
            if (have && !in_range(p, entries, a.err)) have = false;
        }
        if (have) {
            S = a.wl_S[p];
            M = a.wl_M[p];
            n = a.wl_n[p];
            if (kCount) {
                ++searched;
                units += S;
            }
            // pack the stages; feasible upper bound (every stage at its
            // memory run, which the screen guarantees covers L), lower bound
            // (every stage holds one layer), unsaturated continuous balance
            Search q;
            q.lo = 0;
            q.hi = 0;
            float inv = 0.f, cw = 0.f;
            // the entry's row of stage bytes (zero past S), 16 at a time
            uint32_t cw4[8];
            {
                const uint4* row = reinterpret_cast<const uint4*>(a.wl_code + p * kMaxStages);
                const uint4 v0 = __ldg(row);
                const uint4 v1 = S > 16 ? __ldg(row + 1) : make_uint4(0, 0, 0, 0);
                cw4[0] = v0.x; cw4[1] = v0.y; cw4[2] = v0.z; cw4[3] = v0.w;
                cw4[4] = v1.x; cw4[5] = v1.y; cw4[6] = v1.z; cw4[7] = v1.w;
            }
#pragma unroll
            for (int s = 0; s < kMaxStages; ++s) {
                if (s >= S) break;
                const int code = (cw4[s >> 2] >> ((s & 3) * 8)) & 0xff;
                const int next = s + 1 < kMaxStages ? (cw4[(s + 1) >> 2] >> (((s + 1) & 3) * 8)) & 0xff : 0;
                const uint32_t w = stage_word(code, next, s + 1 == S, min(S - s, M), t);
                mysw[s * kEqBlock] = w;
                const int64_t qq = t.q[w & 31], cc = t.p2p[(w >> 5) & 255];
                const int m = (int)(w >> 13) & 255;
                q.hi = max(q.hi, cc + (int64_t)m * qq);
                q.lo = max(q.lo, cc + qq);
                const float rq = t.rq[w & 31];
                inv += rq;
                cw += t.cf[(w >> 5) & 255] * rq;
            }
            // first guess: Newton on the saturating continuous count
            const float flo = u64_to_float(q.lo), fhi = u64_to_float(q.hi);
            float Bf = fmaxf(flo, inv > 0.f ? ((float)L + 0.5f * (float)S + cw) / inv : flo);
            for (int it = 0; it < 3; ++it) {  // the exact probes finish the job
                float sl;
                int below;
                Bf = fminf(Bf, fhi);
                const float cnt = eq_count(t, mysw, S, Bf, sl, below);
                const float tgt = (float)L + 0.5f * (float)below;
                if (cnt >= tgt - 0.25f || sl <= 0.f) break;
                Bf += (tgt - cnt) / sl;
            }
            q.B = (int64_t)float_to_u64(fminf(Bf, fhi));
            q.Blo = q.Bhi = -1;
            q.clo = q.chi = 0;
            q.probes = 0;
            q.mode = -1;
            q.anchor = 0;
            // exact probes until B* is known (one in almost every case),
            // then one more at B* itself if the stored caps are not its own
            if (q.lo < q.hi) {
                while (!eq_step(t, mysw, S, q, a.err)) {
                }
            }
            if (q.mode < 0) {
                Probe pr;
                ++q.probes;
                if (!eq_probe(t, mysw, S, q.hi, pr) || pr.hi != q.hi) atomicOr(a.err, kErrInternal);
                q.chi = pr.tot;
                q.mode = kCapsAsStored;
            }
            if (kCount) probes += q.probes;
            T = eq_evaluate(a, t, mysw, p, S, M, n, q);
        }
        if (a.sv_count) {
            // inside a top-k pricing: the entries whose n*M / T reaches the
            // running threshold (float, below the k-th key by a margin that
            // covers the rounding) go to the top-k's survivor list.  The
            // warp first raises the threshold to its own k-th best key (for
            // k <= 32): any k entries' smallest key is at most the call's
            // final k-th, so the raised value keeps the filter exact
            const uint32_t nM = (uint32_t)n * (uint32_t)M;
            const float key = have && T > 0 ? (float)nM / (float)T : -1.0f;
            const int kk = min(max(__ldg(a.topk_k), 1), kMaxTopK);
            float own = 0.f;
            if (kk <= 32) {
                float v = key;  // bitonic sort of the warp's keys, descending
#pragma unroll
                for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
                    for (int stride2 = size >> 1; stride2 > 0; stride2 >>= 1) {
                        const float o = __shfl_xor_sync(0xffffffffu, v, stride2);
                        const bool desc = (lane & size) == 0 || size == 32;
                        v = (((lane & stride2) == 0) == desc) ? fmaxf(v, o) : fminf(v, o);
                    }
                const float kth = __shfl_sync(0xffffffffu, v, kk - 1);
                if (kth > 0.f) {
                    own = kth * (1.0f - 1.0f / 65536.0f);
                    if (lane == 0) atomicMax(a.thr, __float_as_uint(own));
                }
            }
            const float thr = fmaxf(__uint_as_float(__ldcg(a.thr)), own);
            const bool keep = key > 0.f && key >= thr;
            const unsigned mask = __ballot_sync(0xffffffffu, keep);
            if (mask) {
                int base0 = 0;
                if (lane == __ffs(mask) - 1) base0 = atomicAdd(a.sv_count, __popc(mask));
                const int pos = __shfl_sync(0xffffffffu, base0, __ffs(mask) - 1) + __popc(mask & ((1u << lane) - 1));
                if (keep && pos < a.wl_cap) {
                    a.sv_idx[pos] = a.wl_idx[p];
                    a.sv_T[pos] = T;
                    a.sv_nM[pos] = nM;
                }
            }
        }
    }
    if (kCount) {
        unsigned long long v0 = units, v1 = probes, v2 = searched;
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
    const size_t smem = eq_layout(a.lay.L).bytes;
    int per_sm = 0;
    const cudaError_t e = resident_blocks(reinterpret_cast<const void*>(&eq_search_kernel<kCount>), kEqBlock, smem, &per_sm);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: size for the batch,
    // at most seven of the eight CTAs that fit an SM -- warps fetch further
    // entries when free, and the free slot lets the next chunk's screen
    // start beside this search's last warps
    const int64_t need = (a.n + kEqBlock - 1) / kEqBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * std::min(per_sm, 7));
    eq_search_kernel<kCount><<<grid, kEqBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_eq_search(const PriceArgs& a, int num_sms, cudaStream_t st) {
    return a.counters ? launch<true>(a, num_sms, st) : launch<false>(a, num_sms, st);
}

}  // namespace hd
