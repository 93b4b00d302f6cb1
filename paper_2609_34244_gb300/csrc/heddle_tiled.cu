// heddle_tiled.cu -- expert tiling (§5.3 "Expert tiling").
//
// The 2^j devices of a stage factor as 2^le EP x 2^lt ETP x 2^ld EDP.  ETP
// slices one tensor and stays within the type's largest node; ETP is the
// innermost factor, so an EP group spans e t consecutive devices and uses
// the node NIC once that leaves a node; EDP replicates the experts.  Per
// layer (seconds, IEEE double, left to right, no fused multiply-add):
//   compute  flops / (k * TFLOPS * 1e12)
//   TP       k > 1: + (4 * 2(k-1)/k) * ar_bytes / bw_k     (the dense part)
//   EP       e > 1: + (4 * (e-1)/e) * a2a_bytes / bw_et
//   ETP      t > 1: + (4 * 2(t-1)/t) * a2a_bytes / intra
// quantised to the nearest ns; the slot with EP over all devices is the
// untiled cost.  Memory with EDP degree d: state + (d-1) expert state + f
// act <= mem k.  Gradient sync: ceil(2((n-1) Gd + (n d - 1) Ge) 1e9 /
// (n k bw)), bw the intra-node bandwidth when n = 1 and the stage fits one
// node, else the slowest NIC.
//
// Two kernels: a one-CTA table build (after the main cost tables), and the
// tiled search over the screen's worklist, one thread per entry with the
// tiled image in shared memory:
//   stage time     t_s(i, j) = min over allowed tilings whose memory fits of
//                  P_tiling[j] - P_tiling[i] + c_s (the earliest slot on
//                  ties); monotone under interval inclusion
//   PartitionLayers  threshold search on B with an exact probe: backward
//                  sets C_s of feasible stage-s starts (the smallest
//                  successor in C_{s+1} dominates), snapping the bracket to
//                  the largest accepted / smallest rejected stage time;
//                  the canonical split walks the sets at B* taking the
//                  smallest boundary each time
//   re-selection   per stage and EDP exponent m, the fastest fitting tiling
//                  with EDP exponent <= m; g grows with d, so for a bound Y
//                  on the gradient term each stage's admissible tilings are
//                  such a prefix; T(Y) is evaluated for every Y among the
//                  stages' gradient terms of fitting tilings and the
//                  smallest T wins (the smaller Y on ties).

#include <algorithm>

#include "heddle_tiled.cuh"

namespace hd {
namespace {

constexpr int kTabThreads = 256;
constexpr int64_t kTableLimit = (int64_t)1 << 40;
constexpr int kTBlock = 128;
constexpr int kSetWords = 8;  // 256-bit position sets (L <= 255)
constexpr int kMaxIters = 256;

// Nearest integer of v >= 0, halves away from zero (v - trunc(v) is exact
// below 2^52).
__device__ int64_t nearest_ns(double v) {
    double r = trunc(v);
    if (__dsub_rn(v, r) >= 0.5) r = __dadd_rn(r, 1.0);
    return (int64_t)r;
}

// (le, lt, ld) of slot i of degree 2^j.
__host__ __device__ inline void tiling_of(int j, int i, int& le, int& lt, int& ld) {
    int k = 0;
    for (int d = 0; d <= j; ++d)
        for (int t = 0; t + d <= j; ++t) {
            if (k == i) {
                ld = d;
                lt = t;
                le = j - d - t;
                return;
            }
            ++k;
        }
    le = lt = ld = 0;
}

__device__ inline int degree_of_slot(int slot) { return slot < 1 ? 0 : slot < 4 ? 1 : slot < 10 ? 2 : 3; }

__global__ void __launch_bounds__(kTabThreads) tiled_tables_kernel(TiledTableArgs a) {
    const TiledLayout& y = a.tl;
    const int L = y.L, NT = y.NT;
    const Layout& m = a.lay;
    const int32_t* gmaxn = reinterpret_cast<const int32_t*>(a.img + m.offMaxN);
    const int32_t* ggpus = reinterpret_cast<const int32_t*>(a.img + m.offGpus);
    const int64_t* ginter = reinterpret_cast<const int64_t*>(a.img + m.offInter);
    int64_t* Pt = reinterpret_cast<int64_t*>(a.timg + y.offPt);
    uint8_t* code = a.timg + y.offCode;
    const int tid = threadIdx.x;

    // per-layer entries, parked at Pt[row][l + 1]
    for (int t = tid; t < NT * kTileSlots * L; t += blockDim.x) {
        const int l = t % L;
        const int slot = (t / L) % kTileSlots;
        const int g = t / (kTileSlots * L);
        const int j = degree_of_slot(slot);
        int le, lt, ld;
        tiling_of(j, slot - tile_base(j), le, lt, ld);
        const bool allowed = ggpus[g] > 0 && (1 << lt) <= gmaxn[g];
        int64_t q = 0;
        if (allowed) {
            const heddle_layer ly = a.layers[l];
            const double near = __ll2double_rn(a.types[g].intra_bw), far = __ll2double_rn(ginter[g]);
            const double k = (double)(1 << j);
            double sec = __ddiv_rn(ly.flops, __dmul_rn(__dmul_rn(k, a.types[g].tflops), 1e12));
            if (j > 0) {
                const double bw = (1 << j) <= gmaxn[g] ? near : far;
                const double w = __ddiv_rn(__dmul_rn(2.0, __dsub_rn(k, 1.0)), k);
                sec = __dadd_rn(sec, __ddiv_rn(__dmul_rn(__dmul_rn(4.0, w), __ll2double_rn(ly.ar_bytes)), bw));
            }
            if (le > 0) {
                const double e = (double)(1 << le);
                const double bw = (1 << (le + lt)) <= gmaxn[g] ? near : far;
                const double part = __ddiv_rn(__dsub_rn(e, 1.0), e);
                sec = __dadd_rn(sec, __ddiv_rn(__dmul_rn(__dmul_rn(4.0, part), __ll2double_rn(ly.a2a_bytes)), bw));
            }
            if (lt > 0) {
                const double tt = (double)(1 << lt);
                const double ring = __ddiv_rn(__dmul_rn(2.0, __dsub_rn(tt, 1.0)), tt);
                sec = __dadd_rn(sec, __ddiv_rn(__dmul_rn(__dmul_rn(4.0, ring), __ll2double_rn(ly.a2a_bytes)), near));
            }
            const double ns = __dmul_rn(sec, 1e9);
            if (!(ns >= 0.0) || !(ns < 4.0e18))
                atomicOr(a.flags, kTabBadValue);
            else
                q = nearest_ns(ns);
        }
        Pt[(size_t)(g * kTileSlots + slot) * (L + 1) + l + 1] = q;
    }
    __syncthreads();
    // A tiling is dominated when another allowed tiling of the same degree
    // and EDP degree (hence the same memory and gradient terms) comes first
    // and is no slower on every layer, or is strictly faster on every layer:
    // on every interval it is then never the fastest fitting tiling, nor the
    // earliest among equally fast ones, so the search skips it (bit 6).
    for (int t = tid; t < 8 * kTileSlots; t += blockDim.x) {
        const int slot = t % kTileSlots, g = t / kTileSlots;
        const int j = degree_of_slot(slot);
        int le, lt, ld;
        tiling_of(j, slot - tile_base(j), le, lt, ld);
        const bool allowed = g < NT && ggpus[g] > 0 && (1 << lt) <= gmaxn[g];
        bool dominated = false;
        if (allowed) {
            const int64_t* me = Pt + (size_t)(g * kTileSlots + slot) * (L + 1);
            const int cnt = (j + 1) * (j + 2) / 2;
            for (int o = 0; o < cnt && !dominated; ++o) {
                const int other = tile_base(j) + o;
                int le2, lt2, ld2;
                tiling_of(j, o, le2, lt2, ld2);
                if (other == slot || ld2 != ld || (1 << lt2) > gmaxn[g]) continue;
                const int64_t* ot = Pt + (size_t)(g * kTileSlots + other) * (L + 1);
                bool le_all = true, lt_all = true;
                for (int l = 1; l <= L && le_all; ++l) {
                    le_all = ot[l] <= me[l];
                    lt_all = lt_all && ot[l] < me[l];
                }
                dominated = le_all && (lt_all || other < slot);
            }
        }
        code[t] = (uint8_t)(le | (lt << 2) | (ld << 4) | (dominated ? 0x40 : 0) | (allowed ? 0x80 : 0));
    }
    __syncthreads();
    for (int r = tid; r < NT * kTileSlots; r += blockDim.x) {
        int64_t* row = Pt + (size_t)r * (L + 1);
        row[0] = 0;
        int64_t acc = 0;
        for (int l = 1; l <= L; ++l) {
            acc += row[l];
            if (acc > kTableLimit) {
                atomicOr(a.flags, kTabTooLarge);
                acc = kTableLimit;
            }
            row[l] = acc;
        }
    }
    // byte prefixes and the per-type constants
    if (tid == 0) {
        const int64_t* SA = reinterpret_cast<const int64_t*>(a.img + m.offSA);
        const int64_t* PB = reinterpret_cast<const int64_t*>(a.img + m.offPB);
        int64_t* tSA = reinterpret_cast<int64_t*>(a.timg + y.offSA);
        int64_t* tPB = reinterpret_cast<int64_t*>(a.timg + y.offPB);
        int64_t* ES = reinterpret_cast<int64_t*>(a.timg + y.offES);
        int64_t* PE = reinterpret_cast<int64_t*>(a.timg + y.offPE);
        int64_t es = 0, pe = 0;
        ES[0] = PE[0] = 0;
        for (int l = 0; l <= L; ++l) {
            tSA[2 * l] = SA[2 * l];
            tSA[2 * l + 1] = SA[2 * l + 1];
            tPB[l] = PB[l];
            if (l < L) {
                es += a.expert_state[l];
                pe += a.expert_param[l];
                ES[l + 1] = es;
                PE[l + 1] = pe;
            }
        }
    }
    for (int t = tid; t < 8 * 8 * 2; t += blockDim.x)
        reinterpret_cast<int64_t*>(a.timg + y.offP2P)[t] = reinterpret_cast<const int64_t*>(a.img + m.offP2P)[t];
    if (tid < 8) {
        reinterpret_cast<int64_t*>(a.timg + y.offMem)[tid] = reinterpret_cast<const int64_t*>(a.img + m.offMem)[tid];
        reinterpret_cast<int64_t*>(a.timg + y.offInter)[tid] = ginter[tid];
        reinterpret_cast<int64_t*>(a.timg + y.offIntra)[tid] = tid < NT ? a.types[tid].intra_bw : 0;
        reinterpret_cast<int32_t*>(a.timg + y.offMaxN)[tid] = gmaxn[tid];
    }
}

// ------------------------------------------------------------------ search

struct TTabs {
    const int64_t* Pt;
    const longlong2* SA;
    const int64_t* ES;
    const int64_t* PB;
    const int64_t* PE;
    const int64_t* p2p;
    const int64_t* mem;
    const int64_t* inter;
    const int64_t* intra;
    const int32_t* maxn;
    const uint8_t* code;
    int L;
};

// One stage's constants.
struct TStage {
    int g, j;
    int64_t c;     // P2P to the next stage
    int64_t cap;   // memory per GPU x devices
    int64_t f;     // in-flight micro-batches
};

__device__ __forceinline__ TStage tstage(const TTabs& t, const uint8_t* codes, int s, int S, int M) {
    TStage st;
    const int b = codes[s];
    st.g = b & 7;
    st.j = (b >> 3) & 3;
    st.cap = t.mem[st.g] << st.j;
    st.f = min(S - s, M);
    st.c = 0;
    if (s + 1 < S) {
        const int bn = codes[s + 1];
        const int h = bn & 7, jn = (bn >> 3) & 3;
        const int same = (st.g == h) && ((1 << st.j) + (1 << jn) <= t.maxn[st.g]);
        st.c = t.p2p[(st.g * 8 + h) * 2 + same];
    }
    return st;
}

// Memory of layers [i, e) with EDP exponent ld fits?
__device__ __forceinline__ bool tfits(const TTabs& t, const TStage& st, int i, int e, int ld) {
    const longlong2 a = t.SA[i], b = t.SA[e];
    const int64_t mem = (b.x - a.x) + (((int64_t)1 << ld) - 1) * (t.ES[e] - t.ES[i]) + st.f * (b.y - a.y);
    return mem <= st.cap;
}

// Fastest fitting tiling of layers [i, e) on stage st (kInf if none).
__device__ int64_t ttime(const TTabs& t, const TStage& st, int i, int e) {
    const int base = tile_base(st.j), cnt = (st.j + 1) * (st.j + 2) / 2;
    int64_t best = kInf;
    for (int o = 0; o < cnt; ++o) {
        const int slot = base + o;
        const uint8_t cd = t.code[st.g * kTileSlots + slot];
        if ((cd & 0xc0) != 0x80) continue;  // not allowed, or dominated
        if (!tfits(t, st, i, e, (cd >> 4) & 3)) continue;
        const int64_t* P = t.Pt + (size_t)(st.g * kTileSlots + slot) * (t.L + 1);
        best = min(best, P[e] - P[i] + st.c);
    }
    return best;
}

__device__ __forceinline__ bool has(const uint32_t* C, int i) { return (C[i >> 5] >> (i & 31)) & 1u; }

// smallest set position in [i, hi], -1 if none
__device__ int next_in(const uint32_t* C, int i, int hi) {
    if (i > hi) return -1;
    int w = i >> 5;
    uint32_t m = C[w] & (0xffffffffu << (i & 31));
    while (m == 0) {
        if (++w > (hi >> 5)) return -1;
        m = C[w];
    }
    const int x = (w << 5) + __ffs(m) - 1;
    return x <= hi ? x : -1;
}

// largest set position in [lo, i], -1 if none
__device__ int prev_in(const uint32_t* C, int i, int lo) {
    if (i < lo) return -1;
    int w = i >> 5;
    uint32_t m = C[w] & (0xffffffffu >> (31 - (i & 31)));
    while (m == 0) {
        if (--w < (lo >> 5)) return -1;
        m = C[w];
    }
    const int x = (w << 5) + 31 - __clz(m);
    return x >= lo ? x : -1;
}

// Exact probe of bound B: C[s] = feasible starts of stage s (C[S] = {L}).
// hi / lo: largest accepted / smallest rejected stage time judged.
__device__ bool tprobe(const TTabs& t, const uint8_t* codes, int S, int M, int64_t B, int64_t& hi, int64_t& lo,
                       uint32_t (*C)[kSetWords]) {
    const int L = t.L;
    hi = -1;
    lo = kInf;
    for (int w = 0; w < kSetWords; ++w) C[S][w] = 0;
    C[S][L >> 5] = 1u << (L & 31);
    for (int s = S - 1; s >= 1; --s) {
        for (int w = 0; w < kSetWords; ++w) C[s][w] = 0;
        const TStage st = tstage(t, codes, s, S, M);
        const int imax = L - (S - s);
        int succ = next_in(C[s + 1], imax + 1, L);
        bool any = false;
        int i = imax;
        while (i >= s) {
            if (has(C[s + 1], i + 1)) succ = i + 1;
            // kInf: no successor, or no tiling of [i, succ) fits memory
            const int64_t v = succ < 0 ? kInf : ttime(t, st, i, succ);
            if (v != kInf && v <= B) {
                C[s][i >> 5] |= 1u << (i & 31);
                hi = max(hi, v);
                any = true;
                --i;
                continue;
            }
            if (v != kInf) lo = min(lo, v);
            // [i, succ) is rejected (too slow or out of memory), and so is
            // every longer [i', succ): resume below the next smaller
            // successor
            const int j2 = prev_in(C[s + 1], i, s + 1);
            if (j2 < 0) break;
            succ = j2;
            i = j2 - 1;
        }
        if (!any) return false;
    }
    const int succ0 = S == 1 ? L : next_in(C[1], 1, L);
    if (succ0 < 0) return false;
    const int64_t v = ttime(t, tstage(t, codes, 0, S, M), 0, succ0);
    if (v == kInf) return false;
    if (v <= B) {
        hi = max(hi, v);
        return true;
    }
    lo = min(lo, v);
    return false;
}

__global__ void __launch_bounds__(kTBlock) tiled_search_kernel(PriceArgs a, TiledArgs ta) {
    extern __shared__ __align__(16) unsigned char smem[];
    {
        const uint4* src = reinterpret_cast<const uint4*>(ta.timg);
        uint4* dst = reinterpret_cast<uint4*>(smem);
        for (uint32_t i = threadIdx.x; i < ta.tl.bytes / 16; i += blockDim.x) dst[i] = src[i];
    }
    __syncthreads();
    const TiledLayout& y = ta.tl;
    TTabs t;
    t.Pt = reinterpret_cast<const int64_t*>(smem + y.offPt);
    t.SA = reinterpret_cast<const longlong2*>(smem + y.offSA);
    t.ES = reinterpret_cast<const int64_t*>(smem + y.offES);
    t.PB = reinterpret_cast<const int64_t*>(smem + y.offPB);
    t.PE = reinterpret_cast<const int64_t*>(smem + y.offPE);
    t.p2p = reinterpret_cast<const int64_t*>(smem + y.offP2P);
    t.mem = reinterpret_cast<const int64_t*>(smem + y.offMem);
    t.inter = reinterpret_cast<const int64_t*>(smem + y.offInter);
    t.intra = reinterpret_cast<const int64_t*>(smem + y.offIntra);
    t.maxn = reinterpret_cast<const int32_t*>(smem + y.offMaxN);
    t.code = smem + y.offCode;
    t.L = y.L;
    const int L = y.L;

    uint32_t C[kMaxStages + 1][kSetWords];
    uint8_t codes[kMaxStages];
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < count;
         p += (int64_t)gridDim.x * blockDim.x) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        {
            const uint4* row = reinterpret_cast<const uint4*>(a.wl_code + p * kMaxStages);
            const uint4 v0 = row[0], v1 = row[1];
            const uint32_t w[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            for (int s = 0; s < kMaxStages; ++s) codes[s] = (uint8_t)(w[s >> 2] >> ((s & 3) * 8));
        }
        // memory-only probe: OOM, else a feasible upper bound
        int64_t hi, lo;
        if (!tprobe(t, codes, S, M, kInf, hi, lo, C)) {
            a.T[c] = -1;
            a.B[c] = -1;
            a.ndp[c] = (uint16_t)n;
            a.status[c] = HEDDLE_CAND_OOM;
            if (a.bounds)
                for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = 0;
            a.wl_T[p] = -1;
            continue;
        }
        // first guess: the balanced bound with every stage at its fastest
        // tiling over all layers, then gallop until the bracket closes
        float inv = 0.f, cw = 0.f;
        for (int s = 0; s < S; ++s) {
            const TStage st = tstage(t, codes, s, S, M);
            const int base = tile_base(st.j), cnt = (st.j + 1) * (st.j + 2) / 2;
            int64_t all = kInf;
            for (int o = 0; o < cnt; ++o)
                if ((t.code[st.g * kTileSlots + base + o] & 0xc0) == 0x80)
                    all = min(all, t.Pt[(size_t)(st.g * kTileSlots + base + o) * (L + 1) + L]);
            const float tot = u64_to_float((uint64_t)all) + 1.0f;
            inv += 1.0f / tot;
            cw += u64_to_float((uint64_t)st.c) / tot;
        }
        int64_t Bhi = hi, Blo = 0;
        bool lo_known = false, hi_known = false;
        int64_t B = (int64_t)float_to_u64((1.0f + cw) / inv);
        int64_t step = max((int64_t)1, (int64_t)float_to_u64(u64_to_float(B) * (float)S / (2.0f * (float)L)));
        int it = 0;
        while (Blo < Bhi) {
            B = min(max(B, Blo), Bhi - 1);
            if (tprobe(t, codes, S, M, B, hi, lo, C)) {
                Bhi = hi;
                hi_known = true;
            } else {
                Blo = lo;
                lo_known = true;
            }
            if (Blo >= Bhi) break;
            if (!lo_known) {
                B = Bhi - step;
                step *= 2;
            } else if (!hi_known) {
                B = Blo + step;
                step *= 2;
            } else {
                B = Blo + (Bhi - Blo) / 2;
            }
            if (++it > kMaxIters) {
                atomicOr(a.err, kErrSearchBound);
                break;
            }
        }
        const int64_t Bstar = Bhi;
        if (!tprobe(t, codes, S, M, Bstar, hi, lo, C)) atomicOr(a.err, kErrInternal);
        uint8_t bnd[kMaxStages + 1];
        bnd[0] = 0;
        for (int s = 0; s + 1 < S; ++s) {
            const int x = next_in(C[s + 1], bnd[s] + 1, L);
            if (x < 0) atomicOr(a.err, kErrInternal);
            bnd[s + 1] = (uint8_t)max(x, 0);
        }
        bnd[S] = (uint8_t)L;

        // ---- re-selection on the split: per stage and EDP exponent m the
        //      fastest fitting tiling with EDP exponent <= m, and the
        //      gradient term of each EDP exponent
        int64_t bt[kMaxStages][4], gg[kMaxStages][4];
        uint8_t bc[kMaxStages][4], bl[kMaxStages][4], hd_[kMaxStages];
        for (int s = 0; s < S; ++s) {
            const TStage st = tstage(t, codes, s, S, M);
            const int i0 = bnd[s], i1 = bnd[s + 1];
            const int64_t Ge = t.PE[i1] - t.PE[i0];
            const int64_t Gd = (t.PB[i1] - t.PB[i0]) - Ge;
            const int64_t bw = (n == 1 && (1 << st.j) <= t.maxn[st.g]) ? t.intra[st.g] : t.inter[st.g];
            const int base = tile_base(st.j);
            int64_t best = kInf;
            uint8_t bcode = 0, bld = 0, hasld = 0;
            int o = 0;
            for (int m = 0; m <= st.j; ++m) {
                const u128 vol = (u128)(n - 1) * (u128)Gd + (u128)((n << m) - 1) * (u128)Ge;
                int64_t gv = 0;
                if (vol != 0) {
                    bool ok = true;
                    gv = (int64_t)ceil_div_u128((u128)2 * vol * 1000000000u, (uint64_t)(n << st.j) * (uint64_t)bw, &ok);
                    if (!ok) atomicOr(a.err, kErrInternal);
                }
                gg[s][m] = gv;
                // the slots of EDP exponent m: ETP exponent 0 .. j - m
                for (int lt = 0; lt <= st.j - m; ++lt, ++o) {
                    const uint8_t cd = t.code[st.g * kTileSlots + base + o];
                    if ((cd & 0xc0) != 0x80 || !tfits(t, st, i0, i1, m)) continue;
                    hasld |= (uint8_t)(1 << m);
                    const int64_t* P = t.Pt + (size_t)(st.g * kTileSlots + base + o) * (L + 1);
                    const int64_t v = P[i1] - P[i0] + st.c;
                    if (v < best) {
                        best = v;
                        bcode = cd & 15;
                        bld = (uint8_t)m;
                    }
                }
                bt[s][m] = best;
                bc[s][m] = bcode;
                bl[s][m] = bld;
            }
            hd_[s] = hasld;
        }
        int64_t bestT = kInf, bestY = 0, bestB = 0;
        int ys_best = -1;
        uint8_t pick[kMaxStages];
        for (int ys = 0; ys < S; ++ys) {
            const int jy = (codes[ys] >> 3) & 3;
            for (int my = 0; my <= jy; ++my) {
                if (!((hd_[ys] >> my) & 1)) continue;
                const int64_t Y = gg[ys][my];
                int64_t tm = 0, ts = 0, gm = 0;
                bool all = true;
                for (int s = 0; s < S && all; ++s) {
                    const int js = (codes[s] >> 3) & 3;
                    int mm = -1;
                    while (mm + 1 <= js && gg[s][mm + 1] <= Y) ++mm;
                    if (mm < 0 || bt[s][mm] == kInf) {
                        all = false;
                        break;
                    }
                    tm = max(tm, bt[s][mm]);
                    ts += bt[s][mm];
                    gm = max(gm, gg[s][bl[s][mm]]);
                    pick[s] = (uint8_t)mm;
                }
                if (!all) continue;
                const int64_t T = (int64_t)(M - 1) * tm + ts + gm;
                if (T < bestT || (T == bestT && Y < bestY)) {
                    bestT = T;
                    bestY = Y;
                    bestB = tm;
                    ys_best = ys;
                    if (ta.tiling)
                        for (int s = 0; s < S; ++s) ta.tiling[(int64_t)s * ta.tstride + c] = bc[s][pick[s]];
                }
            }
        }
        if (ys_best < 0) {
            atomicOr(a.err, kErrInternal);
            bestT = -1;
        }
        a.T[c] = bestT;
        a.wl_T[p] = bestT;
        a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
        a.B[c] = bestB;
        a.ndp[c] = (uint16_t)n;
        a.status[c] = HEDDLE_CAND_OK;
        if (a.bounds)
            for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = s <= S ? bnd[s] : 0;
    }
}

}  // namespace

cudaError_t launch_tiled_tables(const TiledTableArgs& a, cudaStream_t st) {
    tiled_tables_kernel<<<1, kTabThreads, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_tiled_search(const PriceArgs& a, const TiledArgs& t, int num_sms, cudaStream_t st) {
    const size_t smem = t.tl.bytes;
    cudaError_t e = cudaFuncSetAttribute(tiled_search_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, tiled_search_kernel, kTBlock, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: size for the batch
    const int64_t need = (a.n + kTBlock - 1) / kTBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    tiled_search_kernel<<<grid, kTBlock, smem, st>>>(a, t);
    return cudaGetLastError();
}

}  // namespace hd
