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
// tiled search over the screen's worklist, one warp per entry with the
// tiled image in shared memory:
//   stage time     t_s(i, j) = min over allowed tilings whose memory fits of
//                  P_tiling[j] - P_tiling[i] + c_s (the earliest slot on
//                  ties); monotone under interval inclusion
//   PartitionLayers  the exact threshold search of the general search, its
//                  probe (heddle_wprobe.cuh) checking 32 positions per round
//                  with this stage time; the canonical split from the sets
//                  at B*
//   re-selection   one lane per stage keeps, per EDP exponent m, the
//                  fastest fitting tiling with EDP exponent <= m and the
//                  gradient term of m; g grows with d, so for a bound Y on
//                  the gradient term each stage's admissible tilings are
//                  such a prefix; T(Y) (warp reductions) is evaluated for
//                  every Y among the stages' gradient terms of fitting
//                  tilings and the smallest T wins (the smaller Y on ties).

#include <algorithm>

#include "heddle_tiled.cuh"
#include "heddle_wprobe.cuh"

namespace hd {
namespace {

constexpr int kTabThreads = 256;
constexpr int64_t kTableLimit = (int64_t)1 << 40;
constexpr int kTBlock = 256;
constexpr int kTWarps = kTBlock / 32;
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
    const int32_t* maxn;
    const int64_t* intra;
    const uint8_t* code;
    int L;
};

// One stage's constants.
struct TLane {
    int g, j;
    int64_t c;    // P2P to the next stage
    int64_t cap;  // memory per GPU x devices
    int64_t f;    // in-flight micro-batches
};

// Memory of layers [i, e) with EDP exponent ld fits?
__device__ __forceinline__ bool tfits(const TTabs& t, const TLane& st, int i, int e, int ld) {
    const longlong2 a = t.SA[i], b = t.SA[e];
    const int64_t mem = (b.x - a.x) + (((int64_t)1 << ld) - 1) * (t.ES[e] - t.ES[i]) + st.f * (b.y - a.y);
    return mem <= st.cap;
}

// The interval test of the tiled search: the fastest allowed, undominated
// tiling whose memory fits (2 if none fits).
struct TiledCheck {
    typedef TLane Stage;
    const TTabs& t;
    TLane mine;  // the stage this lane holds
    __device__ TLane stage(int s) const {
        TLane r;
        r.g = __shfl_sync(wp::kFull, mine.g, s);
        r.j = __shfl_sync(wp::kFull, mine.j, s);
        r.c = __shfl_sync(wp::kFull, mine.c, s);
        r.cap = __shfl_sync(wp::kFull, mine.cap, s);
        r.f = __shfl_sync(wp::kFull, mine.f, s);
        return r;
    }
    // not inlined: the probe calls it from several places, and inlined
    // copies of its loop over the tilings made the kernel wait on
    // instruction fetch
    __device__ __noinline__ int eval(const TLane& st, int i, int e, int64_t B, int64_t* cost) const {
        const int base = tile_base(st.j), cnt = (st.j + 1) * (st.j + 2) / 2;
        int64_t best = kInf;
        for (int o = 0; o < cnt; ++o) {
            const uint8_t cd = t.code[st.g * kTileSlots + base + o];
            if ((cd & 0xc0) != 0x80) continue;  // not allowed, or dominated
            if (!tfits(t, st, i, e, (cd >> 4) & 3)) continue;
            const int64_t* P = t.Pt + (size_t)(st.g * kTileSlots + base + o) * (t.L + 1);
            best = min(best, P[e] - P[i] + st.c);
        }
        if (best == kInf) return 2;
        *cost = best;
        return best <= B ? 0 : 1;
    }
};

// The first guess of B* (warp-collective, after the memory probe found a
// split): each stage at its fastest allowed tiling's average layer cost,
// with its P2P and its memory run from layer 0 without EDP copies (the
// longest any tiling allows); not inlined, so the probe loop around it
// keeps its registers.
__device__ __noinline__ int64_t tiled_guess(const uint8_t* code, const int64_t* Pt, const longlong2* SA, int g, int j,
                                            int64_t c, int64_t cap, int64_t f, bool live, int S, int L, int64_t hi) {
    float rq = 0.f, cf = 0.f, mr = 0.f;
    if (live) {
        const int base = tile_base(j), cnt = (j + 1) * (j + 2) / 2;
        int64_t all = kInf;
        for (int o = 0; o < cnt; ++o)
            if ((code[g * kTileSlots + base + o] & 0xc0) == 0x80)
                all = min(all, Pt[(size_t)(g * kTileSlots + base + o) * (L + 1) + L]);
        rq = all > 0 && all < kInf ? (float)L / u64_to_float((uint64_t)all) : 0.f;
        cf = u64_to_float((uint64_t)c);
        int r0 = 0, r1 = L;  // the largest run [0, r) within memory, no EDP copies
        while (r0 < r1) {
            const int mid = (r0 + r1 + 1) >> 1;
            const longlong2 sm = SA[mid];
            if ((sm.x - SA[0].x) + f * (sm.y - SA[0].y) <= cap) r0 = mid;
            else r1 = mid - 1;
        }
        mr = (float)r0;
    }
    return wp::first_guess(rq, cf, mr, S, L, hi);
}

// element k of a 4-entry register array (k in [0, 3])
template <class T>
__device__ __forceinline__ T pick4(const T (&v)[4], int k) {
    return k == 0 ? v[0] : k == 1 ? v[1] : k == 2 ? v[2] : v[3];
}

__global__ void __launch_bounds__(kTBlock, 3) tiled_search_kernel(PriceArgs a, TiledArgs ta) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    if (!wp::load_image(smem, ta.timg, ta.tl.bytes, &bar, a.err)) return;
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
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    wp::WarpArea& wa = reinterpret_cast<wp::WarpArea*>(smem + ((y.bytes + 127u) & ~127u))[warp];
    unsigned long long checks = 0;
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    // each warp prices its own first entry, then the next untaken one
    // whenever it is free
    const int64_t first = (int64_t)gridDim.x * kTWarps;
    auto take = [&]() {
        int e = 0;
        if (lane == 0) e = atomicAdd(a.wl_count + kWlTakeWarp, 1);
        return first + __shfl_sync(wp::kFull, e, 0);
    };
    for (int64_t p = (int64_t)blockIdx.x * kTWarps + warp; p < count; p = take()) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        if (!in_range(c, a.n, a.err) || !in_range(S - 1, kMaxStages, a.err)) continue;
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        const bool live = lane < S;
        // this lane's stage (lane < S)
        const int code = a.wl_code[p * kMaxStages + lane];
        const int nxt = __shfl_down_sync(wp::kFull, code, 1);
        TLane mine;
        mine.g = code & 7;
        mine.j = (code >> 3) & 3;
        mine.cap = t.mem[mine.g] << mine.j;
        mine.f = live ? min(S - lane, M) : 0;
        mine.c = 0;
        if (lane + 1 < S) {
            const int h = nxt & 7, jn = (nxt >> 3) & 3;
            const int same = (mine.g == h) && ((1 << mine.j) + (1 << jn) <= t.maxn[mine.g]);
            mine.c = t.p2p[(mine.g * 8 + h) * 2 + same];
        }
        const TiledCheck check{t, mine};
        // one probe call site (the probe is large): phase 0 the memory-only
        // probe (OOM, else a feasible upper bound), phase 1 the threshold
        // search galloping from the snapped bounds, phase 2 the probe at B*
        // whose sets give the split
        int64_t Bhi = 0, Blo = 0, B = kInf, step = 1;
        bool lo_known = false, hi_known = false, oom = false;
        int phase = 0, it = 0;
        while (true) {
            int64_t hi, lo;
            const bool feas = wp::probe(check, S, L, B, wa, hi, lo, checks);
            if (phase == 0) {
                if (!feas) {
                    oom = true;
                    break;
                }
                Bhi = hi;
                B = tiled_guess(t.code, t.Pt, t.SA, mine.g, mine.j, mine.c, mine.cap, mine.f, lane < S, S, L, Bhi);
                phase = 1;
            } else if (phase == 1) {
                if (feas) {
                    Bhi = hi;
                    hi_known = true;
                } else {
                    Blo = lo;
                    lo_known = true;
                }
                if (!lo_known) {
                    B = Bhi - step;
                    step *= 2;
                } else if (!hi_known) {
                    B = Blo + step - 1;
                    step *= 2;
                } else {
                    B = Blo + (Bhi - Blo) / 2;
                }
                if (++it > kMaxIters) {
                    if (lane == 0) atomicOr(a.err, kErrSearchBound);
                    Blo = Bhi;
                }
            } else {
                if (!feas && lane == 0) atomicOr(a.err, kErrInternal);
                break;
            }
            if (phase == 1 && Blo >= Bhi) {
                phase = 2;
                B = Bhi;
            } else if (phase == 1) {
                B = min(max(B, Blo), Bhi - 1);
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
        if (!wp::walk(wa, S, L) && lane == 0) atomicOr(a.err, kErrInternal);

        // ---- re-selection on the split, one lane per stage: per EDP
        //      exponent m the fastest fitting tiling with EDP exponent <= m
        //      (bt, its code bc and exponent bl) and the gradient term gg
        int64_t bt[4] = {kInf, kInf, kInf, kInf}, gg[4] = {0, 0, 0, 0};
        int bc[4] = {0, 0, 0, 0}, bl[4] = {0, 0, 0, 0};
        int hasld = 0, a1 = 0;
        if (live) {
            const int i0 = wa.A[lane], i1 = wa.A[lane + 1];
            a1 = i1;
            const int64_t Ge = t.PE[i1] - t.PE[i0];
            const int64_t Gd = (t.PB[i1] - t.PB[i0]) - Ge;
            const int64_t bw = (n == 1 && (1 << mine.j) <= t.maxn[mine.g]) ? t.intra[mine.g] : t.inter[mine.g];
            const int base = tile_base(mine.j);
            int64_t best = kInf;
            int bcode = 0, bld = 0, o = 0;
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                if (m > mine.j) break;
                const u128 vol = (u128)(n - 1) * (u128)Gd + (u128)((n << m) - 1) * (u128)Ge;
                int64_t gv = 0;
                if (vol != 0) {
                    bool okd = true;
                    gv = (int64_t)ceil_div_u128((u128)2 * vol * 1000000000u, (uint64_t)(n << mine.j) * (uint64_t)bw,
                                                &okd);
                    if (!okd) atomicOr(a.err, kErrInternal);
                }
                gg[m] = gv;
                // the slots of EDP exponent m: ETP exponent 0 .. j - m
                for (int lt = 0; lt <= mine.j - m; ++lt, ++o) {
                    const uint8_t cd = t.code[mine.g * kTileSlots + base + o];
                    if ((cd & 0xc0) != 0x80 || !tfits(t, mine, i0, i1, m)) continue;
                    hasld |= 1 << m;
                    const int64_t* P = t.Pt + (size_t)(mine.g * kTileSlots + base + o) * (L + 1);
                    const int64_t v = P[i1] - P[i0] + mine.c;
                    if (v < best) {
                        best = v;
                        bcode = cd & 15;
                        bld = m;
                    }
                }
                bt[m] = best;
                bc[m] = bcode;
                bl[m] = bld;
            }
        }
        int64_t bestT = kInf, bestY = 0, bestB = 0;
        int mycode = 0;
        bool found = false;
        for (int ys = 0; ys < S; ++ys) {
            const int hy = __shfl_sync(wp::kFull, hasld, ys);
#pragma unroll
            for (int my = 0; my < 4; ++my) {
                const int64_t Y = __shfl_sync(wp::kFull, gg[my], ys);
                if (!((hy >> my) & 1)) continue;
                // each stage: its fastest fitting tiling with g <= Y (the
                // admissible EDP exponents are a prefix: g grows with d)
                int mm = -1;
#pragma unroll
                for (int m = 0; m < 4; ++m)
                    if (m <= mine.j && gg[m] <= Y) mm = m;
                const int64_t tv = mm >= 0 ? pick4(bt, mm) : kInf;
                const bool bad = live && tv == kInf;
                if (__any_sync(wp::kFull, bad)) continue;
                const int64_t gsel = live ? pick4(gg, pick4(bl, mm)) : 0;
                const int64_t tm = wp::wmax64(live ? tv : 0), tsum = wp::wsum64(live ? tv : 0);
                const int64_t gm = wp::wmax64(gsel);
                const int64_t T = (int64_t)(M - 1) * tm + tsum + gm;
                if (!found || T < bestT || (T == bestT && Y < bestY)) {
                    found = true;
                    bestT = T;
                    bestY = Y;
                    bestB = tm;
                    mycode = live ? pick4(bc, mm) : 0;
                }
            }
        }
        if (lane == 0) {
            if (!found) atomicOr(a.err, kErrInternal);
            a.T[c] = found ? bestT : -1;
            a.wl_T[p] = found ? bestT : -1;
            a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
            a.B[c] = bestB;
            a.ndp[c] = (uint16_t)n;
            a.status[c] = HEDDLE_CAND_OK;
        }
        if (ta.tiling && live) ta.tiling[(int64_t)lane * ta.tstride + c] = (uint8_t)mycode;
        if (a.bounds) {
            a.bounds[(int64_t)(lane + 1) * a.bstride + c] = live ? (uint8_t)a1 : 0;
            if (lane == 0) a.bounds[c] = 0;
        }
        __syncwarp();  // wa is reused by the next entry
    }
    (void)checks;
}

}  // namespace

cudaError_t launch_tiled_tables(const TiledTableArgs& a, cudaStream_t st) {
    tiled_tables_kernel<<<1, kTabThreads, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_tiled_search(const PriceArgs& a, const TiledArgs& t, int num_sms, cudaStream_t st) {
    const size_t smem = ((t.tl.bytes + 127u) & ~127u) + sizeof(wp::WarpArea) * kTWarps;
    int per_sm = 0;
    const cudaError_t e = resident_blocks(reinterpret_cast<const void*>(&tiled_search_kernel), kTBlock, smem, &per_sm);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: one warp per entry,
    // at most one wave
    const int64_t need = (a.n + kTWarps - 1) / kTWarps;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    tiled_search_kernel<<<grid, kTBlock, smem, st>>>(a, t);
    return cudaGetLastError();
}

}  // namespace hd
