// heddle_price.cu -- pricing kernel: decode + validate (§5.1 masks), DP
// degree (§5.3 packing), PartitionLayers (min-max split, §3.1 listing, with
// the memory validation of §5.2) and Evaluate (1F1B iteration time, §5.3).
//
// Two launches per batch.  The screen kernel (one thread per candidate,
// coalesced) decodes and validates every candidate, computes its DP degree
// and decides memory feasibility from a table of the longest run of layers
// each (type, degree, in-flight count) can hold: if the runs of the stages
// sum below L no split fits (OOM); when every layer has the same state and
// activation bytes, runs summing to at least L (each at least one layer)
// also guarantee a split that fits, so no memory-only probe is needed.
// Candidates that still need PartitionLayers are compacted into a worklist;
// the search kernel (one thread per worklist entry, persistent grid) runs the
// threshold search on them, so cheap and expensive candidates do not share
// warps.  Each search CTA first copies the cost-table image into shared
// memory with one bulk TMA copy (cp.async.bulk, completion on an mbarrier).
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
// itself a stage cost.  The C sets of the probe at B* give the canonical
// split directly: a_{s+1} = min { j in C_{s+1} : j > a_s }, the smallest
// boundary vector attaining B* (the feasible splits form a lattice under
// componentwise min).
//
// Memory layout: the tables live in shared memory; per-thread state that is
// indexed by a stage or a set word (stage codes, the forward bounds U, the
// two position sets the backward pass reads and writes) lives in shared
// memory interleaved by thread (element e of thread t at [e * kBlock + t]),
// so each lane hits its own bank whatever index it uses.  A stage's
// parameters are held in registers while that stage is swept.  Only the last
// probe writes its sets to local memory, for the canonical split.

#include <algorithm>

#include "heddle_tiled.cuh"

namespace hd {
namespace {

constexpr int kBlock = 256;
constexpr int kWords = 8;  // 256-bit position sets (L <= 255)
constexpr int kCodeWords = kMaxStages / 4;
constexpr int kMaxIters = 256;
constexpr long long kStageWaitSpins = 1 << 22;

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
    const int32_t* maxn;
    const int32_t* pow2;
    const int32_t* gpus;
    const int32_t* cap;
    const uint8_t* win;
    int L, NT;
};

// Per-thread views into the interleaved shared-memory arrays (already offset
// by the thread index; element e at [e * kBlock]).
struct Lane {
    uint32_t* code4;  // [kCodeWords] four stage codes per word
    uint8_t* U;       // [kMaxStages + 1]
    uint32_t* C[2];   // [words] two position sets
};

__device__ __forceinline__ int stage_code(const Lane& ln, int s) {
    return (ln.code4[(s >> 2) * kBlock] >> ((s & 3) * 8)) & 0xff;
}

// Parameters of one stage, held in registers while the stage is swept.
struct Stage {
    const int64_t* P;  // prefix row of the stage's (type, degree)
    int64_t c;         // P2P to the next stage
    int64_t capk;      // memory per GPU x group size
    int32_t f;         // in-flight microbatches
};

__device__ __forceinline__ Stage load_stage(const Tabs& t, const Lane& ln, int s, int S, int M) {
    const int code = stage_code(ln, s);
    const int g = code & 7, j = (code >> 3) & 3;
    Stage st;
    st.P = t.P + (g * 4 + j) * (t.L + 1);
    st.capk = t.mem[g] << j;
    st.f = min(S - s, M);
    st.c = 0;
    if (s + 1 < S) {
        const int cn = stage_code(ln, s + 1);
        const int h = cn & 7, jn = (cn >> 3) & 3;
        const int same = (g == h) && ((1 << j) + (1 << jn) <= t.maxn[g]);
        st.c = t.p2p[(g * 8 + h) * 2 + same];
    }
    return st;
}

// Snapping values of the current probe.
struct Snap {
    int64_t hi, lo;
    unsigned long long checks;
};

// Interval [i, j) on stage st with cached prefix values of both ends:
// 0 fits (cost <= B), 1 too slow, 2 out of memory.
__device__ __forceinline__ int judge(const Stage& st, int64_t Pi, longlong2 Si, int64_t Pj, longlong2 Sj,
                                     int64_t B, Snap& sn) {
    ++sn.checks;
    const int64_t mem = (Sj.x - Si.x) + (int64_t)st.f * (Sj.y - Si.y);
    if (mem > st.capk) return 2;
    const int64_t cost = Pj - Pi + st.c;
    if (cost <= B) {
        sn.hi = max(sn.hi, cost);
        return 0;
    }
    sn.lo = min(sn.lo, cost);
    return 1;
}

__device__ __forceinline__ uint32_t word(const uint32_t* C, int w) { return C[w * kBlock]; }

// largest set position in [lo, i], -1 if none
__device__ __forceinline__ int prev_set(const uint32_t* C, int i, int lo) {
    if (i < lo) return -1;
    int wd = i >> 5;
    uint32_t m = word(C, wd) & (0xffffffffu >> (31 - (i & 31)));
    while (m == 0) {
        if (--wd < (lo >> 5)) return -1;
        m = word(C, wd);
    }
    const int x = (wd << 5) + 31 - __clz(m);
    return x >= lo ? x : -1;
}

// smallest set position in [i, hi], -1 if none
__device__ __forceinline__ int next_set(const uint32_t* C, int i, int hi) {
    if (i > hi) return -1;
    int wd = i >> 5;
    uint32_t m = word(C, wd) & (0xffffffffu << (i & 31));
    while (m == 0) {
        if (++wd > (hi >> 5)) return -1;
        m = word(C, wd);
    }
    const int x = (wd << 5) + __ffs(m) - 1;
    return x <= hi ? x : -1;
}

// Sets of the probe at B*, kept for the canonical split (local memory).
struct Final {
    uint32_t w[kMaxStages + 1][kWords];
    int16_t lo[kMaxStages + 1], hi[kMaxStages + 1];
};

template <bool kStore>
__device__ bool probe(const Tabs& t, const Lane& ln, int S, int M, int64_t B, Snap& sn, Final* fin) {
    const int L = t.L;
    sn.hi = -1;
    sn.lo = kInf;
    // forward upper bounds on the boundaries
    int u = 0;
    ln.U[0] = 0;
    for (int s = 0; s + 1 < S; ++s) {
        const Stage st = load_stage(t, ln, s, S, M);
        const int64_t Pi = st.P[u];
        const longlong2 Si = t.SA[u];
        const int lim = L - (S - 1 - s);
        int j = u;
        while (j + 1 <= lim) {
            if (judge(st, Pi, Si, st.P[j + 1], t.SA[j + 1], B, sn) != 0) break;
            ++j;
        }
        if (j < s + 1) return false;
        u = j;
        ln.U[(s + 1) * kBlock] = (uint8_t)j;
    }
    // backward feasible-start sets: C_S = {L}, then stages S-1 .. 1
    int cur = 0;
    {
        uint32_t* CS = ln.C[cur];
        for (int wd = S >> 5; wd < (L >> 5); ++wd) CS[wd * kBlock] = 0;
        CS[(L >> 5) * kBlock] = 1u << (L & 31);
    }
    int nmin = L, nmax = L;
    for (int s = S - 1; s >= 1; --s) {
        const uint32_t* Cn = ln.C[cur];
        uint32_t* Cs = ln.C[cur ^ 1];
        const int top = min((int)ln.U[s * kBlock], nmax - 1);
        if (top < s) return false;
        const Stage st = load_stage(t, ln, s, S, M);
        for (int wd = s >> 5; wd <= (top >> 5); ++wd) Cs[wd * kBlock] = 0;
        int succ = next_set(Cn, top + 1, nmax);
        int64_t Pj = st.P[succ];
        longlong2 Sj = t.SA[succ];
        int i = top, hi = -1, lo = -1;
        int accw = top >> 5;  // word of Cs being assembled
        uint32_t acc = 0;
        int cnw = -1;         // cached word of Cn
        uint32_t cn = 0;
        while (i >= s) {
            const int64_t Pi = st.P[i];
            const longlong2 Si = t.SA[i];
            if (judge(st, Pi, Si, Pj, Sj, B, sn) == 0) {
                if ((i >> 5) != accw) {
                    Cs[accw * kBlock] = acc;
                    accw = i >> 5;
                    acc = 0;
                }
                acc |= 1u << (i & 31);
                if (hi < 0) hi = i;
                lo = i;
                if (i >= nmin) {
                    if ((i >> 5) != cnw) {
                        cnw = i >> 5;
                        cn = word(Cn, cnw);
                    }
                    if ((cn >> (i & 31)) & 1u) {
                        succ = i;
                        Pj = Pi;
                        Sj = Si;
                    }
                }
                --i;
            } else {
                const int j2 = prev_set(Cn, i, nmin);
                if (j2 < 0) break;
                i = j2 - 1;
                succ = j2;
                Pj = st.P[j2];
                Sj = t.SA[j2];
            }
        }
        Cs[accw * kBlock] = acc;
        if (hi < 0) return false;
        if (kStore) {
            for (int wd = lo >> 5; wd <= (hi >> 5); ++wd) fin->w[s][wd] = Cs[wd * kBlock];
            fin->lo[s] = (int16_t)lo;
            fin->hi[s] = (int16_t)hi;
        }
        cur ^= 1;
        nmin = lo;
        nmax = hi;
    }
    const Stage st0 = load_stage(t, ln, 0, S, M);
    return judge(st0, st0.P[0], t.SA[0], st0.P[nmin], t.SA[nmin], B, sn) == 0;
}

__device__ void bind_tables(Tabs& t, const unsigned char* img, const Layout& y) {
    t.P = reinterpret_cast<const int64_t*>(img + y.offP);
    t.SA = reinterpret_cast<const longlong2*>(img + y.offSA);
    t.PB = reinterpret_cast<const int64_t*>(img + y.offPB);
    t.p2p = reinterpret_cast<const int64_t*>(img + y.offP2P);
    t.mem = reinterpret_cast<const int64_t*>(img + y.offMem);
    t.inter = reinterpret_cast<const int64_t*>(img + y.offInter);
    t.maxn = reinterpret_cast<const int32_t*>(img + y.offMaxN);
    t.pow2 = reinterpret_cast<const int32_t*>(img + y.offPow2);
    t.gpus = reinterpret_cast<const int32_t*>(img + y.offGpus);
    t.cap = reinterpret_cast<const int32_t*>(img + y.offCap);
    t.win = img + y.offWin;
    t.L = y.L;
    t.NT = y.NT;
}

__device__ __forceinline__ void write_rejected(const PriceArgs& a, int64_t c, int status, int64_t n) {
    a.T[c] = -1;
    a.B[c] = -1;
    a.ndp[c] = (uint16_t)(status == HEDDLE_CAND_OOM ? n : 0);
    a.status[c] = (uint8_t)status;
    if (a.bounds)
        for (int s = 0; s <= kMaxStages; ++s) a.bounds[(int64_t)s * a.bstride + c] = 0;
}

constexpr int kScreenBlock = 256;

// floor(a / d) for 0 <= a < 2^16 and 1 <= d <= 256 as (a 2^8) ceil(2^24 / d)
// / 2^32: the error a (ceil(2^24/d) - 2^24/d) / 2^24 < 2^-8 stays below 1/d,
// the smallest distance from a / d up to the next integer
__device__ __forceinline__ uint32_t div_small(uint32_t a, uint32_t d, const uint32_t* magic) {
    return __umulhi(a << 8, magic[d]);
}

// Per stage byte: bit 31 inadmissible; bits 24-26 type; bits 16-21 the bit
// position of the stage's GPUs in the type's demand word (degree bits +
// 16 * unit class); bits 0-10 the row (type, degree) of the run table.
__device__ __forceinline__ uint32_t stage_desc(int b, const Layout& y, const unsigned char* img, int moe) {
    const int32_t* gmaxn = reinterpret_cast<const int32_t*>(img + y.offMaxN);
    const int32_t* gpow2 = reinterpret_cast<const int32_t*>(img + y.offPow2);
    const int32_t* ggpus = reinterpret_cast<const int32_t*>(img + y.offGpus);
    const int g = b & 7, j = (b >> 3) & 3;
    if ((b >> 5) != 0 || g >= y.NT || ggpus[g] <= 0 || (!moe && (1 << j) > gmaxn[g])) return 1u << 31;
    const int unit = (1 << j) <= gmaxn[g] ? (1 << j) : gpow2[g];
    const int uc = 31 - __clz(unit);
    return ((uint32_t)g << 24) | ((uint32_t)(j + 16 * uc) << 16) | (uint32_t)((g * 4 + j) * 33);
}

// Steps 1-2 and the memory screen for every candidate of the batch.  Each
// CTA takes 256 consecutive candidates at a time: their S and M, and the
// code planes up to the largest S among them, are copied to shared memory
// (16-byte vector copies when the planes are aligned), the candidates are
// counting-sorted by S, and thread i screens the i-th of that order, so the
// lanes of a warp run stage loops of nearly equal length.
__global__ void __launch_bounds__(kScreenBlock) screen_kernel(PriceArgs a) {
    __shared__ uint32_t desc[256];
    __shared__ uint8_t win[8 * 4 * 33];
    __shared__ uint32_t cap[8 * 4];
    __shared__ uint32_t magic[257];
    __shared__ uint64_t dem[8 * kScreenBlock];  // per-thread GPUs per unit class, 4 x 16 bits per type
    __shared__ __align__(16) uint8_t tile[kMaxStages * kScreenBlock];  // [stage][candidate of the slice]
    __shared__ uint8_t sS[kScreenBlock];
    __shared__ uint16_t sM[kScreenBlock];
    __shared__ uint8_t order[kScreenBlock];
    __shared__ int bins[kMaxStages + 3];
    __shared__ int smax;
    const Layout& y = a.lay;
    const int L = y.L;
    {
        const int32_t* gcap = reinterpret_cast<const int32_t*>(a.img + y.offCap);
        for (int i = threadIdx.x; i < 256; i += blockDim.x) desc[i] = stage_desc(i, y, a.img, a.moe);
        for (int i = threadIdx.x; i < 32; i += blockDim.x) cap[i] = (uint32_t)gcap[i];
        for (int i = threadIdx.x; i < 8 * 4 * 33; i += blockDim.x) win[i] = a.img[y.offWin + i];
        for (int i = threadIdx.x; i < 257; i += blockDim.x) magic[i] = i >= 1 ? ((1u << 24) + i - 1) / i : 0;
    }
    const bool memuni = reinterpret_cast<const int32_t*>(a.img + y.offModel)[0] != 0;
    const int s_lim = min(min(kMaxStages, a.s_max), L);
    const bool vec16 = ((reinterpret_cast<uintptr_t>(a.code) | (uintptr_t)a.stride) & 15) == 0;
    uint64_t* mydem = dem + threadIdx.x;
    const int lane = threadIdx.x & 31;
    for (int64_t c0 = (int64_t)blockIdx.x * kScreenBlock; c0 < a.n; c0 += (int64_t)gridDim.x * kScreenBlock) {
        const int nloc = (int)min((int64_t)kScreenBlock, a.n - c0);
        // ---- S and M of the slice; S = 0 marks a depth or M outside range,
        //      bin kMaxStages + 1 the padding past the batch
        int key = kMaxStages + 1;
        if (threadIdx.x < nloc) {
            const int S = a.S[c0 + threadIdx.x];
            // at micro-batch size 2^shift a replica runs M / 2^shift
            // micro-batches; a size that does not divide M is not priced
            const int Mraw = a.M[c0 + threadIdx.x];
            const int M = Mraw >> a.mbs_shift;
            const bool whole = (Mraw & ((1 << a.mbs_shift) - 1)) == 0;
            key = (S >= 1 && S <= s_lim && M >= 1 && whole) ? S : 0;
            sS[threadIdx.x] = (uint8_t)key;
            sM[threadIdx.x] = (uint16_t)M;
        }
        if (threadIdx.x < kMaxStages + 3) bins[threadIdx.x] = 0;
        if (threadIdx.x == 0) smax = 0;
        __syncthreads();
        atomicAdd(&bins[key], 1);
        if (key <= kMaxStages && key > 0) atomicMax(&smax, key);
        __syncthreads();
        // ---- code planes 0 .. smax-1 of the slice into the tile
        const int np = smax;
        if (vec16 && nloc == kScreenBlock) {
            for (int i = threadIdx.x; i < np * (kScreenBlock / 16); i += kScreenBlock) {
                const int s = i / (kScreenBlock / 16), o = (i % (kScreenBlock / 16)) * 16;
                *reinterpret_cast<uint4*>(tile + s * kScreenBlock + o) =
                    __ldg(reinterpret_cast<const uint4*>(a.code + (int64_t)s * a.stride + c0 + o));
            }
        } else {
            for (int i = threadIdx.x; i < np * kScreenBlock; i += kScreenBlock) {
                const int s = i / kScreenBlock, o = i % kScreenBlock;
                if (o < nloc) tile[i] = __ldg(a.code + (int64_t)s * a.stride + c0 + o);
            }
        }
        if (threadIdx.x < 32) {
            // exclusive scan of bins 0..33 by one warp (lane l: bin l, lane
            // 31 also bins 32 and 33)
            const int v = bins[lane];
            int x = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y2 = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y2;
            }
            const int b32 = bins[32], b33 = bins[33];
            __syncwarp();
            bins[lane] = x - v;
            if (lane == 31) {
                bins[32] = x;
                bins[33] = x + b32;
            }
            (void)b33;
        }
        __syncthreads();
        order[atomicAdd(&bins[key], 1)] = (uint8_t)threadIdx.x;
        __syncthreads();
        const int ci = order[threadIdx.x];
        const bool live = threadIdx.x < nloc;  // padding sorts last
        const int64_t c = c0 + ci;
        int S = 0, M = 0, status = HEDDLE_CAND_INVALID;
        int64_t n = 0;
        if (live) {
            S = sS[ci];
            M = sM[ci];
            if (S > 0) {
#pragma unroll
                for (int g = 0; g < 8; ++g) mydem[g * kScreenBlock] = 0;
                uint32_t bad = 0, present = 0;
                int run_sum = 0, run_min = 255;
                const uint8_t* col = tile + ci;
                for (int s = 0; s < S; ++s) {
                    const uint32_t d = desc[col[s * kScreenBlock]];
                    bad |= d;
                    const int g = (d >> 24) & 7;
                    present |= 1u << g;
                    mydem[g * kScreenBlock] += 1ull << ((d >> 16) & 63);
                    const int w = win[(d & 0x7ff) + min(S - s, M)];
                    run_sum += w;
                    run_min = min(run_min, w);
                }
                if (bad >> 31) {
                    status = HEDDLE_CAND_INVALID;
                } else {
                    // n = min over (type, class e) of capacity / GPUs in units
                    // >= 2^e; a class with no group of its own size is
                    // dominated by the class above it
                    uint32_t nn = 0xffffffffu;
                    while (present) {
                        const int g = __ffs(present) - 1;
                        present &= present - 1;
                        const uint64_t v = mydem[g * kScreenBlock];
                        uint32_t dsum = 0;
#pragma unroll
                        for (int e = 3; e >= 0; --e) {
                            const uint32_t f = (uint32_t)(v >> (16 * e)) & 0xffffu;
                            dsum += f;
                            if (f) nn = min(nn, div_small(cap[g * 4 + e], dsum, magic));
                        }
                    }
                    n = nn;
                    if (n == 0)
                        status = HEDDLE_CAND_NO_FIT;
                    else if (run_min < 1 || run_sum < L)
                        status = HEDDLE_CAND_OOM;
                    else
                        status = HEDDLE_CAND_OK;
                }
            }
            if (status != HEDDLE_CAND_OK) write_rejected(a, c, status, n);
        }
        // compact the candidates that need the search (one atomic per warp)
        const bool take = live && status == HEDDLE_CAND_OK;
        const unsigned mask = __ballot_sync(0xffffffffu, take);
        if (mask) {
            int base = 0;
            if (lane == 0) base = atomicAdd(a.wl_count, __popc(mask));
            base = __shfl_sync(0xffffffffu, base, 0);
            const int p = base + __popc(mask & ((1u << lane) - 1));
            if (take) {
                if (p < a.wl_cap) {
                    a.wl_idx[p] = (int32_t)c;
                    a.wl_n[p] = (uint16_t)n;
                    a.wl_M[p] = (uint16_t)M;
                    a.wl_S[p] = (uint8_t)S;
                    a.wl_memok[p] = memuni ? 1 : 0;
                } else {
                    atomicOr(a.err, kErrInternal);
                }
            }
            if (a.uniform && take) {
                // the entry in its depth's bucket, for the equal-layer
                // search's order by decreasing depth
                const unsigned same = __match_any_sync(mask, S);
                const int leader = __ffs(same) - 1;
                int b0 = 0;
                if (lane == leader) b0 = atomicAdd(a.wl_count + 1 + S, __popc(same));
                const int bpos = __shfl_sync(same, b0, leader) + __popc(same & ((1u << lane) - 1));
                if (p < a.wl_cap && bpos < a.wl_cap) a.wl_bucket[(int64_t)(S - 1) * a.wl_cap + bpos] = p;
            }
            // each taken candidate's row of 32 stage bytes, written by the
            // whole warp (lane = stage; zero past its depth)
            for (unsigned m = mask; m; m &= m - 1) {
                const int src = __ffs(m) - 1;
                const int pc = __shfl_sync(0xffffffffu, p, src);
                const int cc = __shfl_sync(0xffffffffu, ci, src);
                const int Sc = __shfl_sync(0xffffffffu, S, src);
                if (pc < a.wl_cap)
                    a.wl_code[(int64_t)pc * kMaxStages + lane] = lane < Sc ? tile[lane * kScreenBlock + cc] : 0;
            }
        }
        __syncthreads();  // the tile, S, M and order are reused by the next slice
    }
}

// Steps 3-4 for every worklist entry.
template <bool kCount>
__global__ void __launch_bounds__(kBlock) search_kernel(PriceArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    if (!stage_tables(smem, a.img, a.lay.bytes, &bar, a.err)) return;

    const Layout& y = a.lay;
    Tabs t;
    bind_tables(t, smem, y);
    const int L = y.L;
    const int W = (L >> 5) + 1;

    // per-thread interleaved arrays after the table image
    uint32_t* lane_words = reinterpret_cast<uint32_t*>(smem + y.bytes);
    Lane ln;
    ln.code4 = lane_words + threadIdx.x;
    ln.C[0] = lane_words + kCodeWords * kBlock + threadIdx.x;
    ln.C[1] = ln.C[0] + W * kBlock;
    ln.U = reinterpret_cast<uint8_t*>(lane_words + (kCodeWords + 2 * W) * kBlock) + threadIdx.x;

    Snap sn;
    sn.checks = 0;
    unsigned long long probes = 0, priced = 0;
    Final fin;

    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < count; p += stride) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        const bool memok = a.wl_memok[p] != 0;
        {
            // the entry's row of stage bytes, 16 bytes at a time
            const uint4* row = reinterpret_cast<const uint4*>(a.wl_code + p * kMaxStages);
            const uint4 lo = __ldg(row);
            ln.code4[0 * kBlock] = lo.x;
            ln.code4[1 * kBlock] = lo.y;
            ln.code4[2 * kBlock] = lo.z;
            ln.code4[3 * kBlock] = lo.w;
            if (S > 16) {
                const uint4 hi = __ldg(row + 1);
                ln.code4[4 * kBlock] = hi.x;
                ln.code4[5 * kBlock] = hi.y;
                ln.code4[6 * kBlock] = hi.z;
                ln.code4[7 * kBlock] = hi.w;
            }
        }
        if (kCount) ++priced;
        // an upper bound that is feasible whenever memory is: every stage
        // cost of every interval is at most max_s (P_s[L] + c_s)
        int64_t hi = 0;
        float inv = 0.f, cw = 0.f;
        for (int s = 0; s < S; ++s) {
            const Stage st = load_stage(t, ln, s, S, M);
            hi = max(hi, st.P[L] + st.c);
            const float tot = u64_to_float(st.P[L]) + 1.0f;
            inv += 1.0f / tot;
            cw += u64_to_float(st.c) / tot;
        }
        if (!memok) {
            // memory-only probe decides OOM and gives a tighter upper bound
            if (kCount) ++probes;
            if (!probe<false>(t, ln, S, M, kInf, sn, nullptr)) {
                write_rejected(a, c, HEDDLE_CAND_OOM, n);
                a.wl_T[p] = -1;
                continue;
            }
            hi = sn.hi;
        }
        // ---- PartitionLayers: threshold search from the balanced guess
        int64_t lo = 0;
        bool lo_known = false, hi_known = false;
        int64_t B = (int64_t)float_to_u64((1.0f + cw) / inv);
        int64_t step = max((int64_t)1, (int64_t)float_to_u64(u64_to_float(B) * (float)S / (2.0f * (float)L)));
        int it = 0;
        while (lo < hi) {
            B = min(max(B, lo), hi - 1);
            if (kCount) ++probes;
            if (probe<false>(t, ln, S, M, B, sn, nullptr)) {
                hi = sn.hi;
                hi_known = true;
            } else {
                lo = sn.lo;
                lo_known = true;
            }
            if (lo >= hi) break;
            if (!lo_known) {
                B = hi - step;  // gallop down from a feasible guess
                step *= 2;
            } else if (!hi_known) {
                B = lo + step;  // gallop up from an infeasible guess
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
        // the sets of the optimum give the canonical split
        if (kCount) ++probes;
        if (!probe<true>(t, ln, S, M, Bstar, sn, &fin)) atomicOr(a.err, kErrInternal);
        uint8_t bnd[kMaxStages + 1];
        bnd[0] = 0;
        for (int s = 0; s + 1 < S; ++s) {
            const int from = max((int)bnd[s] + 1, (int)fin.lo[s + 1]);
            int wd = from >> 5;
            uint32_t m = fin.w[s + 1][wd] & (0xffffffffu << (from & 31));
            while (m == 0 && wd < (fin.hi[s + 1] >> 5)) m = fin.w[s + 1][++wd];
            bnd[s + 1] = (uint8_t)(m ? (wd << 5) + __ffs(m) - 1 : 0);
        }
        bnd[S] = (uint8_t)L;
        // ---- Evaluate: T = (M-1) max t_s + sum t_s + max g_s
        int64_t tmax = 0, tsum = 0;
        int sg = -1;
        uint64_t bestG = 0, bestD = 1;
        for (int s = 0; s < S; ++s) {
            const Stage st = load_stage(t, ln, s, S, M);
            const int64_t ts = st.P[bnd[s + 1]] - st.P[bnd[s]] + st.c;
            tmax = max(tmax, ts);
            tsum += ts;
            if (n > 1) {
                // stage with the largest G_s / (k_s bw_s), compared exactly
                const int code = stage_code(ln, s);
                const int g = code & 7, j = (code >> 3) & 3;
                const uint64_t G = (uint64_t)(t.PB[bnd[s + 1]] - t.PB[bnd[s]]);
                const uint64_t D = (uint64_t)t.inter[g] << j;
                if (sg < 0 || (u128)G * bestD > (u128)bestG * D) {
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
            // (G < 2^50 and bandwidths < 2^40 keep n k bw below 2^64)
            const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * bestG;
            bool ok = true;
            gmax = (int64_t)ceil_div_u128(num, (uint64_t)n * bestD, &ok);
            if (!ok) atomicOr(a.err, kErrInternal);
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
        unsigned long long v0 = sn.checks, v1 = probes, v2 = priced;
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

// shared memory of the per-thread interleaved arrays
size_t lane_bytes(int L) {
    const int W = (L >> 5) + 1;
    return (size_t)kBlock * (4 * kCodeWords + 4 * 2 * W + (kMaxStages + 1));
}

template <bool kCount>
cudaError_t launch_search(const PriceArgs& a, int num_sms, cudaStream_t st) {
    const size_t smem = a.lay.bytes + lane_bytes(a.lay.L);
    cudaError_t e = cudaFuncSetAttribute(search_kernel<kCount>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, search_kernel<kCount>, kBlock, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // the worklist length is only known on the device: size for the batch
    const int64_t need = (a.n + kBlock - 1) / kBlock;
    const int grid = (int)std::min<int64_t>(need, (int64_t)num_sms * per_sm);
    search_kernel<kCount><<<grid, kBlock, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_screen(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid, int64_t* launches) {
    if (a.n <= 0) return cudaSuccess;
    if (a.n > a.wl_cap) return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(a.wl_count, 0, sizeof(int32_t) * kWlMeta, st);
    if (e != cudaSuccess) return e;
    // one wave of resident CTAs, each looping over slices
    static int screen_per_sm = 0;
    if (screen_per_sm == 0) {
        int v = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, screen_kernel, kScreenBlock, 0);
        if (e != cudaSuccess) return e;
        screen_per_sm = v > 0 ? v : 1;
    }
    const int grid =
        (int)std::min<int64_t>((a.n + kScreenBlock - 1) / kScreenBlock, (int64_t)num_sms * screen_per_sm);
    screen_kernel<<<grid, kScreenBlock, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (launches) launches[0] += 1;
    if (mid && (e = cudaEventRecord(mid, st)) != cudaSuccess) return e;
    return cudaSuccess;
}

cudaError_t launch_price(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid, int64_t* launches) {
    if (a.n <= 0) return cudaSuccess;
    cudaError_t e = launch_screen(a, num_sms, st, mid, launches);
    if (e != cudaSuccess) return e;
    if (launches) launches[1] += 1;
    if (a.split_mode) return launch_distribute(a, num_sms, st);
    if (a.uniform) return launch_eq_search(a, num_sms, st);
    return a.counters ? launch_search<true>(a, num_sms, st) : launch_search<false>(a, num_sms, st);
}

}  // namespace hd
