// heddle_distribute.cu -- the paper's own layer split as a second split mode
// (§5.3 "Layer split and DP degree"): each stage gets layers in proportion
// to its profiled speed; if that split exceeds a stage's memory, a fixed
// list of alternative splits is priced and the fastest one that fits is
// kept.  The hot path's min-max PartitionLayers replaces this rule; this
// mode prices the same candidates the paper's way so the two can be
// compared (the quality gap of the heuristic).
//
// Readings (shared with the oracle only through their statement): the speed
// of stage s is 2^40 divided by the time of all L layers on its type and
// degree, rounded down; the list is (1) in proportion to speed, (2) equal
// layer counts, (3) in proportion to the longest run of consecutive layers
// each stage's memory holds; shares are floors of L w_s / sum w with at
// least one layer per stage, missing layers to the largest remainders (the
// earlier stage on ties), surplus layers off the stage holding the most
// (the later stage on ties); the fastest is the smallest pipeline time
// (M-1) max t_s + sum t_s, the earlier alternative on ties (Algorithm 1
// splits the layers before the fill picks the DP degree, so the choice
// cannot see the gradient term).  No alternative fits: OOM.
//
// One warp per worklist entry, one lane per stage (S <= 32): every
// per-stage quantity lives in the lane's registers, and the split's sums,
// ranks, scans and maxima are warp collectives.  The screen has already
// rejected the candidates no split fits; the small tables are read through
// the L1 cache.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kDistBlock = 128;
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ int64_t warp_sum64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ int64_t warp_max64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, (int64_t)__shfl_xor_sync(kFull, v, o));
    return v;
}

// This lane's layer count when L layers go to the S live lanes in
// proportion to w (sum V > 0): floor of the exact share, at least one;
// missing layers one each to the largest remainders (the earlier stage on
// ties); surplus layers one at a time off the stage holding the most (the
// later stage on ties).
__device__ int share_count(bool live, int S, int L, int64_t w, int64_t V, int lane) {
    int64_t q = 0, rem = 0;
    if (live) {
        const int64_t share = (int64_t)L * w;
        q = share / V;
        rem = share - q * V;
    }
    int cnt = live ? (q < 1 ? 1 : (int)q) : 0;
    int total = __reduce_add_sync(kFull, (unsigned)cnt);
    if (total < L) {
        // the L - total largest remainders gain one layer
        int rank = 0;
        for (int t = 0; t < S; ++t) {
            const int64_t rt = __shfl_sync(kFull, rem, t);
            rank += (rt > rem || (rt == rem && t < lane)) ? 1 : 0;
        }
        if (live && rank < L - total) ++cnt;
    }
    while (total > L) {
        // the stage holding the most (the later one on ties) gives one up
        const int key = live && cnt > 1 ? (cnt << 8) | lane : -1;
        const int top = __reduce_max_sync(kFull, (unsigned)(key + 1)) - 1;
        if (lane == (top & 0xff)) --cnt;
        --total;
    }
    return cnt;
}

__global__ void __launch_bounds__(kDistBlock) distribute_kernel(PriceArgs a) {
    const Layout& y = a.lay;
    const int L = y.L;
    const int64_t* P = reinterpret_cast<const int64_t*>(a.img + y.offP);
    const longlong2* SA = reinterpret_cast<const longlong2*>(a.img + y.offSA);
    const int64_t* PB = reinterpret_cast<const int64_t*>(a.img + y.offPB);
    const int64_t* p2p = reinterpret_cast<const int64_t*>(a.img + y.offP2P);
    const int64_t* mem = reinterpret_cast<const int64_t*>(a.img + y.offMem);
    const int64_t* inter = reinterpret_cast<const int64_t*>(a.img + y.offInter);
    const int32_t* maxn = reinterpret_cast<const int32_t*>(a.img + y.offMaxN);
    const uint8_t* win = a.img + y.offWin;
    const int lane = threadIdx.x & 31;
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    // each warp prices its own first entry, then the next untaken one
    // whenever it is free
    const int64_t first = (int64_t)gridDim.x * (blockDim.x >> 5);
    auto take = [&]() {
        int e = 0;
        if (lane == 0) e = atomicAdd(a.wl_count + kWlTakeWarp, 1);
        return first + __shfl_sync(kFull, e, 0);
    };
    for (int64_t p = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); p < count; p = take()) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        if (!in_range(c, a.n, a.err) || !in_range(S - 1, kMaxStages, a.err)) continue;
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        const bool live = lane < S;
        // this lane's stage: cost row, P2P, memory capacity, in-flight count,
        // NIC x degree, and its weight under each alternative
        const int code = a.wl_code[p * kMaxStages + lane];
        const int nxt = __shfl_down_sync(kFull, code, 1);
        const int g = code & 7, j = (code >> 3) & 3;
        const int row = (g * 4 + j) * (L + 1);
        const int64_t capk = mem[g] << j;
        const int f = min(S - lane, M);
        const uint64_t D = (uint64_t)inter[g] << j;
        int64_t cs = 0;
        if (lane + 1 < S) {
            const int h = nxt & 7, jn = (nxt >> 3) & 3;
            const int same = (g == h) && ((1 << j) + (1 << jn) <= maxn[g]);
            cs = p2p[(g * 8 + h) * 2 + same];
        }
        int64_t w[3] = {0, 0, 0};
        if (live) {
            const int64_t all = P[row + L] - P[row];
            w[0] = all > 0 ? ((int64_t)1 << 40) / all : ((int64_t)1 << 40);
            w[1] = 1;
            w[2] = win[(g * 4 + j) * 33 + f];
        }
        bool found = false;
        int64_t bestPipe = 0, bestB = 0;
        int bestLo = 0, bestHi = 0;  // this lane's stage [bestLo, bestHi) in the chosen split
#pragma unroll
        for (int alt = 0; alt < 3; ++alt) {
            const int64_t V = warp_sum64(w[alt]);
            if (V <= 0) continue;
            const int cnt = share_count(live, S, L, w[alt], V, lane);
            // boundaries: inclusive scan of the counts
            int hi = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(kFull, hi, o);
                if (lane >= o) hi += t;
            }
            const int lo = hi - cnt;
            bool fits = true;
            int64_t t = 0;
            if (live) {
                const longlong2 a0 = SA[lo], a1 = SA[hi];
                fits = (a1.x - a0.x) + (int64_t)f * (a1.y - a0.y) <= capk;
                t = P[row + hi] - P[row + lo] + cs;
            }
            if (!__all_sync(kFull, fits)) continue;
            // the pipeline time of this split decides between alternatives
            const int64_t tmax = warp_max64(t), tsum = warp_sum64(t);
            const int64_t pipe = (int64_t)(M - 1) * tmax + tsum;
            if (!found || pipe < bestPipe) {
                found = true;
                bestPipe = pipe;
                bestB = tmax;
                bestLo = lo;
                bestHi = hi;
            }
        }
        int64_t T = bestPipe;
        if (found && n > 1) {
            // Evaluate adds the gradient term: the stage with the largest
            // G_s / (k_s bw_s), compared exactly, then ceil(2(n-1) G 1e9 / (n k bw))
            uint64_t G = live ? (uint64_t)(PB[bestHi] - PB[bestLo]) : 0;
            uint64_t Dd = live ? D : 1;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const uint64_t G2 = __shfl_xor_sync(kFull, G, o), D2 = __shfl_xor_sync(kFull, Dd, o);
                if ((u128)G2 * Dd > (u128)G * D2) {
                    G = G2;
                    Dd = D2;
                }
            }
            const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * G;
            bool ok = true;
            T += (int64_t)ceil_div_u128(num, (uint64_t)n * Dd, &ok);
            if (!ok && lane == 0) atomicOr(a.err, kErrInternal);
        }
        if (lane == 0) {
            if (found) {
                a.T[c] = T;
                a.B[c] = bestB;
                a.status[c] = HEDDLE_CAND_OK;
                a.wl_T[p] = T;
            } else {
                a.T[c] = -1;
                a.B[c] = -1;
                a.status[c] = HEDDLE_CAND_OOM;
                a.wl_T[p] = -1;
            }
            a.ndp[c] = (uint16_t)n;  // OOM keeps the DP degree
            a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
        }
        if (a.bounds) {
            // plane s + 1 from lane s; plane 0 from lane 31 (always 0)
            const int plane = lane == 31 ? 0 : lane + 1;
            a.bounds[(int64_t)plane * a.bstride + c] = (lane != 31 && found && live) ? (uint8_t)bestHi : 0;
            if (lane == 0) a.bounds[(int64_t)kMaxStages * a.bstride + c] = (found && S == kMaxStages) ? (uint8_t)L : 0;
        }
    }
}

}  // namespace

cudaError_t launch_distribute(const PriceArgs& a, int num_sms, cudaStream_t st) {
    // one warp per entry; the worklist length is only known on the device
    const int grid = (int)std::min<int64_t>((a.n + kDistBlock / 32 - 1) / (kDistBlock / 32), (int64_t)num_sms * 16);
    distribute_kernel<<<grid, kDistBlock, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
