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
// One thread per worklist entry (the screen has already rejected the
// candidates no split fits); the small tables are read through the L1
// cache.  This is a comparison mode, not the hot path: per-stage state
// lives in local arrays.

#include <algorithm>

#include "heddle_internal.cuh"

namespace hd {
namespace {

constexpr int kDistBlock = 128;

// L layers over S stages in proportion to weights w (sum V > 0): boundaries to b.
__device__ void share_split(int S, int L, const int64_t* w, int64_t V, uint8_t* b) {
    int cnt[kMaxStages];
    int64_t rem[kMaxStages];
    int total = 0;
    for (int s = 0; s < S; ++s) {
        const int64_t share = (int64_t)L * w[s];
        const int64_t q = share / V;
        rem[s] = share - q * V;
        cnt[s] = q < 1 ? 1 : (int)q;
        total += cnt[s];
    }
    uint32_t given = 0;
    while (total < L) {
        int best = -1;
        for (int s = 0; s < S; ++s)
            if (!((given >> s) & 1u) && (best < 0 || rem[s] > rem[best])) best = s;
        given |= 1u << best;
        ++cnt[best];
        ++total;
    }
    while (total > L) {
        int best = -1;
        for (int s = 0; s < S; ++s)
            if (cnt[s] > 1 && (best < 0 || cnt[s] >= cnt[best])) best = s;
        --cnt[best];
        --total;
    }
    b[0] = 0;
    for (int s = 0; s < S; ++s) b[s + 1] = (uint8_t)(b[s] + cnt[s]);
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
    const int64_t count = min((int64_t)*a.wl_count, (int64_t)a.wl_cap);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < count; p += stride) {
        const int64_t c = a.wl_idx[p];
        const int S = a.wl_S[p];
        const int M = a.wl_M[p];
        const int64_t n = a.wl_n[p];
        uint8_t code[kMaxStages];
        {
            const uint4* row = reinterpret_cast<const uint4*>(a.wl_code + p * kMaxStages);
            const uint4 v[2] = {__ldg(row), __ldg(row + 1)};
            const uint8_t* bytes = reinterpret_cast<const uint8_t*>(v);
            for (int s = 0; s < kMaxStages; ++s) code[s] = bytes[s];
        }
        // per stage: cost row, P2P, memory capacity, in-flight count, NIC x degree
        int row[kMaxStages];
        int64_t cs[kMaxStages], capk[kMaxStages];
        int fs[kMaxStages];
        uint64_t D[kMaxStages];
        int64_t w[3][kMaxStages];
        int64_t V[3] = {0, 0, 0};
        for (int s = 0; s < S; ++s) {
            const int g = code[s] & 7, j = (code[s] >> 3) & 3;
            row[s] = (g * 4 + j) * (L + 1);
            capk[s] = mem[g] << j;
            fs[s] = min(S - s, M);
            D[s] = (uint64_t)inter[g] << j;
            cs[s] = 0;
            if (s + 1 < S) {
                const int h = code[s + 1] & 7, jn = (code[s + 1] >> 3) & 3;
                const int same = (g == h) && ((1 << j) + (1 << jn) <= maxn[g]);
                cs[s] = p2p[(g * 8 + h) * 2 + same];
            }
            const int64_t all = P[row[s] + L] - P[row[s]];
            w[0][s] = all > 0 ? ((int64_t)1 << 40) / all : ((int64_t)1 << 40);
            w[1][s] = 1;
            w[2][s] = win[(g * 4 + j) * 33 + fs[s]];
            for (int k = 0; k < 3; ++k) V[k] += w[k][s];
        }
        bool found = false;
        int64_t bestT = 0, bestB = 0, bestPipe = 0;
        uint8_t bestb[kMaxStages + 1];
        for (int alt = 0; alt < 3; ++alt) {
            if (V[alt] <= 0) continue;
            uint8_t b[kMaxStages + 1];
            share_split(S, L, w[alt], V[alt], b);
            bool fits = true;
            for (int s = 0; s < S && fits; ++s) {
                const longlong2 lo = SA[b[s]], hi = SA[b[s + 1]];
                fits = (hi.x - lo.x) + (int64_t)fs[s] * (hi.y - lo.y) <= capk[s];
            }
            if (!fits) continue;
            // the pipeline time of this split decides between alternatives
            int64_t tmax = 0, tsum = 0;
            for (int s = 0; s < S; ++s) {
                const int64_t t = P[row[s] + b[s + 1]] - P[row[s] + b[s]] + cs[s];
                tmax = max(tmax, t);
                tsum += t;
            }
            const int64_t pipe = (int64_t)(M - 1) * tmax + tsum;
            if (!found || pipe < bestPipe) {
                found = true;
                bestPipe = pipe;
                bestT = pipe;
                bestB = tmax;
                for (int s = 0; s <= S; ++s) bestb[s] = b[s];
            }
        }
        if (found && n > 1) {
            // Evaluate adds the gradient term: the stage with the largest
            // G_s / (k_s bw_s), compared exactly, then ceil(2(n-1) G 1e9 / (n k bw))
            uint64_t bestG = 0, bestD = 1;
            int sg = -1;
            for (int s = 0; s < S; ++s) {
                const uint64_t G = (uint64_t)(PB[bestb[s + 1]] - PB[bestb[s]]);
                if (sg < 0 || (u128)G * bestD > (u128)bestG * D[s]) {
                    sg = s;
                    bestG = G;
                    bestD = D[s];
                }
            }
            const u128 num = (u128)(2 * (uint64_t)(n - 1) * 1000000000ull) * bestG;
            bool ok = true;
            bestT += (int64_t)ceil_div_u128(num, (uint64_t)n * bestD, &ok);
            if (!ok) atomicOr(a.err, kErrInternal);
        }
        if (found) {
            a.T[c] = bestT;
            a.B[c] = bestB;
            a.ndp[c] = (uint16_t)n;
            a.status[c] = HEDDLE_CAND_OK;
            a.wl_T[p] = bestT;
        } else {
            a.T[c] = -1;
            a.B[c] = -1;
            a.ndp[c] = (uint16_t)n;  // OOM keeps the DP degree
            a.status[c] = HEDDLE_CAND_OOM;
            a.wl_T[p] = -1;
        }
        a.wl_nM[p] = (uint32_t)n * (uint32_t)M;
        if (a.bounds)
            for (int s = 0; s <= kMaxStages; ++s)
                a.bounds[(int64_t)s * a.bstride + c] = (found && s <= S) ? bestb[s] : 0;
    }
}

}  // namespace

cudaError_t launch_distribute(const PriceArgs& a, int num_sms, cudaStream_t st) {
    const int grid = (int)std::min<int64_t>((a.n + kDistBlock - 1) / kDistBlock, (int64_t)num_sms * 16);
    distribute_kernel<<<grid, kDistBlock, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
