// heddle_tables.cu -- cost-table build (step 0 of the pricing path).
//
// One CTA turns the cluster and model descriptions into the integer image the
// pricing kernel stages into shared memory:
//   * per (GPU type g, degree 2^j, layer l) the layer's time in whole ns --
//     the profile entry of the paper's cost model (§5.2: computation plus
//     communication of one layer per GPU type and TP degree), synthesised
//     from FLOPs and link bandwidths or taken from an explicit profile --
//     and its prefix sums over layers;
//   * prefix sums of state, activation and gradient bytes (memory validation
//     of §5.2, gradient synchronisation);
//   * per-type node statistics for the DP packing of §5.1/§5.3;
//   * the P2P constants between consecutive stages.
// Double arithmetic uses explicitly rounded intrinsics (no contraction into
// fused multiply-add) in the order the header documents.

#include <math.h>

#include "heddle_internal.cuh"

namespace hd {
namespace {

typedef unsigned __int128 u128;

constexpr int kThreads = 256;
constexpr int64_t kTableLimit = (int64_t)1 << 40;

// Nearest integer of v >= 0, halves away from zero.  v - trunc(v) is exact
// for every double below 2^52 (and zero above).
__device__ int64_t round_half_away(double v) {
    double r = trunc(v);
    if (__dsub_rn(v, r) >= 0.5) r = __dadd_rn(r, 1.0);
    return (int64_t)r;
}

__device__ int64_t ceil_div(u128 a, u128 b) { return (int64_t)((a + b - 1) / b); }

__global__ void __launch_bounds__(kThreads) build_tables_kernel(TableArgs a) {
    const Layout& y = a.lay;
    const int L = y.L, NT = y.NT;
    int64_t* P = reinterpret_cast<int64_t*>(a.img + y.offP);
    int64_t* SA = reinterpret_cast<int64_t*>(a.img + y.offSA);
    int64_t* PB = reinterpret_cast<int64_t*>(a.img + y.offPB);
    int64_t* p2p = reinterpret_cast<int64_t*>(a.img + y.offP2P);
    int64_t* mem = reinterpret_cast<int64_t*>(a.img + y.offMem);
    int64_t* inter = reinterpret_cast<int64_t*>(a.img + y.offInter);
    int64_t* minq = reinterpret_cast<int64_t*>(a.img + y.offMinQ);
    int32_t* maxn = reinterpret_cast<int32_t*>(a.img + y.offMaxN);
    int32_t* pow2 = reinterpret_cast<int32_t*>(a.img + y.offPow2);
    int32_t* gpus = reinterpret_cast<int32_t*>(a.img + y.offGpus);
    int32_t* cap = reinterpret_cast<int32_t*>(a.img + y.offCap);
    const int tid = threadIdx.x;

    // per-type node statistics (one thread per type; types beyond NT are absent)
    if (tid < kMaxTypes) {
        const int g = tid;
        int64_t cnt = 0, nic = kInf;
        int32_t mx = 0;
        int64_t cp[4] = {0, 0, 0, 0};
        if (g < NT) {
            for (int b = 0; b < a.n_nodes; ++b) {
                const heddle_node nd = a.nodes[b];
                if (nd.type != g) continue;
                cnt += nd.gpus;
                mx = max(mx, nd.gpus);
                nic = min(nic, nd.nic_bw);
                for (int e = 0; e < 4; ++e) cp[e] += (int64_t)(nd.gpus >> e) << e;
            }
        }
        gpus[g] = (int32_t)cnt;
        maxn[g] = mx;
        int p = 1;
        while (p * 2 <= mx && p < 8) p *= 2;
        pow2[g] = cnt ? p : 0;
        inter[g] = cnt ? nic : 0;
        mem[g] = g < NT ? a.types[g].mem_bytes : 0;
        for (int e = 0; e < 4; ++e) cap[g * 4 + e] = (int32_t)cp[e];
    }
    __syncthreads();

    // per-layer cost entries q[g][j][l], parked at P[g][j][l + 1]
    for (int t = tid; t < NT * 4 * L; t += blockDim.x) {
        const int l = t % L;
        const int j = (t / L) % 4;
        const int g = t / (4 * L);
        int64_t q = 0;
        if (gpus[g] > 0) {
            double s;
            if (a.profile) {
                s = a.profile[t];
            } else {
                const heddle_layer ly = a.layers[l];
                const double k = (double)(1 << j);
                s = __ddiv_rn(ly.flops, __dmul_rn(__dmul_rn(k, a.types[g].tflops), 1e12));
                if (j > 0) {
                    const double bw = (1 << j) <= maxn[g] ? __ll2double_rn(a.types[g].intra_bw)
                                                          : __ll2double_rn(inter[g]);
                    const double ring = __ddiv_rn(__dmul_rn(2.0, __dsub_rn(k, 1.0)), k);
                    double u = __dmul_rn(4.0, ring);
                    u = __dmul_rn(u, __ll2double_rn(ly.ar_bytes));
                    u = __ddiv_rn(u, bw);
                    s = __dadd_rn(s, u);
                    const double part = __ddiv_rn(__dsub_rn(k, 1.0), k);
                    u = __dmul_rn(4.0, part);
                    u = __dmul_rn(u, __ll2double_rn(ly.a2a_bytes));
                    u = __ddiv_rn(u, bw);
                    s = __dadd_rn(s, u);
                }
            }
            const double ns = __dmul_rn(s, 1e9);
            if (!(ns >= 0.0) || !(ns < 4.0e18)) {
                atomicOr(a.flags, kTabBadValue);
            } else {
                q = round_half_away(ns);
            }
        }
        a.q[t] = q;
        P[(size_t)(g * 4 + j) * (L + 1) + l + 1] = q;
    }
    __syncthreads();

    // prefix sums per (type, degree) row, cheapest single layer
    for (int r = tid; r < NT * 4; r += blockDim.x) {
        int64_t* row = P + (size_t)r * (L + 1);
        row[0] = 0;
        int64_t acc = 0, mn = kInf;
        for (int l = 1; l <= L; ++l) {
            const int64_t q = row[l];
            mn = min(mn, q);
            acc += q;
            if (acc > kTableLimit) {
                atomicOr(a.flags, kTabTooLarge);
                acc = kTableLimit;
            }
            row[l] = acc;
        }
        minq[r] = mn;
    }
    // equal per-layer cost for every (type, degree) of a present type
    __shared__ int cost_uniform;
    if (tid == 0) cost_uniform = 1;
    __syncthreads();
    for (int t = tid; t < NT * 4 * L; t += blockDim.x) {
        const int l = t % L;
        if (l > 0 && a.q[t] != a.q[t - l]) cost_uniform = 0;
    }
    __syncthreads();
    if (tid == 0) reinterpret_cast<int32_t*>(a.img + y.offModel)[1] = cost_uniform;

    // byte prefixes
    if (tid == 0) {
        int64_t st = 0, ac = 0, pb = 0;
        SA[0] = 0;
        SA[1] = 0;
        PB[0] = 0;
        for (int l = 0; l < L; ++l) {
            st += a.layers[l].state_bytes;
            ac += a.layers[l].act_bytes;
            pb += a.layers[l].param_bytes;
            SA[2 * (l + 1)] = st;
            SA[2 * (l + 1) + 1] = ac;
            PB[l + 1] = pb;
        }
    }

    // longest run of consecutive layers whose state plus f in-flight
    // activations fit one group of (type g, degree 2^j): a two-pointer scan
    // per (g, j, f); a candidate whose stages' runs sum below L cannot fit
    if (tid == 0) {
        bool uni = true;
        for (int l = 1; l < L; ++l)
            uni = uni && a.layers[l].state_bytes == a.layers[0].state_bytes &&
                  a.layers[l].act_bytes == a.layers[0].act_bytes;
        reinterpret_cast<int32_t*>(a.img + y.offModel)[0] = uni ? 1 : 0;
        bool puni = true;
        for (int l = 1; l < L; ++l) puni = puni && a.layers[l].param_bytes == a.layers[0].param_bytes;
        reinterpret_cast<int32_t*>(a.img + y.offModel)[2] = puni ? 1 : 0;
    }
    uint8_t* win = a.img + y.offWin;
    for (int t = tid; t < 8 * 4 * 33; t += blockDim.x) {
        const int f = t % 33;
        const int j = (t / 33) % 4;
        const int g = t / (33 * 4);
        int best = 0;
        if (g < NT && gpus[g] > 0 && f > 0) {
            const int64_t capk = mem[g] << j;
            int e = 0;
            int64_t st = 0, ac = 0;  // bytes of layers [i, e)
            for (int i = 0; i < L; ++i) {
                if (e < i) {
                    e = i;
                    st = ac = 0;
                }
                while (e < L && (st + a.layers[e].state_bytes) + (int64_t)f * (ac + a.layers[e].act_bytes) <= capk) {
                    st += a.layers[e].state_bytes;
                    ac += a.layers[e].act_bytes;
                    ++e;
                }
                best = max(best, e - i);
                if (e > i) {
                    st -= a.layers[i].state_bytes;
                    ac -= a.layers[i].act_bytes;
                }
            }
        }
        win[t] = (uint8_t)best;
    }

    // P2P: forward activation plus backward gradient (2 x boundary bytes)
    // over the intra-node link when the two consecutive groups share a node,
    // else over the slower NIC of the two types
    for (int t = tid; t < 8 * 8 * 2; t += blockDim.x) {
        const int same = t & 1;
        const int h = (t >> 1) & 7;
        const int g = t >> 4;
        int64_t bw = 0;
        if (g < NT && h < NT && gpus[g] > 0 && gpus[h] > 0)
            bw = same ? a.types[g].intra_bw : min(inter[g], inter[h]);
        int64_t c = 0;
        if (bw > 0) {
            c = ceil_div((u128)2 * (u128)a.boundary_bytes * 1000000000u, (u128)bw);
            if (c > kTableLimit) atomicOr(a.flags, kTabTooLarge);
        }
        p2p[t] = c;
    }
}

}  // namespace

cudaError_t launch_tables(const TableArgs& a, cudaStream_t st) {
    build_tables_kernel<<<1, kThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hd
