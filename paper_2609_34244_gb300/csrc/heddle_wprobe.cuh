// heddle_wprobe.cuh -- the exact PartitionLayers probe run by one warp per
// worklist entry, shared by the general search and the expert-tiling search.
//
// probe(B) decides whether a split with every stage time <= B and every
// stage within memory exists:
//   forward:  U_0 = 0, U_{s+1} = the furthest end stage s reaches from U_s
//             (an upper bound on every feasible boundary a_{s+1});
//   backward: C_S = {L}; C_s = { i in [s, U_s] : the smallest j in C_{s+1}
//             above i gives a stage [i, j) that fits }; feasible iff stage 0
//             fits [0, min C_1).
// Stage time and memory grow with the interval, so the smallest successor
// dominates and C_s is exactly the set of feasible stage-s starts below U_s.
// The probe also returns the largest accepted and the smallest rejected
// stage time: every B' in [hi, B] (feasible) or [B, lo) (infeasible) takes
// the same decisions, so a search snaps its bracket to them and ends on B*;
// the sets at B* give the canonical (lexicographically smallest) split.
//
// The 32 lanes check 32 positions at once: a stage's forward reach is the
// first rejection among 32 consecutive ends, and a backward set is built
// one 32-bit word per round -- lane l checks start 32 w + l against its
// smallest successor (a bit scan of the successor set) and the ballot is
// the word.  A check type J supplies the stages and the interval test:
//   typename J::Stage J::stage(int s) const   -- every lane calls it
//   int J::eval(const Stage&, int i, int j, int64_t B, int64_t* cost) const
//       -- 0 fits (cost <= B), 1 too slow, 2 out of memory.

#pragma once

#include "heddle_internal.cuh"

namespace hd {
namespace wp {

constexpr int kSetWords = 8;  // 256-bit position sets (L <= 255)
constexpr unsigned kFull = 0xffffffffu;
// Bounds of the image wait, in global-timer nanoseconds: the copy's own
// wait, then (after raising the error flag) a second wait for the copies
// still in flight.
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr uint64_t kDrainNs = 1000000000ull;

// per-warp shared state: sets C[0..32], forward bounds U, the split A
struct WarpArea {
    uint32_t C[kMaxStages + 1][kSetWords];
    uint8_t U[kMaxStages + 1];
    uint8_t A[kMaxStages + 1];
    uint8_t pad[30];
};

__device__ __forceinline__ uint32_t saddr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait on phase 0 of bar for at most `limit` ns; true once it completed.
__device__ __forceinline__ bool wait_phase0(uint64_t* bar, uint64_t limit) {
    const uint64_t t0 = global_ns();
    for (;;) {
        uint32_t done;
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0; selp.u32 %0, 1, 0, p; }"
            : "=r"(done)
            : "r"(saddr(bar))
            : "memory");
        if (done) return true;
        if (global_ns() - t0 > limit) return false;
    }
}

// A table image into shared memory: one thread arms an mbarrier with the
// byte count (a multiple of 16) and issues bulk asynchronous copies that
// together move exactly that count; all threads wait on phase 0.
//
// No copy outlives this function while the device works: the armed count
// equals the bytes issued, so the phase completes exactly when the last
// copy lands, and the copies depend on nothing but device memory (no other
// thread, CTA or kernel), so they land within microseconds.  The wait is
// still bounded (global timer, kWaitNs): if it runs out the CTA raises the
// error flag and waits once more, again bounded (kDrainNs), for the copies
// in flight before it returns; only a memory system that has stopped
// altogether -- a lost context, where no CTA runs again -- gets past both.
// False (error flag raised) if the first wait ran out.
__device__ inline bool load_image(unsigned char* dst, const unsigned char* src, uint32_t bytes, uint64_t* bar,
                                  uint32_t* err) {
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(saddr(bar)));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(bar)), "r"(bytes)
                     : "memory");
        for (uint32_t o = 0; o < bytes; o += 32768) {
            const uint32_t nb = bytes - o < 32768 ? bytes - o : 32768;
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    saddr(dst + o)),
                "l"(src + o), "r"(nb), "r"(saddr(bar))
                : "memory");
        }
    }
    __syncthreads();
    const bool done = wait_phase0(bar, kWaitNs);
    const int all = __syncthreads_and(done);
    if (!all) {
        if (threadIdx.x == 0) atomicOr(err, kErrStageWait);
        // the copies in flight land before the CTA leaves its shared memory
        if (threadIdx.x == 0) (void)wait_phase0(bar, kDrainNs);
        __syncthreads();
    }
    return all != 0;
}

__device__ __forceinline__ int64_t wmax64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, (int64_t)__shfl_xor_sync(kFull, v, o));
    return v;
}
__device__ __forceinline__ int64_t wmin64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = min(v, (int64_t)__shfl_xor_sync(kFull, v, o));
    return v;
}
__device__ __forceinline__ int64_t wsum64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

// smallest set position of C in (i, L], -1 if none (warp-uniform inputs)
__device__ __forceinline__ int next_above(const uint32_t* C, int i, int L) {
    int w = (i + 1) >> 5;
    if (w > (L >> 5)) return -1;
    uint32_t m = C[w] & (0xffffffffu << ((i + 1) & 31));
    while (m == 0) {
        if (++w > (L >> 5)) return -1;
        m = C[w];
    }
    return (w << 5) + __ffs(m) - 1;
}

// Exact probe of bound B by one warp (all lanes call it; uniform result).
// The sets land in wa; hi / lo are the snap values; checks counts the
// interval checks of this lane.
template <class J>
__device__ bool probe(const J& check, int S, int L, int64_t B, WarpArea& wa, int64_t& hi_out, int64_t& lo_out,
                      unsigned long long& checks) {
    const int lane = threadIdx.x & 31;
    int64_t hi = -1, lo = kInf;
    bool ok = true;
    // forward upper bounds on the boundaries
    int u = 0;
    if (lane == 0) wa.U[0] = 0;
    for (int s = 0; s + 1 < S && ok; ++s) {
        const typename J::Stage st = check.stage(s);
        const int lim = L - (S - 1 - s);
        int reach = u;  // furthest accepted end (u: none yet)
        for (int base = u + 1; base <= lim; base += 32) {
            const int j = base + lane;
            int r = 1;  // beyond lim: treated as a rejection
            int64_t v = 0;
            if (j <= lim) {
                r = check.eval(st, u, j, B, &v);
                ++checks;
                if (r == 0) hi = max(hi, v);
                else if (r == 1) lo = min(lo, v);
            }
            const unsigned rej = __ballot_sync(kFull, r != 0);
            if (rej) {
                reach = base + __ffs(rej) - 2;
                break;
            }
            reach = base + 31;
        }
        if (reach < s + 1) ok = false;
        u = reach;
        if (lane == 0) wa.U[s + 1] = (uint8_t)reach;
    }
    __syncwarp();
    // backward feasible-start sets: C_S = {L}, then stages S-1 .. 1
    if (ok) {
        if (lane < kSetWords) wa.C[S][lane] = lane == (L >> 5) ? 1u << (L & 31) : 0u;
        __syncwarp();
        int nmax = L;
        for (int s = S - 1; s >= 1 && ok; --s) {
            const uint32_t* Cn = wa.C[s + 1];
            if (lane < kSetWords) wa.C[s][lane] = 0;
            __syncwarp();
            const int top = min((int)wa.U[s], nmax - 1);
            if (top < s) {
                ok = false;
                break;
            }
            const typename J::Stage st = check.stage(s);
            int any = 0, newmax = -1;
            for (int w = top >> 5; w >= (s >> 5); --w) {
                const int i = (w << 5) + lane;
                // smallest successor above i: in this word, else beyond it
                const uint32_t cw = Cn[w];
                const uint32_t above = lane == 31 ? 0u : (cw >> (lane + 1)) << (lane + 1);
                int beyond = -1;
                for (int w2 = w + 1; w2 <= (L >> 5); ++w2)
                    if (Cn[w2]) {
                        beyond = (w2 << 5) + __ffs(Cn[w2]) - 1;
                        break;
                    }
                const int succ = above ? (w << 5) + __ffs(above) - 1 : beyond;
                int r = 3;
                int64_t v = 0;
                if (i >= s && i <= top && succ >= 0) {
                    r = check.eval(st, i, succ, B, &v);
                    ++checks;
                    if (r == 0) hi = max(hi, v);
                    else if (r == 1) lo = min(lo, v);
                }
                const unsigned acc = __ballot_sync(kFull, r == 0);
                if (lane == 0) wa.C[s][w] = acc;
                if (acc) {
                    any = 1;
                    if (newmax < 0) newmax = (w << 5) + 31 - __clz(acc);
                }
            }
            __syncwarp();
            if (!any) ok = false;
            nmax = newmax;
        }
    }
    bool feasible = false;
    if (ok) {
        const int succ0 = S == 1 ? L : next_above(wa.C[1], 0, L);
        const typename J::Stage st0 = check.stage(0);
        if (succ0 >= 0 && lane == 0) {
            int64_t v = 0;
            const int r = check.eval(st0, 0, succ0, B, &v);
            ++checks;
            if (r == 0) {
                hi = max(hi, v);
                feasible = true;
            } else if (r == 1) {
                lo = min(lo, v);
            }
        }
        feasible = __shfl_sync(kFull, feasible, 0);
    }
    hi_out = wmax64(hi);
    lo_out = wmin64(lo);
    return feasible;
}

// The forward pass alone, for a bound B at which every stage could hold any
// single layer of the model (its most expensive layer's time plus its P2P
// within B, and the largest single-layer state and activation within its
// memory; the caller checks this).  Then, by induction, the feasible
// stage-s ends form the interval [s, U_s]: positions up to U_{s-1} + 1 are
// reached one layer after their predecessor, those beyond only from U_{s-1}
// (the largest predecessor dominates), so B is feasible iff the last stage
// fits [U_{S-1}, L), and the chain of U_s is a split attaining every
// accepted stage time.  The snap values therefore mean what they mean for
// probe(): every bound in [hi, B] is feasible, every bound in [B, lo) is
// not (the interval property holds at any bound >= B).  No sets are built:
// the canonical split needs probe() at B*.
template <class J>
__device__ bool forward_probe(const J& check, int S, int L, int64_t B, int64_t& hi_out, int64_t& lo_out,
                              unsigned long long& checks) {
    const int lane = threadIdx.x & 31;
    int64_t hi = -1, lo = kInf;
    bool ok = true;
    int u = 0;
    for (int s = 0; s + 1 < S && ok; ++s) {
        const typename J::Stage st = check.stage(s);
        const int lim = L - (S - 1 - s);
        int reach = u;
        for (int base = u + 1; base <= lim; base += 32) {
            const int j = base + lane;
            int r = 1;
            int64_t v = 0;
            if (j <= lim) {
                r = check.eval(st, u, j, B, &v);
                ++checks;
                if (r == 0) hi = max(hi, v);
                else if (r == 1) lo = min(lo, v);
            }
            const unsigned rej = __ballot_sync(kFull, r != 0);
            if (rej) {
                reach = base + __ffs(rej) - 2;
                break;
            }
            reach = base + 31;
        }
        if (reach < s + 1) ok = false;
        u = reach;
    }
    bool feasible = false;
    if (ok) {
        const typename J::Stage st = check.stage(S - 1);
        if (lane == 0) {
            int64_t v = 0;
            const int r = check.eval(st, u, L, B, &v);
            ++checks;
            if (r == 0) {
                hi = max(hi, v);
                feasible = true;
            } else if (r == 1) {
                lo = min(lo, v);
            }
        }
        feasible = __shfl_sync(kFull, feasible, 0);
    }
    hi_out = wmax64(hi);
    lo_out = wmin64(lo);
    return feasible;
}

// The first guess of B* (warp-uniform): the saturating continuous balance
// sum_s min(m_s, (B - c_s) / q_s) = L + (stages below their run) / 2, with
// each lane's stage given by 1 / q_s (rq, its average layer cost), c_s (cf)
// and its memory run m_s (mr); at most three Newton steps from the
// unsaturated balance, clamped to [max_s c_s + q_s, hi].
__device__ inline int64_t first_guess(float rq, float cf, float mr, int S, int L, int64_t hi) {
    const bool st = rq > 0.f;
    float inv = rq, cw = cf * rq, flo = st ? cf + 1.0f / rq : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        inv += __shfl_xor_sync(kFull, inv, o);
        cw += __shfl_xor_sync(kFull, cw, o);
        flo = fmaxf(flo, __shfl_xor_sync(kFull, flo, o));
    }
    const float fhi = u64_to_float((uint64_t)hi);
    float Bf = fmaxf(flo, inv > 0.f ? ((float)L + 0.5f * (float)S + cw) / inv : flo);
    for (int it = 0; it < 3; ++it) {
        Bf = fminf(Bf, fhi);
        const float x = (Bf - cf) * rq;
        const bool sat = !st || x >= mr;
        float cnt = sat ? mr : x, sl = sat ? 0.f : rq, nb = sat ? 0.f : 1.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            cnt += __shfl_xor_sync(kFull, cnt, o);
            sl += __shfl_xor_sync(kFull, sl, o);
            nb += __shfl_xor_sync(kFull, nb, o);
        }
        const float tgt = (float)L + 0.5f * nb;
        if (cnt >= tgt - 0.25f || sl <= 0.f) break;
        Bf += (tgt - cnt) / sl;
    }
    return (int64_t)float_to_u64(fmaxf(fminf(Bf, fhi), 0.f));
}

// The canonical split from the sets of a feasible probe at B*, by lane 0
// into wa.A (a_{s+1} = the smallest element of C_{s+1} above a_s); false if
// a set ran out (never expected after a feasible probe).
__device__ inline bool walk(WarpArea& wa, int S, int L) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) {
        int at = 0;
        wa.A[0] = 0;
        for (int s = 0; s + 1 < S; ++s) {
            const int x = next_above(wa.C[s + 1], at, L);
            if (x < 0) ok = false;
            at = max(x, at + 1);
            wa.A[s + 1] = (uint8_t)at;
        }
        wa.A[S] = (uint8_t)L;
    }
    __syncwarp();
    return __shfl_sync(kFull, ok, 0);
}

}  // namespace wp
}  // namespace hd
