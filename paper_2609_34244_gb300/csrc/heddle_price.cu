// heddle_price.cu -- the screen kernel (decode + validate, §5.1 masks; DP
// degree, §5.3 packing; the memory screen of §5.2) and the dispatch of the
// search over its worklist.
//
// Two launches per chunk.  The screen kernel (one thread per candidate,
// coalesced) decodes and validates every candidate, computes its DP degree
// and decides memory feasibility from a table of the longest run of layers
// each (type, degree, in-flight count) can hold: if the runs of the stages
// sum below L no split fits (OOM); when every layer has the same state and
// activation bytes, runs summing to at least L (each at least one layer)
// also guarantee a split that fits, so no memory-only probe is needed.
// Candidates that still need PartitionLayers are compacted into a worklist,
// which one of the searches then prices: the equal-layer closed form
// (heddle_eqsearch.cu) when every layer costs the same, the paper's split
// rule in that mode (heddle_distribute.cu), else the general exact
// threshold search: one thread per entry while every stage fits any single
// layer (heddle_gsearch.cu), one warp per entry for the rest
// (heddle_wsearch.cu).

#include <algorithm>
#include <mutex>

#include "heddle_tiled.cuh"

namespace hd {
namespace {

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

// Per stage byte: bit 31 inadmissible; bits 24-26 type; bits 16-20 the bit
// that adds the stage's units to its type's demand word; bits 0-10 the row
// (type, degree) of the run table.
__device__ __forceinline__ uint32_t stage_desc(int b, const Layout& y, const unsigned char* img, int moe) {
    const int32_t* gmaxn = reinterpret_cast<const int32_t*>(img + y.offMaxN);
    const int32_t* gpow2 = reinterpret_cast<const int32_t*>(img + y.offPow2);
    const int32_t* ggpus = reinterpret_cast<const int32_t*>(img + y.offGpus);
    const int g = b & 7, j = (b >> 3) & 3;
    if ((b >> 5) != 0 || g >= y.NT || ggpus[g] <= 0 || (!moe && (1 << j) > gmaxn[g])) return 1u << 31;
    const int unit = (1 << j) <= gmaxn[g] ? (1 << j) : gpow2[g];
    const int uc = 31 - __clz(unit);
    // the stage adds 2^(j - uc) units of 2^uc GPUs to field uc of its type's
    // demand word (fields of 9, 8, 7 and 6 bits at bits 0, 9, 17, 24: at
    // most 32 stages x 8 / 2^uc units)
    const int off = uc == 0 ? 0 : uc == 1 ? 9 : uc == 2 ? 17 : 24;
    return ((uint32_t)g << 24) | ((uint32_t)(j - uc + off) << 16) | (uint32_t)((g * 4 + j) * 33);
}

// Steps 1-2 and the memory screen for every candidate of the batch.  Each
// CTA takes 256 consecutive candidates at a time: their S and M, and the
// code planes up to the largest S among them, are copied to shared memory
// (16-byte vector copies when the planes are aligned), the candidates are
// counting-sorted by S, and thread i screens the i-th of that order, so the
// lanes of a warp run stage loops of nearly equal length.
// kGen: the general search follows (the single-fit routing below is live).
template <bool kGen>
__global__ void __launch_bounds__(kScreenBlock) screen_kernel(PriceArgs a) {
    __shared__ uint32_t desc[256];
    __shared__ uint8_t win[8 * 4 * 33];
    __shared__ __align__(16) uint32_t cap[8 * 4];
    __shared__ uint32_t magic[257];
    __shared__ uint32_t dem[8 * kScreenBlock];  // per-thread units per class (see stage_desc), per type
    __shared__ __align__(16) uint8_t tile[kMaxStages * kScreenBlock];  // [stage][candidate of the slice]
    __shared__ uint8_t sS[kScreenBlock];
    __shared__ uint16_t sM[kScreenBlock];
    __shared__ uint8_t order[kScreenBlock];
    __shared__ int bins[kMaxStages + 3];
    __shared__ int smax;
    // general search only: per (type, degree, in-flight count) whether any
    // single layer of the model fits the stage's memory; entries with a
    // stage where not go straight to the warp-per-entry search's list
    __shared__ uint8_t sfit[8 * 4 * 33];
    __shared__ long long single[2];
    const Layout& y = a.lay;
    const int L = y.L;
    constexpr bool gen = kGen;
    if (gen) {
        if (threadIdx.x < 32) {
            const longlong2* SA = reinterpret_cast<const longlong2*>(a.img + y.offSA);
            long long m0 = 0, m1 = 0;
            for (int l = threadIdx.x; l < L; l += 32) {
                const longlong2 u = SA[l], v = SA[l + 1];
                m0 = max(m0, v.x - u.x);
                m1 = max(m1, v.y - u.y);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                m0 = max(m0, __shfl_xor_sync(0xffffffffu, m0, o));
                m1 = max(m1, __shfl_xor_sync(0xffffffffu, m1, o));
            }
            if (threadIdx.x == 0) {
                single[0] = m0;
                single[1] = m1;
            }
        }
        __syncthreads();
        const int64_t* gmem = reinterpret_cast<const int64_t*>(a.img + y.offMem);
        for (int i = threadIdx.x; i < 8 * 4 * 33; i += blockDim.x) {
            const int g = i / 132, j = (i / 33) & 3, f = i % 33;
            sfit[i] = g < y.NT && single[0] + (long long)f * single[1] <= (long long)(gmem[g] << j);
        }
    }
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
    uint32_t* mydem = dem + threadIdx.x;
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
            // a plan's template that the plan cannot reach is priced SKIPPED
            // (bit 7 of its S byte; it sorts with the invalid ones)
            const bool skipped = a.skip && a.skip[c0 + threadIdx.x];
            if (skipped) key = 0;
            sS[threadIdx.x] = (uint8_t)(key | (skipped ? 0x80 : 0));
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
        uint32_t fits1 = 1;  // every stage could hold any single layer (general search)
        int64_t n = 0;
        if (live) {
            S = sS[ci] & 0x3f;
            M = sM[ci];
            if (sS[ci] & 0x80) status = HEDDLE_CAND_SKIPPED;
            if (S > 0) {
#pragma unroll
                for (int g = 0; g < 8; ++g) mydem[g * kScreenBlock] = 0;
                uint32_t bad = 0;
                int run_sum = 0, run_min = 255;
                const uint8_t* col = tile + ci;
                for (int s = 0; s < S; ++s) {
                    const uint32_t d = desc[col[s * kScreenBlock]];
                    bad |= d;
                    const int g = (d >> 24) & 7;
                    mydem[g * kScreenBlock] += 1u << ((d >> 16) & 31);
                    const int wi = (d & 0x7ff) + min(S - s, M);
                    const int w = win[wi];
                    run_sum += w;
                    run_min = min(run_min, w);
                    if (gen) fits1 &= sfit[wi];
                }
                if (bad >> 31) {
                    status = HEDDLE_CAND_INVALID;
                } else {
                    // n = min over (type, class e) of capacity / GPUs in units
                    // >= 2^e; a class with no group of its own size is
                    // dominated by the class above it.  Every type is
                    // visited (an absent type's demand word is zero), so the
                    // eight chains of loads are independent
                    uint32_t nn = 0xffffffffu;
#pragma unroll
                    for (int g = 0; g < 8; ++g) {
                        const uint32_t v = mydem[g * kScreenBlock];
                        const uint4 cg = *reinterpret_cast<const uint4*>(cap + g * 4);
                        // GPUs per class from the unit counts
                        const uint32_t f3 = (v >> 24) << 3, f2 = ((v >> 17) & 0x7fu) << 2;
                        const uint32_t f1 = ((v >> 9) & 0xffu) << 1, f0 = v & 0x1ffu;
                        const uint32_t d3 = f3, d2 = d3 + f2, d1 = d2 + f1, d0 = d1 + f0;
                        const uint32_t q3 = div_small(cg.w, d3, magic), q2 = div_small(cg.z, d2, magic);
                        const uint32_t q1 = div_small(cg.y, d1, magic), q0 = div_small(cg.x, d0, magic);
                        nn = min(nn, min(min(f3 ? q3 : 0xffffffffu, f2 ? q2 : 0xffffffffu),
                                         min(f1 ? q1 : 0xffffffffu, f0 ? q0 : 0xffffffffu)));
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
            // the entry in its depth's bucket, for the searches' order by
            // decreasing depth -- or, for the general search when some
            // stage cannot hold every single layer, in the list of the
            // warp-per-entry search
            const bool listed = gen && take && !fits1;
            const unsigned bmask = __ballot_sync(0xffffffffu, take && !listed);
            const unsigned lmask = __ballot_sync(0xffffffffu, listed);
            if (lmask) {
                int l0 = 0;
                if (lane == __ffs(lmask) - 1) l0 = atomicAdd(a.wl_count + kWlGeneral, __popc(lmask));
                l0 = __shfl_sync(0xffffffffu, l0, __ffs(lmask) - 1) + __popc(lmask & ((1u << lane) - 1));
                if (listed && p < a.wl_cap && l0 < a.wl_cap) a.sv_idx[l0] = p;
            }
            if (take && !listed) {
                const unsigned same = __match_any_sync(bmask, S);
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

}  // namespace

// The general search: one thread per entry where every stage fits any single
// layer (heddle_gsearch.cu), then one warp per entry it left (heddle_wsearch.cu).
cudaError_t launch_thread_search(const PriceArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_warp_search(const PriceArgs& a, int num_sms, cudaStream_t st, bool listed);

cudaError_t launch_screen(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid, int64_t* launches) {
    if (a.n <= 0) return cudaSuccess;
    if (a.n > a.wl_cap) return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(a.wl_count, 0, sizeof(int32_t) * kWlMeta, st);
    if (e != cudaSuccess) return e;
    // one wave of resident CTAs, each looping over slices
    int screen_per_sm = 0;
    e = resident_blocks(reinterpret_cast<const void*>(&screen_kernel<false>), kScreenBlock, 0, &screen_per_sm);
    if (e != cudaSuccess) return e;
    const int grid = (int)std::min<int64_t>((a.n + kScreenBlock - 1) / kScreenBlock,
                                            (int64_t)num_sms * std::max(screen_per_sm, 1));
    if (!a.uniform && !a.split_mode) screen_kernel<true><<<grid, kScreenBlock, 0, st>>>(a);
    else screen_kernel<false><<<grid, kScreenBlock, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (launches) launches[0] += 1;
    if (mid && (e = cudaEventRecord(mid, st)) != cudaSuccess) return e;
    return cudaSuccess;
}

cudaError_t resident_blocks(const void* func, int block, size_t smem, int* per_sm) {
    struct Limit {  // the largest dynamic shared memory a kernel was allowed so far
        const void* func;
        int device;
        size_t smem;
    };
    struct Answer {
        const void* func;
        int device, block;
        size_t smem;
        int per_sm;
    };
    static std::mutex mu;
    static Limit limits[32];
    static Answer answers[128];
    static int n_limits = 0, n_answers = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < n_answers; ++i) {
        const Answer& x = answers[i];
        if (x.func == func && x.device == dev && x.block == block && x.smem == smem) {
            *per_sm = x.per_sm;
            return cudaSuccess;
        }
    }
    // raise (never lower) the kernel's limit: cached launches of larger
    // sizes rely on it.  Past the tables' capacity nothing is cached and
    // the limit is set on every call.
    int li = -1;
    for (int i = 0; i < n_limits; ++i)
        if (limits[i].func == func && limits[i].device == dev) li = i;
    if (li < 0 && n_limits < 32) {
        li = n_limits++;
        limits[li] = Limit{func, dev, 0};
    }
    if (li < 0 || limits[li].smem < smem) {
        e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        if (li >= 0) limits[li].smem = smem;
    }
    int v = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, func, block, smem);
    if (e != cudaSuccess) return e;
    if (li >= 0 && n_answers < 128) answers[n_answers++] = Answer{func, dev, block, smem, v};
    *per_sm = v;
    return cudaSuccess;
}

cudaError_t launch_price(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid, int64_t* launches) {
    if (a.n <= 0) return cudaSuccess;
    cudaError_t e = launch_screen(a, num_sms, st, mid, launches);
    if (e != cudaSuccess) return e;
    if (launches) launches[1] += 1;
    if (a.split_mode) return launch_distribute(a, num_sms, st);
    if (a.uniform) return launch_eq_search(a, num_sms, st);
    // a batch smaller than the thread search's threshold cannot fill its
    // buckets up to it: that kernel would return at once, so it is not launched
    if (a.n >= a.thread_min && (e = launch_thread_search(a, num_sms, st)) != cudaSuccess) return e;
    return launch_warp_search(a, num_sms, st, true);
}

}  // namespace hd
