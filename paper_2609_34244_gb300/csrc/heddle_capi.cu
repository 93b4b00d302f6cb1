// heddle_capi.cu -- the C ABI (include/heddle.h): context, validated loads,
// launches on the caller's stream, and the host-buffer streaming path.

#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "heddle_tiled.cuh"

using hd::Layout;

struct heddle_ctx {
    int device = 0;
    int num_sms = 0;
    char msg[512] = {0};
    // host copies of the descriptions
    std::vector<heddle_gpu_type> types;
    std::vector<heddle_node> nodes;
    std::vector<heddle_layer> layers;
    std::vector<double> profile;
    bool have_cluster = false, have_model = false, have_profile = false;
    int64_t boundary_bytes = 0;
    int32_t moe = 0;
    // device tables
    Layout lay{};
    bool tables_ready = false;
    int32_t model_flags[4] = {0, 0, 0, 0};  // copy of the image's model flags
    int32_t search_mode = HEDDLE_SEARCH_AUTO;
    int32_t thread_min = -1;  // heddle_set_thread_search_min (< 0: the default)
    unsigned char* d_img = nullptr;
    size_t img_cap = 0;
    int64_t* d_q = nullptr;
    size_t q_cap = 0;
    uint32_t* d_flags = nullptr;            // [0] table build, [1] device errors, [2] top-k threshold
    unsigned long long* d_counters = nullptr;  // [3]
    bool count_next = false;
    // search worklist scratch (hd::kWorklistCap candidates); the other
    // sets, the four work streams and their events exist once a call has
    // priced more than one chunk (consecutive chunks rotate over sets and
    // streams, so one chunk's screen and search overlap the earlier
    // chunks' searches and top-k)
    struct Worklist {
        int32_t* count = nullptr;   // hd::kWlMeta ints
        int32_t* bucket = nullptr;  // [32][2^20]
        int32_t* idx = nullptr;
        uint16_t* n = nullptr;
        uint16_t* M = nullptr;
        uint8_t* S = nullptr;
        uint8_t* memok = nullptr;
        uint8_t* code = nullptr;
        int64_t* T = nullptr;
        uint32_t* nM = nullptr;
        // survivors of the top-k threshold (equal-layer search in a top-k pricing)
        int32_t* sv_idx = nullptr;
        int64_t* sv_T = nullptr;
        uint32_t* sv_nM = nullptr;
    };
    // five worklist sets: chunk i uses set i % 5, so it waits for the top-k
    // of chunk i - 5 (the first chunk's, which fills an empty state, is the
    // longest), while four chunks run on the four work streams
    static constexpr int kWlSets = 5;
    Worklist wl[kWlSets];
    bool pipe_ready = false;
    cudaStream_t s_work[4] = {nullptr, nullptr, nullptr, nullptr};
    cudaEvent_t ev_in = nullptr;
    cudaEvent_t ev_searched[kWlSets] = {}, ev_wl_free[kWlSets] = {};
    int64_t chunk = hd::kWorklistCap;
    // top-k merge scratch
    hd::TopkEntry* d_scratch = nullptr;
    int32_t* d_scratch_count = nullptr;
    int scratch_blocks = 0;
    hd::TopkEntry* d_scratch2 = nullptr;
    int32_t* d_scratch2_count = nullptr;
    int32_t* d_tickets = nullptr;  // [17], zero between top-k launches
    // host-buffer path
    cudaStream_t s_h2d = nullptr, s_d2h = nullptr;
    // kStageSets staging sets: a batch's copies in wait only for the batch
    // kStageSets earlier to be merged, so the copy stream keeps running while
    // the two batches before it are still being searched
    static constexpr int kStageSets = 3;
    cudaEvent_t ev_loaded[kStageSets] = {}, ev_priced[kStageSets] = {}, ev_free[kStageSets] = {};
    int64_t stage_cap = 0;
    int32_t stage_smax = 0;
    uint8_t* st_S[kStageSets] = {};
    uint16_t* st_M[kStageSets] = {};
    uint8_t* st_code[kStageSets] = {};
    int64_t* st_T[kStageSets] = {};
    int64_t* st_B[kStageSets] = {};
    uint16_t* st_n[kStageSets] = {};
    uint8_t* st_status[kStageSets] = {};
    uint8_t* st_bounds[kStageSets] = {};
    heddle_topk_state* d_state = nullptr;
    // phase timing: four events per priced chunk (start, after the screen,
    // after the search, after the top-k), recorded while time_phases is set
    bool time_phases = false;
    std::vector<cudaEvent_t> ev_pool;
    struct PhaseRec {
        cudaEvent_t e[5];  // screen start, screen end, search end, top-k start, top-k end
        bool topk;
        int64_t launches[3];
    };
    std::vector<PhaseRec> phase_recs;
    // micro-batch-size fill: one cost-table image per size 2^i (level i),
    // and the results of one level for one chunk
    struct Level {
        Layout lay{};
        unsigned char* img = nullptr;
        size_t img_cap = 0;
        int64_t* q = nullptr;
        size_t q_cap = 0;
        int32_t flags[4] = {0, 0, 0, 0};
    };
    int32_t mbs_levels = 0;
    std::vector<double> mbs_profile;  // [levels][types][4][L] seconds, or empty
    bool mbs_ready = false;
    Level lv[HEDDLE_MAX_MBS_LEVELS];
    // one result set per size above the base (their pricings run as a
    // pipeline, their merges after)
    int64_t* lv_T[HEDDLE_MAX_MBS_LEVELS] = {};
    int64_t* lv_B[HEDDLE_MAX_MBS_LEVELS] = {};
    uint16_t* lv_n[HEDDLE_MAX_MBS_LEVELS] = {};
    uint8_t* lv_status[HEDDLE_MAX_MBS_LEVELS] = {};
    uint8_t* lv_bounds[HEDDLE_MAX_MBS_LEVELS] = {};
    size_t lv_T_cap[HEDDLE_MAX_MBS_LEVELS] = {}, lv_B_cap[HEDDLE_MAX_MBS_LEVELS] = {},
           lv_n_cap[HEDDLE_MAX_MBS_LEVELS] = {}, lv_status_cap[HEDDLE_MAX_MBS_LEVELS] = {},
           lv_bounds_cap[HEDDLE_MAX_MBS_LEVELS] = {};
    // multi-template plans: the cluster's nodes on the device, split bounds
    // of slots whose caller passed none
    int32_t* d_node_type = nullptr;
    int32_t* d_node_gpus = nullptr;
    size_t node_cap = 0, node_cap2 = 0;
    bool nodes_on_device = false;  // d_node_* hold the loaded cluster's nodes
    uint8_t* plan_bounds[HEDDLE_MAX_TEMPLATES] = {nullptr, nullptr, nullptr, nullptr};
    size_t plan_bounds_cap[HEDDLE_MAX_TEMPLATES] = {0, 0, 0, 0};
    uint8_t* skip_mask = nullptr;  // the plan slot being priced: candidates priced SKIPPED
    size_t skip_mask_cap = 0;
    // expert tiling: the experts' byte counts and the tiled image
    bool have_experts = false, tiled_ready = false;
    std::vector<int64_t> expert_state, expert_param;
    hd::TiledLayout tlay{};
    unsigned char* d_timg = nullptr;
    size_t timg_cap = 0;
};

namespace {

heddle_status fail(heddle_ctx* x, heddle_status st, const char* fmt, ...) {
    if (x) {
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(x->msg, sizeof(x->msg), fmt, ap);
        va_end(ap);
    }
    return st;
}

heddle_status ok(heddle_ctx* x) {
    x->msg[0] = 0;
    return HEDDLE_OK;
}

#define CU(call)                                                                           \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess)                                                             \
            return fail(x, HEDDLE_E_CUDA, "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                        __FILE__, __LINE__);                                               \
    } while (0)

// Makes the context's device current for the duration of a call.
struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

template <class T>
cudaError_t grow(T** p, size_t* cap, size_t need) {
    if (*cap >= need && *p) return cudaSuccess;
    if (*p) cudaFree(*p);
    *p = nullptr;
    *cap = 0;
    cudaError_t e = cudaMalloc((void**)p, need);
    if (e == cudaSuccess) *cap = need;
    return e;
}

constexpr int64_t kByteLimit = (int64_t)1 << 42;
constexpr int64_t kBwLimit = (int64_t)1 << 40;
constexpr int64_t kMemLimit = (int64_t)1 << 50;

// Build one cost-table image (and its per-layer cost table) for the given
// layers, profile (nullable: the synthetic formula) and boundary bytes.
heddle_status build_image(heddle_ctx* x, const std::vector<heddle_layer>& layers, const double* profile,
                          int64_t boundary_bytes, Layout& lay, unsigned char** img, size_t* img_cap,
                          int64_t** qtab, size_t* q_cap, int32_t model_flags[4]) {
    const int NT = (int)x->types.size(), L = (int)layers.size();
    // the gradient term stays below 2^56 ns: 2 * sum(param) * 1e9 / slowest NIC
    {
        unsigned __int128 G = 0;
        for (const auto& ly : layers) G += (unsigned __int128)ly.param_bytes;
        for (int g = 0; g < NT; ++g) {
            int64_t nic = INT64_MAX;
            for (const auto& nd : x->nodes)
                if (nd.type == g && nd.nic_bw < nic) nic = nd.nic_bw;
            if (nic == INT64_MAX) continue;
            const unsigned __int128 t = (2 * G * 1000000000u + nic - 1) / (unsigned __int128)nic;
            if (t > ((unsigned __int128)1 << 56))
                return fail(x, HEDDLE_E_LIMIT, "gradient synchronisation of type %d exceeds 2^56 ns", g);
        }
    }
    lay = hd::make_layout(L, NT);
    CU(grow(img, img_cap, lay.bytes));
    CU(grow(qtab, q_cap, sizeof(int64_t) * (size_t)NT * 4 * L));
    heddle_gpu_type* d_types = nullptr;
    heddle_node* d_nodes = nullptr;
    heddle_layer* d_layers = nullptr;
    double* d_prof = nullptr;
    cudaError_t e = cudaMalloc(&d_types, sizeof(heddle_gpu_type) * NT);
    if (e == cudaSuccess) e = cudaMalloc(&d_nodes, sizeof(heddle_node) * x->nodes.size());
    if (e == cudaSuccess) e = cudaMalloc(&d_layers, sizeof(heddle_layer) * L);
    const size_t nprof = (size_t)NT * 4 * L;
    if (e == cudaSuccess && profile) e = cudaMalloc(&d_prof, sizeof(double) * nprof);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_types, x->types.data(), sizeof(heddle_gpu_type) * NT, cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_nodes, x->nodes.data(), sizeof(heddle_node) * x->nodes.size(),
                       cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_layers, layers.data(), sizeof(heddle_layer) * L, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && d_prof) e = cudaMemcpy(d_prof, profile, sizeof(double) * nprof, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemset(*img, 0, lay.bytes);
    if (e == cudaSuccess) e = cudaMemset(x->d_flags, 0, sizeof(uint32_t));
    if (e == cudaSuccess) {
        hd::TableArgs a{};
        a.lay = lay;
        a.types = d_types;
        a.nodes = d_nodes;
        a.n_nodes = (int32_t)x->nodes.size();
        a.layers = d_layers;
        a.profile = d_prof;
        a.boundary_bytes = boundary_bytes;
        a.moe = x->moe;
        a.img = *img;
        a.q = *qtab;
        a.flags = x->d_flags;
        e = hd::launch_tables(a, 0);
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    uint32_t flags = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&flags, x->d_flags, sizeof(uint32_t), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess)
        e = cudaMemcpy(model_flags, *img + lay.offModel, sizeof(int32_t) * 4, cudaMemcpyDeviceToHost);
    cudaFree(d_types);
    cudaFree(d_nodes);
    cudaFree(d_layers);
    if (d_prof) cudaFree(d_prof);
    if (e != cudaSuccess) return fail(x, HEDDLE_E_CUDA, "cost-table build: %s", cudaGetErrorString(e));
    if (flags & hd::kTabBadValue)
        return fail(x, HEDDLE_E_ARG, "a per-layer cost is negative, not finite or above 4e18 ns");
    if (flags & hd::kTabTooLarge)
        return fail(x, HEDDLE_E_LIMIT, "a per-(type, degree) model time or a P2P term exceeds 2^40 ns");
    return ok(x);
}

// The tables of the micro-batch-size fill: level i is the model at
// micro-batch 2^i times the base size -- FLOPs, stored activations, the TP
// all-reduce and EP all-to-all messages and the boundary activation scale
// by 2^i; parameter, gradient and state bytes do not -- with its profile
// slice when per-size profiles were given.
heddle_status build_levels(heddle_ctx* x) {
    x->mbs_ready = false;
    if (x->mbs_levels < 1 || !x->have_cluster || !x->have_model) return ok(x);
    const int NT = (int)x->types.size(), L = (int)x->layers.size();
    const bool prof = !x->mbs_profile.empty();
    if (prof && x->mbs_profile.size() != (size_t)x->mbs_levels * NT * 4 * L)
        return fail(x, HEDDLE_E_STATE, "size profiles cover %zu entries, need %d levels x %d types x 4 x %d layers",
                    x->mbs_profile.size(), x->mbs_levels, NT, L);
    if (!prof && x->have_profile)
        return fail(x, HEDDLE_E_STATE, "the model was loaded with a profile: the fill needs per-size profiles");
    for (int i = 0; i < x->mbs_levels; ++i) {
        const int64_t f = (int64_t)1 << i;
        std::vector<heddle_layer> ly = x->layers;
        for (auto& y : ly) {
            y.flops *= (double)f;
            if (y.act_bytes > kByteLimit / f || y.ar_bytes > kByteLimit / f || y.a2a_bytes > kByteLimit / f)
                return fail(x, HEDDLE_E_LIMIT, "size 2^%d: a byte count exceeds 2^42", i);
            y.act_bytes *= f;
            y.ar_bytes *= f;
            y.a2a_bytes *= f;
        }
        if (x->boundary_bytes > kByteLimit / f)
            return fail(x, HEDDLE_E_LIMIT, "size 2^%d: boundary_bytes exceeds 2^42", i);
        heddle_ctx::Level& v = x->lv[i];
        const double* pr = prof ? x->mbs_profile.data() + (size_t)i * NT * 4 * L : nullptr;
        const heddle_status st =
            build_image(x, ly, pr, x->boundary_bytes * f, v.lay, &v.img, &v.img_cap, &v.q, &v.q_cap, v.flags);
        if (st != HEDDLE_OK) return st;
    }
    x->mbs_ready = true;
    return ok(x);
}

// The tiled image (expert tiling) from the main image, the layers and the
// experts' byte counts.
heddle_status build_tiled(heddle_ctx* x) {
    x->tiled_ready = false;
    if (!x->have_experts || !x->tables_ready) return ok(x);
    if (x->have_profile)
        return fail(x, HEDDLE_E_STATE, "expert tiling needs the synthetic cost model (the model has a profile)");
    const int NT = (int)x->types.size(), L = (int)x->layers.size();
    const hd::TiledLayout tl = hd::make_tiled_layout(L, NT);
    if (tl.bytes > hd::kTiledImageLimit)
        return fail(x, HEDDLE_E_LIMIT, "tiled tables of %d types x %d layers take %u bytes (limit %u)", NT, L,
                    tl.bytes, hd::kTiledImageLimit);
    // gradient terms stay below 2^56 ns on the intra-node path as well
    {
        unsigned __int128 G = 0;
        for (const auto& ly : x->layers) G += (unsigned __int128)ly.param_bytes;
        for (int g = 0; g < NT; ++g) {
            const unsigned __int128 t = (2 * G * 1000000000u + x->types[g].intra_bw - 1) /
                                        (unsigned __int128)x->types[g].intra_bw;
            if (t > ((unsigned __int128)1 << 56))
                return fail(x, HEDDLE_E_LIMIT, "expert gradient synchronisation of type %d exceeds 2^56 ns", g);
        }
    }
    CU(grow(&x->d_timg, &x->timg_cap, tl.bytes));
    heddle_gpu_type* d_types = nullptr;
    heddle_layer* d_layers = nullptr;
    int64_t* d_ex = nullptr;
    cudaError_t e = cudaMalloc(&d_types, sizeof(heddle_gpu_type) * NT);
    if (e == cudaSuccess) e = cudaMalloc(&d_layers, sizeof(heddle_layer) * L);
    if (e == cudaSuccess) e = cudaMalloc(&d_ex, sizeof(int64_t) * 2 * L);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_types, x->types.data(), sizeof(heddle_gpu_type) * NT, cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_layers, x->layers.data(), sizeof(heddle_layer) * L, cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_ex, x->expert_state.data(), sizeof(int64_t) * L, cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d_ex + L, x->expert_param.data(), sizeof(int64_t) * L, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemset(x->d_timg, 0, tl.bytes);
    if (e == cudaSuccess) e = cudaMemset(x->d_flags, 0, sizeof(uint32_t));
    if (e == cudaSuccess) {
        hd::TiledTableArgs a{};
        a.tl = tl;
        a.lay = x->lay;
        a.img = x->d_img;
        a.types = d_types;
        a.layers = d_layers;
        a.expert_state = d_ex;
        a.expert_param = d_ex + L;
        a.timg = x->d_timg;
        a.flags = x->d_flags;
        e = hd::launch_tiled_tables(a, 0);
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    uint32_t flags = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&flags, x->d_flags, sizeof(uint32_t), cudaMemcpyDeviceToHost);
    cudaFree(d_types);
    cudaFree(d_layers);
    cudaFree(d_ex);
    if (e != cudaSuccess) return fail(x, HEDDLE_E_CUDA, "tiled table build: %s", cudaGetErrorString(e));
    if (flags & hd::kTabBadValue)
        return fail(x, HEDDLE_E_ARG, "a tiled per-layer cost is negative, not finite or above 4e18 ns");
    if (flags & hd::kTabTooLarge) return fail(x, HEDDLE_E_LIMIT, "a tiled model time exceeds 2^40 ns");
    x->tlay = tl;
    x->tiled_ready = true;
    return ok(x);
}

heddle_status build_tables(heddle_ctx* x) {
    x->tables_ready = false;
    x->tiled_ready = false;
    x->mbs_ready = false;
    if (!x->have_cluster || !x->have_model) return ok(x);
    const int NT = (int)x->types.size(), L = (int)x->layers.size();
    if (x->have_profile && x->profile.size() != (size_t)NT * 4 * L)
        return fail(x, HEDDLE_E_STATE,
                    "model profile covers %zu entries, cluster needs %d types x 4 x %d layers",
                    x->profile.size(), NT, L);
    heddle_status st = build_image(x, x->layers, x->have_profile ? x->profile.data() : nullptr,
                                   x->boundary_bytes, x->lay, &x->d_img, &x->img_cap, &x->d_q, &x->q_cap,
                                   x->model_flags);
    if (st != HEDDLE_OK) return st;
    x->tables_ready = true;
    if (x->have_experts && (st = build_tiled(x)) != HEDDLE_OK) return st;
    if (x->mbs_levels > 0) return build_levels(x);
    return ok(x);
}

heddle_status check_cands(heddle_ctx* x, const heddle_candidates* c, bool device) {
    if (!c) return fail(x, HEDDLE_E_ARG, "candidates is NULL");
    if (c->n < 0) return fail(x, HEDDLE_E_ARG, "negative candidate count");
    if (c->n == 0) return HEDDLE_OK;
    if (!c->S || !c->M || !c->code) return fail(x, HEDDLE_E_ARG, "null candidate array");
    if (c->plane_stride < c->n) return fail(x, HEDDLE_E_ARG, "plane_stride below n");
    if (c->s_max < 1 || c->s_max > HEDDLE_MAX_STAGES)
        return fail(x, HEDDLE_E_ARG, "s_max must be in [1, %d]", HEDDLE_MAX_STAGES);
    (void)device;
    return HEDDLE_OK;
}

// the equal-layer closed form applies when every layer has the same cost per
// (type, degree) and the same memory, unless the general search is forced
bool equal_layer_search(const heddle_ctx* x, const int32_t* model_flags) {
    return x->search_mode == HEDDLE_SEARCH_AUTO && model_flags[0] && model_flags[1];
}
bool equal_layer_search(const heddle_ctx* x) { return equal_layer_search(x, x->model_flags); }

heddle_status check_ready(heddle_ctx* x) {
    if (!x->have_cluster) return fail(x, HEDDLE_E_STATE, "no cluster loaded");
    if (!x->have_model) return fail(x, HEDDLE_E_STATE, "no model loaded");
    if (!x->tables_ready) return fail(x, HEDDLE_E_STATE, "cost tables are not built");
    return HEDDLE_OK;
}

cudaError_t alloc_worklist(heddle_ctx::Worklist& w) {
    const size_t cap = hd::kWorklistCap;
    cudaError_t e = cudaMalloc(&w.count, sizeof(int32_t) * hd::kWlMeta);
    if (e == cudaSuccess) e = cudaMalloc(&w.bucket, sizeof(int32_t) * HEDDLE_MAX_STAGES * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.idx, sizeof(int32_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.n, sizeof(uint16_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.M, sizeof(uint16_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.S, cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.memok, cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.code, (size_t)HEDDLE_MAX_STAGES * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.T, sizeof(int64_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.nM, sizeof(uint32_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.sv_idx, sizeof(int32_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.sv_T, sizeof(int64_t) * cap);
    if (e == cudaSuccess) e = cudaMalloc(&w.sv_nM, sizeof(uint32_t) * cap);
    return e;
}

void free_worklist(heddle_ctx::Worklist& w) {
    cudaFree(w.count);
    cudaFree(w.bucket);
    cudaFree(w.idx);
    cudaFree(w.n);
    cudaFree(w.M);
    cudaFree(w.S);
    cudaFree(w.memok);
    cudaFree(w.code);
    cudaFree(w.T);
    cudaFree(w.nM);
    cudaFree(w.sv_idx);
    cudaFree(w.sv_T);
    cudaFree(w.sv_nM);
    w = heddle_ctx::Worklist{};
}

}  // namespace

extern "C" {

heddle_status heddle_create(heddle_ctx** out, int32_t device) {
    if (!out) return HEDDLE_E_ARG;
    *out = nullptr;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) return HEDDLE_E_CUDA;
    if (device < 0 || device >= ndev) return HEDDLE_E_ARG;
    heddle_ctx* x = new (std::nothrow) heddle_ctx();
    if (!x) return HEDDLE_E_NOMEM;
    x->device = device;
    DeviceGuard dg(device);
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess) {
        delete x;
        return HEDDLE_E_CUDA;
    }
    x->num_sms = prop.multiProcessorCount;
    x->scratch_blocks = 8 * x->num_sms;  // per-CTA lists of the top-k and of the fused search
    cudaError_t e = cudaMalloc(&x->d_flags, 4 * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaMemset(x->d_flags, 0, 4 * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaMalloc(&x->d_counters, 3 * sizeof(unsigned long long));
    if (e == cudaSuccess) e = cudaMemset(x->d_counters, 0, 3 * sizeof(unsigned long long));
    if (e == cudaSuccess)
        e = cudaMalloc(&x->d_scratch, sizeof(hd::TopkEntry) * hd::kMaxTopK * x->scratch_blocks);
    if (e == cudaSuccess) e = cudaMalloc(&x->d_scratch_count, sizeof(int32_t) * x->scratch_blocks);
    if (e == cudaSuccess) e = alloc_worklist(x->wl[0]);
    const int l2 = (x->scratch_blocks + 31) / 32;
    if (e == cudaSuccess) e = cudaMalloc(&x->d_scratch2, sizeof(hd::TopkEntry) * hd::kMaxTopK * l2);
    if (e == cudaSuccess) e = cudaMalloc(&x->d_scratch2_count, sizeof(int32_t) * l2);
    if (e == cudaSuccess) e = cudaMalloc(&x->d_tickets, sizeof(int32_t) * 17);
    if (e == cudaSuccess) e = cudaMemset(x->d_tickets, 0, sizeof(int32_t) * 17);

    if (e != cudaSuccess) {
        heddle_destroy(x);
        return HEDDLE_E_CUDA;
    }
    *out = x;
    return HEDDLE_OK;
}

void heddle_destroy(heddle_ctx* x) {
    if (!x) return;
    DeviceGuard dg(x->device);
    cudaFree(x->d_img);
    cudaFree(x->d_q);
    cudaFree(x->d_flags);
    cudaFree(x->d_counters);
    cudaFree(x->d_scratch);
    cudaFree(x->d_scratch_count);
    for (int b = 0; b < heddle_ctx::kWlSets; ++b) {
        free_worklist(x->wl[b]);
        if (x->ev_searched[b]) cudaEventDestroy(x->ev_searched[b]);
        if (x->ev_wl_free[b]) cudaEventDestroy(x->ev_wl_free[b]);
    }
    for (int b = 0; b < 4; ++b)
        if (x->s_work[b]) cudaStreamDestroy(x->s_work[b]);
    if (x->ev_in) cudaEventDestroy(x->ev_in);
    cudaFree(x->d_scratch2);
    cudaFree(x->d_scratch2_count);
    cudaFree(x->d_tickets);
    for (int b = 0; b < heddle_ctx::kStageSets; ++b) {
        cudaFree(x->st_S[b]);
        cudaFree(x->st_M[b]);
        cudaFree(x->st_code[b]);
        cudaFree(x->st_T[b]);
        cudaFree(x->st_B[b]);
        cudaFree(x->st_n[b]);
        cudaFree(x->st_status[b]);
        cudaFree(x->st_bounds[b]);
        if (x->ev_loaded[b]) cudaEventDestroy(x->ev_loaded[b]);
        if (x->ev_priced[b]) cudaEventDestroy(x->ev_priced[b]);
        if (x->ev_free[b]) cudaEventDestroy(x->ev_free[b]);
    }
    cudaFree(x->d_state);
    for (auto& v : x->lv) {
        cudaFree(v.img);
        cudaFree(v.q);
    }
    for (int i = 0; i < HEDDLE_MAX_MBS_LEVELS; ++i) {
        cudaFree(x->lv_T[i]);
        cudaFree(x->lv_B[i]);
        cudaFree(x->lv_n[i]);
        cudaFree(x->lv_status[i]);
        cudaFree(x->lv_bounds[i]);
    }
    cudaFree(x->d_timg);
    cudaFree(x->d_node_type);
    cudaFree(x->d_node_gpus);
    for (auto* b : x->plan_bounds) cudaFree(b);
    cudaFree(x->skip_mask);
    for (auto& r : x->phase_recs)
        for (cudaEvent_t ev : r.e) x->ev_pool.push_back(ev);
    for (cudaEvent_t ev : x->ev_pool) cudaEventDestroy(ev);
    if (x->s_h2d) cudaStreamDestroy(x->s_h2d);
    if (x->s_d2h) cudaStreamDestroy(x->s_d2h);
    delete x;
}

const char* heddle_last_error(const heddle_ctx* x) { return x ? x->msg : "null context"; }

heddle_status heddle_load_cluster(heddle_ctx* x, const heddle_gpu_type* types, int32_t n_types,
                                  const heddle_node* nodes, int32_t n_nodes) {
    if (!x) return HEDDLE_E_ARG;
    if (!types || !nodes) return fail(x, HEDDLE_E_ARG, "null cluster array");
    if (n_types < 1 || n_types > HEDDLE_MAX_TYPES)
        return fail(x, HEDDLE_E_LIMIT, "n_types must be in [1, %d]", HEDDLE_MAX_TYPES);
    if (n_nodes < 1) return fail(x, HEDDLE_E_ARG, "no nodes");
    for (int g = 0; g < n_types; ++g) {
        const heddle_gpu_type& t = types[g];
        if (!(t.tflops > 0.0) || !isfinite(t.tflops))
            return fail(x, HEDDLE_E_ARG, "type %d: tflops must be finite and positive", g);
        if (t.mem_bytes < 1 || t.mem_bytes > kMemLimit)
            return fail(x, HEDDLE_E_LIMIT, "type %d: mem_bytes outside [1, 2^50]", g);
        if (t.intra_bw < 1 || t.intra_bw > kBwLimit)
            return fail(x, HEDDLE_E_LIMIT, "type %d: intra_bw outside [1, 2^40]", g);
    }
    int64_t total = 0;
    for (int b = 0; b < n_nodes; ++b) {
        const heddle_node& nd = nodes[b];
        if (nd.type < 0 || nd.type >= n_types) return fail(x, HEDDLE_E_ARG, "node %d: bad type", b);
        if (nd.gpus < 1) return fail(x, HEDDLE_E_ARG, "node %d: gpus must be >= 1", b);
        if (nd.nic_bw < 1 || nd.nic_bw > kBwLimit)
            return fail(x, HEDDLE_E_LIMIT, "node %d: nic_bw outside [1, 2^40]", b);
        total += nd.gpus;
        if (total > HEDDLE_MAX_GPUS) return fail(x, HEDDLE_E_LIMIT, "more than %d GPUs", HEDDLE_MAX_GPUS);
    }
    DeviceGuard dg(x->device);
    x->types.assign(types, types + n_types);
    x->nodes.assign(nodes, nodes + n_nodes);
    x->nodes_on_device = false;
    x->have_cluster = true;
    return build_tables(x);
}

heddle_status heddle_load_model(heddle_ctx* x, const heddle_layer* layers, int32_t n_layers,
                                int64_t boundary_bytes, int32_t flags, const double* profile_s) {
    if (!x) return HEDDLE_E_ARG;
    if (!layers) return fail(x, HEDDLE_E_ARG, "layers is NULL");
    if (n_layers < 1 || n_layers > HEDDLE_MAX_LAYERS)
        return fail(x, HEDDLE_E_LIMIT, "n_layers must be in [1, %d]", HEDDLE_MAX_LAYERS);
    if (boundary_bytes < 0 || boundary_bytes > kByteLimit)
        return fail(x, HEDDLE_E_LIMIT, "boundary_bytes outside [0, 2^42]");
    if (flags & ~HEDDLE_MODEL_MOE) return fail(x, HEDDLE_E_ARG, "unknown model flags");
    for (int l = 0; l < n_layers; ++l) {
        const heddle_layer& ly = layers[l];
        if (!(ly.flops >= 0.0) || !isfinite(ly.flops))
            return fail(x, HEDDLE_E_ARG, "layer %d: flops must be finite and >= 0", l);
        const int64_t v[5] = {ly.param_bytes, ly.state_bytes, ly.act_bytes, ly.ar_bytes, ly.a2a_bytes};
        for (int i = 0; i < 5; ++i)
            if (v[i] < 0 || v[i] > kByteLimit)
                return fail(x, HEDDLE_E_LIMIT, "layer %d: byte count outside [0, 2^42]", l);
    }
    if (profile_s && !x->have_cluster)
        return fail(x, HEDDLE_E_STATE, "a profile needs the cluster loaded first");
    DeviceGuard dg(x->device);
    x->layers.assign(layers, layers + n_layers);
    x->boundary_bytes = boundary_bytes;
    x->moe = (flags & HEDDLE_MODEL_MOE) ? 1 : 0;
    x->have_profile = profile_s != nullptr;
    if (profile_s) {
        const size_t n = (size_t)x->types.size() * 4 * n_layers;
        x->profile.assign(profile_s, profile_s + n);
    } else {
        x->profile.clear();
    }
    x->have_model = true;
    // the experts' byte counts describe the previous model's layers
    x->have_experts = false;
    x->expert_state.clear();
    x->expert_param.clear();
    return build_tables(x);
}

heddle_status heddle_load_experts(heddle_ctx* x, const int64_t* expert_state, const int64_t* expert_param,
                                  int32_t n_layers) {
    if (!x) return HEDDLE_E_ARG;
    if (!expert_state && !expert_param) {
        x->have_experts = x->tiled_ready = false;
        x->expert_state.clear();
        x->expert_param.clear();
        return ok(x);
    }
    if (!expert_state || !expert_param) return fail(x, HEDDLE_E_ARG, "one of the expert arrays is NULL");
    if (!x->have_model) return fail(x, HEDDLE_E_STATE, "no model loaded");
    if (n_layers != (int32_t)x->layers.size())
        return fail(x, HEDDLE_E_ARG, "n_layers %d differs from the model's %zu layers", n_layers, x->layers.size());
    if (x->have_profile)
        return fail(x, HEDDLE_E_STATE, "expert tiling needs the synthetic cost model (the model has a profile)");
    for (int l = 0; l < n_layers; ++l) {
        if (expert_state[l] < 0 || expert_state[l] > x->layers[l].state_bytes)
            return fail(x, HEDDLE_E_ARG, "layer %d: expert_state outside [0, state_bytes]", l);
        if (expert_param[l] < 0 || expert_param[l] > x->layers[l].param_bytes)
            return fail(x, HEDDLE_E_ARG, "layer %d: expert_param outside [0, param_bytes]", l);
    }
    DeviceGuard dg(x->device);
    x->expert_state.assign(expert_state, expert_state + n_layers);
    x->expert_param.assign(expert_param, expert_param + n_layers);
    x->have_experts = true;
    const heddle_status st = build_tiled(x);
    if (st != HEDDLE_OK) {
        x->have_experts = false;
        x->expert_state.clear();
        x->expert_param.clear();
    }
    return st;
}

}  // extern "C"

namespace {

// The other worklist sets, the work streams and their events (once).
heddle_status ensure_pipeline(heddle_ctx* x) {
    if (x->pipe_ready) return HEDDLE_OK;
    cudaError_t e = cudaSuccess;
    for (int b = 1; b < heddle_ctx::kWlSets && e == cudaSuccess; ++b) e = alloc_worklist(x->wl[b]);
    for (int b = 0; b < 4 && e == cudaSuccess; ++b)
        if (!x->s_work[b]) e = cudaStreamCreateWithFlags(&x->s_work[b], cudaStreamNonBlocking);
    for (int b = 0; b < heddle_ctx::kWlSets && e == cudaSuccess; ++b) {
        if (!x->ev_searched[b]) e = cudaEventCreateWithFlags(&x->ev_searched[b], cudaEventDisableTiming);
        if (e == cudaSuccess && !x->ev_wl_free[b])
            e = cudaEventCreateWithFlags(&x->ev_wl_free[b], cudaEventDisableTiming);
    }
    if (e == cudaSuccess && !x->ev_in) e = cudaEventCreateWithFlags(&x->ev_in, cudaEventDisableTiming);
    if (e != cudaSuccess) {
        for (int b = 1; b < heddle_ctx::kWlSets; ++b) free_worklist(x->wl[b]);
        return fail(x, e == cudaErrorMemoryAllocation ? HEDDLE_E_NOMEM : HEDDLE_E_CUDA,
                    "pipeline worklist sets: %s", cudaGetErrorString(e));
    }
    x->pipe_ready = true;
    return HEDDLE_OK;
}

hd::TopkArgs topk_args(heddle_ctx* x, heddle_topk_state* state) {
    hd::TopkArgs a{};
    a.state = state;
    a.scratch = x->d_scratch;
    a.scratch_count = x->d_scratch_count;
    a.max_blocks = x->scratch_blocks;
    a.scratch2 = x->d_scratch2;
    a.scratch2_count = x->d_scratch2_count;
    a.tickets = x->d_tickets;
    return a;
}

// Five timing events for one chunk, from the pool (created on demand).
heddle_status take_phase_rec(heddle_ctx* x, heddle_ctx::PhaseRec* rec) {
    for (int i = 0; i < 5; ++i) {
        if (x->ev_pool.empty()) {
            cudaEvent_t ev;
            CU(cudaEventCreate(&ev));
            x->ev_pool.push_back(ev);
        }
        rec->e[i] = x->ev_pool.back();
        x->ev_pool.pop_back();
    }
    return HEDDLE_OK;
}

// The call-wide fields of the pricing arguments (consumes count_next).
void fill_price_args(heddle_ctx* x, const heddle_candidates* c, const heddle_ctx::Level* lvl, int shift, bool tiled,
                     hd::PriceArgs& a) {
    a.lay = lvl ? lvl->lay : x->lay;
    a.img = lvl ? lvl->img : x->d_img;
    a.mbs_shift = shift;
    a.moe = x->moe;
    a.stride = c->plane_stride;
    a.s_max = c->s_max;
    a.bstride = c->n;
    a.err = x->d_flags + 1;
    a.counters = x->count_next ? x->d_counters : nullptr;
    x->count_next = false;
    a.wl_cap = hd::kWorklistCap;
    a.uniform = !tiled && equal_layer_search(x, lvl ? lvl->flags : x->model_flags) ? 1 : 0;
    a.split_mode = x->search_mode == HEDDLE_SEARCH_DISTRIBUTE ? 1 : 0;
    a.thread_min = x->thread_min < 0 ? hd::thread_search_min(x->num_sms) : x->thread_min;
}

// One chunk [lo, lo + nb) of cands into r: screen and search on `ws` with
// worklist set W, then (with a state) the top-k over the chunk's searched
// candidates on `cs`, after the search when ws != cs.  `a` holds the
// call-wide fields; its chunk fields are set here.
heddle_status price_chunk(heddle_ctx* x, hd::PriceArgs& a, const heddle_candidates* c, const heddle_results* r,
                          int64_t lo, int64_t nb, int set, cudaStream_t ws, heddle_topk_state* state,
                          cudaStream_t cs, bool tiled, uint8_t* tiling) {
    heddle_status st;
    const heddle_ctx::Worklist& W = x->wl[set];
    a.wl_count = W.count;
    a.wl_idx = W.idx;
    a.wl_n = W.n;
    a.wl_M = W.M;
    a.wl_S = W.S;
    a.wl_memok = W.memok;
    a.wl_code = W.code;
    a.wl_bucket = W.bucket;
    a.wl_T = W.T;
    a.wl_nM = W.nM;
    // inside a top-k pricing the equal-layer search hands the top-k only the
    // entries that reach the running threshold
    const bool survivors = state && a.uniform && !a.split_mode && !tiled;
    a.sv_count = survivors ? W.count + hd::kWlSurv : nullptr;
    a.sv_idx = W.sv_idx;
    a.sv_T = W.sv_T;
    a.sv_nM = W.sv_nM;
    a.thr = x->d_flags + 2;
    a.topk_k = state ? &state->k : nullptr;
    a.S = c->S + lo;
    a.M = c->M + lo;
    a.code = c->code + lo;
    a.n = nb;
    a.T = r->T + lo;
    a.B = r->bottleneck + lo;
    a.ndp = r->n_dp + lo;
    a.status = r->status + lo;
    a.bounds = r->bounds ? r->bounds + lo : nullptr;
    heddle_ctx::PhaseRec rec{};
    if (x->time_phases) {
        if ((st = take_phase_rec(x, &rec)) != HEDDLE_OK) return st;
        rec.topk = state != nullptr;
        x->phase_recs.push_back(rec);
        CU(cudaEventRecord(rec.e[0], ws));
    }
    int64_t* nl = x->time_phases ? x->phase_recs.back().launches : nullptr;
    if (tiled) {
        hd::TiledArgs ta{};
        ta.tl = x->tlay;
        ta.timg = x->d_timg;
        ta.tiling = tiling ? tiling + lo : nullptr;
        ta.tstride = c->n;
        CU(hd::launch_screen(a, x->num_sms, ws, x->time_phases ? rec.e[1] : nullptr, nl));
        if (nl) nl[1] += 1;
        CU(hd::launch_tiled_search(a, ta, x->num_sms, ws));
    } else {
        CU(hd::launch_price(a, x->num_sms, ws, x->time_phases ? rec.e[1] : nullptr, nl));
    }
    if (x->time_phases) CU(cudaEventRecord(rec.e[2], ws));
    if (state) {
        if (ws != cs) {
            CU(cudaEventRecord(x->ev_searched[set], ws));
            CU(cudaStreamWaitEvent(cs, x->ev_searched[set], 0));
        }
        if (x->time_phases) CU(cudaEventRecord(rec.e[3], cs));
        // top-k over the searched candidates of this chunk only
        hd::TopkArgs m = topk_args(x, state);
        m.base_index = c->base_index + lo;
        m.wl_count = survivors ? W.count + hd::kWlSurv : W.count;
        m.wl_idx = survivors ? W.sv_idx : W.idx;
        m.wl_T = survivors ? W.sv_T : W.T;
        m.wl_nM = survivors ? W.sv_nM : W.nM;
        m.wl_cap = hd::kWorklistCap;
        m.thr = x->d_flags + 2;
        CU(hd::launch_topk_worklist(m, nb, x->num_sms, cs, nl ? nl + 2 : nullptr));
        if (x->time_phases) CU(cudaEventRecord(rec.e[4], cs));
    }
    return HEDDLE_OK;
}

// Price cands into r; with a state, run the top-k over each chunk's searched
// candidates (the only ones that can be OK) and merge them into *state.
// `lvl` (nullable) selects the tables of one micro-batch size and `shift`
// its log2: the screen then prices each candidate with M >> shift
// micro-batches (invalid where 2^shift does not divide M).
heddle_status price_impl(heddle_ctx* x, const heddle_candidates* c, const heddle_results* r,
                         heddle_topk_state* state, void* stream, const heddle_ctx::Level* lvl = nullptr,
                         int shift = 0, uint8_t* tiling = nullptr) {
    heddle_status st = check_cands(x, c, true);
    if (st != HEDDLE_OK) return st;
    if (!r) return fail(x, HEDDLE_E_ARG, "results is NULL");
    if ((st = check_ready(x)) != HEDDLE_OK) return st;
    if (c->n == 0) return ok(x);
    if (!r->T || !r->bottleneck || !r->n_dp || !r->status)
        return fail(x, HEDDLE_E_ARG, "null result array");
    const bool tiled = x->tiled_ready && !lvl;
    if (tiled && x->search_mode == HEDDLE_SEARCH_DISTRIBUTE)
        return fail(x, HEDDLE_E_STATE, "expert tiling prices the min-max split only (search mode DISTRIBUTE)");
    DeviceGuard dg(x->device);
    if (tiled && tiling) CU(cudaMemsetAsync(tiling, 0, (size_t)HEDDLE_MAX_STAGES * c->n, (cudaStream_t)stream));
    hd::PriceArgs a{};
    fill_price_args(x, c, lvl, shift, tiled, a);
    // chunks of at most x->chunk candidates.  With one chunk everything runs
    // on the caller's stream.  With more, chunk i runs its screen and search
    // on work stream i % 4 with worklist set i % 5 (after the caller's
    // earlier work and after chunk i - 5 released that set), and its top-k
    // on the caller's stream after its search, so the top-k merges stay in
    // chunk order while the next chunks are screened and searched meanwhile
    // (four streams: 1.00e10 candidates/s on 1e7 stress128 candidates in
    // 1e6 chunks, against 9.73e9 with two, 9.90e9 with three, 1.01e10 with
    // six and 9.83e9 with eight).
    const cudaStream_t cs = (cudaStream_t)stream;
    const int64_t chunk = x->chunk;
    const bool pipe = c->n > chunk;
    // the threshold starts at zero for each call: the state may have been
    // reset or replaced since the last one
    if (state) CU(cudaMemsetAsync(x->d_flags + 2, 0, sizeof(uint32_t), cs));
    if (pipe) {
        if ((st = ensure_pipeline(x)) != HEDDLE_OK) return st;
        CU(cudaEventRecord(x->ev_in, cs));
    }
    bool used[heddle_ctx::kWlSets] = {};
    int64_t i = 0;
    for (int64_t lo = 0; lo < c->n; lo += chunk, ++i) {
        const int64_t nb = c->n - lo < chunk ? c->n - lo : chunk;
        const int b = pipe ? (int)(i % heddle_ctx::kWlSets) : 0;
        const cudaStream_t ws = pipe ? x->s_work[i % 4] : cs;
        if (pipe) {
            CU(cudaStreamWaitEvent(ws, x->ev_in, 0));
            if (used[b]) CU(cudaStreamWaitEvent(ws, x->ev_wl_free[b], 0));
            used[b] = true;
        }
        if ((st = price_chunk(x, a, c, r, lo, nb, b, ws, state, cs, tiled, tiling)) != HEDDLE_OK) return st;
        if (pipe) CU(cudaEventRecord(x->ev_wl_free[b], state ? cs : ws));
    }
    if (pipe && !state)
        for (int b = 0; b < heddle_ctx::kWlSets; ++b)
            if (used[b]) CU(cudaStreamWaitEvent(cs, x->ev_wl_free[b], 0));
    return ok(x);
}

// One chunk of a pricing: candidates [lo, lo + nb) of c into r (offsets
// and the bounds plane stride c->n as for a call on c), with the tables of
// lvl (nullable: the main tables) at micro-batch shift `shift`.
struct PriceUnit {
    const heddle_candidates* c;
    const heddle_results* r;
    const heddle_ctx::Level* lvl;
    int shift;
    int64_t lo, nb;
    const uint8_t* skip = nullptr;  // per candidate of c: price it SKIPPED (nullable)
};

// Independent chunk pricings (no top-k, no tiling output) as one pipeline:
// they rotate over the work streams and worklist sets like the chunks of
// one call, and `stream` waits for all of them.  The units are validated
// by the caller.
heddle_status price_units(heddle_ctx* x, const PriceUnit* u, int nu, void* stream) {
    heddle_status st;
    const cudaStream_t cs = (cudaStream_t)stream;
    const bool tiled = x->tiled_ready;
    if (tiled && x->search_mode == HEDDLE_SEARCH_DISTRIBUTE)
        return fail(x, HEDDLE_E_STATE, "expert tiling prices the min-max split only (search mode DISTRIBUTE)");
    DeviceGuard dg(x->device);
    const bool pipe = nu > 1;
    if (pipe) {
        if ((st = ensure_pipeline(x)) != HEDDLE_OK) return st;
        CU(cudaEventRecord(x->ev_in, cs));
    }
    bool used[heddle_ctx::kWlSets] = {};
    for (int k = 0; k < nu; ++k) {
        if (u[k].nb <= 0) continue;
        const int b = pipe ? (k % heddle_ctx::kWlSets) : 0;
        const cudaStream_t ws = pipe ? x->s_work[k % 4] : cs;
        if (pipe) {
            CU(cudaStreamWaitEvent(ws, x->ev_in, 0));
            if (used[b]) CU(cudaStreamWaitEvent(ws, x->ev_wl_free[b], 0));
            used[b] = true;
        }
        const bool t = tiled && !u[k].lvl;
        hd::PriceArgs a{};
        fill_price_args(x, u[k].c, u[k].lvl, u[k].shift, t, a);
        a.skip = u[k].skip ? u[k].skip + u[k].lo : nullptr;
        if ((st = price_chunk(x, a, u[k].c, u[k].r, u[k].lo, u[k].nb, b, ws, nullptr, cs, t, nullptr)) != HEDDLE_OK)
            return st;
        if (pipe) CU(cudaEventRecord(x->ev_wl_free[b], ws));
    }
    if (pipe)
        for (int b = 0; b < heddle_ctx::kWlSets; ++b)
            if (used[b]) CU(cudaStreamWaitEvent(cs, x->ev_wl_free[b], 0));
    return ok(x);
}

}  // namespace

extern "C" {

heddle_status heddle_price_candidates(heddle_ctx* x, const heddle_candidates* c,
                                      const heddle_results* r, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    return price_impl(x, c, r, nullptr, stream);
}

heddle_status heddle_price_tiled(heddle_ctx* x, const heddle_candidates* c, const heddle_results* r,
                                 uint8_t* tiling, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    if (!x->tiled_ready) return fail(x, HEDDLE_E_STATE, "no experts loaded (heddle_load_experts)");
    return price_impl(x, c, r, nullptr, stream, nullptr, 0, tiling);
}

heddle_status heddle_price_topk(heddle_ctx* x, const heddle_candidates* c, const heddle_results* r,
                                heddle_topk_state* state, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    if (!state) return fail(x, HEDDLE_E_ARG, "state is NULL");
    return price_impl(x, c, r, state, stream);
}

heddle_status heddle_topk_reset(heddle_ctx* x, heddle_topk_state* state, int32_t k, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    if (!state) return fail(x, HEDDLE_E_ARG, "state is NULL");
    if (k < 1 || k > HEDDLE_MAX_TOPK) return fail(x, HEDDLE_E_LIMIT, "k must be in [1, %d]", HEDDLE_MAX_TOPK);
    DeviceGuard dg(x->device);
    CU(hd::launch_topk_reset(state, k, (cudaStream_t)stream));
    return ok(x);
}

heddle_status heddle_topk(heddle_ctx* x, const heddle_candidates* c, const heddle_results* r,
                          heddle_topk_state* state, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    heddle_status st = check_cands(x, c, true);
    if (st != HEDDLE_OK) return st;
    if (!r || !state) return fail(x, HEDDLE_E_ARG, "results or state is NULL");
    if (c->n == 0) return ok(x);
    if (!r->T || !r->n_dp || !r->status) return fail(x, HEDDLE_E_ARG, "null result array");
    DeviceGuard dg(x->device);
    hd::TopkArgs a = topk_args(x, state);
    a.M = c->M;
    a.T = r->T;
    a.ndp = r->n_dp;
    a.status = r->status;
    a.n = c->n;
    a.base_index = c->base_index;
    CU(hd::launch_topk(a, x->num_sms, (cudaStream_t)stream));
    return ok(x);
}

heddle_status heddle_price_topk_host(heddle_ctx* x, const heddle_candidates* c,
                                     const heddle_results* r, heddle_topk_state* state,
                                     int64_t batch, void* stream) {
    if (!x) return HEDDLE_E_ARG;
    heddle_status st = check_cands(x, c, false);
    if (st != HEDDLE_OK) return st;
    if (!state) return fail(x, HEDDLE_E_ARG, "state is NULL");
    if (state->k < 1 || state->k > HEDDLE_MAX_TOPK)
        return fail(x, HEDDLE_E_LIMIT, "state k must be in [1, %d]", HEDDLE_MAX_TOPK);
    if (batch < 1) return fail(x, HEDDLE_E_ARG, "batch must be >= 1");
    if (batch > hd::kWorklistCap) return fail(x, HEDDLE_E_LIMIT, "batch must be at most %d", hd::kWorklistCap);
    if ((st = check_ready(x)) != HEDDLE_OK) return st;
    const bool tiled = x->tiled_ready;
    if (tiled && x->search_mode == HEDDLE_SEARCH_DISTRIBUTE)
        return fail(x, HEDDLE_E_STATE, "expert tiling prices the min-max split only (search mode DISTRIBUTE)");
    DeviceGuard dg(x->device);
    if ((st = ensure_pipeline(x)) != HEDDLE_OK) return st;
    cudaStream_t sc = (cudaStream_t)stream;
    const int64_t n = c->n;
    const int64_t nb_max = n < batch ? (n > 0 ? n : 1) : batch;
    // staging buffers (grown on demand) and the copy streams / events
    if (!x->s_h2d) {
        CU(cudaStreamCreateWithFlags(&x->s_h2d, cudaStreamNonBlocking));
        CU(cudaStreamCreateWithFlags(&x->s_d2h, cudaStreamNonBlocking));
        for (int b = 0; b < heddle_ctx::kStageSets; ++b) {
            CU(cudaEventCreateWithFlags(&x->ev_loaded[b], cudaEventDisableTiming));
            CU(cudaEventCreateWithFlags(&x->ev_priced[b], cudaEventDisableTiming));
            CU(cudaEventCreateWithFlags(&x->ev_free[b], cudaEventDisableTiming));
        }
        CU(cudaMalloc(&x->d_state, sizeof(heddle_topk_state)));
    }
    if (x->stage_cap < nb_max || x->stage_smax < c->s_max) {
        CU(cudaDeviceSynchronize());
        const int64_t cap = nb_max > x->stage_cap ? nb_max : x->stage_cap;
        const int32_t sm = c->s_max > x->stage_smax ? c->s_max : x->stage_smax;
        for (int b = 0; b < heddle_ctx::kStageSets; ++b) {
            cudaFree(x->st_S[b]);
            cudaFree(x->st_M[b]);
            cudaFree(x->st_code[b]);
            cudaFree(x->st_T[b]);
            cudaFree(x->st_B[b]);
            cudaFree(x->st_n[b]);
            cudaFree(x->st_status[b]);
            cudaFree(x->st_bounds[b]);
            x->st_S[b] = nullptr;
            x->st_M[b] = nullptr;
            x->st_code[b] = nullptr;
            x->st_T[b] = x->st_B[b] = nullptr;
            x->st_n[b] = nullptr;
            x->st_status[b] = x->st_bounds[b] = nullptr;
            if (cudaMalloc(&x->st_S[b], cap) != cudaSuccess ||
                cudaMalloc(&x->st_M[b], 2 * cap) != cudaSuccess ||
                cudaMalloc(&x->st_code[b], (size_t)sm * cap) != cudaSuccess ||
                cudaMalloc(&x->st_T[b], 8 * cap) != cudaSuccess ||
                cudaMalloc(&x->st_B[b], 8 * cap) != cudaSuccess ||
                cudaMalloc(&x->st_n[b], 2 * cap) != cudaSuccess ||
                cudaMalloc(&x->st_status[b], cap) != cudaSuccess ||
                cudaMalloc(&x->st_bounds[b], (size_t)HEDDLE_BOUND_PLANES * cap) != cudaSuccess) {
                x->stage_cap = 0;
                x->stage_smax = 0;
                return fail(x, HEDDLE_E_NOMEM, "staging buffers for %lld candidates", (long long)cap);
            }
        }
        x->stage_cap = cap;
        x->stage_smax = sm;
    }
    CU(cudaMemcpyAsync(x->d_state, state, sizeof(heddle_topk_state), cudaMemcpyHostToDevice, sc));
    CU(cudaMemsetAsync(x->d_flags + 2, 0, sizeof(uint32_t), sc));
    for (int b = 0; b < heddle_ctx::kStageSets; ++b) CU(cudaEventRecord(x->ev_free[b], sc));
    const bool want_bounds = r && r->bounds;
    // batch k: copies in on s_h2d into staging set k % 3 (free once batch
    // k - 3 is copied out), screen and search on work stream k % 2 (worklist
    // set k % 5, released by batch k - 5's top-k), top-k merge on the
    // caller's stream in batch order, copies out on s_d2h
    bool used[heddle_ctx::kWlSets] = {};
    for (int64_t lo = 0, it = 0; lo < n; lo += batch, ++it) {
        const int b = (int)(it % heddle_ctx::kStageSets);
        const int wb = (int)(it % heddle_ctx::kWlSets);
        const int64_t nb = (n - lo) < batch ? (n - lo) : batch;
        // host -> device on the copy stream once the set is free
        CU(cudaStreamWaitEvent(x->s_h2d, x->ev_free[b], 0));
        CU(cudaMemcpyAsync(x->st_S[b], c->S + lo, nb, cudaMemcpyHostToDevice, x->s_h2d));
        CU(cudaMemcpyAsync(x->st_M[b], c->M + lo, 2 * nb, cudaMemcpyHostToDevice, x->s_h2d));
        CU(cudaMemcpy2DAsync(x->st_code[b], nb, c->code + lo, c->plane_stride, nb, c->s_max,
                             cudaMemcpyHostToDevice, x->s_h2d));
        CU(cudaEventRecord(x->ev_loaded[b], x->s_h2d));
        const cudaStream_t ws = x->s_work[it & 1];
        CU(cudaStreamWaitEvent(ws, x->ev_loaded[b], 0));
        if (used[wb]) CU(cudaStreamWaitEvent(ws, x->ev_wl_free[wb], 0));
        used[wb] = true;
        heddle_candidates cb{};
        cb.S = x->st_S[b];
        cb.M = x->st_M[b];
        cb.code = x->st_code[b];
        cb.n = nb;
        cb.plane_stride = nb;
        cb.s_max = c->s_max;
        cb.base_index = c->base_index + lo;
        heddle_results rb{};
        rb.T = x->st_T[b];
        rb.bottleneck = x->st_B[b];
        rb.n_dp = x->st_n[b];
        rb.status = x->st_status[b];
        rb.bounds = want_bounds ? x->st_bounds[b] : nullptr;
        if (nb > 0) {
            hd::PriceArgs a{};
            fill_price_args(x, &cb, nullptr, 0, tiled, a);
            if ((st = price_chunk(x, a, &cb, &rb, 0, nb, wb, ws, x->d_state, sc, tiled, nullptr)) != HEDDLE_OK)
                return st;
        }
        CU(cudaEventRecord(x->ev_wl_free[wb], sc));
        CU(cudaEventRecord(x->ev_priced[b], sc));
        // device -> host of the requested result fields on the second copy stream
        CU(cudaStreamWaitEvent(x->s_d2h, x->ev_priced[b], 0));
        if (r && r->T) CU(cudaMemcpyAsync(r->T + lo, rb.T, 8 * nb, cudaMemcpyDeviceToHost, x->s_d2h));
        if (r && r->bottleneck)
            CU(cudaMemcpyAsync(r->bottleneck + lo, rb.bottleneck, 8 * nb, cudaMemcpyDeviceToHost, x->s_d2h));
        if (r && r->n_dp) CU(cudaMemcpyAsync(r->n_dp + lo, rb.n_dp, 2 * nb, cudaMemcpyDeviceToHost, x->s_d2h));
        if (r && r->status)
            CU(cudaMemcpyAsync(r->status + lo, rb.status, nb, cudaMemcpyDeviceToHost, x->s_d2h));
        if (want_bounds)
            CU(cudaMemcpy2DAsync(r->bounds + lo, n, rb.bounds, nb, nb, HEDDLE_BOUND_PLANES,
                                 cudaMemcpyDeviceToHost, x->s_d2h));
        CU(cudaEventRecord(x->ev_free[b], x->s_d2h));
    }
    CU(cudaMemcpyAsync(state, x->d_state, sizeof(heddle_topk_state), cudaMemcpyDeviceToHost, sc));
    CU(cudaStreamSynchronize(x->s_d2h));
    CU(cudaStreamSynchronize(x->s_h2d));
    CU(cudaStreamSynchronize(sc));
    return ok(x);
}

heddle_status heddle_get_tables(heddle_ctx* x, int64_t* q, int64_t* p2p) {
    if (!x) return HEDDLE_E_ARG;
    heddle_status st = check_ready(x);
    if (st != HEDDLE_OK) return st;
    DeviceGuard dg(x->device);
    if (q)
        CU(cudaMemcpy(q, x->d_q, sizeof(int64_t) * (size_t)x->lay.NT * 4 * x->lay.L,
                      cudaMemcpyDeviceToHost));
    if (p2p) CU(cudaMemcpy(p2p, x->d_img + x->lay.offP2P, sizeof(int64_t) * 128, cudaMemcpyDeviceToHost));
    return ok(x);
}

heddle_status heddle_device_errors(heddle_ctx* x, uint32_t* flags) {
    if (!x || !flags) return x ? fail(x, HEDDLE_E_ARG, "flags is NULL") : HEDDLE_E_ARG;
    DeviceGuard dg(x->device);
    CU(cudaDeviceSynchronize());
    CU(cudaMemcpy(flags, x->d_flags + 1, sizeof(uint32_t), cudaMemcpyDeviceToHost));
    CU(cudaMemset(x->d_flags + 1, 0, sizeof(uint32_t)));
    return ok(x);
}

heddle_status heddle_set_search(heddle_ctx* x, int32_t mode) {
    if (!x) return HEDDLE_E_ARG;
    if (mode != HEDDLE_SEARCH_AUTO && mode != HEDDLE_SEARCH_GENERAL && mode != HEDDLE_SEARCH_DISTRIBUTE)
        return fail(x, HEDDLE_E_ARG, "unknown search mode %d", mode);
    x->search_mode = mode;
    return ok(x);
}

heddle_status heddle_set_thread_search_min(heddle_ctx* x, int32_t min_entries) {
    if (!x) return HEDDLE_E_ARG;
    x->thread_min = min_entries < 0 ? -1 : min_entries;
    return ok(x);
}

heddle_status heddle_get_search(heddle_ctx* x, int32_t* in_use) {
    if (!x || !in_use) return x ? fail(x, HEDDLE_E_ARG, "in_use is NULL") : HEDDLE_E_ARG;
    heddle_status st = check_ready(x);
    if (st != HEDDLE_OK) return st;
    *in_use = x->search_mode == HEDDLE_SEARCH_DISTRIBUTE ? HEDDLE_SEARCH_DISTRIBUTE
              : x->tiled_ready                        ? HEDDLE_SEARCH_TILED
              : equal_layer_search(x)                 ? HEDDLE_SEARCH_EQUAL_LAYERS
                                                      : HEDDLE_SEARCH_GENERAL;
    return ok(x);
}

heddle_status heddle_count_next(heddle_ctx* x, int32_t enable) {
    if (!x) return HEDDLE_E_ARG;
    x->count_next = enable != 0;
    return ok(x);
}

heddle_status heddle_load_mbs(heddle_ctx* x, int32_t levels, const double* profile_s) {
    if (!x) return HEDDLE_E_ARG;
    if (levels < 0 || levels > HEDDLE_MAX_MBS_LEVELS)
        return fail(x, HEDDLE_E_LIMIT, "levels must be in [0, %d]", HEDDLE_MAX_MBS_LEVELS);
    if (profile_s && (!x->have_cluster || !x->have_model))
        return fail(x, HEDDLE_E_STATE, "size profiles need the cluster and the model loaded first");
    DeviceGuard dg(x->device);
    x->mbs_levels = levels;
    if (profile_s && levels > 0) {
        const size_t n = (size_t)levels * x->types.size() * 4 * x->layers.size();
        for (size_t i = 0; i < n; ++i)
            if (!(profile_s[i] >= 0.0) || !isfinite(profile_s[i]))
                return fail(x, HEDDLE_E_ARG, "size profile entry %zu is negative or not finite", i);
        x->mbs_profile.assign(profile_s, profile_s + n);
    } else {
        x->mbs_profile.clear();
    }
    return build_levels(x);
}

heddle_status heddle_price_mbs(heddle_ctx* x, const heddle_candidates* c, const heddle_results* r, uint8_t* mbs,
                               void* stream) {
    if (!x) return HEDDLE_E_ARG;
    heddle_status st = check_cands(x, c, true);
    if (st != HEDDLE_OK) return st;
    if (!r) return fail(x, HEDDLE_E_ARG, "results is NULL");
    if ((st = check_ready(x)) != HEDDLE_OK) return st;
    if (x->mbs_levels < 1 || !x->mbs_ready) return fail(x, HEDDLE_E_STATE, "no micro-batch sizes loaded");
    if (x->tiled_ready) return fail(x, HEDDLE_E_STATE, "the micro-batch-size fill does not combine with expert tiling");
    if (c->n == 0) return ok(x);
    if (!r->T || !r->bottleneck || !r->n_dp || !r->status) return fail(x, HEDDLE_E_ARG, "null result array");
    DeviceGuard dg(x->device);
    cudaStream_t sm = (cudaStream_t)stream;
    if (mbs) CU(cudaMemsetAsync(mbs, 0, (size_t)c->n, sm));
    const int nl = x->mbs_levels;
    const size_t cap = (size_t)std::min<int64_t>(c->n, x->chunk);
    for (int i = 1; i < nl; ++i) {
        CU(grow(&x->lv_T[i], &x->lv_T_cap[i], sizeof(int64_t) * cap));
        CU(grow(&x->lv_B[i], &x->lv_B_cap[i], sizeof(int64_t) * cap));
        CU(grow(&x->lv_n[i], &x->lv_n_cap[i], sizeof(uint16_t) * cap));
        CU(grow(&x->lv_status[i], &x->lv_status_cap[i], cap));
        if (r->bounds) CU(grow(&x->lv_bounds[i], &x->lv_bounds_cap[i], (size_t)(HEDDLE_MAX_STAGES + 1) * cap));
    }
    // per chunk: every size priced as one pipeline (the base size straight
    // into the caller's results, each larger size into its own set), then
    // the larger sizes folded into the results in order
    for (int64_t lo = 0; lo < c->n; lo += x->chunk) {
        const int64_t nb = std::min<int64_t>(c->n - lo, x->chunk);
        heddle_candidates cc = *c;
        cc.S = c->S + lo;
        cc.M = c->M + lo;
        cc.code = c->code + lo;
        cc.n = nb;
        cc.base_index = c->base_index + lo;
        heddle_results rs[HEDDLE_MAX_MBS_LEVELS];
        PriceUnit units[HEDDLE_MAX_MBS_LEVELS];
        for (int i = 0; i < nl; ++i) {
            if (i == 0) {
                // the base size straight into the caller's results
                units[0] = PriceUnit{c, r, &x->lv[0], 0, lo, nb};
            } else {
                // a larger size into its own set, laid out for this chunk
                rs[i] = heddle_results{x->lv_T[i], x->lv_B[i], x->lv_n[i], x->lv_status[i],
                                       r->bounds ? x->lv_bounds[i] : nullptr};
                units[i] = PriceUnit{&cc, &rs[i], &x->lv[i], i, 0, nb};
            }
        }
        if ((st = price_units(x, units, nl, stream)) != HEDDLE_OK) return st;
        for (int i = 1; i < nl; ++i) {
            hd::MbsMergeArgs m{};
            m.n = nb;
            m.T_l = x->lv_T[i];
            m.B_l = x->lv_B[i];
            m.n_l = x->lv_n[i];
            m.status_l = x->lv_status[i];
            m.bounds_l = r->bounds ? x->lv_bounds[i] : nullptr;
            m.bstride_l = nb;
            m.T = r->T + lo;
            m.B = r->bottleneck + lo;
            m.ndp = r->n_dp + lo;
            m.status = r->status + lo;
            m.bounds = r->bounds ? r->bounds + lo : nullptr;
            m.bstride = c->n;
            m.mbs = mbs ? mbs + lo : nullptr;
            m.level = i;
            CU(hd::launch_mbs_merge(m, x->num_sms, sm));
        }
    }
    return ok(x);
}

heddle_status heddle_price_plans(heddle_ctx* x, const heddle_plans* pl, const heddle_plan_results* pr,
                                 void* stream) {
    if (!x) return HEDDLE_E_ARG;
    if (!pl || !pr) return fail(x, HEDDLE_E_ARG, "plans or results is NULL");
    heddle_status st = check_ready(x);
    if (st != HEDDLE_OK) return st;
    if (x->tiled_ready) return fail(x, HEDDLE_E_STATE, "plan pricing does not combine with expert tiling");
    if (pl->n < 0) return fail(x, HEDDLE_E_ARG, "negative plan count");
    if (pl->n > hd::kWorklistCap) return fail(x, HEDDLE_E_LIMIT, "more than 2^20 plans in one call");
    if (pl->slots < 1 || pl->slots > HEDDLE_MAX_TEMPLATES)
        return fail(x, HEDDLE_E_ARG, "slots must be in [1, %d]", HEDDLE_MAX_TEMPLATES);
    if (pl->n == 0) return ok(x);
    if (!pl->n_templates || !pr->placed || !pr->thr) return fail(x, HEDDLE_E_ARG, "null plan array");
    for (int t = 0; t < pl->slots; ++t) {
        if (pl->t[t].n != pl->n) return fail(x, HEDDLE_E_ARG, "slot %d holds %lld candidates, not n", t,
                                             (long long)pl->t[t].n);
        if ((st = check_cands(x, &pl->t[t], true)) != HEDDLE_OK) return st;
        const heddle_results& r = pr->t[t];
        if (!r.T || !r.bottleneck || !r.n_dp || !r.status) return fail(x, HEDDLE_E_ARG, "null result array, slot %d", t);
    }
    for (const auto& nd : x->nodes)
        if (nd.gpus > HEDDLE_PLAN_MAX_NODE)
            return fail(x, HEDDLE_E_LIMIT, "plans need nodes of at most %d GPUs", HEDDLE_PLAN_MAX_NODE);
    DeviceGuard dg(x->device);
    cudaStream_t sm = (cudaStream_t)stream;
    const size_t nn = x->nodes.size();
    int32_t vmax = 1;
    for (const auto& nd : x->nodes) vmax = std::max(vmax, nd.gpus);
    if (!x->nodes_on_device) {
        // once per loaded cluster (a synchronous copy)
        CU(grow(&x->d_node_type, &x->node_cap, sizeof(int32_t) * nn));
        CU(grow(&x->d_node_gpus, &x->node_cap2, sizeof(int32_t) * nn));
        std::vector<int32_t> ty(nn), gp(nn);
        for (size_t b = 0; b < nn; ++b) {
            ty[b] = x->nodes[b].type;
            gp[b] = x->nodes[b].gpus;
        }
        CU(cudaMemcpy(x->d_node_type, ty.data(), sizeof(int32_t) * nn, cudaMemcpyHostToDevice));
        CU(cudaMemcpy(x->d_node_gpus, gp.data(), sizeof(int32_t) * nn, cudaMemcpyHostToDevice));
        x->nodes_on_device = true;
    }
    hd::PlanArgs a{};
    a.lay = x->lay;
    a.img = x->d_img;
    a.n = pl->n;
    a.slots = pl->slots;
    a.n_tmpl = pl->n_templates;
    a.node_type = x->d_node_type;
    a.node_gpus = x->d_node_gpus;
    a.n_nodes = (int32_t)nn;
    a.vmax = vmax;
    a.placed = pr->placed;
    a.thr = pr->thr;
    a.err = x->d_flags + 1;
    // the slots priced as standalone candidates, slot by slot: slot t only
    // for the plans whose templates 0 .. t-1 are each OK alone (the mask
    // reads slot t - 1's statuses), the chunks of a slot pipelined over the
    // work streams.  The walk re-evaluates templates after the first from
    // their splits, so those slots need bounds
    heddle_results rs[HEDDLE_MAX_TEMPLATES];
    CU(grow(&x->skip_mask, &x->skip_mask_cap, (size_t)pl->n));
    for (int t = 0; t < pl->slots; ++t) {
        rs[t] = pr->t[t];
        if (!rs[t].bounds && t > 0) {
            CU(grow(&x->plan_bounds[t], &x->plan_bounds_cap[t], (size_t)(HEDDLE_MAX_STAGES + 1) * pl->n));
            rs[t].bounds = x->plan_bounds[t];
        }
        CU(hd::launch_plan_mask(pl->n_templates, pl->slots, t, t > 0 ? rs[t - 1].status : nullptr, x->skip_mask,
                                pl->n, x->num_sms, sm));
        std::vector<PriceUnit> units;
        for (int64_t lo = 0; lo < pl->n; lo += x->chunk) {
            PriceUnit u{&pl->t[t], &rs[t], nullptr, 0, lo, std::min<int64_t>(x->chunk, pl->n - lo)};
            u.skip = x->skip_mask;
            units.push_back(u);
        }
        if ((st = price_units(x, units.data(), (int)units.size(), stream)) != HEDDLE_OK) return st;
    }
    for (int t = 0; t < pl->slots; ++t) {
        const heddle_results& r = rs[t];
        hd::PlanSlot& s = a.slot[t];
        s.S = pl->t[t].S;
        s.M = pl->t[t].M;
        s.code = pl->t[t].code;
        s.stride = pl->t[t].plane_stride;
        s.T = r.T;
        s.B = r.bottleneck;
        s.ndp = r.n_dp;
        s.status = r.status;
        s.bounds = r.bounds;
        s.bstride = pl->n;
    }
    CU(hd::launch_plans(a, x->num_sms, sm));
    return ok(x);
}

heddle_status heddle_set_chunk(heddle_ctx* x, int64_t chunk) {
    if (!x) return HEDDLE_E_ARG;
    if (chunk < 1 || chunk > hd::kWorklistCap)
        return fail(x, HEDDLE_E_LIMIT, "chunk must be in [1, %d]", hd::kWorklistCap);
    x->chunk = chunk;
    return ok(x);
}

heddle_status heddle_time_phases(heddle_ctx* x, int32_t enable) {
    if (!x) return HEDDLE_E_ARG;
    x->time_phases = enable != 0;
    return ok(x);
}

heddle_status heddle_phase_times(heddle_ctx* x, double ms[HEDDLE_N_PHASES], int64_t launches[HEDDLE_N_PHASES]) {
    if (!x || !ms || !launches) return x ? fail(x, HEDDLE_E_ARG, "null output") : HEDDLE_E_ARG;
    DeviceGuard dg(x->device);
    for (int p = 0; p < HEDDLE_N_PHASES; ++p) {
        ms[p] = 0.0;
        launches[p] = 0;
    }
    heddle_status st = HEDDLE_OK;
    // screen e0 -> e1, search e1 -> e2, top-k e3 -> e4 (its own start: with
    // several chunks the top-k runs on another stream than the search)
    static const int from[HEDDLE_N_PHASES] = {0, 1, 3}, to[HEDDLE_N_PHASES] = {1, 2, 4};
    for (auto& r : x->phase_recs) {
        const int np = r.topk ? 3 : 2;
        cudaError_t e = cudaEventSynchronize(r.e[r.topk ? 4 : 2]);
        for (int p = 0; p < np && e == cudaSuccess; ++p) {
            float t = 0.f;
            e = cudaEventElapsedTime(&t, r.e[from[p]], r.e[to[p]]);
            ms[p] += t;
            launches[p] += r.launches[p];
        }
        if (e != cudaSuccess && st == HEDDLE_OK)
            st = fail(x, HEDDLE_E_CUDA, "phase timing: %s", cudaGetErrorString(e));
        for (cudaEvent_t ev : r.e) x->ev_pool.push_back(ev);
    }
    x->phase_recs.clear();
    return st == HEDDLE_OK ? ok(x) : st;
}

heddle_status heddle_work_counters(heddle_ctx* x, uint64_t out[3]) {
    if (!x || !out) return x ? fail(x, HEDDLE_E_ARG, "out is NULL") : HEDDLE_E_ARG;
    DeviceGuard dg(x->device);
    unsigned long long v[3];
    CU(cudaDeviceSynchronize());
    CU(cudaMemcpy(v, x->d_counters, sizeof(v), cudaMemcpyDeviceToHost));
    CU(cudaMemset(x->d_counters, 0, sizeof(v)));
    for (int i = 0; i < 3; ++i) out[i] = v[i];
    return ok(x);
}

}  // extern "C"
