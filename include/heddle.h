/*
 * heddle.h -- C ABI of the GB300 (sm_103a) batched candidate-plan pricer.
 *
 * The operation is the inner loop of a parallelism planner (paper
 * arxiv 2609.34244): for every candidate pipeline structure -- a depth S and,
 * per stage, a GPU type and a TP degree (the "structural template" of §5.1) --
 * find the DP replication count the node packing admits (§5.3), split the
 * model's layers into S contiguous stages minimising the slowest stage under
 * per-GPU memory limits (PartitionLayers of the §3.1 search listing, memory
 * validation of §5.2), price the 1F1B iteration time
 *     T = (M - 1) * max_s t_s + sum_s t_s + max_s g_s         (§5.3)
 * with inter-stage P2P inside t_s and the DP gradient synchronisation g_s,
 * and rank the candidates by throughput n * M / T (§5 overview).
 *
 * All pricing arithmetic after the cost-table build is integer: times in
 * int64 nanoseconds, sizes in int64 bytes, bandwidths in int64 bytes/s.
 * Results are bit-exact and independent of launch configuration.
 *
 * Conventions for every entry point:
 *   - returns heddle_status; never aborts the process;
 *   - a context is not thread-safe: one host thread uses it at a time;
 *   - "device" pointers are CUDA device (or managed) memory on the context's
 *     device, owned by the caller; the library keeps no reference after the
 *     call returns (asynchronous calls read and write them on the stream);
 *   - "stream" is a cudaStream_t (NULL = legacy default stream);
 *   - per-candidate problems are data, reported in the status plane, not
 *     call errors.
 */
#ifndef HEDDLE_H
#define HEDDLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define HEDDLE_MAX_TYPES 8      /* GPU types per cluster */
#define HEDDLE_MAX_STAGES 32    /* pipeline depth S */
#define HEDDLE_MAX_LAYERS 255   /* model layers L (boundaries fit in a byte) */
#define HEDDLE_MAX_GPUS 65535   /* GPUs per cluster (DP degree fits in uint16) */
#define HEDDLE_MAX_TOPK 64
#define HEDDLE_BOUND_PLANES (HEDDLE_MAX_STAGES + 1)

typedef enum {
    HEDDLE_OK = 0,
    HEDDLE_E_ARG = 1,    /* null pointer, negative size, malformed record */
    HEDDLE_E_STATE = 2,  /* cluster or model not loaded, or mismatched */
    HEDDLE_E_LIMIT = 3,  /* a size or value exceeds a documented limit */
    HEDDLE_E_CUDA = 4,   /* a CUDA runtime call failed (message has details) */
    HEDDLE_E_NOMEM = 5   /* device or host allocation failed */
} heddle_status;

/* Per-candidate status (uint8 plane). */
enum {
    HEDDLE_CAND_OK = 0,
    HEDDLE_CAND_OOM = 1,     /* no layer split fits the GPUs' memory (§5.2) */
    HEDDLE_CAND_NO_FIT = 2,  /* not one replica can be placed on the nodes */
    HEDDLE_CAND_INVALID = 3, /* masked structure (§5.1): see heddle_price_candidates */
    HEDDLE_CAND_SKIPPED = 4  /* a plan's template after the plan ended (heddle_price_plans) */
};

typedef struct heddle_ctx heddle_ctx;

/* Create a context on CUDA device `device`.  Allocates its device scratch
 * once (about 190 MB: the search worklist of 2^20 candidates with their 32
 * stage bytes, its per-depth index lists and the top-k merge lists) and
 * queries the SM count.
 * *out is NULL on failure. */
heddle_status heddle_create(heddle_ctx** out, int32_t device);

/* Free the context and all device memory it owns.  NULL is ignored. */
void heddle_destroy(heddle_ctx* ctx);

/* Message of the last failed call on ctx (never NULL; "" after success).
 * The buffer belongs to ctx and is overwritten by the next call. */
const char* heddle_last_error(const heddle_ctx* ctx);

/* ------------------------------------------------------------- cluster */

/* One GPU type (§5.1 "normalized hardware attributes"): peak dense TFLOPS,
 * memory per GPU in bytes, intra-node link bandwidth in bytes/s. */
typedef struct {
    double tflops;
    int64_t mem_bytes;
    int64_t intra_bw;
} heddle_gpu_type;

/* One node (§5.1 "a node list per GPU type"): type index, GPU count,
 * inter-node NIC bandwidth in bytes/s. */
typedef struct {
    int32_t type;
    int32_t gpus;
    int64_t nic_bw;
} heddle_node;

/* Load the GPU composition.  Host arrays, copied before return.
 * Limits: 1 <= n_types <= 8; n_nodes >= 1; every node: 0 <= type < n_types,
 * gpus >= 1, 1 <= nic_bw <= 2^40; total GPUs <= 65535; tflops finite > 0;
 * 1 <= mem_bytes <= 2^50; 1 <= intra_bw <= 2^40.  Types without nodes are
 * allowed (candidates using them are INVALID).  Rebuilds the cost tables if
 * a model is loaded (synchronous: the call returns after the device tables
 * are ready). */
heddle_status heddle_load_cluster(heddle_ctx* ctx, const heddle_gpu_type* types,
                                  int32_t n_types, const heddle_node* nodes,
                                  int32_t n_nodes);

/* --------------------------------------------------------------- model */

/* One layer (§5.2 "one layer per repeated structure"):
 *   flops        forward+backward FLOPs for one microbatch
 *   param_bytes  gradient bytes the DP all-reduce synchronises
 *   state_bytes  parameters + gradients + optimizer state held for the layer
 *   act_bytes    activation bytes kept per in-flight microbatch
 *   ar_bytes     message of each of the layer's four TP all-reduces
 *   a2a_bytes    message of each of the layer's four EP all-to-alls (0: dense) */
typedef struct {
    double flops;
    int64_t param_bytes;
    int64_t state_bytes;
    int64_t act_bytes;
    int64_t ar_bytes;
    int64_t a2a_bytes;
} heddle_layer;

#define HEDDLE_MODEL_MOE 1 /* stage degree is an EP degree; may exceed a node */

/* Load the model.  Host arrays, copied before return.
 * boundary_bytes: activation bytes crossing a stage boundary per microbatch.
 * profile_s: nullable [n_types][4][n_layers] seconds per layer at degree
 *   2^j (computation plus communication, §5.2 profile entries); replaces the
 *   synthetic formula and requires the cluster to be loaded first.
 * Per-layer cost in ns (synthetic profile, degree k = 2^j, type g):
 *   s = flops / (k * tflops_g * 1e12)
 *   k > 1: s += 4 * (2(k-1)/k) * ar_bytes / bw  and  s += 4 * ((k-1)/k) * a2a_bytes / bw
 *   bw = intra_bw_g if k <= largest node of g, else the slowest NIC of g
 *   q = nearest integer of s * 1e9, halves away from zero
 * evaluated left to right in IEEE double without fused multiply-add.
 * Limits: 1 <= n_layers <= 255; all byte counts in [0, 2^42]; flops finite
 * >= 0; every per-(type, degree) total of q <= 2^40 ns; P2P and gradient
 * terms must stay below 2^40 / 2^56 ns (E_LIMIT otherwise). */
heddle_status heddle_load_model(heddle_ctx* ctx, const heddle_layer* layers, int32_t n_layers,
                                int64_t boundary_bytes, int32_t flags,
                                const double* profile_s);

/* ---------------------------------------------------------- candidates */

/* Candidate batch, structure of arrays in device memory.
 *   S[n]       stage count (uint8)
 *   M[n]       microbatches per iteration (uint16)
 *   code       stage bytes, stage-major: stage s of candidate c at
 *              code[s * plane_stride + c], for s < s_max; byte = type
 *              (bits 0-2) | log2 degree (bits 3-4); bits 5-7 must be 0
 *   base_index global index of candidate 0 (used by the top-k) */
typedef struct {
    const uint8_t* S;
    const uint16_t* M;
    const uint8_t* code;
    int64_t n;
    int64_t plane_stride;
    int32_t s_max;
    int32_t reserved;
    int64_t base_index;
} heddle_candidates;

/* Per-candidate results in device memory (caller-owned, n entries each).
 *   T           iteration time, ns (-1 unless status OK)
 *   bottleneck  min-max stage time B* = max_s t_s, ns (-1 unless OK)
 *   n_dp        DP replication count (0 for INVALID / NO_FIT)
 *   status      HEDDLE_CAND_*
 *   bounds      nullable, [33][n] uint8: stage boundaries a_0..a_S of the
 *               canonical split (plane s at bounds[s * n + c]); all zero
 *               unless OK.  Among all splits attaining B* the canonical one
 *               is the lexicographically smallest boundary vector. */
typedef struct {
    int64_t* T;
    int64_t* bottleneck;
    uint16_t* n_dp;
    uint8_t* status;
    uint8_t* bounds;
} heddle_results;

/* Price a batch (PartitionLayers + Evaluate, §3.1, §5.2, §5.3).
 * Asynchronous on `stream`; no host round-trip.  Each chunk of the batch
 * (heddle_set_chunk, default and at most 2^20 candidates) takes two
 * launches: a screen (masks, DP degree, memory) that compacts the
 * candidates needing the threshold search into a worklist owned by the
 * context, then the search over that worklist.  A batch of one chunk runs
 * on `stream` and allocates nothing.  A batch of several chunks
 * rotates five worklist sets over four context-owned work streams, so
 * the next chunks are screened and searched while chunk i finishes: each work
 * stream first waits for the work queued on `stream` before the call, any
 * top-k merge runs on `stream` in chunk order, and `stream` waits for every
 * chunk before work queued after the call runs (stream-ordered as a single
 * launch would be).  The first such call allocates the other four sets
 * (~210 MB each) and the streams (E_NOMEM if that fails).  Calls on one context
 * must not overlap on the GPU (use one stream per context, or one context
 * per stream).
 * A candidate is INVALID if S = 0, S > 32, S > s_max, S > L, M = 0, a stage
 * byte has bits 5-7 set, names a type >= n_types or a type without GPUs, or
 * (dense models) asks a degree above the largest node of its type (the TP
 * mask of §5.1).  NO_FIT: DP degree 0.  OOM: no split fits in memory.
 * Errors: E_ARG (null ctx/struct/pointers, n < 0, plane_stride < n,
 * s_max outside [1, 32]), E_STATE (cluster or model missing), E_CUDA (launch
 * failure).  n = 0 is a no-op. */
heddle_status heddle_price_candidates(heddle_ctx* ctx, const heddle_candidates* cands,
                                      const heddle_results* results, void* stream);

/* Chunk size of the pricing calls: 1 <= chunk <= 2^20 (E_LIMIT otherwise).
 * Results never depend on it. */
heddle_status heddle_set_chunk(heddle_ctx* ctx, int64_t chunk);

/* ----------------------------------------------------------------- top-k */

/* Running top-k of OK candidates, best first, caller-owned device memory.
 * Order: higher throughput nM / T first (exact integer comparison
 * nM_a * T_b > nM_b * T_a), equal throughput -> smaller idx first.
 * nM = n_dp * M.  Each candidate index may be merged at most once. */
typedef struct {
    int32_t k;      /* 1..64 */
    int32_t count;  /* entries in use, <= k */
    int64_t idx[HEDDLE_MAX_TOPK];
    int64_t T[HEDDLE_MAX_TOPK];
    uint32_t nM[HEDDLE_MAX_TOPK];
} heddle_topk_state;

/* Set *state (device) to empty with capacity k (1..64).  Asynchronous. */
heddle_status heddle_topk_reset(heddle_ctx* ctx, heddle_topk_state* state, int32_t k,
                                void* stream);

/* Merge the OK candidates of a priced batch into *state (device): a
 * block-level top-k per CTA into context-owned scratch, then merge levels of
 * 16 lists per CTA, the last with the incoming state (two or three
 * launches, no inter-CTA waiting).
 * Asynchronous; reads cands->M, results->T/n_dp/status.  Errors: E_ARG,
 * E_STATE, E_CUDA.  Calls on one context must not overlap on the GPU (they
 * share the scratch): use one stream per context. */
heddle_status heddle_topk(heddle_ctx* ctx, const heddle_candidates* cands,
                          const heddle_results* results, heddle_topk_state* state,
                          void* stream);

/* Price a batch and merge its OK candidates into *state (device): after each
 * chunk's search, one top-k launch runs over that chunk's worklist of
 * searched candidates only (the screen already rejected the rest): per-CTA
 * lists, the last CTA of each group of 16 merges its group and the last
 * group merges the group lists into the state (tickets, no waiting) -- no
 * pass over the full results.
 * Same results and the same state as heddle_price_candidates followed by
 * heddle_topk.  Errors as for both. */
heddle_status heddle_price_topk(heddle_ctx* ctx, const heddle_candidates* cands,
                                const heddle_results* results, heddle_topk_state* state,
                                void* stream);

/* ------------------------------------------------- allocation-free top-k */

/* The top-k merge of heddle_topk for callers that cannot allocate device
 * memory at all -- for example code running inside another framework's
 * memory pool, where every device allocation must go through that pool, or
 * code that must not allocate after start-up -- and therefore cannot create
 * a heddle context either.  The paper has no counterpart: this is a
 * property of the library, not of the method.
 *
 * No context: runs on the calling thread's current device and allocates
 * nothing (no cudaMalloc, no library allocation).  Its scratch is a
 * file-scope device array of 96.25 KB that every device holds from the time
 * the library's device code is loaded until the process exits: 64 lists of
 * 64 entries, one per slice of 65,536 candidates, so a call handles at most
 * HEDDLE_TOPK_NOALLOC_MAX_N = 4,194,304 candidates (E_LIMIT beyond).
 * Every call looks up the array's device address on the current device
 * (cudaGetSymbolAddress; a device reset reloads the library's device code,
 * so an address kept from before it would be stale).  The first call on a
 * device also loads the library's device code there: make that first call
 * before any stream capture.
 * Every call on a device shares the array and overwrites it, so calls whose
 * kernels overlap on the GPU race: serialise them (one stream).
 *
 * Arguments as heddle_topk: merges the OK candidates of a priced batch
 * (cands->M, base_index; results->T, n_dp, status; device memory) into
 * *state (device, as set up by heddle_topk_reset or copied in by the
 * caller).  Same resulting state as heddle_topk.  Asynchronous on `stream`.
 * Errors: E_ARG (null pointers, n < 0), E_LIMIT (n above the maximum),
 * E_CUDA (symbol lookup or launch failed); there is no message buffer. */
#define HEDDLE_TOPK_NOALLOC_MAX_N 4194304
heddle_status heddle_topk_noalloc(const heddle_candidates* cands, const heddle_results* results,
                                  heddle_topk_state* state, void* stream);

/* --------------------------------------------- micro-batch-size fill */

/* §5.3 "Micro-batch size": the micro-batch size comes from the profiled
 * powers of two; every size that fits memory is priced and the one with the
 * shortest iteration time is kept.  The loaded model describes one
 * micro-batch of the base size b0; level i is the size 2^i b0.
 *
 * heddle_load_mbs(ctx, levels, profile_s) prepares levels 0 .. levels-1
 * (1 <= levels <= HEDDLE_MAX_MBS_LEVELS; 0 forgets them) and builds their
 * cost tables (synchronous).  At level i the per-layer FLOPs, stored
 * activations, TP all-reduce and EP all-to-all messages and the boundary
 * activation are 2^i times the model's; parameter, gradient and state
 * bytes are unchanged.  profile_s (nullable, host, copied) gives seconds
 * per layer for every level: [levels][n_types][4][n_layers], degree 2^j, as
 * the profile of heddle_load_model; without it the synthetic formula runs
 * on the scaled FLOPs and messages (E_STATE if the model itself was loaded
 * with a profile).  The levels are rebuilt when the cluster or model is
 * reloaded (their profile must still match the sizes).  Errors: E_ARG
 * (non-finite or negative profile entry), E_STATE, E_LIMIT (a scaled byte
 * count above 2^42, a table total above its limit), E_CUDA.
 *
 * heddle_price_mbs(ctx, cands, results, mbs, stream) prices every candidate
 * at every level: at level i a replica still processes M base micro-batches
 * per iteration, as M / 2^i micro-batches of size 2^i b0, and a level whose
 * size does not divide M is not priced for that candidate.  Each result row
 * holds the level with the smallest T among the levels where the candidate
 * is OK (equal T: the smaller level); a candidate OK at no level keeps the
 * base level's status (memory grows with the size, so a candidate that does
 * not fit at the base size fits at none).  mbs (nullable, device u8[n])
 * receives the chosen level (0 when not OK).  The throughput key of
 * heddle_topk stays n * M / T: M base micro-batches per iteration at any
 * size.  Asynchronous on `stream`; device buffers as heddle_price_candidates
 * (which keeps pricing the base size only).  Errors: E_ARG, E_STATE (no
 * levels loaded), E_CUDA. */
#define HEDDLE_MAX_MBS_LEVELS 4
heddle_status heddle_load_mbs(heddle_ctx* ctx, int32_t levels, const double* profile_s);
heddle_status heddle_price_mbs(heddle_ctx* ctx, const heddle_candidates* cands,
                               const heddle_results* results, uint8_t* mbs, void* stream);

/* ----------------------------------------------- multi-template plans */

/* Algorithm 1 builds a plan as a sequence of structural templates, each
 * holding its own GPUs; the reward of a step is the throughput the new
 * template adds (§5.5, Eq. reward).  heddle_price_plans prices a batch of
 * such plans: template t of a plan is priced against the GPUs templates
 * 0 .. t-1 left.  Its DP degree comes from the free GPUs per node (the
 * closed form of heddle_price_candidates on the free counts); its groups are
 * then placed largest first, each on a node of its type whose free GPUs
 * equal the group size, else on the node with the fewest free GPUs above it
 * (§5.1: a node whose size equals the degree first, else GPUs from a larger
 * node).  The layer split, the bottleneck and OOM do not depend on the DP
 * degree, so each slot is first priced as standalone candidates with the
 * context's search mode, then re-evaluated with the plan's degree (slot t
 * is priced only for the plans whose templates 0 .. t-1 are each OK on
 * their own: no other plan reaches it).  The first template that is not OK
 * (INVALID, NO_FIT on the GPUs left, OOM) ends the plan; later templates
 * are SKIPPED.  The plan's throughput is
 * the sum over its placed templates of n * M * 1e9 / T base micro-batches
 * per second, each term rounded in IEEE double, in template order (so the
 * step rewards are those terms).
 *
 * plans: n plans (0 <= n <= 2^20 per call), slots (1..HEDDLE_MAX_TEMPLATES)
 * template slots; n_templates[c] (device u8) the templates of plan c
 * (values above slots count as slots); t[i] the candidates of slot i
 * (device arrays as heddle_candidates, t[i].n == n).
 * results: per slot device arrays as heddle_results (T, bottleneck, n_dp,
 * status, optional bounds), overwritten with the plan's prices; placed[c]
 * (device u8) the templates placed; thr[c] (device double) the throughput.
 * Asynchronous on `stream`.  Errors: E_ARG, E_STATE, E_LIMIT (n above 2^20,
 * a node of more than HEDDLE_PLAN_MAX_NODE GPUs), E_CUDA, E_NOMEM. */
#define HEDDLE_MAX_TEMPLATES 4
#define HEDDLE_PLAN_MAX_NODE 64
typedef struct {
    int64_t n;
    int32_t slots;
    int32_t reserved;
    const uint8_t* n_templates;
    heddle_candidates t[HEDDLE_MAX_TEMPLATES];
} heddle_plans;
typedef struct {
    heddle_results t[HEDDLE_MAX_TEMPLATES];
    uint8_t* placed;
    double* thr;
} heddle_plan_results;
heddle_status heddle_price_plans(heddle_ctx* ctx, const heddle_plans* plans,
                                 const heddle_plan_results* results, void* stream);

/* ------------------------------------------------------ expert tiling */

/* §5.3 "Expert tiling": the 2^j devices of a stage factor into EP x ETP x
 * EDP (2^le x 2^lt x 2^ld, le + lt + ld = j).  ETP slices one tensor, so it
 * stays within the type's largest node; EP may leave a node; EDP is the
 * rest.  heddle_load_experts(ctx, expert_state, expert_param, n_layers)
 * gives, per layer of the loaded model, the experts' part of its state and
 * gradient bytes (host arrays, copied; 0 for a dense layer, at most the
 * layer's state_bytes / param_bytes) and turns tiling on for every later
 * heddle_price_candidates, heddle_price_topk, heddle_price_topk_host and
 * heddle_price_tiled call (both NULL turn it off; loading a model turns it
 * off).  Synchronous; builds NT x 20 x (L+1) int64 tiled tables, which
 * must fit 160 KB (E_LIMIT otherwise).  Needs the synthetic cost model
 * (E_STATE with a profile).  Readings (the paper names each direction's
 * collectives but prints no formula), per layer in seconds, IEEE double
 * left to right, no fused multiply-add:
 *   s = flops / (k * tflops * 1e12)
 *   k > 1: s += (4 * 2(k-1)/k) * ar_bytes / bw_k     bw_k = intra if k <= largest node, else NIC
 *   e > 1: s += (4 * (e-1)/e) * a2a_bytes / bw_et    ETP innermost: the EP group spans e*t devices
 *   t > 1: s += (4 * 2(t-1)/t) * a2a_bytes / intra
 * q = nearest ns; the tiling e = k, t = d = 1 is the untiled cost.  Memory
 * with EDP d: state + (d-1) expert state + f act <= mem k.  Gradient sync
 * of the stage: ceil(2((n-1) Gd + (n d - 1) Ge) 1e9 / (n k bw)) ns, Gd / Ge
 * the dense / expert gradient bytes of its layers, bw = intra when n = 1
 * and k <= largest node, else the slowest NIC.  PartitionLayers minimises
 * the largest stage time with every stage on its fastest fitting tiling
 * (the earliest slot on ties; slots order EDP exponent ascending, then ETP
 * exponent); the tilings are then re-selected against the whole iteration
 * time (M-1) max t + sum t + max g: for every bound Y among the gradient
 * terms of the fitting tilings each stage takes its fastest fitting tiling
 * with g <= Y, and the smallest T wins (the smaller Y on ties).
 * `bottleneck` is then the plan's largest stage time under the chosen
 * tilings.  Tiling prices the min-max split only: with search mode
 * DISTRIBUTE pricing returns E_STATE, and so do heddle_price_mbs and
 * heddle_price_plans while tiling is on.
 *
 * heddle_price_tiled prices like heddle_price_candidates and also writes
 * the chosen tiling of every stage: tiling (device, nullable) [32][n]
 * bytes, plane s at tiling[s * n + c] = log2 EP | log2 ETP << 2 (0 past S
 * and unless OK).  E_STATE unless experts are loaded. */
heddle_status heddle_load_experts(heddle_ctx* ctx, const int64_t* expert_state, const int64_t* expert_param,
                                  int32_t n_layers);
heddle_status heddle_price_tiled(heddle_ctx* ctx, const heddle_candidates* cands, const heddle_results* results,
                                 uint8_t* tiling, void* stream);

/* -------------------------------------------------------- host buffers */

/* End-to-end convenience for host (ideally pinned) buffers: streams the
 * candidates in batches of `batch` (1 <= batch <= 2^20, E_LIMIT above)
 * through context-owned device staging buffers (three sets), prices them,
 * merges them into *state and copies back every non-NULL field of
 * `results` (host arrays of cands->n entries; bounds uses plane stride
 * cands->n).  Batch k is copied in on a copy stream into staging set k % 3
 * (free once batch k - 3 is copied out), screened and searched
 * on work stream k % 2 with worklist set k % 5, merged on `stream` in batch
 * order and copied out on a second copy stream, so copies, the search of
 * one batch and the screen of the next overlap.  *state is host memory,
 * read on entry (k, and any entries already held) and written on return.
 * Synchronous: returns when all outputs are in host memory.  Grows its
 * staging buffers and creates the other worklist sets on first use
 * (allocation).  Errors as above, plus E_NOMEM. */
heddle_status heddle_price_topk_host(heddle_ctx* ctx, const heddle_candidates* cands,
                                     const heddle_results* results, heddle_topk_state* state,
                                     int64_t batch, void* stream);

/* ------------------------------------------------------- introspection */

/* Copy the quantised cost tables to host memory (synchronous):
 * q[n_types][4][n_layers] per-layer ns at degree 2^j (zero for types
 * without GPUs) and p2p[8][8][2] P2P ns (from type, to type, same-node).
 * Either pointer may be NULL. */
heddle_status heddle_get_tables(heddle_ctx* ctx, int64_t* q, int64_t* p2p);

/* Device-side error flags raised since the last call (synchronises the
 * device first, then clears them): bit 0 a table-staging wait timed out,
 * bit 1 a search exceeded its iteration bound, bit 2 an internal
 * consistency check failed, bit 3 (bounds-checked builds only) an index
 * test failed and the access was skipped.  0 in normal operation. */
heddle_status heddle_device_errors(heddle_ctx* ctx, uint32_t* flags);

/* PartitionLayers search.  AUTO (default) uses the equal-layer closed form
 * when every layer of the loaded model has the same quantised cost for each
 * (type, degree) and the same state and activation bytes -- then a stage of
 * per-layer cost q and memory capacity m holds min(m, floor((B - c) / q))
 * layers at bound B and a probe costs O(S) -- and the general interval
 * search otherwise.  GENERAL forces the general search.  Both are exact and
 * return identical results.  heddle_get_search reports the search the next
 * pricing call will run (GENERAL or EQUAL_LAYERS); E_STATE if the cost
 * tables are not built.
 *
 * DISTRIBUTE replaces PartitionLayers by the paper's own layer split
 * (§5.3 "Layer split and DP degree"), to measure what the exact min-max
 * split gains: layers in proportion to each stage's speed (2^40 / time of
 * all layers on its type and degree, rounded down; largest remainders, at
 * least one layer per stage), else the fastest fitting split of a fixed
 * list -- equal layer counts, layers in proportion to each stage's longest
 * memory-fitting run -- else OOM; "fastest" is the smallest pipeline time
 * (M-1) max t_s + sum t_s (Algorithm 1 splits before it picks the DP
 * degree); then the same Evaluate.  Results, status
 * rules and the top-k are as for the other modes; bottleneck is the chosen
 * split's largest stage time (not B*). */
#define HEDDLE_SEARCH_AUTO 0
#define HEDDLE_SEARCH_GENERAL 1
#define HEDDLE_SEARCH_EQUAL_LAYERS 2
#define HEDDLE_SEARCH_DISTRIBUTE 3
#define HEDDLE_SEARCH_TILED 4 /* reported by heddle_get_search while expert tiling is on */
heddle_status heddle_set_search(heddle_ctx* ctx, int32_t mode);
heddle_status heddle_get_search(heddle_ctx* ctx, int32_t* in_use);

/* Routing of the general search (models whose layers differ, §3.1
 * PartitionLayers) between its two kernels.  The thread-per-entry search
 * takes the worklist entries whose stages could each hold any single layer
 * when there are at least min_entries of them, and the warp-per-entry
 * search prices the rest; with fewer, the warp search prices every entry
 * (a thread search with too few entries runs as long as its longest serial
 * chain).  min_entries < 0 restores the default, 32 x the device's SM
 * count; 0 always runs the thread search.  Both routes return identical
 * results.  Errors: E_ARG (ctx NULL). */
heddle_status heddle_set_thread_search_min(heddle_ctx* ctx, int32_t min_entries);

/* Work counters of the next heddle_price_candidates call on ctx, for the
 * roofline report: when enabled, that call runs the counting variant of the
 * pricing kernel and accumulates, in device memory owned by ctx,
 * [0] interval checks evaluated (general search) or stages of the
 * candidates that reached the search, each counted once (equal-layer
 * search), [1] exact feasibility probes, [2] candidates that reached the
 * search.  heddle_work_counters(ctx, out) copies them out
 * (synchronous) and resets them. */
heddle_status heddle_count_next(heddle_ctx* ctx, int32_t enable);
heddle_status heddle_work_counters(heddle_ctx* ctx, uint64_t out[3]);

/* Device time of each phase of the pricing calls, measured with CUDA events
 * on the caller's stream.  The paper has no counterpart: it is how the
 * roofline report times its kernels without a profiler.  While enabled
 * (heddle_time_phases(ctx, 1); no stream capture meanwhile, the events are
 * created on demand), every chunk that heddle_price_candidates,
 * heddle_price_topk or heddle_price_topk_host prices records events
 * before the screen kernel, between the screen and the search kernel and
 * after the search kernel (on the stream that runs them) and, when the call
 * merges a top-k, before and after the top-k kernels (on `stream`).  With
 * several chunks in flight the phases of neighbouring chunks overlap, so
 * each phase's time is its own kernels' elapsed time while they share the
 * GPU.  heddle_phase_times synchronises on them and returns, per
 * phase (SCREEN, SEARCH, TOPK), the summed elapsed milliseconds and the
 * number of kernels launched in it (one screen, one search and one top-k
 * kernel per chunk), then forgets them.  The events add no work to the
 * kernels; enabling or disabling changes no result.  Errors: E_ARG,
 * E_CUDA. */
#define HEDDLE_PHASE_SCREEN 0
#define HEDDLE_PHASE_SEARCH 1
#define HEDDLE_PHASE_TOPK 2
#define HEDDLE_N_PHASES 3
heddle_status heddle_time_phases(heddle_ctx* ctx, int32_t enable);
heddle_status heddle_phase_times(heddle_ctx* ctx, double ms[HEDDLE_N_PHASES],
                                 int64_t launches[HEDDLE_N_PHASES]);

#ifdef __cplusplus
}
#endif
#endif /* HEDDLE_H */
