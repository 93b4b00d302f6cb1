/*
 * heddle_oracle.h -- CPU oracle for Heddle's batched candidate-plan pricing.
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, obviously-correct
 * restatement of the cost model of the paper (arxiv 2609.34244, §3.1 nested
 * search listing, §5.1 structural templates, §5.2 cost model, §5.3 auto-fill
 * and the 1F1B iteration time).  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline / reference arm may load it.  It shares no code,
 * header, table or helper with the CUDA library; both only read the same
 * seeded input arrays.
 *
 * All inputs are plain arrays (structure of arrays).  Times are int64
 * nanoseconds after quantisation, bytes are int64, bandwidths int64 bytes/s.
 */
#ifndef HEDDLE_ORACLE_H
#define HEDDLE_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORC_OK 0
#define ORC_OOM 1
#define ORC_NO_FIT 2
#define ORC_INVALID 3
#define ORC_SKIPPED 4 /* a plan's template after the plan ended */

typedef struct orc_ctx orc_ctx;

/* Build the oracle's cost model for one cluster and one model.
 * profile_s: nullable [n_types][4][n_layers] seconds per layer at degree 2^j.
 * Returns NULL on malformed input (a message is written to err, 256 bytes). */
orc_ctx* orc_create(int n_types, const double* tflops, const int64_t* mem_bytes,
                    const int64_t* intra_bw, int n_nodes, const int32_t* node_type,
                    const int32_t* node_gpus, const int64_t* node_nic, int n_layers,
                    const double* flops, const int64_t* param_bytes,
                    const int64_t* state_bytes, const int64_t* act_bytes,
                    const int64_t* ar_bytes, const int64_t* a2a_bytes,
                    int64_t boundary_bytes, int moe, const double* profile_s, char* err);
void orc_destroy(orc_ctx* x);

/* Quantised tables: q[n_types][4][L] per-layer ns, p2p[8][8][2] ns
 * (from type, to type, same-node flag), present/maxnode/inter_bw per type. */
void orc_tables(const orc_ctx* x, int64_t* q, int64_t* p2p, int32_t* maxnode,
                int64_t* inter_bw);

/* Price candidates [0, n): S[n], M[n], code[s * plane_stride + c] for
 * s < s_max.  Outputs T, bottleneck, n_dp, status and (nullable) bounds
 * [33][n].  threads <= 0 means one thread.  Returns the threads used. */
int orc_price(const orc_ctx* x, int64_t n, const uint8_t* S, const uint16_t* M,
              const uint8_t* code, int64_t plane_stride, int s_max, int64_t* T,
              int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* bounds,
              int threads);

/* Layer split used by orc_price: 0 (default) the min-max PartitionLayers of
 * the hot path; 1 the paper's own rule (§5.3 "Layer split and DP degree"):
 * layers in proportion to each stage's speed (2^40 / time of all layers on
 * its type and degree, rounded down), else the fastest fitting split of a
 * fixed list -- equal layer counts, layers in proportion to each stage's
 * longest memory-fitting run -- else OOM; "fastest" is the smallest
 * pipeline time (M-1) max t_s + sum t_s (the split precedes the DP degree
 * in Algorithm 1). */
void orc_set_split(orc_ctx* x, int mode);

/* Expert tiling (§5.3 "Expert tiling"): expert_state[l] and expert_param[l]
 * are the expert parts of layer l's state and gradient bytes (0 for a dense
 * layer; at most the layer's totals).  Turns tiling on for orc_price /
 * orc_price_tiled with PartitionLayers (both NULL turn it off).  A stage of
 * 2^j devices may then use every tiling 2^le EP x 2^lt ETP x 2^ld EDP with
 * ETP within the type's largest node: per-layer cost with the EP and ETP
 * collectives, memory with the expert state replicated d times, gradient
 * sync of expert gradients over n d copies; the split minimises the
 * largest stage time at each stage's fastest fitting tiling, and the
 * tilings are re-selected against the whole iteration time.  Needs the
 * synthetic cost model (no explicit profile).  Returns 0, or -1 with a
 * message in err. */
int orc_set_experts(orc_ctx* x, const int64_t* expert_state, const int64_t* expert_param, char* err);

/* Tiled cost tables (after orc_set_experts): Pt[n_types][20][L+1] prefix
 * ns per tiling slot (slots 0, 1-3, 4-9, 10-19 for 1, 2, 4, 8 devices; EDP
 * exponent ascending, then ETP exponent) and valid[n_types][20]. */
void orc_tiled_tables(const orc_ctx* x, int64_t* Pt, int32_t* valid);

/* orc_price plus, when tiling is on, the chosen tiling of every stage:
 * tiling[s * n + c] = log2 EP | log2 ETP << 2 (nullable; 0 past S and
 * unless OK).  Returns -1 if tiling is combined with the paper's split. */
int orc_price_tiled(const orc_ctx* x, int64_t n, const uint8_t* S, const uint16_t* M,
                    const uint8_t* code, int64_t plane_stride, int s_max, int64_t* T,
                    int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* bounds,
                    uint8_t* tiling, int threads);

/* Multi-template plans (Algorithm 1): n_plans plans of up to max_tmpl
 * templates (n_tmpl[c] used); template t of plan c has depth S[t*n + c],
 * micro-batches M[t*n + c] and stage codes code[(t*s_max + s)*n + c].
 * Templates are priced in order against the GPUs the earlier ones left
 * (DP degree from the free GPUs per node; groups placed largest first on a
 * node whose free GPUs equal the group size, else the node with the fewest
 * free GPUs above it); the first template that is not OK ends the plan.
 * Per template [t*n + c]: T, bottleneck, n_dp, status (ORC_SKIPPED past
 * the end); per plan: placed templates and throughput
 * sum n*M*1e9/T (IEEE double, template order).  Single-threaded. */
int orc_price_plans(const orc_ctx* x, int64_t n_plans, int max_tmpl, const uint8_t* n_tmpl,
                    const uint8_t* S, const uint16_t* M, const uint8_t* code, int s_max,
                    int64_t* T, int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* placed,
                    double* thr);

/* Top-k of the OK candidates by throughput n*M/T, ties to the smaller index.
 * idx = base_index + c.  Writes up to k entries; returns how many. */
int orc_topk(int64_t n, int64_t base_index, const int64_t* T, const uint16_t* n_dp,
             const uint16_t* M, const uint8_t* status, int k, int64_t* out_idx,
             int64_t* out_T, uint32_t* out_nM);

/* Min-max contiguous partition of L layers into S non-empty stages, stated
 * on raw integer inputs (test hook).  Stage s costs P[s][j] - P[s][i] + c[s]
 * and fits iff W[s][j] - W[s][i] <= cap[s]; P and W are [S][L+1].
 * Returns 1 and writes B* and the lexicographically smallest optimal
 * boundary vector a[0..S] if a valid partition exists, else returns 0. */
int orc_partition_raw(int S, int L, const int64_t* P, const int64_t* c, const int64_t* W,
                      const int64_t* cap, int64_t* Bstar, int32_t* a);

/* Largest replication count n for which n copies of every group (sizes
 * group_gpus[0..n_groups)) can be placed on nodes of node_gpus[0..n_nodes)
 * without a group crossing a node (one GPU type).  Group sizes must be
 * powers of two. */
int orc_replicas(int n_nodes, const int32_t* node_gpus, int n_groups,
                 const int32_t* group_gpus);

#ifdef __cplusplus
}
#endif
#endif
