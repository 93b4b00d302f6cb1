/*
 * heddle_oracle.c -- CPU oracle for Heddle's batched candidate-plan pricing.
 *
 * TEST INFRASTRUCTURE ONLY (see heddle_oracle.h).  Every step is written as
 * the plain definition it restates, in the order the paper describes it:
 *
 *   cost table   §5.2 "Throughput estimation": one entry per (GPU type, TP
 *                degree) gives the per-layer computation and communication
 *                cost.  Quantised here to whole nanoseconds.
 *   DP degree    §5.3 "Layer split and DP degree" and §5.1 "Non-uniform GPU
 *                composition support": pack each stage's TP group into nodes
 *                of its type, a group never crossing a node; take the largest
 *                replication count the packing admits.  Computed here by
 *                explicit first-fit-decreasing placement.
 *   partition    §3.1 listing, PartitionLayers: split the layers into S
 *                contiguous non-empty stages minimising the largest stage
 *                time, with the memory validation of §5.2.  Computed here by
 *                the textbook O(S L^2) dynamic programme.
 *   evaluate     §5.3 iteration time of a 1F1B pipeline,
 *                (M-1) max_s t_s + sum_s t_s + max_s g_s.
 *   rank, top-k  §5 overview: plans are ranked by predicted throughput.
 *   tiling       §5.3 "Expert tiling" (optional, orc_set_experts): a stage's
 *                expert layers factor its devices into EP x ETP x EDP; every
 *                factorisation that fits memory is priced, the stage keeps
 *                the fastest, and the per-stage choices are re-selected
 *                against the whole iteration time.
 *
 * Readings of points the paper leaves open (quantisation, P2P, memory and
 * gradient-sync formulas, tie-breaks) are the ones listed in the design
 * notes; each is restated beside the code that applies it.
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off (no fused multiply-add, so the
 * double arithmetic of the quantiser is the plain IEEE sequence written).
 */
#include "heddle_oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#define MAXT 8
#define MAXS 32
#define MAXL 255
#define INF INT64_MAX

typedef unsigned __int128 u128;

struct orc_ctx {
    int n_types, L, moe;
    int64_t gpus[MAXT];      /* GPUs of each type */
    int32_t maxnode[MAXT];   /* largest node of each type */
    int64_t inter_bw[MAXT];  /* slowest NIC among the nodes of each type */
    int64_t intra_bw[MAXT];
    int64_t mem[MAXT];
    int n_nodes;
    int32_t* node_type;
    int32_t* node_gpus;
    int64_t* q;      /* [n_types][4][L] quantised per-layer ns */
    int64_t* P;      /* [n_types][4][L+1] prefix sums of q */
    int64_t* state;  /* [L+1] prefix of state bytes */
    int64_t* act;    /* [L+1] prefix of stored activation bytes */
    int64_t* param;  /* [L+1] prefix of gradient (parameter) bytes */
    int64_t p2p[MAXT][MAXT][2];
    int split_mode;  /* 0: min-max PartitionLayers, 1: the paper's Distribute rule */
    /* the layers' cost inputs, kept for the expert-tiling tables */
    double tflops[MAXT];
    double* flops;
    int64_t *ar, *a2a;
    int has_profile;
    /* expert tiling (0: off) */
    int tiled;
    int64_t* estate;  /* [L+1] prefix of the expert part of state bytes */
    int64_t* eparam;  /* [L+1] prefix of the expert part of gradient bytes */
    int64_t* Pt;      /* [n_types][20][L+1] prefix of per-layer ns per tiling slot */
    int tvalid[MAXT][20];
};

/* ---------------------------------------------------------------- tables */

/* Nearest nanosecond, halves away from zero (C99 llround). */
static int64_t to_ns(double seconds) { return (int64_t)llround(seconds * 1e9); }

/* ceil(a / b) for a >= 0, b > 0 in 128-bit arithmetic. */
static int64_t ceil_div128(u128 a, u128 b) { return (int64_t)((a + b - 1) / b); }

/* Per-layer time in seconds of layer l on one GPU group of type g and degree
 * k = 2^j (§5.2: computation plus communication of one layer).  Synthetic
 * stand-in for a profile entry:
 *   compute  flops / (k * TFLOPS * 1e12)
 *   TP       k > 1: four ring all-reduces (two forward, two backward) of
 *            ar_bytes, each moving 2(k-1)/k of the message
 *   EP       k > 1: four all-to-alls (dispatch and combine, forward and
 *            backward) of a2a_bytes, each moving (k-1)/k of the message
 * Both collectives use the type's intra-node bandwidth when the group fits
 * in one node, else the node NIC bandwidth (an EP group may leave a node,
 * §5.3 "Expert tiling"). */
static double layer_seconds(const orc_ctx* x, int g, int j, double flops, int64_t ar,
                            int64_t a2a, double tflops) {
    double k = (double)(1 << j);
    double s = flops / (k * tflops * 1e12);
    if (j > 0) {
        double bw = (1 << j) <= x->maxnode[g] ? (double)x->intra_bw[g] : (double)x->inter_bw[g];
        double ring = (2.0 * (k - 1.0)) / k;
        double t = 4.0 * ring;
        t = t * (double)ar;
        t = t / bw;
        s = s + t;
        double part = (k - 1.0) / k;
        t = 4.0 * part;
        t = t * (double)a2a;
        t = t / bw;
        s = s + t;
    }
    return s;
}

orc_ctx* orc_create(int n_types, const double* tflops, const int64_t* mem_bytes,
                    const int64_t* intra_bw, int n_nodes, const int32_t* node_type,
                    const int32_t* node_gpus, const int64_t* node_nic, int n_layers,
                    const double* flops, const int64_t* param_bytes,
                    const int64_t* state_bytes, const int64_t* act_bytes,
                    const int64_t* ar_bytes, const int64_t* a2a_bytes,
                    int64_t boundary_bytes, int moe, const double* profile_s, char* err) {
    if (n_types < 1 || n_types > MAXT || n_layers < 1 || n_layers > MAXL || n_nodes < 1) {
        if (err) snprintf(err, 256, "size out of range");
        return NULL;
    }
    orc_ctx* x = (orc_ctx*)calloc(1, sizeof(orc_ctx));
    int L = n_layers;
    x->n_types = n_types;
    x->L = L;
    x->moe = moe != 0;
    x->has_profile = profile_s != NULL;
    x->flops = (double*)malloc(sizeof(double) * L);
    x->ar = (int64_t*)malloc(sizeof(int64_t) * L);
    x->a2a = (int64_t*)malloc(sizeof(int64_t) * L);
    for (int l = 0; l < L; ++l) {
        x->flops[l] = flops ? flops[l] : 0.0;
        x->ar[l] = ar_bytes ? ar_bytes[l] : 0;
        x->a2a[l] = a2a_bytes ? a2a_bytes[l] : 0;
    }
    for (int g = 0; g < n_types; ++g) x->tflops[g] = tflops[g];
    x->n_nodes = n_nodes;
    x->node_type = (int32_t*)malloc(sizeof(int32_t) * n_nodes);
    x->node_gpus = (int32_t*)malloc(sizeof(int32_t) * n_nodes);
    memcpy(x->node_type, node_type, sizeof(int32_t) * n_nodes);
    memcpy(x->node_gpus, node_gpus, sizeof(int32_t) * n_nodes);
    for (int g = 0; g < n_types; ++g) {
        x->gpus[g] = 0;
        x->maxnode[g] = 0;
        x->inter_bw[g] = INT64_MAX;
        x->intra_bw[g] = intra_bw[g];
        x->mem[g] = mem_bytes[g];
    }
    for (int b = 0; b < n_nodes; ++b) {
        int g = node_type[b];
        if (g < 0 || g >= n_types || node_gpus[b] < 1) {
            if (err) snprintf(err, 256, "bad node %d", b);
            orc_destroy(x);
            return NULL;
        }
        x->gpus[g] += node_gpus[b];
        if (node_gpus[b] > x->maxnode[g]) x->maxnode[g] = node_gpus[b];
        if (node_nic[b] < x->inter_bw[g]) x->inter_bw[g] = node_nic[b];
    }
    for (int g = 0; g < n_types; ++g)
        if (x->gpus[g] == 0) x->inter_bw[g] = 0; /* absent type: never priced */

    size_t nq = (size_t)n_types * 4 * L;
    x->q = (int64_t*)calloc(nq, sizeof(int64_t));
    x->P = (int64_t*)calloc((size_t)n_types * 4 * (L + 1), sizeof(int64_t));
    for (int g = 0; g < n_types; ++g) {
        if (x->gpus[g] == 0) continue; /* tables of absent types stay zero */
        for (int j = 0; j < 4; ++j) {
            int64_t* q = x->q + ((size_t)g * 4 + j) * L;
            int64_t* P = x->P + ((size_t)g * 4 + j) * (L + 1);
            P[0] = 0;
            for (int l = 0; l < L; ++l) {
                double sec = profile_s
                                 ? profile_s[((size_t)g * 4 + j) * L + l]
                                 : layer_seconds(x, g, j, flops[l], ar_bytes[l], a2a_bytes[l],
                                                 tflops[g]);
                q[l] = to_ns(sec);
                P[l + 1] = P[l] + q[l];
            }
        }
    }
    x->state = (int64_t*)calloc(L + 1, sizeof(int64_t));
    x->act = (int64_t*)calloc(L + 1, sizeof(int64_t));
    x->param = (int64_t*)calloc(L + 1, sizeof(int64_t));
    for (int l = 0; l < L; ++l) {
        x->state[l + 1] = x->state[l] + state_bytes[l];
        x->act[l + 1] = x->act[l] + act_bytes[l];
        x->param[l + 1] = x->param[l] + param_bytes[l];
    }
    /* Inter-stage P2P (reading): forward activation plus backward gradient,
     * 2 * boundary bytes, over the intra-node link when both stages are the
     * same type and the two groups fit in one node, else over the slower of
     * the two types' NICs. */
    for (int g = 0; g < MAXT; ++g)
        for (int h = 0; h < MAXT; ++h)
            for (int same = 0; same < 2; ++same) {
                int64_t bw = 0;
                if (g < n_types && h < n_types && x->gpus[g] && x->gpus[h]) {
                    if (same)
                        bw = x->intra_bw[g];
                    else
                        bw = x->inter_bw[g] < x->inter_bw[h] ? x->inter_bw[g] : x->inter_bw[h];
                }
                x->p2p[g][h][same] =
                    bw > 0 ? ceil_div128((u128)2 * (u128)boundary_bytes * 1000000000u, (u128)bw)
                           : 0;
            }
    return x;
}

void orc_destroy(orc_ctx* x) {
    if (!x) return;
    free(x->node_type);
    free(x->node_gpus);
    free(x->q);
    free(x->P);
    free(x->state);
    free(x->act);
    free(x->param);
    free(x->flops);
    free(x->ar);
    free(x->a2a);
    free(x->estate);
    free(x->eparam);
    free(x->Pt);
    free(x);
}

void orc_tables(const orc_ctx* x, int64_t* q, int64_t* p2p, int32_t* maxnode,
                int64_t* inter_bw) {
    if (q) memcpy(q, x->q, sizeof(int64_t) * (size_t)x->n_types * 4 * x->L);
    if (p2p) memcpy(p2p, x->p2p, sizeof(x->p2p));
    for (int g = 0; g < x->n_types; ++g) {
        if (maxnode) maxnode[g] = x->maxnode[g];
        if (inter_bw) inter_bw[g] = x->inter_bw[g];
    }
}

/* --------------------------------------------------------- expert tiling */

/* §5.3 "Expert tiling": the 2^j devices of a stage factor as EP x ETP x EDP
 * (e t d = 2^j).  With power-of-two degrees a tiling is the exponent pair
 * (le, lt), ld = j - le - lt; the 1 + 3 + 6 + 10 tilings of 1, 2, 4 and 8
 * devices take slots 0, 1-3, 4-9 and 10-19, in the order EDP exponent
 * ascending, then ETP exponent ascending.  Slot 0 of every degree (EP over
 * all devices, no ETP, no EDP) is the untiled stage. */
static const int tile_base[4] = {0, 1, 4, 10};

static void tiling_of(int j, int idx, int* le, int* lt, int* ld) {
    int k = 0;
    for (int d = 0; d <= j; ++d)
        for (int t = 0; t + d <= j; ++t) {
            if (k == idx) {
                *ld = d;
                *lt = t;
                *le = j - d - t;
                return;
            }
            ++k;
        }
}

/* Per-layer seconds of layer l on a stage of type g with 2^j devices tiled
 * as (2^le EP, 2^lt ETP, 2^(j-le-lt) EDP).  Readings (the paper names the
 * collectives of each direction but prints no formula):
 *   compute  flops / (k * TFLOPS * 1e12): every tiling spreads the layer's
 *            work over all k devices
 *   TP       k > 1: the dense part's four ring all-reduces of ar_bytes over
 *            the k devices, as for an untiled stage
 *   EP       e > 1: four all-to-alls of a2a_bytes, each moving (e-1)/e; ETP
 *            is the innermost factor, so an EP group spans e * t
 *            consecutive devices and uses the NIC once that leaves a node
 *   ETP      t > 1: four ring all-reduces of a2a_bytes (the expert output),
 *            2(t-1)/t each, inside a node (ETP carries TP's node bound)
 *   EDP      no per-micro-batch traffic; it replicates the expert state
 *            (memory) and synchronises expert gradients (evaluate)
 * The untiled slot reproduces the untiled cost bit for bit. */
static double tiled_seconds(const orc_ctx* x, int g, int j, int le, int lt, int l) {
    double k = (double)(1 << j);
    double sec = x->flops[l] / (k * x->tflops[g] * 1e12);
    double near = (double)x->intra_bw[g], far = (double)x->inter_bw[g];
    if (j > 0) {
        double bw = (1 << j) <= x->maxnode[g] ? near : far;
        double w = (2.0 * (k - 1.0)) / k;
        sec = sec + ((4.0 * w) * (double)x->ar[l]) / bw;
    }
    if (le > 0) {
        double e = (double)(1 << le);
        double bw = (1 << (le + lt)) <= x->maxnode[g] ? near : far;
        sec = sec + ((4.0 * ((e - 1.0) / e)) * (double)x->a2a[l]) / bw;
    }
    if (lt > 0) {
        double t = (double)(1 << lt);
        sec = sec + ((4.0 * ((2.0 * (t - 1.0)) / t)) * (double)x->a2a[l]) / near;
    }
    return sec;
}

int orc_set_experts(orc_ctx* x, const int64_t* expert_state, const int64_t* expert_param, char* err) {
    int L = x->L;
    free(x->estate);
    free(x->eparam);
    free(x->Pt);
    x->estate = x->eparam = x->Pt = NULL;
    x->tiled = 0;
    if (!expert_state && !expert_param) return 0;
    if (!expert_state || !expert_param || x->has_profile) {
        if (err) snprintf(err, 256, "expert tiling needs both byte arrays and the synthetic cost model");
        return -1;
    }
    for (int l = 0; l < L; ++l) {
        int64_t st = x->state[l + 1] - x->state[l], pb = x->param[l + 1] - x->param[l];
        if (expert_state[l] < 0 || expert_state[l] > st || expert_param[l] < 0 || expert_param[l] > pb) {
            if (err) snprintf(err, 256, "expert bytes of layer %d outside [0, layer bytes]", l);
            return -1;
        }
    }
    x->estate = (int64_t*)calloc(L + 1, sizeof(int64_t));
    x->eparam = (int64_t*)calloc(L + 1, sizeof(int64_t));
    for (int l = 0; l < L; ++l) {
        x->estate[l + 1] = x->estate[l] + expert_state[l];
        x->eparam[l + 1] = x->eparam[l] + expert_param[l];
    }
    x->Pt = (int64_t*)calloc((size_t)x->n_types * 20 * (L + 1), sizeof(int64_t));
    for (int g = 0; g < x->n_types; ++g)
        for (int j = 0; j < 4; ++j)
            for (int i = 0; i < (j + 1) * (j + 2) / 2; ++i) {
                int le = 0, lt = 0, ld = 0, slot = tile_base[j] + i;
                tiling_of(j, i, &le, &lt, &ld);
                /* ETP slices one tensor, so it stays inside a node */
                x->tvalid[g][slot] = x->gpus[g] > 0 && (1 << lt) <= x->maxnode[g];
                int64_t* P = x->Pt + ((size_t)g * 20 + slot) * (L + 1);
                P[0] = 0;
                for (int l = 0; l < L; ++l)
                    P[l + 1] = P[l] + (x->tvalid[g][slot] ? to_ns(tiled_seconds(x, g, j, le, lt, l)) : 0);
            }
    x->tiled = 1;
    return 0;
}

void orc_tiled_tables(const orc_ctx* x, int64_t* Pt, int32_t* valid) {
    if (!x->tiled) return;
    if (Pt) memcpy(Pt, x->Pt, sizeof(int64_t) * (size_t)x->n_types * 20 * (x->L + 1));
    if (valid)
        for (int g = 0; g < x->n_types; ++g)
            for (int t = 0; t < 20; ++t) valid[g * 20 + t] = x->tvalid[g][t];
}

/* ------------------------------------------------------------- DP degree */

/* Can n replicas of the groups be placed?  First-fit decreasing: groups are
 * taken from the largest size down, each into the first node (in list order)
 * with enough free GPUs.  Equal-size groups are placed as a batch, which is
 * what placing them one at a time first-fit does. */
static int ffd_fits(int n_nodes, const int32_t* node_gpus, const int64_t* count_by_size,
                    int64_t n) {
    int64_t* rem = (int64_t*)malloc(sizeof(int64_t) * (n_nodes > 0 ? n_nodes : 1));
    for (int b = 0; b < n_nodes; ++b) rem[b] = node_gpus[b];
    int ok = 1;
    for (int e = 3; e >= 0 && ok; --e) {
        int64_t w = (int64_t)1 << e;
        int64_t left = count_by_size[e] * n;
        for (int b = 0; b < n_nodes && left > 0; ++b) {
            int64_t take = rem[b] / w;
            if (take > left) take = left;
            rem[b] -= take * w;
            left -= take;
        }
        if (left > 0) ok = 0;
    }
    free(rem);
    return ok;
}

/* Largest n such that n replicas fit (0 if not even one does). */
static int64_t replicas(int n_nodes, const int32_t* node_gpus, const int64_t* count_by_size) {
    int64_t any = 0, total = 0;
    for (int e = 0; e < 4; ++e) any += count_by_size[e];
    for (int b = 0; b < n_nodes; ++b) total += node_gpus[b];
    if (any == 0) return INT64_MAX; /* this type hosts no stage */
    int64_t n = 0;
    while (n < total && ffd_fits(n_nodes, node_gpus, count_by_size, n + 1)) ++n;
    return n;
}

int orc_replicas(int n_nodes, const int32_t* node_gpus, int n_groups,
                 const int32_t* group_gpus) {
    int64_t cnt[4] = {0, 0, 0, 0};
    for (int i = 0; i < n_groups; ++i) {
        int e = 0;
        while (e < 3 && (1 << e) < group_gpus[i]) ++e;
        cnt[e] += 1;
    }
    int64_t n = replicas(n_nodes, node_gpus, cnt);
    return n == INT64_MAX ? 0 : (int)n;
}

/* DP degree of a candidate: the replication count every GPU type admits.
 * A stage group of degree k larger than the largest node of its type (only
 * possible for an EP degree, §5.3) is placed as k/p blocks of p GPUs, p the
 * largest power of two not above that node size (reading). */
static int64_t dp_degree(const orc_ctx* x, int S, const int* g, const int* j, const int32_t* node_free) {
    int64_t best = INT64_MAX;
    int32_t* ng = (int32_t*)malloc(sizeof(int32_t) * x->n_nodes);
    for (int t = 0; t < x->n_types; ++t) {
        int64_t cnt[4] = {0, 0, 0, 0};
        int used = 0;
        for (int s = 0; s < S; ++s) {
            if (g[s] != t) continue;
            used = 1;
            int k = 1 << j[s];
            int e = j[s];
            while ((1 << e) > x->maxnode[t]) --e;
            cnt[e] += k >> e;
        }
        if (!used) continue;
        int nn = 0;
        for (int b = 0; b < x->n_nodes; ++b)
            if (x->node_type[b] == t) ng[nn++] = node_free ? node_free[b] : x->node_gpus[b];
        int64_t r = replicas(nn, ng, cnt);
        if (r < best) best = r;
    }
    free(ng);
    return best == INT64_MAX ? 0 : best;
}

/* --------------------------------------------------------- PartitionLayers */

/* f[s][i]: smallest achievable largest stage time of stages s..S-1 covering
 * layers [i, L), INF if they cannot.  B* = f[0][0].  The canonical optimum is
 * the lexicographically smallest boundary vector: walk s = 0..S-1 taking the
 * smallest next boundary j whose stage fits, costs at most B*, and whose
 * remainder can still finish within B*. */
static int partition(int S, int L, const int64_t* const* P, const int64_t* c,
                     const int64_t* const* W, const int64_t* cap, int64_t* f,
                     int64_t* Bstar, int32_t* a) {
#define F(s, i) f[(size_t)(s) * (L + 1) + (i)]
    for (int i = 0; i <= L; ++i) F(S, i) = (i == L) ? 0 : INF;
    for (int s = S - 1; s >= 0; --s) {
        for (int i = 0; i <= L; ++i) {
            int64_t best = INF;
            for (int j = i + 1; j <= L; ++j) {
                if (F(s + 1, j) == INF) continue;
                if (W[s][j] - W[s][i] > cap[s]) continue;
                int64_t t = P[s][j] - P[s][i] + c[s];
                int64_t v = t > F(s + 1, j) ? t : F(s + 1, j);
                if (v < best) best = v;
            }
            F(s, i) = best;
        }
    }
    int64_t B = F(0, 0);
    if (B == INF) return 0;
    *Bstar = B;
    a[0] = 0;
    for (int s = 0; s < S; ++s) {
        int i = a[s], chosen = -1;
        for (int j = i + 1; j <= L; ++j) {
            if (F(s + 1, j) > B) continue;
            if (W[s][j] - W[s][i] > cap[s]) continue;
            if (P[s][j] - P[s][i] + c[s] > B) continue;
            chosen = j;
            break;
        }
        a[s + 1] = chosen; /* exists because f[s][a_s] <= B */
    }
    return 1;
#undef F
}

int orc_partition_raw(int S, int L, const int64_t* P, const int64_t* c, const int64_t* W,
                      const int64_t* cap, int64_t* Bstar, int32_t* a) {
    if (S < 1 || L < 1) return 0;
    const int64_t** Pp = (const int64_t**)malloc(sizeof(int64_t*) * S);
    const int64_t** Wp = (const int64_t**)malloc(sizeof(int64_t*) * S);
    for (int s = 0; s < S; ++s) {
        Pp[s] = P + (size_t)s * (L + 1);
        Wp[s] = W + (size_t)s * (L + 1);
    }
    int64_t* f = (int64_t*)malloc(sizeof(int64_t) * (size_t)(S + 1) * (L + 1));
    int ok = partition(S, L, Pp, c, Wp, cap, f, Bstar, a);
    free(f);
    free(Pp);
    free(Wp);
    return ok;
}

/* ------------------------------------------------------ price one candidate */

typedef struct {
    int64_t T, B;
    int64_t n;
    int status;
    int32_t a[MAXS + 1];
    uint8_t tile[MAXS]; /* expert tiling per stage: log2 EP | log2 ETP << 2 */
} priced;

/* Evaluate (§5.3): T = (M-1) max t_s + sum t_s + max g_s for the split a;
 * writes max t_s to *tmax_out. */
static int64_t evaluate(const orc_ctx* x, int S, int M, int64_t n, const int64_t* const* P, const int64_t* c,
                        const int* j, const int* g, const int32_t* a, int64_t* tmax_out) {
    int64_t tmax = 0, tsum = 0, gmax = 0;
    for (int s = 0; s < S; ++s) {
        int64_t t = P[s][a[s + 1]] - P[s][a[s]] + c[s];
        if (t > tmax) tmax = t;
        tsum += t;
        /* DP gradient synchronisation of stage s (reading): a ring all-reduce
         * over the n replicas of the stage's gradient shard (G_s / k bytes),
         * 2(n-1)/n of it over the slowest NIC of the type, in whole ns
         * rounded up; zero without replication */
        int64_t gs = 0;
        if (n > 1) {
            int64_t G = x->param[a[s + 1]] - x->param[a[s]];
            u128 num = (u128)2 * (u128)(n - 1) * (u128)G * 1000000000u;
            u128 den = (u128)n * (u128)(1 << j[s]) * (u128)x->inter_bw[g[s]];
            gs = ceil_div128(num, den);
        }
        if (gs > gmax) gmax = gs;
    }
    *tmax_out = tmax;
    return (int64_t)(M - 1) * tmax + tsum + gmax;
}

/* ------------------------------------------- tiled PartitionLayers, Evaluate */

/* The tilings a stage may use: prefix row, EDP degree minus one, code. */
typedef struct {
    int n;
    const int64_t* P[10];
    int64_t d1[10];
    uint8_t code[10];
} tiles;

/* Stage time of layers [i, j) under expert tiling: the fastest tiling whose
 * memory fits (§5.3: every factorisation that fits per-GPU memory is priced
 * and the shortest kept; the earliest slot on ties), INF if none fits.
 * Memory (reading): per device, dense state / k + expert state / (e t) +
 * f activations / k; with e t = k / d that is state + (d - 1) expert state
 * + f act <= capacity * k.  *which gets the option index. */
static int64_t tiled_time(const orc_ctx* x, const tiles* tl, int64_t c, int64_t f, int64_t cap, int i, int j,
                          int* which) {
    int64_t fastest = INF;
    for (int o = 0; o < tl->n; ++o) {
        int64_t mem = (x->state[j] - x->state[i]) + tl->d1[o] * (x->estate[j] - x->estate[i]) +
                      f * (x->act[j] - x->act[i]);
        if (mem > cap) continue;
        int64_t t = tl->P[o][j] - tl->P[o][i] + c;
        if (t < fastest) {
            fastest = t;
            if (which) *which = o;
        }
    }
    return fastest;
}

/* The dynamic programme of partition() over the tiled stage time.  The
 * fastest fitting tiling of an interval is no slower on a sub-interval
 * (each tiling that fits the interval fits the sub-interval and costs
 * less), so stage time stays monotone under inclusion and the canonical
 * (lexicographically smallest) optimal split is defined as before. */
static int partition_tiled(const orc_ctx* x, int S, const tiles* tl, const int64_t* c, const int64_t* f_s,
                           const int64_t* cap, int64_t* f, int64_t* Bstar, int32_t* a) {
    int L = x->L;
#define FT(s, i) f[(size_t)(s) * (L + 1) + (i)]
    for (int i = 0; i <= L; ++i) FT(S, i) = (i == L) ? 0 : INF;
    for (int s = S - 1; s >= 0; --s)
        for (int i = 0; i <= L; ++i) {
            int64_t lowest = INF;
            for (int j = i + 1; j <= L; ++j) {
                if (FT(s + 1, j) == INF) continue;
                int64_t t = tiled_time(x, &tl[s], c[s], f_s[s], cap[s], i, j, NULL);
                if (t == INF) continue;
                int64_t v = t > FT(s + 1, j) ? t : FT(s + 1, j);
                if (v < lowest) lowest = v;
            }
            FT(s, i) = lowest;
        }
    int64_t B = FT(0, 0);
    if (B == INF) return 0;
    *Bstar = B;
    a[0] = 0;
    for (int s = 0; s < S; ++s) {
        int chosen = -1;
        for (int j = a[s] + 1; j <= L && chosen < 0; ++j)
            if (FT(s + 1, j) <= B && tiled_time(x, &tl[s], c[s], f_s[s], cap[s], a[s], j, NULL) <= B) chosen = j;
        a[s + 1] = chosen;
    }
    return 1;
#undef FT
}

/* Gradient synchronisation of a tiled stage over layers [lo, hi) (reading):
 * the dense gradients are all-reduced over the n replicas as in evaluate();
 * the expert gradients over the n d copies of each expert shard (d EDP
 * copies in each replica).  Per device that is Gd / k and Ge / (e t) =
 * d Ge / k bytes, each ring moving 2(r-1)/r of it for r participants, so
 *   g = ceil(2 ((n-1) Gd + (n d - 1) Ge) 1e9 / (n k bw))  ns,
 * bw the type's intra-node bandwidth when n = 1 and the stage's devices fit
 * in one node (the EDP copies alone, inside the node), else its slowest
 * NIC.  With d = 1 this is the untiled formula. */
static int64_t tiled_sync(const orc_ctx* x, int g, int j, int64_t n, int64_t d, int32_t lo, int32_t hi) {
    int64_t Ge = x->eparam[hi] - x->eparam[lo];
    int64_t Gd = (x->param[hi] - x->param[lo]) - Ge;
    u128 vol = (u128)(n - 1) * (u128)Gd + (u128)(n * d - 1) * (u128)Ge;
    if (vol == 0) return 0;
    int64_t bw = (n == 1 && (1 << j) <= x->maxnode[g]) ? x->intra_bw[g] : x->inter_bw[g];
    return ceil_div128((u128)2 * vol * 1000000000u, (u128)n * (u128)(1 << j) * (u128)bw);
}

/* §5.3: the per-stage fastest tilings are the starting point and the
 * choice is re-selected against the whole iteration time on the split a.
 * Exact form (reading): for a bound Y on the gradient term every stage
 * takes its fastest fitting tiling with g_s <= Y (the earliest on ties),
 * giving T(Y) = (M-1) max t_s + sum t_s + max g_s; the result is the
 * smallest T(Y) over Y among the g values of all options, the smaller Y on
 * ties.  A combination whose largest gradient term is Y* is matched or
 * beaten by T(Y*), so this is the minimum of T over all combinations.
 * Writes the plan's largest stage time and the chosen tilings. */
static int64_t evaluate_tiled(const orc_ctx* x, int S, int M, int64_t n, const tiles* tl, const int64_t* c,
                              const int64_t* f_s, const int64_t* cap, const int* g, const int* j, const int32_t* a,
                              int64_t* B_out, uint8_t* tile_out) {
    int64_t ot[MAXS][10], og[MAXS][10];
    int fits[MAXS][10];
    for (int s = 0; s < S; ++s)
        for (int o = 0; o < tl[s].n; ++o) {
            int64_t mem = (x->state[a[s + 1]] - x->state[a[s]]) +
                          tl[s].d1[o] * (x->estate[a[s + 1]] - x->estate[a[s]]) +
                          f_s[s] * (x->act[a[s + 1]] - x->act[a[s]]);
            fits[s][o] = mem <= cap[s];
            ot[s][o] = tl[s].P[o][a[s + 1]] - tl[s].P[o][a[s]] + c[s];
            og[s][o] = tiled_sync(x, g[s], j[s], n, tl[s].d1[o] + 1, a[s], a[s + 1]);
        }
    int64_t bestT = INF, bestY = 0, bestB = 0;
    for (int ys = 0; ys < S; ++ys)
        for (int yo = 0; yo < tl[ys].n; ++yo) {
            if (!fits[ys][yo]) continue;
            int64_t Y = og[ys][yo];
            int64_t tm = 0, ts = 0, gm = 0;
            int pick[MAXS], all = 1;
            for (int s = 0; s < S && all; ++s) {
                pick[s] = -1;
                for (int o = 0; o < tl[s].n; ++o)
                    if (fits[s][o] && og[s][o] <= Y && (pick[s] < 0 || ot[s][o] < ot[s][pick[s]])) pick[s] = o;
                if (pick[s] < 0) {
                    all = 0;
                    break;
                }
                if (ot[s][pick[s]] > tm) tm = ot[s][pick[s]];
                ts += ot[s][pick[s]];
                if (og[s][pick[s]] > gm) gm = og[s][pick[s]];
            }
            if (!all) continue;
            int64_t T = (int64_t)(M - 1) * tm + ts + gm;
            if (T < bestT || (T == bestT && Y < bestY)) {
                bestT = T;
                bestY = Y;
                bestB = tm;
                for (int s = 0; s < S; ++s) tile_out[s] = tl[s].code[pick[s]];
            }
        }
    *B_out = bestB;
    return bestT;
}

/* ---------------------------------------------- the paper's split rule */

/* §5.3 "Layer split and DP degree": the paper's planner gives each stage
 * layers in proportion to its profiled speed; if that split exceeds a
 * stage's memory it prices a fixed list of alternative splits and keeps the
 * fastest that fits.  Readings: the speed of stage s is 2^40 divided by the
 * time of all L layers on its type and degree, rounded down; the list is
 * (1) in proportion to speed, (2) equal layer counts, (3) in proportion to
 * the longest run of consecutive layers each stage's memory holds; the
 * fastest is the smallest pipeline time (M-1) max t_s + sum t_s, the
 * earlier alternative on ties -- Algorithm 1 splits the layers before the
 * fill picks the DP degree, so the choice cannot see the gradient term. */

/* L layers over S stages in proportion to weights w >= 0 (sum > 0): floor
 * of the exact share, at least one layer per stage; missing layers go one
 * each to the largest remainders (the earlier stage on ties); surplus
 * layers (the one-layer minimum can overshoot) come one at a time off the
 * stage holding the most (the later stage on ties).  Boundaries to a. */
static void proportional_split(int S, int L, const int64_t* w, int32_t* a) {
    int64_t V = 0;
    for (int s = 0; s < S; ++s) V += w[s];
    int64_t cnt[MAXS], rem[MAXS];
    int64_t total = 0;
    for (int s = 0; s < S; ++s) {
        int64_t share = (int64_t)L * w[s];
        cnt[s] = share / V;
        rem[s] = share % V;
        if (cnt[s] < 1) cnt[s] = 1;
        total += cnt[s];
    }
    int given[MAXS] = {0};
    while (total < L) {
        int best = -1;
        for (int s = 0; s < S; ++s)
            if (!given[s] && (best < 0 || rem[s] > rem[best])) best = s;
        given[best] = 1;
        cnt[best] += 1;
        total += 1;
    }
    while (total > L) {
        int best = -1;
        for (int s = 0; s < S; ++s)
            if (cnt[s] > 1 && (best < 0 || cnt[s] >= cnt[best])) best = s;
        cnt[best] -= 1;
        total -= 1;
    }
    a[0] = 0;
    for (int s = 0; s < S; ++s) a[s + 1] = a[s] + (int32_t)cnt[s];
}

/* Longest run of consecutive layers [i, j) with W[j] - W[i] <= cap. */
static int64_t longest_run(const int64_t* W, int L, int64_t cap) {
    int64_t best = 0;
    for (int i = 0; i < L; ++i)
        for (int j = i + 1; j <= L && W[j] - W[i] <= cap; ++j)
            if (j - i > best) best = j - i;
    return best;
}

/* The paper's rule: returns 1 and the chosen split in a (with its T and
 * max t_s) if one of the alternatives fits, else 0. */
static int distribute(const orc_ctx* x, int S, int L, int M, int64_t n, const int64_t* const* P,
                      const int64_t* c, const int64_t* const* W, const int64_t* cap, const int* g,
                      const int* j, int32_t* a, int64_t* T_out, int64_t* B_out) {
    int64_t w[3][MAXS];
    for (int s = 0; s < S; ++s) {
        int64_t all = P[s][L];
        w[0][s] = all > 0 ? ((int64_t)1 << 40) / all : ((int64_t)1 << 40);
        w[1][s] = 1;
        w[2][s] = longest_run(W[s], L, cap[s]);
    }
    int found = 0;
    int64_t best_pipe = 0;
    for (int alt = 0; alt < 3; ++alt) {
        int64_t V = 0;
        for (int s = 0; s < S; ++s) V += w[alt][s];
        if (V <= 0) continue;
        int32_t b[MAXS + 1];
        proportional_split(S, L, w[alt], b);
        int fits = 1;
        for (int s = 0; s < S && fits; ++s)
            if (W[s][b[s + 1]] - W[s][b[s]] > cap[s]) fits = 0;
        if (!fits) continue;
        int64_t tmax = 0, tsum = 0;
        for (int s = 0; s < S; ++s) {
            int64_t t = P[s][b[s + 1]] - P[s][b[s]] + c[s];
            if (t > tmax) tmax = t;
            tsum += t;
        }
        int64_t pipe = (int64_t)(M - 1) * tmax + tsum;
        if (!found || pipe < best_pipe) {
            found = 1;
            best_pipe = pipe;
            for (int s = 0; s <= S; ++s) a[s] = b[s];
        }
    }
    if (found) *T_out = evaluate(x, S, M, n, P, c, j, g, a, B_out);
    return found;
}

/* Price one candidate; node_free (nullable) replaces the cluster's GPUs per
 * node for the DP degree (the GPUs a plan has left, Algorithm 1). */
static void price_one(const orc_ctx* x, int S, int M, const uint8_t* codes, int64_t* f,
                      int64_t* Wbuf, priced* out, const int32_t* node_free) {
    int L = x->L;
    memset(out, 0, sizeof(*out));
    out->T = -1;
    out->B = -1;
    /* decode and validate the structural template (§5.1 masks) */
    int g[MAXS], j[MAXS];
    if (S < 1 || S > MAXS || S > L || M < 1) {
        out->status = ORC_INVALID;
        return;
    }
    for (int s = 0; s < S; ++s) {
        int b = codes[s];
        g[s] = b & 7;
        j[s] = (b >> 3) & 3;
        if ((b >> 5) != 0 || g[s] >= x->n_types || x->gpus[g[s]] == 0 ||
            (!x->moe && (1 << j[s]) > x->maxnode[g[s]])) {
            out->status = ORC_INVALID;
            return;
        }
    }
    /* DP degree (§5.3) */
    int64_t n = dp_degree(x, S, g, j, node_free);
    if (n == 0) {
        out->status = ORC_NO_FIT;
        return;
    }
    out->n = n;
    /* stage views for PartitionLayers */
    const int64_t* P[MAXS];
    const int64_t* W[MAXS];
    int64_t c[MAXS], cap[MAXS];
    for (int s = 0; s < S; ++s) {
        P[s] = x->P + ((size_t)g[s] * 4 + j[s]) * (L + 1);
        if (s + 1 < S) {
            int same = g[s] == g[s + 1] && (1 << j[s]) + (1 << j[s + 1]) <= x->maxnode[g[s]];
            c[s] = x->p2p[g[s]][g[s + 1]][same];
        } else {
            c[s] = 0;
        }
        /* memory (§5.2): parameters, gradients and optimizer state of the
         * stage's layers plus the activations of its in-flight microbatches
         * (1F1B keeps min(S - s, M) on stage s), all split over the k GPUs of
         * the group; compared as total <= capacity * k */
        int64_t inflight = (S - s) < M ? (S - s) : M;
        int64_t* w = Wbuf + (size_t)s * (L + 1);
        for (int i = 0; i <= L; ++i) w[i] = x->state[i] + inflight * x->act[i];
        W[s] = w;
        cap[s] = x->mem[g[s]] * (int64_t)(1 << j[s]);
    }
    if (x->tiled) {
        /* expert tiling (§5.3): every stage may use each valid tiling of
         * its devices */
        tiles tl[MAXS];
        int64_t fs[MAXS];
        for (int s = 0; s < S; ++s) {
            tl[s].n = 0;
            for (int i = 0; i < (j[s] + 1) * (j[s] + 2) / 2; ++i) {
                int slot = tile_base[j[s]] + i, le = 0, lt = 0, ld = 0;
                if (!x->tvalid[g[s]][slot]) continue;
                tiling_of(j[s], i, &le, &lt, &ld);
                tl[s].P[tl[s].n] = x->Pt + ((size_t)g[s] * 20 + slot) * (L + 1);
                tl[s].d1[tl[s].n] = ((int64_t)1 << ld) - 1;
                tl[s].code[tl[s].n] = (uint8_t)(le | (lt << 2));
                tl[s].n += 1;
            }
            fs[s] = (S - s) < M ? (S - s) : M;
        }
        int64_t Bt;
        if (!partition_tiled(x, S, tl, c, fs, cap, f, &Bt, out->a)) {
            out->status = ORC_OOM;
            return;
        }
        out->T = evaluate_tiled(x, S, M, n, tl, c, fs, cap, g, j, out->a, &out->B, out->tile);
        out->status = ORC_OK;
        return;
    }
    if (x->split_mode == 1) {
        /* the paper's split rule instead of PartitionLayers */
        if (!distribute(x, S, L, M, n, P, c, W, cap, g, j, out->a, &out->T, &out->B)) {
            out->status = ORC_OOM;
            out->T = out->B = -1;
            return;
        }
        out->status = ORC_OK;
        return;
    }
    int64_t B;
    if (!partition(S, L, P, c, W, cap, f, &B, out->a)) {
        out->status = ORC_OOM;
        return;
    }
    int64_t tmax;
    out->B = B;
    out->T = evaluate(x, S, M, n, P, c, j, g, out->a, &tmax);
    out->status = ORC_OK;
}

void orc_set_split(orc_ctx* x, int mode) { x->split_mode = mode; }

typedef struct {
    const orc_ctx* x;
    int64_t lo, hi;
    const uint8_t* S;
    const uint16_t* M;
    const uint8_t* code;
    int64_t stride;
    int s_max;
    int64_t *T, *B;
    uint16_t* n_dp;
    uint8_t *status, *bounds, *tiling;
    int64_t n_all;
} job;

static void* run_job(void* arg) {
    job* jb = (job*)arg;
    const orc_ctx* x = jb->x;
    int L = x->L;
    int64_t* f = (int64_t*)malloc(sizeof(int64_t) * (size_t)(MAXS + 1) * (L + 1));
    int64_t* Wbuf = (int64_t*)malloc(sizeof(int64_t) * (size_t)MAXS * (L + 1));
    uint8_t codes[MAXS];
    for (int64_t c = jb->lo; c < jb->hi; ++c) {
        int S = jb->S[c];
        priced r;
        if (S > jb->s_max) {
            memset(&r, 0, sizeof(r));
            r.T = r.B = -1;
            r.status = ORC_INVALID;
        } else {
            for (int s = 0; s < S && s < MAXS; ++s) codes[s] = jb->code[(int64_t)s * jb->stride + c];
            price_one(x, S, jb->M[c], codes, f, Wbuf, &r, NULL);
        }
        jb->T[c] = r.T;
        jb->B[c] = r.B;
        jb->n_dp[c] = (uint16_t)(r.status == ORC_OK || r.status == ORC_OOM ? r.n : 0);
        jb->status[c] = (uint8_t)r.status;
        if (jb->bounds) {
            for (int s = 0; s <= MAXS; ++s)
                jb->bounds[(int64_t)s * jb->n_all + c] =
                    (r.status == ORC_OK && s <= S) ? (uint8_t)r.a[s] : 0;
        }
        if (jb->tiling) {
            for (int s = 0; s < MAXS; ++s)
                jb->tiling[(int64_t)s * jb->n_all + c] = (r.status == ORC_OK && s < S) ? r.tile[s] : 0;
        }
    }
    free(f);
    free(Wbuf);
    return NULL;
}

int orc_price_tiled(const orc_ctx* x, int64_t n, const uint8_t* S, const uint16_t* M,
                    const uint8_t* code, int64_t plane_stride, int s_max, int64_t* T,
                    int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* bounds,
                    uint8_t* tiling, int threads) {
    if (x->tiled && x->split_mode != 0) return -1; /* tiling prices the min-max split only */
    if (threads < 1) threads = 1;
    if (threads > n) threads = n > 0 ? (int)n : 1;
    job* jobs = (job*)calloc(threads, sizeof(job));
    pthread_t* tid = (pthread_t*)calloc(threads, sizeof(pthread_t));
    for (int t = 0; t < threads; ++t) {
        job* jb = &jobs[t];
        jb->x = x;
        jb->lo = n * t / threads;
        jb->hi = n * (t + 1) / threads;
        jb->S = S;
        jb->M = M;
        jb->code = code;
        jb->stride = plane_stride;
        jb->s_max = s_max;
        jb->T = T;
        jb->B = bottleneck;
        jb->n_dp = n_dp;
        jb->status = status;
        jb->bounds = bounds;
        jb->tiling = tiling;
        jb->n_all = n;
    }
    if (threads == 1) {
        run_job(&jobs[0]);
    } else {
        for (int t = 0; t < threads; ++t) pthread_create(&tid[t], NULL, run_job, &jobs[t]);
        for (int t = 0; t < threads; ++t) pthread_join(tid[t], NULL);
    }
    free(jobs);
    free(tid);
    return threads;
}

int orc_price(const orc_ctx* x, int64_t n, const uint8_t* S, const uint16_t* M,
              const uint8_t* code, int64_t plane_stride, int s_max, int64_t* T,
              int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* bounds,
              int threads) {
    return orc_price_tiled(x, n, S, M, code, plane_stride, s_max, T, bottleneck, n_dp, status, bounds,
                           NULL, threads);
}

/* ------------------------------------------------- multi-template plans */

/* Algorithm 1 builds a plan as a sequence of structural templates, each
 * holding its own GPUs (§5 "Planning as autoregressive construction"); the
 * reward of a step is the throughput the new template adds (§5.5,
 * Eq. reward).  A plan is priced template by template against the GPUs the
 * earlier templates left: the template's DP degree comes from the free
 * GPUs per node, its groups are then placed -- largest first, each on a
 * node of its type whose free GPUs equal the group size, else on the node
 * with the fewest free GPUs above it (§5.1: a node whose size equals the
 * requested degree first, else GPUs from a larger node; the earliest node
 * on ties) -- and a template that does not fit (OOM, NO_FIT, INVALID) ends
 * the plan at the templates placed so far.  Plan throughput (reading): the
 * sum over placed templates of n M 1e9 / T base micro-batches per second,
 * each term rounded in IEEE double, in template order. */
static void place_groups(const orc_ctx* x, int S, const int* g, const int* j, int64_t n, int32_t* node_free) {
    for (int e = 3; e >= 0; --e) {
        int32_t w = 1 << e;
        for (int s = 0; s < S; ++s) {
            int k = 1 << j[s];
            int eb = j[s];
            while ((1 << eb) > x->maxnode[g[s]]) --eb;
            if (eb != e) continue;
            int64_t blocks = (int64_t)(k >> eb) * n;
            for (int64_t b = 0; b < blocks; ++b) {
                int pick = -1;
                for (int d = 0; d < x->n_nodes; ++d)
                    if (x->node_type[d] == g[s] && node_free[d] == w) {
                        pick = d;
                        break;
                    }
                if (pick < 0)
                    for (int d = 0; d < x->n_nodes; ++d)
                        if (x->node_type[d] == g[s] && node_free[d] > w &&
                            (pick < 0 || node_free[d] < node_free[pick]))
                            pick = d;
                if (pick < 0) return; /* cannot happen: n came from these nodes */
                node_free[pick] -= w;
            }
        }
    }
}

int orc_price_plans(const orc_ctx* x, int64_t n_plans, int max_tmpl, const uint8_t* n_tmpl,
                    const uint8_t* S, const uint16_t* M, const uint8_t* code, int s_max,
                    int64_t* T, int64_t* bottleneck, uint16_t* n_dp, uint8_t* status, uint8_t* placed,
                    double* thr) {
    int L = x->L;
    int64_t* f = (int64_t*)malloc(sizeof(int64_t) * (size_t)(MAXS + 1) * (L + 1));
    int64_t* Wbuf = (int64_t*)malloc(sizeof(int64_t) * (size_t)MAXS * (L + 1));
    int32_t* node_free = (int32_t*)malloc(sizeof(int32_t) * (x->n_nodes > 0 ? x->n_nodes : 1));
    for (int64_t c = 0; c < n_plans; ++c) {
        for (int d = 0; d < x->n_nodes; ++d) node_free[d] = x->node_gpus[d];
        int ended = 0, nt = n_tmpl[c] < max_tmpl ? n_tmpl[c] : max_tmpl;
        double sum = 0.0;
        placed[c] = 0;
        for (int t = 0; t < max_tmpl; ++t) {
            int64_t o = (int64_t)t * n_plans + c;
            T[o] = -1;
            bottleneck[o] = -1;
            n_dp[o] = 0;
            if (ended || t >= nt) {
                status[o] = ORC_SKIPPED;
                continue;
            }
            int St = S[o];
            uint8_t codes[MAXS];
            priced r;
            if (St > s_max) {
                memset(&r, 0, sizeof(r));
                r.status = ORC_INVALID;
            } else {
                for (int s = 0; s < St && s < MAXS; ++s) codes[s] = code[((int64_t)t * s_max + s) * n_plans + c];
                price_one(x, St, M[o], codes, f, Wbuf, &r, node_free);
            }
            status[o] = (uint8_t)r.status;
            if (r.status != ORC_OK) {
                n_dp[o] = (uint16_t)(r.status == ORC_OOM ? r.n : 0);
                ended = 1;
                continue;
            }
            T[o] = r.T;
            bottleneck[o] = r.B;
            n_dp[o] = (uint16_t)r.n;
            sum = sum + ((double)(r.n * (int64_t)M[o]) * 1e9) / (double)r.T;
            placed[c] = (uint8_t)(t + 1);
            int g[MAXS], j[MAXS];
            for (int s = 0; s < St; ++s) {
                g[s] = codes[s] & 7;
                j[s] = (codes[s] >> 3) & 3;
            }
            place_groups(x, St, g, j, r.n, node_free);
        }
        thr[c] = sum;
    }
    free(f);
    free(Wbuf);
    free(node_free);
    return 0;
}

/* ------------------------------------------------------------ rank, top-k */

typedef struct {
    int64_t idx, T;
    uint32_t nM;
} entry;

/* a before b: higher throughput nM/T, compared exactly as nM_a*T_b vs
 * nM_b*T_a; equal throughput goes to the smaller index. */
static int better_first(const void* pa, const void* pb) {
    const entry* a = (const entry*)pa;
    const entry* b = (const entry*)pb;
    u128 lhs = (u128)a->nM * (u128)b->T;
    u128 rhs = (u128)b->nM * (u128)a->T;
    if (lhs != rhs) return lhs > rhs ? -1 : 1;
    return a->idx < b->idx ? -1 : (a->idx > b->idx ? 1 : 0);
}

int orc_topk(int64_t n, int64_t base_index, const int64_t* T, const uint16_t* n_dp,
             const uint16_t* M, const uint8_t* status, int k, int64_t* out_idx,
             int64_t* out_T, uint32_t* out_nM) {
    entry* e = (entry*)malloc(sizeof(entry) * (size_t)(n > 0 ? n : 1));
    int64_t m = 0;
    for (int64_t c = 0; c < n; ++c) {
        if (status[c] != ORC_OK) continue;
        e[m].idx = base_index + c;
        e[m].T = T[c];
        e[m].nM = (uint32_t)n_dp[c] * (uint32_t)M[c];
        ++m;
    }
    qsort(e, (size_t)m, sizeof(entry), better_first);
    int cnt = (int)(m < k ? m : k);
    for (int i = 0; i < cnt; ++i) {
        out_idx[i] = e[i].idx;
        out_T[i] = e[i].T;
        out_nM[i] = e[i].nM;
    }
    free(e);
    return cnt;
}
