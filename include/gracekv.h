/*
 * gracekv.h -- C ABI of the GraceKV prefill-time KV-cache compression pass
 * (arxiv 2608.07001, "Every Cache Entry Earns Its Place: Global Allocation of
 * Resolution and Coverage for KV Cache Compression"), implemented as
 * hand-written CUDA kernels for sm_103a (GB300).
 *
 * The pass follows the problem statement of Sec. 3.1 / App. A.1: after one
 * prefill, the cache K, V of every layer l and KV head g is compressed into a
 * ragged cache of at most B_total entries (one entry = one stored K/V pair).
 * Four calls, in this order, on one context:
 *
 *   gracekv_segment      curvature-guided slot partition      (App. B.2-B.3)
 *   gracekv_build_trees  prototype trees, node values, gains  (App. A.3-A.5)
 *   gracekv_allocate     global greedy Add/Split allocation   (App. A.5, C.3)
 *   gracekv_gather       ragged compressed cache + index map  (App. A.5)
 *
 * Decoding on the result (gracekv_decode_*, App. A.3 Eq. app_decode_logit)
 * follows at the end of this header.
 *
 * Conventions for every call:
 *   - Tensor arguments are DEVICE pointers to contiguous row-major arrays owned
 *     by the caller; the library never frees or retains them past the call.
 *     Arguments named *_host are host pointers.
 *   - K and V have layout [L][G][T][d] (G = number of KV heads); Q (the
 *     observation-window queries, placed after the input at positions
 *     T..T+W-1, all seeing [0, T)) has layout [L][Hq][W][d]; query head h
 *     belongs to KV head h / (Hq / G).  Element type = params.dtype
 *     (fp32 or bf16) for K, V, Q, K_out and V_out.
 *   - K, V, Q, K_out and V_out must start on a 16-byte boundary (they are
 *     read and written as 16-byte vectors); int32/float arrays on 4 bytes,
 *     int64 arrays on 8.  A misaligned pointer returns GKV_EINVAL.
 *   - `stream` is a cudaStream_t passed as void*; work is enqueued on it.
 *     Calls that return a host count (*_host) synchronise that stream once.
 *   - Every call returns a gkv_status and never aborts or throws.  A CUDA
 *     error makes the context sticky-failed (GKV_ECUDA on every later call);
 *     gracekv_last_error() describes the first failure.
 *   - Calls out of order return GKV_ESTATE without enqueuing work.
 *   - A context and its workspace belong to one device (the device current
 *     at gracekv_create); calls on one context must not overlap.
 */
#ifndef GRACEKV_H
#define GRACEKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GRACEKV_ABI_VERSION 4

typedef enum {
    GKV_OK = 0,
    GKV_EINVAL = 1,        /* bad shape, pointer or hyper-parameter */
    GKV_EBUDGET = 2,       /* budget cannot hold L*G*4 recent entries, or no context left */
    GKV_ENOMEM = 3,        /* device workspace allocation failed */
    GKV_ECUDA = 4,         /* a CUDA call failed (context is now sticky-failed) */
    GKV_ETIMEOUT = 5,      /* a bounded device-side wait gave up */
    GKV_ENONFINITE = 6,    /* a NaN/Inf input or intermediate was found */
    GKV_ESTATE = 7,        /* call out of order, or context already failed */
    GKV_EUNSUPPORTED = 8,  /* valid per the paper but not built here (see message) */
    GKV_ECAPACITY = 9      /* an output buffer is too small */
} gkv_status;

typedef enum { GKV_F32 = 0, GKV_BF16 = 1 } gkv_dtype;

typedef struct gracekv_ctx gracekv_ctx;

/*
 * Shapes and hyper-parameters.  Defaults (gracekv_default_params) are the
 * paper's: App. A.1 (recent window 32), App. B.2 (windows {4,8,16},
 * lambda_stab 0.25, lambda_s 0.15, segmentation layers at relative depths
 * 0.33/0.50/0.67), App. B.3 (n_min 16, n_max 128, n0 64, lambda_d 0.25,
 * lambda_n 0.10, c_cut 1.0), App. B.4 (K = 16 split candidates), App. A.3
 * (lambda_kappa 0.05, lambda_Z 0.25, lambda_M 0.75, value base 0.1), App. B.2
 * (epsilon 1e-6).
 */
typedef struct {
    int32_t L, G, Hq, T, d, W;     /* layers, KV heads, query heads, tokens, head dim, probes */
    int32_t dtype;                 /* gkv_dtype of K, V, Q, K_out, V_out */
    int32_t ctx_start, ctx_end;    /* context [c_s, c_e) inside [0, T) (App. A.1) */
    int32_t recent;                /* requested recent window r (shrinks to fit the budget) */
    int64_t budget;                /* B_total = floor(L G N_ctx / x), App. A.1 Eq. app_total_budget */
    double rope_base;              /* RoPE base of the keys (0: keys carry no RoPE) */
    int32_t n_min, n_max, n0;      /* slot length bounds and target (App. B.3) */
    double lambda_stab, lambda_s, lambda_d, lambda_n, c_cut;
    int32_t seg_layers[8];         /* explicit segmentation layers, or n_seg_layers = 0 */
    int32_t n_seg_layers;          /*   for the relative-depth rule of App. B.2 */
    int32_t windows[4];            /* curvature window scales (App. B.2) */
    int32_t n_windows;
    int32_t k_cand;                /* top-K curvature split candidates (App. B.4); 0..16 */
    double lambda_kappa, lambda_Z, lambda_M, eps, base_frac;
    double lambda_graph;           /* multi-hop weight (App. A.4; the paper's value 0.3, 0: direct
                                      relevance only); > 0 needs gracekv_set_graph_queries */
    double alpha_floor;            /* singleton-floor cap alpha (App. A.5 Stage I, Eq. app_floor_cap);
                                      0: no floor (the paper's "w/o SF"); the paper's value is 0.6 */
    /* The paper's ablations (App. B.4 last paragraph, App. C.1); 0 = the method.
     * seg_mode 1 ("w/o CS" with k_cand = 0 and lambda_kappa = 0): uniform slots
     *   of target length n0 over the compressible context -- J = max(1,
     *   round-half-up(N_c / n0)) slots, slot j starting at c_s + floor(j N_c / J)
     *   -- and curvature 0 everywhere (k_cand = 0 leaves the midpoint as the
     *   only binary cut, lambda_kappa = 0 drops the curvature reward).
     * quota_alloc 1 ("w/o GA"): each (l, g) gets the fixed capacity
     *   floor(B_free / LG) (+1 for the first B_free mod LG pairs) and cannot use
     *   capacity another pair leaves; trees are then built completely. */
    int32_t seg_mode;
    int32_t quota_alloc;
    /* Singleton floor (used when alpha_floor > 0; App. A.5 Stage I, App. C.4):
     * consensus weight c (0.5), gate gamma (1.2, f >= gamma / N_c), value mass
     * eta (0.95), max-pool half width (3: width 7).  Candidates of an (l, g):
     * f descending (ties: lower t) up to the longest prefix whose token values
     * sum to at most eta.  When their joint cost C0 (per slot: the frontier
     * size after isolating them) exceeds cap = floor(alpha B_free), each (l, g)
     * keeps its first max(1, floor(n cap / C0)); each then walks those in
     * order and accepts every one whose path still fits what is left of its
     * share floor(cap n' / sum n'), skipping those that do not.  Accepted
     * positions become singleton leaves by forced extraction, and the floor's
     * Adds and extractions are executed before the auction.  Not combined with
     * quota_alloc (GKV_EUNSUPPORTED). */
    double floor_c, floor_gamma, floor_eta;
    int32_t floor_half;
    /* Multi-hop relevance (lambda_graph > 0; App. A.4): seed mass eta_seed
     * (0.9), at most m_seed seeds per hop (64, at most 64), r_hop hops (2),
     * inter-hop decay rho_hop (0.5).  Graph layers at relative depths 0.50 and
     * 0.75.  Needs bf16, d in {64, 128} and N_c <= 131072 (GKV_EUNSUPPORTED). */
    double eta_seed, rho_hop;
    int32_t m_seed, r_hop;
    /* Execution of the segmentation DP (App. B.3 Eq. app_dp_recurrence); the
     * slots do not depend on it.  The recurrence runs in chunks of 32 steps of
     * min(n_min, 16) endpoints on separate CTAs, each started dp_warmup tokens
     * early from a flat state; a chunk whose state at its start is not the
     * previous chunk's up to a constant is run again, in order, from the
     * previous chunk's exact state.  0: 512 tokens (rounded up to whole steps);
     * negative: one chunk, the plain sequential recurrence on one CTA. */
    int32_t dp_warmup;
} gkv_params;

/* Fill *p with the paper's defaults; shapes and budget are left zero.  Host only. */
gkv_status gracekv_default_params(gkv_params *p);

/* B_total = floor(L * G * n_ctx / x) for compression ratio x >= 1
 * (App. A.1 Eq. app_total_budget).  Returns -1 for invalid arguments.  Host only. */
int64_t gracekv_budget_for_ratio(int32_t L, int32_t G, int32_t n_ctx, double x);

/* The graph layers of the multi-hop relevance (App. A.4; their depths are
 * stated in App. A.1): the distinct layers floor(0.50 L) and floor(0.75 L)
 * (each at most L - 1), ascending, written to out[0 .. n-1] (nullable; room
 * for 2).  Returns n (1 or 2), or -1 for L <= 0.  Host only. */
int32_t gracekv_graph_layers(int32_t L, int32_t *out);

/* Validate *p, resolve the recent window against the budget (r = 32, shrunk to
 * floor(B_total / (L G)) when L G r > B_total, never below 4: App. A.1) and
 * allocate the device workspace on the current device.  On success *out owns
 * it; release with gracekv_destroy.  Errors: GKV_EINVAL, GKV_EBUDGET,
 * GKV_EUNSUPPORTED (d not in {64, 128}, W > 64, n_max above 128, G d above
 * 2048, a compressible region whose segmentation DP does not fit one CTA's
 * shared memory -- about 630,000 tokens with the default n_min and n_max,
 * about 170,000 with a negative dp_warmup; lambda_graph > 0 with fp32 inputs
 * or N_c above 131072; alpha_floor > 0 together with quota_alloc), GKV_ENOMEM,
 * GKV_ECUDA. */
gkv_status gracekv_create(const gkv_params *p, gracekv_ctx **out);
void gracekv_destroy(gracekv_ctx *ctx);
const char *gracekv_last_error(const gracekv_ctx *ctx);
const char *gracekv_status_string(gkv_status s);

/* Resolved quantities: effective recent window r, compressible length
 * N_c = c_e - r - c_s, free budget B_free = B_total - L G r (App. A.1
 * Eq. app_free_budget), and the number of slots of the last segmentation. */
gkv_status gracekv_query(const gracekv_ctx *ctx, int32_t *recent, int32_t *n_c,
                         int64_t *b_free, int32_t *n_slots);

/*
 * Stage 1 -- curvature-guided segmentation (App. B.2-B.3).
 * Trajectory h^(l)_t = concat_g V[l][g][t][:] at the segmentation layers
 * (or `hidden` [n_seg][T][Dh] fp32 when given, Dh a multiple of 8 up to
 * 2048, 16-byte aligned), multi-scale curvature
 * (Eq. app_local_curvature), stabilised curvature (Eq.
 * app_stabilized_curvature), robust-z boundary score (Eq. app_boundary_score,
 * surprisal [T] fp32 optional, 0 when NULL), and the length-constrained DP
 * (Eq. app_dp_recurrence with the terminal relaxation of Eq.
 * app_terminal_predecessor) over the compressible region [c_s, c_e - r).
 * Outputs: slot_starts (device, [cap + 1] int32, absolute positions,
 * slot_starts[J] = c_e - r), *n_slots_host = J (synchronises `stream`),
 * kappa (device, nullable, [T] fp32 stabilised curvature).
 * Errors: GKV_EINVAL, GKV_ECAPACITY (J > cap), GKV_ENONFINITE, GKV_ECUDA.
 */
gkv_status gracekv_segment(gracekv_ctx *ctx, const void *V, const float *hidden, int32_t Dh,
                           const float *surprisal, int32_t *slot_starts, int32_t cap,
                           int32_t *n_slots_host, float *kappa, void *stream);

/*
 * Stage 2a (optional) -- the observation-query score passes of stage 2: row
 * statistics (max logit, partition over [0, T), partition over the
 * compressible region) of every probe row (l, h, u), and the token values of
 * the compressible region (App. A.3 max-logit shift; App. A.4 Eqs.
 * app_attention_probability, app_direct_relevance, app_bottom_up_value).
 * They read K and Q only, so they can overlap the segmentation: the passes
 * are enqueued on `stream` (which should differ from the segmentation's) --
 * right away when a segmentation has been done and its trees not yet built,
 * otherwise by the next gracekv_segment, after an event recorded on its
 * stream before its first kernel.  The next gracekv_build_trees with
 * the same K and Q pointers uses these results instead of recomputing them,
 * after making its own stream wait for them; K and Q must not change until
 * then.  Asynchronous.
 * Errors: GKV_EINVAL (null or misaligned pointer), GKV_ESTATE, GKV_ECUDA.
 */
gkv_status gracekv_score(gracekv_ctx *ctx, const void *K, const void *Q, void *stream);

/*
 * Stage 2 -- prototype trees (App. A.3), token and node values (App. A.4),
 * gains (App. A.5 Eq. app_operation_gains).  Requires a prior
 * gracekv_segment (its curvature drives the split candidates).  If
 * slot_starts (device, [n_slots + 1] int32 absolute) is non-NULL it replaces
 * the segmentation's slots (externally supplied partition of [c_s, c_e - r));
 * omega (device [L][G] fp32, nullable = all ones) is the head sensitivity.
 * Row statistics (max logit, partition over [0, T), partition over the
 * compressible region) are computed for every probe row (l, h, u); the trees
 * stay in the context's workspace.  In order, after the token values: with
 * lambda_graph > 0 the multi-hop relevance (App. A.4) mixes into them, from
 * the queries of the last gracekv_set_graph_queries; with alpha_floor > 0
 * the singleton floor (App. A.5 Stage I) is chosen from the (mixed) values;
 * then the trees are built, floor positions extracted first.  A supplied
 * slot may hold 1 to 16384 tokens (the segmentation's hold n_min..n_max);
 * every tree recurses to single-token leaves whatever its slot's length.
 * Errors: GKV_EINVAL (also: lambda_graph > 0 without graph queries, supplied
 * slots that do not partition the region), GKV_ESTATE, GKV_EUNSUPPORTED (a
 * supplied slot longer than 16384 tokens), GKV_ENOMEM, GKV_ECUDA.
 */
gkv_status gracekv_build_trees(gracekv_ctx *ctx, const void *K, const void *V, const void *Q,
                               const float *omega, const int32_t *slot_starts, int32_t n_slots,
                               void *stream);

/*
 * Stage 3 -- global greedy allocation (App. A.5 Stage II, App. C.3): the
 * result equals a max-priority queue keyed by U = Delta / c with order
 * (U desc, unit (l, g, j) asc, node (a asc, b desc)), seeded with every Add,
 * discarding unaffordable pops, under B_free.  *n_entries_host receives the
 * number of cache entries E = L G (T - N_c) + used (synchronises `stream`).
 * Errors: GKV_ESTATE, GKV_ENONFINITE, GKV_ECUDA.
 */
gkv_status gracekv_allocate(gracekv_ctx *ctx, int64_t *n_entries_host, void *stream);

/*
 * Stage 4 -- packing (App. A.5 "Frontier updates and physical packing").
 * Per (l, g), in this order: prefix tokens [0, c_s), the frontier nodes of
 * every covered slot in ascending position, the recent window and the
 * suffix [c_e - r, T).  Non-singleton nodes store (ktil, vtil, p, log m_eff)
 * (Eqs. app_rope_prototype, app_value_prototype,
 * app_effective_multiplicity); single tokens store their original K/V bits,
 * position and log m = 0.  Outputs (device): K_out, V_out [cap][d] dtype,
 * pos [cap] int32, log_m [cap] fp32, src_lo / src_hi [cap] int32 (the token
 * interval each entry covers), offsets [L G + 1] int64 (entry range of each
 * (l, g)).  cap must be >= the count returned by gracekv_allocate.
 * Errors: GKV_ESTATE, GKV_ECAPACITY, GKV_ECUDA.
 */
gkv_status gracekv_gather(gracekv_ctx *ctx, const void *K, const void *V, void *K_out,
                          void *V_out, int32_t *pos, float *log_m, int32_t *src_lo,
                          int32_t *src_hi, int64_t *offsets, int64_t cap, void *stream);

/*
 * The whole pass from host buffers: K, V [L][G][T][d] and Q [L][Hq][W][d]
 * (dtype of the params; page-locked host memory gives the full copy rate),
 * omega (host [L][G] fp32, nullable).  The inputs are copied to device
 * buffers the context keeps (allocated on the first call), layer group by
 * layer group on a copy stream of the context, and the work that needs only
 * the layers already copied starts as they land: the segmentation after Q
 * and its layers of V, the score passes and the first tree-building launch
 * of each layer group after that group (tensor-core score path; otherwise
 * after the last group); the pruning passes, the allocation and the packing
 * follow on `stream`.  The cache is then copied to the host arrays (layouts
 * of gracekv_gather; capacity `cap` entries, offsets [L G + 1]).
 * Synchronous: returns when the host arrays hold the cache; *n_entries_host
 * receives E.  No hidden states, surprisal, supplied slots or graph queries
 * (use the stage calls for those).  Errors: those of the stage calls,
 * GKV_ECAPACITY (E > cap), GKV_ENOMEM (device copies of the inputs),
 * GKV_EUNSUPPORTED (lambda_graph > 0).
 */
gkv_status gracekv_compress_host(gracekv_ctx *ctx, const void *K, const void *V, const void *Q,
                                 const float *omega, void *K_out, void *V_out, int32_t *pos, float *log_m,
                                 int32_t *src_lo, int32_t *src_hi, int64_t *offsets, int64_t cap,
                                 int64_t *n_entries_host, void *stream);

/*
 * Introspection for tests and tools (not needed to compress).  Copies the
 * current trees and selection to caller-owned HOST arrays (synchronises
 * `stream`).  Node records of all units are packed unit after unit, unit
 * order (l, g, j); within a unit in creation order (breadth-first for slots
 * of at most 128 tokens; a longer slot's tree is created level by level,
 * each node of at most 128 tokens getting slots reserved for its subtree).
 *   unit_first [L G J + 1] int64: node range of each unit
 *   unit_Uadd, unit_Ddrop [L G J] fp32; add_sel [L G J] uint8
 *   per node (capacity node_cap): a, b, child0 (index within the unit, -1 for
 *   leaves), nchild (-1: pending, not evaluated; -2: an unused reserved
 *   slot, to be skipped), cost int32; D, R, U, kappa fp32; split_sel uint8
 *   row stats (nullable) [L][Hq][W] fp32: max logit, Z over [0,T), Z over C
 *   rtok (nullable) [L][G][N_c] fp32 token values
 * *n_nodes_host receives the node count (GKV_ECAPACITY if > node_cap).
 */
gkv_status gracekv_export(gracekv_ctx *ctx, int64_t node_cap, int64_t *n_nodes_host,
                          int64_t *unit_first, float *unit_Uadd, float *unit_Ddrop,
                          uint8_t *add_sel, int32_t *a, int32_t *b, int32_t *child0,
                          int32_t *nchild, int32_t *cost, float *D, float *R, float *U,
                          float *kappa, uint8_t *split_sel, float *row_m, float *row_Z,
                          float *row_ZC, float *rtok, void *stream);

/*
 * The queries of every position at the graph layers, for the multi-hop
 * relevance of the next gracekv_build_trees (App. A.4, Eqs.
 * app_global_seed_score, app_hop_propagation, app_diffused_relevance):
 * Qg [n_graph][Hq][T][d] bf16 (device; the caller keeps it alive until the
 * build returns), n_graph = the number of graph layers (the distinct layers
 * floor(0.50 L) and floor(0.75 L)), in ascending layer order.  The seeds'
 * rows attend to their causal range [0, u]; the token values become
 * R = (1 - lambda_graph) s-hat + lambda_graph d-hat.  Errors: GKV_EINVAL,
 * GKV_ESTATE (lambda_graph = 0).
 */
gkv_status gracekv_set_graph_queries(gracekv_ctx *ctx, const void *Qg, int32_t n_graph);

/*
 * Layer-KV-head sensitivity omega (App. A.4, Eqs. app_head_sensitivity_raw,
 * app_head_sensitivity), the per-(l, g) multiplier the pass takes as its
 * omega input.  No context, no allocation.
 *   W_O [L][D][Hq d] bf16: each layer's attention output projection, row-major
 *     (out_features x in_features); column block h (d columns) is W_O^{l,h}.
 *   o [L][Hq][U][d] bf16: the heads' attention outputs at the U question
 *     probes, before the projection (U <= 64).
 *   omega [L][G] fp32 (device, output); scratch: L G 65 fp32 (device).
 * static = (sum_{h in H(g)} ||W_O^{l,h}||_F^2)^{1/2}, input = mean_u
 * ||sum_{h in H(g)} W_O^{l,h} o_u^{l,h}||_2, raw = sqrt(static input),
 * omega = raw / (mean raw + 1e-6).  Products on the tensor cores (exact bf16
 * products, fp32 sums).  Errors: GKV_EINVAL, GKV_EUNSUPPORTED (dtype other
 * than bf16, d not in {64, 128}, U > 64, D not a multiple of 8), GKV_ECUDA.
 */
gkv_status gracekv_head_sensitivity(const void *W_O, const void *o, int32_t L, int32_t G, int32_t Hq,
                                    int32_t d, int32_t D, int32_t U, int32_t dtype, float *omega,
                                    float *scratch, void *stream);

/*
 * The singleton floor of the last gracekv_build_trees (alpha_floor > 0), to
 * caller-owned HOST arrays (synchronises `stream`): accepted [L G][N_c] uint8
 * (1 = a floor singleton), f [L G][N_c] fp32 floor scores (nullable),
 * *B_floor_host the entries the floor's ops take.  GKV_ESTATE without a floor.
 */
gkv_status gracekv_export_floor(gracekv_ctx *ctx, uint8_t *accepted, float *f, int64_t *B_floor_host,
                                void *stream);

/*
 * Measurement support (not needed to compress).  gracekv_profile(ctx, 1)
 * makes every later stage call record CUDA events on its stream around each
 * kernel group: 0 segmentation, 1 row statistics, 2 token values, 3 unit
 * trees, 4 allocation, 5 gather, 6 singleton floor, 7 multi-hop relevance.
 * gracekv_stats synchronises the events of the calls made since the last
 * gracekv_stats / gracekv_profile and returns
 * the summed milliseconds per group in stage_ms[0 .. n_stages-1] (nullable);
 * *launches (nullable) receives the number of kernels this context has
 * launched since it was created; work[0 .. n_work-1] (nullable) receives the
 * tree-building work of the last gracekv_build_trees: [0] probe-scan token
 * steps, [1] candidate intervals evaluated, [2] sum of candidate lengths,
 * [3] units built, [4] chunks of the last segmentation DP, [5] of those, the
 * chunks that were run again from the exact state (their warm-up had not
 * reached the true state up to a constant).
 */
#define GRACEKV_N_STAGES 8
gkv_status gracekv_profile(gracekv_ctx *ctx, int32_t enable);
gkv_status gracekv_stats(gracekv_ctx *ctx, float *stage_ms, int32_t n_stages, int64_t *launches,
                         uint64_t *work, int32_t n_work);

/*
 * Allocation-free row statistics (the paper has no counterpart: this is a
 * deployment entry point).  For callers that must not call cudaMalloc -- an
 * engine that reserves the whole device for its own memory pool, or a
 * latency-critical loop that cannot take the device synchronisation an
 * allocation may cause -- this call computes, without a context and without
 * allocating, the same per-probe-row statistics as gracekv_build_trees: for
 * every row (l, h, u) the max logit m over [0, T), Z = sum exp(x - m) over
 * [0, T) and Z^C over the range [c_lo, c_hi).  K [L][G][T][d] and Q
 * [L][Hq][W][d] (dtype GKV_F32 / GKV_BF16) are device inputs; row_m, row_Z,
 * row_ZC [L][Hq][W] fp32 are device outputs; work is enqueued on `stream`.
 *   Scratch: a fixed 4 MiB device array inside this library (held by every
 *   GPU that loads it until the process exits); L * Hq * W above 349525 rows
 *   returns GKV_ECAPACITY.  The first call on a device resolves the array's
 *   device address; make that first call before any stream capture.
 *   Calls share the array: calls that overlap on the GPU (other streams,
 *   other threads) race and must be serialised by the caller.
 *   Non-finite inputs are not detected: a NaN or Inf in K or Q gives NaN or
 *   Inf rows and the call still returns GKV_OK (it never synchronises, so it
 *   has no point at which to report a device-side check); a caller whose
 *   inputs may be non-finite checks the outputs.
 *   Errors: GKV_EINVAL (shapes, pointers, L * G above 65535), GKV_ECAPACITY,
 *   GKV_ECUDA.
 */
gkv_status gracekv_row_stats_noalloc(const void *K, const void *Q, int32_t L, int32_t G,
                                     int32_t Hq, int32_t T, int32_t d, int32_t W, int32_t dtype,
                                     int32_t c_lo, int32_t c_hi, float *row_m, float *row_Z,
                                     float *row_ZC, void *stream);

/*
 * Decoding on the compressed cache (App. A.3, Eq. app_decode_logit, and the
 * packing paragraph of App. A.5).  The packed cache of gracekv_gather stays
 * read-only while decoding; every token generated afterwards is appended to
 * its (l, g) with effective multiplicity 1 (log m = 0), in an append area the
 * caller owns.  For layer l, query head h of KV head g = h / (Hq / G):
 *     x_e = q_h . k_e / sqrt(d) + log m_e  over the entries e of (l, g),
 *     out_h = sum_e softmax(x)_e v_e ;
 * the entries of (l, g) are the packed ones [offsets[lg], offsets[lg + 1])
 * followed by the first n_app appended rows.  An (l, g) with no entry gives a
 * zero output.  These calls need no context and never allocate.
 *
 * gkv_decode_cache describes the cache (all pointers DEVICE memory, owned by
 * the caller): L, G, Hq, d and dtype as at compression (d in {64, 128},
 * Hq / G in {1, 2, 4, 8}, else GKV_EUNSUPPORTED); K, V [n_entries][d] dtype
 * (16-byte aligned), log_m [n_entries] fp32 and offsets [L G + 1] int64 as
 * written by gracekv_gather, n_entries = E its count (below 2^31; offsets past
 * it make gracekv_decode_status report GKV_EINVAL and nothing is read);
 * K_app, V_app [L][G][app_cap][d] dtype (16-byte aligned; nullable when
 * app_cap = 0).
 */
typedef struct {
    int32_t L, G, Hq, d, dtype;
    const void *K, *V;
    const float *log_m;
    const int64_t *offsets;
    int64_t n_entries;
    void *K_app, *V_app;
    int32_t app_cap;
} gkv_decode_cache;

/* Bytes of the device workspace gracekv_decode_attention needs for this
 * cache geometry (the per-piece partials, a counter per (l, g) and a status
 * word).  The caller allocates it 256-byte aligned and zeroes it once; every
 * call leaves it zeroed again (the status word aside, see
 * gracekv_decode_status).  One workspace serves one stream at a time. */
gkv_status gracekv_decode_workspace_size(const gkv_decode_cache *c, size_t *bytes);

/* Append the new token of layers [l0, l0 + n_layers): k_new, v_new
 * [n_layers][G][d] dtype (device, 16-byte aligned) become row n_app of the
 * append area of each (l, g).  The caller then counts n_app + 1 rows.
 * Errors: GKV_EINVAL, GKV_ECAPACITY (n_app >= app_cap), GKV_ECUDA. */
gkv_status gracekv_decode_append(const gkv_decode_cache *c, int32_t l0, int32_t n_layers,
                                 int32_t n_app, const void *k_new, const void *v_new, void *stream);

/* Decoding attention of layers [l0, l0 + n_layers) over the packed entries
 * and the first n_app appended rows.  q [n_layers][Hq][d] dtype (device,
 * already rotated for the current position, like the cached keys); out
 * [n_layers][Hq][d] fp32 (device, 16-byte aligned).  Asynchronous on
 * `stream`; a device-side failure sets the workspace's status word, which
 * gracekv_decode_status reports.  Errors: GKV_EINVAL (shapes, pointers,
 * n_app > app_cap), GKV_EUNSUPPORTED, GKV_ECUDA. */
gkv_status gracekv_decode_attention(const gkv_decode_cache *c, int32_t l0, int32_t n_layers,
                                    int32_t n_app, const void *q, float *out, void *workspace,
                                    void *stream);

/* Synchronises `stream` and reports (then clears) the workspace's status
 * word: GKV_ETIMEOUT when a bounded device-side wait of an earlier
 * gracekv_decode_attention on this workspace gave up, GKV_EINVAL when the
 * offsets of a call pointed past n_entries, else GKV_OK. */
gkv_status gracekv_decode_status(void *workspace, void *stream);

#ifdef __cplusplus
}
#endif
#endif
