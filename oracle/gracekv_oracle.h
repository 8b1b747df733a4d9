/*
 * gracekv_oracle.h -- plain CPU oracle of the GraceKV prefill-time compression
 * pass (arxiv 2608.07001, "Every Cache Entry Earns Its Place").
 *
 * TEST INFRASTRUCTURE ONLY.  This oracle exists to check the CUDA path; only
 * tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load it.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Everything is single-threaded fp64 arithmetic on the exact input values
 * (bf16/fp32 inputs are widened to double by the caller), written as plain
 * loops that follow the paper's definitions in the paper's order:
 *
 *   budget            Sec. App. A.1, Eq. (app_total_budget), (app_free_budget)
 *   curvature         App. B.2, Eqs. (app_hidden_normalization) ..
 *                     (app_stabilized_curvature)
 *   boundary score    App. B.2, Eqs. (app_robust_z), (app_mad), (app_boundary_score)
 *   DP segmentation   App. B.3, Eqs. (app_adjacent_difference) ..
 *                     (app_terminal_predecessor)
 *   row statistics    App. A.3 "Prototype distortion" (max-logit shift),
 *                     App. A.4 Eq. (app_attention_probability)
 *   token values      App. A.4 Eqs. (app_direct_relevance), (app_bottom_up_value)
 *   prototypes        App. A.3 Eqs. (app_rope_prototype), (app_value_prototype),
 *                     (app_effective_multiplicity)
 *   distortion        App. A.3 Eqs. (app_original_attention_stats) ..
 *                     (app_node_and_drop_distortion)
 *   refinement        App. A.3 Eqs. (app_binary_split) .. (app_split_choice),
 *                     App. B.4 Eq. (app_tree_split_candidates)
 *   gains / costs     App. A.5 Eqs. (app_operation_gains) .. (app_unit_utility)
 *   greedy allocation App. A.5 Stage II, App. C.3 (max-priority queue)
 *   packing           App. A.5 "Frontier updates and physical packing"
 *   head sensitivity  App. A.4 Eqs. (app_head_sensitivity_raw), (app_head_sensitivity)
 *   decoding          App. A.3 Eq. (app_decode_logit) over the packed cache
 *                     plus appended tokens at multiplicity 1 (App. A.5)
 *
 * Readings of silent or ambiguous passages:
 *   R1  trajectory h^(l)_t = concat_g v^(l,g)_t unless hidden states are given;
 *       surprisal defaults to 0; omega defaults to 1; lambda_graph = 0.
 *   R2  visible range of every probe = [0, T); probes = the W observation
 *       queries; distortion probe u uses query head H(g)[u mod |H(g)|].
 *   R3  b_i rewards a cut between positions i and i+1.
 *   R4  median = lower median (rank floor((n-1)/2)).
 *   R5  DP ties -> first maximum in ascending predecessor a.
 *   R6  split candidates: top-K positions t in [a, b-2] by kappa (ties: lower
 *       t), cut xi = t+1, plus midpoint xi = a + floor(n/2); kappa-hat is the
 *       min-max normalisation of kappa over [a, b-2] (0 when flat); cut ties
 *       -> smallest xi; extraction p* = argmax R_tok (ties: lower t);
 *       binary wins a rho tie.
 *   R7  normalisation of the mass weight = the probe's full partition over
 *       [0, T) with the same max-logit shift.
 *   R8  epsilon = 1e-6 wherever the paper writes epsilon without a value.
 *   R9  p_v = round half to even of the mean position.
 *   R10 single-token intervals store the original K/V, p = t, m = 1, D = 0.
 *   R11 RoPE: half-split pairs (i, i + d/2), theta_i = base^(-2i/d),
 *       RoPE^-1(k, t) = RoPE(k, -t); base 0 means keys carry no rotation.
 *   R12 gains are clamped at 0; heap order (U desc, unit asc, a asc, b desc);
 *       an unaffordable pop is discarded for good.
 *   R13 "w/o CS": J = max(1, round-half-up(N_c / n0)) slots, slot j starting at
 *       c_s + floor(j N_c / J) (lengths differ by at most one); curvature is
 *       taken as 0 everywhere; the split candidates and the curvature reward
 *       are removed with k_cand = 0 and lambda_kappa = 0 (midpoint only).
 *   R14 "w/o GA": (l, g) number lg gets the capacity floor(B_free / LG), plus
 *       one for lg < B_free mod LG; the heap pops as before and discards an op
 *       its (l, g) cannot afford; a pair's unused capacity is lost.
 *   R16 multi-hop relevance (App. A.4): graph layers at the relative depths
 *       0.50 and 0.75 that App. A.1 states, read as floor(rho L) with
 *       duplicates dropped; seeds of a hop = tokens
 *       of C in order of their score descending (ties: lower t), taken while
 *       fewer than m_seed are taken and their running mass is below eta_seed
 *       (the seed that reaches eta is included); hop 1 scores = S-hat (Eq.
 *       app_global_seed_score), later hops = the previous hop's propagation
 *       score normalised over C; a hop's seed weights are its scores over
 *       the seed set, normalised to sum 1 (uniform when they sum to 0); seed u
 *       attends to [0, u] (its causal visible range); the propagation score
 *       of a hop is zeroed at that hop's and all earlier seeds.
 *   R15 singleton floor (App. A.5 Stage I, App. C.4): R = the token values
 *       after the multi-hop mix (the direct ones when lambda_graph = 0); the
 *       consensus is the mean over all (l, g); the
 *       max-pool window is clipped to the compressible context.  Candidates
 *       of an (l, g): f descending (ties: lower t), while f >= gamma / N_c,
 *       stopping before the running sum of R would exceed eta.  Joint cost
 *       of a set S in a slot = the slot's frontier size after isolating S =
 *       |S| + number of maximal runs of slot positions outside S.  When the
 *       joint cost C0 of all candidates exceeds cap = floor(alpha B_base)
 *       (B_base = the auction budget without a floor), every (l, g) with
 *       n >= 1 candidates keeps its first n' = max(1, floor(n cap / C0)).
 *       Per-head safeguard: an (l, g) may use cap_h = floor(cap n' / sum n')
 *       entries (its share of the cap by kept candidates; the shares sum to at
 *       most cap, so the global cap holds).  An (l, g) walks its kept
 *       candidates in order and accepts each one whose complete path still
 *       fits cap_h; one that does not fit is skipped and the walk goes on,
 *       so a later, cheaper candidate can still be accepted (App. A.5: a
 *       candidate is accepted only when its path remains feasible, and the
 *       floor is not switched off for a head when the budget is tight).  A
 *       candidate's path costs 1 for its slot's Add if the slot is still
 *       uncovered, plus the new entries of extracting it from its current
 *       frontier interval [lo, hi]: [lo, t) and (t, hi] when non-empty.
 *       A node whose interval holds accepted positions is extracted at the one
 *       with the largest f (ties: lower t); the floor ops (the Adds of slots
 *       with an accepted position and these extractions) execute before the
 *       auction, which gets B_base - B_floor.
 *
 * Parity is pinned for every function here (see tests/test_oracle_*.py);
 * no function is "parity unpinned".
 */
#ifndef GRACEKV_ORACLE_H
#define GRACEKV_ORACLE_H
#include <stdint.h>

typedef struct {
    int32_t L, G, Hq, T, d, W;
    int32_t ctx_start, ctx_end;   /* context [c_s, c_e) inside [0, T) */
    int32_t recent;               /* requested recent window r */
    double rope_base;             /* 0: keys carry no RoPE */
    int32_t n_min, n_max, n0;
    double lambda_stab, lambda_s, lambda_d, lambda_n, c_cut;
    int32_t seg_layers[8];
    int32_t n_seg_layers;
    int32_t windows[4];
    int32_t n_windows;
    int32_t k_cand;
    double lambda_kappa, lambda_Z, lambda_M, eps, base_frac;
    int32_t disp_mode;            /* 0: definition, 1: paper's prefix form */
    double alpha_floor;           /* singleton-floor cap alpha (0: no floor, "w/o SF") */
    double floor_c, floor_gamma, floor_eta;   /* consensus weight, gate, cumulative value */
    int32_t floor_half;           /* max-pool half width (7 = 2 * 3 + 1) */
    double lambda_graph;          /* multi-hop weight (0: direct relevance only) */
    double eta_seed, rho_hop;     /* seed mass, inter-hop decay */
    int32_t m_seed, r_hop;        /* at most m_seed seeds per hop, r_hop hops */
    int32_t seg_mode;             /* 0: curvature DP; 1: uniform slots of target length n0
                                     and curvature 0 (the "w/o CS" ablation, App. B.4 end) */
    int32_t quota_alloc;          /* 0: one shared budget; 1: fixed per-(l, g) capacity
                                     B_free / LG (the "w/o GA" ablation, App. C.1) */
} orc_params;

/* Per-node records of all trees (flat, capacity = L*G*2*N_c). */
typedef struct {
    int64_t cap;
    int64_t count;      /* out */
    int32_t *lg, *slot, *a, *b, *parent, *child0, *nchild, *form, *cost;
    int32_t *floor_op;  /* 1: a forced extraction of the singleton floor */
    double *D, *Ddrop, *R, *U, *kappa, *kscale;
    double *m_cut, *m_form, *m_topk, *m_ext;
} orc_nodes;

int orc_budget(const orc_params *p, int64_t B_total, int32_t *r_eff, int64_t *B_free);

int orc_curvature(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                  double *kappa_out, double *kappa_lw_out);
int orc_robust_z(const double *a, int32_t n, double *z);
int orc_segment(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                const double *surprisal, double *kappa_out, double *b_out,
                int32_t *slot_starts, int32_t cap, int32_t *n_slots,
                double *dp_best, double *dp_second);

int orc_uniform_slots(const orc_params *p, int32_t *slot_starts, int32_t cap, int32_t *n_slots);

int orc_dp_weights(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                   const double *b, int32_t n, const int32_t *a_rel, const int32_t *i_rel,
                   double *w_out);

int orc_row_stats(const orc_params *p, const double *Q, const double *K,
                  double *m, double *Z, double *ZC);
int orc_token_values(const orc_params *p, const double *Q, const double *K,
                     const double *m, const double *Z, double *rtok);

int orc_eval_interval(const orc_params *p, const double *K, const double *V,
                      const double *Q, const double *m, const double *Z,
                      const double *rtok, int32_t l, int32_t g, int32_t a, int32_t b,
                      double *D, double *Ddrop, double *ktil, double *vtil,
                      int32_t *pos, double *logm);

/* Singleton floor (reading R15).  rtok [L G][N_c]; outputs f [L G][N_c],
 * accepted [L G][N_c] (1 = an accepted floor position), *B_floor (its
 * entries) and *n_cand (initial candidates before the cap). */
int orc_floor(const orc_params *p, const double *rtok, const int32_t *slot_starts, int32_t n_slots,
              int64_t B_base, double *f, uint8_t *accepted, int64_t *B_floor, int64_t *n_cand);

/* floor_acc / floor_f (nullable): the accepted floor positions and their
 * scores; nodes holding one are extracted there (floor_op = 1). */
int orc_build_trees(const orc_params *p, const double *K, const double *V, const double *Q,
                    const double *omega, const double *kappa, const int32_t *slot_starts,
                    int32_t n_slots, const double *m, const double *Z, const double *rtok,
                    const uint8_t *floor_acc, const double *floor_f,
                    orc_nodes *nodes, double *unit_Uadd, int64_t *unit_root);

/* unit_floor (nullable): 1 for a slot whose Add is a floor op.  The floor ops
 * execute first; *used counts them and the auction's entries. */
int orc_allocate(const orc_params *p, int64_t B_free, int32_t n_slots,
                 const orc_nodes *nodes, const double *unit_Uadd, const int64_t *unit_root,
                 const uint8_t *unit_floor, uint8_t *add_sel, uint8_t *split_sel, int64_t *used);

int orc_gather(const orc_params *p, const double *K, const double *V, const double *rtok,
               int32_t n_slots, const orc_nodes *nodes, const int64_t *unit_root,
               const uint8_t *add_sel, const uint8_t *split_sel, int64_t cap,
               double *K_out, double *V_out, int32_t *pos, double *log_m,
               int32_t *src_lo, int32_t *src_hi, int64_t *offsets, int64_t *n_entries);

/* Multi-hop relevance, App. A.4 Eqs. (app_global_seed_score),
 * (app_hop_propagation), (app_diffused_relevance), reading R16.  shat
 * [L G][N_c] the direct relevance (Eq. app_direct_relevance); Qg
 * [n_graph][Hq][T][d] the queries of every position at the graph layers
 * graph_l[]; K [L][G][T][d].  Output dhat [N_c]; seeds [r_hop][m_seed]
 * (absolute positions, -1 padded) and their weights (nullable). */
int orc_multihop(const orc_params *p, const double *shat, const double *Qg, const int32_t *graph_l,
                 int32_t n_graph, const double *K, double *dhat, int32_t *seeds, double *seed_w);
int orc_graph_layers(const orc_params *p, int32_t *out);

/* Layer-KV-head sensitivity, App. A.4 Eqs. (app_head_sensitivity_raw),
 * (app_head_sensitivity).  W_O [L][D][Hq d] (the output projection of each
 * layer, row-major: column block h is W_O^{l,h}); o [L][Hq][U][d] (attention
 * outputs of the U question probes before the projection); omega [L][G]. */
int orc_head_sensitivity(int32_t L, int32_t G, int32_t Hq, int32_t d, int32_t D, int32_t U,
                         const double *W_O, const double *o, double eps, double *omega);

/* q [nl][Hq][d] for layers l0 .. l0 + nl - 1; packed cache K, V [E][d],
 * log_m [E], off [L G + 1]; appended rows K_app, V_app [L][G][app_cap][d]
 * (the first n_app of each (l, g) are valid); out [nl][Hq][d]. */
int orc_decode_attention(int32_t L, int32_t G, int32_t Hq, int32_t d, int32_t l0, int32_t nl,
                         const double *q, const double *K, const double *V, const double *log_m,
                         const int64_t *off, const double *K_app, const double *V_app,
                         int32_t app_cap, int32_t n_app, double *out);

#endif
