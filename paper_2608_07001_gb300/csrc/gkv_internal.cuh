// gkv_internal.cuh -- internal declarations shared by the CUDA translation
// units of the GraceKV compression library (context, workspace, launchers,
// small device helpers).  Not part of the public ABI (include/gracekv.h).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <string>
#include <vector>

#include "../../include/gracekv.h"

namespace gkv {

constexpr int kMaxUnit = 128;       // longest slot a unit kernel holds in shared memory
constexpr int kMaxSlot = 16384;     // longest slot of a supplied partition (longer ones: long units, build_long.cu)
constexpr int kStPipeTimeout = 32;   // status bit: a bounded wait of a tensor-core pipeline gave up
constexpr int kStLongCap = 64;       // status bit: the long-unit work items exceeded their capacity
constexpr int kScoreStatus = 8;      // dev_int word of the score passes' status bits
constexpr int kDpRerun = 9;          // dev_int word: segmentation DP chunks re-run from the exact state
constexpr int kMaxSegLayers = 8;
constexpr int kMaxWindows = 4;

// ---------------------------------------------------------------------------
// Workspace owned by a context.  All arrays are device memory.
// ---------------------------------------------------------------------------
struct Workspace {
    // RoPE rotation table: (cos, sin)(t * theta_i) for t in [0, T), i < d/2.
    float2 *rope = nullptr;
    float2 *rope_rel = nullptr;    // [2 kMaxSlot - 1][d/2] rotations by the offsets -(kMaxSlot-1)..kMaxSlot-1
    int4 *ent = nullptr;           // [B_total + L G (T - N_c)] frontier entry descriptors of the gather
    // segmentation
    float *inv_norm = nullptr;     // [n_seg][T] 1 / max(||h_t||, eps)
    float *nrm2 = nullptr;         // [n_seg][T] ||hbar_t||^2
    double *klw = nullptr;         // [n_seg * n_win][T] curvature per (layer, window)
    double *kappa = nullptr;       // [T] stabilised curvature
    double *bscore = nullptr;      // [T] boundary score
    double *zbuf = nullptr;        // [T] scratch for robust z
    unsigned long long *zdev = nullptr;   // [T] keys of the absolute deviations (robust z)
    double *p2 = nullptr;          // [N_c + 1] prefix of sum_l ||d_t||^2
    float *ew = nullptr;           // [(N_c + 1) * nbp] DP edge weights (len n_min..n_max), rows padded to 4
    float2 *ewt = nullptr;         // [n_max + 1] terminal edge weights (len 1..n_max) at i = N_c
    int32_t *slots = nullptr;      // [N_c + 2] slot starts (absolute)
    uint8_t *dp_len = nullptr;     // [N_c + 16] DP: chosen slot length of every endpoint
    float2 *dp_head = nullptr;     // [chunks][128] DP state (double-float) on the window ending at a chunk's start
    float2 *dp_tail = nullptr;     // [chunks][256] DP state on the window ending at a chunk's end
    uint8_t *dp_tab = nullptr;     // [chunks][n_max] DP: where the path leaves a chunk, per entry point
    int32_t *dev_int = nullptr;    // [16] small device scalars (J, status, counts, ...)
    unsigned long long *sel_state = nullptr;   // [4] radix-select state of the robust z
    unsigned int *sel_hist = nullptr;          // [2048] its global digit histogram
    // row statistics and token values
    float *row_m = nullptr, *row_Z = nullptr, *row_ZC = nullptr;  // [L*Hq*W]
    float *rowp = nullptr;         // [3][L*Hq*W][n_chunks] pass-A partials
    float *row_mneg = nullptr;     // [L*Hq*W] -(m log2 e + log2 Z): pass-B exponent offset
    float *Eg = nullptr;           // [L*G][N_c][32][2] probe weights exp(q_u.k_t / sqrt(d) - m_u) of every
                                   // compressible token, (u, u + 32) pairs (written by the tensor-core pass B)
    short *qperm = nullptr;        // [gq W] rows of a KV head in pass B's column order: probe rows first
    double *lg_scale = nullptr;    // [L*G] pass-B normaliser 1 / (sum_r Z^C_r / Z_r + eps)
    float *rtok = nullptr;         // [L*G*N_c]
    // node records, indexed lg*2*N_c + 2*(slot start - c_s) + k
    int32_t *nd_a = nullptr, *nd_b = nullptr, *nd_child0 = nullptr;
    int32_t *nd_parent = nullptr;  // global index of the parent; roots: -2 - unit id
    int32_t *nd_unit = nullptr;    // unit id lg * J + j
    int8_t *nd_nchild = nullptr, *nd_cost = nullptr;
    float *nd_D = nullptr;         // distortion D(I_v) of every node (resumed nodes read
                                   // exactly the value their parent computed)
    float *nd_R = nullptr, *nd_U = nullptr, *nd_kappa = nullptr;
    uint8_t *nd_sel = nullptr;     // split selected (1), discarded tie (2)
    // singleton floor (alpha_floor > 0)
    float *fl_rbar = nullptr;      // [N_c] consensus token value
    float *fl_f = nullptr;         // [L G][N_c] floor scores
    uint8_t *fl_acc = nullptr;     // [L G][N_c] accepted floor positions
    unsigned long long *fl_head = nullptr;   // [L G][8] per (l, g) selection state
    unsigned long long *fl_glob = nullptr;   // [4] joint cost, kept candidates, floor entries
    uint8_t *u_floor = nullptr;    // [units_cap] slots whose Add is a floor op
    // multi-hop relevance (lambda_graph > 0)
    float *mh_sc = nullptr, *mh_acc = nullptr;   // [N_c] seed scores, accumulated propagation
    float *mh_dpart = nullptr;     // [n_graph Hq][N_c] propagation per (graph layer, head)
    float *mh_stat = nullptr;      // [n_graph Hq][chunks][64][2] row statistics per chunk
    float *mh_rowmz = nullptr;     // [n_graph Hq][64][2]
    uint8_t *mh_was = nullptr;     // [N_c]
    int32_t *mh_seeds = nullptr, *mh_nseed = nullptr, *mh_graph_l = nullptr;
    float *mh_w = nullptr, *mh_red = nullptr;
    uint64_t *mh_pkeys = nullptr;  // [N_c / 2048][64] seed candidates of every part
    float *mh_psum = nullptr;      // [N_c / 2048] score sums of every part
    uint2 *ops = nullptr;          // [node_cap / 2] Split ops built so far: (key bits, node << 1 | cost - 1)
    unsigned int *n_ops = nullptr; // [1] entries of ops
    // per-unit arrays (capacity units_cap), unit id = lg * J + j
    int64_t units_cap = 0;
    int32_t *u_nnodes = nullptr;
    float *u_Uadd = nullptr, *u_Ddrop = nullptr;
    float *u_pend = nullptr;       // largest key bound of the unit's pending nodes (-1: none)
    uint8_t *u_sel = nullptr;      // Add selected (1), discarded tie (2)
    int32_t *u_count = nullptr;    // frontier entries per unit
    int64_t *u_off = nullptr;      // entry offset of each unit's frontier
    int32_t *u_list = nullptr;     // compacted unit ids (ties)
    long long *u_bsum = nullptr;   // [units_cap / 1024 + 2] block sums of the gather's offset scan
    long long *tie_bsum = nullptr; // [units_cap / 1024 + L G + 2] chunk sums of the allocation's tie scan
    // allocation
    unsigned long long *hist = nullptr;        // [2048] cost-weighted histogram
    unsigned long long *alloc_state = nullptr; // see alloc.cu
    unsigned long long *work = nullptr;        // [4] tree-building work counters
    // bound-ordered expansion of pending nodes
    unsigned int *pend_hist = nullptr;         // [65536] units per bound bin
    float *pend_cut = nullptr;                 // [1] lower bound of the next pass
    unsigned int *pend_n = nullptr;            // [1] units that reach the threshold
    unsigned long long *pend_pot = nullptr;    // [1] entries a full expansion of those units could take
    // trees of long units (slots above kMaxUnit tokens, build_long.cu): one
    // level's work items, per listed unit its block of them, the unit lists
    int64_t long_cap = 0;          // work items
    int64_t long_units_cap = 0;    // listed units
    int64_t *long_gv = nullptr, *long_uid = nullptr;
    float *long_kin = nullptr;
    uint8_t *long_ufl = nullptr;
    void *long_res = nullptr;      // [long_cap] results (long_res_bytes() each)
    int32_t *long_start = nullptr, *long_cnt = nullptr;   // [long_units_cap]
    unsigned int *long_n = nullptr;                       // [4] the level's work items, small subtrees, next item
                                                          //     of <= kShortUnit and <= kMaxUnit tokens
    int32_t *long_sub = nullptr;    // [2][long_cap] the small subtrees' root nodes (global indices)
    int32_t *long_slots = nullptr;  // [N_c + 1] slot indices of the long slots
    int32_t *long_list = nullptr;   // [units_cap] long units to resume
};

struct Ctx {
    gkv_params p;
    int device = 0;
    int num_sms = 148;
    int32_t r = 0, Nc = 0, c_end = 0, nseg = 0, nwin = 0;
    int32_t seg_layers[kMaxSegLayers];
    int64_t B_free = 0;
    int64_t used = 0;              // budget spent by the last allocation
    int32_t J = 0;                 // slots of the last segmentation / build
    int stage = 0;                 // 0 created, 1 segmented, 2 built, 3 allocated
    gkv_status sticky = GKV_OK;
    std::string err;
    Workspace w;
    int64_t node_cap = 0;          // L*G*2*N_c
    int n_chunks = 0;              // pass-A chunks per row
    // measurement
    int64_t launches = 0;          // kernels launched (host count)
    const void *mh_Qg = nullptr;   // graph layers' queries of the next build (multi-hop relevance)
    const void *mh_K = nullptr;    // the keys of the build in progress
    int mh_ngraph = 0;
    int build_passes = 1;          // unit-kernel launches of the last build (pruning passes)
    int n_long = 0;                // slots of the last build longer than kMaxUnit (w.long_slots)
    int dp_chunks = 0, dp_rerun = 0;   // last segmentation: DP chunks, chunks re-run from the exact state
    // score passes issued ahead by gracekv_score (consumed by the next build);
    // requested before a segmentation, they are enqueued when its dynamic
    // program (one block) starts, so that they overlap it
    bool scored = false, score_pending = false;
    const void *score_K = nullptr, *score_Q = nullptr;
    cudaStream_t score_stream = nullptr;
    cudaEvent_t score_ev = nullptr;
    cudaEvent_t dp_ev = nullptr;   // recorded on the segmentation stream where it starts
    // host pipeline (gracekv_compress_host): device copies of the inputs, the
    // cache before its copy to the host, a copy stream and its events
    void *hK = nullptr, *hV = nullptr, *hQ = nullptr;
    float *hOm = nullptr;
    int32_t *hSlots = nullptr;
    void *oK = nullptr, *oV = nullptr;
    int32_t *opos = nullptr, *olo = nullptr, *ohi = nullptr;
    float *ologm = nullptr;
    int64_t *ooff = nullptr;
    int64_t ocap = 0;
    cudaStream_t copy_stream = nullptr;
    std::vector<cudaEvent_t> copy_ev;   // [0] start, [1] Q and the segmentation layers, [2 + g] layer group g
    bool profile = false;
    std::vector<cudaEvent_t> ev_pool;          // recorded (begin, end) pairs
    std::vector<int> ev_stage;                 // stage of each pair
    size_t ev_used = 0;
};

// RAII helper: records a (begin, end) event pair around a kernel group when
// profiling is on.
struct StageTimer {
    Ctx &c;
    cudaStream_t s;
    cudaEvent_t e1 = nullptr;
    StageTimer(Ctx &c_, int stage, cudaStream_t s_) : c(c_), s(s_) {
        if (!c.profile) return;
        if (c.ev_used + 2 > c.ev_pool.size()) {
            for (int k = 0; k < 64; k++) {
                cudaEvent_t e;
                if (cudaEventCreate(&e) != cudaSuccess) return;
                c.ev_pool.push_back(e);
            }
        }
        cudaEvent_t e0 = c.ev_pool[c.ev_used];
        e1 = c.ev_pool[c.ev_used + 1];
        c.ev_used += 2;
        c.ev_stage.push_back(stage);
        cudaEventRecord(e0, s);
    }
    ~StageTimer() {
        if (e1) cudaEventRecord(e1, s);
    }
};

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> struct Vec8;   // 8 consecutive elements
template <> struct Vec8<float> {
    float v[8];
    __device__ __forceinline__ void load(const float *p) {
        float4 a = reinterpret_cast<const float4 *>(p)[0];
        float4 b = reinterpret_cast<const float4 *>(p)[1];
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
};
template <> struct Vec8<__nv_bfloat16> {
    float v[8];
    __device__ __forceinline__ void load(const __nv_bfloat16 *p) {
        uint4 u = reinterpret_cast<const uint4 *>(p)[0];
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            float2 f = __bfloat1622float2(h[i]);
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// D += A B on the tensor cores: one m16n8k16 tile, bf16 operands (exact
// products), fp32 accumulation.  a: row-major 16x16 fragment, b0/b1: the
// column-major 16x8 fragment, c: the 16x8 accumulator (PTX ISA fragment
// layouts for mma.m16n8k16 with .bf16 operands).
__device__ __forceinline__ void mma_bf16(float c[4], const uint32_t a[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// 16-byte global -> shared copy that bypasses registers (zero-fills when
// pred is false), its commit and its wait.
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool pred) {
    unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    int n = pred ? 16 : 0;   // zero-fill past the end
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem, bool pred) {
    unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    int n = pred ? 4 : 0;   // zero-fill when not pred
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// Two independent fp32 fused multiply-adds in one instruction (Blackwell's
// packed f32x2 FMA; each lane is an ordinary round-to-nearest FMA).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

// Two floats (exactly representable in bf16) packed as a bf16x2 operand word.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

// Monotone 32-bit key of a non-negative float (larger value -> larger key).
__device__ __forceinline__ uint32_t fkey(float x) { return __float_as_uint(x); }

// ---------------------------------------------------------------------------
// Launchers (each returns the launch error, cudaSuccess otherwise)
// ---------------------------------------------------------------------------
cudaError_t launch_rope_table(Ctx &c, cudaStream_t s);

cudaError_t launch_segment(Ctx &c, const void *V, const float *hidden, int Dh,
                           const float *surprisal, float *kappa_out, cudaStream_t s);
// chunks of the segmentation DP over N endpoints: endpoints per chunk, warm-up tokens, count
void dp_chunking(const gkv_params &p, int N, int *S, int *Wu, int *nch);
// shared memory of the DP's finish kernel (bytes) for N endpoints (the larger of its two kernels)
size_t dp_smem_bytes(const gkv_params &p, int N);

// layers [l0, l1) (l1 < 0: all); a partial range needs use_tc(c)
cudaError_t launch_row_stats(Ctx &c, const void *K, const void *Q, cudaStream_t s, int l0 = 0, int l1 = -1);
// tcgen05 score passes (score_tc.cu): applicable to bf16, d in {64, 128}, at
// most 256 probe rows per KV head; row-statistics partials per row = tc_row_chunks.
bool use_tc(const Ctx &c);
int tc_row_chunks(const Ctx &c);
cudaError_t launch_row_stats_tc(Ctx &c, const void *K, const void *Q, cudaStream_t s, int lg0, int nlg);
cudaError_t launch_token_values_tc(Ctx &c, const void *K, const void *Q, cudaStream_t s, int lg0, int nlg);
cudaError_t launch_token_values(Ctx &c, const void *K, const void *Q, cudaStream_t s, int l0 = 0, int l1 = -1);
// Slots of at most kShortUnit tokens run on the unit kernel instance that fits
// two CTAs per SM; the work lists hold them (slot indices for a fresh build,
// unit ids for a resumed one) separately from the longer ones.
constexpr int kShortUnit = 64;
cudaError_t launch_unit_build(Ctx &c, const void *K, const void *V, const void *Q,
                              const float *omega, const int32_t *slots, int J, int resume,
                              int root_only, int max_levels, float tau, const int32_t *list_short,
                              int n_short, const int32_t *list_long, int n_long, cudaStream_t s,
                              int lg0 = 0, int nlg = -1);   // fresh launches: (l, g) in [lg0, lg0 + nlg);
// Subtree mode of the unit kernel (build.cu): the listed pending nodes of
// long units (global node indices; at most kShortUnit tokens in list_short,
// at most kMaxUnit in list_long) each get their subtree built to the leaves
// into the node slots reserved for it (its child0, unit-relative), except the
// children whose key bound is below tau_prune (the threshold of the ops built
// so far: it only rises, so they can never be selected); they stay pending.
cudaError_t launch_unit_subtrees(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                                 const int32_t *slots, int J, const int32_t *list_short, int n_short,
                                 const int32_t *list_long, int n_long, float tau_prune, cudaStream_t s);
// Slot indices split by length class: short ones at list[0, count[0]), those
// of kShortUnit + 1 .. kMaxUnit tokens at list[J - count[1], J), longer ones
// at long_slots[0, count[2]); count[3] receives the tokens of the longer ones.
cudaError_t launch_slot_classes(Ctx &c, const int32_t *slots, int J, int32_t *list, int *count,
                                int32_t *long_slots, cudaStream_t s);
// One level of the trees of long units (build_long.cu): with fresh = 1 the
// roots of the listed slots for (l, g) in [lg0, lg0 + nlg) (root_only: their
// own distortion and Add gain, the split left pending), else the pending
// nodes of the listed units whose key bound reaches tau.  The subtrees of
// its nodes of at most kMaxUnit tokens prune against tau_prune (the
// allocation threshold of the ops built so far, -inf when none; never a
// scheduling cut, since a node pruned inside a subtree is not resumed).  With
// n_items_host the level's work-item count is read back (synchronises s) and
// a level without work launches nothing more.
cudaError_t launch_long_level(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                              const int32_t *slots, int J, int fresh, int root_only, float tau,
                              const int32_t *list, int n_list, int lg0, int nlg, cudaStream_t s,
                              unsigned int *n_items_host, float tau_prune = -INFINITY);
size_t long_res_bytes();
// out[q nlg + i] = the unit id of long slot long_slots[q] for (l, g) = lg0 + i.
cudaError_t launch_long_units(Ctx &c, const int32_t *long_slots, int n_long, int lg0, int nlg, int J,
                              int32_t *out, cudaStream_t s);
// Allocation threshold tau over the ops built so far (alloc_state prefix /
// all-fit flag), and the units whose largest pending key bound reaches
// max(tau, cut), split by slot length class: short units at list[0, count[0]),
// those of up to kMaxUnit tokens at list[n_units - count[1], n_units), longer
// ones at long_list[0, count[2]); *pend_pot receives the entries a complete
// expansion of every unit reaching tau could take.
cudaError_t launch_threshold(Ctx &c, int J, cudaStream_t s);
cudaError_t launch_prune_list(Ctx &c, const int32_t *slots, int J, int32_t *list, int *count,
                              int32_t *long_list, cudaStream_t s);
// Bound-ordered expansion: among the units whose largest pending key bound
// reaches the threshold, the cut that keeps about `m` of them (the lower edge
// of the bin of the m-th largest bound; -inf when fewer qualify), written to
// *cut, with the number that qualify at the threshold in *n_qual.  The prune
// list then uses max(threshold, *cut).
cudaError_t launch_pend_cut(Ctx &c, int J, int m, float *cut, unsigned int *n_qual, cudaStream_t s);

cudaError_t launch_allocate(Ctx &c, int J, cudaStream_t s);
// singleton floor (floor.cu): candidates, cap and accepted positions of every (l, g)
cudaError_t launch_floor(Ctx &c, int J, cudaStream_t s);
// multi-hop relevance (relevance.cu): d-hat mixed into the token values
cudaError_t launch_multihop(Ctx &c, cudaStream_t s);
int multihop_chunks(int T);
int multihop_max_context();
int floor_head_words();
cudaError_t launch_gather(Ctx &c, const void *K, const void *V, const int32_t *slots, int J,
                          void *K_out, void *V_out, int32_t *pos, float *log_m,
                          int32_t *src_lo, int32_t *src_hi, int64_t *offsets, cudaStream_t s);

// Node index base of slot j of (l, g).
__host__ __device__ __forceinline__ int64_t node_base(int lg, int slot_start, int cs, int Nc) {
    return (int64_t)lg * 2 * Nc + 2 * (int64_t)(slot_start - cs);
}

}  // namespace gkv
