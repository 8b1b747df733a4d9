// build.cu -- stage 2 of the GraceKV pass: one prototype tree per
// layer-KV-head-slot unit (App. A.2 atomic units), built level by level by one
// CTA that keeps the whole slot in shared memory.
//
// Per unit (l, g, j), slot [sa, sb), n <= 128 tokens:
//   E[t][u] = exp(q_u . k_t / sqrt d - m_u)   distortion probe u uses query
//             head H(g)[u mod |H(g)|] (App. A.3, GQA round robin), m_u its
//             max logit over [0, T)
//   k_circ_t = RoPE^-1(k_t, t)                 (Eq. app_rope_prototype)
// For every node I = [a, b) of a level, the candidate children are prefixes
// [a, xi) and suffixes [xi, b) of I for the binary cuts X_v (top-16 positions
// by curvature in [a, b-2], cut xi = t + 1, plus the midpoint; App. B.4
// Eq. app_tree_split_candidates) and the two sides of the salient-token
// extraction at p* = argmax R_tok (Eq. app_extract_split).  For each
// candidate J the prototype (ktil, vtil, m_eff; Eqs. app_rope_prototype,
// app_value_prototype, app_effective_multiplicity) is formed by direct sums
// over J; then a forward scan (prefixes) and a backward scan (suffixes) over
// the node's tokens accumulate Z_u(J) and M_u(J) (Eq.
// app_original_attention_stats) for every probe and evaluate D_u (Eq.
// app_probe_distortion) at each candidate end, weighted by the attention mass
// Z_u(J) / Z_u (Eq. app_node_and_drop_distortion).  The refinement form
// follows Eqs. app_binary_split .. app_split_choice; gains, costs and
// utilities follow Eqs. app_operation_gains .. app_unit_utility (clamped at
// 0); each Split op also gets its bottleneck key kappa = min(U, kappa of the
// op that created the node), which the allocator's threshold select uses.
//
// Pruned construction.  A launch evaluates at most `max_levels` levels; the
// nodes below stay pending (child count -1, no Split op yet) and each unit
// reports the largest key of the ops that created its pending nodes.  The
// host then computes the allocation threshold tau over the ops built so far
// -- tau can only grow as ops are added, so it never exceeds the final
// threshold -- and resumes only the pending nodes whose creator has a key
// >= tau: a node whose creator's key is below the final threshold never
// reaches the frontier before the allocation stops, so its own Split is never
// needed.  Resuming repeats until no pending node qualifies.  Within a launch
// a child whose bound is below the launch's tau stays pending as well, so a
// resume launch may build several levels without expanding what its tau
// already rules out.
//
// Layout.  256 threads; thread (p, c) owns the probes p and p + 32 and the
// elements 4 c + 32 g + j (j < 4) of every d-vector: each value, prototype or
// key chunk it reads from shared memory serves two probes, and 8 consecutive
// threads read 128 contiguous bytes (one wavefront, no bank conflicts).
// Slots of up to 64 tokens use a 64-token instance whose footprint allows two
// CTAs per SM; longer slots use the 128-token instance.
#include "gkv_internal.cuh"

#include <cfloat>

#include <type_traits>

namespace gkv {
namespace {

constexpr int kMaxCuts = 18;     // K + midpoint, K <= 16 (+1 spare)
constexpr int kNT = 256;         // threads per CTA
constexpr int kNPP = 32;         // probe pairs: thread handles probes p and p + 32 (W <= 64)
constexpr int kNCL = 8;          // threads per probe pair (4-element groups, interleaved)
constexpr int kPPW = 32 / kNCL;  // probe pairs per warp: lane = 4 c + (pair % 4), so that the
                                 // 4 lanes reading one 16-byte chunk are adjacent (one shared-
                                 // memory wavefront serves them; lanes 8 apart would not merge)
constexpr int kNCD = 19;         // candidate intervals per direction and batch: 17 cuts + p* side + whole node

struct BuildArgs {
    const void *K, *V, *Q;
    const int32_t *slots;
    const float2 *rope;
    const double *kappa;
    const float *rtok, *row_m, *row_Z, *omega;
    const float *Eg;             // nullable: [L G][N_c][32][2] probe weights of every token (score pass B)
    const uint8_t *fl_acc;       // nullable: [L G][N_c] accepted singleton-floor positions
    const float *fl_f;           //           and their floor scores
    int L, G, Hq, T, d, W, gq, cs, Nc, J, k_cand;
    float inv_sqrt_d, lamZ, lamM, eps;
    float lam_kappa, base_frac;
    // work list: fresh launches index (slot list entry, lg), resume launches units
    int resume;                  // 0: build from the root, 1: resume pending nodes
    int subtree;                 // 1: the list holds pending nodes of at most NMAX tokens inside
                                 //    long units (build_long.cu), as global node indices; each CTA
                                 //    builds its node's subtree to the leaves into the node slots
                                 //    reserved for it (the unit-relative index in its child0)
    int root_only;               // fresh: evaluate only the root's own distortion (split stays pending)
    int max_levels;              // levels evaluated by this launch
    float tau;                   // resume: evaluate pending nodes whose key bound >= tau
    const int32_t *list;         // fresh: slot indices; resume: unit ids
    int lg0, nlg;                // fresh: the (l, g) range [lg0, lg0 + nlg) of the launch
    // outputs
    int32_t *nd_a, *nd_b, *nd_child0, *nd_parent, *nd_unit;
    int8_t *nd_nchild, *nd_cost;
    float *nd_D;
    float *nd_R, *nd_U, *nd_kappa;
    uint8_t *nd_sel;
    uint2 *ops;                  // compact list of the Split ops (allocation input)
    unsigned int *n_ops;
    int32_t *u_nnodes;
    float *u_Uadd, *u_Ddrop, *u_pend;
    uint8_t *u_sel;
    int *status;
    unsigned long long *work;
};

struct NodeS {
    float D;
    float kin;                   // bottleneck key of the op that created the node
    short a, b, parent, child0;
    signed char nchild;          // -1: pending (not evaluated)
};

struct BatchNode {
    int node;
    int ncut;
    int8_t cut[kMaxCuts];    // local cut positions xi (ascending)
    int8_t pidx[kMaxCuts];   // candidate index of [a, xi) (-1: single token)
    int8_t sidx[kMaxCuts];   // candidate index of [xi, b) (-1: single token)
    int pstar, eL, eR, whole;
    int forced;              // extraction at a singleton-floor position (a floor op)
    int pre_b, pre_e, suf_b, suf_e;   // prefixes (ascending end) in [0, NCD),
                                      // suffixes (descending start) in [NCD, 2 NCD)
    int pre_r, suf_r;                 // ends of the reserved ranges (unused entries empty)
    double kmin;             // smallest curvature over the node's cut positions
    float krange;            // 1 / (largest - smallest), 0 when they are equal
    int nchild, ca[3], cb[3];
    float cD[3];
};

struct Cand {
    int a, b;        // local interval (a == b: unused entry)
    float meff;
};

// Upper bound of a split's utility: U = omega R (D - sum D_children) / cost
// <= omega R D, since every D >= 0 and cost >= 1 (Eqs. app_operation_gains,
// app_unit_utility).  Rounded up by 1e-5 of its value: the R that the bound
// uses (one fp32 sum over the node's tokens) and the R of the later gain (the
// sum of its children's sums) differ by at most ~1.3e-6 of R, and the products
// add a few ulp, so rounding never makes a bound fall below the utility it bounds.
__device__ __forceinline__ float key_bound(float x) {
    return x + fabsf(x) * 1e-5f;
}

// Order-preserving 64-bit key of a double (larger value -> larger key), so
// that curvature ranks compare exactly like the fp64 values with integer ops.
__device__ __forceinline__ unsigned long long okey(double x) {
    unsigned long long u = (unsigned long long)__double_as_longlong(x);
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
__device__ __forceinline__ double okey_inv(unsigned long long k) {
    unsigned long long u = (k >> 63) ? (k & 0x7fffffffffffffffull) : ~k;
    return __longlong_as_double((long long)u);
}

// 8 consecutive input elements held raw in registers (the load is issued
// first, the conversion to fp32 happens at get).
template <typename T> struct Raw8;
template <> struct Raw8<float> {
    float4 a, b;
    __device__ __forceinline__ void load(const float *p) {
        a = reinterpret_cast<const float4 *>(p)[0];
        b = reinterpret_cast<const float4 *>(p)[1];
    }
    __device__ __forceinline__ void get(float v[8]) const {
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
};
template <> struct Raw8<__nv_bfloat16> {
    uint4 u;
    __device__ __forceinline__ void load(const __nv_bfloat16 *p) { u = *reinterpret_cast<const uint4 *>(p); }
    __device__ __forceinline__ void get(float v[8]) const {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; i++) {   // bf16 -> fp32 is exact: the bits move to the high half
            v[2 * i] = __uint_as_float(w[i] << 16);
            v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
};

__device__ __forceinline__ int round_half_even_mid(int a, int b) {
    int s = a + b - 1;
    if ((s & 1) == 0) return s >> 1;
    int lo = (s - 1) >> 1;
    return (lo & 1) == 0 ? lo : lo + 1;
}

// 8 consecutive elements of a shared-memory row as floats (one or two 16-byte loads).
__device__ __forceinline__ void ld8(const float *p, float v[8]) {
    float4 a = reinterpret_cast<const float4 *>(p)[0], b = reinterpret_cast<const float4 *>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void ld8(const __nv_bfloat16 *p, float v[8]) {
    uint4 u = reinterpret_cast<const uint4 *>(p)[0];
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
    for (int i = 0; i < 4; i++) {
        float2 f = __bfloat1622float2(h[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// 4 consecutive elements (8- or 16-byte aligned) as floats.
__device__ __forceinline__ float4 ld4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 ld4(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
}

// 8 consecutive elements of a shared-memory row as 4 float pairs.
__device__ __forceinline__ void ld8x2(const float *p, float2 v[4]) {
    const float4 a = reinterpret_cast<const float4 *>(p)[0], b = reinterpret_cast<const float4 *>(p)[1];
    v[0] = make_float2(a.x, a.y); v[1] = make_float2(a.z, a.w);
    v[2] = make_float2(b.x, b.y); v[3] = make_float2(b.z, b.w);
}
__device__ __forceinline__ void ld8x2(const __nv_bfloat16 *p, float2 v[4]) {
    const uint4 u = reinterpret_cast<const uint4 *>(p)[0];
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
    for (int i = 0; i < 4; i++) v[i] = __bfloat1622float2(h[i]);
}

// N consecutive elements of a shared-memory row as floats (N = 1 or 2).
template <int N>
__device__ __forceinline__ void ld_pairs(const float *p, float v[N]) {
    if constexpr (N == 2) {
        const float2 x = *reinterpret_cast<const float2 *>(p);
        v[0] = x.x; v[1] = x.y;
    } else {
#pragma unroll
        for (int j = 0; j < N; j++) v[j] = p[j];
    }
}
template <int N>
__device__ __forceinline__ void ld_pairs(const __nv_bfloat16 *p, float v[N]) {
    if constexpr (N == 2) {
        const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(p));
        v[0] = x.x; v[1] = x.y;
    } else {
#pragma unroll
        for (int j = 0; j < N; j++) v[j] = __bfloat162float(p[j]);
    }
}

template <int DH, typename Tin, int NMAX>
struct Smem {
    static constexpr int NWARPS = kNT / 32;
    static constexpr int NB = 16;            // nodes per batch
    static constexpr int MAXNODES = 2 * NMAX;
    float kc[NMAX][DH + 8];                  // rows padded by 32 B: the probe-weight MMA reads
                                             // 8 rows at once, which then fall in distinct banks
    float vv[NMAX][DH];                      // values, converted once to fp32
    float2 E[NMAX][kNPP];                    // probe weights of probes (p, p + 32)
    float ktil[kNCD][DH];                    // prototypes of one direction at a time
    float vtil[kNCD][DH];
    float Rt[NMAX];
    float Ff[NMAX];                          // floor score of an accepted floor position, -inf elsewhere
    float kn[NMAX];
    unsigned long long kap[NMAX];            // order-preserving keys of the curvature
    float redD[2 * kNCD][NWARPS];
    float redP[2 * kNCD][NWARPS];
    float candD[2 * kNCD], candP[2 * kNCD];  // per-candidate D and drop mass
    Cand cand[2 * kNCD];
    NodeS nodes[MAXNODES];
    BatchNode bn[NB];
    short lvl[2][MAXNODES];
    int nlvl[2];
    int nnodes;
    int batch_n, batch_next, batch_pre, batch_suf;   // candidate entries reserved per direction
    unsigned long long wcnt[kNT / 32][3];   // per-warp work counters
    float pend;
    float rootR;                             // R of a fresh root
};

// SUB: the subtree mode (BuildArgs::subtree) as a compile-time flag, so that
// the other instances carry none of its index mapping
template <int DH, typename Tin, int NMAX, bool SUB>
__global__ void __launch_bounds__(kNT, NMAX <= 64 ? 2 : 1) unit_build_kernel(BuildArgs A) {
    using S = Smem<DH, Tin, NMAX>;
    // thread (p, c): probes p and p + 32, elements 4 c + 32 g + j (g < NG, j < 4)
    constexpr int HALF = DH / 2, NWARPS = S::NWARPS, NG = DH / (4 * kNCL), CH = 4 * NG;
    static_assert(kNPP * kNCL == kNT && DH % (4 * kNCL) == 0, "probe layout");
    extern __shared__ __align__(16) unsigned char smem_raw[];
    S &sm = *reinterpret_cast<S *>(smem_raw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int j, lg;
    int64_t gv_sub = -1;         // subtree mode: the pending node whose subtree this CTA builds
    if constexpr (SUB) {
        gv_sub = A.list[blockIdx.x];
        const int uidr = A.nd_unit[gv_sub];
        lg = uidr / A.J;
        j = uidr - lg * A.J;
    } else if (A.resume) {
        const int uidr = A.list[blockIdx.x];
        lg = uidr / A.J;
        j = uidr - lg * A.J;
    } else {
        j = A.list[blockIdx.x / A.nlg];   // slot-major: the units of a slot share its table rows
        lg = A.lg0 + blockIdx.x % A.nlg;
    }
    const bool fresh = !A.resume && !SUB;
    const int l = lg / A.G, g = lg - l * A.G;
    const int64_t uid = (int64_t)lg * A.J + j;
    const int64_t nbase = node_base(lg, A.slots[j], A.cs, A.Nc);   // the unit's node slots
    // the tokens held: the slot, or in subtree mode the node's interval
    const int sa = SUB ? A.nd_a[gv_sub] : A.slots[j];
    const int sb = SUB ? A.nd_b[gv_sub] : A.slots[j + 1];
    const int n = sb - sa;
    // global node index of local node k, and its index inside the unit: the
    // local nodes of a subtree are its root and then its reserved slots
    const int64_t sub_res = SUB ? (int64_t)A.nd_child0[gv_sub] : 0;
    auto gidx = [&](int k) -> int64_t {
        if constexpr (SUB) return k == 0 ? gv_sub : nbase + sub_res + (k - 1);
        else return nbase + k;
    };
    if (n < 1 || n > NMAX) {
        if (tid == 0) atomicOr(A.status, 4);
        return;
    }
    const Tin *Kp = static_cast<const Tin *>(A.K) + ((size_t)lg * A.T + sa) * DH;
    const Tin *Vp = static_cast<const Tin *>(A.V) + ((size_t)lg * A.T + sa) * DH;
    const float om = A.omega ? A.omega[lg] : 1.0f;

    // Probe weights E[t][u] (Eq. app_probe_distortion), stored at E[t][u % 32].x
    // (u < 32) or .y (u >= 32).  When the score pass wrote them for every token
    // they are copied in with the slot (cp.async, 4 bytes each); otherwise
    // they are formed below from the raw keys.
    float *Ef = reinterpret_cast<float *>(&sm.E[0][0]);
    auto eidx = [](int t, int u) { return t * 2 * kNPP + 2 * (u & (kNPP - 1)) + (u >> 5); };
    if (A.Eg) {   // the same layout, n rows of 256 bytes: 16-byte copies
        const float *Eu = A.Eg + ((size_t)lg * A.Nc + (sa - A.cs)) * (2 * kNPP);
        for (int idx = tid; idx < n * (2 * kNPP / 4); idx += kNT) cp_async16(Ef + 4 * idx, Eu + 4 * idx, true);
        cp_async_commit();
    }
    // ---- load the slot ------------------------------------------------------
    // Every global load of a group is issued before any is used.  DH / 8
    // consecutive threads hold a token; they also form ||k_t||, which equals
    // ||k_circ_t|| (a rotation keeps the norm).
    {
        const bool own = tid < n;
        const double kapv = own ? A.kappa[sa + tid] : 0.0;
        const float rtv = own ? A.rtok[(size_t)lg * A.Nc + (sa - A.cs) + tid] : 0.f;
        constexpr int TPT = DH / 8, GRP = 4;
        const int iters = (n * DH + kNT * 8 - 1) / (kNT * 8);
        for (int i0 = 0; i0 < iters; i0 += GRP) {   // the same trip counts for every thread
            Raw8<Tin> kr[GRP], vr[GRP];
#pragma unroll
            for (int q = 0; q < GRP; q++) {
                const int e = (i0 + q) * kNT * 8 + tid * 8;
                if (i0 + q < iters && e < n * DH) {
                    kr[q].load(Kp + e);
                    vr[q].load(Vp + e);
                }
            }
#pragma unroll
            for (int q = 0; q < GRP; q++) {
                if (i0 + q >= iters) break;
                const int e = (i0 + q) * kNT * 8 + tid * 8;
                const bool in = e < n * DH;
                const int t = e / DH, i = e - t * DH;
                float ss = 0.f;
                if (in) {
                    float kx[8], vx[8];
                    kr[q].get(kx);
                    vr[q].get(vx);
#pragma unroll
                    for (int u = 0; u < 8; u++) {
                        sm.kc[t][i + u] = kx[u];
                        sm.vv[t][i + u] = vx[u];
                        ss = fmaf(kx[u], kx[u], ss);
                    }
                }
#pragma unroll
                for (int o = 1; o < TPT; o <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
                if (in && i == 0) sm.kn[t] = sqrtf(ss);
            }
        }
        for (int t = tid; t < n; t += kNT) {
            sm.kap[t] = okey(t == tid ? kapv : A.kappa[sa + t]);
            sm.Rt[t] = t == tid ? rtv : A.rtok[(size_t)lg * A.Nc + (sa - A.cs) + t];
        }
    }
    // probe registers: thread (pp, c) owns probes pp and pp + 32, elements
    // 4 c + 32 g + j; the 8 chunk lanes of a pair read 128 contiguous bytes
    const int c = lane / kPPW, pp = warp * kPPW + (lane & (kPPW - 1));
    float2 qa0[CH / 2], qa1[CH / 2];   // q of the two probes as element pairs
    float mu0 = 0.f, mu1 = 0.f, invZ0 = 0.f, invZ1 = 0.f;
#pragma unroll
    for (int h = 0; h < 2; h++) {
        const int u = pp + kNPP * h;
        float2 *qd = h ? qa1 : qa0;
        if (u < A.W) {
            const size_t row = ((size_t)l * A.Hq + g * A.gq + (u % A.gq)) * A.W + u;
            const Tin *qp = static_cast<const Tin *>(A.Q) + row * DH + 4 * c;
#pragma unroll
            for (int gi = 0; gi < NG; gi++) {
                float4 x = ld4(qp + 32 * gi);
                qd[2 * gi] = make_float2(x.x, x.y);
                qd[2 * gi + 1] = make_float2(x.z, x.w);
            }
            (h ? mu1 : mu0) = A.row_m[row];
            (h ? invZ1 : invZ0) = 1.0f / A.row_Z[row];
        } else {
#pragma unroll
            for (int q = 0; q < CH / 2; q++) qd[q] = make_float2(0.f, 0.f);
        }
    }
    __syncthreads();

    // ---- E[t][u] from the raw (post-RoPE) keys -------------------------------
    if (A.Eg) {
        cp_async_wait<0>();   // the copies above have landed (each thread its own)
    } else if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
        // Tensor cores: logits = Q_probes (64 x DH) . K_slot^T, one 16x8 tile
        // per (probe block, token block); warp w keeps probe block w % 4.
        constexpr int MT = 4, WSTEP = NWARPS / MT;
        const int gr = lane >> 2, c2 = 2 * (lane & 3);
        const int mt = warp % MT;
        const int u0 = mt * 16 + gr, u1 = u0 + 8;
        const __nv_bfloat16 *Qb = static_cast<const __nv_bfloat16 *>(A.Q);
        const size_t r0 = ((size_t)l * A.Hq + g * A.gq + u0 % A.gq) * A.W + u0;
        const size_t r1 = ((size_t)l * A.Hq + g * A.gq + u1 % A.gq) * A.W + u1;
        const bool ok0 = u0 < A.W, ok1 = u1 < A.W;
        uint32_t qa[DH / 16][4];
#pragma unroll
        for (int ks = 0; ks < DH / 16; ks++) {
            const __nv_bfloat16 *p0 = Qb + r0 * DH + ks * 16 + c2, *p1 = Qb + r1 * DH + ks * 16 + c2;
            qa[ks][0] = ok0 ? *reinterpret_cast<const uint32_t *>(p0) : 0u;
            qa[ks][1] = ok1 ? *reinterpret_cast<const uint32_t *>(p1) : 0u;
            qa[ks][2] = ok0 ? *reinterpret_cast<const uint32_t *>(p0 + 8) : 0u;
            qa[ks][3] = ok1 ? *reinterpret_cast<const uint32_t *>(p1 + 8) : 0u;
        }
        const float m0 = ok0 ? A.row_m[r0] : 0.f, m1 = ok1 ? A.row_m[r1] : 0.f;
        const int ntn = (n + 7) / 8;
        for (int nt = warp / MT; nt < ntn; nt += WSTEP) {
            float acc[4] = {0.f, 0.f, 0.f, 0.f};
            const float *kr = &sm.kc[nt * 8 + gr][c2];
#pragma unroll
            for (int ks = 0; ks < DH / 16; ks++) {
                const float2 x0 = *reinterpret_cast<const float2 *>(kr + ks * 16);
                const float2 x1 = *reinterpret_cast<const float2 *>(kr + ks * 16 + 8);
                mma_bf16(acc, qa[ks], pack_bf16x2(x0.x, x0.y), pack_bf16x2(x1.x, x1.y));
            }
            const int t0 = nt * 8 + c2;
            if (t0 < n) {
                Ef[eidx(t0, u0)] = ok0 ? expf(acc[0] * A.inv_sqrt_d - m0) : 0.f;
                Ef[eidx(t0, u1)] = ok1 ? expf(acc[2] * A.inv_sqrt_d - m1) : 0.f;
            }
            if (t0 + 1 < n) {
                Ef[eidx(t0 + 1, u0)] = ok0 ? expf(acc[1] * A.inv_sqrt_d - m0) : 0.f;
                Ef[eidx(t0 + 1, u1)] = ok1 ? expf(acc[3] * A.inv_sqrt_d - m1) : 0.f;
            }
        }
    } else {
        for (int t = 0; t < n; t++) {
            float2 x0 = make_float2(0.f, 0.f), x1 = make_float2(0.f, 0.f);
#pragma unroll
            for (int gi = 0; gi < NG; gi++) {
                const float4 kv = *reinterpret_cast<const float4 *>(&sm.kc[t][4 * c + 32 * gi]);
                const float2 ka = make_float2(kv.x, kv.y), kb = make_float2(kv.z, kv.w);
                x0 = ffma2(qa0[2 * gi], ka, x0); x0 = ffma2(qa0[2 * gi + 1], kb, x0);
                x1 = ffma2(qa1[2 * gi], ka, x1); x1 = ffma2(qa1[2 * gi + 1], kb, x1);
            }
            float y0 = x0.x + x0.y, y1 = x1.x + x1.y;
#pragma unroll
            for (int o = kPPW; o < 32; o <<= 1) {   // over the pair's chunk lanes
                y0 += __shfl_xor_sync(0xffffffffu, y0, o);
                y1 += __shfl_xor_sync(0xffffffffu, y1, o);
            }
            if (c == 0)
                sm.E[t][pp] = make_float2(pp < A.W ? expf(y0 * A.inv_sqrt_d - mu0) : 0.f,
                                          pp + kNPP < A.W ? expf(y1 * A.inv_sqrt_d - mu1) : 0.f);
        }
    }
    __syncthreads();
    // Non-finite probe weights or token values (NaN/Inf in K, Q or the row
    // statistics) make every decision of the unit meaningless: record the
    // unit as a single uncovered leaf with zero gain and flag the error, which
    // the host reports as GKV_ENONFINITE at the allocation's count sync.
    {
        bool bad = false;
        for (int e = tid; e < n * 2 * kNPP; e += kNT) bad |= !isfinite(Ef[e]);
        for (int t = tid; t < n; t += kNT) bad |= !isfinite(sm.Rt[t]);
        if (__syncthreads_or(bad)) {
            if constexpr (SUB) {   // the node stays a leaf; the unit is reported
                if (tid == 0) {
                    atomicOr(A.status, 8);
                    A.nd_nchild[gv_sub] = 0; A.nd_child0[gv_sub] = -1; A.nd_cost[gv_sub] = 0;
                    A.nd_U[gv_sub] = 0.f; A.nd_kappa[gv_sub] = 0.f;
                }
                return;
            }
            if (tid == 0) {
                atomicOr(A.status, 8);
                A.nd_a[nbase] = sa; A.nd_b[nbase] = sb; A.nd_R[nbase] = 0.f; A.nd_D[nbase] = 0.f;
                A.nd_parent[nbase] = (int32_t)(-2 - uid); A.nd_unit[nbase] = (int32_t)uid;
                A.nd_child0[nbase] = -1; A.nd_nchild[nbase] = 0; A.nd_U[nbase] = 0.f;
                A.nd_kappa[nbase] = 0.f; A.nd_sel[nbase] = 0;
                A.u_nnodes[uid] = 1; A.u_Uadd[uid] = 0.f; A.u_Ddrop[uid] = 0.f; A.u_sel[uid] = 0;
                A.u_pend[uid] = -1.f;
            }
            for (int k = tid; k < 2 * n; k += kNT) A.nd_cost[nbase + k] = 0;
            return;
        }
    }
    // Singleton floor (App. A.5 Stage I): the accepted positions of this slot
    // and their scores; a node holding one is extracted at the one of largest
    // score, and the floor's ops carry the largest key (they execute first).
    bool ufl = false;
    if (A.fl_acc) {
        bool any = false;
        for (int t = tid; t < n; t += kNT) {
            const size_t q = (size_t)lg * A.Nc + (sa - A.cs) + t;
            const bool ac = A.fl_acc[q] != 0;
            sm.Ff[t] = ac ? A.fl_f[q] : -INFINITY;
            any |= ac;
        }
        ufl = __syncthreads_or(any);
    }
    // ---- k_circ = RoPE^-1(k, t) ----------------------------------------------
    // batches of RB rotation-table loads are issued before any is used
    {
        constexpr int RB = 8;
        for (int e0 = tid; e0 < n * HALF; e0 += kNT * RB) {
            float2 cs[RB];
#pragma unroll
            for (int q = 0; q < RB; q++) {
                const int e = e0 + q * kNT;
                if (e < n * HALF) {
                    const int t = e / HALF, i = e - t * HALF;
                    cs[q] = A.rope[(size_t)(sa + t) * HALF + i];
                }
            }
#pragma unroll
            for (int q = 0; q < RB; q++) {
                const int e = e0 + q * kNT;
                if (e < n * HALF) {
                    const int t = e / HALF, i = e - t * HALF;
                    const float x = sm.kc[t][i], y = sm.kc[t][i + HALF];
                    sm.kc[t][i] = x * cs[q].x + y * cs[q].y;
                    sm.kc[t][i + HALF] = y * cs[q].x - x * cs[q].y;
                }
            }
        }
    }
    // ---- tree state: a fresh root, a subtree's root, or the unit's records so far
    if constexpr (SUB) {
        if (tid == 0) {
            NodeS &nd = sm.nodes[0];
            nd.a = 0; nd.b = (short)n; nd.parent = -1; nd.child0 = -1; nd.nchild = -1;
            nd.D = A.nd_D[gv_sub];
            const int32_t pg = A.nd_parent[gv_sub];   // a node of the long unit, already evaluated
            nd.kin = pg < 0 ? FLT_MAX : A.nd_kappa[pg];
            sm.nnodes = 1;
            sm.lvl[0][0] = 0;
            sm.nlvl[0] = 1;
            sm.pend = -1.f;
        }
    } else if (!A.resume) {
        if (warp == 0) {
            float r = 0.f;
            for (int t = lane; t < n; t += 32) r += sm.Rt[t];
            r = warp_sum(r);
            if (lane == 0) {
                NodeS &nd = sm.nodes[0];
                nd.a = 0; nd.b = (short)n; nd.parent = -1; nd.child0 = -1; nd.nchild = 0;
                nd.D = 0.f; nd.kin = 0.f;
                sm.rootR = r;
                sm.nnodes = 1;
                sm.lvl[0][0] = 0;
                sm.nlvl[0] = 1;
                sm.pend = -1.f;
                A.nd_a[nbase] = sa; A.nd_b[nbase] = sb; A.nd_R[nbase] = (float)r;
                A.nd_parent[nbase] = (int32_t)(-2 - uid);
                A.nd_unit[nbase] = (int32_t)uid;
            }
        }
    } else {
        const int nn = A.u_nnodes[uid];
        float *bnd_stage = &sm.redD[0][0];   // scratch until the first evaluation
        static_assert(sizeof(sm.redD) >= sizeof(float) * S::MAXNODES, "bound staging");
        for (int k = tid; k < nn; k += kNT) {
            const int64_t v = nbase + k;
            NodeS &nd = sm.nodes[k];
            nd.a = (short)(A.nd_a[v] - sa);
            nd.b = (short)(A.nd_b[v] - sa);
            int32_t pg = A.nd_parent[v];
            nd.parent = pg < 0 ? (short)-1 : (short)(pg - nbase);
            nd.child0 = (short)A.nd_child0[v];
            nd.nchild = A.nd_nchild[v];
            nd.D = A.nd_D[v];
            nd.kin = pg < 0 ? (ufl ? FLT_MAX : A.u_Uadd[uid]) : A.nd_kappa[pg];
            bnd_stage[k] = nd.nchild == -1 ? A.nd_U[v] : -1.f;   // key bound of a pending node
        }
        if (tid == 0) { sm.nnodes = nn; sm.nlvl[0] = 0; sm.pend = -1.f; }
        __syncthreads();
        if (tid == 0) {   // pending nodes that qualify, in creation order
            for (int k = 0; k < nn; k++) {
                if (sm.nodes[k].nchild != -1) continue;
                if (bnd_stage[k] >= A.tau) sm.lvl[0][sm.nlvl[0]++] = (short)k;
                else sm.pend = fmaxf(sm.pend, bnd_stage[k]);
            }
        }
    }
    __syncthreads();

    unsigned long long w_scan = 0, w_eval = 0, w_len = 0;   // work counters (lane 0 of each warp)

    // Prototypes of the batch's prefix (or suffix) candidates, warp per
    // candidate; reserved entries a node did not use are empty and skipped.
    auto prototypes = [&](bool suffix) {
        const int kb = suffix ? kNCD : 0, ke = suffix ? kNCD + sm.batch_suf : sm.batch_pre;
        for (int k = kb + warp; k < ke; k += NWARPS) {
            const int row = k - kb;
            const int ja = sm.cand[k].a, jb = sm.cand[k].b, nJ = jb - ja;
            if (nJ <= 0) continue;
            const int p = round_half_even_mid(sa + ja, sa + jb);   // absolute positions
            // lane owns the rotation pairs (i, i + d/2), i = PPL lane + j; the
            // rotation to p is loaded first so that its latency overlaps the sums
            constexpr int PPL = HALF / 32;
            const int i0 = lane * PPL;
            float2 rot[PPL];
#pragma unroll
            for (int j = 0; j < PPL; j++) rot[j] = A.rope[(size_t)p * HALF + i0 + j];
            // one pass over the tokens: sum k_circ, sum R v and sum v (the weights
            // R_t + beta need the mean R, so sum (R + beta) v = sum R v + beta sum v),
            // and the scalars sum R, sum ||k_circ|| (the same in every lane)
            float m0[PPL], m1[PPL], r0[PPL], r1[PPL], s0[PPL], s1[PPL];
            float rs = 0.f, ks = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) m0[j] = m1[j] = r0[j] = r1[j] = s0[j] = s1[j] = 0.f;
#pragma unroll 8
            for (int t = ja; t < jb; t++) {
                float k0[PPL], k1[PPL], x0[PPL], x1[PPL];
                ld_pairs<PPL>(&sm.kc[t][i0], k0);
                ld_pairs<PPL>(&sm.kc[t][i0 + HALF], k1);
                ld_pairs<PPL>(&sm.vv[t][i0], x0);
                ld_pairs<PPL>(&sm.vv[t][i0 + HALF], x1);
                const float rt = sm.Rt[t];
                rs += rt;
                ks += sm.kn[t];
#pragma unroll
                for (int j = 0; j < PPL; j++) {
                    m0[j] += k0[j];
                    m1[j] += k1[j];
                    r0[j] = fmaf(rt, x0[j], r0[j]);
                    r1[j] = fmaf(rt, x1[j], r1[j]);
                    s0[j] += x0[j];
                    s1[j] += x1[j];
                }
            }
            const float ninv = 1.0f / (float)nJ;
            const float beta = (float)A.base_frac * (rs * ninv);
            const float winv = 1.0f / ((rs + (float)nJ * beta) + A.eps);
            float mu2 = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) {
                const float a0 = m0[j] * ninv, a1 = m1[j] * ninv;
                mu2 = fmaf(a0, a0, fmaf(a1, a1, mu2));
                const float2 cs = rot[j];
                sm.ktil[row][i0 + j] = a0 * cs.x - a1 * cs.y;
                sm.ktil[row][i0 + j + HALF] = a0 * cs.y + a1 * cs.x;
                sm.vtil[row][i0 + j] = fmaf(beta, s0[j], r0[j]) * winv;
                sm.vtil[row][i0 + j + HALF] = fmaf(beta, s1[j], r1[j]) * winv;
            }
            mu2 = warp_sum(mu2);
            if (lane == 0) {
                const float coh = sqrtf(mu2) / (ks * ninv + A.eps);
                const float me = (float)nJ * coh * coh;
                sm.cand[k].meff = me < 1.0f ? 1.0f : (me > (float)nJ ? (float)nJ : me);
            }
        }
    };
    // D_u of candidate k (prototype row `row`) from the probe statistics Z, M
    // of its interval; per-warp partial sums of pi_u D_u and pi_u.
    const float inv_sqrt_d = A.inv_sqrt_d, lamZ = A.lamZ, lamM = A.lamM, epsf = A.eps;
    // D_u of candidate k (prototype row `row`) for the thread's two probes from
    // their running statistics Z, M; per-warp partial sums of pi_u D_u and pi_u.
    auto evaluate = [&](int k, int row, float Z0, float Z1, const float2 *M0, const float2 *M1) {
        float2 kt[CH / 2];
#pragma unroll
        for (int gi = 0; gi < NG; gi++) {
            const float4 x = *reinterpret_cast<const float4 *>(&sm.ktil[row][4 * c + 32 * gi]);
            kt[2 * gi] = make_float2(x.x, x.y);
            kt[2 * gi + 1] = make_float2(x.z, x.w);
        }
        float2 xa = make_float2(0.f, 0.f), xb = make_float2(0.f, 0.f);
#pragma unroll
        for (int q = 0; q < CH / 2; q++) {
            xa = ffma2(qa0[q], kt[q], xa);
            xb = ffma2(qa1[q], kt[q], xb);
        }
        float x0 = xa.x + xa.y, x1 = xb.x + xb.y;
#pragma unroll
        for (int o = kPPW; o < 32; o <<= 1) {   // over the pair's chunk lanes
            x0 += __shfl_xor_sync(0xffffffffu, x0, o);
            x1 += __shfl_xor_sync(0xffffffffu, x1, o);
        }
        const float me = sm.cand[k].meff;
        const float zt0 = me * expf(x0 * inv_sqrt_d - mu0), zt1 = me * expf(x1 * inv_sqrt_d - mu1);
        const float2 nz0 = make_float2(-zt0, -zt0), nz1 = make_float2(-zt1, -zt1);
        float2 r0 = make_float2(0.f, 0.f), r1 = r0, m0 = r0, m1 = r0;
#pragma unroll
        for (int gi = 0; gi < NG; gi++) {
            const float4 x = *reinterpret_cast<const float4 *>(&sm.vtil[row][4 * c + 32 * gi]);
            const float2 va = make_float2(x.x, x.y), vb = make_float2(x.z, x.w);
#pragma unroll
            for (int h = 0; h < 2; h++) {
                const int q = 2 * gi + h;
                const float2 vt = h ? vb : va;
                const float2 d0 = ffma2(nz0, vt, M0[q]), d1 = ffma2(nz1, vt, M1[q]);   // M - zt vtil
                r0 = ffma2(d0, d0, r0);
                r1 = ffma2(d1, d1, r1);
                m0 = ffma2(M0[q], M0[q], m0);
                m1 = ffma2(M1[q], M1[q], m1);
            }
        }
        float res0 = r0.x + r0.y, res1 = r1.x + r1.y, mm0 = m0.x + m0.y, mm1 = m1.x + m1.y;
#pragma unroll
        for (int o = kPPW; o < 32; o <<= 1) {
            res0 += __shfl_xor_sync(0xffffffffu, res0, o);
            res1 += __shfl_xor_sync(0xffffffffu, res1, o);
            mm0 += __shfl_xor_sync(0xffffffffu, mm0, o);
            mm1 += __shfl_xor_sync(0xffffffffu, mm1, o);
        }
        // D_u (Eq. app_probe_distortion), weighted by the probe's attention
        // mass; probes past W have E = 0 and invZ = 0, so they add nothing.
        // Fast division: at most 2 ulp, far below the distortion tolerance.
        const float dz0 = Z0 - zt0, dz1 = Z1 - zt1;
        const float D0 = lamZ * __fdividef(dz0 * dz0, fmaf(Z0, Z0, epsf)) + lamM * __fdividef(res0, mm0 + epsf);
        const float D1 = lamZ * __fdividef(dz1 * dz1, fmaf(Z1, Z1, epsf)) + lamM * __fdividef(res1, mm1 + epsf);
        const float p0 = Z0 * invZ0, p1 = Z1 * invZ1;
        float pd = fmaf(p0, D0, p1 * D1), pw = p0 + p1;
#pragma unroll
        for (int o = 1; o < kPPW; o <<= 1) {   // over the warp's probe pairs
            pd += __shfl_xor_sync(0xffffffffu, pd, o);
            pw += __shfl_xor_sync(0xffffffffu, pw, o);
        }
        if (lane == 0) { sm.redD[k][warp] = pd; sm.redP[k][warp] = pw; }
    };
    // Probe scan of one node in one direction (SUF: suffixes, descending),
    // evaluating each candidate when the running sums reach its far end.
    auto scan = [&](const BatchNode &B, auto SUF) {
        constexpr bool suffix = decltype(SUF)::value;
        const int a = sm.nodes[B.node].a, b = sm.nodes[B.node].b;
        int k = suffix ? B.suf_b : B.pre_b;
        const int ke = suffix ? B.suf_e : B.pre_e;
        if (k >= ke) return;
        float2 M0[CH / 2], M1[CH / 2];
        float Z0 = 0.f, Z1 = 0.f;
#pragma unroll
        for (int q = 0; q < CH / 2; q++) M0[q] = M1[q] = make_float2(0.f, 0.f);
        auto add = [&](int t) {
            const float2 e = sm.E[t][pp];
            const float2 e0 = make_float2(e.x, e.x), e1 = make_float2(e.y, e.y);
            Z0 += e.x;
            Z1 += e.y;
#pragma unroll
            for (int gi = 0; gi < NG; gi++) {
                const float4 x = *reinterpret_cast<const float4 *>(&sm.vv[t][4 * c + 32 * gi]);
                const float2 va = make_float2(x.x, x.y), vb = make_float2(x.z, x.w);
                M0[2 * gi] = ffma2(e0, va, M0[2 * gi]);
                M0[2 * gi + 1] = ffma2(e0, vb, M0[2 * gi + 1]);
                M1[2 * gi] = ffma2(e1, va, M1[2 * gi]);
                M1[2 * gi + 1] = ffma2(e1, vb, M1[2 * gi + 1]);
            }
        };
        int t = suffix ? b - 1 : a;   // next token to add
        for (; k < ke; k++) {
            if (suffix) {
                const int stop = sm.cand[k].a;   // candidates in descending start, all >= a
#pragma unroll 1
                for (; t >= stop; t--) add(t);
                evaluate(k, k - kNCD, Z0, Z1, M0, M1);
            } else {
                const int stop = sm.cand[k].b;   // candidates in ascending end, all <= b
#pragma unroll 1
                for (; t < stop; t++) add(t);
                evaluate(k, k, Z0, Z1, M0, M1);
            }
        }
    };

    int cur = 0;
    int levels_left = A.max_levels;
    while (sm.nlvl[cur] > 0) {
        const int nl = sm.nlvl[cur];
        if (levels_left == 0) {   // depth limit: the level's nodes stay pending
            if (tid == 0) {
                float pm = sm.pend;
                for (int k = 0; k < nl; k++) {
                    const int v = sm.lvl[cur][k];
                    A.nd_nchild[gidx(v)] = -1;
                    pm = fmaxf(pm, A.nd_U[gidx(v)]);   // the key bound written at its creation
                }
                sm.pend = pm;
            }
            break;
        }
        levels_left--;
        if (tid == 0) { sm.nlvl[cur ^ 1] = 0; sm.batch_next = 0; }
        __syncthreads();
        while (sm.batch_next < nl) {
            // ---- batch assignment (thread 0) --------------------------------
            if (tid == 0) {
                int nb = 0, upre = 0, usuf = 0, k = sm.batch_next;
                while (k < nl && nb < S::NB) {
                    const int v = sm.lvl[cur][k];
                    const int nv = sm.nodes[v].b - sm.nodes[v].a;
                    const bool root = v == 0 && fresh;
                    const int nc = (nv >= 3 && !(root && A.root_only)) ? min(A.k_cand + 1, nv - 1) + 1 : 0;
                    const int bp = nc + (root ? 1 : 0), bs = nc;
                    if (upre + bp > kNCD || usuf + bs > kNCD) break;
                    sm.bn[nb].node = v;
                    sm.bn[nb].pre_b = upre;
                    sm.bn[nb].suf_b = kNCD + usuf;
                    upre += bp;
                    usuf += bs;
                    sm.bn[nb].pre_r = upre;
                    sm.bn[nb].suf_r = kNCD + usuf;
                    nb++;
                    k++;
                }
                sm.batch_n = nb;
                sm.batch_next = k;
                sm.batch_pre = upre;
                sm.batch_suf = usuf;
            }
            __syncthreads();
            const int nb = sm.batch_n;
            // ---- phase A: cut candidates per node (warp per node) ------------
            for (int bi = warp; bi < nb; bi += NWARPS) {
                BatchNode &B = sm.bn[bi];
                const int v = B.node;
                const int a = sm.nodes[v].a, b = sm.nodes[v].b, nv = b - a;
                const bool ronly = v == 0 && fresh && A.root_only;   // only the node's own distortion
                // top-K by curvature over positions [a, b-2] (ties: lower t)
                unsigned sel[NMAX / 32];
                unsigned long long kmin = ~0ull, kmax = 0ull;
#pragma unroll
                for (int w = 0; w < NMAX / 32; w++) {
                    int t = a + w * 32 + lane;
                    bool in = !ronly && t <= b - 2;
                    bool s = false;
                    if (in) {
                        const unsigned long long kt = sm.kap[t];
                        kmin = min(kmin, kt);
                        kmax = max(kmax, kt);
                        int rank = 0;
                        for (int q = a; q <= b - 2; q++) {
                            const unsigned long long kq = sm.kap[q];
                            rank += (kq > kt) || (kq == kt && q < t);
                        }
                        s = rank < A.k_cand || t == a + nv / 2 - 1;   // + midpoint
                    }
                    sel[w] = __ballot_sync(0xffffffffu, s);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
                    kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
                }
                // salient token p* = argmax R_tok over [a, b) (ties: lower t)
                float rb = -INFINITY;
                int pb = 0x7fffffff;
                for (int t = a + lane; t < b; t += 32) {
                    float r = sm.Rt[t];
                    if (r > rb) { rb = r; pb = t; }
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    float r2 = __shfl_xor_sync(0xffffffffu, rb, o);
                    int p2 = __shfl_xor_sync(0xffffffffu, pb, o);
                    if (r2 > rb || (r2 == rb && p2 < pb)) { rb = r2; pb = p2; }
                }
                if (pb < a || pb >= b) pb = a;   // only reachable with non-finite values
                // a node holding an accepted floor position is extracted at the one
                // of largest floor score (ties: lower t)
                int forced = 0;
                if (ufl) {
                    float fb = -INFINITY;
                    int fpos = 0x7fffffff;
                    for (int t = a + lane; t < b; t += 32) {
                        const float fv = sm.Ff[t];
                        if (fv > fb) { fb = fv; fpos = t; }
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
                        const float f2 = __shfl_xor_sync(0xffffffffu, fb, o);
                        const int p2 = __shfl_xor_sync(0xffffffffu, fpos, o);
                        if (f2 > fb || (f2 == fb && p2 < fpos)) { fb = f2; fpos = p2; }
                    }
                    if (fb > -INFINITY) { pb = fpos; forced = 1; }
                }
                // Candidate lists, lane-parallel (ranks from ballots): cuts xi in
                // ascending order; prefixes [a, xi) (xi - a >= 2) and the
                // extraction's left side [a, p*) in ascending end, then the whole
                // node (fresh roots); suffixes [xi, b) (b - xi >= 2) and the right
                // side [p*+1, b) in descending start.  A side equal to a cut's
                // interval shares its candidate.
                const unsigned FULL = 0xffffffffu;
                const bool cands = nv >= 3 && !ronly;
                const int maxc = cands ? min(A.k_cand + 1, nv - 1) : 0;
                int ncut = 0;
#pragma unroll
                for (int w = 0; w < NMAX / 32; w++) {
                    const unsigned m = sel[w];
                    const int q = ncut + __popc(m & ((1u << lane) - 1u));
                    if (((m >> lane) & 1u) && q < maxc) B.cut[q] = (int8_t)(a + w * 32 + lane + 1);
                    ncut += __popc(m);
                }
                ncut = min(ncut, maxc);
                __syncwarp();
                const bool hq = lane < ncut;
                const int xi = hq ? B.cut[lane] : 0;
                const unsigned lt = (1u << lane) - 1u, gt = ~((2u << lane) - 1u);
                // prefixes
                const bool pv = hq && xi - a >= 2;
                const unsigned pm = __ballot_sync(FULL, pv);
                const unsigned pbm = __ballot_sync(FULL, hq && xi == pb);
                const bool el_cand = cands && pb - a >= 2;
                const bool el_sep = el_cand && pbm == 0u;
                const int pidx = pv ? B.pre_b + __popc(pm & lt) + (el_sep && pb < xi ? 1 : 0) : -1;
                const int eL_sep = B.pre_b + __popc(__ballot_sync(FULL, pv && xi < pb));
                const int eL_cut = __shfl_sync(FULL, pidx, pbm ? __ffs(pbm) - 1 : 0);
                if (hq) B.pidx[lane] = (int8_t)pidx;
                if (pv) sm.cand[pidx] = {a, xi, 0.f};
                // suffixes
                const int er = pb + 1;
                const bool sv = hq && b - xi >= 2;
                const unsigned smk = __ballot_sync(FULL, sv);
                const unsigned erm = __ballot_sync(FULL, hq && xi == er);
                const bool er_cand = cands && b - er >= 2;
                const bool er_sep = er_cand && erm == 0u;
                const int sidx = sv ? B.suf_b + __popc(smk & gt) + (er_sep && er > xi ? 1 : 0) : -1;
                const int eR_sep = B.suf_b + __popc(__ballot_sync(FULL, sv && xi > er));
                const int eR_cut = __shfl_sync(FULL, sidx, erm ? __ffs(erm) - 1 : 0);
                if (hq) B.sidx[lane] = (int8_t)sidx;
                if (sv) sm.cand[sidx] = {xi, b, 0.f};
                // work counters: tokens swept, candidates evaluated, their lengths
                int len = (pv ? xi - a : 0) + (sv ? b - xi : 0);
                int pe = pv ? xi : a, ss = sv ? xi : b;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    len += __shfl_xor_sync(FULL, len, o);
                    pe = max(pe, __shfl_xor_sync(FULL, pe, o));
                    ss = min(ss, __shfl_xor_sync(FULL, ss, o));
                }
                if (lane == 0) {
                    const double kmn = nv >= 2 ? okey_inv(kmin) : 0.0, kmx = nv >= 2 ? okey_inv(kmax) : 0.0;
                    B.kmin = kmn;
                    B.krange = kmx > kmn ? 1.0f / (float)(kmx - kmn) : 0.f;
                    B.pstar = pb;
                    B.forced = forced;
                    B.ncut = ncut;
                    B.eL = el_sep ? eL_sep : (el_cand ? eL_cut : -1);
                    if (el_sep) sm.cand[eL_sep] = {a, pb, 0.f};
                    int k = B.pre_b + __popc(pm) + (el_sep ? 1 : 0);
                    const bool whole = v == 0 && fresh;
                    B.whole = -1;
                    if (whole) { sm.cand[k] = {a, b, 0.f}; B.whole = k++; }
                    B.pre_e = k;
                    B.eR = er_sep ? eR_sep : (er_cand ? eR_cut : -1);
                    if (er_sep) sm.cand[eR_sep] = {er, b, 0.f};
                    B.suf_e = B.suf_b + __popc(smk) + (er_sep ? 1 : 0);
                    for (int q = B.pre_e; q < B.pre_r; q++) sm.cand[q].a = sm.cand[q].b = 0;
                    for (int q = B.suf_e; q < B.suf_r; q++) sm.cand[q].a = sm.cand[q].b = 0;
                    if (el_sep) { pe = max(pe, pb); len += pb - a; }
                    if (er_sep) { ss = min(ss, er); len += b - er; }
                    if (whole) { pe = b; len += b - a; }
                    w_scan += (pe - a) + (b - ss);
                    w_eval += (B.pre_e - B.pre_b) + (B.suf_e - B.suf_b);
                    w_len += len;
                }
            }
            __syncthreads();
            // ---- phases B/C: prefixes, then suffixes ---------------------------
            prototypes(false);
            __syncthreads();
            for (int bi = 0; bi < nb; bi++) scan(sm.bn[bi], std::false_type());
            __syncthreads();
            prototypes(true);
            __syncthreads();
            for (int bi = 0; bi < nb; bi++) scan(sm.bn[bi], std::true_type());
            __syncthreads();
            // ---- phase D1: candidate sums and decisions (warp per node) -------------
            for (int bi = warp; bi < nb; bi += NWARPS) {
                BatchNode &B = sm.bn[bi];
                NodeS &nd = sm.nodes[B.node];
                const int a = nd.a, b = nd.b, nv = b - a;
                // D and drop mass of this node's candidates: mean over the W probes
                // of the per-warp partial sums
                const float invW = 1.0f / A.W;
                for (int k = lane; k < 2 * kNCD; k += 32) {
                    const bool mine = k < kNCD ? (k >= B.pre_b && k < B.pre_e) : (k >= B.suf_b && k < B.suf_e);
                    if (!mine) continue;
                    float d = 0.f, pw = 0.f;
#pragma unroll
                    for (int w = 0; w < NWARPS; w++) { d += sm.redD[k][w]; pw += sm.redP[k][w]; }
                    sm.candD[k] = d * invW;
                    sm.candP[k] = pw * invW;
                }
                __syncwarp();
                if (B.whole >= 0 && lane == 0) {   // root: D, Ddrop, Add gain (Eq. app_operation_gains)
                    const float Pd = sm.candP[B.whole];
                    const float D = nv >= 2 ? sm.candD[B.whole] : 0.f;
                    nd.D = D;
                    float gain = om * sm.rootR * (Pd - D);
                    if (gain < 0.f) gain = 0.f;
                    nd.kin = ufl ? FLT_MAX : gain;   // a floor slot's Add is a floor op
                    A.u_Uadd[uid] = gain;
                    A.u_Ddrop[uid] = Pd;
                    A.nd_D[gidx(0)] = D;
                }
                __syncwarp();
                if (A.root_only && B.whole >= 0 && nv >= 2) {   // its split is decided later
                    if (lane == 0) B.nchild = -1;
                    continue;
                }
                if (nv < 3) {
                    if (lane == 0) {
                        B.nchild = 0;
                        if (nv == 2) {
                            B.nchild = 2;
                            B.ca[0] = a; B.cb[0] = a + 1; B.cD[0] = 0.f;
                            B.ca[1] = a + 1; B.cb[1] = b; B.cD[1] = 0.f;
                        }
                    }
                    continue;
                }
                const float DI = nd.D;
                // binary cut: lane q evaluates cut q; max G_bin, ties -> smallest xi
                float best = -INFINITY;
                int bq = 0x7fffffff;
                if (lane < B.ncut) {
                    const int xi = B.cut[lane];
                    const float DL = B.pidx[lane] >= 0 ? sm.candD[B.pidx[lane]] : 0.f;
                    const float DR = B.sidx[lane] >= 0 ? sm.candD[B.sidx[lane]] : 0.f;
                    // normalised curvature: the difference is taken in fp64 (the
                    // curvatures may be close), the rest in fp32
                    const float kh = (float)(okey_inv(sm.kap[xi - 1]) - B.kmin) * B.krange;
                    best = ((DI - DL) - DR) + A.lam_kappa * kh;
                    bq = lane;
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    float ov = __shfl_xor_sync(0xffffffffu, best, o);
                    int oq = __shfl_xor_sync(0xffffffffu, bq, o);
                    if (ov > best || (ov == best && oq < bq)) { best = ov; bq = oq; }
                }
                if (lane) continue;
                int bxi = -1;
                float bL = 0.f, bR = 0.f;
                if (bq < B.ncut && best > -INFINITY) {
                    bxi = B.cut[bq];
                    bL = B.pidx[bq] >= 0 ? sm.candD[B.pidx[bq]] : 0.f;
                    bR = B.sidx[bq] >= 0 ? sm.candD[B.sidx[bq]] : 0.f;
                }
                // extraction at p*
                const int ps = B.pstar;
                int ea[3], eb[3], ne = 0;
                float eD[3];
                if (ps > a) { ea[ne] = a; eb[ne] = ps; eD[ne] = ps - a >= 2 ? sm.candD[B.eL] : 0.f; ne++; }
                ea[ne] = ps; eb[ne] = ps + 1; eD[ne] = 0.f; ne++;
                if (ps + 1 < b) { ea[ne] = ps + 1; eb[ne] = b; eD[ne] = b - ps - 1 >= 2 ? sm.candD[B.eR] : 0.f; ne++; }
                float gext = DI;
                for (int q = 0; q < ne; q++) gext -= eD[q];
                if (bxi < 0) {   // only reachable with non-finite gains
                    bxi = B.cut[0];
                    bL = B.pidx[0] >= 0 ? sm.candD[B.pidx[0]] : 0.f;
                    bR = B.sidx[0] >= 0 ? sm.candD[B.sidx[0]] : 0.f;
                }
                const float rho_ext = ne == 3 ? 0.5f * gext : gext;   // G_ext / (|children| - 1), exact
                if (B.forced || rho_ext > best) {
                    B.nchild = ne;
                    for (int q = 0; q < ne; q++) { B.ca[q] = ea[q]; B.cb[q] = eb[q]; B.cD[q] = eD[q]; }
                } else {
                    B.nchild = 2;
                    B.ca[0] = a; B.cb[0] = bxi; B.cD[0] = bL;
                    B.ca[1] = bxi; B.cb[1] = b; B.cD[1] = bR;
                }
            }
            __syncthreads();
            // ---- phase D2: numbering, children, gains, keys (warp per node) --------
            // Child indices are deterministic: the batch's nodes in order, after the
            // nodes created before this batch.
            for (int bi = warp; bi < nb; bi += NWARPS) {
                const BatchNode &B = sm.bn[bi];
                NodeS &nd = sm.nodes[B.node];
                const int64_t gv = gidx(B.node);
                int before = lane < bi ? max(sm.bn[lane].nchild, 0) : 0;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) before += __shfl_xor_sync(0xffffffffu, before, o);
                const int nch = B.nchild;
                if (nch < 0) {   // pending root: its split key is at most min(U_add, omega R D)
                    if (lane == 0) {
                        const float bnd = B.forced ? FLT_MAX : fminf(nd.kin, key_bound(om * sm.rootR * nd.D));
                        nd.nchild = -1; nd.child0 = -1;
                        A.nd_child0[gv] = -1; A.nd_nchild[gv] = -1; A.nd_cost[gv] = 0;
                        A.nd_U[gv] = bnd; A.nd_kappa[gv] = 0.f; A.nd_sel[gv] = 0;
                        atomicMax(reinterpret_cast<int *>(&sm.pend), __float_as_int(bnd));
                    }
                    continue;
                }
                const int child0 = nch ? sm.nnodes + before : -1;
                if (nch == 0) {
                    if (lane == 0) {
                        nd.nchild = 0; nd.child0 = -1;
                        A.nd_child0[gv] = -1; A.nd_nchild[gv] = 0; A.nd_cost[gv] = 0;
                        A.nd_U[gv] = 0.f; A.nd_kappa[gv] = 0.f; A.nd_sel[gv] = 0;
                    }
                    continue;
                }
                float rch[3] = {0.f, 0.f, 0.f};
                for (int q = 0; q < nch; q++) {
                    float r = 0.f;
                    for (int t = B.ca[q] + lane; t < B.cb[q]; t += 32) r += sm.Rt[t];
                    rch[q] = warp_sum(r);
                }
                const float rnode = (rch[0] + rch[1]) + rch[2];   // R of the node = sum over its children
                const float dsum = (B.cD[0] + B.cD[1]) + (nch == 3 ? B.cD[2] : 0.f);
                const int cost = nch - 1;
                float gain = om * rnode * (nd.D - dsum);
                if (gain < 0.f) gain = 0.f;
                const float U = cost == 2 ? 0.5f * gain : gain;
                const float kap = B.forced ? FLT_MAX : fminf(U, nd.kin);
                if (lane == 0) {
                    nd.nchild = (signed char)nch;
                    nd.child0 = (short)child0;
                    A.nd_child0[gv] = (int32_t)(gidx(child0) - nbase); A.nd_nchild[gv] = (int8_t)nch;
                    A.nd_cost[gv] = (int8_t)cost; A.nd_U[gv] = U; A.nd_kappa[gv] = kap;
                    A.nd_sel[gv] = 0;
                    A.ops[atomicAdd(A.n_ops, 1u)] = make_uint2(__float_as_uint(kap), ((uint32_t)gv << 1) | (uint32_t)(cost - 1));
                }
                if (lane < nch) {   // lane q writes child q
                    const int q = lane, ci = child0 + q;
                    const float rq = q == 0 ? rch[0] : (q == 1 ? rch[1] : rch[2]);
                    NodeS &ch = sm.nodes[ci];
                    ch.a = (short)B.ca[q]; ch.b = (short)B.cb[q]; ch.parent = (short)B.node;
                    ch.child0 = -1; ch.nchild = 0; ch.D = B.cD[q]; ch.kin = kap;
                    const int64_t gc = gidx(ci);
                    A.nd_a[gc] = sa + B.ca[q]; A.nd_b[gc] = sa + B.cb[q];
                    A.nd_parent[gc] = (int32_t)gv; A.nd_unit[gc] = (int32_t)uid;
                    A.nd_D[gc] = B.cD[q]; A.nd_R[gc] = (float)rq;
                    A.nd_child0[gc] = -1; A.nd_nchild[gc] = 0; A.nd_cost[gc] = 0;
                    // until the child is evaluated, nd_U holds the bound of its split key
                    // (the largest key when it holds a floor position: a floor op)
                    bool chf = false;
                    if (ufl)
                        for (int t = B.ca[q]; t < B.cb[q] && !chf; t++) chf = sm.Ff[t] > -INFINITY;
                    const float cbnd = B.cb[q] - B.ca[q] >= 2 ? (chf ? FLT_MAX : fminf(kap, key_bound(om * rq * B.cD[q]))) : 0.f;
                    A.nd_U[gc] = cbnd;
                    A.nd_kappa[gc] = 0.f; A.nd_sel[gc] = 0;
                    if (B.cb[q] - B.ca[q] >= 2) {
                        if (cbnd >= A.tau) {   // evaluated at the next level of this launch
                            const int pos = atomicAdd(&sm.nlvl[cur ^ 1], 1);
                            sm.lvl[cur ^ 1][pos] = (short)ci;
                        } else {   // its key cannot reach this pass's threshold: it stays pending
                            ch.nchild = -1;
                            A.nd_nchild[gc] = -1;
                            atomicMax(reinterpret_cast<int *>(&sm.pend), __float_as_int(cbnd));
                        }
                    }
                }
            }
            __syncthreads();
            if (tid == 0) {   // nodes created by this batch (read by the next batch's D2)
                int total = 0;
                for (int bi = 0; bi < nb; bi++) total += max(sm.bn[bi].nchild, 0);
                sm.nnodes += total;
            }
            __syncthreads();
        }
        // keep the next level in creation order (atomic appends may permute it)
        if (tid == 0) {
            int nx = cur ^ 1, m = sm.nlvl[nx];
            for (int x = 1; x < m; x++) {
                short v = sm.lvl[nx][x];
                int y = x - 1;
                while (y >= 0 && sm.lvl[nx][y] > v) { sm.lvl[nx][y + 1] = sm.lvl[nx][y]; y--; }
                sm.lvl[nx][y + 1] = v;
            }
        }
        __syncthreads();
        cur ^= 1;
    }
    if (lane == 0) { sm.wcnt[warp][0] = w_scan; sm.wcnt[warp][1] = w_eval; sm.wcnt[warp][2] = w_len; }
    __syncthreads();
    if (tid == 0) {
        if constexpr (!SUB) {   // a subtree stays inside its reserved slots; what it left pending is never needed
            A.u_nnodes[uid] = sm.nnodes;
            A.u_pend[uid] = sm.pend;
        }
        if (fresh) A.u_sel[uid] = 0;
        unsigned long long tot[3] = {0, 0, 0};
        for (int w = 0; w < NWARPS; w++)
            for (int q = 0; q < 3; q++) tot[q] += sm.wcnt[w][q];
        atomicAdd(&A.work[0], tot[0]);
        atomicAdd(&A.work[1], tot[1]);
        atomicAdd(&A.work[2], tot[2]);
        atomicAdd(&A.work[3], 1ull);
    }
    // unused node slots of the unit carry cost 0 (no op)
    if (fresh)
        for (int k = sm.nnodes + tid; k < 2 * n; k += kNT) A.nd_cost[nbase + k] = 0;
}

template <int DH, typename Tin, int NMAX, bool SUB = false>
cudaError_t launch_t(Ctx &c, BuildArgs &A, unsigned grid, cudaStream_t s) {
    using S = Smem<DH, Tin, NMAX>;
    static_assert(sizeof(S) <= 227 * 1024, "unit kernel shared memory above the per-CTA limit");
    if (grid == 0) return cudaSuccess;
    size_t sm = sizeof(S);
    cudaError_t e = cudaFuncSetAttribute(unit_build_kernel<DH, Tin, NMAX, SUB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    unit_build_kernel<DH, Tin, NMAX, SUB><<<grid, kNT, sm, s>>>(A);
    c.launches += 1;
    return cudaGetLastError();
}

template <typename Tin, int NMAX, bool SUB = false>
cudaError_t launch_dt(Ctx &c, BuildArgs &A, unsigned grid, cudaStream_t s) {
    return c.p.d == 128 ? launch_t<128, Tin, NMAX, SUB>(c, A, grid, s) : launch_t<64, Tin, NMAX, SUB>(c, A, grid, s);
}

}  // namespace

cudaError_t launch_unit_build(Ctx &c, const void *K, const void *V, const void *Q,
                              const float *omega, const int32_t *slots, int J, int resume,
                              int root_only, int max_levels, float tau, const int32_t *list_short, int n_short,
                              const int32_t *list_long, int n_long, cudaStream_t s, int lg0, int nlg) {
    const gkv_params &p = c.p;
    BuildArgs A;
    A.K = K; A.V = V; A.Q = Q;
    A.slots = slots; A.rope = c.w.rope; A.kappa = c.w.kappa;
    A.rtok = c.w.rtok; A.row_m = c.w.row_m; A.row_Z = c.w.row_Z; A.omega = omega;
    A.Eg = use_tc(c) ? c.w.Eg : nullptr;
    A.fl_acc = c.p.alpha_floor > 0.0 ? c.w.fl_acc : nullptr;
    A.fl_f = c.w.fl_f;   // written by the tensor-core pass B
    A.L = p.L; A.G = p.G; A.Hq = p.Hq; A.T = p.T; A.d = p.d; A.W = p.W; A.gq = p.Hq / p.G;
    A.cs = p.ctx_start; A.Nc = c.Nc; A.J = J; A.k_cand = p.k_cand;
    A.inv_sqrt_d = (float)(1.0 / sqrt((double)p.d));
    A.lamZ = (float)p.lambda_Z; A.lamM = (float)p.lambda_M; A.eps = (float)p.eps;
    A.lam_kappa = p.lambda_kappa; A.base_frac = p.base_frac;
    A.resume = resume; A.subtree = 0; A.root_only = root_only; A.max_levels = max_levels; A.tau = tau;
    A.nd_a = c.w.nd_a; A.nd_b = c.w.nd_b; A.nd_child0 = c.w.nd_child0;
    A.nd_parent = c.w.nd_parent; A.nd_unit = c.w.nd_unit;
    A.nd_nchild = c.w.nd_nchild; A.nd_cost = c.w.nd_cost;
    A.ops = c.w.ops; A.n_ops = c.w.n_ops;
    A.nd_D = c.w.nd_D; A.nd_R = c.w.nd_R; A.nd_U = c.w.nd_U; A.nd_kappa = c.w.nd_kappa;
    A.nd_sel = c.w.nd_sel;
    A.u_nnodes = c.w.u_nnodes; A.u_Uadd = c.w.u_Uadd; A.u_Ddrop = c.w.u_Ddrop; A.u_sel = c.w.u_sel;
    A.u_pend = c.w.u_pend;
    A.status = c.w.dev_int + 1;
    A.work = c.w.work;
    if (nlg < 0) nlg = p.L * p.G - lg0;
    A.lg0 = lg0;
    A.nlg = nlg;
    const unsigned LG = (unsigned)nlg;
    const bool bf = p.dtype == GKV_BF16;
    // short slots (<= 64 tokens) on the two-CTA-per-SM instance, the rest on the 128-token one
    A.list = list_short;
    unsigned g1 = resume ? (unsigned)n_short : (unsigned)n_short * LG;
    cudaError_t e = bf ? launch_dt<__nv_bfloat16, 64>(c, A, g1, s) : launch_dt<float, 64>(c, A, g1, s);
    if (e != cudaSuccess) return e;
    A.list = list_long;
    unsigned g2 = resume ? (unsigned)n_long : (unsigned)n_long * LG;
    return bf ? launch_dt<__nv_bfloat16, kMaxUnit>(c, A, g2, s) : launch_dt<float, kMaxUnit>(c, A, g2, s);
}

cudaError_t launch_unit_subtrees(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                                 const int32_t *slots, int J, const int32_t *list_short, int n_short,
                                 const int32_t *list_long, int n_long, float tau_prune, cudaStream_t s) {
    if (n_short + n_long == 0) return cudaSuccess;
    cudaError_t e;
    const gkv_params &p = c.p;
    BuildArgs A;
    A.K = K; A.V = V; A.Q = Q;
    A.slots = slots; A.rope = c.w.rope; A.kappa = c.w.kappa;
    A.rtok = c.w.rtok; A.row_m = c.w.row_m; A.row_Z = c.w.row_Z; A.omega = omega;
    A.Eg = use_tc(c) ? c.w.Eg : nullptr;
    A.fl_acc = p.alpha_floor > 0.0 ? c.w.fl_acc : nullptr;
    A.fl_f = c.w.fl_f;
    A.L = p.L; A.G = p.G; A.Hq = p.Hq; A.T = p.T; A.d = p.d; A.W = p.W; A.gq = p.Hq / p.G;
    A.cs = p.ctx_start; A.Nc = c.Nc; A.J = J; A.k_cand = p.k_cand;
    A.inv_sqrt_d = (float)(1.0 / sqrt((double)p.d));
    A.lamZ = (float)p.lambda_Z; A.lamM = (float)p.lambda_M; A.eps = (float)p.eps;
    A.lam_kappa = p.lambda_kappa; A.base_frac = p.base_frac;
    A.resume = 0; A.subtree = 1; A.root_only = 0; A.max_levels = 4 * kMaxUnit; A.tau = tau_prune;
    A.nd_a = c.w.nd_a; A.nd_b = c.w.nd_b; A.nd_child0 = c.w.nd_child0;
    A.nd_parent = c.w.nd_parent; A.nd_unit = c.w.nd_unit;
    A.nd_nchild = c.w.nd_nchild; A.nd_cost = c.w.nd_cost;
    A.ops = c.w.ops; A.n_ops = c.w.n_ops;
    A.nd_D = c.w.nd_D; A.nd_R = c.w.nd_R; A.nd_U = c.w.nd_U; A.nd_kappa = c.w.nd_kappa;
    A.nd_sel = c.w.nd_sel;
    A.u_nnodes = c.w.u_nnodes; A.u_Uadd = c.w.u_Uadd; A.u_Ddrop = c.w.u_Ddrop; A.u_sel = c.w.u_sel;
    A.u_pend = c.w.u_pend;
    A.status = c.w.dev_int + 1;
    A.work = c.w.work;
    A.lg0 = 0;
    A.nlg = p.L * p.G;
    const bool bf = p.dtype == GKV_BF16;
    A.list = list_short;
    e = bf ? launch_dt<__nv_bfloat16, 64, true>(c, A, (unsigned)n_short, s)
           : launch_dt<float, 64, true>(c, A, (unsigned)n_short, s);
    if (e != cudaSuccess) return e;
    A.list = list_long;
    return bf ? launch_dt<__nv_bfloat16, kMaxUnit, true>(c, A, (unsigned)n_long, s)
              : launch_dt<float, kMaxUnit, true>(c, A, (unsigned)n_long, s);
}

}  // namespace gkv
