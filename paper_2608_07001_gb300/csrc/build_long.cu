// build_long.cu -- the prototype trees of units whose slot is longer than the
// 128 tokens the unit kernel (build.cu) keeps in shared memory: supplied
// partitions may hold slots of thousands of tokens (App. A.2 atomic units are
// whatever slots the partition gives; the trees still recurse to single-token
// leaves, App. A.3 "Recursive refinement rule").
//
// The arithmetic is the unit kernel's, node by node: for a node I = [a, b) the
// binary cuts X_v (top-K positions by curvature in [a, b-2], cut xi = t + 1,
// plus the midpoint a + floor(n/2); App. B.4 Eq. app_tree_split_candidates),
// the salient-token extraction at p* = argmax R_tok (or the singleton-floor
// position of largest score, forced), candidate intervals that are prefixes
// [a, xi) and suffixes [xi, b) of I, RoPE-consistent prototypes (Eqs.
// app_rope_prototype, app_value_prototype, app_effective_multiplicity), the
// probe statistics Z_u, M_u of every candidate from one forward and one
// backward scan over the node (Eq. app_original_attention_stats), D_u and the
// mass-weighted D (Eqs. app_probe_distortion, app_node_and_drop_distortion),
// the refinement decision (Eqs. app_binary_split .. app_split_choice), gains,
// costs, utilities clamped at 0 and bottleneck keys (Eqs.
// app_operation_gains .. app_unit_utility), with the same node records, op
// list and pending-node key bounds, so the allocation, the pruning passes and
// the gather treat both kinds of unit alike.
//
// What differs is the work split.  The tree of a long unit is built one level
// per launch sequence, across CTAs:
//   long_collect  (CTA per listed unit) the nodes to evaluate -- a fresh root,
//                 or the pending nodes whose key bound reaches tau -- as one
//                 contiguous, ordered block of work items per unit;
//   long_eval     (CTA per work item, grid-stride) one node: cut candidates,
//                 per-segment sums between the candidate boundaries (at most
//                 20 segments; each candidate's prototype sums are the sum of
//                 its segments), the probe scans reading K, V and the token
//                 values from global memory, the decision;
//   long_commit   (warp per unit) children numbered in work-item order after
//                 the unit's existing nodes (deterministic), records, Split ops,
//                 pending bounds.
// The probe scans fold their fp32 running sums every 32 tokens (and at every
// candidate end) into a second fp32 sum, so that sums over thousands of
// tokens keep the rounding of short ones.
#include "gkv_internal.cuh"

#include <algorithm>
#include <cfloat>

#include <type_traits>

namespace gkv {
namespace {

constexpr int kLT = 256;          // threads per CTA
constexpr int kLPP = 32;          // probe pairs: thread handles probes p and p + 32 (W <= 64)
constexpr int kLCL = 8;           // threads per probe pair (4-element groups, interleaved)
constexpr int kLPPW = 32 / kLCL;  // probe pairs per warp
constexpr int kLNW = kLT / 32;    // warps
constexpr int kLNCD = 20;         // candidate rows per direction (17 cuts + p* side + whole node)
constexpr int kLMaxCut = 18;      // K + midpoint, K <= 16 (+1 spare)
constexpr int kLMaxSeg = 24;      // segments between the boundaries a, b, the cuts, p*, p* + 1
constexpr int kLFold = 32;        // tokens per fp32 partial sum of a scan
constexpr int kLChunk = 32;       // tokens per staged chunk of a scan

struct LongRes {
    int nch;               // -1: pending (root only), 0: leaf (non-finite inputs), 2 or 3
    int ca[3], cb[3];      // children, absolute positions
    float cD[3], rch[3];   // their distortion and value
    float bnd[3];          // key bound of a child left pending (n >= 2)
    float U, kap;          // the node's split utility and bottleneck key
    float bound;           // pending root: the bound of its split key
};

struct LongArgs {
    const void *K, *V, *Q;
    const int32_t *slots;
    const float2 *rope;
    const double *kappa;
    const float *rtok, *row_m, *row_Z, *omega;
    const float2 *Eg;              // nullable: [L G][N_c][32] probe weights (u, u + 32) of every token
    const uint8_t *fl_acc;         // nullable: [L G][N_c] accepted singleton-floor positions
    const float *fl_f;             //           and their floor scores
    int L, G, Hq, T, d, W, gq, cs, Nc, J, k_cand;
    float inv_sqrt_d, lamZ, lamM, eps, lam_kappa, base_frac;
    int fresh;                     // 1: the roots of the listed slots; 0: pending nodes of listed units
    int root_only;                 // fresh: only the root's own distortion (its split stays pending)
    float tau;                     // resume: evaluate pending nodes whose key bound >= tau
    const int32_t *list;           // fresh: slot indices; resume: unit ids
    int n_list, lg0, nlg;          // fresh units: slot list x (l, g) in [lg0, lg0 + nlg)
    // work items of the level
    int64_t *it_gv, *it_uid;
    float *it_kin;                 // bottleneck key of the op that created the node
    uint8_t *it_ufl;               // the node's unit holds a singleton-floor position
    LongRes *res;
    int32_t *u_start, *u_cnt;      // per listed unit: its block of work items
    unsigned int *n_items;         // [3]: work items, small subtrees (<= kShortUnit, <= kMaxUnit tokens)
    unsigned int *it_next;         // the next work item to take (zero at the level's start)
    int32_t *sub;                  // [2][cap_items] small subtrees' roots (global node indices)
    int64_t cap_items;
    // node records and unit arrays (build.cu's layout)
    int32_t *nd_a, *nd_b, *nd_child0, *nd_parent, *nd_unit;
    int8_t *nd_nchild, *nd_cost;
    float *nd_D, *nd_R, *nd_U, *nd_kappa;
    uint8_t *nd_sel;
    uint2 *ops;
    unsigned int *n_ops;
    int32_t *u_nnodes;
    float *u_Uadd, *u_Ddrop, *u_pend;
    uint8_t *u_sel;
    int *status;
    unsigned long long *work;
};

// Upper bound of a split's utility (see build.cu: U <= omega R D, rounded up).
__device__ __forceinline__ float lkey_bound(float x) { return x + fabsf(x) * 1e-5f; }

__device__ __forceinline__ unsigned long long lokey(double x) {
    unsigned long long u = (unsigned long long)__double_as_longlong(x);
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
__device__ __forceinline__ double lokey_inv(unsigned long long k) {
    unsigned long long u = (k >> 63) ? (k & 0x7fffffffffffffffull) : ~k;
    return __longlong_as_double((long long)u);
}

__device__ __forceinline__ int lround_half_even_mid(int a, int b) {
    int s = a + b - 1;
    if ((s & 1) == 0) return s >> 1;
    int lo = (s - 1) >> 1;
    return (lo & 1) == 0 ? lo : lo + 1;
}

__device__ __forceinline__ float4 lld4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 lld4(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
}
template <int N>
__device__ __forceinline__ void lld_pairs(const float *p, float v[N]) {
#pragma unroll
    for (int j = 0; j < N; j++) v[j] = p[j];
}
template <int N>
__device__ __forceinline__ void lld_pairs(const __nv_bfloat16 *p, float v[N]) {
#pragma unroll
    for (int j = 0; j < N; j++) v[j] = __bfloat162float(p[j]);
}

// Block-wide best (key descending, position ascending); pos = INT_MAX: none.
// Every thread returns the winner.  scratch: kLNW keys and positions.
__device__ __forceinline__ void block_best(unsigned long long &key, int &pos, unsigned long long *sk, int *sp) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long k2 = __shfl_xor_sync(0xffffffffu, key, o);
        const int p2 = __shfl_xor_sync(0xffffffffu, pos, o);
        if (p2 != INT_MAX && (pos == INT_MAX || k2 > key || (k2 == key && p2 < pos))) { key = k2; pos = p2; }
    }
    if (lane == 0) { sk[warp] = key; sp[warp] = pos; }
    __syncthreads();
    key = sk[0];
    pos = sp[0];
    for (int w = 1; w < kLNW; w++) {
        const unsigned long long k2 = sk[w];
        const int p2 = sp[w];
        if (p2 != INT_MAX && (pos == INT_MAX || k2 > key || (k2 == key && p2 < pos))) { key = k2; pos = p2; }
    }
    __syncthreads();
}

// Block-wide sum of a float (fixed order: lanes, then warps ascending).
__device__ __forceinline__ float block_sum(float v, float *sf) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    if (lane == 0) sf[warp] = v;
    __syncthreads();
    float s = 0.f;
    for (int w = 0; w < kLNW; w++) s += sf[w];
    __syncthreads();
    return s;
}

// ---------------------------------------------------------------------------
// long_collect: the level's work items of one listed unit (CTA per unit)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void unit_of(const LongArgs &A, int i, int64_t &uid, int &lg, int &j) {
    if (A.fresh) {
        j = A.list[i / A.nlg];
        lg = A.lg0 + i % A.nlg;
        uid = (int64_t)lg * A.J + j;
    } else {
        uid = A.list[i];
        lg = (int)(uid / A.J);
        j = (int)(uid - (int64_t)lg * A.J);
    }
}

__global__ void __launch_bounds__(kLT) long_collect_kernel(LongArgs A) {
    __shared__ float sf[kLNW];
    __shared__ int wcnt[kLNW];
    __shared__ int base_s;
    const int i = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int64_t uid;
    int lg, j;
    unit_of(A, i, uid, lg, j);
    const int sa = A.slots[j], sb = A.slots[j + 1], n = sb - sa;
    const int64_t nbase = node_base(lg, sa, A.cs, A.Nc);
    const size_t rbase = (size_t)lg * A.Nc + (sa - A.cs);
    // does the slot hold an accepted singleton-floor position (its Add is then a floor op)
    int ufl = 0;
    if (A.fl_acc) {
        int any = 0;
        for (int t = tid; t < n; t += kLT) any |= A.fl_acc[rbase + t];
        ufl = __syncthreads_or(any);
    }
    if (A.fresh) {
        float r = 0.f;
        for (int t = tid; t < n; t += kLT) r += A.rtok[rbase + t];
        const float rootR = block_sum(r, sf);
        for (int k = tid; k < 2 * n; k += kLT) A.nd_cost[nbase + k] = 0;   // unused slots carry no op
        if (tid == 0) {
            const unsigned int pos = atomicAdd(&A.n_items[0], 1u);
            if ((int64_t)pos < A.cap_items) {
                A.it_gv[pos] = nbase;
                A.it_uid[pos] = uid;
                A.it_kin[pos] = 0.f;   // a fresh root's creator is its Add, formed by long_eval
                A.it_ufl[pos] = (uint8_t)ufl;
                A.u_start[i] = (int32_t)pos;
                A.u_cnt[i] = 1;
            } else {
                atomicOr(A.status, 64);
                A.u_start[i] = 0;
                A.u_cnt[i] = 0;
            }
            A.nd_a[nbase] = sa; A.nd_b[nbase] = sb; A.nd_R[nbase] = rootR; A.nd_D[nbase] = 0.f;
            A.nd_parent[nbase] = (int32_t)(-2 - uid); A.nd_unit[nbase] = (int32_t)uid;
            A.nd_child0[nbase] = -1; A.nd_nchild[nbase] = 0; A.nd_U[nbase] = 0.f;
            A.nd_kappa[nbase] = 0.f; A.nd_sel[nbase] = 0;
            A.u_nnodes[uid] = 1; A.u_pend[uid] = -1.f; A.u_sel[uid] = 0;
            A.u_Uadd[uid] = 0.f; A.u_Ddrop[uid] = 0.f;
        }
        return;
    }
    // resume: pending nodes (child count -1) whose key bound reaches tau, in
    // node order; the others keep the unit's largest pending bound
    const int nn = A.u_nnodes[uid];
    int cnt = 0;
    float pend = -1.f;
    for (int k = tid; k < nn; k += kLT) {
        const int64_t v = nbase + k;
        if (A.nd_nchild[v] != -1) continue;
        const float bnd = A.nd_U[v];
        if (bnd < A.tau) { pend = fmaxf(pend, bnd); continue; }
        const int len = A.nd_b[v] - A.nd_a[v];
        if (len > kMaxUnit) { cnt++; continue; }
        // a small node: its subtree goes to the unit kernel (subtree mode), into
        // the slots reserved for it.  A node the unit kernel left pending inside
        // a subtree has none, but its bound is below a threshold that only
        // rises, so it never reaches this point; it is skipped all the same.
        if (A.nd_child0[v] < 0) continue;
        const int cls = len <= kShortUnit ? 0 : 1;
        const unsigned int pos = atomicAdd(&A.n_items[1 + cls], 1u);
        if ((int64_t)pos < A.cap_items) A.sub[(size_t)cls * A.cap_items + pos] = (int32_t)v;
        else atomicOr(A.status, 64);
    }
    pend = warp_max(pend);
    if (lane == 0) sf[warp] = pend;
    cnt = (int)block_sum((float)cnt, reinterpret_cast<float *>(wcnt));   // counts are far below 2^24
    if (tid == 0) {
        float pm = -1.f;
        for (int w = 0; w < kLNW; w++) pm = fmaxf(pm, sf[w]);
        A.u_pend[uid] = pm;
        int b0 = 0;
        if (cnt > 0) {
            const unsigned int pos = atomicAdd(&A.n_items[0], (unsigned)cnt);
            if ((int64_t)pos + cnt <= A.cap_items) {
                b0 = (int)pos;
            } else {
                atomicOr(A.status, 64);
                cnt = 0;
            }
        }
        A.u_start[i] = b0;
        A.u_cnt[i] = cnt;
        base_s = cnt > 0 ? b0 : -1;
    }
    __syncthreads();
    if (base_s < 0) return;
    // ordered compaction, 256 nodes at a time
    int out = base_s;
    for (int k0 = 0; k0 < nn; k0 += kLT) {
        const int k = k0 + tid;
        bool q = false;
        if (k < nn && A.nd_nchild[nbase + k] == -1)
            q = A.nd_U[nbase + k] >= A.tau && A.nd_b[nbase + k] - A.nd_a[nbase + k] > kMaxUnit;
        const unsigned bal = __ballot_sync(0xffffffffu, q);
        if (lane == 0) wcnt[warp] = __popc(bal);
        __syncthreads();
        int before = 0, tot = 0;
        for (int w = 0; w < kLNW; w++) {
            before += w < warp ? wcnt[w] : 0;
            tot += wcnt[w];
        }
        if (q) {
            const int pos = out + before + __popc(bal & ((1u << lane) - 1u));
            const int64_t v = nbase + k;
            const int32_t pg = A.nd_parent[v];
            A.it_gv[pos] = v;
            A.it_uid[pos] = uid;
            A.it_kin[pos] = pg < 0 ? (ufl ? FLT_MAX : A.u_Uadd[uid]) : A.nd_kappa[pg];
            A.it_ufl[pos] = (uint8_t)ufl;
        }
        out += tot;
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// long_eval: one node per CTA (grid-stride over the level's work items)
// ---------------------------------------------------------------------------
template <int DH>
struct LongSmem {
    float sk[kLMaxSeg][DH];          // per segment: sum of k_circ
    float srv[kLMaxSeg][DH];         //              sum of R v
    float ssv[kLMaxSeg][DH];         //              sum of v
    float sR[kLMaxSeg], sKn[kLMaxSeg];
    int sF[kLMaxSeg];                // accepted floor positions in the segment
    float red[kLNW][3 * DH + 2];     // per-warp partials of one segment
    float ktil[2 * kLNCD][DH], vtil[2 * kLNCD][DH];
    float redD[2 * kLNCD][kLNW], redP[2 * kLNCD][kLNW];
    float candD[2 * kLNCD], candP[2 * kLNCD], meff[2 * kLNCD];
    // the probe scans' staging ring: per buffer kLChunk value rows, then as
    // many probe-weight rows (32 float2) or key rows
    __align__(16) unsigned char ring[2][kLChunk * DH * 4 * 2];
    int ca[2 * kLNCD], cb[2 * kLNCD];   // prefixes at [0, npre) by ascending end, suffixes at
                                        // [kLNCD, kLNCD + nsuf) by descending start (absolute)
    int segb[kLMaxSeg + 1];
    int nseg;
    int sel[kLMaxCut], cut[kLMaxCut], pidx[kLMaxCut], sidx[kLMaxCut];
    int ncut, npre, nsuf, eL, eR, whole, pstar, forced;
    double kmin;
    float krange;
    unsigned long long bk[kLNW];
    int bp[kLNW];
    float bf[kLNW];
    int bad;
};

// Order-preserving 32-bit key of a float, widened (larger value -> larger key).
__device__ __forceinline__ unsigned long long fokey(float x) {
    const uint32_t u = __float_as_uint(x);
    return (u >> 31) ? (unsigned long long)(~u) : (unsigned long long)(u | 0x80000000u);
}

// Sort the rows [r0, r0 + m) of (ca, cb) by key (ascending), remapping the
// indices in idx[0 .. ni) that point into them.  Thread 0 only; m <= kLNCD.
__device__ void sort_rows(int *ca, int *cb, int r0, int m, bool by_end_asc, int *const *idx, int ni) {
    int perm[kLNCD], inv[kLNCD], ta[kLNCD], tb[kLNCD];
    for (int q = 0; q < m; q++) perm[q] = q;
    auto key = [&](int q) { return by_end_asc ? cb[r0 + q] : -ca[r0 + q]; };
    for (int x = 1; x < m; x++) {
        const int v = perm[x];
        int y = x - 1;
        while (y >= 0 && key(perm[y]) > key(v)) { perm[y + 1] = perm[y]; y--; }
        perm[y + 1] = v;
    }
    for (int q = 0; q < m; q++) { inv[perm[q]] = q; ta[q] = ca[r0 + perm[q]]; tb[q] = cb[r0 + perm[q]]; }
    for (int q = 0; q < m; q++) { ca[r0 + q] = ta[q]; cb[r0 + q] = tb[q]; }
    for (int k = 0; k < ni; k++)
        if (*idx[k] >= r0 && *idx[k] < r0 + m) *idx[k] = r0 + inv[*idx[k] - r0];
}

template <int DH, typename Tin>
__global__ void __launch_bounds__(kLT, 1) long_eval_kernel(LongArgs A) {
    using S = LongSmem<DH>;
    constexpr int HALF = DH / 2, NG = DH / (4 * kLCL), CH = 4 * NG, PPL = HALF / 32;
    static_assert(kLPP * kLCL == kLT && DH % (4 * kLCL) == 0 && HALF % 32 == 0, "layout");
    extern __shared__ __align__(16) unsigned char lsm_raw[];
    S &sm = *reinterpret_cast<S *>(lsm_raw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c = lane / kLPPW, pp = warp * kLPPW + (lane & (kLPPW - 1));
    const int64_t n_items = min((int64_t)*A.n_items, A.cap_items);
    const float inv_sqrt_d = A.inv_sqrt_d, lamZ = A.lamZ, lamM = A.lamM, epsf = A.eps;
    // work items are taken from a counter, so that CTAs finishing short nodes
    // take the next ones (the nodes of a level range from 129 to 16384 tokens)
    __shared__ long long s_it;
    for (;;) {
        __syncthreads();   // the previous item's reads of s_it are done
        if (tid == 0) s_it = (long long)atomicAdd(A.it_next, 1u);
        __syncthreads();
        const int64_t it = s_it;
        if (it >= n_items) break;
        const int64_t gv = A.it_gv[it], uid = A.it_uid[it];
        const int lg = (int)(uid / A.J), l = lg / A.G, g = lg - l * A.G;
        const int a = A.nd_a[gv], b = A.nd_b[gv], n = b - a;
        const bool root = A.fresh != 0, ronly = root && A.root_only != 0;
        const bool cands = n >= 3 && !ronly;
        const float om = A.omega ? A.omega[lg] : 1.0f;
        const float *Rg = A.rtok + (size_t)lg * A.Nc - A.cs;   // Rg[t]: token value at absolute t
        const Tin *Kl = static_cast<const Tin *>(A.K) + (size_t)lg * A.T * DH;
        const Tin *Vl = static_cast<const Tin *>(A.V) + (size_t)lg * A.T * DH;
        if (tid == 0) sm.bad = 0;
        // ---- phase A: cut candidates, curvature range, p*, forced floor position
        {
            unsigned long long kmin = ~0ull, kmax = 0ull;
            for (int t = a + tid; t <= b - 2; t += kLT) {
                const unsigned long long k = lokey(A.kappa[t]);
                kmin = min(kmin, k);
                kmax = max(kmax, k);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
                kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
            }
            if (lane == 0) { sm.bk[warp] = kmin; sm.bp[warp] = (int)0; }
            __syncthreads();
            if (tid == 0) {
                unsigned long long mn = ~0ull;
                for (int w = 0; w < kLNW; w++) mn = min(mn, sm.bk[w]);
                sm.kmin = n >= 2 ? lokey_inv(mn) : 0.0;
            }
            __syncthreads();
            if (lane == 0) sm.bk[warp] = kmax;
            __syncthreads();
            if (tid == 0) {
                unsigned long long mx = 0ull;
                for (int w = 0; w < kLNW; w++) mx = max(mx, sm.bk[w]);
                const double kmx = n >= 2 ? lokey_inv(mx) : 0.0;
                sm.krange = kmx > sm.kmin ? 1.0f / (float)(kmx - sm.kmin) : 0.f;
            }
            __syncthreads();
        }
        // top-K positions of [a, b-2] by (kappa descending, position ascending)
        const int K = cands ? min(A.k_cand, n - 1) : 0;
        unsigned long long pk = 0ull;
        int ppos = -1, nsel = 0;
        for (int r = 0; r < K; r++) {
            unsigned long long bkey = 0ull;
            int bpos = INT_MAX;
            for (int t = a + tid; t <= b - 2; t += kLT) {
                const unsigned long long k = lokey(A.kappa[t]);
                if (r > 0 && !(k < pk || (k == pk && t > ppos))) continue;   // taken in an earlier round
                if (bpos == INT_MAX || k > bkey || (k == bkey && t < bpos)) { bkey = k; bpos = t; }
            }
            block_best(bkey, bpos, sm.bk, sm.bp);
            if (bpos == INT_MAX) break;
            if (tid == 0) sm.sel[r] = bpos;
            pk = bkey;
            ppos = bpos;
            nsel++;
        }
        // salient token p* = argmax R_tok over [a, b) (ties: lower t)
        {
            unsigned long long bkey = 0ull;
            int bpos = INT_MAX;
            for (int t = a + tid; t < b; t += kLT) {
                const float r = Rg[t];
                if (!isfinite(r)) sm.bad = 1;
                const unsigned long long k = fokey(r);
                if (bpos == INT_MAX || k > bkey) { bkey = k; bpos = t; }
            }
            block_best(bkey, bpos, sm.bk, sm.bp);
            if (tid == 0) sm.pstar = (bpos >= a && bpos < b) ? bpos : a;
        }
        // a node holding an accepted floor position is extracted at the one of
        // largest floor score (ties: lower t)
        {
            int fpos = INT_MAX;
            if (A.fl_acc) {
                unsigned long long bkey = 0ull;
                for (int t = a + tid; t < b; t += kLT) {
                    const size_t q = (size_t)lg * A.Nc + (t - A.cs);
                    if (!A.fl_acc[q]) continue;
                    const unsigned long long k = fokey(A.fl_f[q]);
                    if (fpos == INT_MAX || k > bkey) { bkey = k; fpos = t; }
                }
                block_best(bkey, fpos, sm.bk, sm.bp);
            }
            if (tid == 0) {
                sm.forced = fpos != INT_MAX ? 1 : 0;
                if (fpos != INT_MAX) sm.pstar = fpos;
            }
        }
        __syncthreads();
        // candidate lists and segment boundaries (thread 0)
        if (tid == 0) {
            int nc = 0;
            if (cands) {
                const int mid = a + n / 2;
                bool have = false;
                for (int r = 0; r < nsel; r++) { sm.cut[nc++] = sm.sel[r] + 1; have |= sm.sel[r] + 1 == mid; }
                if (!have) sm.cut[nc++] = mid;
                for (int x = 1; x < nc; x++) {
                    const int v = sm.cut[x];
                    int y = x - 1;
                    while (y >= 0 && sm.cut[y] > v) { sm.cut[y + 1] = sm.cut[y]; y--; }
                    sm.cut[y + 1] = v;
                }
            }
            sm.ncut = nc;
            const int ps = sm.pstar, er = ps + 1;
            int npre = 0, nsuf = 0;
            for (int q = 0; q < nc; q++) {
                const int xi = sm.cut[q];
                sm.pidx[q] = -1;
                if (xi - a >= 2) { sm.ca[npre] = a; sm.cb[npre] = xi; sm.pidx[q] = npre++; }
            }
            int eL = -1, eR = -1, whole = -1;
            if (cands && ps - a >= 2) {
                for (int q = 0; q < nc; q++) if (sm.cut[q] == ps && sm.pidx[q] >= 0) eL = sm.pidx[q];
                if (eL < 0) { sm.ca[npre] = a; sm.cb[npre] = ps; eL = npre++; }
            }
            if (root) { sm.ca[npre] = a; sm.cb[npre] = b; whole = npre++; }
            for (int q = 0; q < nc; q++) {
                const int xi = sm.cut[q];
                sm.sidx[q] = -1;
                if (b - xi >= 2) { sm.ca[kLNCD + nsuf] = xi; sm.cb[kLNCD + nsuf] = b; sm.sidx[q] = kLNCD + nsuf++; }
            }
            if (cands && b - er >= 2) {
                for (int q = 0; q < nc; q++) if (sm.cut[q] == er && sm.sidx[q] >= 0) eR = sm.sidx[q];
                if (eR < 0) { sm.ca[kLNCD + nsuf] = er; sm.cb[kLNCD + nsuf] = b; eR = kLNCD + nsuf++; }
            }
            {
                int *pi[kLMaxCut + 2];
                int ni = 0;
                for (int q = 0; q < nc; q++) pi[ni++] = &sm.pidx[q];
                pi[ni++] = &eL;
                pi[ni++] = &whole;
                sort_rows(sm.ca, sm.cb, 0, npre, true, pi, ni);
                ni = 0;
                for (int q = 0; q < nc; q++) pi[ni++] = &sm.sidx[q];
                pi[ni++] = &eR;
                sort_rows(sm.ca, sm.cb, kLNCD, nsuf, false, pi, ni);
            }
            sm.npre = npre; sm.nsuf = nsuf; sm.eL = eL; sm.eR = eR; sm.whole = whole;
            // segment boundaries: a, b, the cuts, p*, p* + 1
            int bd[kLMaxCut + 4], nb = 0;
            bd[nb++] = a;
            bd[nb++] = b;
            for (int q = 0; q < nc; q++) bd[nb++] = sm.cut[q];
            if (ps > a) bd[nb++] = ps;
            if (er < b) bd[nb++] = er;
            for (int x = 1; x < nb; x++) {
                const int v = bd[x];
                int y = x - 1;
                while (y >= 0 && bd[y] > v) { bd[y + 1] = bd[y]; y--; }
                bd[y + 1] = v;
            }
            int m = 0;
            for (int x = 0; x < nb; x++) if (m == 0 || bd[x] != sm.segb[m - 1]) sm.segb[m++] = bd[x];
            sm.nseg = m - 1;
        }
        __syncthreads();
        // ---- phase B: per-segment sums of k_circ, R v, v, R, ||k|| and floor positions
        // Warp w takes the tokens x + w, x + w + 8, ...; lane owns the rotation
        // pairs (i, i + d/2), i = PPL lane + j.  Each warp's running sums are
        // folded every kLFold of its tokens.
        const int nseg = sm.nseg;
        for (int s = 0; s < nseg; s++) {
            const int x = sm.segb[s], y = sm.segb[s + 1];
            const int i0 = lane * PPL;
            float tk0[PPL], tk1[PPL], tr0[PPL], tr1[PPL], tv0[PPL], tv1[PPL];
            float ck0[PPL], ck1[PPL], cr0[PPL], cr1[PPL], cv0[PPL], cv1[PPL];
            float trs = 0.f, tks = 0.f, crs = 0.f, cks = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) tk0[j] = tk1[j] = tr0[j] = tr1[j] = tv0[j] = tv1[j] = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) ck0[j] = ck1[j] = cr0[j] = cr1[j] = cv0[j] = cv1[j] = 0.f;
            int fold = 0;
            for (int t = x + warp; t < y; t += kLNW) {
                float k0[PPL], k1[PPL], v0[PPL], v1[PPL];
                lld_pairs<PPL>(Kl + (size_t)t * DH + i0, k0);
                lld_pairs<PPL>(Kl + (size_t)t * DH + i0 + HALF, k1);
                lld_pairs<PPL>(Vl + (size_t)t * DH + i0, v0);
                lld_pairs<PPL>(Vl + (size_t)t * DH + i0 + HALF, v1);
                const float rt = Rg[t];
                float nn = 0.f;
#pragma unroll
                for (int j = 0; j < PPL; j++) {
                    nn = fmaf(k0[j], k0[j], fmaf(k1[j], k1[j], nn));
                    const float2 cs = A.rope[(size_t)t * HALF + i0 + j];
                    // k_circ = RoPE^-1(k, t): rotation by -t
                    ck0[j] += k0[j] * cs.x + k1[j] * cs.y;
                    ck1[j] += k1[j] * cs.x - k0[j] * cs.y;
                    cr0[j] = fmaf(rt, v0[j], cr0[j]);
                    cr1[j] = fmaf(rt, v1[j], cr1[j]);
                    cv0[j] += v0[j];
                    cv1[j] += v1[j];
                }
                nn = warp_sum(nn);
                crs += rt;
                cks += sqrtf(nn);
                if (++fold == kLFold) {
#pragma unroll
                    for (int j = 0; j < PPL; j++) {
                        tk0[j] += ck0[j]; tk1[j] += ck1[j]; tr0[j] += cr0[j]; tr1[j] += cr1[j];
                        tv0[j] += cv0[j]; tv1[j] += cv1[j];
                        ck0[j] = ck1[j] = cr0[j] = cr1[j] = cv0[j] = cv1[j] = 0.f;
                    }
                    trs += crs; tks += cks; crs = cks = 0.f;
                    fold = 0;
                }
            }
            float *rw = sm.red[warp];
#pragma unroll
            for (int j = 0; j < PPL; j++) {
                rw[i0 + j] = tk0[j] + ck0[j];
                rw[i0 + j + HALF] = tk1[j] + ck1[j];
                rw[DH + i0 + j] = tr0[j] + cr0[j];
                rw[DH + i0 + j + HALF] = tr1[j] + cr1[j];
                rw[2 * DH + i0 + j] = tv0[j] + cv0[j];
                rw[2 * DH + i0 + j + HALF] = tv1[j] + cv1[j];
            }
            if (lane == 0) { rw[3 * DH] = trs + crs; rw[3 * DH + 1] = tks + cks; }
            int fc = 0;
            if (A.fl_acc)
                for (int t = x + tid; t < y; t += kLT) fc += A.fl_acc[(size_t)lg * A.Nc + (t - A.cs)] ? 1 : 0;
            fc = __syncthreads_count(fc != 0);   // also orders the partials above
            for (int e = tid; e < 3 * DH + 2; e += kLT) {
                float v = 0.f;
#pragma unroll
                for (int w = 0; w < kLNW; w++) v += sm.red[w][e];
                if (e < DH) sm.sk[s][e] = v;
                else if (e < 2 * DH) sm.srv[s][e - DH] = v;
                else if (e < 3 * DH) sm.ssv[s][e - 2 * DH] = v;
                else if (e == 3 * DH) sm.sR[s] = v;
                else sm.sKn[s] = v;
            }
            if (tid == 0) sm.sF[s] = fc;
            __syncthreads();
        }
        // ---- phase C: candidate prototypes from their segments (warp per candidate)
        auto seg_of = [&](int pos) {   // index of the boundary at pos (every candidate end is one)
            int s = 0;
            while (s < nseg && sm.segb[s] != pos) s++;
            return s;
        };
        const int npre = sm.npre, nsuf = sm.nsuf;
        for (int q = warp; q < npre + nsuf; q += kLNW) {
            const int k = q < npre ? q : kLNCD + (q - npre);
            const int x = sm.ca[k], y = sm.cb[k], nJ = y - x;
            const int s0 = seg_of(x), s1 = seg_of(y);
            const int p = lround_half_even_mid(x, y);
            const int i0 = lane * PPL;
            float2 rot[PPL];
#pragma unroll
            for (int j = 0; j < PPL; j++) rot[j] = A.rope[(size_t)p * HALF + i0 + j];
            float m0[PPL], m1[PPL], r0[PPL], r1[PPL], v0[PPL], v1[PPL];
            float rs = 0.f, ks = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) m0[j] = m1[j] = r0[j] = r1[j] = v0[j] = v1[j] = 0.f;
            for (int s = s0; s < s1; s++) {
#pragma unroll
                for (int j = 0; j < PPL; j++) {
                    m0[j] += sm.sk[s][i0 + j];  m1[j] += sm.sk[s][i0 + j + HALF];
                    r0[j] += sm.srv[s][i0 + j]; r1[j] += sm.srv[s][i0 + j + HALF];
                    v0[j] += sm.ssv[s][i0 + j]; v1[j] += sm.ssv[s][i0 + j + HALF];
                }
                rs += sm.sR[s];
                ks += sm.sKn[s];
            }
            const float ninv = 1.0f / (float)nJ;
            const float beta = A.base_frac * (rs * ninv);
            const float winv = 1.0f / ((rs + (float)nJ * beta) + epsf);
            float mu2 = 0.f;
#pragma unroll
            for (int j = 0; j < PPL; j++) {
                const float a0 = m0[j] * ninv, a1 = m1[j] * ninv;
                mu2 = fmaf(a0, a0, fmaf(a1, a1, mu2));
                sm.ktil[k][i0 + j] = a0 * rot[j].x - a1 * rot[j].y;
                sm.ktil[k][i0 + j + HALF] = a0 * rot[j].y + a1 * rot[j].x;
                sm.vtil[k][i0 + j] = fmaf(beta, v0[j], r0[j]) * winv;
                sm.vtil[k][i0 + j + HALF] = fmaf(beta, v1[j], r1[j]) * winv;
            }
            mu2 = warp_sum(mu2);
            if (lane == 0) {
                const float coh = sqrtf(mu2) / (ks * ninv + epsf);
                const float me = (float)nJ * coh * coh;
                sm.meff[k] = me < 1.0f ? 1.0f : (me > (float)nJ ? (float)nJ : me);
            }
        }
        __syncthreads();
        // ---- phase D: probe scans --------------------------------------------
        // thread (pp, c): probes pp and pp + 32, elements 4 c + 32 gi + j
        float2 qa0[CH / 2], qa1[CH / 2];
        float mu0 = 0.f, mu1 = 0.f, invZ0 = 0.f, invZ1 = 0.f;
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int u = pp + kLPP * h;
            float2 *qd = h ? qa1 : qa0;
            if (u < A.W) {
                const size_t row = ((size_t)l * A.Hq + g * A.gq + (u % A.gq)) * A.W + u;
                const Tin *qp = static_cast<const Tin *>(A.Q) + row * DH + 4 * c;
#pragma unroll
                for (int gi = 0; gi < NG; gi++) {
                    const float4 x = lld4(qp + 32 * gi);
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
        const bool has0 = pp < A.W, has1 = pp + kLPP < A.W;
        // D_u of candidate row k from the running statistics, weighted by the
        // probe's attention mass; per-warp partial sums (as in build.cu)
        auto evaluate = [&](int k, float Z0, float Z1, const float2 *M0, const float2 *M1) {
            float2 kt[CH / 2];
#pragma unroll
            for (int gi = 0; gi < NG; gi++) {
                const float4 x = *reinterpret_cast<const float4 *>(&sm.ktil[k][4 * c + 32 * gi]);
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
            for (int o = kLPPW; o < 32; o <<= 1) {
                x0 += __shfl_xor_sync(0xffffffffu, x0, o);
                x1 += __shfl_xor_sync(0xffffffffu, x1, o);
            }
            const float me = sm.meff[k];
            const float zt0 = me * expf(x0 * inv_sqrt_d - mu0), zt1 = me * expf(x1 * inv_sqrt_d - mu1);
            const float2 nz0 = make_float2(-zt0, -zt0), nz1 = make_float2(-zt1, -zt1);
            float2 r0 = make_float2(0.f, 0.f), r1 = r0, m0 = r0, m1 = r0;
#pragma unroll
            for (int gi = 0; gi < NG; gi++) {
                const float4 x = *reinterpret_cast<const float4 *>(&sm.vtil[k][4 * c + 32 * gi]);
                const float2 va = make_float2(x.x, x.y), vb = make_float2(x.z, x.w);
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const int q = 2 * gi + h;
                    const float2 vt = h ? vb : va;
                    const float2 d0 = ffma2(nz0, vt, M0[q]), d1 = ffma2(nz1, vt, M1[q]);
                    r0 = ffma2(d0, d0, r0);
                    r1 = ffma2(d1, d1, r1);
                    m0 = ffma2(M0[q], M0[q], m0);
                    m1 = ffma2(M1[q], M1[q], m1);
                }
            }
            float res0 = r0.x + r0.y, res1 = r1.x + r1.y, mm0 = m0.x + m0.y, mm1 = m1.x + m1.y;
#pragma unroll
            for (int o = kLPPW; o < 32; o <<= 1) {
                res0 += __shfl_xor_sync(0xffffffffu, res0, o);
                res1 += __shfl_xor_sync(0xffffffffu, res1, o);
                mm0 += __shfl_xor_sync(0xffffffffu, mm0, o);
                mm1 += __shfl_xor_sync(0xffffffffu, mm1, o);
            }
            const float dz0 = Z0 - zt0, dz1 = Z1 - zt1;
            const float D0 = lamZ * __fdividef(dz0 * dz0, fmaf(Z0, Z0, epsf)) + lamM * __fdividef(res0, mm0 + epsf);
            const float D1 = lamZ * __fdividef(dz1 * dz1, fmaf(Z1, Z1, epsf)) + lamM * __fdividef(res1, mm1 + epsf);
            const float p0 = Z0 * invZ0, p1 = Z1 * invZ1;
            float pd = fmaf(p0, D0, p1 * D1), pw = p0 + p1;
#pragma unroll
            for (int o = 1; o < kLPPW; o <<= 1) {
                pd += __shfl_xor_sync(0xffffffffu, pd, o);
                pw += __shfl_xor_sync(0xffffffffu, pw, o);
            }
            if (lane == 0) { sm.redD[k][warp] = pd; sm.redP[k][warp] = pw; }
        };
        // one direction: the running sums over the node's tokens, folded every
        // kLFold tokens and at every candidate end, evaluated at each end.  The
        // tokens are staged kLChunk at a time in a two-buffer cp.async ring:
        // their value rows and their probe weights (pass B) or key rows.
        auto scan = [&](bool suffix) {
            const int nk = suffix ? nsuf : npre;
            if (nk == 0) return;
            // tokens of the scan: forward a, a + 1, ..; backward b - 1, b - 2, ..
            int last = suffix ? b : a;     // the farthest candidate end
            for (int k = 0; k < nk; k++) {
                const int kr = suffix ? kLNCD + k : k;
                last = suffix ? min(last, sm.ca[kr]) : max(last, sm.cb[kr]);
            }
            const int ntok = suffix ? b - last : last - a;
            float2 Mt0[CH / 2], Mt1[CH / 2], Mc0[CH / 2], Mc1[CH / 2];
            float Zt0 = 0.f, Zt1 = 0.f, Zc0 = 0.f, Zc1 = 0.f;
#pragma unroll
            for (int q = 0; q < CH / 2; q++) Mt0[q] = Mt1[q] = Mc0[q] = Mc1[q] = make_float2(0.f, 0.f);
            auto fold_in = [&]() {
#pragma unroll
                for (int q = 0; q < CH / 2; q++) {
                    Mt0[q].x += Mc0[q].x; Mt0[q].y += Mc0[q].y; Mt1[q].x += Mc1[q].x; Mt1[q].y += Mc1[q].y;
                    Mc0[q] = Mc1[q] = make_float2(0.f, 0.f);
                }
                Zt0 += Zc0; Zt1 += Zc1; Zc0 = Zc1 = 0.f;
            };
            // chunk c holds the scan's tokens [c kLChunk, (c + 1) kLChunk): rows
            // tlo .. tlo + m - 1 of the input, tlo the smallest position
            auto chunk_rows = [&](int c0, int &tlo, int &m) {
                m = min(kLChunk, ntok - c0);
                tlo = suffix ? b - c0 - m : a + c0;
            };
            auto issue = [&](int c0, int buf) {
                if (c0 < ntok) {
                    int tlo, m;
                    chunk_rows(c0, tlo, m);
                    unsigned char *dst = sm.ring[buf];
                    constexpr int RB = DH * (int)sizeof(Tin);             // bytes of a K or V row
                    const char *vsrc = reinterpret_cast<const char *>(Vl + (size_t)tlo * DH);
                    for (int q = tid; q < m * RB / 16; q += kLT) cp_async16(dst + 16 * q, vsrc + 16 * q, true);
                    unsigned char *dst2 = dst + kLChunk * RB;
                    if (A.Eg) {
                        const char *esrc = reinterpret_cast<const char *>(A.Eg + ((size_t)lg * A.Nc + (tlo - A.cs)) * kLPP);
                        for (int q = tid; q < m * kLPP * 8 / 16; q += kLT) cp_async16(dst2 + 16 * q, esrc + 16 * q, true);
                    } else {
                        const char *ksrc = reinterpret_cast<const char *>(Kl + (size_t)tlo * DH);
                        for (int q = tid; q < m * RB / 16; q += kLT) cp_async16(dst2 + 16 * q, ksrc + 16 * q, true);
                    }
                }
                cp_async_commit();
            };
            int kk = 0, fold = 0;
            bool badt = false;
            issue(0, 0);
            for (int c0 = 0, buf = 0; c0 < ntok; c0 += kLChunk, buf ^= 1) {
                issue(c0 + kLChunk, buf ^ 1);
                cp_async_wait<1>();   // this chunk's copies have landed (each thread its own)
                __syncthreads();
                int tlo, m;
                chunk_rows(c0, tlo, m);
                const Tin *vrow0 = reinterpret_cast<const Tin *>(sm.ring[buf]);
                const unsigned char *aux = sm.ring[buf] + kLChunk * DH * (int)sizeof(Tin);
                for (int i = 0; i < m; i++) {
                    const int r = suffix ? m - 1 - i : i;   // row of the scan's token c0 + i
                    float e0, e1;
                    if (A.Eg) {
                        const float2 e = reinterpret_cast<const float2 *>(aux)[r * kLPP + pp];
                        e0 = has0 ? e.x : 0.f;
                        e1 = has1 ? e.y : 0.f;
                    } else {
                        const Tin *krow = reinterpret_cast<const Tin *>(aux) + (size_t)r * DH;
                        float2 ya = make_float2(0.f, 0.f), yb = ya;
#pragma unroll
                        for (int gi = 0; gi < NG; gi++) {
                            const float4 kv = lld4(krow + 4 * c + 32 * gi);
                            const float2 ka = make_float2(kv.x, kv.y), kb = make_float2(kv.z, kv.w);
                            ya = ffma2(qa0[2 * gi], ka, ya); ya = ffma2(qa0[2 * gi + 1], kb, ya);
                            yb = ffma2(qa1[2 * gi], ka, yb); yb = ffma2(qa1[2 * gi + 1], kb, yb);
                        }
                        float y0 = ya.x + ya.y, y1 = yb.x + yb.y;
#pragma unroll
                        for (int o = kLPPW; o < 32; o <<= 1) {
                            y0 += __shfl_xor_sync(0xffffffffu, y0, o);
                            y1 += __shfl_xor_sync(0xffffffffu, y1, o);
                        }
                        e0 = has0 ? expf(y0 * inv_sqrt_d - mu0) : 0.f;
                        e1 = has1 ? expf(y1 * inv_sqrt_d - mu1) : 0.f;
                    }
                    badt |= !isfinite(e0) || !isfinite(e1);
                    const float2 ee0 = make_float2(e0, e0), ee1 = make_float2(e1, e1);
                    Zc0 += e0;
                    Zc1 += e1;
                    const Tin *vrow = vrow0 + (size_t)r * DH;
#pragma unroll
                    for (int gi = 0; gi < NG; gi++) {
                        const float4 x = lld4(vrow + 4 * c + 32 * gi);
                        const float2 va = make_float2(x.x, x.y), vb = make_float2(x.z, x.w);
                        Mc0[2 * gi] = ffma2(ee0, va, Mc0[2 * gi]);
                        Mc0[2 * gi + 1] = ffma2(ee0, vb, Mc0[2 * gi + 1]);
                        Mc1[2 * gi] = ffma2(ee1, va, Mc1[2 * gi]);
                        Mc1[2 * gi + 1] = ffma2(ee1, vb, Mc1[2 * gi + 1]);
                    }
                    if (++fold == kLFold) { fold_in(); fold = 0; }
                    // candidates whose far end is this token
                    const int t = suffix ? b - 1 - (c0 + i) : a + c0 + i;
                    while (kk < nk) {
                        const int kr = suffix ? kLNCD + kk : kk;
                        if ((suffix ? sm.ca[kr] : sm.cb[kr] - 1) != t) break;
                        fold_in();
                        fold = 0;
                        evaluate(kr, Zt0, Zt1, Mt0, Mt1);
                        kk++;
                    }
                }
                __syncthreads();   // the buffer is refilled by the next issue
            }
            cp_async_wait<0>();
            if (badt) sm.bad = 1;
        };
        scan(false);
        scan(true);
        __syncthreads();
        // ---- phase E: candidate D, the decision, gains and keys -----------------
        const float invW = 1.0f / (float)A.W;
        for (int q = tid; q < npre + nsuf; q += kLT) {
            const int k = q < npre ? q : kLNCD + (q - npre);
            float d = 0.f, pw = 0.f;
#pragma unroll
            for (int w = 0; w < kLNW; w++) { d += sm.redD[k][w]; pw += sm.redP[k][w]; }
            sm.candD[k] = d * invW;
            sm.candP[k] = pw * invW;
        }
        __syncthreads();
        if (warp == 0) {
            LongRes rs;
            rs.nch = 0;
            rs.U = rs.kap = rs.bound = 0.f;
            for (int q = 0; q < 3; q++) { rs.ca[q] = rs.cb[q] = 0; rs.cD[q] = rs.rch[q] = rs.bnd[q] = 0.f; }
            const int forced = sm.forced, ps = sm.pstar, ncut = sm.ncut;
            const bool ufl = A.it_ufl[it] != 0;
            float kin = A.it_kin[it];
            float DI;
            const float nodeR = A.nd_R[gv];
            if (root) {   // D, D_drop and the Add gain of the slot (Eq. app_operation_gains)
                const float Pd = sm.candP[sm.whole];
                DI = sm.candD[sm.whole];
                float gain = om * nodeR * (Pd - DI);
                if (gain < 0.f) gain = 0.f;
                kin = ufl ? FLT_MAX : gain;   // a floor slot's Add is a floor op
                if (lane == 0) {
                    A.u_Uadd[uid] = sm.bad ? 0.f : gain;
                    A.u_Ddrop[uid] = sm.bad ? 0.f : Pd;
                    A.nd_D[gv] = sm.bad ? 0.f : DI;
                }
            } else {
                DI = A.nd_D[gv];
            }
            // value of [x, y) from the segment sums; does it hold a floor position
            auto seg_sum = [&](int x, int y, float &r, bool &fl) {   // x, y are boundaries
                int s = 0;
                while (s < nseg && sm.segb[s] != x) s++;
                r = 0.f;
                fl = false;
                for (; s < nseg && sm.segb[s] != y; s++) { r += sm.sR[s]; fl |= sm.sF[s] != 0; }
            };
            if (sm.bad) {
                if (lane == 0) atomicOr(A.status, 8);   // non-finite: a leaf with zero gain
                rs.nch = 0;
            } else if (ronly) {   // the root's split is decided later: bound its key
                rs.nch = -1;
                rs.bound = forced ? FLT_MAX : fminf(kin, lkey_bound(om * nodeR * DI));
            } else {
                int nch;
                if (n == 2) {
                    nch = 2;
                    rs.ca[0] = a; rs.cb[0] = a + 1; rs.cD[0] = 0.f;
                    rs.ca[1] = a + 1; rs.cb[1] = b; rs.cD[1] = 0.f;
                } else {
                    // binary cut: lane q evaluates cut q; max G_bin, ties -> smallest xi
                    float best = -INFINITY;
                    int bq = 0x7fffffff;
                    if (lane < ncut) {
                        const int xi = sm.cut[lane];
                        const float DL = sm.pidx[lane] >= 0 ? sm.candD[sm.pidx[lane]] : 0.f;
                        const float DR = sm.sidx[lane] >= 0 ? sm.candD[sm.sidx[lane]] : 0.f;
                        const float kh = (float)(A.kappa[xi - 1] - sm.kmin) * sm.krange;
                        best = ((DI - DL) - DR) + A.lam_kappa * kh;
                        bq = lane;
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
                        const float ov = __shfl_xor_sync(0xffffffffu, best, o);
                        const int oq = __shfl_xor_sync(0xffffffffu, bq, o);
                        if (ov > best || (ov == best && oq < bq)) { best = ov; bq = oq; }
                    }
                    int bxi = -1;
                    float bL = 0.f, bR = 0.f;
                    if (bq < ncut && best > -INFINITY) {
                        bxi = sm.cut[bq];
                        bL = sm.pidx[bq] >= 0 ? sm.candD[sm.pidx[bq]] : 0.f;
                        bR = sm.sidx[bq] >= 0 ? sm.candD[sm.sidx[bq]] : 0.f;
                    }
                    // extraction at p*
                    int ea[3], eb[3], ne = 0;
                    float eD[3];
                    if (ps > a) { ea[ne] = a; eb[ne] = ps; eD[ne] = ps - a >= 2 ? sm.candD[sm.eL] : 0.f; ne++; }
                    ea[ne] = ps; eb[ne] = ps + 1; eD[ne] = 0.f; ne++;
                    if (ps + 1 < b) { ea[ne] = ps + 1; eb[ne] = b; eD[ne] = b - ps - 1 >= 2 ? sm.candD[sm.eR] : 0.f; ne++; }
                    float gext = DI;
                    for (int q = 0; q < ne; q++) gext -= eD[q];
                    if (bxi < 0) {   // only reachable with non-finite gains
                        bxi = sm.cut[0];
                        bL = sm.pidx[0] >= 0 ? sm.candD[sm.pidx[0]] : 0.f;
                        bR = sm.sidx[0] >= 0 ? sm.candD[sm.sidx[0]] : 0.f;
                    }
                    const float rho_ext = ne == 3 ? 0.5f * gext : gext;   // G_ext / (|children| - 1)
                    if (forced || rho_ext > best) {
                        nch = ne;
                        for (int q = 0; q < ne; q++) { rs.ca[q] = ea[q]; rs.cb[q] = eb[q]; rs.cD[q] = eD[q]; }
                    } else {
                        nch = 2;
                        rs.ca[0] = a; rs.cb[0] = bxi; rs.cD[0] = bL;
                        rs.ca[1] = bxi; rs.cb[1] = b; rs.cD[1] = bR;
                    }
                }
                bool chf[3] = {false, false, false};
                for (int q = 0; q < nch; q++) seg_sum(rs.ca[q], rs.cb[q], rs.rch[q], chf[q]);
                const float rnode = (rs.rch[0] + rs.rch[1]) + rs.rch[2];   // R of the node = sum over its children
                const float dsum = (rs.cD[0] + rs.cD[1]) + (nch == 3 ? rs.cD[2] : 0.f);
                const int cost = nch - 1;
                float gain = om * rnode * (DI - dsum);
                if (gain < 0.f) gain = 0.f;
                rs.U = cost == 2 ? 0.5f * gain : gain;
                rs.kap = forced ? FLT_MAX : fminf(rs.U, kin);
                for (int q = 0; q < nch; q++)
                    rs.bnd[q] = rs.cb[q] - rs.ca[q] >= 2
                                    ? (chf[q] ? FLT_MAX : fminf(rs.kap, lkey_bound(om * rs.rch[q] * rs.cD[q])))
                                    : 0.f;
                rs.nch = nch;
            }
            if (lane == 0) {
                A.res[it] = rs;
                int pe = a, ssn = b, len = 0;
                for (int q = 0; q < npre; q++) { pe = max(pe, sm.cb[q]); len += sm.cb[q] - sm.ca[q]; }
                for (int q = 0; q < nsuf; q++) { ssn = min(ssn, sm.ca[kLNCD + q]); len += sm.cb[kLNCD + q] - sm.ca[kLNCD + q]; }
                atomicAdd(&A.work[0], (unsigned long long)((pe - a) + (b - ssn)));
                atomicAdd(&A.work[1], (unsigned long long)(npre + nsuf));
                atomicAdd(&A.work[2], (unsigned long long)len);
                atomicAdd(&A.work[3], 1ull);
            }
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// long_commit: children numbered after the unit's nodes, in work-item order
// (warp per listed unit)
// ---------------------------------------------------------------------------
__global__ void long_commit_kernel(LongArgs A) {
    const int i = blockIdx.x, lane = threadIdx.x;
    const int start = A.u_start[i], cnt = A.u_cnt[i];
    if (cnt <= 0) return;
    const int64_t uid = A.it_uid[start];
    const int lg = (int)(uid / A.J), j = (int)(uid - (int64_t)lg * A.J);
    const int64_t nbase = node_base(lg, A.slots[j], A.cs, A.Nc);
    int base = A.u_nnodes[uid];
    float pend = A.u_pend[uid];
    for (int k0 = 0; k0 < cnt; k0 += 32) {
        const int k = k0 + lane;
        const bool in = k < cnt;
        LongRes rs;
        int64_t gv = 0;
        int nch = 0, used = 0;
        if (in) {
            rs = A.res[start + k];
            gv = A.it_gv[start + k];
            nch = rs.nch > 0 ? rs.nch : 0;
            // the children's slots, then for each child of 2 .. kMaxUnit tokens the
            // 2 len - 2 slots its subtree can need (the unit kernel fills them)
            used = nch;
            for (int q = 0; q < nch; q++) {
                const int len = rs.cb[q] - rs.ca[q];
                if (len >= 2 && len <= kMaxUnit) used += 2 * len - 2;
            }
        }
        int incl = used;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        const int tot = __shfl_sync(0xffffffffu, incl, 31);
        if (in) {
            if (rs.nch < 0) {   // pending root: its split key is bounded
                A.nd_child0[gv] = -1; A.nd_nchild[gv] = -1; A.nd_cost[gv] = 0;
                A.nd_U[gv] = rs.bound; A.nd_kappa[gv] = 0.f; A.nd_sel[gv] = 0;
                pend = fmaxf(pend, rs.bound);
            } else if (rs.nch == 0) {
                A.nd_child0[gv] = -1; A.nd_nchild[gv] = 0; A.nd_cost[gv] = 0;
                A.nd_U[gv] = 0.f; A.nd_kappa[gv] = 0.f; A.nd_sel[gv] = 0;
            } else {
                const int child0 = base + incl - used;   // unit-relative index
                const int cost = nch - 1;
                A.nd_child0[gv] = child0; A.nd_nchild[gv] = (int8_t)nch; A.nd_cost[gv] = (int8_t)cost;
                A.nd_U[gv] = rs.U; A.nd_kappa[gv] = rs.kap; A.nd_sel[gv] = 0;
                A.ops[atomicAdd(A.n_ops, 1u)] =
                    make_uint2(__float_as_uint(rs.kap), ((uint32_t)gv << 1) | (uint32_t)(cost - 1));
                int res = child0 + nch;
                for (int q = 0; q < nch; q++) {
                    const int64_t gc = nbase + child0 + q;
                    const int len = rs.cb[q] - rs.ca[q];
                    const bool pending = len >= 2;
                    A.nd_a[gc] = rs.ca[q]; A.nd_b[gc] = rs.cb[q];
                    A.nd_parent[gc] = (int32_t)gv; A.nd_unit[gc] = (int32_t)uid;
                    A.nd_D[gc] = rs.cD[q]; A.nd_R[gc] = rs.rch[q];
                    // a pending child of at most kMaxUnit tokens keeps its reservation in
                    // child0; the reserved slots are marked unused (child count -2) until
                    // the unit kernel fills them
                    A.nd_child0[gc] = (pending && len <= kMaxUnit) ? res : -1;
                    if (pending && len <= kMaxUnit) {
                        for (int r = res; r < res + 2 * len - 2; r++) {
                            A.nd_nchild[nbase + r] = -2; A.nd_cost[nbase + r] = 0; A.nd_sel[nbase + r] = 0;
                        }
                        res += 2 * len - 2;
                    }
                    A.nd_nchild[gc] = pending ? -1 : 0; A.nd_cost[gc] = 0;
                    A.nd_U[gc] = pending ? rs.bnd[q] : 0.f;   // a pending node's key bound
                    A.nd_kappa[gc] = 0.f; A.nd_sel[gc] = 0;
                    if (pending) pend = fmaxf(pend, rs.bnd[q]);
                }
            }
        }
        base += tot;
    }
    pend = warp_max(pend);
    if (lane == 0) {
        A.u_nnodes[uid] = base;
        A.u_pend[uid] = pend;
    }
}

// CTAs of long_eval resident per SM (its shared memory set as at launch)
template <int DH, typename Tin>
int eval_occupancy() {
    using S = LongSmem<DH>;
    if (cudaFuncSetAttribute(long_eval_kernel<DH, Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)sizeof(S)) != cudaSuccess)
        return 1;
    int n = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, long_eval_kernel<DH, Tin>, kLT, sizeof(S)) != cudaSuccess)
        return 1;
    return n;
}

template <int DH, typename Tin>
cudaError_t launch_eval(Ctx &c, const LongArgs &A, unsigned grid, cudaStream_t s) {
    using S = LongSmem<DH>;
    static_assert(sizeof(S) <= 227 * 1024, "long-unit kernel shared memory above the per-CTA limit");
    const size_t sm = sizeof(S);
    cudaError_t e = cudaFuncSetAttribute(long_eval_kernel<DH, Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)sm);
    if (e != cudaSuccess) return e;
    long_eval_kernel<DH, Tin><<<grid, kLT, sm, s>>>(A);
    c.launches += 1;
    return cudaGetLastError();
}

__global__ void long_units_kernel(const int32_t *long_slots, int n_long, int lg0, int nlg, int J, int32_t *out) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= n_long * nlg) return;
    const int q = k / nlg, i = k - q * nlg;
    out[k] = (lg0 + i) * J + long_slots[q];
}

}  // namespace

size_t long_res_bytes() { return sizeof(LongRes); }

cudaError_t launch_long_units(Ctx &c, const int32_t *long_slots, int n_long, int lg0, int nlg, int J,
                              int32_t *out, cudaStream_t s) {
    const int n = n_long * nlg;
    if (n <= 0) return cudaSuccess;
    long_units_kernel<<<(n + 255) / 256, 256, 0, s>>>(long_slots, n_long, lg0, nlg, J, out);
    c.launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_long_level(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                              const int32_t *slots, int J, int fresh, int root_only, float tau,
                              const int32_t *list, int n_list, int lg0, int nlg, cudaStream_t s,
                              unsigned int *n_items_host, float tau_prune) {
    const gkv_params &p = c.p;
    Workspace &w = c.w;
    if (nlg < 0) nlg = p.L * p.G - lg0;
    const int64_t n_units = fresh ? (int64_t)n_list * nlg : (int64_t)n_list;
    if (n_items_host) *n_items_host = 0;
    if (n_units <= 0) return cudaSuccess;
    if (n_units > w.long_units_cap) return cudaErrorInvalidValue;
    LongArgs A;
    A.K = K; A.V = V; A.Q = Q;
    A.slots = slots; A.rope = w.rope; A.kappa = w.kappa;
    A.rtok = w.rtok; A.row_m = w.row_m; A.row_Z = w.row_Z; A.omega = omega;
    A.Eg = use_tc(c) ? reinterpret_cast<const float2 *>(w.Eg) : nullptr;
    A.fl_acc = p.alpha_floor > 0.0 ? w.fl_acc : nullptr;
    A.fl_f = w.fl_f;
    A.L = p.L; A.G = p.G; A.Hq = p.Hq; A.T = p.T; A.d = p.d; A.W = p.W; A.gq = p.Hq / p.G;
    A.cs = p.ctx_start; A.Nc = c.Nc; A.J = J; A.k_cand = p.k_cand;
    A.inv_sqrt_d = (float)(1.0 / sqrt((double)p.d));
    A.lamZ = (float)p.lambda_Z; A.lamM = (float)p.lambda_M; A.eps = (float)p.eps;
    A.lam_kappa = (float)p.lambda_kappa; A.base_frac = (float)p.base_frac;
    A.fresh = fresh; A.root_only = root_only; A.tau = tau;
    A.list = list; A.n_list = n_list; A.lg0 = lg0; A.nlg = nlg;
    A.it_gv = w.long_gv; A.it_uid = w.long_uid; A.it_kin = w.long_kin; A.it_ufl = w.long_ufl;
    A.res = static_cast<LongRes *>(w.long_res);
    A.u_start = w.long_start; A.u_cnt = w.long_cnt; A.n_items = w.long_n; A.cap_items = w.long_cap;
    A.nd_a = w.nd_a; A.nd_b = w.nd_b; A.nd_child0 = w.nd_child0; A.nd_parent = w.nd_parent;
    A.nd_unit = w.nd_unit; A.nd_nchild = w.nd_nchild; A.nd_cost = w.nd_cost;
    A.nd_D = w.nd_D; A.nd_R = w.nd_R; A.nd_U = w.nd_U; A.nd_kappa = w.nd_kappa; A.nd_sel = w.nd_sel;
    A.ops = w.ops; A.n_ops = w.n_ops;
    A.u_nnodes = w.u_nnodes; A.u_Uadd = w.u_Uadd; A.u_Ddrop = w.u_Ddrop; A.u_pend = w.u_pend;
    A.u_sel = w.u_sel;
    A.status = w.dev_int + 1;
    A.work = w.work;
    A.sub = w.long_sub;
    A.it_next = w.long_n + 3;
    cudaError_t e = cudaMemsetAsync(w.long_n, 0, 4 * sizeof(unsigned int), s);
    if (e != cudaSuccess) return e;
    long_collect_kernel<<<(unsigned)n_units, kLT, 0, s>>>(A);
    c.launches += 1;
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // the level's counts: long work items, small subtrees of each class
    unsigned int cnt[3] = {0, 0, 0};
    e = cudaMemcpyAsync(cnt, w.long_n, sizeof cnt, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return e;
    for (int q = 0; q < 3; q++) cnt[q] = (unsigned)std::min<int64_t>((int64_t)cnt[q], w.long_cap);
    if (n_items_host) *n_items_host = cnt[0] + cnt[1] + cnt[2];
    if (cnt[0] > 0) {
        // one resident wave: items are taken dynamically
        int occ = 1;
        if (p.d == 128) occ = p.dtype == GKV_BF16 ? eval_occupancy<128, __nv_bfloat16>() : eval_occupancy<128, float>();
        else occ = p.dtype == GKV_BF16 ? eval_occupancy<64, __nv_bfloat16>() : eval_occupancy<64, float>();
        const unsigned grid = (unsigned)std::min<int64_t>((int64_t)c.num_sms * std::max(occ, 1), (int64_t)cnt[0]);
        e = p.dtype == GKV_BF16
                ? (p.d == 128 ? launch_eval<128, __nv_bfloat16>(c, A, grid, s) : launch_eval<64, __nv_bfloat16>(c, A, grid, s))
                : (p.d == 128 ? launch_eval<128, float>(c, A, grid, s) : launch_eval<64, float>(c, A, grid, s));
        if (e != cudaSuccess) return e;
        long_commit_kernel<<<(unsigned)n_units, 32, 0, s>>>(A);
        c.launches += 1;
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    // nodes of at most kMaxUnit tokens: their subtrees on the unit kernel
    return launch_unit_subtrees(c, K, V, Q, omega, slots, J, w.long_sub, (int)cnt[1], w.long_sub + w.long_cap,
                                (int)cnt[2], tau_prune, s);
}

}  // namespace gkv
