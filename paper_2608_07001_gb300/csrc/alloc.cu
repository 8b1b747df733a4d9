// alloc.cu -- stage 3 of the GraceKV pass: global greedy Add/Split allocation
// (App. A.5 Stage II, App. C.3), computed on the device without a priority
// queue.
//
// The heap of the paper pops ops in non-increasing order of their bottleneck
// key kappa(op) = min(U(op), kappa(op that exposed it)) (kappa(Add) = U(Add)):
// an op is exposed only after its creator, and a child whose U exceeds its
// creator's key is popped right after it.  Hence, with tau the cost-weighted
// threshold cost{kappa > tau} <= B_free < cost{kappa >= tau}:
//   1. every op with kappa > tau is executed (they fit and are
//      prerequisite-closed, since kappa never increases down a path);
//   2. ops with kappa == tau are executed in the heap's order, which visits
//      units in ascending order and, inside a unit, follows the unit's own
//      queue (U desc, a asc, b desc); an op that does not fit the remaining
//      budget is discarded with its subtree (App. C.3);
//   3. if one budget unit is left, the best exposed cost-1 op under the heap's
//      order (U desc, unit asc, a asc, b desc) takes it.
// Ties in U are therefore resolved exactly as the heap resolves them.
//
// With fixed per-(l, g) capacities (the "w/o GA" ablation, App. C.1) the heap
// decomposes into one independent heap per (l, g) with budget
// floor(B_free / LG) (+1 for the first B_free mod LG pairs): every step above
// then runs per (l, g) "segment", each with its own state words and histogram
// (nseg = LG; nseg = 1 is the shared budget).
//
// The ops are the Add of every unit and the Split ops of the compact list the
// unit kernel appends to as it evaluates nodes.
// Kernels: alloc_hist (cost-weighted histogram of the 32-bit keys, three
// passes of 11/11/10 bits), alloc_scan (pick the digit, one block), alloc_mark
// (main set + units holding ties), alloc_ties (one block, units in order),
// alloc_end_max / alloc_end_key / alloc_end_pick (endgame).
#include "gkv_internal.cuh"

#include <algorithm>
#include <cfloat>

namespace gkv {
namespace {

// alloc_state layout (unsigned long long)
enum { ST_PREFIX = 0, ST_ABOVE, ST_ALL, ST_R, ST_ENDU, ST_ENDKEY, ST_TOTAL, ST_USED, ST_CROSS, ST_NTIE, ST_N };
static_assert(ST_N <= 16, "alloc_state holds 16 words per segment");

struct AllocArgs {
    int64_t n_units;
    const uint2 *ops;        // Split ops built so far: (key bits, node index << 1 | cost - 1)
    const unsigned int *n_ops;
    const float *u_U;        // Add keys (kappa = U)
    const float *nd_kappa;
    const int8_t *nd_cost;
    const float *nd_U;
    const int32_t *nd_a, *nd_b, *nd_parent, *nd_unit, *nd_child0;
    const int8_t *nd_nchild;
    const int32_t *u_nnodes;
    const int32_t *slots;
    int J, LG, cs, Nc;
    uint8_t *u_sel, *nd_sel;
    int32_t *u_flag;         // units holding ties (alloc_mark), then their tie state (alloc_tie_scan)
    int64_t *u_tcost;        // cost of each unit's tie closure
    unsigned long long *hist, *st;
    int64_t B_free;
    int *status;
    int nseg;                // 1: one shared budget; L G: a fixed capacity per (l, g)
    const uint8_t *u_floor;  // nullable: slots whose Add is a singleton-floor op (largest key)
};

// State words, histogram and budget of segment seg.  With one segment the
// state sits at st[0 .. ST_N); with per-(l, g) capacities st[0 .. ST_N) holds
// the totals and segment seg uses st[ST_N (1 + seg) ..].
__device__ __forceinline__ unsigned long long *seg_st(const AllocArgs &A, int seg) {
    return A.nseg > 1 ? A.st + ST_N * (1 + seg) : A.st;
}
__device__ __forceinline__ unsigned long long *seg_hist(const AllocArgs &A, int seg) {
    return A.hist + (size_t)2048 * seg;
}
__device__ __forceinline__ long long seg_budget(const AllocArgs &A, int seg) {
    if (A.nseg == 1) return A.B_free;
    return A.B_free / A.nseg + (seg < A.B_free % A.nseg ? 1 : 0);
}
// Segment of op i (unit i for an Add, the unit of node v for a Split).
__device__ __forceinline__ int op_seg(const AllocArgs &A, int64_t i, int64_t v) {
    if (A.nseg == 1) return 0;
    return (int)((v < 0 ? i : (int64_t)A.nd_unit[v]) / A.J);
}

// Op i of the enumeration: the Add of unit i (i < n_units), else Split op
// i - n_units of the compact list; v receives the node index (-1 for an Add).
__device__ __forceinline__ void op_key(const AllocArgs &A, int64_t i, uint32_t &key, int &cost, int64_t &v) {
    if (i < A.n_units) {
        key = (A.u_floor && A.u_floor[i]) ? __float_as_uint(FLT_MAX) : __float_as_uint(A.u_U[i]);
        cost = 1;
        v = -1;
    } else {
        const uint2 o = A.ops[i - A.n_units];
        key = o.x;
        cost = (int)(o.y & 1u) + 1;
        v = (int64_t)(o.y >> 1);
    }
    const float x = __uint_as_float(key);
    if (!(x >= 0.f) || isinf(x)) atomicOr(A.status, 8);
}

__global__ void alloc_hist_kernel(AllocArgs A, int shift, int nbits, uint32_t mask) {
    __shared__ unsigned int sh[2048];
    const int nbin = 1 << nbits;
    for (int b = threadIdx.x; b < nbin; b += blockDim.x) sh[b] = 0;
    __syncthreads();
    const uint32_t prefix = (uint32_t)A.st[ST_PREFIX];
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t w0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
    unsigned int tot = 0;
    // whole warps consume items together so that equal bins are combined first
    // (keys cluster in few bins: one shared atomic per distinct bin and warp)
    auto consume = [&](bool op, uint32_t key, int cost) {
        tot += op ? cost : 0;
        const int bin = op && (key & mask) == prefix ? (int)((key >> shift) & (nbin - 1)) : -1;
        const unsigned grp = __match_any_sync(0xffffffffu, bin);
        const unsigned sum = __reduce_add_sync(grp, (unsigned)(op ? cost : 0));
        if (bin >= 0 && lane == __ffs(grp) - 1) atomicAdd(&sh[bin], sum);
    };
    for (int64_t i0 = w0; i0 < A.n_units; i0 += stride) {   // Add ops, cost 1
        const int64_t i = i0 + lane;
        const bool in = i < A.n_units;
        const float x = in ? ((A.u_floor && A.u_floor[i]) ? FLT_MAX : A.u_U[i]) : 0.f;
        if (in && (!(x >= 0.f) || isinf(x))) atomicOr(A.status, 8);
        consume(in, __float_as_uint(x), 1);
    }
    // Split ops of the compact list
    const int64_t nops = *A.n_ops;
    for (int64_t i0 = w0; i0 < nops; i0 += stride) {
        const int64_t i = i0 + lane;
        const bool in = i < nops;
        const uint2 o = in ? A.ops[i] : make_uint2(0u, 0u);
        const float x = __uint_as_float(o.x);
        if (in && (!(x >= 0.f) || isinf(x))) atomicOr(A.status, 8);
        consume(in, o.x, (int)(o.y & 1u) + 1);
    }
    __syncthreads();
    for (int b = threadIdx.x; b < nbin; b += blockDim.x)
        if (sh[b]) atomicAdd(&A.hist[b], (unsigned long long)sh[b]);
    if (shift == 21) {   // first pass: total cost of all ops
        tot = __reduce_add_sync(0xffffffffu, tot);
        if (lane == 0 && tot) atomicAdd(&A.st[ST_TOTAL], (unsigned long long)tot);
    }
}

// The same histogram per segment (per-(l, g) capacities): global atomics,
// combined per warp over equal (segment, bin) pairs.
__global__ void alloc_hist_seg_kernel(AllocArgs A, int shift, int nbits, uint32_t mask) {
    const int nbin = 1 << nbits;
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t w0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
    const int64_t n = A.n_units + *A.n_ops;
    for (int64_t i0 = w0; i0 < n; i0 += stride) {
        const int64_t i = i0 + lane;
        const bool in = i < n;
        uint32_t key = 0;
        int cost = 0;
        int64_t v = -1;
        int seg = 0;
        if (in) {
            op_key(A, i, key, cost, v);
            seg = op_seg(A, i, v);
        }
        unsigned long long *st = seg_st(A, seg);
        const uint32_t prefix = in ? (uint32_t)st[ST_PREFIX] : 0u;
        const int bin = in && (key & mask) == prefix ? (int)((key >> shift) & (nbin - 1)) : -1;
        const long long tag = bin >= 0 ? ((long long)seg << 11) | bin : -1;
        const unsigned grp = __match_any_sync(0xffffffffu, tag);
        const unsigned sum = __reduce_add_sync(grp, (unsigned)(bin >= 0 ? cost : 0));
        if (bin >= 0 && lane == __ffs(grp) - 1) atomicAdd(seg_hist(A, seg) + bin, (unsigned long long)sum);
        if (shift == 21) {   // first pass: total cost per segment
            const int stag = in ? seg : -1;
            const unsigned g2 = __match_any_sync(0xffffffffu, stag);
            const unsigned tot = __reduce_add_sync(g2, (unsigned)(in ? cost : 0));
            if (in && lane == __ffs(g2) - 1) atomicAdd(&st[ST_TOTAL], (unsigned long long)tot);
        }
    }
}

// Pick the digit of this pass: scanning bins from the top, the bin where the
// cost of higher keys first exceeds the budget.  One block of 1024 threads
// per segment; thread t owns bins nbin-1-2t and nbin-2-2t.
__global__ void __launch_bounds__(1024) alloc_scan_kernel(AllocArgs A, int shift, int nbits) {
    __shared__ unsigned long long wsum[32];
    const int nbin = 1 << nbits;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int seg = blockIdx.x;
    unsigned long long *st = seg_st(A, seg), *hist = seg_hist(A, seg);
    const unsigned long long B = (unsigned long long)seg_budget(A, seg);
    const bool all = (shift == 21) ? (st[ST_TOTAL] <= B) : (st[ST_ALL] != 0);
    const int b0 = nbin - 1 - 2 * tid, b1 = b0 - 1;
    unsigned long long h0 = b0 >= 0 ? hist[b0] : 0ull, h1 = b1 >= 0 ? hist[b1] : 0ull;
    // exclusive scan of (h0 + h1) over threads, in descending bin order
    unsigned long long x = h0 + h1, incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        unsigned long long v = wsum[lane], iv = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            unsigned long long y = __shfl_up_sync(0xffffffffu, iv, o);
            if (lane >= o) iv += y;
        }
        wsum[lane] = iv - v;   // exclusive prefix of warp totals
    }
    __syncthreads();
    const unsigned long long above = st[ST_ABOVE];
    const unsigned long long before = above + wsum[warp] + (incl - x);
    __syncthreads();
    if (all) {
        if (tid == 0 && shift == 21) st[ST_ALL] = 1;
    } else {
        // the crossing bin is unique: above + cost(higher bins) <= B < ... + h
        if (b0 >= 0 && before <= B && before + h0 > B) {
            st[ST_PREFIX] |= ((unsigned long long)b0 << shift);
            st[ST_ABOVE] = before;
        } else if (b1 >= 0 && before + h0 <= B && before + h0 + h1 > B) {
            st[ST_PREFIX] |= ((unsigned long long)b1 << shift);
            st[ST_ABOVE] = before + h0;
        }
    }
    if (b0 >= 0) hist[b0] = 0;
    if (b1 >= 0) hist[b1] = 0;
}

// Main set (kappa > tau, or everything when it fits) and units holding ties.
__global__ void alloc_mark_kernel(AllocArgs A) {
    const int64_t n = A.n_units + *A.n_ops;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t key;
        int cost;
        int64_t v;
        op_key(A, i, key, cost, v);
        const unsigned long long *st = seg_st(A, op_seg(A, i, v));
        const bool all = st[ST_ALL] != 0;
        const uint32_t tau = (uint32_t)st[ST_PREFIX];
        uint8_t s = (all || key > tau) ? 1 : 0;
        if (v < 0) {
            A.u_sel[i] = s;
            if (!all && key == tau) A.u_flag[i] = 1;
        } else {
            A.nd_sel[v] = s;
            if (!all && key == tau) A.u_flag[A.nd_unit[v]] = 1;
        }
    }
}

// ---------------------------------------------------------------------------
// Ties (ops whose key equals tau).  The heap takes them unit by unit in
// ascending unit order, each unit's in its own heap order, while budget is
// left.  A unit whose tie ops all fit executes every tie op reachable from
// the main set (its tie closure), so:
//   alloc_tie_cost   every unit's closure and its cost, in parallel (a
//                    closure op is marked 3; parents precede children in a
//                    unit's node order, so one pass in that order suffices)
//   alloc_tie_scan   per segment, the ordered prefix of the costs: units
//                    whose closure fits select it whole, the first that does
//                    not is the crossing unit, with the budget left for it
//   alloc_tie_apply  the closures of the units before it selected (3 -> 1),
//                    the others cleared (3 -> 0)
//   alloc_ties       the crossing unit and the ones after it, while budget is
//                    left, replayed op by op (block-wide argmax per pop).
// ---------------------------------------------------------------------------
__global__ void alloc_tie_cost_kernel(AllocArgs A) {
    const int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= A.n_units) return;
    int64_t cost = 0;
    if (A.u_flag[u]) {
        const unsigned long long *st = seg_st(A, A.nseg > 1 ? (int)(u / A.J) : 0);
        const uint32_t tau = (uint32_t)st[ST_PREFIX];
        const int lg = (int)(u / A.J), j = (int)(u - (int64_t)lg * A.J);
        const int64_t nb = node_base(lg, A.slots[j], A.cs, A.Nc);
        const bool addtie = A.u_sel[u] == 0 && !(A.u_floor && A.u_floor[u]) && __float_as_uint(A.u_U[u]) == tau;
        if (addtie) { A.u_sel[u] = 3; cost += 1; }
        const bool root_open = A.u_sel[u] == 1 || A.u_sel[u] == 3;
        const int nn = A.u_nnodes[u];
        for (int k = 0; k < nn; k++) {
            const int64_t v = nb + k;
            if (A.nd_cost[v] <= 0 || A.nd_sel[v] != 0 || __float_as_uint(A.nd_kappa[v]) != tau) continue;
            const int32_t pg = A.nd_parent[v];
            const bool open = pg < 0 ? root_open : (A.nd_sel[pg] == 1 || A.nd_sel[pg] == 3);
            if (!open) continue;
            A.nd_sel[v] = 3;
            cost += A.nd_cost[v];
        }
    }
    A.u_tcost[u] = cost;
    if (cost > 0) atomicAdd(&seg_st(A, A.nseg > 1 ? (int)(u / A.J) : 0)[ST_NTIE], 1ull);
}

// Ordered scan of the closure costs per segment, in three steps over chunks
// of 1024 units (chunk c of segment seg covers units u_lo + 1024 c ..):
// chunk sums, an exclusive scan of a segment's chunk sums, then each unit's
// state -- 1: its whole closure fits, 2: the crossing unit (ST_CROSS, with the
// budget left for it in ST_R), 0: otherwise.
constexpr int kTieChunk = 1024;
__device__ __forceinline__ void seg_units(const AllocArgs &A, int seg, int64_t &u_lo, int64_t &u_hi) {
    u_lo = A.nseg > 1 ? (int64_t)seg * A.J : 0;
    u_hi = A.nseg > 1 ? u_lo + A.J : A.n_units;
}
__device__ __forceinline__ long long block_incl_scan(long long c, long long *wsum, long long &total) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    long long incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    long long before = 0;
    total = 0;
    for (int w = 0; w < 32; w++) {
        if (w < warp) before += wsum[w];
        total += wsum[w];
    }
    __syncthreads();
    return before + incl;
}

// grid (chunks per segment, segments)
__global__ void __launch_bounds__(kTieChunk) alloc_tie_bsum_kernel(AllocArgs A, long long *bsum, int nch) {
    __shared__ long long wsum[32];
    const int seg = blockIdx.y, c = blockIdx.x;
    const unsigned long long *st = seg_st(A, seg);
    if (st[ST_ALL] || st[ST_NTIE] == 0) return;
    int64_t u_lo, u_hi;
    seg_units(A, seg, u_lo, u_hi);
    const int64_t u = u_lo + (int64_t)c * kTieChunk + threadIdx.x;
    long long tot;
    block_incl_scan(u < u_hi ? (long long)A.u_tcost[u] : 0, wsum, tot);
    if (threadIdx.x == 0) bsum[(size_t)seg * nch + c] = tot;
}

// one block per segment: exclusive prefix of its chunk sums
__global__ void __launch_bounds__(kTieChunk) alloc_tie_bscan_kernel(AllocArgs A, long long *bsum, int nch) {
    __shared__ long long wsum[32];
    __shared__ long long carry;
    const int seg = blockIdx.x;
    unsigned long long *st = seg_st(A, seg);
    if (st[ST_ALL]) return;
    const long long R = seg_budget(A, seg) - (long long)st[ST_ABOVE];
    if (st[ST_NTIE] == 0) {   // no tie op is exposed: nothing to order
        if (threadIdx.x == 0) st[ST_R] = (unsigned long long)R;
        return;
    }
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    long long *b = bsum + (size_t)seg * nch;
    for (int c0 = 0; c0 < nch; c0 += kTieChunk) {
        const int c = c0 + threadIdx.x;
        const long long x = c < nch ? b[c] : 0;
        long long tot;
        const long long incl = block_incl_scan(x, wsum, tot);
        if (c < nch) b[c] = carry + incl - x;
        __syncthreads();
        if (threadIdx.x == 0) carry += tot;
        __syncthreads();
    }
    if (threadIdx.x == 0 && carry <= R) st[ST_R] = (unsigned long long)(R - carry);   // every closure fits
}

// grid (chunks per segment, segments): each unit's state and the crossing unit
__global__ void __launch_bounds__(kTieChunk) alloc_tie_scan_kernel(AllocArgs A, const long long *bsum, int nch) {
    __shared__ long long wsum[32];
    const int seg = blockIdx.y, c = blockIdx.x;
    unsigned long long *st = seg_st(A, seg);
    if (st[ST_ALL] || st[ST_NTIE] == 0) return;
    const long long R = seg_budget(A, seg) - (long long)st[ST_ABOVE];
    int64_t u_lo, u_hi;
    seg_units(A, seg, u_lo, u_hi);
    const int64_t u = u_lo + (int64_t)c * kTieChunk + threadIdx.x;
    const long long cost = u < u_hi ? (long long)A.u_tcost[u] : 0;
    long long tot;
    const long long hi = bsum[(size_t)seg * nch + c] + block_incl_scan(cost, wsum, tot), lo = hi - cost;
    if (u < u_hi) {
        int state = 0;
        if (cost > 0 && hi <= R) state = 1;                 // its whole closure fits
        else if (cost > 0 && lo <= R && hi > R) {           // the crossing unit (at most one)
            state = 2;
            st[ST_CROSS] = (unsigned long long)u;
            st[ST_R] = (unsigned long long)(R - lo);
        }
        A.u_flag[u] = state;
    }
}

__global__ void alloc_tie_apply_kernel(AllocArgs A) {
    const int64_t n = A.n_units + *A.n_ops;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        if (i < A.n_units) {
            if (A.u_sel[i] == 3) A.u_sel[i] = A.u_flag[i] == 1 ? 1 : 0;
        } else {
            const int64_t v = (int64_t)(A.ops[i - A.n_units].y >> 1);
            if (A.nd_sel[v] == 3) A.nd_sel[v] = A.u_flag[A.nd_unit[v]] == 1 ? 1 : 0;
        }
    }
}

// Node index base of unit uid.
__device__ __forceinline__ int64_t unit_base(const AllocArgs &A, int64_t uid) {
    int lg = (int)(uid / A.J), j = (int)(uid - (int64_t)lg * A.J);
    return node_base(lg, A.slots[j], A.cs, A.Nc);
}

// One block per segment: from its crossing unit on, while budget is left,
// each unit holding ties is replayed with its own queue restricted to tie ops
// (U descending, then the node's position ascending and length descending);
// each pop is a block-wide argmax over the unit's nodes.  An op costing more
// than the budget left is discarded (2): its subtree is never exposed.
__global__ void __launch_bounds__(1024) alloc_ties_kernel(AllocArgs A) {
    __shared__ unsigned long long wk[32];
    __shared__ int wi[32];
    __shared__ long long Rs;
    __shared__ unsigned long long bkey;
    __shared__ int bidx;
    const int seg = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned long long *st = seg_st(A, seg);
    if (st[ST_ALL]) {
        if (tid == 0) st[ST_R] = 0, st[ST_USED] = st[ST_TOTAL];
        return;
    }
    if (st[ST_CROSS] == ~0ull) return;   // every tie closure fit (alloc_tie_scan set ST_R)
    const uint32_t tau = (uint32_t)st[ST_PREFIX];
    const int64_t u_hi = A.nseg > 1 ? (int64_t)seg * A.J + A.J : A.n_units;
    if (tid == 0) Rs = (long long)st[ST_R];
    __syncthreads();
    for (int64_t u = (int64_t)st[ST_CROSS]; u < u_hi && Rs > 0; u++) {
        if (A.u_tcost[u] <= 0) continue;            // no tie op exposed in this unit
        const int lg = (int)(u / A.J), j = (int)(u - (int64_t)lg * A.J);
        const int sa = A.slots[j];
        const int64_t nb = node_base(lg, sa, A.cs, A.Nc);
        const int nn = A.u_nnodes[u];
        for (;;) {
            // key: U bits (32) | 2^15 - 1 - (a - sa) (15) | b - a (15); -1 node: the Add
            unsigned long long best = 0ull;
            int bi = -2;
            if (tid == 0 && A.u_sel[u] == 0 && !(A.u_floor && A.u_floor[u]) &&
                __float_as_uint(A.u_U[u]) == tau) {
                best = ((unsigned long long)__float_as_uint(A.u_U[u]) << 32) |
                       ((unsigned long long)(32767u) << 15) | (unsigned long long)(A.nd_b[nb] - A.nd_a[nb]);
                bi = -1;
            }
            for (int k = tid; k < nn; k += 1024) {
                const int64_t v = nb + k;
                if (A.nd_cost[v] <= 0 || A.nd_sel[v] != 0 || __float_as_uint(A.nd_kappa[v]) != tau) continue;
                const int32_t pg = A.nd_parent[v];
                const bool exposed = pg < 0 ? A.u_sel[u] == 1 : A.nd_sel[pg] == 1;
                if (!exposed) continue;
                const unsigned long long key = ((unsigned long long)__float_as_uint(A.nd_U[v]) << 32) |
                                               ((unsigned long long)(32767u - (uint32_t)(A.nd_a[v] - sa)) << 15) |
                                               (unsigned long long)(A.nd_b[v] - A.nd_a[v]);
                if (bi == -2 || key > best) { best = key; bi = k; }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const unsigned long long k2 = __shfl_xor_sync(0xffffffffu, best, o);
                const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
                if (i2 != -2 && (bi == -2 || k2 > best)) { best = k2; bi = i2; }
            }
            if (lane == 0) { wk[warp] = best; wi[warp] = bi; }
            __syncthreads();
            if (tid == 0) {
                unsigned long long b = 0ull;
                int ix = -2;
                for (int w = 0; w < 32; w++)
                    if (wi[w] != -2 && (ix == -2 || wk[w] > b)) { b = wk[w]; ix = wi[w]; }
                bkey = b;
                bidx = ix;
                if (ix != -2) {
                    const int cost = ix == -1 ? 1 : A.nd_cost[nb + ix];
                    const uint8_t sv = cost > Rs ? 2 : 1;   // 2 = discarded (subtree never exposed)
                    if (sv == 1) Rs -= cost;
                    if (ix == -1) A.u_sel[u] = sv;
                    else A.nd_sel[nb + ix] = sv;
                }
            }
            __syncthreads();
            if (bidx == -2 || Rs <= 0) break;
        }
    }
    if (tid == 0) st[ST_R] = (unsigned long long)Rs;
}

// Endgame: when exactly one budget unit is left, the best exposed cost-1 op.
__device__ __forceinline__ bool end_cand(const AllocArgs &A, int64_t i, float &U,
                                         unsigned long long &key) {
    if (i < A.n_units) {
        if (A.u_sel[i] != 0) return false;
        int64_t nb = unit_base(A, i);
        U = A.u_U[i];
        int a = A.nd_a[nb], b = A.nd_b[nb];
        key = ((unsigned long long)i << 37) | ((unsigned long long)a << 17) | (0x1FFFFull - (unsigned)(b - a));
        return true;
    }
    const int64_t v = (int64_t)(A.ops[i - A.n_units].y >> 1);
    if (A.nd_cost[v] != 1 || A.nd_sel[v] != 0) return false;
    int32_t p = A.nd_parent[v];
    bool exposed = p < 0 ? A.u_sel[-2 - p] == 1 : A.nd_sel[p] == 1;
    if (!exposed) return false;
    U = A.nd_U[v];
    int a = A.nd_a[v], b = A.nd_b[v];
    key = ((unsigned long long)A.nd_unit[v] << 37) | ((unsigned long long)a << 17) |
          (0x1FFFFull - (unsigned)(b - a));
    return true;
}

// Segment of endgame candidate i (its unit's (l, g) with per-pair capacities).
__device__ __forceinline__ int end_seg(const AllocArgs &A, int64_t i) {
    if (A.nseg == 1) return 0;
    return op_seg(A, i, i < A.n_units ? -1 : (int64_t)(A.ops[i - A.n_units].y >> 1));
}

__global__ void alloc_end_max_kernel(AllocArgs A) {
    const int64_t n = A.n_units + *A.n_ops;
    if (A.nseg == 1 && A.st[ST_R] != 1) return;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        unsigned long long *st = seg_st(A, end_seg(A, i));
        if (st[ST_R] != 1) continue;
        float U;
        unsigned long long k;
        if (!end_cand(A, i, U, k)) continue;
        const unsigned b = __float_as_uint(U) + 1u;     // +1: distinguish "no candidate" (0)
        if (b > (unsigned)st[ST_ENDU]) atomicMax(&st[ST_ENDU], (unsigned long long)b);
    }
}

__global__ void alloc_end_key_kernel(AllocArgs A) {
    const int64_t n = A.n_units + *A.n_ops;
    if (A.nseg == 1 && (A.st[ST_R] != 1 || A.st[ST_ENDU] == 0)) return;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        unsigned long long *st = seg_st(A, end_seg(A, i));
        if (st[ST_R] != 1 || st[ST_ENDU] == 0) continue;
        float U;
        unsigned long long k;
        if (!end_cand(A, i, U, k)) continue;
        if (__float_as_uint(U) != (unsigned)st[ST_ENDU] - 1u) continue;
        if (k < st[ST_ENDKEY]) atomicMin(&st[ST_ENDKEY], k);
    }
}

__global__ void alloc_end_pick_kernel(AllocArgs A) {
    const int64_t n = A.n_units + *A.n_ops;
    if (A.nseg == 1 && (A.st[ST_R] != 1 || A.st[ST_ENDU] == 0)) return;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const unsigned long long *st = seg_st(A, end_seg(A, i));
        if (st[ST_R] != 1 || st[ST_ENDU] == 0) continue;
        float U;
        unsigned long long k;
        if (!end_cand(A, i, U, k)) continue;
        if (k != st[ST_ENDKEY] || __float_as_uint(U) + 1u != (unsigned)st[ST_ENDU]) continue;
        if (i < A.n_units) A.u_sel[i] = 1;
        else A.nd_sel[A.ops[i - A.n_units].y >> 1] = 1;
    }
}

// Budget left and used per segment; with per-pair capacities the totals add
// up into st[ST_USED].
__global__ void alloc_final_kernel(AllocArgs A) {
    for (int seg = blockIdx.x * blockDim.x + threadIdx.x; seg < A.nseg; seg += gridDim.x * blockDim.x) {
        unsigned long long *st = seg_st(A, seg);
        long long R = (long long)st[ST_R];
        if (!st[ST_ALL] && R == 1 && st[ST_ENDU] != 0) R = 0;
        st[ST_R] = (unsigned long long)R;
        if (!st[ST_ALL]) st[ST_USED] = (unsigned long long)(seg_budget(A, seg) - R);
        if (A.nseg > 1) atomicAdd(&A.st[ST_USED], st[ST_USED]);
    }
}

__global__ void alloc_init_kernel(unsigned long long *st, unsigned long long *hist, int nseg) {
    const int nst = ST_N * (nseg > 1 ? nseg + 1 : 1);
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nst; i += gridDim.x * blockDim.x)
        st[i] = (i % ST_N == ST_ENDKEY || i % ST_N == ST_CROSS) ? ~0ull : 0ull;
    for (int64_t b = blockIdx.x * blockDim.x + threadIdx.x; b < (int64_t)2048 * nseg; b += gridDim.x * blockDim.x)
        hist[b] = 0;
}


AllocArgs make_args(Ctx &c, int J) {
    Workspace &w = c.w;
    AllocArgs A;
    A.n_units = (int64_t)c.p.L * c.p.G * J;
    A.ops = w.ops; A.n_ops = w.n_ops;
    A.u_U = w.u_Uadd; A.nd_kappa = w.nd_kappa; A.nd_cost = w.nd_cost; A.nd_U = w.nd_U;
    A.nd_a = w.nd_a; A.nd_b = w.nd_b; A.nd_parent = w.nd_parent; A.nd_unit = w.nd_unit;
    A.nd_child0 = w.nd_child0; A.nd_nchild = w.nd_nchild; A.u_nnodes = w.u_nnodes;
    A.slots = w.slots;
    A.J = J; A.LG = c.p.L * c.p.G; A.cs = c.p.ctx_start; A.Nc = c.Nc;
    A.u_sel = w.u_sel; A.nd_sel = w.nd_sel; A.u_flag = w.u_count;
    A.u_tcost = w.u_off;     // scratch until the gather writes the entry offsets
    A.hist = w.hist; A.st = w.alloc_state; A.B_free = c.B_free; A.status = w.dev_int + 1;
    A.nseg = c.p.quota_alloc ? c.p.L * c.p.G : 1;
    A.u_floor = c.p.alpha_floor > 0.0 ? w.u_floor : nullptr;
    return A;
}

int grid_for(const Ctx &c, int64_t n) {
    int blocks = (int)std::min<int64_t>((n + 255) / 256, (int64_t)c.num_sms * 8);
    return blocks < 1 ? 1 : blocks;
}

// Units with a pending node whose creator key is >= tau (all of them when
// every op built so far fits the budget).
__global__ void prune_list_kernel(const float *u_pend, const int32_t *slots, int J, int64_t n_units,
                                  const unsigned long long *st, const float *cut, int32_t *list,
                                  int *count, int32_t *long_list, unsigned long long *potential) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n_units) return;
    float p = u_pend[i];
    if (!(p >= 0.f)) return;   // -1: no pending node
    const bool all = st[ST_ALL] != 0;
    const bool above = all || __float_as_uint(p) >= (uint32_t)st[ST_PREFIX];
    if (above) {   // cost of expanding the unit completely: n - 1 entries at most
        const int j = (int)(i % J);
        atomicAdd(potential, (unsigned long long)(slots[j + 1] - slots[j] - 1));
    }
    if (above && p >= *cut) {
        const int j = (int)(i % J);
        const int n = slots[j + 1] - slots[j];
        if (n <= kShortUnit) list[atomicAdd(count, 1)] = (int32_t)i;
        else if (n <= kMaxUnit) list[n_units - 1 - atomicAdd(count + 1, 1)] = (int32_t)i;
        else long_list[atomicAdd(count + 2, 1)] = (int32_t)i;
    }
}

// Histogram (top 16 bits of the non-negative float keys) of the largest
// pending key bound of every unit that reaches the threshold.
constexpr int kPendBins = 1 << 16;
__global__ void pend_hist_kernel(const float *u_pend, int64_t n_units, const unsigned long long *st,
                                 unsigned int *hist) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n_units) return;
    const float p = u_pend[i];
    if (!(p >= 0.f)) return;
    const bool all = st[ST_ALL] != 0;
    if (all || __float_as_uint(p) >= (uint32_t)st[ST_PREFIX]) atomicAdd(&hist[__float_as_uint(p) >> 16], 1u);
}

// One block of 1024 threads: thread t owns the 64 bins below kPendBins - 64 t;
// the bin where the count of larger-or-equal bounds first reaches m gives the cut.
__global__ void __launch_bounds__(1024) pend_cut_kernel(const unsigned int *hist, int m, float *cut,
                                                        unsigned int *n_qual) {
    __shared__ unsigned int wsum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int hi = kPendBins - 64 * tid;   // bins [hi - 64, hi), descending
    unsigned int own = 0;
    for (int b = hi - 1; b >= hi - 64; b--) own += hist[b];
    unsigned int incl = own;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        unsigned int w = wsum[lane], wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        wsum[lane] = wi - w;   // exclusive over warps
    }
    __syncthreads();
    const unsigned int before = wsum[warp] + incl - own;   // bounds in bins >= hi
    if (tid == 1023) *n_qual = before + own;
    if (before < (unsigned)m && before + own >= (unsigned)m) {
        unsigned int acc = before;
        for (int b = hi - 1; b >= hi - 64; b--) {
            acc += hist[b];
            if (acc >= (unsigned)m) { *cut = __uint_as_float((unsigned)b << 16); break; }
        }
    }
    if (tid == 1023 && before + own < (unsigned)m) *cut = -INFINITY;   // fewer than m qualify: no cut
}

__global__ void slot_classes_kernel(const int32_t *slots, int J, int32_t *list, int *count,
                                    int32_t *long_slots) {
    int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= J) return;
    const int n = slots[j + 1] - slots[j];
    if (n <= kShortUnit) list[atomicAdd(count, 1)] = j;
    else if (n <= kMaxUnit) list[J - 1 - atomicAdd(count + 1, 1)] = j;
    else {
        long_slots[atomicAdd(count + 2, 1)] = j;
        atomicAdd(count + 3, n);
    }
}

}  // namespace

cudaError_t launch_threshold(Ctx &c, int J, cudaStream_t s) {
    AllocArgs A = make_args(c, J);
    alloc_init_kernel<<<A.nseg > 1 ? 256 : 1, 256, 0, s>>>(c.w.alloc_state, c.w.hist, A.nseg);
    const int blocks = grid_for(c, A.n_units + c.node_cap / 2);
    const int shifts[3] = {21, 10, 0};
    const int bits[3] = {11, 11, 10};
    uint32_t mask = 0;
    for (int ps = 0; ps < 3; ps++) {
        if (A.nseg > 1)
            alloc_hist_seg_kernel<<<blocks, 256, 0, s>>>(A, shifts[ps], bits[ps], mask);
        else
            alloc_hist_kernel<<<blocks, 256, 0, s>>>(A, shifts[ps], bits[ps], mask);
        alloc_scan_kernel<<<A.nseg, 1024, 0, s>>>(A, shifts[ps], bits[ps]);
        mask |= ((1u << bits[ps]) - 1u) << shifts[ps];
    }
    c.launches += 7;
    return cudaGetLastError();
}

cudaError_t launch_prune_list(Ctx &c, const int32_t *slots, int J, int32_t *list, int *count,
                              int32_t *long_list, cudaStream_t s) {
    const int64_t nu = (int64_t)c.p.L * c.p.G * J;
    cudaError_t e = cudaMemsetAsync(count, 0, 3 * sizeof(int), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(c.w.pend_pot, 0, sizeof(unsigned long long), s);
    if (e != cudaSuccess) return e;
    prune_list_kernel<<<(unsigned)((nu + 255) / 256), 256, 0, s>>>(c.w.u_pend, slots, J, nu,
                                                                    c.w.alloc_state, c.w.pend_cut, list,
                                                                    count, long_list, c.w.pend_pot);
    c.launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_pend_cut(Ctx &c, int J, int m, float *cut, unsigned int *n_qual, cudaStream_t s) {
    const int64_t nu = (int64_t)c.p.L * c.p.G * J;
    cudaError_t e = cudaMemsetAsync(c.w.pend_hist, 0, sizeof(unsigned int) * kPendBins, s);
    if (e != cudaSuccess) return e;
    pend_hist_kernel<<<(unsigned)((nu + 255) / 256), 256, 0, s>>>(c.w.u_pend, nu, c.w.alloc_state,
                                                                   c.w.pend_hist);
    pend_cut_kernel<<<1, 1024, 0, s>>>(c.w.pend_hist, m, cut, n_qual);
    c.launches += 2;
    return cudaGetLastError();
}

cudaError_t launch_slot_classes(Ctx &c, const int32_t *slots, int J, int32_t *list, int *count,
                                int32_t *long_slots, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(count, 0, 4 * sizeof(int), s);
    if (e != cudaSuccess) return e;
    slot_classes_kernel<<<(J + 255) / 256, 256, 0, s>>>(slots, J, list, count, long_slots);
    c.launches += 1;
    return cudaGetLastError();
}

cudaError_t launch_allocate(Ctx &c, int J, cudaStream_t s) {
    Workspace &w = c.w;
    AllocArgs A = make_args(c, J);
    cudaMemsetAsync(w.u_count, 0, sizeof(int32_t) * A.n_units, s);
    cudaError_t e = launch_threshold(c, J, s);
    if (e != cudaSuccess) return e;
    const int blocks = grid_for(c, A.n_units + c.node_cap / 2);
    alloc_mark_kernel<<<blocks, 256, 0, s>>>(A);
    alloc_tie_cost_kernel<<<(unsigned)((A.n_units + 255) / 256), 256, 0, s>>>(A);
    {
        const int64_t seg_len = A.nseg > 1 ? (int64_t)J : A.n_units;
        const int nch = (int)((seg_len + kTieChunk - 1) / kTieChunk);
        const dim3 g((unsigned)std::max(nch, 1), (unsigned)A.nseg);
        alloc_tie_bsum_kernel<<<g, kTieChunk, 0, s>>>(A, w.tie_bsum, nch);
        alloc_tie_bscan_kernel<<<A.nseg, kTieChunk, 0, s>>>(A, w.tie_bsum, nch);
        alloc_tie_scan_kernel<<<g, kTieChunk, 0, s>>>(A, w.tie_bsum, nch);
    }
    alloc_tie_apply_kernel<<<blocks, 256, 0, s>>>(A);
    alloc_ties_kernel<<<A.nseg, 1024, 0, s>>>(A);
    alloc_end_max_kernel<<<blocks, 256, 0, s>>>(A);
    alloc_end_key_kernel<<<blocks, 256, 0, s>>>(A);
    alloc_end_pick_kernel<<<blocks, 256, 0, s>>>(A);
    alloc_final_kernel<<<(A.nseg + 255) / 256, 256, 0, s>>>(A);
    c.launches += 11;
    return cudaGetLastError();
}

}  // namespace gkv
