// floor.cu -- the Stage I singleton floor (App. A.5 Stage I, Eqs.
// app_floor_score, app_floor_gate, app_floor_cap; App. C.4), between the
// token values and the tree build.
//
//   f_{l,g,t} = max_{|tau - t| <= 3, tau in C} [(1 - c) R_{l,g,tau} + c mean_{l,g} R_{l,g,tau}]
//
// For every (l, g) the candidates are the tokens in order f descending (ties:
// lower t) that pass the gate f >= gamma / N_c, up to the longest prefix whose
// value sum stays <= eta.  The cap is floor(alpha B_base).  When the joint
// cost C0 of all candidates -- per slot, the frontier size after isolating
// them: |S| + maximal runs outside S -- exceeds it, each (l, g) keeps its first
// max(1, floor(n cap / C0)) candidates; each (l, g) then has the share
// floor(cap n' / sum n') and walks its kept candidates in order, accepting
// each one whose complete path still fits the share and skipping the others
// (App. A.5 Stage I: a candidate is accepted only when its path remains
// feasible).  The tree build then extracts every accepted position as a
// singleton (forced extraction); the floor's ops carry the largest key.
//
// One CTA per (l, g) finds the candidate and kept prefixes with a block-wide
// weighted radix select on the key (~bits(f) << 32 | t): three 11/11/10-bit
// passes over the f part, then an ordered scan over t among the tokens of the
// crossing f.  Token values enter the select as fixed-point integers (2^-40
// units), so the sums are exact and independent of the order of
// accumulation.  The acceptance walk takes the kept candidates 1024 at a time
// in key order (the same select, by count), sorts each chunk in shared
// memory, and one warp walks it against a bitmap of the accepted positions.
#include "gkv_internal.cuh"

#include <cfloat>

namespace gkv {
namespace {

constexpr int kFlThreads = 1024;
constexpr double kFlFix = 1099511627776.0;   // 2^40

struct FloorArgs {
    const float *rtok;        // [LG][Nc]
    const int32_t *slots;     // [J + 1] absolute slot starts
    float *rbar;              // [Nc]
    float *f;                 // [LG][Nc]
    uint8_t *acc;             // [LG][Nc] accepted floor positions
    uint8_t *u_floor;         // [LG J] slots holding an accepted position
    unsigned long long *head; // [LG][kFlHead] per (l, g) state
    unsigned long long *glob; // [4]: C0, sum n', B_floor
    int LG, Nc, J, cs, half;
    float c, gate;
    unsigned long long eta_fx;
    long long cap;
};
enum { FH_CUT = 0, FH_N, FH_COST0, FH_KEEP, FH_CUTK, FH_USED, kFlHead };
enum { FG_C0 = 0, FG_NKEEP, FG_USED };

__device__ __forceinline__ uint64_t fl_key(float f, int t) {
    return ((uint64_t)(~__float_as_uint(f)) << 32) | (uint32_t)t;
}

// Block-wide weighted select over the tokens t in [0, n) whose key is below
// lim: the key cut such that the tokens with key < cut weigh at most budget and
// the token with key == cut would exceed it; ~0 when all of them fit.
// wt(t) is the token's integer weight.  Every thread returns the same cut.
template <class W>
__device__ uint64_t block_wselect(const float *f, int n, uint64_t lim, unsigned long long budget, W wt,
                                  unsigned long long *hist, unsigned long long *wsum, unsigned long long *bc) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // stage 1: the f part of the key, 11 / 11 / 10 bits from the top
    uint32_t prefix = 0, mask = 0;
    unsigned long long below = 0;
    const int shifts[3] = {21, 10, 0}, bits[3] = {11, 11, 10};
    bool all_fit = false;
    for (int ps = 0; ps < 3; ps++) {
        const int nbin = 1 << bits[ps];
        for (int b = tid; b < 2048; b += kFlThreads) hist[b] = 0;
        __syncthreads();
        for (int t = tid; t < n; t += kFlThreads) {
            const uint64_t k = fl_key(f[t], t);
            if (k >= lim) continue;
            const uint32_t k32 = (uint32_t)(k >> 32);
            if ((k32 & mask) != prefix) continue;
            const unsigned long long w = wt(t);
            if (w) atomicAdd(&hist[(k32 >> shifts[ps]) & (nbin - 1)], w);
        }
        __syncthreads();
        // ascending bins: thread t owns bins 2t, 2t + 1
        const int b0 = 2 * tid, b1 = b0 + 1;
        const unsigned long long h0 = b0 < nbin ? hist[b0] : 0ull, h1 = b1 < nbin ? hist[b1] : 0ull;
        unsigned long long x = h0 + h1, incl = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const unsigned long long v = wsum[lane];
            unsigned long long iv = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned long long y = __shfl_up_sync(0xffffffffu, iv, o);
                if (lane >= o) iv += y;
            }
            wsum[lane] = iv - v;
            if (lane == 31) bc[1] = iv;      // total weight of this pass's tokens
        }
        __syncthreads();
        const unsigned long long before = below + wsum[warp] + (incl - x);
        if (ps == 0 && tid == 0) bc[0] = 0xFFFFFFFFull;   // no crossing bin yet
        __syncthreads();
        if (below + bc[1] <= budget) {
            all_fit = true;        // (only possible in the first pass: later passes keep one crossing bin)
            break;
        }
        if (b0 < nbin && before <= budget && before + h0 > budget) { bc[0] = (unsigned)b0; bc[2] = before; }
        else if (b1 < nbin && before + h0 <= budget && before + h0 + h1 > budget) { bc[0] = (unsigned)b1; bc[2] = before + h0; }
        __syncthreads();
        prefix |= (uint32_t)bc[0] << shifts[ps];
        mask |= (uint32_t)(nbin - 1) << shifts[ps];
        below = bc[2];
        __syncthreads();
    }
    if (all_fit) return ~0ull;
    // stage 2: tokens whose f part equals the crossing value, in t order
    const unsigned long long rem = budget - below;
    unsigned long long carry = 0;
    if (tid == 0) bc[3] = ~0ull;
    __syncthreads();
    for (int t0 = 0; t0 < n; t0 += kFlThreads) {
        const int t = t0 + tid;
        unsigned long long w = 0;
        if (t < n) {
            const uint64_t k = fl_key(f[t], t);
            if (k < lim && (uint32_t)(k >> 32) == prefix) w = wt(t);
        }
        unsigned long long incl = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const unsigned long long v = wsum[lane];
            unsigned long long iv = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned long long y = __shfl_up_sync(0xffffffffu, iv, o);
                if (lane >= o) iv += y;
            }
            wsum[lane] = iv - v;
            if (lane == 31) bc[1] = iv;
        }
        __syncthreads();
        const unsigned long long cum = carry + wsum[warp] + incl;   // inclusive, in t order
        if (w && cum > rem && cum - w <= rem) atomicMin(&bc[3], ((unsigned long long)prefix << 32) | (uint32_t)t);
        carry += bc[1];
        __syncthreads();
        if (bc[3] != ~0ull) break;
    }
    __syncthreads();
    return bc[3];
}

// Joint cost of the tokens with key < cut inside one (l, g): per slot, |S| +
// the maximal runs of slot positions outside S (0 for a slot without any).
__device__ unsigned long long block_joint_cost(const FloorArgs &a, const float *f, uint64_t cut,
                                               unsigned long long *wsum) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned long long tot = 0;
    for (int j = warp; j < a.J; j += kFlThreads / 32) {
        const int sa = a.slots[j] - a.cs, sb = a.slots[j + 1] - a.cs;
        int k = 0, runs = 0;
        bool prev_in = true;       // position sa - 1 counts as inside: a run may start at sa
        for (int t0 = sa; t0 < sb; t0 += 32) {
            const int t = t0 + lane;
            const bool in = t < sb && fl_key(f[t], t) < cut;
            const unsigned m = __ballot_sync(0xffffffffu, in);
            const unsigned valid = __ballot_sync(0xffffffffu, t < sb);
            // position t starts a run when it is outside S and t - 1 is inside (or t = sa)
            const unsigned prev = (m << 1) | (prev_in ? 1u : 0u);
            runs += __popc(~m & valid & prev);
            k += __popc(m);
            prev_in = (m >> 31) & 1u;
            if (sb - t0 < 32) prev_in = (m >> (sb - t0 - 1)) & 1u;
        }
        if (lane == 0 && k) tot += (unsigned long long)(k + runs);
    }
    if (lane == 0) wsum[warp] = tot;
    __syncthreads();
    unsigned long long s = 0;
    if (tid == 0)
        for (int w = 0; w < kFlThreads / 32; w++) s += wsum[w];
    __syncthreads();
    if (tid == 0) wsum[0] = s;
    __syncthreads();
    s = wsum[0];
    __syncthreads();
    return s;
}

__global__ void floor_rbar_kernel(FloorArgs a) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= a.Nc) return;
    double s = 0.0;
    for (int lg = 0; lg < a.LG; lg++) s += a.rtok[(size_t)lg * a.Nc + t];
    a.rbar[t] = (float)(s / a.LG);
}

__global__ void floor_score_kernel(FloorArgs a) {
    const int lg = blockIdx.y;
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= a.Nc) return;
    const float *R = a.rtok + (size_t)lg * a.Nc;
    float m = -INFINITY;
    for (int u = max(t - a.half, 0); u <= min(t + a.half, a.Nc - 1); u++)
        m = fmaxf(m, (1.f - a.c) * R[u] + a.c * a.rbar[u]);
    a.f[(size_t)lg * a.Nc + t] = m;
}

// Candidates of each (l, g): the eta prefix among the gated tokens.
__global__ void __launch_bounds__(kFlThreads) floor_cand_kernel(FloorArgs a) {
    __shared__ unsigned long long hist[2048], wsum[32], bc[4];
    const int lg = blockIdx.x;
    const float *f = a.f + (size_t)lg * a.Nc;
    const float *R = a.rtok + (size_t)lg * a.Nc;
    const uint64_t gate_lim = ((uint64_t)(~__float_as_uint(a.gate)) + 1ull) << 32;   // f >= gate
    const uint64_t cut = block_wselect(f, a.Nc, gate_lim, a.eta_fx,
                                       [&](int t) { return (unsigned long long)((double)R[t] * kFlFix); },
                                       hist, wsum, bc);
    const uint64_t lim = cut < gate_lim ? cut : gate_lim;
    unsigned long long n = 0;
    for (int t = threadIdx.x; t < a.Nc; t += kFlThreads) n += fl_key(f[t], t) < lim;
    n = __reduce_add_sync(0xffffffffu, (unsigned)n);
    if ((threadIdx.x & 31) == 0 && n) atomicAdd(&a.head[(size_t)lg * kFlHead + FH_N], n);
    if (threadIdx.x == 0) a.head[(size_t)lg * kFlHead + FH_CUT] = lim;
    __syncthreads();
    const unsigned long long c0 = block_joint_cost(a, f, lim, wsum);
    if (threadIdx.x == 0) {
        a.head[(size_t)lg * kFlHead + FH_COST0] = c0;
        if (c0) atomicAdd(&a.glob[FG_C0], c0);
    }
}

// Proportional reduction when the joint cost of all candidates exceeds the cap.
__global__ void __launch_bounds__(kFlThreads) floor_keep_kernel(FloorArgs a) {
    __shared__ unsigned long long hist[2048], wsum[32], bc[4];
    const int lg = blockIdx.x;
    unsigned long long *h = a.head + (size_t)lg * kFlHead;
    const float *f = a.f + (size_t)lg * a.Nc;
    const unsigned long long n = h[FH_N], C0 = a.glob[FG_C0];
    const unsigned long long cap = (unsigned long long)a.cap;
    unsigned long long keep = n;
    uint64_t cut = h[FH_CUT];
    if (n && C0 > cap) {
        keep = n * cap / C0;
        if (keep < 1) keep = 1;
        if (keep < n) cut = block_wselect(f, a.Nc, cut, keep, [](int) { return 1ull; }, hist, wsum, bc);
    }
    if (threadIdx.x == 0) {
        h[FH_KEEP] = keep;
        h[FH_CUTK] = cut;
        if (keep) atomicAdd(&a.glob[FG_NKEEP], keep);
    }
}

// Nearest accepted position of [lo, hi] (context-relative, lo <= hi) in the
// bitmap: the largest one when from_top, else the smallest; -1 when none.
// Called by a whole warp; every lane returns the same value.
__device__ __forceinline__ int fl_nearest(const uint32_t *bits, int lo, int hi, bool from_top) {
    const int lane = threadIdx.x & 31, wlo = lo >> 5, whi = hi >> 5;
    const uint32_t mlo = ~0u << (lo & 31), mhi = (2u << (hi & 31)) - 1u;   // bits >= lo, <= hi
    for (int w0 = from_top ? whi : wlo; from_top ? w0 >= wlo : w0 <= whi; w0 += from_top ? -32 : 32) {
        const int w = from_top ? w0 - lane : w0 + lane;
        uint32_t x = 0;
        if (w >= wlo && w <= whi) {
            x = bits[w];
            if (w == wlo) x &= mlo;
            if (w == whi) x &= mhi;
        }
        const unsigned bal = __ballot_sync(0xffffffffu, x != 0);
        if (bal) {
            const int src = __ffs(bal) - 1;          // the lane nearest the start
            const uint32_t xs = __shfl_sync(0xffffffffu, x, src);
            const int ws = from_top ? w0 - src : w0 + src;
            return from_top ? ws * 32 + 31 - __clz(xs) : ws * 32 + __ffs(xs) - 1;
        }
    }
    return -1;
}

// Acceptance: walk the kept candidates in order (f descending, ties lower t);
// accept each one whose path fits what is left of the head's share, skip the
// others.  A candidate's path costs 1 for its slot's Add when no accepted
// position is in the slot yet, plus one entry for each non-empty side of it
// inside its current frontier interval (bounded by the nearest accepted
// positions of the slot, else by the slot's ends).  Dynamic shared memory: the
// accepted positions as a bitmap of ceil(N_c / 32) words.
__global__ void __launch_bounds__(kFlThreads) floor_accept_kernel(FloorArgs a) {
    __shared__ unsigned long long hist[2048], wsum[32], bc[4];
    __shared__ int cnt;
    extern __shared__ uint32_t acc_bits[];
    const int lg = blockIdx.x, tid = threadIdx.x;
    unsigned long long *h = a.head + (size_t)lg * kFlHead;
    const float *f = a.f + (size_t)lg * a.Nc;
    const int nw = (a.Nc + 31) >> 5;
    for (int w = tid; w < nw; w += kFlThreads) acc_bits[w] = 0u;
    const unsigned long long keep = h[FH_KEEP], nkeep = a.glob[FG_NKEEP];
    const unsigned long long share = keep ? (unsigned long long)a.cap * keep / nkeep : 0ull;
    const uint64_t kcut = h[FH_CUTK];
    // the chunk lives in hist between two selects: keys, then slot bounds
    uint64_t *ck = reinterpret_cast<uint64_t *>(hist);
    int *ca = reinterpret_cast<int *>(hist + kFlThreads);
    int *cb = ca + kFlThreads;
    unsigned long long used = 0, done = 0;      // used: meaningful in warp 0
    uint64_t lo_cut = 0;
    __syncthreads();
    while (done < keep) {
        const unsigned long long m = keep - done < (unsigned long long)kFlThreads ? keep - done
                                                                                 : (unsigned long long)kFlThreads;
        const uint64_t hi_cut = done + m >= keep
            ? kcut : block_wselect(f, a.Nc, kcut, done + m, [](int) { return 1ull; }, hist, wsum, bc);
        ck[tid] = ~0ull;
        if (tid == 0) cnt = 0;
        __syncthreads();
        for (int t = tid; t < a.Nc; t += kFlThreads) {
            const uint64_t k = fl_key(f[t], t);
            if (k >= lo_cut && k < hi_cut) {
                const int i = atomicAdd(&cnt, 1);
                if (i < kFlThreads) ck[i] = k;
            }
        }
        __syncthreads();
        // bitonic sort of the chunk's keys, ascending (unused entries are ~0)
        for (int k2 = 2; k2 <= kFlThreads; k2 <<= 1)
            for (int j2 = k2 >> 1; j2 > 0; j2 >>= 1) {
                const int ix = tid ^ j2;
                if (ix > tid) {
                    const uint64_t x = ck[tid], y = ck[ix];
                    if ((x > y) == ((tid & k2) == 0)) { ck[tid] = y; ck[ix] = x; }
                }
                __syncthreads();
            }
        const int mc = min((int)m, min(cnt, kFlThreads));   // keys collected (m when the select is exact)
        if (tid < mc) {
            const int t = (int)(uint32_t)ck[tid];
            int lo = 0, hi = a.J;                  // the last j with slots[j] - cs <= t
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (a.slots[mid] - a.cs <= t) lo = mid; else hi = mid;
            }
            ca[tid] = a.slots[lo] - a.cs;
            cb[tid] = a.slots[lo + 1] - a.cs;
        }
        __syncthreads();
        if (tid < 32) {
            for (int i = 0; i < mc; i++) {
                const int t = (int)(uint32_t)ck[i], sa = ca[i], sb = cb[i];
                const int left = t > sa ? fl_nearest(acc_bits, sa, t - 1, true) : -1;
                const int right = t < sb - 1 ? fl_nearest(acc_bits, t + 1, sb - 1, false) : -1;
                const int lo = left >= 0 ? left + 1 : sa, hi = right >= 0 ? right - 1 : sb - 1;
                const unsigned long long cost =
                    (left < 0 && right < 0 ? 1ull : 0ull) + (lo < t ? 1ull : 0ull) + (t < hi ? 1ull : 0ull);
                if (used + cost <= share) {
                    used += cost;
                    if (tid == 0) acc_bits[t >> 5] |= 1u << (t & 31);
                }
                __syncwarp();
            }
        }
        __syncthreads();
        lo_cut = hi_cut;
        done += m;
    }
    uint8_t *acc = a.acc + (size_t)lg * a.Nc;
    for (int t = tid; t < a.Nc; t += kFlThreads) acc[t] = (uint8_t)((acc_bits[t >> 5] >> (t & 31)) & 1u);
    for (int j = tid; j < a.J; j += kFlThreads) {
        uint8_t any = 0;
        for (int t = a.slots[j] - a.cs; t < a.slots[j + 1] - a.cs && !any; t++)
            any = (uint8_t)((acc_bits[t >> 5] >> (t & 31)) & 1u);
        a.u_floor[(size_t)lg * a.J + j] = any;
    }
    if (tid == 0) {
        h[FH_USED] = used;
        if (used) atomicAdd(&a.glob[FG_USED], used);
    }
}

}  // namespace

cudaError_t launch_floor(Ctx &c, int J, cudaStream_t s) {
    Workspace &w = c.w;
    const gkv_params &p = c.p;
    FloorArgs a;
    a.rtok = w.rtok;
    a.slots = w.slots;
    a.rbar = w.fl_rbar;
    a.f = w.fl_f;
    a.acc = w.fl_acc;
    a.u_floor = w.u_floor;
    a.head = w.fl_head;
    a.glob = w.fl_glob;
    a.LG = p.L * p.G;
    a.Nc = c.Nc;
    a.J = J;
    a.cs = p.ctx_start;
    a.half = p.floor_half;
    a.c = (float)p.floor_c;
    a.gate = (float)(p.floor_gamma / c.Nc);
    a.eta_fx = (unsigned long long)(p.floor_eta * kFlFix);
    a.cap = (long long)floor(p.alpha_floor * (double)c.B_free);
    cudaError_t e = cudaMemsetAsync(w.fl_head, 0, sizeof(unsigned long long) * kFlHead * a.LG, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(w.fl_glob, 0, sizeof(unsigned long long) * 4, s);
    if (e != cudaSuccess) return e;
    floor_rbar_kernel<<<(a.Nc + 255) / 256, 256, 0, s>>>(a);
    floor_score_kernel<<<dim3((a.Nc + 255) / 256, a.LG), 256, 0, s>>>(a);
    floor_cand_kernel<<<a.LG, kFlThreads, 0, s>>>(a);
    floor_keep_kernel<<<a.LG, kFlThreads, 0, s>>>(a);
    const size_t bits_bytes = sizeof(uint32_t) * (size_t)((a.Nc + 31) / 32);
    e = cudaFuncSetAttribute(floor_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bits_bytes);
    if (e != cudaSuccess) return e;
    floor_accept_kernel<<<a.LG, kFlThreads, bits_bytes, s>>>(a);
    c.launches += 5;
    return cudaGetLastError();
}

int floor_head_words() { return kFlHead; }

}  // namespace gkv
