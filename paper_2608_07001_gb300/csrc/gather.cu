// gather.cu -- stage 4 of the GraceKV pass: packing of the retained frontier
// into a ragged cache (App. A.5 "Frontier updates and physical packing").
//
// A node is on the frontier when the op that created it was executed (the
// Add for a root, the parent's Split otherwise) and its own Split was not.
// Per (l, g) the cache holds, in ascending position: the prefix [0, c_s),
// the frontier nodes of every covered slot, then the recent window and the
// suffix [c_e - r, T).  Single tokens keep their original K/V bits, position
// and log m = 0; other nodes store the prototype (ktil, vtil, p, log m_eff) of
// Eqs. app_rope_prototype, app_value_prototype, app_effective_multiplicity,
// recomputed here from K, V and the token values.
//
// Kernels: gather_count (frontier entries per unit), gather_bsum /
// gather_bscan / gather_offs (ordered exclusive scan -> per-unit and per-(l, g)
// offsets), gather_list
// (warp per unit, depth-first in ascending position: entry descriptors by
// output position), gather_emit (persistent warps, one entry at a time, rows
// streamed through a per-warp cp.async ring: prototypes or single-token
// copies), gather_tokens (prefix / recent / suffix copies).
#include "gkv_internal.cuh"

#include <algorithm>

namespace gkv {
namespace {

struct GatherArgs {
    const void *K, *V;
    const float *rtok;
    const float2 *rope;
    const float2 *rope_rel;    // [2 kMaxSlot - 1][d/2]: rotation by the offset p - t
    int4 *ent;                 // [entries]: (a, b, lg, 1) of every frontier entry, by output position
    const int32_t *slots;
    const int32_t *nd_a, *nd_b, *nd_child0, *nd_parent;
    const int8_t *nd_nchild;
    const uint8_t *nd_sel, *u_sel;
    const int32_t *u_nnodes;
    int32_t *u_count;
    int64_t *u_off;
    int L, G, T, d, J, cs, cend, Nc;
    double base_frac, eps;
    void *K_out, *V_out;
    int32_t *pos, *src_lo, *src_hi;
    float *log_m;
    int64_t *offsets;
};

__device__ __forceinline__ int round_half_even_mid(int a, int b) {
    int s = a + b - 1;
    if ((s & 1) == 0) return s >> 1;
    int lo = (s - 1) >> 1;
    return (lo & 1) == 0 ? lo : lo + 1;
}


__global__ void gather_count_kernel(GatherArgs A) {
    int64_t nu = (int64_t)A.L * A.G * A.J;
    int64_t uid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (uid >= nu) return;
    int lg = (int)(uid / A.J), j = (int)(uid - (int64_t)lg * A.J);
    int cnt = 0;
    if (A.u_sel[uid] == 1) {
        int64_t nb = node_base(lg, A.slots[j], A.cs, A.Nc);
        int nn = A.u_nnodes[uid];
        // frontier count = 1 + sum over executed splits of (|child| - 1)
        cnt = 1;
        for (int k = 0; k < nn; k++)
            if (A.nd_sel[nb + k] == 1) cnt += A.nd_nchild[nb + k] - 1;
    }
    A.u_count[uid] = cnt;
}

// Ordered exclusive scan of the per-unit counts in three steps (block sums,
// one block scanning the block sums, block-local scans); unit offsets include
// the prefix tokens of its (l, g) and the prefix + tail tokens of earlier (l, g).
constexpr int kScanB = 1024;

__global__ void __launch_bounds__(kScanB) gather_bsum_kernel(const int32_t *cnt, int64_t nu, long long *bsum) {
    __shared__ long long ws[kScanB / 32];
    const int64_t i = (int64_t)blockIdx.x * kScanB + threadIdx.x;
    long long v = i < nu ? cnt[i] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x < 32) {
        long long w = ws[threadIdx.x];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) w += __shfl_xor_sync(0xffffffffu, w, o);
        if (threadIdx.x == 0) bsum[blockIdx.x] = w;
    }
}

// In place: bsum[b] becomes the exclusive prefix of the block sums; bsum[nb]
// the total.  One block; thread t scans a contiguous run of blocks.
__global__ void __launch_bounds__(kScanB) gather_bscan_kernel(long long *bsum, int nb) {
    __shared__ long long part[kScanB];
    const int tid = threadIdx.x;
    const int per = (nb + kScanB - 1) / kScanB;
    const int b0 = tid * per, b1 = min(nb, b0 + per);
    long long s = 0;
    for (int q = b0; q < b1; q++) s += bsum[q];
    part[tid] = s;
    __syncthreads();
    if (tid == 0) {
        long long acc = 0;
        for (int k = 0; k < kScanB; k++) { const long long v = part[k]; part[k] = acc; acc += v; }
        bsum[nb] = acc;
    }
    __syncthreads();
    long long acc = part[tid];
    for (int q = b0; q < b1; q++) { const long long v = bsum[q]; bsum[q] = acc; acc += v; }
}

__global__ void __launch_bounds__(kScanB) gather_offs_kernel(GatherArgs A, const long long *bsum, int nb) {
    __shared__ long long ws[kScanB / 32];
    const int64_t nu = (int64_t)A.L * A.G * A.J;
    const int64_t i = (int64_t)blockIdx.x * kScanB + threadIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const long long v = i < nu ? A.u_count[i] : 0;
    long long incl = v;   // inclusive warp scan
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) ws[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const long long w = ws[lane];
        long long wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        ws[lane] = wi - w;   // exclusive over the block's warps
    }
    __syncthreads();
    const long long extra = (long long)A.cs + (A.T - A.cend);   // uncompressed entries per (l, g)
    if (i < nu) {
        const long long excl = bsum[blockIdx.x] + ws[warp] + incl - v;
        const int lg = (int)(i / A.J), j = (int)(i - (int64_t)lg * A.J);
        const long long off = excl + (long long)lg * extra + A.cs;
        A.u_off[i] = off;
        if (j == 0) A.offsets[lg] = off - A.cs;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) A.offsets[A.L * A.G] = bsum[nb] + (long long)A.L * A.G * extra;
}

// No covered unit at all: every (l, g) holds only its uncompressed tokens.
__global__ void gather_offs_empty_kernel(GatherArgs A) {
    const long long extra = (long long)A.cs + (A.T - A.cend);
    for (int lg = threadIdx.x; lg <= A.L * A.G; lg += blockDim.x) A.offsets[lg] = (long long)lg * extra;
}

// 8 consecutive elements held raw (loaded from shared memory, converted to
// fp32 on get, or stored back bit for bit).
template <typename T> struct Raw8;
template <> struct Raw8<float> {
    float4 a, b;
    __device__ __forceinline__ void load_shared(const float *p) {
        a = reinterpret_cast<const float4 *>(p)[0];
        b = reinterpret_cast<const float4 *>(p)[1];
    }
    __device__ __forceinline__ void get(float v[8]) const {
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    __device__ __forceinline__ void store(float *p) const {
        reinterpret_cast<float4 *>(p)[0] = a;
        reinterpret_cast<float4 *>(p)[1] = b;
    }
};
template <> struct Raw8<__nv_bfloat16> {
    uint4 u;
    __device__ __forceinline__ void load_shared(const __nv_bfloat16 *p) { u = *reinterpret_cast<const uint4 *>(p); }
    __device__ __forceinline__ void get(float v[8]) const {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; i++) {   // bf16 -> fp32 is exact: the bits move to the high half
            v[2 * i] = __uint_as_float(w[i] << 16);
            v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
    __device__ __forceinline__ void store(__nv_bfloat16 *p) const { *reinterpret_cast<uint4 *>(p) = u; }
};

// 4 consecutive elements held raw.
template <typename T> struct Raw4;
template <> struct Raw4<float> {
    float4 a;
    __device__ __forceinline__ void load_shared(const float *p) { a = *reinterpret_cast<const float4 *>(p); }
    __device__ __forceinline__ void get(float v[4]) const { v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; }
    __device__ __forceinline__ void store(float *p) const { *reinterpret_cast<float4 *>(p) = a; }
};
template <> struct Raw4<__nv_bfloat16> {
    uint2 u;
    __device__ __forceinline__ void load_shared(const __nv_bfloat16 *p) { u = *reinterpret_cast<const uint2 *>(p); }
    __device__ __forceinline__ void get(float v[4]) const {
        v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xFFFF0000u);
        v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xFFFF0000u);
    }
    __device__ __forceinline__ void store(__nv_bfloat16 *p) const { *reinterpret_cast<uint2 *>(p) = u; }
};
__device__ __forceinline__ void store4(__nv_bfloat16 *dst, const float v[4]) {
    uint2 u;
    __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&u);
    h[0] = __floats2bfloat162_rn(v[0], v[1]);
    h[1] = __floats2bfloat162_rn(v[2], v[3]);
    *reinterpret_cast<uint2 *>(dst) = u;
}
__device__ __forceinline__ void store4(float *dst, const float v[4]) {
    *reinterpret_cast<float4 *>(dst) = make_float4(v[0], v[1], v[2], v[3]);
}

// 8 consecutive elements copied bit for bit.
__device__ __forceinline__ void copy8(__nv_bfloat16 *dst, const __nv_bfloat16 *src) {
    *reinterpret_cast<uint4 *>(dst) = *reinterpret_cast<const uint4 *>(src);
}
__device__ __forceinline__ void copy8(float *dst, const float *src) {
    reinterpret_cast<uint4 *>(dst)[0] = reinterpret_cast<const uint4 *>(src)[0];
    reinterpret_cast<uint4 *>(dst)[1] = reinterpret_cast<const uint4 *>(src)[1];
}
__device__ __forceinline__ void store8(__nv_bfloat16 *dst, const float v[8]) {
    uint4 u;
    __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&u);
#pragma unroll
    for (int j = 0; j < 4; j++) h[j] = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
    *reinterpret_cast<uint4 *>(dst) = u;
}
__device__ __forceinline__ void store8(float *dst, const float v[8]) {
    reinterpret_cast<float4 *>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4 *>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// Frontier entries of every covered unit in ascending position (warp per
// unit, depth-first over the executed splits, children in ascending
// position): the descriptor of each entry goes to its output position.
__global__ void gather_list_kernel(GatherArgs A) {
    __shared__ short stack[8][kMaxUnit + 4];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nu = (int64_t)A.L * A.G * A.J;
    const int64_t uid = (int64_t)blockIdx.x * 8 + warp;
    if (uid >= nu || A.u_sel[uid] != 1 || lane != 0) return;
    const int lg = (int)(uid / A.J), j = (int)(uid - (int64_t)lg * A.J);
    if (A.slots[j + 1] - A.slots[j] > kMaxUnit) return;   // a long unit: gather_list_long
    const int64_t nb = node_base(lg, A.slots[j], A.cs, A.Nc);
    int64_t e = A.u_off[uid];
    short *st = stack[warp];
    int sp = 0;
    st[sp++] = 0;
    while (sp > 0) {
        const int x = st[--sp];
        const int64_t v = nb + x;
        if (A.nd_sel[v] == 1) {
            const int c0 = A.nd_child0[v], nc = A.nd_nchild[v];
            for (int q = nc - 1; q >= 0; q--) st[sp++] = (short)(c0 + q);   // leftmost on top
            continue;
        }
        A.ent[e++] = make_int4(A.nd_a[v], A.nd_b[v], lg, 1);
    }
}

// The same for the units of slots longer than kMaxUnit (CTA per unit): a node
// is a frontier entry when it is reached (the root with its Add selected, or a
// child of a selected split) and its own split is not selected; the entries of
// a unit are disjoint intervals, so an entry's output rank is the number of
// entry starts before its own, counted over a bitmap of the slot's positions.
__global__ void __launch_bounds__(256) gather_list_long_kernel(GatherArgs A, const int32_t *long_slots) {
    __shared__ uint32_t bits[kMaxSlot / 32];
    __shared__ int wpre[kMaxSlot / 32];
    __shared__ int warp_tot[8];
    const int LG = A.L * A.G;
    const int lg = blockIdx.x % LG, j = long_slots[blockIdx.x / LG];
    const int64_t uid = (int64_t)lg * A.J + j;
    if (A.u_sel[uid] != 1) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int sa = A.slots[j], n = A.slots[j + 1] - sa;
    const int nw = (n + 31) / 32;
    const int64_t nb = node_base(lg, sa, A.cs, A.Nc);
    const int nn = A.u_nnodes[uid];
    for (int w = tid; w < nw; w += 256) bits[w] = 0u;
    __syncthreads();
    auto frontier = [&](int k) {
        const int64_t v = nb + k;
        if (A.nd_sel[v] == 1 || A.nd_nchild[v] == -2) return false;   // selected, or an unused slot
        const int32_t pg = A.nd_parent[v];
        return pg < 0 ? true : A.nd_sel[pg] == 1;   // the root is reached: its Add is selected
    };
    for (int k = tid; k < nn; k += 256)
        if (frontier(k)) {
            const int off = A.nd_a[nb + k] - sa;
            atomicOr(&bits[off >> 5], 1u << (off & 31));
        }
    __syncthreads();
    // exclusive prefix of the set bits in word order (thread t: words 2 t, 2 t + 1)
    const int w0 = 2 * tid;
    const int c0 = w0 < nw ? __popc(bits[w0]) : 0, c1 = w0 + 1 < nw ? __popc(bits[w0 + 1]) : 0;
    const int x = c0 + c1;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    int before = 0;
    for (int w = 0; w < warp; w++) before += warp_tot[w];
    const int ex = before + incl - x;
    if (w0 < nw) wpre[w0] = ex;
    if (w0 + 1 < nw) wpre[w0 + 1] = ex + c0;
    __syncthreads();
    const int64_t e0 = A.u_off[uid];
    for (int k = tid; k < nn; k += 256)
        if (frontier(k)) {
            const int off = A.nd_a[nb + k] - sa;
            const int rank = wpre[off >> 5] + __popc(bits[off >> 5] & ((1u << (off & 31)) - 1u));
            A.ent[e0 + rank] = make_int4(A.nd_a[nb + k], A.nd_b[nb + k], lg, 1);
        }
}

// Prototypes of the listed entries (one warp per entry; rows read as
// 8-element chunks, LPR = d / 8 lanes per row and RPW = 32 / LPR rows per step).
// Each warp walks its entries (warp id, + number of warps, ...) as one stream of
// steps; the K and V rows and token values of step s + D - 1 are copied into
// the warp's ring of D steps (cp.async, zero-filled past an entry's end) while
// step s is consumed, so D - 1 steps of loads stay in flight across entry
// boundaries.  Lane c of a row holds the key's rotation pairs (i, i + d/2) for
// i = 4 c .. 4 c + 3 and the value elements 8 c .. 8 c + 7.  The key prototype RoPE(mean_t RoPE^-1(k_t, t),
// p) is formed as mean_t of k_t rotated by p - t (rotations compose), from a
// table of the offsets -(kMaxSlot - 1) .. kMaxSlot - 1; its norm equals the norm of the mean
// inverse-rotated key.  The value prototype uses sum_t (R_t + beta) v_t =
// sum R v + beta sum v.  All arithmetic is fp32.
constexpr int kRingSteps = 8;

template <typename Tin, int DH>
struct EmitGeom {
    static constexpr int LPR = DH / 8, RPW = 32 / LPR;
    static constexpr int KB = DH * (int)sizeof(Tin);      // bytes of a K (or V) row
    static constexpr int RB = 2 * KB;                      // ring bytes of a row: K, then V
    static constexpr int CPR = RB / 16;                    // 16-byte chunks of a ring row
    static constexpr int WARP_BYTES = kRingSteps * RPW * (RB + 4);
};

template <typename Tin, int DH>
__global__ void __launch_bounds__(256, 2) gather_emit_kernel(GatherArgs A, int64_t n_ent) {
    using Gm = EmitGeom<Tin, DH>;
    constexpr int HALF = DH / 2, LPR = Gm::LPR, RPW = Gm::RPW, RB = Gm::RB, CPR = Gm::CPR;
    const float base_frac = (float)A.base_frac, eps = (float)A.eps;
    constexpr int D = kRingSteps;
    extern __shared__ __align__(16) unsigned char gsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *ring = gsm + (size_t)warp * Gm::WARP_BYTES;
    float *rring = reinterpret_cast<float *>(ring + D * RPW * RB);
    const int64_t nw = (int64_t)gridDim.x * 8;
    const int r = lane / LPR, c = lane - r * LPR;
    const int i0 = 4 * c;                      // the lane's rotation pairs i0 .. i0 + 3 (both halves)

    struct Cur { int64_t e; int s, nst, lg, a, b; };
    // first compressible entry at or after e in this warp's sequence
    auto seek = [&](Cur &cu, int64_t e) {
        for (; e < n_ent; e += nw) {
            const int4 en = A.ent[e];
            if (en.w == 0) continue;   // prefix / recent / suffix token (gather_tokens)
            cu.e = e; cu.s = 0; cu.lg = en.z; cu.a = en.x; cu.b = en.y;
            cu.nst = (en.y - en.x + RPW - 1) / RPW;
            return;
        }
        cu.e = n_ent;
    };
    Cur pf, cs;
    seek(pf, (int64_t)blockIdx.x * 8 + warp);
    cs = pf;
    // copy the prefetch cursor's step into ring slot `slot` and advance it
    auto issue = [&](int slot) {
        if (pf.e < n_ent) {
            const char *K = static_cast<const char *>(A.K) + (size_t)pf.lg * A.T * Gm::KB;
            const char *V = static_cast<const char *>(A.V) + (size_t)pf.lg * A.T * Gm::KB;
            const int t0 = pf.a + pf.s * RPW;
#pragma unroll
            for (int q = lane; q < RPW * CPR; q += 32) {
                const int rr = q / CPR, ch = q - rr * CPR;
                const int t = t0 + rr;
                const bool ok = t < pf.b;
                const size_t row = (size_t)(ok ? t : pf.a) * Gm::KB;
                const char *src = ch < CPR / 2 ? K + row + ch * 16 : V + row + (ch - CPR / 2) * 16;
                cp_async16(ring + ((size_t)slot * RPW + rr) * RB + ch * 16, src, ok);
            }
            if (lane < RPW) {
                const int t = t0 + lane;
                const bool ok = t < pf.b;
                cp_async4(&rring[slot * RPW + lane], A.rtok + (size_t)pf.lg * A.Nc + ((ok ? t : pf.a) - A.cs), ok);
            }
            if (++pf.s == pf.nst) seek(pf, pf.e + nw);
        }
        cp_async_commit();
    };
    for (int q = 0; q < D - 1; q++) issue(q);
    int slot = 0;
    while (cs.e < n_ent) {
        const int lg = cs.lg, a = cs.a, b = cs.b, n = b - a;
        const int64_t e = cs.e;
        Tin *Ko = static_cast<Tin *>(A.K_out) + (size_t)e * DH;
        Tin *Vo = static_cast<Tin *>(A.V_out) + (size_t)e * DH;
        const int p = round_half_even_mid(a, b);
        float mk[8], sv[8], srv[8], kn = 0.f, rs = 0.f;   // mk: pairs i0 + j (j < 4) and their partners
#pragma unroll
        for (int j = 0; j < 8; j++) mk[j] = sv[j] = srv[j] = 0.f;
        for (int st = 0; st < cs.nst; st++) {
            issue((slot + D - 1) % D);   // the slot consumed last
            cp_async_wait<D - 1>();      // this step's group has landed
            __syncwarp();
            const unsigned char *row = ring + ((size_t)slot * RPW + r) * RB;
            Raw4<Tin> klo, khi;
            Raw8<Tin> vraw;
            klo.load_shared(reinterpret_cast<const Tin *>(row) + i0);
            khi.load_shared(reinterpret_cast<const Tin *>(row) + HALF + i0);
            vraw.load_shared(reinterpret_cast<const Tin *>(row + Gm::KB) + 8 * c);
            const float rr = rring[slot * RPW + r];
            const int t = a + st * RPW + r;
            const int tt = t < b ? t : b - 1;   // rows past b are zero
            if (n == 1) {   // single token: original bits, p = t, log m = 0
                if (lane < LPR) {
                    klo.store(Ko + i0);
                    khi.store(Ko + HALF + i0);
                    vraw.store(Vo + 8 * c);
                }
            } else {
                float x[4], y[4], vx[8], nn = 0.f;
                klo.get(x);
                khi.get(y);
                vraw.get(vx);
#pragma unroll
                for (int j = 0; j < 4; j++) nn = fmaf(x[j], x[j], fmaf(y[j], y[j], nn));
#pragma unroll
                for (int o = 1; o < LPR; o <<= 1) nn += __shfl_xor_sync(0xffffffffu, nn, o);
                if (c == 0) kn += sqrtf(nn);   // |k_t|
                rs += rr;
                const float4 *cs4 = reinterpret_cast<const float4 *>(
                    A.rope_rel + (size_t)(p - tt + kMaxSlot - 1) * HALF + i0);
#pragma unroll
                for (int j2 = 0; j2 < 2; j2++) {
                    const float4 q = cs4[j2];          // (cos, sin) of pairs i0 + 2 j2, i0 + 2 j2 + 1
                    const float cc[2] = {q.x, q.z}, sn[2] = {q.y, q.w};
#pragma unroll
                    for (int h = 0; h < 2; h++) {
                        const int j = 2 * j2 + h;
                        // rotation by p - t: x' = x cos - y sin, y' = x sin + y cos
                        mk[j] = fmaf(x[j], cc[h], fmaf(-y[j], sn[h], mk[j]));
                        mk[4 + j] = fmaf(x[j], sn[h], fmaf(y[j], cc[h], mk[4 + j]));
                    }
                }
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    sv[j] += vx[j];
                    srv[j] = fmaf(rr, vx[j], srv[j]);
                }
            }
            __syncwarp();   // the slot may be refilled by the next issue
            slot = slot + 1 == D ? 0 : slot + 1;
        }
        if (n == 1) {
            if (lane == 0) { A.pos[e] = a; A.log_m[e] = 0.f; A.src_lo[e] = a; A.src_hi[e] = b; }
        } else {
            // combine the row groups
#pragma unroll
            for (int o = LPR; o < 32; o <<= 1) {
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    mk[j] += __shfl_xor_sync(0xffffffffu, mk[j], o);
                    sv[j] += __shfl_xor_sync(0xffffffffu, sv[j], o);
                    srv[j] += __shfl_xor_sync(0xffffffffu, srv[j], o);
                }
                kn += __shfl_xor_sync(0xffffffffu, kn, o);
                rs += __shfl_xor_sync(0xffffffffu, rs, o);
            }
            kn = __shfl_sync(0xffffffffu, kn, 0);
            const float ninv = 1.0f / (float)n;
            const float beta = base_frac * (rs * ninv);
            const float winv = 1.0f / (rs + (float)n * beta + eps);
            float ko[8], vo[8], mu2 = 0.f;
#pragma unroll
            for (int j = 0; j < 8; j++) {
                ko[j] = mk[j] * ninv;
                vo[j] = fmaf(beta, sv[j], srv[j]) * winv;
                mu2 = fmaf(ko[j], ko[j], mu2);
            }
#pragma unroll
            for (int o = 1; o < LPR; o <<= 1) mu2 += __shfl_xor_sync(0xffffffffu, mu2, o);
            if (lane < LPR) {
                store4(Ko + i0, ko);
                store4(Ko + HALF + i0, ko + 4);
                store8(Vo + 8 * c, vo);
            }
            if (lane == 0) {
                const float coh = sqrtf(mu2) / (kn * ninv + eps);
                float me = (float)n * coh * coh;
                me = me < 1.0f ? 1.0f : (me > (float)n ? (float)n : me);
                A.pos[e] = p;
                A.log_m[e] = logf(me);
                A.src_lo[e] = a;
                A.src_hi[e] = b;
            }
        }
        seek(cs, cs.e + nw);
    }
    cp_async_wait<0>();
}

template <typename Tin>
__global__ void gather_tokens_kernel(GatherArgs A) {
    const int lg = blockIdx.y;
    const int ntail = A.T - A.cend;
    const int k = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (k >= A.cs + ntail) return;
    int t;
    int64_t e;
    if (k < A.cs) { t = k; e = A.offsets[lg] + k; }
    else { t = A.cend + (k - A.cs); e = A.offsets[lg + 1] - ntail + (k - A.cs); }
    const Tin *K = static_cast<const Tin *>(A.K) + ((size_t)lg * A.T + t) * A.d;
    const Tin *V = static_cast<const Tin *>(A.V) + ((size_t)lg * A.T + t) * A.d;
    Tin *Ko = static_cast<Tin *>(A.K_out) + (size_t)e * A.d;
    Tin *Vo = static_cast<Tin *>(A.V_out) + (size_t)e * A.d;
    for (int i = lane; i < A.d; i += 32) { Ko[i] = K[i]; Vo[i] = V[i]; }
    if (lane == 0) { A.pos[e] = t; A.log_m[e] = 0.f; A.src_lo[e] = t; A.src_hi[e] = t + 1; }
}

// Persistent grid: as many blocks as fit on the device at once.
template <typename Tin, int DH>
cudaError_t launch_emit(const Ctx &c, const GatherArgs &A, int64_t n_ent, cudaStream_t s) {
    const size_t smem = 8 * (size_t)EmitGeom<Tin, DH>::WARP_BYTES;
    cudaError_t e = cudaFuncSetAttribute(gather_emit_kernel<Tin, DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_emit_kernel<Tin, DH>, 256, smem);
    if (e != cudaSuccess) return e;
    const int64_t want = std::max<int64_t>(1, (int64_t)c.num_sms * std::max(per_sm, 1));
    const unsigned ge = (unsigned)std::min<int64_t>((n_ent + 7) / 8, want);
    gather_emit_kernel<Tin, DH><<<ge, 256, smem, s>>>(A, n_ent);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gather(Ctx &c, const void *K, const void *V, const int32_t *slots, int J,
                          void *K_out, void *V_out, int32_t *pos, float *log_m,
                          int32_t *src_lo, int32_t *src_hi, int64_t *offsets, cudaStream_t s) {
    GatherArgs A;
    A.K = K; A.V = V; A.rtok = c.w.rtok; A.rope = c.w.rope; A.rope_rel = c.w.rope_rel; A.ent = c.w.ent;
    A.slots = slots;
    A.nd_a = c.w.nd_a; A.nd_b = c.w.nd_b; A.nd_child0 = c.w.nd_child0; A.nd_parent = c.w.nd_parent;
    A.nd_nchild = c.w.nd_nchild;
    A.nd_sel = c.w.nd_sel; A.u_sel = c.w.u_sel; A.u_nnodes = c.w.u_nnodes;
    A.u_count = c.w.u_count; A.u_off = c.w.u_off;
    A.L = c.p.L; A.G = c.p.G; A.T = c.p.T; A.d = c.p.d; A.J = J; A.cs = c.p.ctx_start;
    A.cend = c.c_end; A.Nc = c.Nc; A.base_frac = c.p.base_frac; A.eps = c.p.eps;
    A.K_out = K_out; A.V_out = V_out; A.pos = pos; A.log_m = log_m; A.src_lo = src_lo;
    A.src_hi = src_hi; A.offsets = offsets;
    const int64_t nu = (int64_t)c.p.L * c.p.G * J;
    const int nb = (int)((nu + kScanB - 1) / kScanB);
    if (nu > 0) {
        gather_count_kernel<<<(unsigned)((nu + 255) / 256), 256, 0, s>>>(A);
        gather_bsum_kernel<<<nb, kScanB, 0, s>>>(c.w.u_count, nu, c.w.u_bsum);
        gather_bscan_kernel<<<1, kScanB, 0, s>>>(c.w.u_bsum, nb);
        gather_offs_kernel<<<nb, kScanB, 0, s>>>(A, c.w.u_bsum, nb);
    } else {
        gather_offs_empty_kernel<<<1, 256, 0, s>>>(A);
    }
    const bool bf = c.p.dtype == GKV_BF16;
    unsigned gu = (unsigned)((nu + 7) / 8);
    // descriptors by output position; positions of uncompressed tokens stay 0
    const int64_t n_ent = c.p.L * (int64_t)c.p.G * (c.p.T - c.Nc) + c.used;
    cudaError_t me = cudaMemsetAsync(A.ent, 0, sizeof(int4) * (size_t)n_ent, s);
    if (me != cudaSuccess) return me;
    if (gu) {
        gather_list_kernel<<<gu, 256, 0, s>>>(A);
        if (c.n_long > 0) {
            gather_list_long_kernel<<<(unsigned)(c.n_long * c.p.L * c.p.G), 256, 0, s>>>(A, c.w.long_slots);
            c.launches += 1;
        }
        cudaError_t le;
        if (c.p.d == 128) {
            if (bf) le = launch_emit<__nv_bfloat16, 128>(c, A, n_ent, s);
            else le = launch_emit<float, 128>(c, A, n_ent, s);
        } else {
            if (bf) le = launch_emit<__nv_bfloat16, 64>(c, A, n_ent, s);
            else le = launch_emit<float, 64>(c, A, n_ent, s);
        }
        if (le != cudaSuccess) return le;
    }
    int ntok = c.p.ctx_start + (c.p.T - c.c_end);
    c.launches += (nu > 0 ? 4 : 1) + (gu ? 2 : 0) + (ntok > 0 ? 1 : 0);
    if (ntok > 0) {
        dim3 g((ntok + 7) / 8, c.p.L * c.p.G);
        if (bf) gather_tokens_kernel<__nv_bfloat16><<<g, 256, 0, s>>>(A);
        else gather_tokens_kernel<float><<<g, 256, 0, s>>>(A);
    }
    return cudaGetLastError();
}

}  // namespace gkv
