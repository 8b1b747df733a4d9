// decode.cu -- decoding attention on the packed compressed cache.
//
// App. A.3, Eq. (app_decode_logit): a packed entry v of (layer l, KV head g)
// enters the attention of query head h (g = h / (Hq / G)) with the logit
//     x_v = q_h . k~_v / sqrt(d) + log m_v^eff ,
// and every token generated after the compression is appended to its (l, g)
// with effective multiplicity 1, i.e. log m = 0 (App. A.5, "Frontier updates
// and physical packing").  The output of head h is sum_v softmax(x)_v v~_v.
//
// The work is one read of the cache: 2 d elements per entry plus log m, with
// O(gq d) arithmetic per entry (gq = Hq / G query heads share one KV head).
// So the kernels are built for HBM bandwidth:
//
//   * The entries of the launch -- for every (l, g) its packed range
//     [off[lg], off[lg+1]) followed by its first n_app appended rows -- form one
//     virtual sequence that is cut into equal contiguous chunks, one per CTA,
//     whatever the per-head lengths (the global allocation makes them very
//     uneven).  A chunk meets one or more (l, g); each meeting is a "piece".
//   * One producer lane streams the rows of a piece through a ring of shared
//     memory, completion on mbarriers: the keys of a sub-chunk, then its
//     values; packed rows and appended rows go to separate stages.  bf16
//     caches arrive as 2-D TMA tiles with the 128-byte swizzle; fp32 caches as
//     1-D bulk copies of whole rows.  Keys and values are read from HBM once.
//   * bf16 (decode_tc_kernel): eight consumer warps run both products on the
//     tensor cores (m16n8k16, exact bf16 products, fp32 sums).  Logits: the
//     keys are the 16-row operand and the gq queries the 8-column one.  After
//     the sub-chunk maximum, the fp32 weights p = 2^(x - M) are split exactly
//     enough into three bf16 parts (hi + mid + lo, residual below 2^-26 p)
//     that form the 8-column operand of the value product, whose 16-row
//     operand is a 16-channel slice of the values (ldmatrix.trans); each warp
//     owns one channel slice, so its accumulator is the piece's result.
//   * fp32 (decode_cc_kernel): the same flow on CUDA cores -- packed fp32x2
//     FMA, a butterfly across the lanes of a row for the logits.
//   * A piece leaves (max, sum of weights, weighted value sum) per head.  The
//     CTA that finishes the last piece of an (l, g) -- found with an atomic
//     counter after a memory fence, nothing waits on anything -- merges the
//     pieces and writes the output; a head met by a single piece is written
//     directly.
//
// Every wait on an mbarrier is bounded in time; a wait that gives up records
// a status bit, lets the others run out without waiting and the CTA exits
// after the copies it issued have landed (or their own wait gave up).
#include "../../include/gracekv.h"
#include "tc.cuh"

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <atomic>
#include <cstring>

namespace gkv {
namespace {

constexpr int kDecWarps = 8;                         // consumer warps
constexpr int kDecThreads = (kDecWarps + 1) * 32;    // + one producer warp
constexpr int kDecStages = 8;                        // ring depth
constexpr int kDecStageBytes = 8192;                 // bytes per ring stage
constexpr int kDecMaxGrid = 1024;                    // partial slots beyond the heads
constexpr int kDecMaxHeads = 1023;                   // (l, g) heads of one launch (offsets in shared memory)
constexpr int kDecMinRows = 128;                     // rows a CTA takes at least (small launches)
constexpr int kDecStatusTimeout = 1;
constexpr int kDecStatusRange = 2;                   // offsets point past n_entries
constexpr uint64_t kDecWaitNs = 2000000000ull;
constexpr float kLog2e = 1.4426950408889634f;

// Floats of one piece's partial: the weighted value sums [gq][d], then the
// maxima [gq] and the weight sums [gq], padded so that every partial starts
// on a 64-byte boundary (the merge reads the sums as float4).
__host__ __device__ constexpr int dec_part_floats(int gq, int d) { return gq * d + 16; }

struct DecArgs {
    const char *K, *V;          // packed rows [E][d]
    const float *log_m;         // [E]
    const int64_t *off;         // [L G + 1]
    int64_t n_entries;          // rows of K, V, log_m
    const char *Ka, *Va;        // appended rows [L][G][app_cap][d]
    const void *q;              // [n_layers][Hq][d]
    float *out;                 // [n_layers][Hq][d]
    float *part;                // piece partials
    int *cnt;                   // [L G] pieces finished per head (reset by the merging CTA)
    int *status;
    int G, Hq, app_cap, n_app, s0, nS;
    float qscale;               // log2(e) / sqrt(d)
};

// Tensor maps of the bf16 path: [rows][d] with boxes of [RPS rows][64 columns]
// and the 128-byte swizzle, for the packed and the appended keys and values.
struct DecMaps {
    CUtensorMap K, V, Ka, Va;
};

template <typename T, int D, int GQ>
struct DecCfg {
    static constexpr bool TC = sizeof(T) == 2;               // bf16: tensor cores, swizzled tiles
    static constexpr int RB = D * (int)sizeof(T);            // bytes per row
    static constexpr int RPS = kDecStageBytes / RB;          // rows per ring stage
    static constexpr int SUB = TC ? (GQ < 8 ? 512 : 256) : 2048 / GQ;   // entries per sub-chunk
    static constexpr int EPT = SUB / (kDecWarps * 32);       // sub-chunk entries per consumer thread
    // tensor-core path
    static constexpr int NB = D / 64;                        // 64-column boxes per row
    static constexpr int TPS = RPS / 16;                     // 16-row steps per stage
    static constexpr int MAXST = SUB / RPS + 1;              // stages of one sub-chunk, at most
    static constexpr int NMT = D / 16;                       // 16-channel slices of the values
    static constexpr int WPM = kDecWarps / NMT;              // warps per slice
    static constexpr int FRW = MAXST * TPS * 3 * 64;         // words of the weight operands
    // CUDA-core path
    static constexpr int CPR = RB / 16;                      // 16-byte chunks per row
    static constexpr int LPR = CPR < 16 ? CPR : 16;          // lanes per row
    static constexpr int CPL = CPR / LPR;                    // chunks per lane
    static constexpr int EPC = 16 / (int)sizeof(T);          // elements per chunk
    static constexpr int EPL = CPL * EPC;                    // elements per lane
    static constexpr int RPW = 32 / LPR;                     // rows per warp step
    // shared memory after the head and the ring (floats)
    static constexpr int LGF = TC ? SUB * GQ : 2 * SUB * GQ; // logits (two buffers on CUDA cores)
    static constexpr int FRF = TC ? FRW : 0;
    static constexpr int REDF = TC ? (WPM > 1 ? WPM * GQ * D : 0) : kDecWarps * GQ * D;
    static constexpr int SUMF = GQ * D;
    static constexpr int VOFF = kDecMaxHeads + 1;            // the launch's offsets (int32, relative)
    static constexpr size_t SMEM =
        1024 + (size_t)kDecStages * kDecStageBytes + (size_t)(LGF + FRF + REDF + SUMF + VOFF) * sizeof(float);
    static_assert(SUB % RPS == 0 && SUB % (kDecWarps * 32) == 0, "decode sub-chunk");
    static_assert(!TC || (RPS % 16 == 0 && kDecWarps % NMT == 0 && TPS % WPM == 0), "decode tensor tiles");
    static_assert(TC || (GQ <= LPR && LPR * RPW == 32 && RPS % (kDecWarps * RPW) == 0), "decode lanes");
};

struct alignas(16) DecSmemHead {
    uint64_t full[kDecStages];
    uint64_t empty[kDecStages];
    float wmax[kDecWarps][8];
    float wsum[kDecWarps][8];
    float hsum[8];
    int abort;
    int last;
};

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t a[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t a[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float c[4], const uint32_t a[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Two floats rounded to bf16 (lo -> bits 0..15, hi -> bits 16..31).
__device__ __forceinline__ uint32_t bf16x2_rn(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Byte offset, inside a bf16 stage, of the 16-byte chunk `ch` of row r: the
// stage holds NB boxes of [RPS][128 B] written by TMA with the 128-byte
// swizzle (chunk ^ row % 8; stages are 1024-byte aligned).
template <int RPS>
__device__ __forceinline__ uint32_t sw_off(int r, int ch) {
    return (uint32_t)((ch >> 3) * RPS * 128 + r * 128 + (((ch & 7) ^ (r & 7)) << 4));
}

// Bounded wait that also gives up at once when another thread has given up.
__device__ __forceinline__ bool dec_wait(uint32_t bar, uint32_t parity, DecSmemHead &h, int *status) {
    if (tc::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = tc::globaltimer_ns();
    for (uint32_t it = 0;; it++) {
        if (tc::mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 63u) {
            if (*(volatile int *)&h.abort) return false;
            if (tc::globaltimer_ns() - t0 > kDecWaitNs) {
                atomicOr(status, kDecStatusTimeout);
                atomicExch(&h.abort, 1);
                return false;
            }
        }
    }
}

__device__ __forceinline__ void consumer_sync() {
    asm volatile("bar.sync 1, %0;" ::"r"(kDecWarps * 32) : "memory");
}

// The launch's heads as the CTA sees them: voff (shared memory) holds
// off[s] - off[s0] for s in [s0, s0 + nS].
struct DecView {
    const int *voff;
    int64_t base;               // off[s0]
    int s0, n_app;
    // virtual start of head s: its packed entries come first, then its appended rows
    __device__ __forceinline__ int64_t vstart(int s) const {
        return (int64_t)voff[s - s0] + (int64_t)(s - s0) * n_app;
    }
    __device__ __forceinline__ int64_t packed(int s) const { return voff[s + 1 - s0] - voff[s - s0]; }
    __device__ __forceinline__ int64_t first_row(int s) const { return base + voff[s - s0]; }
};
// Chunk (CTA) holding virtual index i when `total` entries are cut into
// `nc` chunks [floor(c total / nc), floor((c + 1) total / nc)).
__device__ __forceinline__ int chunk_of(int64_t i, int64_t total, int64_t nc) {
    return (int)(((i + 1) * nc + total - 1) / total - 1);
}

// The CTA's share of the launch: chunk [lo, hi) of the virtual sequence, the
// first head it meets, the number of chunks.  Loads the launch's offsets into
// shared memory first (one coalesced pass instead of a chain of dependent
// loads); block 0 also writes the zero outputs of heads without any entry.
// Returns false when the CTA has no work (or the offsets do not fit the cache).
template <int D, int GQ>
__device__ __forceinline__ bool dec_setup(const DecArgs &a, int *voff, DecView &v, int64_t &lo, int64_t &hi,
                                          int64_t &total, int64_t &nc, int &s_first) {
    const int tid = threadIdx.x;
    const int64_t base = a.off[a.s0];
    for (int i = tid; i <= a.nS; i += kDecThreads) voff[i] = (int)(a.off[a.s0 + i] - base);
    __syncthreads();
    v.voff = voff;
    v.base = base;
    v.s0 = a.s0;
    v.n_app = a.n_app;
    if (base + voff[a.nS] > a.n_entries) {      // the offsets do not fit the cache
        if (blockIdx.x == 0 && tid == 0) atomicOr(a.status, kDecStatusRange);
        return false;
    }
    total = v.vstart(a.s0 + a.nS);
    nc = total < (int64_t)gridDim.x ? total : (int64_t)gridDim.x;
    if (blockIdx.x == 0 && a.n_app == 0)
        for (int s = a.s0 + tid; s < a.s0 + a.nS; s += kDecThreads)
            if (v.packed(s) == 0) {
                float *o = a.out + ((size_t)(s / a.G - a.s0 / a.G) * a.Hq + (size_t)(s % a.G) * GQ) * D;
                for (int i = 0; i < GQ * D; i++) o[i] = 0.f;
            }
    if ((int64_t)blockIdx.x >= nc) return false;
    lo = (int64_t)blockIdx.x * total / nc;
    hi = ((int64_t)blockIdx.x + 1) * total / nc;
    int sb = a.s0, se = a.s0 + a.nS;              // the last s with vstart(s) <= lo
    while (se - sb > 1) {
        const int mid = (sb + se) >> 1;
        if (v.vstart(mid) <= lo) sb = mid; else se = mid;
    }
    s_first = sb;
    return true;
}

__device__ __forceinline__ void dec_init_barriers(DecSmemHead &hd) {
    if (threadIdx.x == 0) {
        for (int i = 0; i < kDecStages; i++) {
            tc::mbar_init(tc::smem_u32(&hd.full[i]), 1);
            tc::mbar_init(tc::smem_u32(&hd.empty[i]), kDecWarps);
        }
        hd.abort = 0;
        tc::fence_barrier_init();
    }
    __syncthreads();
}

// Producer lane: every stage of every piece of the chunk, in the order the
// consumers take them -- per sub-chunk the key stages, then the value stages;
// within each, the packed rows and then the appended rows, RPS rows a stage.
template <typename T, int D, int GQ>
__device__ void dec_produce(const DecArgs &a, const DecMaps &maps, const DecView &v, DecSmemHead &hd,
                            unsigned char *ring, int64_t lo, int64_t hi, int s_first) {
    using C = DecCfg<T, D, GQ>;
    if constexpr (C::TC) {
        tc::tma_prefetch_desc(&maps.K);
        tc::tma_prefetch_desc(&maps.V);
        tc::tma_prefetch_desc(&maps.Ka);
        tc::tma_prefetch_desc(&maps.Va);
    }
    uint32_t it = 0;
    bool ok = true;
    for (int s = s_first; ok && s < a.s0 + a.nS; s++) {
        const int64_t vs = v.vstart(s), ve = v.vstart(s + 1);
        if (vs >= hi) break;
        if (ve <= lo || ve == vs) continue;      // before the chunk, or no entry
        const int64_t pa = (lo > vs ? lo : vs) - vs, pb = (hi < ve ? hi : ve) - vs;
        const int64_t npk = v.packed(s);
        for (int64_t sa = pa; ok && sa < pb; sa += C::SUB) {
            const int64_t sbnd = sa + C::SUB < pb ? sa + C::SUB : pb;
            for (int kv = 0; ok && kv < 2; kv++)
                for (int part = 0; ok && part < 2; part++) {
                    const int64_t p0 = part ? (sa > npk ? sa : npk) : sa;
                    const int64_t p1 = part ? sbnd : (sbnd < npk ? sbnd : npk);
                    for (int64_t r0 = p0; r0 < p1; r0 += C::RPS, it++) {
                        const int st = it % kDecStages;
                        if (*(volatile int *)&hd.abort ||
                            !dec_wait(tc::smem_u32(&hd.empty[st]), ((it / kDecStages) & 1) ^ 1, hd, a.status)) {
                            ok = false;
                            break;
                        }
                        const int64_t nr = p1 - r0 < C::RPS ? p1 - r0 : C::RPS;
                        const int64_t row = part ? (int64_t)s * a.app_cap + (r0 - npk) : v.first_row(s) + r0;
                        const uint32_t fb = tc::smem_u32(&hd.full[st]);
                        const uint32_t dst = tc::smem_u32(ring + st * kDecStageBytes);
                        if constexpr (C::TC) {
                            // whole boxes (rows past the tensor read as zeros)
                            const CUtensorMap *mp = part ? (kv ? &maps.Va : &maps.Ka) : (kv ? &maps.V : &maps.K);
                            tc::mbar_expect_tx(fb, (uint32_t)(C::NB * C::RPS * 128));
#pragma unroll
                            for (int b = 0; b < C::NB; b++)
                                tc::tma_load_2d(dst + (uint32_t)(b * C::RPS * 128), mp, b * 64, (int)row, fb);
                        } else {
                            const char *src = part ? (kv ? a.Va : a.Ka) : (kv ? a.V : a.K);
                            tc::mbar_expect_tx(fb, (uint32_t)(nr * C::RB));
                            bulk_g2s(dst, src + row * C::RB, (uint32_t)(nr * C::RB), fb);
                        }
                    }
                }
        }
    }
    // the copies still in flight land before the block exits
    for (uint32_t i = it > kDecStages ? it - kDecStages : 0; i < it; i++)
        tc::mbar_wait(tc::smem_u32(&hd.full[i % kDecStages]), (i / kDecStages) & 1, kDecWaitNs);
}

// End of a piece: sums [GQ][D] (weighted value sums) and hd.hsum (sums of the
// weights) in shared memory, mrun the running maxima (base 2).  Writes the
// output when the piece is the whole head, else the piece's partial; the CTA
// finishing the head's last piece merges all of them, in parallel over the
// pieces and the outputs (scratch: at least 1024 floats of shared memory).
template <int D, int GQ>
__device__ __forceinline__ void dec_finish(const DecArgs &a, DecSmemHead &hd, const float *sums,
                                           const float (&mrun)[GQ], int s, int64_t vs, int64_t ve, int64_t total,
                                           int64_t nc, float *scratch) {
    constexpr int PART = dec_part_floats(GQ, D);
    static_assert(PART % 16 == 0 && 2 * GQ <= 16, "decode partial layout");
    constexpr int NT = kDecWarps * 32;
    constexpr int NQ = GQ * D / 4;                   // float4 groups of one partial's sums
    constexpr int NG = NT / NQ > 0 ? NT / NQ : 1;    // pieces taken at once
    static_assert(NG * GQ * D <= 1024 && (NQ <= NT ? NT % NQ == 0 : NQ % NT == 0), "decode merge tiling");
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int l_rel = s / a.G - a.s0 / a.G, g = s % a.G;
    const int c_lo = chunk_of(vs, total, nc), c_hi = chunk_of(ve - 1, total, nc);
    float *o_base = a.out + ((size_t)l_rel * a.Hq + (size_t)g * GQ) * D;
    if (c_lo == c_hi) {
        for (int i = tid; i < GQ * D; i += NT) o_base[i] = sums[i] / hd.hsum[i / D];
    } else {
        float *pp = a.part + (size_t)((s - a.s0) + (int)blockIdx.x) * PART;
        for (int i = tid; i < GQ * D; i += NT) pp[i] = sums[i];
#pragma unroll
        for (int h = 0; h < GQ; h++)
            if (tid == h) {
                pp[GQ * D + h] = mrun[h];
                pp[GQ * D + GQ + h] = hd.hsum[h];
            }
        __threadfence();
        consumer_sync();
        if (tid == 0) hd.last = (atomicAdd(a.cnt + s, 1) == c_hi - c_lo);
        consumer_sync();
        if (hd.last) {
            __threadfence();
            const int np = c_hi - c_lo + 1;
            const float *p0 = a.part + (size_t)((s - a.s0) + c_lo) * PART;   // the head's pieces, consecutive
            // overall maximum per head
            float mx[GQ];
#pragma unroll
            for (int h = 0; h < GQ; h++) mx[h] = -INFINITY;
            for (int p = tid; p < np; p += NT)
#pragma unroll
                for (int h = 0; h < GQ; h++) mx[h] = fmaxf(mx[h], __ldcg(p0 + (size_t)p * PART + GQ * D + h));
#pragma unroll
            for (int h = 0; h < GQ; h++) {
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], o));
                if (lane == 0) hd.wmax[warp][h] = mx[h];
            }
            consumer_sync();
            float M[GQ], den[GQ];
#pragma unroll
            for (int h = 0; h < GQ; h++) {
                M[h] = hd.wmax[0][h];
#pragma unroll
                for (int w = 1; w < kDecWarps; w++) M[h] = fmaxf(M[h], hd.wmax[w][h]);
                den[h] = 0.f;
            }
            // weight sums: pieces spread over the threads
            for (int p = tid; p < np; p += NT)
#pragma unroll
                for (int h = 0; h < GQ; h++) {
                    const float *q = p0 + (size_t)p * PART + GQ * D;
                    den[h] += tc::ex2(__ldcg(q + h) - M[h]) * __ldcg(q + GQ + h);
                }
            // value sums: thread = (group of NG pieces, float4 of the sums)
            for (int qd = tid % NQ; qd < NQ; qd += NT) {
                const int h = qd * 4 / D;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
                for (int p = tid / NQ; p < np; p += NG) {
                    const float *q = p0 + (size_t)p * PART;
                    const float w = tc::ex2(__ldcg(q + GQ * D + h) - M[h]);
                    const float4 x = __ldcg(reinterpret_cast<const float4 *>(q) + qd);
                    acc.x += w * x.x; acc.y += w * x.y; acc.z += w * x.z; acc.w += w * x.w;
                }
                if (tid / NQ < NG) reinterpret_cast<float4 *>(scratch)[(tid / NQ) * NQ + qd] = acc;
            }
#pragma unroll
            for (int h = 0; h < GQ; h++) {
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) den[h] += __shfl_xor_sync(0xffffffffu, den[h], o);
                if (lane == 0) hd.wsum[warp][h] = den[h];
            }
            consumer_sync();
            for (int i = tid; i < GQ * D; i += NT) {
                const int h = i / D;
                float num = 0.f, dd = 0.f;
#pragma unroll
                for (int k = 0; k < NG; k++) num += scratch[k * GQ * D + i];
#pragma unroll
                for (int w = 0; w < kDecWarps; w++) dd += hd.wsum[w][h];
                o_base[i] = num / dd;
            }
            if (tid == 0) a.cnt[s] = 0;
        }
    }
    consumer_sync();                 // the sums, the scratch and the head words are reused next
}

// Sub-chunk maximum of the base-2 logits (log m added into lg in place) and
// the rescaling factors of the running sums; returns via mrun / alpha.
template <int GQ, int EPT>
__device__ __forceinline__ void dec_subchunk_max(DecSmemHead &hd, float *lg, const float (&lmv)[EPT], int nsub,
                                                 float (&mrun)[GQ], float (&alpha)[GQ]) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    float mx[GQ];
#pragma unroll
    for (int h = 0; h < GQ; h++) mx[h] = -INFINITY;
#pragma unroll
    for (int i = 0; i < EPT; i++) {
        const int e = tid + i * (kDecWarps * 32);
        if (e < nsub) {
#pragma unroll
            for (int h = 0; h < GQ; h++) {
                const float x = lg[e * GQ + h] + lmv[i];
                lg[e * GQ + h] = x;
                mx[h] = fmaxf(mx[h], x);
            }
        }
    }
#pragma unroll
    for (int h = 0; h < GQ; h++) {
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], o));
        if (lane == 0) hd.wmax[warp][h] = mx[h];
    }
    consumer_sync();
#pragma unroll
    for (int h = 0; h < GQ; h++) {
        float m = hd.wmax[0][h];
#pragma unroll
        for (int w = 1; w < kDecWarps; w++) m = fmaxf(m, hd.wmax[w][h]);
        const float mn = fmaxf(mrun[h], m);
        alpha[h] = tc::ex2(mrun[h] - mn);          // 0 on the first sub-chunk
        mrun[h] = mn;
    }
}

// ============================ bf16: tensor cores ============================
template <int D, int GQ>
__global__ void __launch_bounds__(kDecThreads, 2)
    decode_tc_kernel(const DecArgs a, const __grid_constant__ DecMaps maps) {
    using C = DecCfg<__nv_bfloat16, D, GQ>;
    extern __shared__ __align__(1024) unsigned char dsm[];
    DecSmemHead &hd = *reinterpret_cast<DecSmemHead *>(dsm);
    unsigned char *ring = dsm + 1024;          // 1024-byte aligned stages (swizzle atoms)
    float *lg = reinterpret_cast<float *>(ring + kDecStages * kDecStageBytes);
    uint32_t *fr = reinterpret_cast<uint32_t *>(lg + C::LGF);
    float *red = reinterpret_cast<float *>(fr + C::FRF);
    float *sums = red + C::REDF;
    int *voff = reinterpret_cast<int *>(sums + C::SUMF);

    int64_t lo, hi, total, nc;
    int s_first;
    DecView v;
    if (!dec_setup<D, GQ>(a, voff, v, lo, hi, total, nc, s_first)) return;
    dec_init_barriers(hd);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (warp == kDecWarps) {
        if (lane == 0) dec_produce<__nv_bfloat16, D, GQ>(a, maps, v, hd, ring, lo, hi, s_first);
        return;
    }

    const int hq = lane >> 2, tq = lane & 3;               // MMA fragment row group / column pair
    const int mt = warp % C::NMT, kg = warp / C::NMT;      // this warp's value channels / row steps
    const int fl = (tid >> 1) % (4 * GQ);                  // lane of the weight operand this thread fills
    const int hs = fl >> 2;                                // ... and its head
    uint32_t it = 0;

    for (int s = s_first; s < a.s0 + a.nS; s++) {
        const int64_t vs = v.vstart(s), ve = v.vstart(s + 1);
        if (vs >= hi) break;
        if (ve <= lo || ve == vs) continue;
        const int64_t pa = (lo > vs ? lo : vs) - vs, pb = (hi < ve ? hi : ve) - vs;
        const int64_t npk = v.packed(s);
        const int l_rel = s / a.G - a.s0 / a.G, g = s % a.G;

        // the queries as the logit MMA's 16 x 8 column operand: column n = head
        // n (zero past GQ), k = channel, per 16-channel step
        uint32_t qb[D / 16][2];
        {
            const uint32_t *qh = reinterpret_cast<const uint32_t *>(
                static_cast<const __nv_bfloat16 *>(a.q) + ((size_t)l_rel * a.Hq + (size_t)g * GQ + (hq < GQ ? hq : 0)) * D);
#pragma unroll
            for (int kk = 0; kk < D / 16; kk++) {
                qb[kk][0] = hq < GQ ? __ldg(qh + kk * 8 + tq) : 0u;
                qb[kk][1] = hq < GQ ? __ldg(qh + kk * 8 + 4 + tq) : 0u;
            }
        }
        float acc[4] = {0.f, 0.f, 0.f, 0.f};   // channels 16 mt + hq (+8) x heads 2 tq, 2 tq + 1
        float mrun[GQ], lsum = 0.f;            // lsum: head hs
#pragma unroll
        for (int h = 0; h < GQ; h++) mrun[h] = -INFINITY;

        for (int64_t sa = pa; sa < pb; sa += C::SUB) {
            const int64_t sbnd = sa + C::SUB < pb ? sa + C::SUB : pb;
            const int nsub = (int)(sbnd - sa);
            const int pk_rel = (int)(npk - sa < 0 ? 0 : (npk - sa < nsub ? npk - sa : nsub));
            const int n_pk_st = (pk_rel + C::RPS - 1) / C::RPS;
            const int n_st = n_pk_st + (nsub - pk_rel + C::RPS - 1) / C::RPS;
            float lmv[C::EPT];
#pragma unroll
            for (int i = 0; i < C::EPT; i++) {
                const int64_t k = sa + tid + i * (kDecWarps * 32);
                lmv[i] = (k < sbnd && k < npk) ? __ldg(a.log_m + v.first_row(s) + k) * kLog2e : 0.f;
            }
            // ---- keys: lg[row][head] = q . k log2(e) / sqrt(d)
            for (int st = 0; st < n_st; st++, it++) {
                const int slot = it % kDecStages;
                dec_wait(tc::smem_u32(&hd.full[slot]), (it / kDecStages) & 1, hd, a.status);
                const int r0 = st < n_pk_st ? st * C::RPS : pk_rel + (st - n_pk_st) * C::RPS;
                const int nr = min(C::RPS, (st < n_pk_st ? pk_rel : nsub) - r0);
                const uint32_t sbase = tc::smem_u32(ring + slot * kDecStageBytes);
                const int mi = lane >> 3, ri = lane & 7;
#pragma unroll
                for (int t = 0; t < C::TPS; t++) {
                    if ((int)((it * C::TPS + t) % kDecWarps) != warp || t * 16 >= nr) continue;
                    float c[4] = {0.f, 0.f, 0.f, 0.f};
                    const int ar = t * 16 + ri + (mi & 1) * 8;     // row this lane addresses
#pragma unroll
                    for (int kk = 0; kk < D / 16; kk++) {
                        uint32_t af[4];
                        ldsm_x4(sbase + sw_off<C::RPS>(ar, kk * 2 + (mi >> 1)), af);
                        mma16816(c, af, qb[kk][0], qb[kk][1]);
                    }
                    // c[0], c[1]: row hq, heads 2 tq, 2 tq + 1; c[2], c[3]: row hq + 8
                    const int h0 = 2 * tq, ra = t * 16 + hq, rb = ra + 8;
                    if (h0 < GQ) {
                        if (ra < nr) lg[(r0 + ra) * GQ + h0] = c[0] * a.qscale;
                        if (rb < nr) lg[(r0 + rb) * GQ + h0] = c[2] * a.qscale;
                    }
                    if (h0 + 1 < GQ) {
                        if (ra < nr) lg[(r0 + ra) * GQ + h0 + 1] = c[1] * a.qscale;
                        if (rb < nr) lg[(r0 + rb) * GQ + h0 + 1] = c[3] * a.qscale;
                    }
                }
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(tc::smem_u32(&hd.empty[slot]));
            }
            consumer_sync();
            float alpha[GQ];
            dec_subchunk_max<GQ, C::EPT>(hd, lg, lmv, nsub, mrun, alpha);
            float ahs = alpha[0], Mh = mrun[0];            // this thread's head (no dynamic indexing)
#pragma unroll
            for (int h = 1; h < GQ; h++)
                if (h == hs) { ahs = alpha[h]; Mh = mrun[h]; }
            lsum *= ahs;
            {
                float a0 = 0.f, a1 = 0.f;                  // heads 2 tq, 2 tq + 1 (0 past GQ)
#pragma unroll
                for (int h = 0; h < GQ; h++) {
                    if (h == 2 * tq) a0 = alpha[h];
                    if (h == 2 * tq + 1) a1 = alpha[h];
                }
                acc[0] *= a0; acc[1] *= a1; acc[2] *= a0; acc[3] *= a1;
            }
            // ---- weights as the value MMA's column operand: for each stage and
            // 16-row step, lane (head h, tq) holds rows 2 tq, 2 tq + 1 (word 0)
            // and 2 tq + 8, 2 tq + 9 (word 1); p = hi + mid + lo in bf16
            {
                const int reg = tid & 1, t4 = fl & 3;
                const int nw = n_st * C::TPS * 8 * GQ;          // words of this sub-chunk
                for (int w = tid; w < nw; w += kDecWarps * 32) {
                    const int ksst = (w >> 1) / (4 * GQ);
                    const int ks = ksst % C::TPS, st = ksst / C::TPS;
                    const int r0 = st < n_pk_st ? st * C::RPS : pk_rel + (st - n_pk_st) * C::RPS;
                    const int nr = min(C::RPS, (st < n_pk_st ? pk_rel : nsub) - r0);
                    const int rr = ks * 16 + reg * 8 + 2 * t4;
                    const float p0 = rr < nr ? tc::ex2(lg[(r0 + rr) * GQ + hs] - Mh) : 0.f;
                    const float p1 = rr + 1 < nr ? tc::ex2(lg[(r0 + rr + 1) * GQ + hs] - Mh) : 0.f;
                    lsum += p0 + p1;
                    const uint32_t w_hi = bf16x2_rn(p0, p1);
                    const float r10 = p0 - __uint_as_float(w_hi << 16), r11 = p1 - __uint_as_float(w_hi & 0xffff0000u);
                    const uint32_t w_mid = bf16x2_rn(r10, r11);
                    const float r20 = r10 - __uint_as_float(w_mid << 16), r21 = r11 - __uint_as_float(w_mid & 0xffff0000u);
                    const uint32_t w_lo = bf16x2_rn(r20, r21);
                    uint32_t *dst = fr + (size_t)(st * C::TPS + ks) * 3 * 64 + fl * 2 + reg;
                    dst[0] = w_hi;
                    dst[64] = w_mid;
                    dst[128] = w_lo;
                }
            }
            consumer_sync();
            // ---- values: acc[channels][heads] += V^T P over this warp's row steps
            for (int st = 0; st < n_st; st++, it++) {
                const int slot = it % kDecStages;
                dec_wait(tc::smem_u32(&hd.full[slot]), (it / kDecStages) & 1, hd, a.status);
                const uint32_t sbase = tc::smem_u32(ring + slot * kDecStageBytes);
                const int mi = lane >> 3;
#pragma unroll
                for (int ks = 0; ks < C::TPS; ks++) {
                    if (ks % C::WPM != kg) continue;
                    uint32_t af[4];
                    // rows 16 ks + (lane & 7) + 8 (mi >> 1), channels 16 mt + 8 (mi & 1) .. + 7
                    ldsm_x4_t(sbase + sw_off<C::RPS>(ks * 16 + (lane & 7) + (mi >> 1) * 8, mt * 2 + (mi & 1)), af);
                    const uint32_t *b = fr + (size_t)(st * C::TPS + ks) * 3 * 64 + lane * 2;
#pragma unroll
                    for (int part = 0; part < 3; part++) {
                        const uint2 bw = *reinterpret_cast<const uint2 *>(b + part * 64);
                        mma16816(acc, af, bw.x, bw.y);
                    }
                }
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(tc::smem_u32(&hd.empty[slot]));
            }
        }

        // ---- piece result: weight sums per head, value sums per (head, channel)
        // lanes 8k .. 8k + 7 of warp w share the head (4 w + k) % GQ
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
        if ((lane & 7) == 0) hd.wsum[warp][lane >> 3] = lsum;
        {
            const int d0 = mt * 16 + hq, h0 = 2 * tq;
            float *dst = C::WPM > 1 ? red + (size_t)kg * GQ * D : sums;
            if (h0 < GQ) { dst[h0 * D + d0] = acc[0]; dst[h0 * D + d0 + 8] = acc[2]; }
            if (h0 + 1 < GQ) { dst[(h0 + 1) * D + d0] = acc[1]; dst[(h0 + 1) * D + d0 + 8] = acc[3]; }
        }
        consumer_sync();
        if (tid < GQ) {                  // fixed order: results do not depend on timing
            float v = 0.f;
#pragma unroll
            for (int w = 0; w < kDecWarps; w++)
#pragma unroll
                for (int k = 0; k < 4; k++)
                    if ((4 * w + k) % GQ == tid) v += hd.wsum[w][k];
            hd.hsum[tid] = v;
        }
        if constexpr (C::WPM > 1) {
            for (int i = tid; i < GQ * D; i += kDecWarps * 32) {
                float v = 0.f;
#pragma unroll
                for (int k = 0; k < C::WPM; k++) v += red[(size_t)k * GQ * D + i];
                sums[i] = v;
            }
        }
        consumer_sync();
        dec_finish<D, GQ>(a, hd, sums, mrun, s, vs, ve, total, nc, reinterpret_cast<float *>(fr));
    }
}

// ============================ fp32: CUDA cores ==============================
template <typename T>
__device__ __forceinline__ void chunk_to_float(const uint4 &u, float *f) {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
}

template <int D, int GQ>
__global__ void __launch_bounds__(kDecThreads, 2)
    decode_cc_kernel(const DecArgs a, const __grid_constant__ DecMaps maps) {
    using T = float;
    using C = DecCfg<T, D, GQ>;
    extern __shared__ __align__(1024) unsigned char dsm[];
    DecSmemHead &hd = *reinterpret_cast<DecSmemHead *>(dsm);
    unsigned char *ring = dsm + 1024;
    float *lgb = reinterpret_cast<float *>(ring + kDecStages * kDecStageBytes);
    float *red = lgb + C::LGF;
    float *sums = red + C::REDF;
    int *voff = reinterpret_cast<int *>(sums + C::SUMF);

    int64_t lo, hi, total, nc;
    int s_first;
    DecView v;
    if (!dec_setup<D, GQ>(a, voff, v, lo, hi, total, nc, s_first)) return;
    dec_init_barriers(hd);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (warp == kDecWarps) {
        if (lane == 0) dec_produce<T, D, GQ>(a, maps, v, hd, ring, lo, hi, s_first);
        return;
    }

    const int rg = lane / C::LPR, j = lane % C::LPR;
    const int hsel = j / (C::LPR / GQ);                 // head whose logit this lane ends with
    const bool writer = (j % (C::LPR / GQ)) == 0;
    uint32_t it = 0;
    int buf = 0;

    for (int s = s_first; s < a.s0 + a.nS; s++) {
        const int64_t vs = v.vstart(s), ve = v.vstart(s + 1);
        if (vs >= hi) break;
        if (ve <= lo || ve == vs) continue;
        const int64_t pa = (lo > vs ? lo : vs) - vs, pb = (hi < ve ? hi : ve) - vs;
        const int64_t npk = v.packed(s);
        const int l_rel = s / a.G - a.s0 / a.G, g = s % a.G;

        // this lane's elements of the GQ queries, pre-scaled to base 2
        float2 q2[GQ][C::EPL / 2];
#pragma unroll
        for (int h = 0; h < GQ; h++) {
            const T *qh = static_cast<const T *>(a.q) + ((size_t)l_rel * a.Hq + (size_t)g * GQ + h) * D;
#pragma unroll
            for (int c = 0; c < C::CPL; c++) {
                float f[C::EPC];
                chunk_to_float<T>(__ldg(reinterpret_cast<const uint4 *>(qh) + j + C::LPR * c), f);
#pragma unroll
                for (int e = 0; e < C::EPC; e += 2)
                    q2[h][(c * C::EPC + e) / 2] = make_float2(f[e] * a.qscale, f[e + 1] * a.qscale);
            }
        }
        float2 acc[GQ][C::EPL / 2];
#pragma unroll
        for (int h = 0; h < GQ; h++)
#pragma unroll
            for (int e = 0; e < C::EPL / 2; e++) acc[h][e] = make_float2(0.f, 0.f);
        float mrun[GQ], lsum[GQ];
#pragma unroll
        for (int h = 0; h < GQ; h++) { mrun[h] = -INFINITY; lsum[h] = 0.f; }

        for (int64_t sa = pa; sa < pb; sa += C::SUB) {
            const int64_t sbnd = sa + C::SUB < pb ? sa + C::SUB : pb;
            const int nsub = (int)(sbnd - sa);
            float *lg = lgb + buf * (C::SUB * GQ);
            buf ^= 1;
            float lmv[C::EPT];
#pragma unroll
            for (int i = 0; i < C::EPT; i++) {
                const int64_t k = sa + tid + i * (kDecWarps * 32);
                lmv[i] = (k < sbnd && k < npk) ? __ldg(a.log_m + v.first_row(s) + k) * kLog2e : 0.f;
            }
            // ---- keys: base-2 logits into lg[row][head]
            for (int part = 0; part < 2; part++) {
                const int64_t p0 = part ? (sa > npk ? sa : npk) : sa;
                const int64_t p1 = part ? sbnd : (sbnd < npk ? sbnd : npk);
                for (int64_t r0l = p0; r0l < p1; r0l += C::RPS, it++) {
                    const int slot = it % kDecStages;
                    dec_wait(tc::smem_u32(&hd.full[slot]), (it / kDecStages) & 1, hd, a.status);
                    const int nr = (int)(p1 - r0l < C::RPS ? p1 - r0l : C::RPS);
                    const int r0 = (int)(r0l - sa);
                    const unsigned char *stage = ring + slot * kDecStageBytes;
#pragma unroll
                    for (int k = 0; k < C::RPS / (kDecWarps * C::RPW); k++) {
                        const int r = (k * kDecWarps + warp) * C::RPW + rg;
                        if ((k * kDecWarps + warp) * C::RPW >= nr) break;
                        float v[GQ];
#pragma unroll
                        for (int h = 0; h < GQ; h++) v[h] = 0.f;
#pragma unroll
                        for (int c = 0; c < C::CPL; c++) {
                            const uint4 u = *reinterpret_cast<const uint4 *>(stage + r * C::RB + (j + C::LPR * c) * 16);
                            float f[C::EPC];
                            chunk_to_float<T>(u, f);
#pragma unroll
                            for (int h = 0; h < GQ; h++) {
                                float2 p2 = make_float2(0.f, 0.f);
#pragma unroll
                                for (int e = 0; e < C::EPC; e += 2)
                                    p2 = __ffma2_rn(q2[h][(c * C::EPC + e) / 2], make_float2(f[e], f[e + 1]), p2);
                                v[h] += p2.x + p2.y;
                            }
                        }
                        // butterfly over the lanes of the row: each step halves the
                        // heads a lane keeps until every lane holds one full sum
#pragma unroll
                        for (int step = 0; (C::LPR >> (step + 1)) >= 1; step++) {
                            const int o = C::LPR >> (step + 1);
                            const int nv = (GQ >> step) > 1 ? (GQ >> step) : 1;
                            if (nv > 1) {
                                const bool up = (lane & o) != 0;
#pragma unroll
                                for (int i = 0; i < nv / 2; i++) {
                                    const float send = up ? v[i] : v[i + nv / 2];
                                    const float keep = up ? v[i + nv / 2] : v[i];
                                    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                                }
                            } else {
                                v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
                            }
                        }
                        if (writer && r < nr) lg[(r0 + r) * GQ + hsel] = v[0];
                    }
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(tc::smem_u32(&hd.empty[slot]));
                }
            }
            consumer_sync();
            float alpha[GQ];
            dec_subchunk_max<GQ, C::EPT>(hd, lg, lmv, nsub, mrun, alpha);
#pragma unroll
            for (int h = 0; h < GQ; h++) lsum[h] *= alpha[h];
            // ---- weights p = 2^(x - M) in place of the logits
#pragma unroll
            for (int i = 0; i < C::EPT; i++) {
                const int e = tid + i * (kDecWarps * 32);
                if (e < nsub) {
#pragma unroll
                    for (int h = 0; h < GQ; h++) {
                        const float p = tc::ex2(lg[e * GQ + h] - mrun[h]);
                        lsum[h] += p;
                        lg[e * GQ + h] = p;
                    }
                }
            }
#pragma unroll
            for (int h = 0; h < GQ; h++)
#pragma unroll
                for (int e = 0; e < C::EPL / 2; e++) {
                    acc[h][e].x *= alpha[h];
                    acc[h][e].y *= alpha[h];
                }
            consumer_sync();
            // ---- values: acc[h] += p[h] v
            for (int part = 0; part < 2; part++) {
                const int64_t p0 = part ? (sa > npk ? sa : npk) : sa;
                const int64_t p1 = part ? sbnd : (sbnd < npk ? sbnd : npk);
                for (int64_t r0l = p0; r0l < p1; r0l += C::RPS, it++) {
                    const int slot = it % kDecStages;
                    dec_wait(tc::smem_u32(&hd.full[slot]), (it / kDecStages) & 1, hd, a.status);
                    const int nr = (int)(p1 - r0l < C::RPS ? p1 - r0l : C::RPS);
                    const int r0 = (int)(r0l - sa);
                    const unsigned char *stage = ring + slot * kDecStageBytes;
#pragma unroll
                    for (int k = 0; k < C::RPS / (kDecWarps * C::RPW); k++) {
                        const int r = (k * kDecWarps + warp) * C::RPW + rg;
                        if ((k * kDecWarps + warp) * C::RPW >= nr) break;
                        if (r < nr) {
                            float p[GQ];
#pragma unroll
                            for (int h = 0; h < GQ; h++) p[h] = lg[(r0 + r) * GQ + h];
#pragma unroll
                            for (int c = 0; c < C::CPL; c++) {
                                const uint4 u = *reinterpret_cast<const uint4 *>(stage + r * C::RB + (j + C::LPR * c) * 16);
                                float f[C::EPC];
                                chunk_to_float<T>(u, f);
#pragma unroll
                                for (int h = 0; h < GQ; h++)
#pragma unroll
                                    for (int e = 0; e < C::EPC; e += 2)
                                        acc[h][(c * C::EPC + e) / 2] =
                                            __ffma2_rn(make_float2(p[h], p[h]), make_float2(f[e], f[e + 1]),
                                                       acc[h][(c * C::EPC + e) / 2]);
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(tc::smem_u32(&hd.empty[slot]));
                }
            }
        }

        // ---- piece result: sum the row groups of each warp, then the warps
#pragma unroll
        for (int o = C::LPR; o < 32; o <<= 1)
#pragma unroll
            for (int h = 0; h < GQ; h++)
#pragma unroll
                for (int e = 0; e < C::EPL / 2; e++) {
                    acc[h][e].x += __shfl_xor_sync(0xffffffffu, acc[h][e].x, o);
                    acc[h][e].y += __shfl_xor_sync(0xffffffffu, acc[h][e].y, o);
                }
#pragma unroll
        for (int h = 0; h < GQ; h++) {
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) lsum[h] += __shfl_xor_sync(0xffffffffu, lsum[h], o);
            if (lane == 0) hd.wsum[warp][h] = lsum[h];
        }
        consumer_sync();                 // the last values pass is done with the logit buffers
        if (rg == 0) {
#pragma unroll
            for (int h = 0; h < GQ; h++)
#pragma unroll
                for (int c = 0; c < C::CPL; c++)
#pragma unroll
                    for (int e = 0; e < C::EPC; e += 2)
                        *reinterpret_cast<float2 *>(red + ((size_t)warp * GQ + h) * D + (j + C::LPR * c) * C::EPC + e) =
                            acc[h][(c * C::EPC + e) / 2];
        }
        consumer_sync();
        for (int i = tid; i < GQ * D; i += kDecWarps * 32) {
            float v = 0.f;
#pragma unroll
            for (int w = 0; w < kDecWarps; w++) v += red[(size_t)w * GQ * D + i];
            sums[i] = v;
        }
        if (tid < GQ) {
            float v = 0.f;
#pragma unroll
            for (int w = 0; w < kDecWarps; w++) v += hd.wsum[w][tid];
            hd.hsum[tid] = v;
        }
        consumer_sync();
        dec_finish<D, GQ>(a, hd, sums, mrun, s, vs, ve, total, nc, lgb);
    }
}

__global__ void decode_append_kernel(const uint4 *k_new, const uint4 *v_new, uint4 *Ka, uint4 *Va, int G,
                                     int l0, int app_cap, int row, int row_chunks, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const int rlg = i / row_chunks, c = i % row_chunks;         // rlg = (l - l0) G + g
    const size_t dst = ((size_t)(l0 * G + rlg) * app_cap + row) * row_chunks + c;
    Ka[dst] = k_new[i];
    Va[dst] = v_new[i];
}

constexpr int kDecMaxDevices = 64;

// Grid of one launch: as many CTAs as fit on the device at once (set up once
// per device and instantiation; the shared-memory opt-in is per device).
// Grid of one launch: as many CTAs as fit on the device at once (set up once
// per device and instantiation; the shared-memory opt-in is per device), fewer
// when the launch holds fewer than kDecMinRows rows per CTA (estimated from
// the average head length): small launches then split each head into fewer
// pieces, which shortens the merge.
template <typename T, int D, int GQ>
cudaError_t launch_decode(const DecArgs &a, const DecMaps &m, int64_t rows_est, int dev, cudaStream_t s) {
    using C = DecCfg<T, D, GQ>;
    static std::atomic<int> grid_of[kDecMaxDevices];
    const size_t smem = C::SMEM;
    static_assert(sizeof(DecSmemHead) <= 1024, "decode shared-memory head");
    auto kern = C::TC ? decode_tc_kernel<D, GQ> : decode_cc_kernel<D, GQ>;
    if (dev < 0 || dev >= kDecMaxDevices) return cudaErrorInvalidDevice;
    int grid = grid_of[dev].load(std::memory_order_relaxed);
    if (grid == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        int per_sm = 1, sms = 1;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kDecThreads, smem);
        if (e != cudaSuccess) return e;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        grid = std::min(kDecMaxGrid, std::max(1, per_sm) * sms);
        grid_of[dev].store(grid, std::memory_order_relaxed);
    }
    grid = (int)std::max<int64_t>(1, std::min<int64_t>(grid, (rows_est + kDecMinRows - 1) / kDecMinRows));
    kern<<<grid, kDecThreads, smem, s>>>(a, m);
    return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_decode_gq(const DecArgs &a, const DecMaps &m, int gq, int64_t rows, int dev, cudaStream_t s) {
    switch (gq) {
        case 1: return launch_decode<T, D, 1>(a, m, rows, dev, s);
        case 2: return launch_decode<T, D, 2>(a, m, rows, dev, s);
        case 4: return launch_decode<T, D, 4>(a, m, rows, dev, s);
        case 8: return launch_decode<T, D, 8>(a, m, rows, dev, s);
        default: return cudaErrorInvalidValue;
    }
}

// [rows][d] bf16 rows, boxes of [box_rows][64 columns], 128-byte swizzle.
bool dec_map(CUtensorMap *m, const void *p, int64_t rows, int d, int box_rows) {
    auto enc = tc::tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)(rows > 0 ? rows : 1)};
    cuuint64_t gstr[1] = {(cuuint64_t)d * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p), gdim, gstr, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool al(const void *p, uintptr_t m) { return (reinterpret_cast<uintptr_t>(p) & (m - 1)) == 0; }

gkv_status check_cache(const gkv_decode_cache *c) {
    if (!c) return GKV_EINVAL;
    if (c->L <= 0 || c->G <= 0 || c->Hq <= 0 || c->Hq % c->G || c->app_cap < 0) return GKV_EINVAL;
    if (c->dtype != GKV_F32 && c->dtype != GKV_BF16) return GKV_EINVAL;
    const int gq = c->Hq / c->G;
    if ((c->d != 64 && c->d != 128) || (gq != 1 && gq != 2 && gq != 4 && gq != 8)) return GKV_EUNSUPPORTED;
    if (!c->K || !c->V || !c->log_m || !c->offsets || c->n_entries < 0 || c->n_entries >= (1LL << 31))
        return GKV_EINVAL;
    if (!al(c->K, 16) || !al(c->V, 16) || !al(c->log_m, 4) || !al(c->offsets, 8)) return GKV_EINVAL;
    if (c->app_cap > 0 && (!c->K_app || !c->V_app || !al(c->K_app, 16) || !al(c->V_app, 16))) return GKV_EINVAL;
    return GKV_OK;
}

size_t part_floats(const gkv_decode_cache *c) {
    return (size_t)((int64_t)c->L * c->G + kDecMaxGrid) * dec_part_floats(c->Hq / c->G, c->d);
}
constexpr size_t kWsHeadBytes = 256;    // status word + padding
size_t cnt_bytes(const gkv_decode_cache *c) { return (((size_t)c->L * c->G * sizeof(int)) + 255) / 256 * 256; }

}  // namespace
}  // namespace gkv

using namespace gkv;

extern "C" gkv_status gracekv_decode_workspace_size(const gkv_decode_cache *c, size_t *bytes) {
    const gkv_status st = check_cache(c);
    if (st != GKV_OK) return st;
    if (!bytes) return GKV_EINVAL;
    *bytes = kWsHeadBytes + cnt_bytes(c) + part_floats(c) * sizeof(float);
    return GKV_OK;
}

extern "C" gkv_status gracekv_decode_append(const gkv_decode_cache *c, int32_t l0, int32_t n_layers,
                                            int32_t n_app, const void *k_new, const void *v_new, void *stream) {
    const gkv_status st = check_cache(c);
    if (st != GKV_OK) return st;
    if (l0 < 0 || n_layers <= 0 || l0 + n_layers > c->L || n_app < 0) return GKV_EINVAL;
    if (n_app >= c->app_cap) return GKV_ECAPACITY;
    if (!k_new || !v_new || !al(k_new, 16) || !al(v_new, 16)) return GKV_EINVAL;
    const int row_chunks = c->d * (c->dtype == GKV_BF16 ? 2 : 4) / 16;
    const int n = n_layers * c->G * row_chunks;
    decode_append_kernel<<<(n + 255) / 256, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(k_new), static_cast<const uint4 *>(v_new), static_cast<uint4 *>(c->K_app),
        static_cast<uint4 *>(c->V_app), c->G, l0, c->app_cap, n_app, row_chunks, n);
    return cudaGetLastError() == cudaSuccess ? GKV_OK : GKV_ECUDA;
}

extern "C" gkv_status gracekv_decode_attention(const gkv_decode_cache *c, int32_t l0, int32_t n_layers,
                                               int32_t n_app, const void *q, float *out, void *workspace,
                                               void *stream) {
    const gkv_status st = check_cache(c);
    if (st != GKV_OK) return st;
    if (l0 < 0 || n_layers <= 0 || l0 + n_layers > c->L || n_app < 0 || n_app > c->app_cap) return GKV_EINVAL;
    if (!q || !out || !workspace || !al(q, 16) || !al(out, 16) || !al(workspace, 256)) return GKV_EINVAL;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GKV_ECUDA;
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    DecArgs a;
    a.K = static_cast<const char *>(c->K);
    a.V = static_cast<const char *>(c->V);
    a.log_m = c->log_m;
    a.off = c->offsets;
    a.n_entries = c->n_entries;
    a.Ka = static_cast<const char *>(c->K_app);
    a.Va = static_cast<const char *>(c->V_app);
    a.q = q;
    a.out = out;
    a.status = reinterpret_cast<int *>(ws);
    a.cnt = reinterpret_cast<int *>(ws + kWsHeadBytes);
    a.part = reinterpret_cast<float *>(ws + kWsHeadBytes + cnt_bytes(c));
    a.G = c->G;
    a.Hq = c->Hq;
    a.app_cap = c->app_cap;
    a.n_app = n_app;
    a.s0 = l0 * c->G;
    a.nS = n_layers * c->G;
    a.qscale = (float)(1.4426950408889634 / sqrt((double)c->d));
    const int gq = c->Hq / c->G;
    if (c->G > kDecMaxHeads) return GKV_EUNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DecMaps m;
    memset(&m, 0, sizeof(m));
    cudaError_t e = cudaSuccess;
    if (c->dtype == GKV_BF16) {
        const int box_rows = kDecStageBytes / (c->d * 2);
        const int64_t app_rows = (int64_t)c->L * c->G * c->app_cap;
        const void *ka = c->app_cap > 0 ? c->K_app : c->K, *va = c->app_cap > 0 ? c->V_app : c->V;
        if (!dec_map(&m.K, c->K, c->n_entries, c->d, box_rows) || !dec_map(&m.V, c->V, c->n_entries, c->d, box_rows) ||
            !dec_map(&m.Ka, ka, c->app_cap > 0 ? app_rows : 1, c->d, box_rows) ||
            !dec_map(&m.Va, va, c->app_cap > 0 ? app_rows : 1, c->d, box_rows))
            return GKV_ECUDA;
    }
    // one launch covers at most kDecMaxHeads heads (its offsets sit in shared
    // memory): longer layer ranges run as consecutive launches
    const int lpl = kDecMaxHeads / c->G;
    const size_t esz = c->dtype == GKV_BF16 ? 2 : 4;
    for (int lb = 0; lb < n_layers; lb += lpl) {
        const int nl = std::min(lpl, n_layers - lb);
        DecArgs b = a;
        b.s0 = (l0 + lb) * c->G;
        b.nS = nl * c->G;
        b.q = static_cast<const char *>(q) + (size_t)lb * c->Hq * c->d * esz;
        b.out = out + (size_t)lb * c->Hq * c->d;
        const int64_t rows = c->n_entries * b.nS / ((int64_t)c->L * c->G) + (int64_t)b.nS * n_app;
        if (c->dtype == GKV_BF16)
            e = c->d == 128 ? launch_decode_gq<__nv_bfloat16, 128>(b, m, gq, rows, dev, s)
                            : launch_decode_gq<__nv_bfloat16, 64>(b, m, gq, rows, dev, s);
        else
            e = c->d == 128 ? launch_decode_gq<float, 128>(b, m, gq, rows, dev, s)
                            : launch_decode_gq<float, 64>(b, m, gq, rows, dev, s);
        if (e != cudaSuccess) return GKV_ECUDA;
    }
    return GKV_OK;
}

extern "C" gkv_status gracekv_decode_status(void *workspace, void *stream) {
    if (!workspace || !al(workspace, 256)) return GKV_EINVAL;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int h = 0;
    if (cudaMemcpyAsync(&h, workspace, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return GKV_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return GKV_ECUDA;
    if (h == 0) return GKV_OK;
    if (cudaMemsetAsync(workspace, 0, sizeof(int), s) != cudaSuccess) return GKV_ECUDA;
    return (h & kDecStatusRange) ? GKV_EINVAL : GKV_ETIMEOUT;
}
