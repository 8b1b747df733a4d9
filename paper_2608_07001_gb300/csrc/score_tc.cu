// score_tc.cu -- the two observation-query x key score passes on the
// tensor cores of the sm_100 family (tcgen05.mma with accumulators in TMEM,
// operands staged by TMA), for bf16 inputs with d in {64, 128} and at most
// 256 probe rows per KV head.
//
//   row_stats_tc     pass A (App. A.3 max-logit shift; App. A.4 Eq.
//                    app_attention_probability denominators).  For every probe
//                    row r of KV head (l, g) and token chunk: the max logit
//                    m_r = max_t q_r.k_t / sqrt(d), Z_r = sum_t exp(x_rt - m_r) and
//                    Z^C_r, the same sum over the chunk's part of the compressible
//                    context C.  S = Q K^T with the rows in TMEM lanes (two halves
//                    of 128 rows) and 128 tokens per tile in columns: one thread
//                    owns one row and keeps its running (max, Z, Z^C).
//   token_values_tc  pass B (App. A.4 Eqs. app_direct_relevance,
//                    app_bottom_up_value with lambda_graph = 0).
//                    s_t = sum_r exp(x_rt - m_r) / Z_r and
//                    shat_t = s_t / (sum_r Z^C_r / Z_r + eps).  S^T = K Q^T with 128
//                    tokens in TMEM lanes and the rows in columns: one thread owns
//                    one token and sums over its rows.
//
// Warp roles (320 threads): warps 0-7 read the accumulators (warp w reaches
// TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31), warp 8 issues the TMA loads, and
// warp 9 allocates TMEM and issues the MMAs.  Key tiles of 128 tokens stream
// through a 4-stage ring of shared memory.  The accumulator is double-buffered
// in TMEM, so the MMA of tile i + 1 overlaps the exponentials of tile i
// (pass B: warps 0-3 take the even tiles and warps 4-7 the odd ones).
// Products of bf16 values are exact and the sums are fp32, as in the mma.sync
// kernels of score.cu.  Exponentials run in base 2 on logits pre-scaled by
// log2(e) / sqrt(d).
//
// Every wait is bounded (tc::mbar_wait): a wait that gives up sets the status
// bit kStPipeTimeout, lets the other roles run out, waits for the copies and
// MMAs already issued and frees TMEM before the block exits.
#include "gkv_internal.cuh"
#include "tc.cuh"

#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

namespace gkv {
namespace {

constexpr int kTcTile = 128;           // tokens per key tile
constexpr int kTcStages = 4;           // key tiles in flight
constexpr int kTcThreads = 320;        // 8 accumulator warps + TMA warp + MMA warp
constexpr int kTcWarpTma = 8, kTcWarpMma = 9;
constexpr uint32_t kBox = 128 * 128;   // bytes of one [128 rows][64 bf16] swizzled box
constexpr uint64_t kWaitNs = 2000000000ull;
constexpr float kLog2e = 1.4426950408889634f;

struct TcArgs {
    int T, G, Hq, W, gq, Rg, cs, cend, Nc, nrow_all;
    int t_lo, t_hi;          // token range the pass covers for every (l, g)
    int chunk_tiles, nch;    // tiles per block, blocks per (l, g)
    int nq;                  // probe rows staged: 128 * halves (pass A) or the padded width N (pass B)
    int lg0;                 // first (l, g) of the launch (grid.y covers the following ones)
    float scale;             // log2(e) / sqrt(d)
};

__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

struct TcBars {
    unsigned long long full[kTcStages], empty[kTcStages], accfull[2], accempty[2], qfull;
    uint32_t tbase;
    int abort;
};

// MODE 0: pass A (row statistics); MODE 1: pass B (token values).
template <int DH, int MODE>
__global__ void __launch_bounds__(kTcThreads, 1) score_tc_kernel(
        const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapQ,
        const __grid_constant__ CUtensorMap mapQ1, const short *qperm, TcArgs a,
        const float *rmneg, const double *lg_scale, float *part, float *rtok, int *status,
        const float *rm, float *Eg) {
    constexpr int NKB = DH / 64;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char *sbase = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                             ~static_cast<uintptr_t>(1023));
    const int QR = (a.nq + 127) & ~127;                     // staged Q rows (whole boxes)
    unsigned char *Qs = sbase;                              // [NKB][QR][128 B]
    unsigned char *Ks = sbase + (size_t)NKB * QR * 128;     // [stage][NKB][128][128 B]
    __shared__ TcBars sb;
    __shared__ __align__(16) float mneg[256];   // pass B: -(m_r log2 e + log2 Z_r), -inf past the rows
    __shared__ float eoff[64];                  // pass B: -m_r log2 e of probe u's row (columns 0 .. W-1)
    __shared__ float scale_s;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int lg = a.lg0 + blockIdx.y, l = lg / a.G, g = lg - l * a.G;
    const int t_begin = a.t_lo + blockIdx.x * a.chunk_tiles * kTcTile;
    const int t_end = min(a.t_hi, t_begin + a.chunk_tiles * kTcTile);
    const int ntile = t_end > t_begin ? (t_end - t_begin + kTcTile - 1) / kTcTile : 0;
    const int rowbase = (l * a.Hq + g * a.gq) * a.W;        // first probe row of (l, g) in [L][Hq][W]
    const int nhalf = MODE == 0 ? a.nq / 128 : 1;
    const uint32_t acc_cols = (uint32_t)a.nq;   // TMEM columns of one accumulator buffer
    uint32_t tcols = 32;
    while (tcols < 2 * acc_cols) tcols <<= 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kTcStages; s++) {
            tc::mbar_init(tc::smem_u32(&sb.full[s]), 1);
            tc::mbar_init(tc::smem_u32(&sb.empty[s]), 1);
        }
        for (int b = 0; b < 2; b++) {
            tc::mbar_init(tc::smem_u32(&sb.accfull[b]), 1);
            tc::mbar_init(tc::smem_u32(&sb.accempty[b]), MODE == 0 ? 4 * nhalf : 4);
        }
        tc::mbar_init(tc::smem_u32(&sb.qfull), 1);
        sb.abort = 0;
        tc::fence_barrier_init();
    }
    if (MODE == 1) {
        // column n of pass B holds row qperm[n] of the KV head: the probe rows
        // (u mod gq) W + u first (n = u < W), then the other rows
        for (int n = threadIdx.x; n < 256; n += kTcThreads) {
            const int r = n < a.Rg ? qperm[n] : -1;
            mneg[n] = r >= 0 ? rmneg[rowbase + r] : -INFINITY;
            if (n < 64) eoff[n] = n < a.W ? (float)(-(double)rm[rowbase + r] * 1.4426950408889634) : 0.f;
        }
        if (threadIdx.x == 0) scale_s = (float)lg_scale[lg];
    }
    if (warp == kTcWarpMma) {
        tc::tmem_alloc(tc::smem_u32(&sb.tbase), tcols);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = sb.tbase;

    if (warp == kTcWarpTma) {
        // ---------------- producer ----------------
        if (MODE == 1) {   // probe rows first: one-row boxes, placed by qperm, spread over the warp
            const uint32_t qbar = tc::smem_u32(&sb.qfull);
            if (lane == 0) tc::mbar_expect_tx(qbar, (uint32_t)(NKB * QR * 128));
            __syncwarp();
            for (int e = lane; e < NKB * QR; e += 32) {
                const int kb = e / QR, n = e - kb * QR;
                const int r = n < a.Rg ? qperm[n] : 0;   // rows past Rg: any row (their columns are masked)
                tc::tma_load_2d(tc::smem_u32(Qs + ((size_t)kb * QR + n) * 128), &mapQ1, kb * 64, rowbase + r, qbar);
            }
        }
        if (lane == 0) {
            tc::tma_prefetch_desc(&mapK);
            tc::tma_prefetch_desc(&mapQ);
            const uint32_t qbar = tc::smem_u32(&sb.qfull);
            if (MODE == 0) {
                tc::mbar_expect_tx(qbar, (uint32_t)(NKB * QR * 128));
                for (int kb = 0; kb < NKB; kb++)
                    for (int j = 0; j < QR; j += 128)
                        tc::tma_load_2d(tc::smem_u32(Qs + ((size_t)kb * QR + j) * 128), &mapQ, kb * 64, rowbase + j, qbar);
            }
            const int krow = lg * a.T + t_begin;
            int issued = 0;
            (void)krow;
            for (int i = 0; i < ntile; i++) {
                const int st = i % kTcStages, r = i / kTcStages;
                if (*(volatile int *)&sb.abort) break;
                if (!tc::mbar_wait(tc::smem_u32(&sb.empty[st]), (r & 1) ^ 1, kWaitNs)) {
                    atomicOr(status, kStPipeTimeout);
                    atomicExch(&sb.abort, 1);
                    break;
                }
                const uint32_t fbar = tc::smem_u32(&sb.full[st]);
                tc::mbar_expect_tx(fbar, (uint32_t)(NKB * kBox));
                for (int kb = 0; kb < NKB; kb++)
                    tc::tma_load_2d(tc::smem_u32(Ks + ((size_t)st * NKB + kb) * kBox), &mapK, kb * 64,
                                    krow + i * kTcTile, fbar);
                issued++;
            }
            // the copies still in flight land before the block exits
            for (int i = max(0, issued - kTcStages); i < issued; i++)
                tc::mbar_wait(tc::smem_u32(&sb.full[i % kTcStages]), (i / kTcStages) & 1, kWaitNs);
            tc::mbar_wait(qbar, 0, kWaitNs);
        }
    } else if (warp == kTcWarpMma) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            int done = 0;
            bool ok = tc::mbar_wait(tc::smem_u32(&sb.qfull), 0, kWaitNs);
            const uint32_t qaddr = tc::smem_u32(Qs), kaddr = tc::smem_u32(Ks);
            for (int i = 0; ok && i < ntile; i++) {
                const int st = i % kTcStages, r = i / kTcStages, b = i & 1, ra = i >> 1;
                if (*(volatile int *)&sb.abort) break;
                ok = tc::mbar_wait(tc::smem_u32(&sb.full[st]), r & 1, kWaitNs) &&
                     tc::mbar_wait(tc::smem_u32(&sb.accempty[b]), (ra & 1) ^ 1, kWaitNs);
                if (!ok) break;
                tc::tc_fence_after();
                const uint32_t kst = kaddr + (uint32_t)(st * NKB) * kBox;
                if (MODE == 0) {
                    constexpr uint32_t idesc = tc::idesc_bf16_f32(128, kTcTile);
                    for (int h = 0; h < nhalf; h++) {
                        const uint32_t d = tb + (uint32_t)b * acc_cols + (uint32_t)h * 128;
#pragma unroll
                        for (int kb = 0; kb < NKB; kb++)
#pragma unroll
                            for (int s = 0; s < 4; s++)
                                tc::mma_bf16(d, tc::sdesc_sw128(qaddr + (uint32_t)(kb * QR + h * 128) * 128 + 32 * s),
                                             tc::sdesc_sw128(kst + kb * kBox + 32 * s), idesc, (kb | s) != 0);
                    }
                } else {
                    const uint32_t idesc = tc::idesc_bf16_f32(128, a.nq);
                    const uint32_t d = tb + (uint32_t)b * acc_cols;
#pragma unroll
                    for (int kb = 0; kb < NKB; kb++)
#pragma unroll
                        for (int s = 0; s < 4; s++)
                            tc::mma_bf16(d, tc::sdesc_sw128(kst + kb * kBox + 32 * s),
                                         tc::sdesc_sw128(qaddr + (uint32_t)(kb * QR) * 128 + 32 * s), idesc,
                                         (kb | s) != 0);
                }
                tc::mma_commit(tc::smem_u32(&sb.empty[st]));
                tc::mma_commit(tc::smem_u32(&sb.accfull[b]));
                done++;
            }
            if (!ok) {
                atomicOr(status, kStPipeTimeout);
                atomicExch(&sb.abort, 1);
            }
            // the last commit covers every MMA issued: wait for it before TMEM is freed
            if (done > 0) tc::mbar_wait(tc::smem_u32(&sb.accfull[(done - 1) & 1]), ((done - 1) >> 1) & 1, kWaitNs);
        }
    } else if (MODE == 0) {
        // ---------------- pass A: one thread per probe row ----------------
        const int q = warp & 3, h = warp >> 2;
        if (h < nhalf) {
            const float scale = a.scale;
            float m2 = -INFINITY, z = 0.f, zc = 0.f;      // base-2 running max, sums
            for (int i = 0; i < ntile; i++) {
                const int b = i & 1;
                if (!tc::mbar_wait(tc::smem_u32(&sb.accfull[b]), (i >> 1) & 1, kWaitNs)) {
                    atomicOr(status, kStPipeTimeout);
                    atomicExch(&sb.abort, 1);
                    break;
                }
                tc::tc_fence_after();
                const int t0 = t_begin + i * kTcTile;
                const uint32_t tcol = tb + ((uint32_t)(q * 32) << 16) + (uint32_t)b * acc_cols + (uint32_t)h * 128;
#pragma unroll 1
                for (int c = 0; c < kTcTile / 32; c++) {
                    float v[32];
                    tc::tmem_ld32(tcol + 32 * c, v);
                    if (c == kTcTile / 32 - 1) {   // the buffer is free for the MMA of tile i + 2
                        tc::tc_fence_before();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(tc::smem_u32(&sb.accempty[b]));
                    }
                    const int tc0 = t0 + 32 * c;
                    if (tc0 >= t_end) continue;
                    const int nv = min(32, t_end - tc0);
                    float cm = -INFINITY;
                    if (nv == 32) {
#pragma unroll
                        for (int j = 0; j < 32; j++) cm = fmaxf(cm, v[j]);
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; j++)
                            if (j < nv) cm = fmaxf(cm, v[j]);
                    }
                    const float nm = fmaxf(m2, cm * scale);
                    if (nm > m2) {
                        const float corr = tc::ex2(m2 - nm);
                        z *= corr;
                        zc *= corr;
                        m2 = nm;
                    }
                    const float2 sc2 = make_float2(scale, scale), nm2 = make_float2(-m2, -m2);
                    float2 acc = make_float2(0.f, 0.f);
                    const bool inC = tc0 >= a.cs && tc0 + nv <= a.cend;
                    if (nv == 32 && (inC || tc0 >= a.cend || tc0 + 32 <= a.cs)) {
#pragma unroll
                        for (int j = 0; j < 32; j += 2) {
                            const float2 y = ffma2(make_float2(v[j], v[j + 1]), sc2, nm2);
                            acc = fadd2(acc, make_float2(tc::ex2(y.x), tc::ex2(y.y)));
                        }
                        const float s = acc.x + acc.y;
                        z += s;
                        if (inC) zc += s;
                    } else {   // a chunk that ends the range or straddles a bound of C
                        float s = 0.f, sc = 0.f;
#pragma unroll
                        for (int j = 0; j < 32; j++) {
                            if (j < nv) {
                                const float e = tc::ex2(fmaf(v[j], scale, -m2));
                                s += e;
                                const int t = tc0 + j;
                                if (t >= a.cs && t < a.cend) sc += e;
                            }
                        }
                        z += s;
                        zc += sc;
                    }
                }
            }
            const int r = h * 128 + q * 32 + lane;
            if (r < a.Rg) {
                const size_t row = (size_t)rowbase + r;
                part[((size_t)0 * a.nrow_all + row) * a.nch + blockIdx.x] =
                    m2 == -INFINITY ? -INFINITY : m2 * (1.0f / kLog2e);
                part[((size_t)1 * a.nrow_all + row) * a.nch + blockIdx.x] = z;
                part[((size_t)2 * a.nrow_all + row) * a.nch + blockIdx.x] = zc;
            }
        }
    } else {
        // ---------------- pass B: one thread per token ----------------
        // warps 0-3 take the even tiles (buffer 0), warps 4-7 the odd ones (buffer 1)
        const int q = warp & 3, b = warp >> 2;
        const float2 sc2 = make_float2(a.scale, a.scale);
        for (int i = b; i < ntile; i += 2) {
            if (!tc::mbar_wait(tc::smem_u32(&sb.accfull[b]), (i >> 1) & 1, kWaitNs)) {
                atomicOr(status, kStPipeTimeout);
                atomicExch(&sb.abort, 1);
                break;
            }
            tc::tc_fence_after();
            const uint32_t tcol = tb + ((uint32_t)(q * 32) << 16) + (uint32_t)b * acc_cols;
            float2 acc0 = make_float2(0.f, 0.f), acc1 = acc0;
            const int t = t_begin + i * kTcTile + q * 32 + lane;
            // 32 columns of the accumulator: their probabilities into acc0 / acc1
            auto chunk = [&](const float v[32], int c) {
                const float *mn = &mneg[c];
#pragma unroll
                for (int j = 0; j < 32; j += 4) {
                    const float4 m4 = *reinterpret_cast<const float4 *>(mn + j);
                    const float2 y0 = ffma2(make_float2(v[j], v[j + 1]), sc2, make_float2(m4.x, m4.y));
                    const float2 y1 = ffma2(make_float2(v[j + 2], v[j + 3]), sc2, make_float2(m4.z, m4.w));
                    acc0 = fadd2(acc0, make_float2(tc::ex2(y0.x), tc::ex2(y0.y)));
                    acc1 = fadd2(acc1, make_float2(tc::ex2(y1.x), tc::ex2(y1.y)));
                }
            };
            auto release = [&](int c) {   // after the last load: the buffer is free for tile i + 2
                if (c + 32 >= a.nq) {
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(tc::smem_u32(&sb.accempty[b]));
                }
            };
            {   // columns 0 .. 63 are the probes u: their weights E (no 1 / Z), stored
                // token-major as the unit kernel keeps them, (E_u, E_{u+32}) pairs
                float v0[32], v1[32];
                tc::tmem_ld32(tcol, v0);
                release(0);
                tc::tmem_ld32(tcol + 32, v1);
                release(32);
                if (Eg && t < t_end) {
                    float4 *dst = reinterpret_cast<float4 *>(Eg + ((size_t)lg * a.Nc + (t - a.cs)) * 64);
#pragma unroll
                    for (int j = 0; j < 32; j += 2) {
                        const float e0 = tc::ex2(fmaf(v0[j], a.scale, eoff[j]));
                        const float e1 = tc::ex2(fmaf(v1[j], a.scale, eoff[32 + j]));
                        const float e2 = tc::ex2(fmaf(v0[j + 1], a.scale, eoff[j + 1]));
                        const float e3 = tc::ex2(fmaf(v1[j + 1], a.scale, eoff[33 + j]));
                        dst[j >> 1] = make_float4(j < a.W ? e0 : 0.f, j + 32 < a.W ? e1 : 0.f,
                                                  j + 1 < a.W ? e2 : 0.f, j + 33 < a.W ? e3 : 0.f);
                    }
                }
                chunk(v0, 0);
                chunk(v1, 32);
            }
#pragma unroll 1
            for (int c = 64; c < a.nq; c += 32) {
                float v[32];
                tc::tmem_ld32(tcol + c, v);
                release(c);
                chunk(v, c);
            }
            const float s = (acc0.x + acc0.y) + (acc1.x + acc1.y);
            if (t < t_end) rtok[(size_t)lg * a.Nc + (t - a.cs)] = s * scale_s;
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == kTcWarpMma) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, tcols);
    }
}

// ---- host side -------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encoder() { return tc::tensor_map_encoder(); }

// [rows][DH] row-major bf16, boxes of [128 rows][64 columns], 128-byte swizzle.
bool make_map(CUtensorMap *m, const void *p, int64_t rows, int DH, int box_rows = 128) {
    auto enc = encoder();
    if (!enc) return false;
    cuuint64_t gdim[2] = {(cuuint64_t)DH, (cuuint64_t)rows};
    cuuint64_t gstr[1] = {(cuuint64_t)DH * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p), gdim, gstr, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t tc_smem(int DH, int nq) {
    const int QR = (nq + 127) & ~127;
    return 1024 + (size_t)(DH / 64) * QR * 128 + (size_t)kTcStages * (DH / 64) * kBox;
}

template <int DH, int MODE>
cudaError_t launch_tc(const TcArgs &a, int LG, const void *K, const void *Q, int64_t krows, int64_t qrows,
                      const float *rmneg, const double *lg_scale, float *part, float *rtok, int *status,
                      cudaStream_t s, const float *rm = nullptr, float *Eg = nullptr, const short *qperm = nullptr) {
    CUtensorMap mk, mq, mq1;
    if (!make_map(&mk, K, krows, DH) || !make_map(&mq, Q, qrows, DH) || !make_map(&mq1, Q, qrows, DH, 1))
        return cudaErrorNotSupported;
    const size_t smem = tc_smem(DH, a.nq);
    cudaError_t e = cudaFuncSetAttribute(score_tc_kernel<DH, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)tc_smem(DH, 256));
    if (e != cudaSuccess) return e;
    dim3 grid(a.nch, LG);
    score_tc_kernel<DH, MODE><<<grid, kTcThreads, smem, s>>>(mk, mq, mq1, qperm, a, rmneg, lg_scale, part, rtok, status,
                                                               rm, Eg);
    return cudaGetLastError();
}

// Blocks per (l, g) for a range of ntiles key tiles: about 32 waves of
// one-block-per-SM over the whole device, at least 8 tiles per block.
void split(int ntiles, int LG, int num_sms, int *chunk_tiles, int *nch) {
    int64_t want = std::max<int64_t>(1, (32LL * num_sms + LG / 2) / LG);
    want = std::min<int64_t>(want, std::max(1, ntiles / 8));
    *chunk_tiles = (int)((ntiles + want - 1) / want);
    *nch = std::max(1, (ntiles + *chunk_tiles - 1) / *chunk_tiles);
}

TcArgs base_args(const Ctx &c) {
    TcArgs a;
    a.T = c.p.T; a.G = c.p.G; a.Hq = c.p.Hq; a.W = c.p.W;
    a.gq = c.p.Hq / c.p.G;
    a.Rg = a.gq * a.W;
    a.cs = c.p.ctx_start; a.cend = c.c_end; a.Nc = c.Nc;
    a.nrow_all = c.p.L * c.p.Hq * c.p.W;
    a.scale = (float)(1.4426950408889634 / sqrt((double)c.p.d));
    return a;
}

}  // namespace

bool use_tc(const Ctx &c) {
    const int Rg = (c.p.Hq / c.p.G) * c.p.W;
    return c.p.dtype == GKV_BF16 && (c.p.d == 64 || c.p.d == 128) && Rg <= 256 &&
           (int64_t)c.p.L * c.p.G * c.p.T < (1LL << 31) && encoder() != nullptr;
}

int tc_row_chunks(const Ctx &c) {
    int ct, nch;
    split((c.p.T + kTcTile - 1) / kTcTile, c.p.L * c.p.G, c.num_sms, &ct, &nch);
    return nch;
}

cudaError_t launch_row_stats_tc(Ctx &c, const void *K, const void *Q, cudaStream_t s, int lg0, int nlg) {
    TcArgs a = base_args(c);
    a.t_lo = 0;
    a.t_hi = c.p.T;
    split((c.p.T + kTcTile - 1) / kTcTile, c.p.L * c.p.G, c.num_sms, &a.chunk_tiles, &a.nch);
    if (a.nch > c.n_chunks) return cudaErrorInvalidValue;   // the partial buffer holds n_chunks per row
    a.nq = a.Rg <= 128 ? 128 : 256;
    a.lg0 = lg0;
    const int LG = nlg;
    const int64_t krows = (int64_t)c.p.L * c.p.G * c.p.T, qrows = (int64_t)a.nrow_all;
    cudaError_t e = c.p.d == 128
        ? launch_tc<128, 0>(a, LG, K, Q, krows, qrows, nullptr, nullptr, c.w.rowp, nullptr, c.w.dev_int + kScoreStatus, s)
        : launch_tc<64, 0>(a, LG, K, Q, krows, qrows, nullptr, nullptr, c.w.rowp, nullptr, c.w.dev_int + kScoreStatus, s);
    if (e == cudaSuccess) c.launches += 1;
    return e;
}

cudaError_t launch_token_values_tc(Ctx &c, const void *K, const void *Q, cudaStream_t s, int lg0, int nlg) {
    TcArgs a = base_args(c);
    a.t_lo = c.p.ctx_start;
    a.t_hi = c.c_end;
    split((c.Nc + kTcTile - 1) / kTcTile, c.p.L * c.p.G, c.num_sms, &a.chunk_tiles, &a.nch);
    a.nq = (a.Rg + 63) / 64 * 64;
    a.lg0 = lg0;
    const int LG = nlg;
    const int64_t krows = (int64_t)c.p.L * c.p.G * c.p.T, qrows = (int64_t)a.nrow_all;
    cudaError_t e = c.p.d == 128
        ? launch_tc<128, 1>(a, LG, K, Q, krows, qrows, c.w.row_mneg, c.w.lg_scale, nullptr, c.w.rtok,
                            c.w.dev_int + kScoreStatus, s, c.w.row_m, c.w.Eg, c.w.qperm)
        : launch_tc<64, 1>(a, LG, K, Q, krows, qrows, c.w.row_mneg, c.w.lg_scale, nullptr, c.w.rtok,
                           c.w.dev_int + kScoreStatus, s, c.w.row_m, c.w.Eg, c.w.qperm);
    if (e == cudaSuccess) c.launches += 1;
    return e;
}

}  // namespace gkv
