// score.cu -- observation-query x key score passes of the GraceKV pass.
//
//   rope_table     (cos, sin)(t theta_i), theta_i = base^(-2i/d), built in fp64
//                  (RoPE convention: half-split pairs (i, i + d/2)).
//   row_stats      pass A: for every probe row r = (l, h, u) the max logit
//                  m_r = max_t q.k_t / sqrt(d) over the visible range [0, T),
//                  Z_r = sum_t exp(x - m_r) and Z^C_r = the same sum over the
//                  compressible context C (App. A.3 max-logit shift; App. A.4
//                  Eq. app_attention_probability denominators).
//   token_values   pass B: s_t = sum_r exp(x_rt - m_r) / Z_r over the rows of
//                  KV head g, shat_t = s_t / (sum_r Z^C_r / Z_r + eps) for t in C
//                  (App. A.4 Eqs. app_direct_relevance, app_bottom_up_value with
//                  lambda_graph = 0).
//
// Both passes contract a [rows x d] query block with [tokens x d] keys.  bf16
// inputs with d in {64, 128} run on the tcgen05 tensor cores (score_tc.cu);
// other bf16 shapes on mma.sync tiles below; fp32 inputs in 64 x 64 FFMA tiles.
// All accumulate in fp32 from exact products of the inputs.
#include "gkv_internal.cuh"

#include <algorithm>
#include <mutex>

namespace gkv {
namespace {

// (cos, sin) of the rotation angle (t0 + row) theta_i, theta_i = base^(-2i/d).
__global__ void rope_table_kernel(int T, int d, double base, float2 *tab, int t0) {
    int half = d / 2;
    int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)T * half) return;
    int t = (int)(e / half), i = (int)(e - (int64_t)t * half);
    t += t0;
    if (base == 0.0) {
        tab[e] = make_float2(1.f, 0.f);
        return;
    }
    double theta = pow(base, -2.0 * (double)i / (double)d);
    double s, c;
    sincos((double)t * theta, &s, &c);
    tab[e] = make_float2((float)c, (float)s);
}

constexpr int kTR = 64;   // rows per tile
constexpr int kTT = 64;   // tokens per tile
constexpr int kKC = 32;   // head-dim chunk

struct ScoreArgs {
    int L, G, Hq, T, d, W, gq, Rg, cs, cend, Nc;
    float inv_sqrt_d;
};

// Accumulate the 64 x 64 score tile of (rows rbase.., tokens tbase..) into
// acc[i][j] (row ty + 16 i, token tx + 16 j); Qs / Ks are [kKC][64] staging.
template <typename Tin>
__device__ __forceinline__ void score_tile(const Tin *Qblk, const Tin *Kblk, int nrows, int ntok,
                                           int d, float *Qs, float *Ks, float acc[4][4]) {
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
#pragma unroll
    for (int i = 0; i < 4; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < d; k0 += kKC) {
        __syncthreads();
        for (int e = tid; e < kTR * kKC; e += 256) {
            int r = e / kKC, k = e - r * kKC;
            Qs[k * kTR + r] = (r < nrows && k0 + k < d) ? to_f(Qblk[(size_t)r * d + k0 + k]) : 0.f;
            Ks[k * kTT + r] = (r < ntok && k0 + k < d) ? to_f(Kblk[(size_t)r * d + k0 + k]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int k = 0; k < kKC; k++) {
            float q[4], kv[4];
#pragma unroll
            for (int i = 0; i < 4; i++) q[i] = Qs[k * kTR + ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; j++) kv[j] = Ks[k * kTT + tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; i++)
#pragma unroll
                for (int j = 0; j < 4; j++) acc[i][j] = fmaf(q[i], kv[j], acc[i][j]);
        }
    }
}

// Pass A.  grid = (token chunks, row tiles, L*G); writes per-chunk partials.
template <typename Tin>
__global__ void __launch_bounds__(256) row_stats_kernel(const Tin *K, const Tin *Q, ScoreArgs a,
                                                        int chunk, int nchunks, float *part) {
    __shared__ float Qs[kKC * kTR], Ks[kKC * kTT];
    const int lg = blockIdx.z, l = lg / a.G, g = lg - l * a.G;
    const int r0 = blockIdx.y * kTR;
    const int t_begin = blockIdx.x * chunk, t_end = min(a.T, t_begin + chunk);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const Tin *Qblk = Q + ((size_t)(l * a.Hq + g * a.gq) * a.W + r0) * a.d;
    const Tin *Kl = K + (size_t)lg * a.T * a.d;
    const int nrows = min(kTR, a.Rg - r0);
    float m[4], z[4], zc[4];
#pragma unroll
    for (int i = 0; i < 4; i++) { m[i] = -INFINITY; z[i] = 0.f; zc[i] = 0.f; }
    for (int t0 = t_begin; t0 < t_end; t0 += kTT) {
        int ntok = min(kTT, t_end - t0);
        float acc[4][4];
        score_tile(Qblk, Kl + (size_t)t0 * a.d, nrows, ntok, a.d, Qs, Ks, acc);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            float x[4], tm = -INFINITY;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                x[j] = (tx + 16 * j < ntok) ? acc[i][j] * a.inv_sqrt_d : -INFINITY;
                tm = fmaxf(tm, x[j]);
            }
#pragma unroll
            for (int o = 1; o < 16; o <<= 1) tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, o));
            float nm = fmaxf(m[i], tm);
            float sz = 0.f, szc = 0.f;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                int t = t0 + tx + 16 * j;
                if (tx + 16 * j < ntok) {
                    float e = expf(x[j] - nm);
                    sz += e;
                    if (t >= a.cs && t < a.cend) szc += e;
                }
            }
#pragma unroll
            for (int o = 1; o < 16; o <<= 1) {
                sz += __shfl_xor_sync(0xffffffffu, sz, o);
                szc += __shfl_xor_sync(0xffffffffu, szc, o);
            }
            float sc = (m[i] == -INFINITY) ? 0.f : expf(m[i] - nm);
            z[i] = z[i] * sc + sz;
            zc[i] = zc[i] * sc + szc;
            m[i] = nm;
        }
    }
    if (tx == 0) {
        const int nrow_all = a.L * a.Hq * a.W;
#pragma unroll
        for (int i = 0; i < 4; i++) {
            int r = ty + 16 * i;
            if (r >= nrows) continue;
            size_t row = (size_t)(l * a.Hq + g * a.gq) * a.W + r0 + r;   // index into [L][Hq][W]
            part[((size_t)0 * nrow_all + row) * nchunks + blockIdx.x] = m[i];
            part[((size_t)1 * nrow_all + row) * nchunks + blockIdx.x] = z[i];
            part[((size_t)2 * nrow_all + row) * nchunks + blockIdx.x] = zc[i];
        }
    }
}

// Combines the per-chunk partials of every row; rmneg (nullable) receives
// -(m_r log2 e + log2 Z_r), the base-2 exponent offset of exp(x - m_r) / Z_r.
__global__ void row_combine_kernel(const float *part, int nrow, int nchunks, float *rm, float *rz,
                                   float *rzc, int *status, float *rmneg, int row0 = 0, int row1 = -1) {
    const int row = row0 + blockIdx.x * blockDim.x + threadIdx.x;   // rows [row0, row1) of nrow
    if (row >= (row1 < 0 ? nrow : row1)) return;
    const float *pm = part + (size_t)row * nchunks;
    const float *pz = part + ((size_t)nrow + row) * nchunks;
    const float *pc = part + ((size_t)2 * nrow + row) * nchunks;
    float M = -INFINITY;
    for (int c = 0; c < nchunks; c++) M = fmaxf(M, pm[c]);
    double Z = 0.0, ZC = 0.0;
    for (int c = 0; c < nchunks; c++) {
        if (pm[c] == -INFINITY) continue;
        double s = exp((double)pm[c] - (double)M);
        Z += pz[c] * s;
        ZC += pc[c] * s;
    }
    if (!isfinite(M) || !isfinite(Z)) atomicOr(status, 2);
    rm[row] = M;
    rz[row] = (float)Z;
    rzc[row] = (float)ZC;
    if (rmneg) rmneg[row] = (float)(-((double)M * 1.4426950408889634 + log2((double)(float)Z)));
}

// Pass-B normaliser of every KV head: 1 / (sum_r Z^C_r / Z_r + eps) over its rows.
__global__ void lg_scale_kernel(const float *rz, const float *rzc, int G, int Hq, int W, int gq, double eps,
                                double *out, int lg0) {
    const int lg = lg0 + blockIdx.x, l = lg / G, g = lg - l * G;
    const size_t rowbase = (size_t)(l * Hq + g * gq) * W;
    double s = 0.0;
    for (int r = threadIdx.x; r < gq * W; r += 32) s += (double)rzc[rowbase + r] / (double)rz[rowbase + r];
    s = warp_sum(s);
    if (threadIdx.x == 0) out[lg] = 1.0 / (s + eps);
}

// Pass B.  grid = (token tiles over C, L*G).  Loops over the row tiles of the
// KV head, accumulating s_t for the 64 tokens of the tile.
template <typename Tin>
__global__ void __launch_bounds__(256) token_values_kernel(const Tin *K, const Tin *Q, ScoreArgs a,
                                                           const float *rm, const float *rz,
                                                           const float *rzc, float eps,
                                                           float *rtok) {
    __shared__ float Qs[kKC * kTR], Ks[kKC * kTT];
    __shared__ float colpart[16][kTT];
    __shared__ float rowm[kTR], rowiz[kTR];
    __shared__ double scale_s;
    const int lg = blockIdx.y, l = lg / a.G, g = lg - l * a.G;
    const int t0 = a.cs + blockIdx.x * kTT;
    const int ntok = min(kTT, a.cend - t0);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const size_t rowbase = (size_t)(l * a.Hq + g * a.gq) * a.W;
    if (tid < 32) {
        double s = 0.0;
        for (int r = tid; r < a.Rg; r += 32) s += (double)rzc[rowbase + r] / (double)rz[rowbase + r];
        s = warp_sum(s);
        if (tid == 0) scale_s = 1.0 / (s + (double)eps);
    }
    float s_tok[4] = {0.f, 0.f, 0.f, 0.f};
    const Tin *Kl = K + ((size_t)lg * a.T + t0) * a.d;
    for (int r0 = 0; r0 < a.Rg; r0 += kTR) {
        int nrows = min(kTR, a.Rg - r0);
        __syncthreads();
        if (tid < kTR) {
            bool ok = tid < nrows;
            rowm[tid] = ok ? rm[rowbase + r0 + tid] : 0.f;
            rowiz[tid] = ok ? 1.0f / rz[rowbase + r0 + tid] : 0.f;
        }
        float acc[4][4];
        score_tile(Q + (rowbase + r0) * a.d, Kl, nrows, ntok, a.d, Qs, Ks, acc);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            int r = ty + 16 * i;
            if (r >= nrows) continue;
#pragma unroll
            for (int j = 0; j < 4; j++)
                s_tok[j] += expf(acc[i][j] * a.inv_sqrt_d - rowm[r]) * rowiz[r];
        }
    }
#pragma unroll
    for (int j = 0; j < 4; j++) colpart[ty][tx + 16 * j] = s_tok[j];
    __syncthreads();
    if (tid < ntok) {
        float s = 0.f;
        for (int q = 0; q < 16; q++) s += colpart[q][tid];
        rtok[(size_t)lg * a.Nc + (t0 - a.cs) + tid] = (float)((double)s * scale_s);
    }
}

// ---------------------------------------------------------------------------
// Tensor-core (bf16 mma.sync m16n8k16, fp32 accumulation) versions of both
// passes for bf16 inputs: products of bf16 values are exact, sums are fp32.
// 16 warps per CTA, warp w owns probe rows 16 w .. 16 w + 15 of the KV head
// (its Q fragments stay in registers); 64-token key tiles are staged in
// shared memory (row stride d + 8 halves: conflict-free fragment reads) with
// cp.async double buffering.  Exponentials run in base 2 on pre-scaled logits.
// ---------------------------------------------------------------------------
constexpr int kMT = 64;           // tokens per tile
constexpr int kMmaWarps = 16;
constexpr float kLog2e = 1.4426950408889634f;

// Stage tokens [t0, t0 + 64) of K (row-major [T][DH]) into a padded tile.
template <int DH>
__device__ __forceinline__ void stage_tile(__nv_bfloat16 *tile, const __nv_bfloat16 *Kl, int t0, int tend) {
    constexpr int CPR = DH / 8;            // 16-byte chunks per row
    for (int e = threadIdx.x; e < kMT * CPR; e += blockDim.x) {
        int r = e / CPR, cc = e - r * CPR;
        int t = t0 + r;
        bool ok = t < tend;
        const __nv_bfloat16 *src = Kl + (size_t)(ok ? t : t0) * DH + cc * 8;
        cp_async16(tile + r * (DH + 8) + cc * 8, src, ok);
    }
}

// Load the A fragments of rows [r0, r0 + 16) of a row-major [rows][DH] block.
template <int DH>
__device__ __forceinline__ void load_qfrag(uint32_t qa[DH / 16][4], const __nv_bfloat16 *Qrows, int lane) {
    const int r = lane >> 2, k = 2 * (lane & 3);
#pragma unroll
    for (int ks = 0; ks < DH / 16; ks++) {
        const __nv_bfloat16 *p0 = Qrows + (size_t)r * DH + ks * 16 + k;
        const __nv_bfloat16 *p1 = Qrows + (size_t)(r + 8) * DH + ks * 16 + k;
        qa[ks][0] = *reinterpret_cast<const uint32_t *>(p0);
        qa[ks][1] = *reinterpret_cast<const uint32_t *>(p1);
        qa[ks][2] = *reinterpret_cast<const uint32_t *>(p0 + 8);
        qa[ks][3] = *reinterpret_cast<const uint32_t *>(p1 + 8);
    }
}

// Scores of the warp's 16 rows against the 64 tokens of a staged tile.
template <int DH>
__device__ __forceinline__ void tile_scores(float c[8][4], const uint32_t qa[DH / 16][4],
                                            const __nv_bfloat16 *tile, int lane) {
    const int n = lane >> 2, k = 2 * (lane & 3);
#pragma unroll
    for (int nt = 0; nt < 8; nt++) {
        c[nt][0] = c[nt][1] = c[nt][2] = c[nt][3] = 0.f;
        const __nv_bfloat16 *row = tile + (nt * 8 + n) * (DH + 8) + k;
#pragma unroll
        for (int ks = 0; ks < DH / 16; ks++) {
            uint32_t b0 = *reinterpret_cast<const uint32_t *>(row + ks * 16);
            uint32_t b1 = *reinterpret_cast<const uint32_t *>(row + ks * 16 + 8);
            mma_bf16(c[nt], qa[ks], b0, b1);
        }
    }
}

// Pass A on tensor cores.  grid = (token chunks, 1, L*G); rows = 16 * warps.
template <int DH>
__global__ void __launch_bounds__(kMmaWarps * 32) row_stats_mma_kernel(
        const __nv_bfloat16 *K, const __nv_bfloat16 *Q, ScoreArgs a, int chunk, int nchunks,
        float *part) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __nv_bfloat16 *tiles = reinterpret_cast<__nv_bfloat16 *>(smem_raw);   // [2][64][DH + 8]
    const int lg = blockIdx.z, l = lg / a.G, g = lg - l * a.G;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t_begin = blockIdx.x * chunk, t_end = min(a.T, t_begin + chunk);
    const __nv_bfloat16 *Kl = K + (size_t)lg * a.T * DH;
    const size_t rowbase = (size_t)(l * a.Hq + g * a.gq) * a.W;
    const bool wact = warp * 16 < a.Rg;
    uint32_t qa[DH / 16][4];
    if (wact) load_qfrag<DH>(qa, Q + (rowbase + warp * 16) * DH, lane);
    const float scale = a.inv_sqrt_d * kLog2e;     // logits in base-2 units
    float m[2] = {-INFINITY, -INFINITY}, z[2] = {0.f, 0.f}, zc[2] = {0.f, 0.f};
    const int ntile = (t_end - t_begin + kMT - 1) / kMT;
    if (ntile > 0) stage_tile<DH>(tiles, Kl, t_begin, t_end);
    cp_async_commit();
    for (int it = 0; it < ntile; it++) {
        const int t0 = t_begin + it * kMT;
        if (it + 1 < ntile) stage_tile<DH>(tiles + ((it + 1) & 1) * kMT * (DH + 8), Kl, t0 + kMT, t_end);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (wact) {
            float c[8][4];
            tile_scores<DH>(c, qa, tiles + (it & 1) * kMT * (DH + 8), lane);
#pragma unroll
            for (int h = 0; h < 2; h++) {          // h = 0: row lane/4, h = 1: row lane/4 + 8
                float tm = -INFINITY;
#pragma unroll
                for (int nt = 0; nt < 8; nt++)
#pragma unroll
                    for (int q = 0; q < 2; q++) {
                        int t = t0 + nt * 8 + 2 * (lane & 3) + q;
                        float x = c[nt][2 * h + q] * scale;
                        c[nt][2 * h + q] = x;
                        if (t < t_end) tm = fmaxf(tm, x);
                    }
                tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, 1));
                tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, 2));
                const float nm = fmaxf(m[h], tm);
                float sz = 0.f, szc = 0.f;
#pragma unroll
                for (int nt = 0; nt < 8; nt++)
#pragma unroll
                    for (int q = 0; q < 2; q++) {
                        int t = t0 + nt * 8 + 2 * (lane & 3) + q;
                        if (t < t_end) {
                            float e = exp2f(c[nt][2 * h + q] - nm);
                            sz += e;
                            if (t >= a.cs && t < a.cend) szc += e;
                        }
                    }
                sz += __shfl_xor_sync(0xffffffffu, sz, 1);
                sz += __shfl_xor_sync(0xffffffffu, sz, 2);
                szc += __shfl_xor_sync(0xffffffffu, szc, 1);
                szc += __shfl_xor_sync(0xffffffffu, szc, 2);
                const float sc = m[h] == -INFINITY ? 0.f : exp2f(m[h] - nm);
                z[h] = z[h] * sc + sz;
                zc[h] = zc[h] * sc + szc;
                m[h] = nm;
            }
        }
        __syncthreads();
    }
    if (wact && (lane & 3) == 0) {
        const int nrow_all = a.L * a.Hq * a.W;
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const size_t row = rowbase + warp * 16 + (lane >> 2) + 8 * h;
            part[((size_t)0 * nrow_all + row) * nchunks + blockIdx.x] =
                m[h] == -INFINITY ? -INFINITY : m[h] * (1.0f / kLog2e);
            part[((size_t)1 * nrow_all + row) * nchunks + blockIdx.x] = z[h];
            part[((size_t)2 * nrow_all + row) * nchunks + blockIdx.x] = zc[h];
        }
    }
}

// Pass B on tensor cores.  grid = (token chunks over C, L*G).
template <int DH>
__global__ void __launch_bounds__(kMmaWarps * 32) token_values_mma_kernel(
        const __nv_bfloat16 *K, const __nv_bfloat16 *Q, ScoreArgs a, int chunk, const float *rm,
        const float *rz, const float *rzc, float eps, float *rtok) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __nv_bfloat16 *tiles = reinterpret_cast<__nv_bfloat16 *>(smem_raw);   // [2][64][DH + 8]
    float *colpart = reinterpret_cast<float *>(tiles + 2 * kMT * (DH + 8));  // [16][64]
    __shared__ double scale_s;
    const int lg = blockIdx.y, l = lg / a.G, g = lg - l * a.G;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t_begin = a.cs + blockIdx.x * chunk, t_end = min(a.cend, t_begin + chunk);
    const __nv_bfloat16 *Kl = K + (size_t)lg * a.T * DH;
    const size_t rowbase = (size_t)(l * a.Hq + g * a.gq) * a.W;
    const bool wact = warp * 16 < a.Rg;
    if (warp == 0) {
        double sum = 0.0;
        for (int r = lane; r < a.Rg; r += 32) sum += (double)rzc[rowbase + r] / (double)rz[rowbase + r];
        sum = warp_sum(sum);
        if (lane == 0) scale_s = 1.0 / (sum + (double)eps);
    }
    uint32_t qa[DH / 16][4];
    float rmh[2] = {0.f, 0.f}, rih[2] = {0.f, 0.f};
    if (wact) {
        load_qfrag<DH>(qa, Q + (rowbase + warp * 16) * DH, lane);
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const size_t row = rowbase + warp * 16 + (lane >> 2) + 8 * h;
            rmh[h] = rm[row] * kLog2e;
            rih[h] = 1.0f / rz[row];
        }
    }
    const float scale = a.inv_sqrt_d * kLog2e;
    const int ntile = (t_end - t_begin + kMT - 1) / kMT;
    if (ntile > 0) stage_tile<DH>(tiles, Kl, t_begin, t_end);
    cp_async_commit();
    for (int it = 0; it < ntile; it++) {
        const int t0 = t_begin + it * kMT;
        if (it + 1 < ntile) stage_tile<DH>(tiles + ((it + 1) & 1) * kMT * (DH + 8), Kl, t0 + kMT, t_end);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        float col[16];
#pragma unroll
        for (int q = 0; q < 16; q++) col[q] = 0.f;
        if (wact) {
            float c[8][4];
            tile_scores<DH>(c, qa, tiles + (it & 1) * kMT * (DH + 8), lane);
#pragma unroll
            for (int nt = 0; nt < 8; nt++)
#pragma unroll
                for (int q = 0; q < 2; q++)
                    col[2 * nt + q] = exp2f(c[nt][q] * scale - rmh[0]) * rih[0] +
                                      exp2f(c[nt][2 + q] * scale - rmh[1]) * rih[1];
        }
#pragma unroll
        for (int q = 0; q < 16; q++) {
            float v = col[q];
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            col[q] = v;
        }
        if (lane < 4) {
#pragma unroll
            for (int nt = 0; nt < 8; nt++)
#pragma unroll
                for (int q = 0; q < 2; q++) colpart[warp * kMT + nt * 8 + 2 * lane + q] = col[2 * nt + q];
        }
        __syncthreads();
        if (threadIdx.x < kMT) {
            const int t = t0 + threadIdx.x;
            if (t < t_end) {
                float sum = 0.f;
                for (int w = 0; w < kMmaWarps; w++) sum += colpart[w * kMT + threadIdx.x];
                rtok[(size_t)lg * a.Nc + (t - a.cs)] = (float)((double)sum * scale_s);
            }
        }
    }
}

ScoreArgs make_args(const Ctx &c) {
    ScoreArgs a;
    a.L = c.p.L; a.G = c.p.G; a.Hq = c.p.Hq; a.T = c.p.T; a.d = c.p.d; a.W = c.p.W;
    a.gq = c.p.Hq / c.p.G;
    a.Rg = a.gq * a.W;
    a.cs = c.p.ctx_start;
    a.cend = c.c_end;
    a.Nc = c.Nc;
    a.inv_sqrt_d = (float)(1.0 / sqrt((double)c.p.d));
    return a;
}

}  // namespace

cudaError_t launch_rope_table(Ctx &c, cudaStream_t s) {
    int64_t n = (int64_t)c.p.T * (c.p.d / 2);
    rope_table_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(c.p.T, c.p.d, c.p.rope_base, c.w.rope, 0);
    // rotations by the offsets -(kMaxSlot - 1) .. kMaxSlot - 1 (prototype position minus token position)
    int64_t nr = (int64_t)(2 * kMaxSlot - 1) * (c.p.d / 2);
    rope_table_kernel<<<(unsigned)((nr + 255) / 256), 256, 0, s>>>(2 * kMaxSlot - 1, c.p.d, c.p.rope_base,
                                                                   c.w.rope_rel, -(kMaxSlot - 1));
    return cudaGetLastError();
}

bool use_mma(const Ctx &c, const ScoreArgs &a) {
    return c.p.dtype == GKV_BF16 && (c.p.d == 64 || c.p.d == 128) && a.Rg % 16 == 0 &&
           a.Rg <= 16 * kMmaWarps;
}

template <int DH>
void launch_mma_a(const Ctx &c, const ScoreArgs &a, const void *K, const void *Q, int chunk, cudaStream_t s) {
    size_t sm = 2 * kMT * (DH + 8) * sizeof(__nv_bfloat16);
    dim3 grid(c.n_chunks, 1, a.L * a.G);
    row_stats_mma_kernel<DH><<<grid, kMmaWarps * 32, sm, s>>>(
        static_cast<const __nv_bfloat16 *>(K), static_cast<const __nv_bfloat16 *>(Q), a, chunk,
        c.n_chunks, c.w.rowp);
}

template <int DH>
void launch_mma_b(const Ctx &c, const ScoreArgs &a, const void *K, const void *Q, int chunk, float eps,
                  cudaStream_t s) {
    size_t sm = 2 * kMT * (DH + 8) * sizeof(__nv_bfloat16) + kMmaWarps * kMT * sizeof(float);
    dim3 grid((c.Nc + chunk - 1) / chunk, a.L * a.G);
    token_values_mma_kernel<DH><<<grid, kMmaWarps * 32, sm, s>>>(
        static_cast<const __nv_bfloat16 *>(K), static_cast<const __nv_bfloat16 *>(Q), a, chunk,
        c.w.row_m, c.w.row_Z, c.w.row_ZC, eps, c.w.rtok);
}

cudaError_t launch_row_stats(Ctx &c, const void *K, const void *Q, cudaStream_t s, int l0, int l1) {
    ScoreArgs a = make_args(c);
    if (l1 < 0) l1 = a.L;
    if (use_tc(c)) {   // tcgen05 pass (score_tc.cu) over layers [l0, l1), then the same combine
        cudaError_t e = launch_row_stats_tc(c, K, Q, s, l0 * a.G, (l1 - l0) * a.G);
        if (e != cudaSuccess) return e;
        const int nrow = a.L * a.Hq * a.W, r0 = l0 * a.Hq * a.W, r1 = l1 * a.Hq * a.W;
        row_combine_kernel<<<(r1 - r0 + 255) / 256, 256, 0, s>>>(c.w.rowp, nrow, tc_row_chunks(c), c.w.row_m,
                                                                 c.w.row_Z, c.w.row_ZC, c.w.dev_int + kScoreStatus,
                                                                 c.w.row_mneg, r0, r1);
        lg_scale_kernel<<<(l1 - l0) * a.G, 32, 0, s>>>(c.w.row_Z, c.w.row_ZC, a.G, a.Hq, a.W, a.gq, (double)c.p.eps,
                                                        c.w.lg_scale, l0 * a.G);
        c.launches += 1;
        c.launches += 1;
        return cudaGetLastError();
    }
    if (l0 != 0 || l1 != a.L) return cudaErrorInvalidValue;   // layer ranges: tensor-core path only
    int chunk = (c.p.T + c.n_chunks - 1) / c.n_chunks;
    chunk = (chunk + kTT - 1) / kTT * kTT;
    if (use_mma(c, a)) {
        if (c.p.d == 128) launch_mma_a<128>(c, a, K, Q, chunk, s);
        else launch_mma_a<64>(c, a, K, Q, chunk, s);
        int nrow = a.L * a.Hq * a.W;
        row_combine_kernel<<<(nrow + 255) / 256, 256, 0, s>>>(c.w.rowp, nrow, c.n_chunks, c.w.row_m,
                                                              c.w.row_Z, c.w.row_ZC, c.w.dev_int + kScoreStatus, nullptr);
        c.launches += 2;
        return cudaGetLastError();
    }
    dim3 grid(c.n_chunks, (a.Rg + kTR - 1) / kTR, a.L * a.G);
    if (c.p.dtype == GKV_BF16)
        row_stats_kernel<<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(K),
                                              static_cast<const __nv_bfloat16 *>(Q), a, chunk,
                                              c.n_chunks, c.w.rowp);
    else
        row_stats_kernel<<<grid, 256, 0, s>>>(static_cast<const float *>(K),
                                              static_cast<const float *>(Q), a, chunk, c.n_chunks,
                                              c.w.rowp);
    int nrow = a.L * a.Hq * a.W;
    row_combine_kernel<<<(nrow + 255) / 256, 256, 0, s>>>(c.w.rowp, nrow, c.n_chunks, c.w.row_m,
                                                          c.w.row_Z, c.w.row_ZC, c.w.dev_int + kScoreStatus, nullptr);
    c.launches += 2;
    return cudaGetLastError();
}

cudaError_t launch_token_values(Ctx &c, const void *K, const void *Q, cudaStream_t s, int l0, int l1) {
    ScoreArgs a = make_args(c);
    dim3 grid((c.Nc + kTT - 1) / kTT, a.L * a.G);
    float eps = (float)c.p.eps;
    if (l1 < 0) l1 = a.L;
    if (use_tc(c)) return launch_token_values_tc(c, K, Q, s, l0 * a.G, (l1 - l0) * a.G);
    if (l0 != 0 || l1 != a.L) return cudaErrorInvalidValue;   // layer ranges: tensor-core path only
    if (use_mma(c, a)) {
        // about 4 CTAs of 16 warps per SM-pass over the compressible region
        int64_t want = 4LL * c.num_sms;
        int64_t per = std::max<int64_t>(1, ((int64_t)a.L * a.G * c.Nc) / want);
        int chunk = (int)std::min<int64_t>(std::max<int64_t>(kMT, (per + kMT - 1) / kMT * kMT), 4096);
        if (c.p.d == 128) launch_mma_b<128>(c, a, K, Q, chunk, eps, s);
        else launch_mma_b<64>(c, a, K, Q, chunk, eps, s);
        c.launches += 1;
        return cudaGetLastError();
    }
    if (c.p.dtype == GKV_BF16)
        token_values_kernel<<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(K),
                                                 static_cast<const __nv_bfloat16 *>(Q), a,
                                                 c.w.row_m, c.w.row_Z, c.w.row_ZC, eps, c.w.rtok);
    else
        token_values_kernel<<<grid, 256, 0, s>>>(static_cast<const float *>(K),
                                                 static_cast<const float *>(Q), a, c.w.row_m,
                                                 c.w.row_Z, c.w.row_ZC, eps, c.w.rtok);
    c.launches += 1;
    return cudaGetLastError();
}

}  // namespace gkv

// ---------------------------------------------------------------------------
// Allocation-free row statistics.
//
// Some callers cannot call cudaMalloc: a serving engine or framework that
// reserves the whole device for its own memory pool, or a latency-critical
// loop that cannot accept the implicit device synchronisation an allocation
// can cause.  gracekv_row_stats_noalloc gives them the row statistics pass
// without a context: its scratch (the per-chunk partial maxima and sums, and
// a status word) lives in the fixed array below, which every GPU that loads
// this library keeps for the life of the process.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchFloats = (size_t)1 << 20;   // 4 MiB of fp32 scratch
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float *g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array for the current device, resolved once
// per device (host code cannot use the array's name as a device address).
cudaError_t noalloc_scratch(int dev, float **out) {
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = static_cast<float *>(p);
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" gkv_status gracekv_row_stats_noalloc(const void *K, const void *Q, int32_t L, int32_t G,
                                                int32_t Hq, int32_t T, int32_t d, int32_t W,
                                                int32_t dtype, int32_t c_lo, int32_t c_hi,
                                                float *row_m, float *row_Z, float *row_ZC,
                                                void *stream) {
    if (!K || !Q || !row_m || !row_Z || !row_ZC) return GKV_EINVAL;
    if ((reinterpret_cast<uintptr_t>(K) & 15u) || (reinterpret_cast<uintptr_t>(Q) & 15u) ||
        (reinterpret_cast<uintptr_t>(row_m) & 3u) || (reinterpret_cast<uintptr_t>(row_Z) & 3u) ||
        (reinterpret_cast<uintptr_t>(row_ZC) & 3u))
        return GKV_EINVAL;
    if (L <= 0 || G <= 0 || Hq <= 0 || T <= 0 || d <= 0 || W <= 0 || Hq % G || d % 8) return GKV_EINVAL;
    if ((int64_t)L * G > 65535) return GKV_EINVAL;     // one grid z-slice per (l, g)
    if (dtype != GKV_F32 && dtype != GKV_BF16) return GKV_EINVAL;
    if (c_lo < 0 || c_hi > T || c_lo > c_hi) return GKV_EINVAL;
    const int64_t nrow = (int64_t)L * Hq * W;
    // three partials per (row, chunk) plus one status word must fit the array
    if (3 * nrow + 1 > (int64_t)kNoAllocScratchFloats) return GKV_ECAPACITY;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GKV_ECUDA;
    float *scratch = nullptr;
    if (noalloc_scratch(dev, &scratch) != cudaSuccess) return GKV_ECUDA;
    int sms = 148;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    gkv::ScoreArgs a;
    a.L = L; a.G = G; a.Hq = Hq; a.T = T; a.d = d; a.W = W;
    a.gq = Hq / G;
    a.Rg = a.gq * W;
    a.cs = c_lo; a.cend = c_hi; a.Nc = c_hi - c_lo;
    a.inv_sqrt_d = (float)(1.0 / sqrt((double)d));
    const int64_t base = (int64_t)L * G * ((a.Rg + 63) / 64);
    int64_t nch = (4 * (int64_t)sms + base - 1) / base;
    nch = std::max<int64_t>(1, std::min<int64_t>(nch, std::max(1, T / 256)));
    while (nch > 1 && 3 * nrow * nch + 1 > (int64_t)kNoAllocScratchFloats) nch--;
    const int nchunks = (int)nch;
    int chunk = (T + nchunks - 1) / nchunks;
    chunk = (chunk + gkv::kTT - 1) / gkv::kTT * gkv::kTT;
    int *status = reinterpret_cast<int *>(scratch + 3 * nrow * nchunks);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // every (row, chunk) partial is overwritten by the pass; only the status
    // word has to start at zero.  The combine kernel flags non-finite rows in
    // it, but this entry point does not read it back: such rows come out
    // NaN / Inf with GKV_OK (documented at the declaration).
    if (cudaMemsetAsync(status, 0, sizeof(int), s) != cudaSuccess) return GKV_ECUDA;
    dim3 grid(nchunks, (a.Rg + gkv::kTR - 1) / gkv::kTR, L * G);
    if (dtype == GKV_BF16)
        gkv::row_stats_kernel<<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(K),
                                                   static_cast<const __nv_bfloat16 *>(Q), a, chunk,
                                                   nchunks, scratch);
    else
        gkv::row_stats_kernel<<<grid, 256, 0, s>>>(static_cast<const float *>(K),
                                                   static_cast<const float *>(Q), a, chunk, nchunks,
                                                   scratch);
    gkv::row_combine_kernel<<<(unsigned)((nrow + 255) / 256), 256, 0, s>>>(scratch, (int)nrow, nchunks,
                                                                            row_m, row_Z, row_ZC, status, nullptr);
    return cudaGetLastError() == cudaSuccess ? GKV_OK : GKV_ECUDA;
}
