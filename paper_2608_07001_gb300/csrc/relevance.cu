// relevance.cu -- multi-hop relevance (App. A.4, Eqs. app_global_seed_score,
// app_hop_propagation, app_diffused_relevance) mixed into the token values
// (Eq. app_bottom_up_value: R = (1 - lambda) s-hat + lambda d-hat).
//
// Per hop: the seeds are the tokens of the context in order of their score
// descending (ties: lower t), taken while fewer than m_seed are taken and
// their running mass stays below eta_seed (the one reaching it included);
// hop 1 scores S-hat (the mean direct relevance over all (l, g)), later hops
// the previous hop's propagation score.  A seed u attends, at every graph
// layer and query head, to its causal range [0, u]:
//   d_t = sum_{l, g, h in H(g), u} w_u pi^{l,h,g}_{u,t},
// zeroed at this and the earlier hops' seeds; d = sum_k rho^(k-1) d^(k),
// d-hat = d / (sum_C d + eps).
//
// The seed rows of one (graph layer, query head) form a 64-row query tile;
// key tiles of 64 tokens stream through shared memory (cp.async, two
// stages) and the logits come from the tensor cores (mma.sync m16n8k16,
// exact bf16 products, fp32 sums), in base 2.  A statistics pass forms each
// row's maximum and partition sum over its range chunk by chunk, a combine
// pass merges the chunks, and a sums pass adds w_u 2^(x - m) / Z over the
// rows of every key column, per (graph layer, head) into its own array,
// reduced afterwards in a fixed order (deterministic).
#include "gkv_internal.cuh"
#include "tc.cuh"

#include <cfloat>

namespace gkv {
namespace {

constexpr int kMhRows = 64;        // seeds per tile (m_seed <= 64)
constexpr int kMhKeys = 64;        // keys per tile
constexpr int kMhChunk = 4096;     // keys per CTA
constexpr int kMhPad = 8;
constexpr float kMhLog2e = 1.4426950408889634f;

struct MhArgs {
    const __nv_bfloat16 *K, *Qg;    // K [L][G][T][d]; Qg [n_graph][Hq][T][d]
    const int32_t *graph_l;         // [n_graph]
    int n_graph, L, G, Hq, T, d, cs, Nc, n_chunks, m_seed;
    float scale2, eta, eps;
    float *rtok;                    // [L G][N_c]: s-hat in, R out
    float *sc;                      // [N_c] scores of the hop's seed choice
    float *acc;                     // [N_c] sum_k rho^(k-1) d^(k)
    float *dpart;                   // [n_graph Hq][N_c]
    float *stat;                    // [n_graph Hq][n_chunks][64][2]
    float *rowmz;                   // [n_graph Hq][64][2]
    uint8_t *was;                   // [N_c] seeds of this or an earlier hop
    int32_t *seeds;                 // [64] C-relative positions
    uint64_t *pkeys;                // [parts][64] the best keys of every part
    float *psum;                    // [parts] score sums
    float *w;                       // [64]
    int *nseed;
    float *red;                     // [2] scratch sums
};

template <int D>
struct MhSmem {
    __nv_bfloat16 Qs[kMhRows][D + kMhPad];
    __nv_bfloat16 Ks[2][kMhKeys][D + kMhPad];
    float colsum[4][kMhKeys];
};

__device__ __forceinline__ void mh_ldsm_x4(uint32_t addr, uint32_t a[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
                 : "r"(addr));
}

// S-hat numerator: the mean direct relevance over all (l, g).
__global__ void mh_mean_kernel(MhArgs a) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= a.Nc) return;
    float s = 0.f;
    for (int lg = 0; lg < a.L * a.G; lg++) s += a.rtok[(size_t)lg * a.Nc + t];
    a.sc[t] = s / (a.L * a.G);
    a.acc[t] = 0.f;
    a.was[t] = 0;
}

// The seeds come from a top-64 selection: the order "score descending, ties
// lower t" is the descending order of the 64-bit key (order-preserving bits
// of the score) << 32 | ~t, so the first m_seed keys of the sorted context
// are the seeds that m_seed successive argmax picks would give.  A part
// kernel sorts 2048-token chunks in shared memory (bitonic) and keeps each
// chunk's best 64 and its score sum; one CTA sorts the survivors and applies
// the mass rule to the head of the list.
constexpr int kMhMaxNc = 4096 * 32;       // context tokens (N_c) the selection supports
constexpr int kMhPart = 2048;             // tokens per part CTA
constexpr int kMhMaxParts = kMhMaxNc / kMhPart;
constexpr int kMhTop = 64;                // survivors per part (>= m_seed)
static_assert(kMhMaxParts * kMhTop == 64 * 64, "workspace sizes of the seed candidates");

__device__ __forceinline__ uint64_t mh_key(float v, int t) {
    uint32_t b = __float_as_uint(v);
    b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return ((uint64_t)b << 32) | (uint32_t)(~(uint32_t)t);
}
__device__ __forceinline__ float mh_key_value(uint64_t k) {
    uint32_t b = (uint32_t)(k >> 32);
    b = (b & 0x80000000u) ? (b & 0x7fffffffu) : ~b;
    return __uint_as_float(b);
}

// Descending bitonic sort of n (a power of two) keys in shared memory by the
// whole block; ends with a barrier.
__device__ void mh_bitonic_desc(uint64_t *x, int n) {
    for (int k = 2; k <= n; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n / 2; i += blockDim.x) {
                const int lo = 2 * i - (i & (j - 1)), hi = lo + j;
                const uint64_t p = x[lo], q = x[hi];
                if ((p < q) == ((lo & k) == 0)) { x[lo] = q; x[hi] = p; }
            }
            __syncthreads();
        }
}

// Block sum in a fixed order (warp shuffles, then the warps in order).
__device__ float mh_block_sum(float v, float *wv) {
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) wv[threadIdx.x >> 5] = v;
    __syncthreads();
    float s = 0.f;
    for (int k = 0; k < (int)(blockDim.x >> 5); k++) s += wv[k];
    __syncthreads();
    return s;
}

__global__ void __launch_bounds__(1024) mh_top_part_kernel(MhArgs a) {
    __shared__ uint64_t key[kMhPart];
    __shared__ float wv[32];
    const int t0 = blockIdx.x * kMhPart;
    float part = 0.f;
    for (int i = threadIdx.x; i < kMhPart; i += 1024) {
        const int t = t0 + i;
        uint64_t k = 0;                               // below every token's key
        if (t < a.Nc) {
            const float v = a.sc[t];
            part += v;
            k = mh_key(v, t);
        }
        key[i] = k;
    }
    const float tot = mh_block_sum(part, wv);
    mh_bitonic_desc(key, kMhPart);
    if (threadIdx.x < kMhTop) a.pkeys[(size_t)blockIdx.x * kMhTop + threadIdx.x] = key[threadIdx.x];
    if (threadIdx.x == 0) a.psum[blockIdx.x] = tot;
}

// One CTA: the hop's seeds.  hop1: the scores are S (normalised with eps,
// Eq. app_global_seed_score), else a propagation score (normalised by its
// sum).  Seeds are taken while fewer than m_seed are taken and the running
// mass is below eta_seed.
__global__ void __launch_bounds__(1024) mh_seeds_kernel(MhArgs a, int n_parts, int hop1) {
    __shared__ uint64_t key[kMhMaxParts * kMhTop];
    __shared__ float tot_s;
    __shared__ int n_s;
    int n = kMhTop;
    while (n < n_parts * kMhTop) n <<= 1;
    for (int i = threadIdx.x; i < n; i += 1024) key[i] = i < n_parts * kMhTop ? a.pkeys[i] : 0ull;
    if (threadIdx.x == 0) {
        float s = 0.f;
        for (int p = 0; p < n_parts; p++) s += a.psum[p];
        tot_s = s;
    }
    __syncthreads();
    mh_bitonic_desc(key, n);
    if (threadIdx.x == 0) {
        const float tot = tot_s;
        const float inv = hop1 ? 1.f / (tot + a.eps) : (tot > 0.f ? 1.f / tot : 0.f);
        float cum = 0.f, wsum = 0.f;
        int m = 0;
        while (m < a.m_seed && m < a.Nc && cum < a.eta) {
            const uint64_t k = key[m];
            const float v = mh_key_value(k);
            a.seeds[m] = (int)(~(uint32_t)k);
            a.w[m] = v;
            cum += v * inv;
            wsum += v;
            m++;
        }
        for (int k = 0; k < m; k++) a.w[k] = wsum > 0.f ? a.w[k] / wsum : 1.f / m;
        *a.nseed = m;
        n_s = m;
    }
    __syncthreads();
    if (threadIdx.x < n_s) a.was[a.seeds[threadIdx.x]] = 1;
}

// Logit tiles of the seed rows of (graph layer gi, query head h) against the
// keys [k0, k0 + kMhChunk) (MODE 0: row statistics per chunk; MODE 1: the
// weighted column sums over the context keys).
template <int D, int MODE>
__global__ void __launch_bounds__(128) mh_tile_kernel(MhArgs a) {
    extern __shared__ __align__(16) unsigned char mh_raw[];
    MhSmem<D> &sm = *reinterpret_cast<MhSmem<D> *>(mh_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gh = blockIdx.y, gi = gh / a.Hq, h = gh % a.Hq, g = h / (a.Hq / a.G);
    const int l = a.graph_l[gi];
    const int ns = *a.nseed;
    int umax = -1;
    for (int s = 0; s < ns; s++) umax = max(umax, a.cs + a.seeds[s]);
    // keys of this CTA: MODE 0 [0, umax]; MODE 1 the context keys up to umax
    const int base = MODE ? a.cs : 0;
    const int k0 = base + blockIdx.x * kMhChunk;
    const int kend = min(min(k0 + kMhChunk, MODE ? a.cs + a.Nc : a.T), umax + 1);
    if (k0 >= kend || ns == 0) {
        if (MODE == 0)
            for (int r = tid; r < kMhRows; r += 128) {
                float *st = a.stat + (((size_t)gh * a.n_chunks + blockIdx.x) * kMhRows + r) * 2;
                st[0] = -INFINITY;
                st[1] = 0.f;
            }
        else
            for (int t = k0 + tid; t < min(k0 + kMhChunk, a.cs + a.Nc); t += 128)
                a.dpart[(size_t)gh * a.Nc + (t - a.cs)] = 0.f;
        return;
    }
    const __nv_bfloat16 *Kl = a.K + ((size_t)l * a.G + g) * a.T * D;
    // seed query rows (zero past the seed count)
    for (int e = tid; e < kMhRows * D / 8; e += 128) {
        const int r = e / (D / 8), c = e % (D / 8);
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r < ns)
            v = *reinterpret_cast<const uint4 *>(a.Qg + (((size_t)gi * a.Hq + h) * a.T + a.cs + a.seeds[r]) * D + 8 * c);
        *reinterpret_cast<uint4 *>(&sm.Qs[r][8 * c]) = v;
    }
    auto issue = [&](int kt, int st) {
        for (int e = tid; e < kMhKeys * D / 8; e += 128) {
            const int r = e / (D / 8), c = e % (D / 8);
            const bool in = kt + r < kend;
            cp_async16(&sm.Ks[st][r][8 * c], in ? Kl + (size_t)(kt + r) * D + 8 * c : Kl, in);
        }
        cp_async_commit();
    };
    // this thread's rows: 16 warp + hq (+8); the seeds' positions and statistics
    const int hq = lane >> 2, tq = lane & 3, mi = lane >> 3, ri = lane & 7;
    const int r0 = warp * 16 + hq, r1 = r0 + 8;
    const int u0 = r0 < ns ? a.cs + a.seeds[r0] : -1, u1 = r1 < ns ? a.cs + a.seeds[r1] : -1;
    float m0 = -INFINITY, m1 = -INFINITY, z0 = 0.f, z1 = 0.f;    // MODE 0: running
    float w0 = 0.f, w1 = 0.f;                                     // MODE 1: w_u / Z, maxima
    if (MODE == 1) {
        if (r0 < ns) { m0 = a.rowmz[((size_t)gh * kMhRows + r0) * 2]; w0 = a.w[r0] / a.rowmz[((size_t)gh * kMhRows + r0) * 2 + 1]; }
        if (r1 < ns) { m1 = a.rowmz[((size_t)gh * kMhRows + r1) * 2]; w1 = a.w[r1] / a.rowmz[((size_t)gh * kMhRows + r1) * 2 + 1]; }
    }
    issue(k0, 0);
    for (int kt = k0, st = 0; kt < kend; kt += kMhKeys, st ^= 1) {
        if (kt + kMhKeys < kend) {
            issue(kt + kMhKeys, st ^ 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        float c[kMhKeys / 8][4];
#pragma unroll
        for (int n = 0; n < kMhKeys / 8; n++) c[n][0] = c[n][1] = c[n][2] = c[n][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < D / 16; ks++) {
            uint32_t af[4];
            mh_ldsm_x4(static_cast<uint32_t>(__cvta_generic_to_shared(
                           &sm.Qs[warp * 16 + ri + (mi & 1) * 8][ks * 16 + (mi >> 1) * 8])),
                       af);
#pragma unroll
            for (int n = 0; n < kMhKeys / 8; n++) {
                const uint32_t b0 = *reinterpret_cast<const uint32_t *>(&sm.Ks[st][n * 8 + hq][ks * 16 + 2 * tq]);
                const uint32_t b1 = *reinterpret_cast<const uint32_t *>(&sm.Ks[st][n * 8 + hq][ks * 16 + 8 + 2 * tq]);
                mma_bf16(c[n], af, b0, b1);
            }
        }
        // c[n][0], c[n][1]: row r0, keys kt + 8 n + 2 tq (+1); c[n][2], c[n][3]: row r1
        if (MODE == 0) {
#pragma unroll
            for (int n = 0; n < kMhKeys / 8; n++)
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    const int key = kt + n * 8 + 2 * tq + (q & 1);
                    const int u = q < 2 ? u0 : u1;
                    if (key > u || key >= kend) continue;
                    const float x = c[n][q] * a.scale2;
                    float &m = q < 2 ? m0 : m1;
                    float &z = q < 2 ? z0 : z1;
                    if (x > m) { z = z * tc::ex2(m - x) + 1.f; m = x; }
                    else z += tc::ex2(x - m);
                }
        } else {
            float cs_[kMhKeys / 8][2];
#pragma unroll
            for (int n = 0; n < kMhKeys / 8; n++)
#pragma unroll
                for (int e = 0; e < 2; e++) {
                    const int key = kt + n * 8 + 2 * tq + e;
                    float v = 0.f;
                    if (key <= u0 && key < kend) v += w0 * tc::ex2(c[n][e] * a.scale2 - m0);
                    if (key <= u1 && key < kend) v += w1 * tc::ex2(c[n][2 + e] * a.scale2 - m1);
                    cs_[n][e] = v;
                }
            // sum over the warp's 16 rows (lanes of equal tq), then over the warps
#pragma unroll
            for (int n = 0; n < kMhKeys / 8; n++)
#pragma unroll
                for (int e = 0; e < 2; e++) {
                    float v = cs_[n][e];
#pragma unroll
                    for (int o = 4; o < 32; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    if (hq == 0) sm.colsum[warp][n * 8 + 2 * tq + e] = v;
                }
            __syncthreads();
            for (int k = tid; k < kMhKeys; k += 128) {
                const int key = kt + k;
                if (key < kend) {
                    const float v = (sm.colsum[0][k] + sm.colsum[1][k]) + (sm.colsum[2][k] + sm.colsum[3][k]);
                    a.dpart[(size_t)gh * a.Nc + (key - a.cs)] = v;
                }
            }
        }
        __syncthreads();
    }
    if (MODE == 0) {
        // merge the 4 lanes of a row (equal hq), then write the chunk's partials
#pragma unroll
        for (int o = 1; o < 4; o <<= 1) {
            const float mo0 = __shfl_xor_sync(0xffffffffu, m0, o), zo0 = __shfl_xor_sync(0xffffffffu, z0, o);
            const float mo1 = __shfl_xor_sync(0xffffffffu, m1, o), zo1 = __shfl_xor_sync(0xffffffffu, z1, o);
            const float n0 = fmaxf(m0, mo0), n1 = fmaxf(m1, mo1);
            z0 = (m0 > -INFINITY ? z0 * tc::ex2(m0 - n0) : 0.f) + (mo0 > -INFINITY ? zo0 * tc::ex2(mo0 - n0) : 0.f);
            z1 = (m1 > -INFINITY ? z1 * tc::ex2(m1 - n1) : 0.f) + (mo1 > -INFINITY ? zo1 * tc::ex2(mo1 - n1) : 0.f);
            m0 = n0;
            m1 = n1;
        }
        if (tq == 0) {
            float *st0 = a.stat + (((size_t)gh * a.n_chunks + blockIdx.x) * kMhRows + r0) * 2;
            float *st1 = a.stat + (((size_t)gh * a.n_chunks + blockIdx.x) * kMhRows + r1) * 2;
            st0[0] = m0; st0[1] = z0;
            st1[0] = m1; st1[1] = z1;
        }
    } else {
        // context keys past the last seed stay zero
        for (int t = max(kend, k0) + tid; t < min(k0 + kMhChunk, a.cs + a.Nc); t += 128)
            a.dpart[(size_t)gh * a.Nc + (t - a.cs)] = 0.f;
    }
}

// Row maxima and partition sums over the chunks.
__global__ void mh_combine_kernel(MhArgs a) {
    const int gh = blockIdx.x, r = threadIdx.x;
    if (r >= kMhRows) return;
    float m = -INFINITY, z = 0.f;
    for (int c = 0; c < a.n_chunks; c++) {
        const float *st = a.stat + (((size_t)gh * a.n_chunks + c) * kMhRows + r) * 2;
        const float mc = st[0], zc = st[1];
        if (mc == -INFINITY) continue;
        const float nm = fmaxf(m, mc);
        z = (m > -INFINITY ? z * tc::ex2(m - nm) : 0.f) + zc * tc::ex2(mc - nm);
        m = nm;
    }
    a.rowmz[((size_t)gh * kMhRows + r) * 2] = m;
    a.rowmz[((size_t)gh * kMhRows + r) * 2 + 1] = z > 0.f ? z : 1.f;
}

// d^(k) = sum over (graph layer, head) in a fixed order, zeroed at the seeds;
// acc += decay d^(k); the next hop's scores.
__global__ void mh_reduce_kernel(MhArgs a, float decay) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= a.Nc) return;
    float v = 0.f;
    for (int gh = 0; gh < a.n_graph * a.Hq; gh++) v += a.dpart[(size_t)gh * a.Nc + t];
    if (a.was[t]) v = 0.f;
    a.acc[t] += decay * v;
    a.sc[t] = v;
}

// d-hat = acc / (sum acc + eps); R = (1 - lambda) s-hat + lambda d-hat.
__global__ void __launch_bounds__(1024) mh_total_kernel(MhArgs a) {
    __shared__ float wv[32];
    float part = 0.f;
    for (int t = threadIdx.x; t < a.Nc; t += 1024) part += a.acc[t];
    part = warp_sum(part);
    if ((threadIdx.x & 31) == 0) wv[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = 0.f;
        for (int k = 0; k < 32; k++) s += wv[k];
        a.red[0] = s;
    }
}

__global__ void mh_mix_kernel(MhArgs a, float lambda) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (size_t)a.L * a.G * a.Nc) return;
    const int t = (int)(i % a.Nc);
    const float dh = a.acc[t] / (a.red[0] + a.eps);
    a.rtok[i] = (1.f - lambda) * a.rtok[i] + lambda * dh;
}

template <int D, int MODE>
cudaError_t launch_mh_tile(const MhArgs &a, dim3 grid, cudaStream_t s) {
    constexpr size_t smem = sizeof(MhSmem<D>);
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(mh_tile_kernel<D, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    mh_tile_kernel<D, MODE><<<grid, 128, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

int multihop_chunks(int T) { return (T + kMhChunk - 1) / kMhChunk; }
int multihop_max_context() { return kMhMaxNc; }

cudaError_t launch_multihop(Ctx &c, cudaStream_t s) {
    Workspace &w = c.w;
    const gkv_params &p = c.p;
    MhArgs a;
    a.K = static_cast<const __nv_bfloat16 *>(c.mh_K);
    a.Qg = static_cast<const __nv_bfloat16 *>(c.mh_Qg);
    a.graph_l = w.mh_graph_l;
    a.n_graph = c.mh_ngraph;
    a.L = p.L; a.G = p.G; a.Hq = p.Hq; a.T = p.T; a.d = p.d;
    a.cs = p.ctx_start; a.Nc = c.Nc;
    a.n_chunks = multihop_chunks(p.T);
    a.m_seed = p.m_seed;
    a.scale2 = (float)(1.4426950408889634 / sqrt((double)p.d));
    a.eta = (float)p.eta_seed;
    a.eps = (float)p.eps;
    a.rtok = w.rtok; a.sc = w.mh_sc; a.acc = w.mh_acc; a.dpart = w.mh_dpart; a.stat = w.mh_stat;
    a.rowmz = w.mh_rowmz; a.was = w.mh_was; a.seeds = w.mh_seeds; a.w = w.mh_w; a.nseed = w.mh_nseed;
    a.pkeys = w.mh_pkeys; a.psum = w.mh_psum;
    a.red = w.mh_red;
    mh_mean_kernel<<<(a.Nc + 255) / 256, 256, 0, s>>>(a);
    c.launches += 1;
    float decay = 1.f;
    const int GH = a.n_graph * a.Hq;
    const int nc_ctx = (a.Nc + kMhChunk - 1) / kMhChunk;
    const int n_parts = (a.Nc + kMhPart - 1) / kMhPart;
    for (int k = 0; k < p.r_hop; k++) {
        mh_top_part_kernel<<<n_parts, 1024, 0, s>>>(a);
        mh_seeds_kernel<<<1, 1024, 0, s>>>(a, n_parts, k == 0);
        cudaError_t e = p.d == 128 ? launch_mh_tile<128, 0>(a, dim3(a.n_chunks, GH), s)
                                   : launch_mh_tile<64, 0>(a, dim3(a.n_chunks, GH), s);
        if (e != cudaSuccess) return e;
        mh_combine_kernel<<<GH, kMhRows, 0, s>>>(a);
        e = p.d == 128 ? launch_mh_tile<128, 1>(a, dim3(nc_ctx, GH), s) : launch_mh_tile<64, 1>(a, dim3(nc_ctx, GH), s);
        if (e != cudaSuccess) return e;
        mh_reduce_kernel<<<(a.Nc + 255) / 256, 256, 0, s>>>(a, decay);
        decay *= (float)p.rho_hop;
        c.launches += 6;
    }
    mh_total_kernel<<<1, 1024, 0, s>>>(a);
    const size_t n = (size_t)p.L * p.G * a.Nc;
    mh_mix_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(a, (float)p.lambda_graph);
    c.launches += 2;
    return cudaGetLastError();
}

}  // namespace gkv
