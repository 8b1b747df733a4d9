// segment.cu -- stage 1 of the GraceKV pass: curvature-guided slot
// segmentation (App. B.2 multi-layer multi-scale curvature, robust boundary
// score; App. B.3 length-constrained dynamic program).
//
// Kernels, in launch order:
//   seg_norm      1 / max(||h_t||, eps) and ||hbar_t||^2 per segmentation layer
//                 (Eq. app_hidden_normalization)
//   seg_curv      kappa^(l,w)_i with sliding window sums (Eqs. app_local_means ..
//                 app_local_curvature), zero unless w <= i < T - w
//   seg_combine   kappa_i = Mean - lambda_stab PopStd (Eq. app_stabilized_curvature)
//   seg_robust_z  exact lower median / MAD by radix select, boundary score
//                 b_i = z(kappa)_i + lambda_s z(surprisal)_i (Eqs. app_robust_z,
//                 app_mad, app_boundary_score)
//   seg_dd, seg_scan   prefix of sum_l ||d_t||^2 (Eq. app_adjacent_difference)
//   seg_band      DP edge weights Gamma(a) - lambda_d Disp([a,i)) - lambda_n
//                 ((i-a-n0)/n0)^2 with Disp in the form of Eq. app_prefix_dispersion,
//                 sum d_t = hbar_{e-1} - hbar_a (the differences telescope)
//   seg_dp        F[i] = max_a F[a] + w(a, i) over n_min <= i-a <= n_max (Eq.
//                 app_dp_recurrence), terminal relaxation (Eq.
//                 app_terminal_predecessor), backtracking to slot starts.
#include "gkv_internal.cuh"

#include <cfloat>

namespace gkv {
namespace {

constexpr double kEps = 1e-6;   // App. B.2: epsilon of the normalisations and of robust z

// Double-float numbers (value = hi + lo, |lo| <= ulp(hi) / 2): the DP state is
// carried in ~48-bit precision on the fp32 units, because fp64 throughput on
// GB300 is very low.  Additions use the error-free two-sum of Knuth.
struct df2 {
    float hi, lo;
};
__device__ __forceinline__ float2 df_split(double x) {
    float hi = (float)x;
    return make_float2(hi, (float)(x - (double)hi));
}
__device__ __forceinline__ df2 df_add(df2 a, float2 b) {
    float s = a.hi + b.x;
    float bb = s - a.hi;
    float e = (a.hi - (s - bb)) + (b.x - bb);
    e += a.lo + b.y;
    float hi = s + e;
    return df2{hi, e - (hi - s)};
}
__device__ __forceinline__ bool df_gt(df2 a, df2 b) { return a.hi > b.hi || (a.hi == b.hi && a.lo > b.lo); }
__device__ __forceinline__ bool df_eq(df2 a, df2 b) { return a.hi == b.hi && a.lo == b.lo; }

// Element (channel c of the trajectory) of h^(l)_t: concat over KV heads of V.
template <typename Tin>
__device__ __forceinline__ float traj_elem(const Tin *V, const float *hidden, int Dh, int G,
                                           int T, int d, int l, int li, int t, int c) {
    if (hidden) return hidden[((size_t)li * T + t) * Dh + c];
    int g = c / d, i = c - g * d;
    return to_f(V[(((size_t)l * G + g) * T + t) * d + i]);
}

struct SegArgs {
    int L, G, T, d, D, Dh, nseg, nwin, cs, N;
    int layers[kMaxSegLayers];
    int windows[kMaxWindows];
};

// ---------------------------------------------------------------------------
// Norms: one warp per (layer, position).
// ---------------------------------------------------------------------------
template <typename Tin>
__global__ void seg_norm_kernel(const Tin *V, const float *hidden, SegArgs a, float *inv_norm,
                                float *nrm2) {
    int li = blockIdx.y;
    int t = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    int lane = threadIdx.x & 31;
    if (t >= a.T) return;
    int l = a.layers[li];
    float s = 0.f;
    if (!hidden && (a.d % 8) == 0) {
        for (int c = lane * 8; c < a.D; c += 256) {
            int g = c / a.d, i = c - g * a.d;
            Vec8<Tin> x;
            x.load(V + (((size_t)l * a.G + g) * a.T + t) * a.d + i);
            float f = 0.f;
#pragma unroll
            for (int k = 0; k < 8; k++) f = fmaf(x.v[k], x.v[k], f);
            s += f;
        }
    } else {
        for (int c = lane; c < a.D; c += 32) {
            float x = traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, t, c);
            s = fmaf(x, x, s);
        }
    }
    s = warp_sum(s);
    if (lane == 0) {
        const float n = sqrtf(s);
        const float den = n > (float)kEps ? n : (float)kEps;
        inv_norm[(size_t)li * a.T + t] = 1.0f / den;
        nrm2[(size_t)li * a.T + t] = s / (den * den);
    }
}

// ---------------------------------------------------------------------------
// Curvature.  Block = 256 threads = 512 consecutive positions (two adjacent
// ones per thread) of one segmentation layer.  The trajectory channels are
// staged in chunks of kCurvCC channels, already normalised (hbar = h /
// max(|h|, eps)), channel-major in shared memory so that the threads of a
// warp read consecutive rows.  A thread loads the 34 rows around its two
// positions with 8-byte loads, forms each position's window sums directly
// (running sums outward from the position, left window [i-w+1, i], right
// window [i+1, i+w]) and accumulates |d-|^2, |d+|^2 and d-.d+ over all
// channels in registers: no cross-thread reduction.
// ---------------------------------------------------------------------------
constexpr int kHalo = 16;                       // largest window
constexpr int kCurvPP = 2;                      // positions per thread
constexpr int kCurvPT = 256 * kCurvPP;          // positions per block
constexpr int kCurvRows = kCurvPT + 2 * kHalo;  // staged rows
constexpr int kCurvRS = kCurvRows + 2;          // row stride (even: 8-byte row loads)
constexpr int kCurvCC = 32;                     // channels per stage
constexpr size_t kCurvSmem = ((size_t)kCurvCC * kCurvRS + kCurvRows) * sizeof(float);

// 8 consecutive trajectory channels c .. c+7 (c % 8 == 0) of row t, or zeros
// outside [0, T).
template <typename Tin>
__device__ __forceinline__ void traj_load8(const Tin *V, const float *hidden, const SegArgs &a,
                                           int l, int li, int t, int c, float v[8]) {
    if (t < 0 || t >= a.T) {
#pragma unroll
        for (int j = 0; j < 8; j++) v[j] = 0.f;
        return;
    }
    if (hidden) {
        const float4 *p = reinterpret_cast<const float4 *>(hidden + ((size_t)li * a.T + t) * a.Dh + c);
        const float4 x = p[0], y = p[1];
        v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w; v[4] = y.x; v[5] = y.y; v[6] = y.z; v[7] = y.w;
        return;
    }
    const int g = c / a.d, i = c - g * a.d;
    Vec8<Tin> x;
    x.load(V + (((size_t)l * a.G + g) * a.T + t) * a.d + i);
#pragma unroll
    for (int j = 0; j < 8; j++) v[j] = x.v[j];
}

template <typename Tin, bool kDefaultWindows>
__global__ void __launch_bounds__(256) seg_curv_kernel(const Tin *V, const float *hidden,
                                                       SegArgs a, const float *inv_norm,
                                                       double *klw) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float *P = reinterpret_cast<float *>(smem_raw);   // [kCurvCC][kCurvRS] normalised values
    float *inv_s = P + (size_t)kCurvCC * kCurvRS;     // [kCurvRows]
    const int li = blockIdx.y, l = a.layers[li];
    const int i0 = blockIdx.x * kCurvPT, row0 = i0 - kHalo;
    const int tid = threadIdx.x;
    for (int r = tid; r < kCurvRows; r += 256) {
        const int t = row0 + r;
        inv_s[r] = (t >= 0 && t < a.T) ? inv_norm[(size_t)li * a.T + t] : 0.f;
    }
    const int nw = a.nwin;
    int wv[kMaxWindows];
    float inv_w[kMaxWindows];
#pragma unroll
    for (int wi = 0; wi < kMaxWindows; wi++) {
        wv[wi] = kDefaultWindows ? (4 << wi) : a.windows[wi];
        inv_w[wi] = 1.0f / (float)wv[wi];
    }
    float acc[kCurvPP][kMaxWindows][3];
#pragma unroll
    for (int pp = 0; pp < kCurvPP; pp++)
#pragma unroll
        for (int wi = 0; wi < kMaxWindows; wi++) acc[pp][wi][0] = acc[pp][wi][1] = acc[pp][wi][2] = 0.f;
    // this thread's positions sit at staged rows kHalo + 2 tid (+1); it reads
    // rows 2 tid .. 2 tid + 33 (x[k] = row 2 tid + k)
    constexpr int NX = kCurvPP + 2 * kHalo;
    for (int c0 = 0; c0 < a.D; c0 += kCurvCC) {
        const int nq = min(kCurvCC, a.D - c0) >> 3;   // 8-channel chunks in this stage
        __syncthreads();
        // stage: the loads of 4 row chunks are issued before any is stored
        for (int e0 = tid; e0 < kCurvRows * nq; e0 += 256 * 4) {
            float v[4][8];
#pragma unroll
            for (int u = 0; u < 4; u++) {
                const int e = e0 + 256 * u;
                if (e < kCurvRows * nq) {
                    const int r = e / nq, q = e - r * nq;
                    traj_load8(V, hidden, a, l, li, row0 + r, c0 + 8 * q, v[u]);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; u++) {
                const int e = e0 + 256 * u;
                if (e < kCurvRows * nq) {
                    const int r = e / nq, q = e - r * nq;
                    const float sc = inv_s[r];
#pragma unroll
                    for (int j = 0; j < 8; j++) P[(size_t)(8 * q + j) * kCurvRS + r] = v[u][j] * sc;
                }
            }
        }
        __syncthreads();
        for (int c = 0; c < 8 * nq; c++) {
            const float2 *rp = reinterpret_cast<const float2 *>(P + (size_t)c * kCurvRS + 2 * tid);
            float x[NX];
#pragma unroll
            for (int k = 0; k < NX / 2; k++) {
                const float2 y = rp[k];
                x[2 * k] = y.x;
                x[2 * k + 1] = y.y;
            }
#pragma unroll
            for (int pp = 0; pp < kCurvPP; pp++) {
                const int R = kHalo + pp;   // the position's index in x
                const float h = x[R];
                float sl = h, sr = 0.f;
                float SL[kMaxWindows], SR[kMaxWindows];
#pragma unroll
                for (int wi = 0; wi < kMaxWindows; wi++) SL[wi] = SR[wi] = 0.f;
#pragma unroll
                for (int tau = 1; tau <= kHalo; tau++) {
                    // left sum over tau' < tau, right sum over 1 .. tau
                    if (kDefaultWindows) {
                        if (tau == 4) SL[0] = sl;
                        if (tau == 8) SL[1] = sl;
                        if (tau == 16) SL[2] = sl;
                    } else {
#pragma unroll
                        for (int wi = 0; wi < kMaxWindows; wi++) SL[wi] = wv[wi] == tau ? sl : SL[wi];
                    }
                    if (tau < kHalo) sl += x[R - tau];
                    sr += x[R + tau];
                    if (kDefaultWindows) {
                        if (tau == 4) SR[0] = sr;
                        if (tau == 8) SR[1] = sr;
                        if (tau == 16) SR[2] = sr;
                    } else {
#pragma unroll
                        for (int wi = 0; wi < kMaxWindows; wi++) SR[wi] = wv[wi] == tau ? sr : SR[wi];
                    }
                }
#pragma unroll
                for (int wi = 0; wi < kMaxWindows; wi++) {
                    if (wi >= nw) break;
                    const float dm = h - SL[wi] * inv_w[wi];   // h_i - mean of the left window
                    const float dp = SR[wi] * inv_w[wi] - h;   // mean of the right window - h_i
                    acc[pp][wi][0] = fmaf(dm, dm, acc[pp][wi][0]);
                    acc[pp][wi][1] = fmaf(dp, dp, acc[pp][wi][1]);
                    acc[pp][wi][2] = fmaf(dm, dp, acc[pp][wi][2]);
                }
            }
        }
    }
#pragma unroll
    for (int pp = 0; pp < kCurvPP; pp++) {
        const int i = i0 + kCurvPP * tid + pp;
        if (i >= a.T) continue;
#pragma unroll
        for (int wi = 0; wi < kMaxWindows; wi++) {
            if (wi >= nw) break;
            const int w = wv[wi];
            double k = 0.0;
            if (i >= w && i < a.T - w) {
                const double xv = sqrt((double)acc[pp][wi][0]), yv = sqrt((double)acc[pp][wi][1]);
                k = 1.0 - (double)acc[pp][wi][2] / ((xv > kEps ? xv : kEps) * (yv > kEps ? yv : kEps));
            }
            klw[((size_t)li * nw + wi) * a.T + i] = k;
        }
    }
}

__global__ void seg_combine_kernel(const double *klw, int nk, int T, double lambda_stab,
                                   double *kappa, float *kappa_out, int *status) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= T) return;
    double m = 0.0;
    for (int k = 0; k < nk; k++) m += klw[(size_t)k * T + i];
    m /= nk;
    double v = 0.0;
    for (int k = 0; k < nk; k++) {
        double x = klw[(size_t)k * T + i] - m;
        v += x * x;
    }
    v /= nk;
    double kk = m - lambda_stab * sqrt(v);
    if (!isfinite(kk)) atomicOr(status, 1);
    kappa[i] = kk;
    if (kappa_out) kappa_out[i] = (float)kk;
}

// ---------------------------------------------------------------------------
// Robust z: exact lower median and MAD by radix select over the ordered
// 64-bit keys of doubles; one block of 1024 threads.
// ---------------------------------------------------------------------------
__device__ __forceinline__ unsigned long long dkey(double x) {
    unsigned long long u = (unsigned long long)__double_as_longlong(x);
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
__device__ __forceinline__ double dkey_inv(unsigned long long k) {
    unsigned long long u = (k >> 63) ? (k & 0x7fffffffffffffffull) : ~k;
    return __longlong_as_double((long long)u);
}

// Select the element of ascending rank `rank` of n keys by radix select over
// 11-bit digits (6 passes).  Each pass: every block counts the keys that
// match the digits fixed so far into a shared-memory histogram (updates
// aggregated per warp, one atomic per distinct bin, since the keys of a pass
// crowd into few bins) and adds it to a global one; one block then scans the
// global histogram, fixes the digit that holds the rank and clears it.  The
// keys are dkey(x[i]) (the median) or dev[i] (the MAD).
constexpr int kSelBits = 11, kSelBins = 1 << kSelBits, kSelU = 8, kSelT = 256;

struct SelState {           // in global memory (4 words)
    unsigned long long prefix, mask;
    long long rank;
    double med;
};

template <bool kDev>
__global__ void __launch_bounds__(kSelT) zsel_hist_kernel(const double *x, const unsigned long long *dev, int n,
                                                         const SelState *st, int shift, int bits,
                                                         unsigned int *ghist) {
    __shared__ unsigned int hist[kSelBins];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const unsigned int nbin = 1u << bits;
    for (int bq = tid; bq < (int)nbin; bq += kSelT) hist[bq] = 0;
    const unsigned long long prefix = st->prefix, mask = st->mask;
    __syncthreads();
    const int per_warp = 32 * kSelU, stride = gridDim.x * (kSelT / 32) * per_warp;
    for (int i0 = (blockIdx.x * (kSelT / 32) + warp) * per_warp; i0 < n; i0 += stride) {   // whole warps
        unsigned long long kk[kSelU];
#pragma unroll
        for (int u = 0; u < kSelU; u++) {
            const int i = i0 + 32 * u + lane;
            kk[u] = i < n ? (kDev ? dev[i] : dkey(x[i])) : 0ull;
        }
#pragma unroll
        for (int u = 0; u < kSelU; u++) {
            const int i = i0 + 32 * u + lane;
            int bin = -1;
            if (i < n && (kk[u] & mask) == prefix) bin = (int)((kk[u] >> shift) & (nbin - 1));
            const unsigned grp = __match_any_sync(0xffffffffu, bin);
            if (bin >= 0 && lane == __ffs(grp) - 1) atomicAdd(&hist[bin], (unsigned)__popc(grp));
        }
    }
    __syncthreads();
    for (int bq = tid; bq < (int)nbin; bq += kSelT)
        if (hist[bq]) atomicAdd(&ghist[bq], hist[bq]);
}

// The digit of this pass: thread t owns bins 2t, 2t + 1 (ascending order).
__global__ void __launch_bounds__(1024) zsel_pick_kernel(SelState *st, unsigned int *ghist, int shift, int bits) {
    __shared__ unsigned int wsum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const unsigned int nbin = 1u << bits;
    const long long r = st->rank;
    const unsigned int h0 = 2 * tid < (int)nbin ? ghist[2 * tid] : 0u;
    const unsigned int h1 = 2 * tid + 1 < (int)nbin ? ghist[2 * tid + 1] : 0u;
    unsigned int incl = h0 + h1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const unsigned int wv = lane < (int)(blockDim.x >> 5) ? wsum[lane] : 0u;
        unsigned int wi = wv;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        wsum[lane] = wi - wv;
    }
    __syncthreads();
    const long long before = (long long)wsum[warp] + incl - (h0 + h1);   // keys in lower bins
    if (r >= before && r < before + h0) {
        st->prefix |= (unsigned long long)(2 * tid) << shift;
        st->rank = r - before;
    } else if (r >= before + h0 && r < before + h0 + h1) {
        st->prefix |= (unsigned long long)(2 * tid + 1) << shift;
        st->rank = r - (before + h0);
    }
    if (tid == 0) st->mask |= (unsigned long long)(nbin - 1) << shift;
    if (2 * tid < (int)nbin) ghist[2 * tid] = 0;
    if (2 * tid + 1 < (int)nbin) ghist[2 * tid + 1] = 0;
}

// A fresh select of rank `rank`; with `keep_med`, the median found by the
// select before it is kept in st->med.
__global__ void zsel_init_kernel(SelState *st, unsigned int *ghist, long long rank, int keep_med) {
    if (threadIdx.x == 0) {
        if (keep_med) st->med = dkey_inv(st->prefix);
        st->prefix = 0;
        st->mask = 0;
        st->rank = rank;
    }
    for (int bq = threadIdx.x; bq < kSelBins; bq += blockDim.x) ghist[bq] = 0;
}

__global__ void zsel_dev_kernel(const double *x, int n, const SelState *st, unsigned long long *dev) {
    const double med = st->med;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        dev[i] = dkey(fabs(x[i] - med));
}

// out[i] (+)= scale * (x[i] - median) / (1.4826 MAD + eps), with one fp64
// division (fp64 division is slow on this part; the product differs from the
// quotient by at most one rounding).
__global__ void zsel_z_kernel(const double *x, int n, const SelState *st, double scale, int accumulate,
                              double *out) {
    const double med = st->med, inv_den = 1.0 / (1.4826 * dkey_inv(st->prefix) + kEps);
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const double z = scale * ((x[i] - med) * inv_den);
        out[i] = accumulate ? out[i] + z : z;
    }
}

// The robust z of x (Eq. app_robust_z), scaled by `scale`, written to or added
// to `out`: lower median and lower median of the absolute deviations.
void robust_z(const double *x, int n, double scale, int accumulate, double *out, unsigned long long *dev,
              SelState *st, unsigned int *ghist, int n_sms, int64_t *launches, cudaStream_t s) {
    const long long rank = (n - 1) / 2;
    const int hb = (int)std::max<long long>(1, std::min<long long>(2LL * n_sms, ((long long)n + kSelT * kSelU - 1) / (kSelT * kSelU)));
    const int eb = (int)std::max<long long>(1, std::min<long long>(4LL * n_sms, ((long long)n + 255) / 256));
    zsel_init_kernel<<<1, 256, 0, s>>>(st, ghist, rank, 0);
    for (int pass = 0; pass < 2; pass++) {
        for (int top = 64; top > 0; top -= kSelBits) {
            const int shift = top > kSelBits ? top - kSelBits : 0, bits = top - shift;
            if (pass == 0) zsel_hist_kernel<false><<<hb, kSelT, 0, s>>>(x, dev, n, st, shift, bits, ghist);
            else zsel_hist_kernel<true><<<hb, kSelT, 0, s>>>(x, dev, n, st, shift, bits, ghist);
            zsel_pick_kernel<<<1, 1024, 0, s>>>(st, ghist, shift, bits);
            *launches += 2;
        }
        if (pass == 0) {
            zsel_init_kernel<<<1, 256, 0, s>>>(st, ghist, rank, 1);
            zsel_dev_kernel<<<eb, 256, 0, s>>>(x, n, st, dev);
            *launches += 2;
        }
    }
    zsel_z_kernel<<<eb, 256, 0, s>>>(x, n, st, scale, accumulate, out);
    *launches += 2;   // with the first init
}

__global__ void f32_to_f64_kernel(const float *x, int n, double *y) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) y[i] = x[i];
}

// ---------------------------------------------------------------------------
// Adjacent differences: dd[t] = sum_l ||hbar_{cs+t+1} - hbar_{cs+t}||^2,
// t in [0, N-1); warp per t.
// ---------------------------------------------------------------------------
template <typename Tin>
__global__ void seg_dd_kernel(const Tin *V, const float *hidden, SegArgs a, const float *inv_norm,
                              double *dd) {
    int t = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    int lane = threadIdx.x & 31;
    if (t >= a.N - 1) return;
    double s = 0.0;
    for (int li = 0; li < a.nseg; li++) {
        int l = a.layers[li];
        int p0 = a.cs + t, p1 = p0 + 1;
        float i0 = inv_norm[(size_t)li * a.T + p0], i1 = inv_norm[(size_t)li * a.T + p1];
        float f = 0.f;
        for (int c = lane * 8; c < a.D; c += 256) {
            float x0[8], x1[8];
            traj_load8(V, hidden, a, l, li, p0, c, x0);
            traj_load8(V, hidden, a, l, li, p1, c, x1);
#pragma unroll
            for (int j = 0; j < 8; j++) {
                const float df = x1[j] * i1 - x0[j] * i0;
                f = fmaf(df, df, f);
            }
        }
        s += (double)warp_sum(f);
    }
    if (lane == 0) dd[t] = s;
}

// Exclusive prefix sum of n doubles, deterministic: out[0] = 0,
// out[t] = sum_{s<t} in[s], t <= n.  Block b owns elements [b C, (b + 1) C),
// C = kScanC; the first kernel reduces each block's elements, the second
// adds the totals of the blocks before it (in order, by one warp) to the
// block's own scan.  Sums of one block follow a fixed tree (thread-local
// runs of kScanPer elements, then warp and block scans).
constexpr int kScanT = 256, kScanPer = 8, kScanC = kScanT * kScanPer;

__device__ double block_scan_excl(double v, double *wtot, double *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    double incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wtot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const double wv = lane < kScanT / 32 ? wtot[lane] : 0.0;
        double wi = wv;
#pragma unroll
        for (int o = 1; o < kScanT / 32; o <<= 1) {
            const double y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        if (lane < kScanT / 32) wtot[lane] = wi - wv;
        if (lane == kScanT / 32 - 1) *total = wi;
    }
    __syncthreads();
    return wtot[warp] + (incl - v);
}

__device__ __forceinline__ double scan_run(const double *in, int n, int base, double r[kScanPer]) {
    double s = 0.0;
#pragma unroll
    for (int j = 0; j < kScanPer; j++) {
        const int i = base + j;
        r[j] = i < n ? in[i] : 0.0;
    }
#pragma unroll
    for (int j = 0; j < kScanPer; j++) s += r[j];
    return s;
}

__global__ void __launch_bounds__(kScanT) seg_scan_part_kernel(const double *in, int n, double *btot) {
    __shared__ double wtot[kScanT / 32];
    __shared__ double total;
    double r[kScanPer];
    const double s = scan_run(in, n, blockIdx.x * kScanC + threadIdx.x * kScanPer, r);
    block_scan_excl(s, wtot, &total);
    if (threadIdx.x == 0) btot[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanT) seg_scan_kernel(const double *in, int n, const double *btot, double *out) {
    __shared__ double wtot[kScanT / 32];
    __shared__ double total, off;
    if (threadIdx.x < 32) {   // the totals of the blocks before this one, in order
        double o = 0.0;
        if (threadIdx.x == 0)
            for (int q = 0; q < (int)blockIdx.x; q++) o += btot[q];
        if (threadIdx.x == 0) off = o;
    }
    double r[kScanPer];
    const int base = blockIdx.x * kScanC + threadIdx.x * kScanPer;
    const double s = scan_run(in, n, base, r);
    double acc = block_scan_excl(s, wtot, &total) + off;
#pragma unroll
    for (int j = 0; j < kScanPer; j++) {
        const int i = base + j;
        if (i <= n) out[i] = acc;
        acc += r[j];
    }
    if (n == 0 && blockIdx.x == 0 && threadIdx.x == 0) out[0] = 0.0;
}

// ---------------------------------------------------------------------------
// DP edge weights.  Block handles RB = 32 consecutive endpoints i (last slot
// position e' = i - 1) and all predecessors a = i - len, len in [n_min, n_max];
// the banded dot products hbar_{cs+e'} . hbar_{cs+a} are formed tile-wise.
// ---------------------------------------------------------------------------
struct BandArgs {
    SegArgs s;
    int n_min, n_max, n0;
    double lambda_d, lambda_n, c_cut;
};

// Row stride of the DP edge weights: n_max - n_min + 1 floats padded to a
// multiple of 4, so that every row starts on a 16-byte boundary.
__host__ __device__ constexpr int dp_row(int nb) { return (nb + 3) & ~3; }

constexpr int kRB = 32;
constexpr int kKC = 32;   // channel chunk

template <typename Tin>
__global__ void __launch_bounds__(256) seg_band_kernel(const Tin *V, const float *hidden, BandArgs b,
                                                       const float *inv_norm, const float *nrm2,
                                                       const double *p2, const double *bscore,
                                                       float *ew) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const SegArgs &a = b.s;
    const int nb = b.n_max - b.n_min + 1, nbp = dp_row(nb);
    const int ncol = kRB + nb - 1;                   // predecessors a in [E0+1-n_max, E0+RB-n_min]
    float *As = reinterpret_cast<float *>(smem_raw); // [kKC][kRB] (conflict-free reads)
    float *Bs = As + kRB * kKC;                      // [ncol][kKC]
    const int E0 = blockIdx.x * kRB;                 // first e' of the block
    const int a0 = E0 + 1 - b.n_max;                 // first predecessor (relative, may be < 0)
    const int tid = threadIdx.x;
    const int r = tid & 31;                          // row (e' = E0 + r)
    const int cg = tid >> 5;                         // column group: columns cg, cg + 8, ...
    constexpr int kMaxCols = 24;                     // ncol <= 8 * 24
    float sd[kMaxCols];
#pragma unroll
    for (int k = 0; k < kMaxCols; k++) sd[k] = 0.f;
    for (int li = 0; li < a.nseg; li++) {
        int l = a.layers[li];
        float acc[kMaxCols];
#pragma unroll
        for (int k = 0; k < kMaxCols; k++) acc[k] = 0.f;
        for (int c0 = 0; c0 < a.D; c0 += kKC) {
            __syncthreads();
            for (int e = tid; e < kRB * kKC; e += 256) {
                int rr = e / kKC, cc = e % kKC;
                int ep = E0 + rr, c = c0 + cc;
                As[cc * kRB + rr] = (ep < a.N && c < a.D)
                            ? traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, a.cs + ep, c) : 0.f;
            }
            for (int e = tid; e < ncol * kKC; e += 256) {
                int rr = e / kKC, cc = e % kKC;
                int ap = a0 + rr, c = c0 + cc;
                Bs[e] = (ap >= 0 && ap < a.N && c < a.D)
                            ? traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, a.cs + ap, c) : 0.f;
            }
            __syncthreads();
#pragma unroll 4
            for (int cc = 0; cc < kKC; cc++) {
                float x = As[cc * kRB + r];
#pragma unroll
                for (int k = 0; k < kMaxCols; k++) {
                    int col = cg + 8 * k;
                    if (col < ncol) acc[k] = fmaf(x, Bs[col * kKC + cc], acc[k]);
                }
            }
        }
        int ep = E0 + r;
        if (ep < a.N) {
            float ie = inv_norm[(size_t)li * a.T + a.cs + ep];
            float ne = nrm2[(size_t)li * a.T + a.cs + ep];
#pragma unroll
            for (int k = 0; k < kMaxCols; k++) {
                int col = cg + 8 * k;
                int ap = a0 + col;
                if (col < ncol && ap >= 0 && ap <= ep) {
                    float ia = inv_norm[(size_t)li * a.T + a.cs + ap];
                    float na = nrm2[(size_t)li * a.T + a.cs + ap];
                    sd[k] += ne + na - 2.f * (ie * ia * acc[k]);
                }
            }
        }
    }
    // edge weights for endpoint i = ep + 1 and len = i - ap
    int ep = E0 + r;
    if (ep >= a.N) return;
    int i = ep + 1;
#pragma unroll
    for (int k = 0; k < kMaxCols; k++) {
        int col = cg + 8 * k;
        if (col >= ncol) continue;
        int ap = a0 + col;
        int len = i - ap;
        if (len < b.n_min || len > b.n_max) continue;
        double w;
        if (ap < 0) {
            ew[(size_t)i * nbp + (len - b.n_min)] = -INFINITY;
            continue;
        } else {
            int nS = len - 1;
            double disp = 0.0;
            if (nS >= 2) {
                double s2 = p2[ep] - p2[ap];     // sum_{t=ap}^{ep-1} ||d_t||^2
                disp = (s2 - (double)sd[k] / nS) / (double)(nS - 1) / a.nseg;
            }
            double gam = ap == 0 ? 0.0 : bscore[a.cs + ap - 1] - b.c_cut;
            double pen = (double)(len - b.n0) / b.n0;
            w = gam - b.lambda_d * disp - b.lambda_n * pen * pen;
        }
        ew[(size_t)i * nbp + (len - b.n_min)] = (float)w;
    }
}

// Tensor-core version for bf16 V trajectories.  Block = 64 endpoints (rows
// e' = E0 .. E0 + 63) x their predecessor band (columns a = a0 .. a0 + ncol - 1,
// ncol = 64 + nb - 1).  The raw bf16 rows are staged 64 channels at a time
// with cp.async (double buffered, row stride 72 halves: conflict-free fragment
// reads) and multiplied with mma.sync m16n8k16 (exact bf16 products, fp32
// sums); after each segmentation layer the Gram entries are folded into
// |hbar_e - hbar_a|^2 = |hbar_e|^2 + |hbar_a|^2 - 2 inv_e inv_a (h_e . h_a).
// Warp w owns row tile w % 4 and every other column tile of that row tile's
// band (the column tiles [2 mt, (16 mt + 15 + nb - 1) / 8]).
// ---------------------------------------------------------------------------
constexpr int kBM = 64;               // endpoints per block
constexpr int kBK = 64;               // channels per stage
constexpr int kBStride = kBK + 8;     // staged row stride (halves)
constexpr int kBNtW = 9;              // column tiles per warp: ceil(18 / 2) for nb <= 128

__host__ __device__ constexpr int band_ncol_tiles(int nb) { return (kBM + nb - 1 + 7) / 8; }
__host__ __device__ constexpr size_t band_mma_smem(int nb) {
    return (size_t)2 * (kBM + 8 * band_ncol_tiles(nb)) * kBStride * sizeof(__nv_bfloat16) +
           (size_t)2 * (kBM + 8 * band_ncol_tiles(nb)) * sizeof(float) + (size_t)3 * 128 * sizeof(double);
}

__global__ void __launch_bounds__(256) seg_band_mma_kernel(const __nv_bfloat16 *V, BandArgs b,
                                                           const float *inv_norm, const float *nrm2,
                                                           const double *p2, const double *bscore,
                                                           float *ew) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const SegArgs &a = b.s;
    const int nb = b.n_max - b.n_min + 1, nbp = dp_row(nb);
    const int nct = band_ncol_tiles(nb);
    const int nrs = kBM + 8 * nct;                      // staged rows: A rows, then B rows
    __nv_bfloat16 *stg = reinterpret_cast<__nv_bfloat16 *>(smem_raw);   // [2][nrs][kBStride]
    float *inv_r = reinterpret_cast<float *>(stg + (size_t)2 * nrs * kBStride);   // [nrs]
    float *nrm_r = inv_r + nrs;                                                    // [nrs]
    // per slot length len = n_min + k: 1 / nS, 1 / ((nS - 1) n_seg) (nS = len - 1)
    // and lambda_n pen^2, so that the edge weights need no fp64 division
    double *t_ins = reinterpret_cast<double *>(nrm_r + nrs);   // [128] (8-byte aligned: 296 nrs bytes in)
    double *t_idn = t_ins + 128, *t_pen = t_idn + 128;
    for (int k = threadIdx.x; k < nb; k += blockDim.x) {
        const int len = b.n_min + k, nS = len - 1;
        t_ins[k] = nS >= 1 ? 1.0 / nS : 0.0;
        t_idn[k] = nS >= 2 ? 1.0 / (double)(nS - 1) / a.nseg : 0.0;
        const double pen = (double)(len - b.n0) / b.n0;
        t_pen[k] = b.lambda_n * pen * pen;
    }
    const int E0 = blockIdx.x * kBM;
    const int a0 = E0 + 1 - b.n_max;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int gr = lane >> 2, c2 = 2 * (lane & 3);
    const int mt = warp & 3, hw = warp >> 2;
    const int nt_lo = 2 * mt, nt_hi = min(nct - 1, (16 * mt + 15 + nb - 1) / 8);
    // relative position (index into the compressible region) of staged row r
    auto rel = [&](int r) { return r < kBM ? E0 + r : a0 + (r - kBM); };
    auto valid = [&](int x) { return x >= 0 && x < a.N; };

    float acc[kBNtW][4], sd[kBNtW][4];
#pragma unroll
    for (int q = 0; q < kBNtW; q++)
#pragma unroll
        for (int h = 0; h < 4; h++) acc[q][h] = sd[q][h] = 0.f;

    const int nchunk = a.D / kBK;
    const int nstage = a.nseg * nchunk;
    auto stage = [&](int st) {
        const int li = st / nchunk, c0 = (st - li * nchunk) * kBK;
        const int l = a.layers[li], g = c0 / a.d, i = c0 - g * a.d;
        __nv_bfloat16 *dst = stg + (size_t)(st & 1) * nrs * kBStride;
        for (int e = tid; e < nrs * (kBK / 8); e += 256) {
            const int r = e >> 3, q = e & 7;
            const int x = rel(r);
            const bool ok = valid(x);
            const __nv_bfloat16 *src = V + (((size_t)l * a.G + g) * a.T + a.cs + (ok ? x : 0)) * a.d + i + 8 * q;
            cp_async16(dst + (size_t)r * kBStride + 8 * q, src, ok);
        }
        cp_async_commit();
    };
    stage(0);
    for (int st = 0; st < nstage; st++) {
        const int li = st / nchunk, ch = st - li * nchunk;
        if (ch == 0) {   // this layer's norms of the staged rows
            for (int r = tid; r < nrs; r += 256) {
                const int x = rel(r);
                const bool ok = valid(x);
                inv_r[r] = ok ? inv_norm[(size_t)li * a.T + a.cs + x] : 0.f;
                nrm_r[r] = ok ? nrm2[(size_t)li * a.T + a.cs + x] : 0.f;
            }
        }
        if (st + 1 < nstage) {
            stage(st + 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const __nv_bfloat16 *As = stg + (size_t)(st & 1) * nrs * kBStride;
        const __nv_bfloat16 *Bs = As + (size_t)kBM * kBStride;
#pragma unroll
        for (int ks = 0; ks < kBK / 16; ks++) {
            uint32_t af[4];
            const __nv_bfloat16 *ar = As + (size_t)(16 * mt + gr) * kBStride + ks * 16 + c2;
            af[0] = *reinterpret_cast<const uint32_t *>(ar);
            af[1] = *reinterpret_cast<const uint32_t *>(ar + 8 * kBStride);
            af[2] = *reinterpret_cast<const uint32_t *>(ar + 8);
            af[3] = *reinterpret_cast<const uint32_t *>(ar + 8 * kBStride + 8);
#pragma unroll
            for (int q = 0; q < kBNtW; q++) {
                const int nt = nt_lo + 2 * q + hw;
                if (nt > nt_hi) break;
                const __nv_bfloat16 *br = Bs + (size_t)(nt * 8 + gr) * kBStride + ks * 16 + c2;
                mma_bf16(acc[q], af, *reinterpret_cast<const uint32_t *>(br),
                         *reinterpret_cast<const uint32_t *>(br + 8));
            }
        }
        if (ch == nchunk - 1) {   // fold this layer: sd += |hbar_e|^2 + |hbar_a|^2 - 2 hbar_e . hbar_a
#pragma unroll
            for (int q = 0; q < kBNtW; q++) {
                const int nt = nt_lo + 2 * q + hw;
                if (nt > nt_hi) break;
#pragma unroll
                for (int h = 0; h < 4; h++) {
                    const int row = 16 * mt + gr + (h >= 2 ? 8 : 0);
                    const int col = nt * 8 + c2 + (h & 1);
                    const float ie = inv_r[row], ne = nrm_r[row];
                    const float ia = inv_r[kBM + col], na = nrm_r[kBM + col];
                    sd[q][h] += ne + na - 2.f * (ie * ia * acc[q][h]);
                    acc[q][h] = 0.f;
                }
            }
        }
        __syncthreads();   // buffer st & 1 and the norms are reused
    }
    // edge weights for endpoint i = ep + 1 and len = i - ap
#pragma unroll
    for (int q = 0; q < kBNtW; q++) {
        const int nt = nt_lo + 2 * q + hw;
        if (nt > nt_hi) break;
#pragma unroll
        for (int h = 0; h < 4; h++) {
            const int row = 16 * mt + gr + (h >= 2 ? 8 : 0);
            const int col = nt * 8 + c2 + (h & 1);
            const int ep = E0 + row, ap = a0 + col;
            if (ep >= a.N) continue;
            const int i = ep + 1, len = i - ap;
            if (len < b.n_min || len > b.n_max) continue;
            if (ap < 0) {
                ew[(size_t)i * nbp + (len - b.n_min)] = -INFINITY;
                continue;
            }
            const int nS = len - 1, kl = len - b.n_min;
            double disp = 0.0;
            if (nS >= 2) {
                const double s2 = p2[ep] - p2[ap];     // sum_{t=ap}^{ep-1} ||d_t||^2
                disp = (s2 - (double)sd[q][h] * t_ins[kl]) * t_idn[kl];
            }
            const double gam = ap == 0 ? 0.0 : bscore[a.cs + ap - 1] - b.c_cut;
            ew[(size_t)i * nbp + kl] = (float)(gam - b.lambda_d * disp - t_pen[kl]);
        }
    }
}

// Terminal relaxation weights at i = N: len in [1, n_max]; warp per len.
template <typename Tin>
__global__ void seg_band_terminal_kernel(const Tin *V, const float *hidden, BandArgs b,
                                         const float *inv_norm, const float *nrm2,
                                         const double *p2, const double *bscore, float2 *ewt) {
    const SegArgs &a = b.s;
    int len = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32 + 1;
    int lane = threadIdx.x & 31;
    if (len > b.n_max) return;
    int i = a.N, ep = i - 1, ap = i - len;
    if (ap < 0) {
        if (lane == 0) ewt[len] = make_float2(-INFINITY, 0.f);
        return;
    }
    double sd = 0.0;
    for (int li = 0; li < a.nseg; li++) {
        int l = a.layers[li];
        float f = 0.f;
        for (int c = lane; c < a.D; c += 32)
            f = fmaf(traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, a.cs + ep, c),
                     traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, a.cs + ap, c), f);
        f = warp_sum(f);
        float ie = inv_norm[(size_t)li * a.T + a.cs + ep], ia = inv_norm[(size_t)li * a.T + a.cs + ap];
        sd += nrm2[(size_t)li * a.T + a.cs + ep] + nrm2[(size_t)li * a.T + a.cs + ap] - 2.f * (ie * ia * f);
    }
    if (lane) return;
    int nS = len - 1;
    double disp = 0.0;
    if (nS >= 2) disp = ((p2[ep] - p2[ap]) - sd / nS) / (double)(nS - 1) / a.nseg;
    double gam = ap == 0 ? 0.0 : bscore[a.cs + ap - 1] - b.c_cut;
    double pen = (double)(len - b.n0) / b.n0;
    ewt[len] = df_split(gam - b.lambda_d * disp - b.lambda_n * pen * pen);
}

// ---------------------------------------------------------------------------
// DP (App. B.3 Eq. app_dp_recurrence): F[i] = max over lengths of
// F[i - len] + w(i - len, i), lengths in [n_min, n_max], ties to the lower
// predecessor.  The chain is cut into chunks that run on separate CTAs.
//
// Inside a CTA, one warp per endpoint: endpoints are processed 16 (or n_min,
// if smaller) at a time -- F[i..i+15] only read F[< i] because i - a >= n_min,
// so one barrier per step suffices.  Lane handles the lengths n_min + lane +
// 32 j; the warp reduces its candidates (value desc, a asc) with shuffles.
// The edge weights do not depend on F: each warp streams its own endpoint
// rows kDpPD steps ahead into a private shared-memory ring with cp.async.
// The state F is a double-float; the edge weights are fp32 (their rounding,
// ~1e-7 of a weight, is far below the DP's near-tie margin).
//
// Across CTAs: chunk c owns the endpoints (e_c, e_c+1], e_c = c S.  Its run
// starts Wu tokens before e_c from F = 0 on a window of n_max positions
// instead of the true state.  The decisions read only differences of F inside
// the window, and once the optimal paths from the window have coalesced, the
// run's F is the true F plus a constant: products of max-plus transition
// matrices converge to rank one (Maleki, Musuvathi and Mytkowicz, PPoPP 2014,
// "Parallelizing dynamic programming through rank convergence").  Each chunk
// records its state on the kDpWin positions ending at e_c (its head) and its
// ring at the end of the run (its tail).  Chunk c's decisions are the true ones
// when chunk c - 1's are and the previous tail minus this head is constant over
// the window: checked in fp64 to kDpTol relative, nine orders below any
// decision margin the tests accept as distinct (a run that has not converged
// differs by whole edge weights).  Chunk 0, and every chunk whose warm-up
// would reach back to the context start, runs from the true state F[0] = 0.
// The finish kernel checks every boundary, re-runs in order each chunk whose
// check fails from the previous tail (then exact), and backtracks.
// ---------------------------------------------------------------------------
constexpr int kDpRing = 256;
constexpr int kDpEp = 16;         // endpoints per step (warps)
constexpr int kDpPD = 8;          // steps of edge weights in flight per warp
constexpr int kDpLen = 4;         // lengths per lane: n_max - n_min + 1 <= 128
constexpr int kDpWin = 128;       // state window compared at a boundary (>= n_max)
constexpr int kDpChunkSteps = 32; // steps per chunk
constexpr double kDpTol = 1e-9;   // boundary check: relative spread of tail - head

__host__ __device__ constexpr size_t dp_smem_base(int nb) {
    return (size_t)kDpRing * 8 + (size_t)kDpEp * kDpPD * dp_row(nb) * 4;
}
// chunk kernel: the base plus the chunk's chosen lengths [S + 1]
__host__ __device__ constexpr size_t dp_smem_chunk(int nb, int S) {
    return dp_smem_base(nb) + (((size_t)S + 1 + 15) & ~(size_t)15);
}
// finish kernel: the base, the boundary flags [nch] and the exit table
// [nch][n_max] (uint8), the chunks' entries and counts [nch] (int32)
__host__ __device__ constexpr size_t dp_smem(int nb, int nch, int n_max) {
    return dp_smem_base(nb) + (((size_t)nch + 15) & ~(size_t)15) + (((size_t)nch * n_max + 15) & ~(size_t)15) +
           (size_t)nch * 8;
}

__device__ __forceinline__ bool better(df2 v, int a, df2 bv, int ba) {
    return df_gt(v, bv) || (df_eq(v, bv) && a < ba);
}

// A chunk's run starts from the true state when its warm-up would begin
// within kDpWin tokens of the context start.
__host__ __device__ __forceinline__ bool dp_exact(int c, int S, int Wu) {
    return c == 0 || (long long)c * S - Wu < kDpWin;
}

// Runs the recurrence for the endpoints i_lo + 1 .. i_hi, step at a time.  On
// entry the ring holds F of the positions i_lo - n_max .. i_lo; on exit the
// positions i_hi - kDpRing + 1 .. i_hi.  The chosen length of endpoint i is
// stored to len_out[i - len_from] for i > len_from.  With head non-null, the kDpWin
// ring entries ending at head_at are copied there once endpoint head_at is
// done (head_at - i_lo a multiple of step).  All threads of the block call it.
__device__ void dp_run(const float *ew, int N, int n_min, int n_max, int i_lo, int i_hi,
                       df2 *ring, float *wbuf, uint8_t *len_out, int len_from,
                       int head_at, df2 *head) {
    const int nb = n_max - n_min + 1, nbp = dp_row(nb);
    const int tid = threadIdx.x, lane = tid & 31, k = tid >> 5;
    const int step = min(n_min, kDpEp);
    const df2 NEG = df2{-INFINITY, 0.f};
    float *mybuf = wbuf + (size_t)k * kDpPD * nbp;
    // row of endpoint i into stage q of this warp's ring (16-byte chunks)
    auto fetch = [&](int i, int q) {
        const bool ok = k < step && i <= i_hi;
        for (int c4 = lane; c4 < nbp / 4; c4 += 32)
            cp_async16(mybuf + (size_t)q * nbp + 4 * c4, ew + (size_t)(ok ? i : 0) * nbp + 4 * c4, ok);
        cp_async_commit();
    };
#pragma unroll
    for (int q = 0; q < kDpPD; q++) fetch(i_lo + 1 + q * step + k, q);
    __syncthreads();
    int q = 0;
    for (int i0 = i_lo + 1; i0 <= i_hi; i0 += step) {
        const int i = i0 + k;
        const bool act = k < step && i <= i_hi;
        cp_async_wait<kDpPD - 1>();   // this step's row (the oldest group) has landed
        __syncwarp();
        const float *wr = mybuf + (size_t)q * nbp;
        // the lane's candidates are independent: form them all, then keep the best
        df2 v[kDpLen];
        int av[kDpLen];
#pragma unroll
        for (int j = 0; j < kDpLen; j++) {
            const int len = n_min + lane + 32 * j;
            const int a = i - len;
            const bool ok = act && len <= n_max && a >= 0;
            const df2 fa = ring[ok ? (a & (kDpRing - 1)) : 0];
            const float w = wr[ok ? len - n_min : 0];
            const bool live = ok && fa.hi != -INFINITY;
            v[j] = live ? df_add(fa, make_float2(w, 0.f)) : NEG;
            av[j] = live ? a : 0x7fffffff;
        }
        df2 best = v[0];
        int ba = av[0];
#pragma unroll
        for (int j = 1; j < kDpLen; j++)
            if (better(v[j], av[j], best, ba)) { best = v[j]; ba = av[j]; }
        __syncwarp();
        fetch(i0 + kDpPD * step + k, q);   // reuse the stage for kDpPD steps ahead
        q = q + 1 == kDpPD ? 0 : q + 1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            df2 ov;
            ov.hi = __shfl_xor_sync(0xffffffffu, best.hi, o);
            ov.lo = __shfl_xor_sync(0xffffffffu, best.lo, o);
            const int oa = __shfl_xor_sync(0xffffffffu, ba, o);
            if (better(ov, oa, best, ba)) { best = ov; ba = oa; }
        }
        if (lane == 0 && act) {
            ring[i & (kDpRing - 1)] = best;
            if (i > len_from) len_out[i - len_from] = best.hi == -INFINITY ? 0 : (uint8_t)(i - ba);
        }
        __syncthreads();
        if (head && i0 + step - 1 == head_at && tid < kDpWin) {
            const int x = head_at - kDpWin + 1 + tid;
            head[tid] = x < 0 ? NEG : ring[x & (kDpRing - 1)];
        }
    }
    cp_async_wait<0>();
    __syncthreads();
}

// The ring, in position order, ending at position e (entries before the
// context start read as unreachable).
__device__ __forceinline__ void dp_save_ring(const df2 *ring, int e, df2 *out) {
    for (int t = threadIdx.x; t < kDpRing; t += blockDim.x) {
        const int x = e - kDpRing + 1 + t;
        out[t] = x < 0 ? df2{-INFINITY, 0.f} : ring[x & (kDpRing - 1)];
    }
}

// Exit table of chunk c (endpoints (e0, e1]): for q < n_max, following the
// chosen lengths from z = e1 - q down, the first position <= e0 is
// e0 - tab[q] (z itself when z <= e0); 255 when the walk meets an
// unreachable endpoint or z < 0.  len(i) is the chosen length of i in (e0, e1].
template <typename LenF>
__device__ __forceinline__ uint8_t dp_exit(int e0, int e1, int q, LenF len) {
    int z = e1 - q;
    if (z < 0) return 255;
    while (z > e0) {
        const int l = len(z);
        if (l == 0) return 255;
        z -= l;
    }
    return (uint8_t)(e0 - z);   // < n_max: the last step into (e0 - n_max, e0], or z = 0 with e0 < n_max
}

__global__ void __launch_bounds__(kDpEp * 32) seg_dp_chunk_kernel(const float *ew, int N, int n_min, int n_max,
                                                                int S, int Wu, uint8_t *len_g, df2 *head,
                                                                df2 *tail, uint8_t *tab_g) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    df2 *ring = reinterpret_cast<df2 *>(smem_raw);          // [kDpRing]
    float *wbuf = reinterpret_cast<float *>(ring + kDpRing); // [kDpEp][kDpPD][nbp]
    uint8_t *lloc = smem_raw + dp_smem_base(n_max - n_min + 1);   // [S + 1] lengths of (e0, e1]
    const int c = blockIdx.x;
    const int e0 = c * S, e1 = min(N, e0 + S);
    const bool exact = dp_exact(c, S, Wu);
    const int s0 = exact ? 0 : e0 - Wu;
    for (int t = threadIdx.x; t < kDpRing; t += blockDim.x)
        ring[t] = exact ? df2{t == 0 ? 0.f : -INFINITY, 0.f} : df2{0.f, 0.f};
    __syncthreads();
    dp_run(ew, N, n_min, n_max, s0, e1, ring, wbuf, lloc, e0, exact ? -1 : e0,
           exact ? nullptr : head + (size_t)c * kDpWin);
    dp_save_ring(ring, e1, tail + (size_t)c * kDpRing);
    for (int i = e0 + 1 + threadIdx.x; i <= e1; i += blockDim.x) len_g[i] = lloc[i - e0];
    for (int q = threadIdx.x; q < n_max; q += blockDim.x)
        tab_g[(size_t)c * n_max + q] = dp_exit(e0, e1, q, [&](int z) { return (int)lloc[z - e0]; });
}

// Difference of two double-float numbers in double-float (two-sum of the
// high parts, then the low parts added).
__device__ __forceinline__ df2 df_sub(df2 a, df2 b) {
    const float s = a.hi - b.hi;
    const float bb = s - a.hi;
    float e = (a.hi - (s - bb)) + (-b.hi - bb);
    e += a.lo - b.lo;
    const float hi = s + e;
    return df2{hi, e - (hi - s)};
}

// Whether the state window `b` (a chunk's head) equals `a` (the previous
// tail's last kDpWin entries) up to a constant on its last n_max positions,
// the only ones the endpoints after the boundary read.  The differences are
// formed in double-float (fp64 is slow on this part).  One warp; the result
// is returned to every lane.
__device__ bool dp_match(const df2 *a, const df2 *b, int n_max, int lane) {
    df2 dmin = df2{INFINITY, 0.f}, dmax = df2{-INFINITY, 0.f};
    float scale = 0.f;
    bool bad = false;
    for (int t = kDpWin - n_max + lane; t < kDpWin; t += 32) {   // the positions later endpoints read
        const df2 x = a[t], y = b[t];
        const bool xi = x.hi == -INFINITY, yi = y.hi == -INFINITY;
        if (xi && yi) continue;
        const df2 dv = df_sub(x, y);
        if (xi != yi || !(fabsf(dv.hi) <= FLT_MAX)) { bad = true; continue; }   // also NaN / Inf
        if (df_gt(dmin, dv)) dmin = dv;
        if (df_gt(dv, dmax)) dmax = dv;
        scale = fmaxf(scale, fmaxf(fabsf(x.hi), fabsf(y.hi)));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        df2 v;
        v.hi = __shfl_xor_sync(0xffffffffu, dmin.hi, o);
        v.lo = __shfl_xor_sync(0xffffffffu, dmin.lo, o);
        if (df_gt(dmin, v)) dmin = v;
        v.hi = __shfl_xor_sync(0xffffffffu, dmax.hi, o);
        v.lo = __shfl_xor_sync(0xffffffffu, dmax.lo, o);
        if (df_gt(v, dmax)) dmax = v;
        scale = fmaxf(scale, __shfl_xor_sync(0xffffffffu, scale, o));
    }
    if (__any_sync(0xffffffffu, bad)) return false;
    if (dmax.hi == -INFINITY) return true;   // nothing reachable on either side
    return df_sub(dmax, dmin).hi <= (float)kDpTol * (1.f + scale);
}

__global__ void __launch_bounds__(kDpEp * 32) seg_dp_finish_kernel(const float *ew, const float2 *ewt, int N,
                                                                 int n_min, int n_max, int S, int Wu, int nch,
                                                                 uint8_t *len_g, const df2 *head, df2 *tail,
                                                                 const uint8_t *tab_g, int cs, int32_t *slots,
                                                                 int *dev_int) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int nb = n_max - n_min + 1;
    df2 *ring = reinterpret_cast<df2 *>(smem_raw);
    float *wbuf = reinterpret_cast<float *>(ring + kDpRing);
    uint8_t *ok = smem_raw + dp_smem_base(nb);                                  // [nch]
    uint8_t *tab = ok + (((size_t)nch + 15) & ~(size_t)15);                      // [nch][n_max]
    int *ent = reinterpret_cast<int *>(tab + (((size_t)nch * n_max + 15) & ~(size_t)15));   // [nch]
    int *cnt = ent + nch;                                                       // [nch]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    for (int q = tid; q < nch * n_max; q += blockDim.x) tab[q] = tab_g[q];
    for (int c = warp; c < nch; c += nw) {
        const bool m = dp_exact(c, S, Wu) ||
                       dp_match(tail + (size_t)(c - 1) * kDpRing + (kDpRing - kDpWin), head + (size_t)c * kDpWin, n_max, lane);
        if (lane == 0) ok[c] = m;
    }
    __syncthreads();
    // chunks in order: a chunk re-run changes its tail, so the next boundary is checked again
    int rerun = 0;
    bool prev = false;
    for (int c = 1; c < nch; c++) {
        if (prev) {
            if (warp == 0) {
                const bool m = dp_exact(c, S, Wu) ||
                               dp_match(tail + (size_t)(c - 1) * kDpRing + (kDpRing - kDpWin),
                                        head + (size_t)c * kDpWin, n_max, lane);
                if (lane == 0) ok[c] = m;
            }
            __syncthreads();
        }
        prev = !ok[c];
        if (!prev) continue;
        const int e0 = c * S, e1 = min(N, e0 + S);
        for (int t = tid; t < kDpRing; t += blockDim.x)
            ring[(e0 - kDpRing + 1 + t) & (kDpRing - 1)] = tail[(size_t)(c - 1) * kDpRing + t];
        __syncthreads();
        dp_run(ew, N, n_min, n_max, e0, e1, ring, wbuf, len_g + e0, e0, -1, nullptr);
        dp_save_ring(ring, e1, tail + (size_t)c * kDpRing);
        __threadfence_block();
        __syncthreads();
        for (int q = tid; q < n_max; q += blockDim.x)   // the chunk's exit table, from its new lengths
            tab[(size_t)c * n_max + q] = dp_exit(e0, e1, q, [&](int z) { return (int)len_g[z]; });
        __syncthreads();
        rerun++;
    }
    __shared__ int sJ;
    if (tid == 0) {
        dev_int[kDpRerun] = rerun;
        const df2 *F = tail + (size_t)(nch - 1) * kDpRing;   // F(N - kDpRing + 1 + t) = F[t]
        if (F[kDpRing - 1].hi == -INFINITY) {
            // terminal relaxation (Eq. app_terminal_predecessor): 1 <= N - a <= n_max,
            // read after every F[< N] has been written
            df2 best = df2{-INFINITY, 0.f};
            int ba = 0x7fffffff;
            for (int len = 1; len <= n_max; len++) {
                int a = N - len;
                if (a < 0) break;
                df2 fa = F[kDpRing - 1 - len];
                if (fa.hi == -INFINITY || ewt[len].x == -INFINITY) continue;
                df2 v = df_add(fa, ewt[len]);
                if (better(v, a, best, ba)) { best = v; ba = a; }
            }
            len_g[N] = best.hi == -INFINITY ? 0 : (uint8_t)(N - ba);
        }
        // the path's first endpoint in each chunk, from the top: the last chunk
        // is walked from N itself (its relaxed length), the others by their tables
        int z = N, bad = 0;
        for (int c = nch - 1; c >= 0; c--) {
            ent[c] = z;
            if (z == 0) continue;
            const int e0 = c * S, e1 = min(N, e0 + S), q = e1 - z;
            if (q < 0 || q >= n_max) { bad = 1; break; }
            const uint8_t o = c == nch - 1 ? dp_exit(e0, e1, 0, [&](int y) { return (int)len_g[y]; })
                                           : tab[(size_t)c * n_max + q];
            if (o == 255) { bad = 1; break; }
            z = e0 - o;
        }
        sJ = bad ? -1 : 0;
    }
    __syncthreads();
    if (sJ < 0) {
        if (tid == 0) dev_int[0] = -1;
        return;
    }
    // endpoints of the path inside each chunk, then their offsets from the top
    for (int c = tid; c < nch; c += blockDim.x) {
        const int e0 = c * S;
        int k = 0;
        for (int z = ent[c]; z > e0 && z > 0;) {   // every length on it is >= 1 (checked above)
            const int l = len_g[z];
            if (l == 0) break;
            k++;
            z -= l;
        }
        cnt[c] = k;
    }
    __syncthreads();
    if (tid == 0) {   // exclusive offsets from the top chunk down; J = all of them
        int acc = 0;
        for (int c = nch - 1; c >= 0; c--) {
            const int k = cnt[c];
            cnt[c] = acc;
            acc += k;
        }
        sJ = acc;
    }
    __syncthreads();
    const int J = sJ;
    for (int c = tid; c < nch; c += blockDim.x) {   // the m-th endpoint from the top is slot start J - m
        const int e0 = c * S;
        int m = cnt[c];
        for (int z = ent[c]; z > e0 && z > 0;) {
            const int l = len_g[z];
            if (l == 0) break;
            slots[J - m++] = cs + z;
            z -= l;
        }
    }
    if (tid == 0) {
        slots[0] = cs;
        dev_int[0] = J;
    }
}

}  // namespace

// Chunks of the segmentation DP: S endpoints per chunk (kDpChunkSteps steps),
// a warm-up of Wu tokens (p.dp_warmup rounded up to whole steps, default 512;
// negative: one chunk, the plain sequential recurrence).
void dp_chunking(const gkv_params &p, int N, int *S, int *Wu, int *nch) {
    const int step = std::min(p.n_min, kDpEp);
    if (p.dp_warmup < 0) {
        *S = std::max(step, (N + step - 1) / step * step);
        *Wu = step;
        *nch = 1;
        return;
    }
    const int w = p.dp_warmup == 0 ? 512 : std::min(p.dp_warmup, std::max(N, 1));
    *S = kDpChunkSteps * step;
    *Wu = std::max(step, (w + step - 1) / step * step);
    *nch = std::max(1, (N + *S - 1) / *S);
}

size_t dp_smem_bytes(const gkv_params &p, int N) {
    int S, Wu, nch;
    dp_chunking(p, N, &S, &Wu, &nch);
    const int nb = p.n_max - p.n_min + 1;
    return std::max(dp_smem_chunk(nb, S), dp_smem(nb, nch, p.n_max));
}

// ---------------------------------------------------------------------------
cudaError_t launch_segment(Ctx &c, const void *V, const float *hidden, int Dh,
                           const float *surprisal, float *kappa_out, cudaStream_t s) {
    const gkv_params &p = c.p;
    Workspace &w = c.w;
    SegArgs a;
    a.L = p.L; a.G = p.G; a.T = p.T; a.d = p.d;
    a.D = hidden ? Dh : p.G * p.d;
    a.Dh = Dh;
    a.nseg = c.nseg; a.nwin = c.nwin;
    a.cs = p.ctx_start; a.N = c.Nc;
    for (int i = 0; i < kMaxSegLayers; i++) a.layers[i] = i < c.nseg ? c.seg_layers[i] : 0;
    for (int i = 0; i < kMaxWindows; i++) a.windows[i] = i < c.nwin ? p.windows[i] : 1;
    const bool bf = p.dtype == GKV_BF16;
    const __nv_bfloat16 *Vb = static_cast<const __nv_bfloat16 *>(V);
    const float *Vf = static_cast<const float *>(V);

    dim3 gn((p.T + 7) / 8, c.nseg);
    if (bf) seg_norm_kernel<<<gn, 256, 0, s>>>(Vb, hidden, a, w.inv_norm, w.nrm2);
    else seg_norm_kernel<<<gn, 256, 0, s>>>(Vf, hidden, a, w.inv_norm, w.nrm2);

    // curvature: one thread per position, staged normalised channels
    {
        const bool defw = c.nwin == 3 && p.windows[0] == 4 && p.windows[1] == 8 && p.windows[2] == 16;
        dim3 gc((p.T + kCurvPT - 1) / kCurvPT, c.nseg);
        const int sm = (int)kCurvSmem;
        if (bf && !hidden) {
            if (defw) {
                cudaFuncSetAttribute(seg_curv_kernel<__nv_bfloat16, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
                seg_curv_kernel<__nv_bfloat16, true><<<gc, 256, sm, s>>>(Vb, hidden, a, w.inv_norm, w.klw);
            } else {
                cudaFuncSetAttribute(seg_curv_kernel<__nv_bfloat16, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
                seg_curv_kernel<__nv_bfloat16, false><<<gc, 256, sm, s>>>(Vb, hidden, a, w.inv_norm, w.klw);
            }
        } else {
            const float *Vx = bf ? nullptr : Vf;
            if (defw) {
                cudaFuncSetAttribute(seg_curv_kernel<float, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
                seg_curv_kernel<float, true><<<gc, 256, sm, s>>>(Vx, hidden, a, w.inv_norm, w.klw);
            } else {
                cudaFuncSetAttribute(seg_curv_kernel<float, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
                seg_curv_kernel<float, false><<<gc, 256, sm, s>>>(Vx, hidden, a, w.inv_norm, w.klw);
            }
        }
    }
    seg_combine_kernel<<<(p.T + 255) / 256, 256, 0, s>>>(w.klw, c.nseg * c.nwin, p.T, p.lambda_stab,
                                                          w.kappa, kappa_out, w.dev_int + 1);
    // boundary score b = z(kappa) + lambda_s z(surprisal)
    SelState *st = reinterpret_cast<SelState *>(w.sel_state);
    robust_z(w.kappa, p.T, 1.0, 0, w.bscore, w.zdev, st, w.sel_hist, c.num_sms, &c.launches, s);
    if (surprisal) {
        f32_to_f64_kernel<<<(p.T + 255) / 256, 256, 0, s>>>(surprisal, p.T, w.zbuf);
        robust_z(w.zbuf, p.T, p.lambda_s, 1, w.bscore, w.zdev, st, w.sel_hist, c.num_sms, &c.launches, s);
    }
    // prefix of sum_l ||d_t||^2 over the compressible region
    int N = c.Nc;
    if (N > 1) {
        int nw8 = (N - 1 + 7) / 8;
        if (bf) seg_dd_kernel<<<nw8, 256, 0, s>>>(Vb, hidden, a, w.inv_norm, w.zbuf);
        else seg_dd_kernel<<<nw8, 256, 0, s>>>(Vf, hidden, a, w.inv_norm, w.zbuf);
    }
    {
        const int ns = N > 1 ? N - 1 : 0, nbs = ns / kScanC + 1;   // blocks cover [0, ns]
        double *btot = reinterpret_cast<double *>(w.zdev);   // free after the robust z (nbs <= T)
        seg_scan_part_kernel<<<nbs, kScanT, 0, s>>>(w.zbuf, ns, btot);
        seg_scan_kernel<<<nbs, kScanT, 0, s>>>(w.zbuf, ns, btot, w.p2);
    }
    // edge weights
    BandArgs b;
    b.s = a;
    b.n_min = p.n_min; b.n_max = p.n_max; b.n0 = p.n0;
    b.lambda_d = p.lambda_d; b.lambda_n = p.lambda_n; b.c_cut = p.c_cut;
    int nb = p.n_max - p.n_min + 1;
    int ncol = kRB + nb - 1;
    if (ncol > 8 * 24) return cudaErrorInvalidConfiguration;
    size_t smb = (size_t)(kRB + ncol) * kKC * 4;
    int gb = (N + kRB - 1) / kRB;
    if (bf && !hidden && a.D % kBK == 0 && a.d % kBK == 0 && nb <= 128) {
        const int gm = (N + kBM - 1) / kBM;
        const int smm = (int)band_mma_smem(nb);
        cudaFuncSetAttribute(seg_band_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smm);
        seg_band_mma_kernel<<<gm, 256, smm, s>>>(Vb, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ew);
        seg_band_terminal_kernel<<<(p.n_max + 7) / 8, 256, 0, s>>>(Vb, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ewt);
    } else if (bf) {
        seg_band_kernel<<<gb, 256, smb, s>>>(Vb, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ew);
        seg_band_terminal_kernel<<<(p.n_max + 7) / 8, 256, 0, s>>>(Vb, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ewt);
    } else {
        seg_band_kernel<<<gb, 256, smb, s>>>(Vf, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ew);
        seg_band_terminal_kernel<<<(p.n_max + 7) / 8, 256, 0, s>>>(Vf, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ewt);
    }
    int S, Wu, nch;
    dp_chunking(p, N, &S, &Wu, &nch);
    const size_t smc = dp_smem_chunk(nb, S), smd = dp_smem(nb, nch, p.n_max);
    if (std::max(smc, smd) > 227 * 1024 - 64 || nb > 32 * kDpLen) return cudaErrorInvalidConfiguration;   // 64: static shared
    cudaFuncSetAttribute(seg_dp_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smc);
    cudaFuncSetAttribute(seg_dp_finish_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smd);
    df2 *head = reinterpret_cast<df2 *>(w.dp_head), *tail = reinterpret_cast<df2 *>(w.dp_tail);
    seg_dp_chunk_kernel<<<nch, kDpEp * 32, smc, s>>>(w.ew, N, p.n_min, p.n_max, S, Wu, w.dp_len, head, tail,
                                                      w.dp_tab);
    seg_dp_finish_kernel<<<1, kDpEp * 32, smd, s>>>(w.ew, w.ewt, N, p.n_min, p.n_max, S, Wu, nch, w.dp_len,
                                                    head, tail, w.dp_tab, p.ctx_start, w.slots, w.dev_int);
    c.launches += 9 + (surprisal ? 1 : 0) + (N > 1 ? 1 : 0);   // and the robust z's own
    return cudaGetLastError();
}

}  // namespace gkv
