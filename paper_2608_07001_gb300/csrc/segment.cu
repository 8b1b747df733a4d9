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
    double s = 0.0;
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
            s += (double)x * x;
        }
    }
    s = warp_sum(s);
    if (lane == 0) {
        double n = sqrt(s);
        double den = n > kEps ? n : kEps;
        inv_norm[(size_t)li * a.T + t] = (float)(1.0 / den);
        nrm2[(size_t)li * a.T + t] = (float)(s / (den * den));
    }
}

// ---------------------------------------------------------------------------
// Curvature.  Block = 256 threads, tile of PT positions of one layer.  The
// raw rows [i0 - 16, i0 + PT + 16) are staged in shared memory; every thread
// owns channels c = tid, tid + 256, ... and slides the window sums of its
// channels along the tile; per position the 9 dot products (3 windows x
// {||d-||^2, ||d+||^2, d-.d+}, up to 4 windows) are reduced per warp into shared memory and
// combined across warps once per tile.
// ---------------------------------------------------------------------------
constexpr int kHalo = 16;

template <typename Tin>
__global__ void __launch_bounds__(256) seg_curv_kernel(const Tin *V, const float *hidden,
                                                       SegArgs a, const float *inv_norm,
                                                       int PT, double *klw) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int li = blockIdx.y;
    const int l = a.layers[li];
    const int i0 = blockIdx.x * PT;
    const int rows = PT + 2 * kHalo;
    const int row0 = i0 - kHalo;
    float *inv_s = reinterpret_cast<float *>(smem_raw);                       // [rows]
    float *red = inv_s + rows;                                                // [PT][8][12]
    Tin *hraw = reinterpret_cast<Tin *>(red + (size_t)PT * 8 * 12);           // [rows][D]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int r = tid; r < rows; r += 256) {
        int t = row0 + r;
        inv_s[r] = (t >= 0 && t < a.T) ? inv_norm[(size_t)li * a.T + t] : 0.f;
    }
    for (size_t e = tid; e < (size_t)rows * a.D; e += 256) {
        int r = (int)(e / a.D), c = (int)(e - (size_t)r * a.D);
        int t = row0 + r;
        float x = (t >= 0 && t < a.T) ? traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, t, c) : 0.f;
        hraw[e] = (Tin)x;
    }
    __syncthreads();
    auto H = [&](int r, int c) -> float { return to_f(hraw[(size_t)r * a.D + c]) * inv_s[r]; };

    const int nw = a.nwin;
    const int npos = min(PT, a.T - i0);
    constexpr int kMaxCh = 8;                      // D <= 2048
    float SL[kMaxCh][kMaxWindows], SR[kMaxCh][kMaxWindows];
    const int nch = (a.D - tid + 255) / 256;
#pragma unroll
    for (int k = 0; k < kMaxCh; k++) {
        if (k >= nch) break;
        int c = tid + 256 * k;
#pragma unroll
        for (int wi = 0; wi < kMaxWindows; wi++) {
            float sl = 0.f, sr = 0.f;
            if (wi < nw) {
                int w = a.windows[wi];
                for (int tau = 0; tau < w; tau++) sl += H(kHalo - tau, c);
                for (int tau = 1; tau <= w; tau++) sr += H(kHalo + tau, c);
            }
            SL[k][wi] = sl;
            SR[k][wi] = sr;
        }
    }
    for (int p = 0; p < npos; p++) {
        const int rr = kHalo + p;       // row of position i0 + p
        float acc[kMaxWindows][3];
#pragma unroll
        for (int wi = 0; wi < kMaxWindows; wi++) acc[wi][0] = acc[wi][1] = acc[wi][2] = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxCh; k++) {
            if (k >= nch) break;
            int c = tid + 256 * k;
            float hi = H(rr, c);
#pragma unroll
            for (int wi = 0; wi < kMaxWindows; wi++) {
                if (wi >= nw) break;
                int w = a.windows[wi];
                if (p > 0) {   // slide from position p-1 to p
                    SL[k][wi] += hi - H(rr - w, c);
                    SR[k][wi] += H(rr + w, c) - hi;
                }
                float inv_w = 1.0f / (float)w;
                float dm = hi - SL[k][wi] * inv_w;
                float dp = SR[k][wi] * inv_w - hi;
                acc[wi][0] = fmaf(dm, dm, acc[wi][0]);
                acc[wi][1] = fmaf(dp, dp, acc[wi][1]);
                acc[wi][2] = fmaf(dm, dp, acc[wi][2]);
            }
        }
#pragma unroll
        for (int wi = 0; wi < kMaxWindows; wi++) {
            if (wi >= nw) break;
#pragma unroll
            for (int q = 0; q < 3; q++) {
                float v = warp_sum(acc[wi][q]);
                if (lane == 0) red[((size_t)p * 8 + warp) * 12 + wi * 3 + q] = v;
            }
        }
    }
    __syncthreads();
    for (int e = tid; e < npos * nw; e += 256) {
        int p = e / nw, wi = e - p * nw;
        int i = i0 + p, w = a.windows[wi];
        double nm = 0, np_ = 0, dt = 0;
        for (int q = 0; q < 8; q++) {
            const float *rp = red + ((size_t)p * 8 + q) * 12 + wi * 3;
            nm += rp[0];
            np_ += rp[1];
            dt += rp[2];
        }
        double k = 0.0;
        if (i >= w && i < a.T - w) {
            double x = sqrt(nm), y = sqrt(np_);
            k = 1.0 - dt / ((x > kEps ? x : kEps) * (y > kEps ? y : kEps));
        }
        klw[((size_t)li * nw + wi) * a.T + i] = k;
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
// Robust z: exact lower median and MAD by 8-bit radix select over the ordered
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

// Select the element of ascending rank `rank` of f(i) over i < n, where f is
// x[i] (mode 0) or |x[i] - center| (mode 1).
__device__ double block_select(const double *x, int n, int rank, int mode, double center,
                               unsigned int *hist, unsigned long long *shared_prefix,
                               int *shared_rank) {
    unsigned long long prefix = 0, mask = 0;
    int r = rank;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            double v = mode ? fabs(x[i] - center) : x[i];
            unsigned long long k = dkey(v);
            if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int acc = 0, b = 0;
            for (; b < 256; b++) {
                if (acc + (int)hist[b] > r) break;
                acc += hist[b];
            }
            *shared_prefix = prefix | ((unsigned long long)b << shift);
            *shared_rank = r - acc;
        }
        __syncthreads();
        prefix = *shared_prefix;
        r = *shared_rank;
        mask |= (255ull << shift);
        __syncthreads();
    }
    return dkey_inv(prefix);
}

// out[i] (+)= scale * (x[i] - median) / (1.4826 MAD + eps)
__global__ void __launch_bounds__(1024) seg_robust_z_kernel(const double *x, int n, double scale,
                                                            int accumulate, double *out) {
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long sp;
    __shared__ int sr;
    int rank = (n - 1) / 2;
    double med = block_select(x, n, rank, 0, 0.0, hist, &sp, &sr);
    double mad = block_select(x, n, rank, 1, med, hist, &sp, &sr);
    double den = 1.4826 * mad + kEps;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        double z = scale * ((x[i] - med) / den);
        out[i] = accumulate ? out[i] + z : z;
    }
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
        for (int c = lane; c < a.D; c += 32) {
            float x0 = traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, p0, c) * i0;
            float x1 = traj_elem(V, hidden, a.Dh, a.G, a.T, a.d, l, li, p1, c) * i1;
            float df = x1 - x0;
            f = fmaf(df, df, f);
        }
        s += (double)f;
    }
    s = warp_sum(s);
    if (lane == 0) dd[t] = s;
}

// Exclusive prefix sum of n doubles (single block, deterministic): out[0] = 0,
// out[t] = sum_{s<t} in[s], t <= n.
__global__ void __launch_bounds__(1024) seg_scan_kernel(const double *in, int n, double *out) {
    __shared__ double part[1024];
    int tid = threadIdx.x;
    int per = (n + 1023) / 1024;
    int b = tid * per, e = min(n, b + per);
    double s = 0.0;
    for (int i = b; i < e; i++) s += in[i];
    part[tid] = s;
    __syncthreads();
    if (tid == 0) {
        double acc = 0.0;
        for (int k = 0; k < 1024; k++) {
            double v = part[k];
            part[k] = acc;
            acc += v;
        }
    }
    __syncthreads();
    double acc = part[tid];
    for (int i = b; i < e; i++) {
        out[i] = acc;
        acc += in[i];
    }
    if (e == n && b < e) out[n] = acc;
    if (n == 0 && tid == 0) out[0] = 0.0;
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

constexpr int kRB = 32;
constexpr int kKC = 32;   // channel chunk

template <typename Tin>
__global__ void __launch_bounds__(256) seg_band_kernel(const Tin *V, const float *hidden, BandArgs b,
                                                       const float *inv_norm, const float *nrm2,
                                                       const double *p2, const double *bscore,
                                                       float2 *ew) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const SegArgs &a = b.s;
    const int nb = b.n_max - b.n_min + 1;
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
            ew[(size_t)i * nb + (len - b.n_min)] = make_float2(-INFINITY, 0.f);
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
        ew[(size_t)i * nb + (len - b.n_min)] = df_split(w);
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
// DP: one block of 1024 threads.  Endpoints are processed 16 (or n_min, if
// smaller) at a time: F[i..i+nb-1] only read F[< i] because i - a >= n_min.
// 64 threads per endpoint reduce its candidates (value desc, a asc).  The
// chosen slot length of every endpoint is kept in shared memory (uint8) so
// the backtracking runs without global round trips.
// ---------------------------------------------------------------------------
constexpr int kDpRing = 256;
constexpr int kDpEp = 16;
constexpr int kDpTpe = 64;

__device__ __forceinline__ bool better(df2 v, int a, df2 bv, int ba) {
    return df_gt(v, bv) || (df_eq(v, bv) && a < ba);
}

__global__ void __launch_bounds__(1024) seg_dp_kernel(const float2 *ew, const float2 *ewt, int N,
                                                      int n_min, int n_max, int cs, double *Fout,
                                                      int32_t *slots, int *dev_int) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    df2 *ring = reinterpret_cast<df2 *>(smem_raw);                       // [kDpRing]
    df2 *rv = ring + kDpRing;                                            // [32] per-warp best value
    int *ra = reinterpret_cast<int *>(rv + 32);                          // [32] per-warp best a
    uint8_t *lenarr = reinterpret_cast<uint8_t *>(ra + 32);              // [N + 1]
    const int nb = n_max - n_min + 1;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int k = tid / kDpTpe, sub = tid % kDpTpe;
    const int step = min(n_min, kDpEp);
    const df2 NEG = df2{-INFINITY, 0.f};
    if (tid == 0) {
        ring[0] = df2{0.f, 0.f};
        Fout[0] = 0.0;
        lenarr[0] = 0;
    }
    __syncthreads();
    for (int i0 = 1; i0 <= N; i0 += step) {
        int i = i0 + k;
        bool act = k < step && i <= N;
        df2 best = NEG;
        int ba = 0x7fffffff;
        if (act) {
            for (int len = n_min + sub; len <= n_max; len += kDpTpe) {
                int a = i - len;
                if (a < 0) break;
                df2 fa = ring[a % kDpRing];
                if (fa.hi == -INFINITY) continue;
                float2 w = ew[(size_t)i * nb + (len - n_min)];
                df2 v = df_add(fa, w);
                if (better(v, a, best, ba)) { best = v; ba = a; }
            }
        }
        // reduce over the 64 threads of the endpoint (2 warps)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            df2 ov;
            ov.hi = __shfl_xor_sync(0xffffffffu, best.hi, o);
            ov.lo = __shfl_xor_sync(0xffffffffu, best.lo, o);
            int oa = __shfl_xor_sync(0xffffffffu, ba, o);
            if (better(ov, oa, best, ba)) { best = ov; ba = oa; }
        }
        if (lane == 0) { rv[warp] = best; ra[warp] = ba; }
        __syncthreads();
        if (sub == 0 && act) {
            df2 v2 = rv[warp + 1];
            int a2 = ra[warp + 1];
            if (better(v2, a2, best, ba)) { best = v2; ba = a2; }
            ring[i % kDpRing] = best;
            Fout[i] = (double)best.hi + (double)best.lo;
            lenarr[i] = best.hi == -INFINITY ? 0 : (uint8_t)(i - ba);
        }
        __syncthreads();
    }
    if (tid == 0 && ring[N % kDpRing].hi == -INFINITY) {
        // terminal relaxation (Eq. app_terminal_predecessor): 1 <= N - a <= n_max,
        // read after every F[< N] has been written
        df2 best = NEG;
        int ba = 0x7fffffff;
        for (int len = 1; len <= n_max; len++) {
            int a = N - len;
            if (a < 0) break;
            df2 fa = ring[a % kDpRing];
            if (fa.hi == -INFINITY || ewt[len].x == -INFINITY) continue;
            df2 v = df_add(fa, ewt[len]);
            if (better(v, a, best, ba)) { best = v; ba = a; }
        }
        Fout[N] = (double)best.hi + (double)best.lo;
        lenarr[N] = best.hi == -INFINITY ? 0 : (uint8_t)(N - ba);
    }
    if (tid == 0) {
        int J = 0, ok = 1;
        for (int i = N; i > 0;) {
            int len = lenarr[i];
            if (len == 0) { ok = 0; break; }
            i -= len;
            J++;
        }
        if (!ok) {
            dev_int[0] = -1;
            return;
        }
        dev_int[0] = J;
        slots[J] = cs + N;
        int j = J;
        for (int i = N; i > 0;) {
            i -= lenarr[i];
            slots[--j] = cs + i;
        }
    }
}

}  // namespace

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

    // curvature tile: staged raw rows (input element type, fp32 for hidden
    // states) + inverse norms + per-warp reductions
    const bool stage_bf = bf && !hidden;
    const size_t esz = stage_bf ? 2 : 4;
    const size_t budget = 224 * 1024;
    int PT = 64;
    auto cur_smem = [&](int pt) {
        return (size_t)(pt + 2 * kHalo) * 4 + (size_t)pt * 8 * 12 * 4 + (size_t)(pt + 2 * kHalo) * a.D * esz;
    };
    while (PT > 8 && cur_smem(PT) > budget) PT /= 2;
    if (cur_smem(PT) > budget) return cudaErrorInvalidConfiguration;
    size_t sm = cur_smem(PT);
    dim3 gc((p.T + PT - 1) / PT, c.nseg);
    if (stage_bf) {
        cudaFuncSetAttribute(seg_curv_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        seg_curv_kernel<<<gc, 256, sm, s>>>(Vb, hidden, a, w.inv_norm, PT, w.klw);
    } else {
        cudaFuncSetAttribute(seg_curv_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        seg_curv_kernel<<<gc, 256, sm, s>>>(bf ? nullptr : Vf, hidden, a, w.inv_norm, PT, w.klw);
    }
    seg_combine_kernel<<<(p.T + 255) / 256, 256, 0, s>>>(w.klw, c.nseg * c.nwin, p.T, p.lambda_stab,
                                                          w.kappa, kappa_out, w.dev_int + 1);
    // boundary score b = z(kappa) + lambda_s z(surprisal)
    seg_robust_z_kernel<<<1, 1024, 0, s>>>(w.kappa, p.T, 1.0, 0, w.bscore);
    if (surprisal) {
        f32_to_f64_kernel<<<(p.T + 255) / 256, 256, 0, s>>>(surprisal, p.T, w.zbuf);
        seg_robust_z_kernel<<<1, 1024, 0, s>>>(w.zbuf, p.T, p.lambda_s, 1, w.bscore);
    }
    // prefix of sum_l ||d_t||^2 over the compressible region
    int N = c.Nc;
    if (N > 1) {
        int nw8 = (N - 1 + 7) / 8;
        if (bf) seg_dd_kernel<<<nw8, 256, 0, s>>>(Vb, hidden, a, w.inv_norm, w.zbuf);
        else seg_dd_kernel<<<nw8, 256, 0, s>>>(Vf, hidden, a, w.inv_norm, w.zbuf);
    }
    seg_scan_kernel<<<1, 1024, 0, s>>>(w.zbuf, N > 1 ? N - 1 : 0, w.p2);
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
    if (bf) {
        seg_band_kernel<<<gb, 256, smb, s>>>(Vb, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ew);
        seg_band_terminal_kernel<<<(p.n_max + 7) / 8, 256, 0, s>>>(Vb, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ewt);
    } else {
        seg_band_kernel<<<gb, 256, smb, s>>>(Vf, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ew);
        seg_band_terminal_kernel<<<(p.n_max + 7) / 8, 256, 0, s>>>(Vf, hidden, b, w.inv_norm, w.nrm2, w.p2, w.bscore, w.ewt);
    }
    size_t smd = kDpRing * sizeof(df2) + 32 * sizeof(df2) + 32 * 4 + (size_t)(N + 1);
    smd = (smd + 15) & ~(size_t)15;
    if (smd > 227 * 1024) return cudaErrorInvalidConfiguration;
    cudaFuncSetAttribute(seg_dp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smd);
    seg_dp_kernel<<<1, 1024, smd, s>>>(w.ew, w.ewt, N, p.n_min, p.n_max, p.ctx_start, w.dpF,
                                       w.slots, w.dev_int);
    c.launches += 8 + (surprisal ? 2 : 0) + (N > 1 ? 1 : 0);
    return cudaGetLastError();
}

}  // namespace gkv
