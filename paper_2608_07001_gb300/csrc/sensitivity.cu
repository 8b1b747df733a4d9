// sensitivity.cu -- layer-KV-head sensitivity omega (App. A.4, Eqs.
// app_head_sensitivity_raw and app_head_sensitivity):
//
//   static_{l,g} = ( sum_{h in H(g)} ||W_O^{l,h}||_F^2 )^{1/2}
//   input_{l,g}  = Mean_u || sum_{h in H(g)} W_O^{l,h} o_u^{l,h} ||_2
//   omega_{l,g}  = sqrt(static input) / (Mean sqrt(static input) + eps)
//
// W_O [L][D][Hq d] is each layer's output projection (column block h is the
// head's D x d block) and o [L][Hq][U][d] the heads' attention outputs at the
// U question probes.  sum_{h in H(g)} W_O^{l,h} o_u^{l,h} is one product of
// the group's D x (gq d) column block with the concatenated outputs, so one
// CTA computes a 128-row tile of Y = W_g X_g (X_g: gq d x U) on the tensor
// cores (mma.sync m16n8k16, bf16 operands -- exact products -- and fp32
// sums), squares it and sums over its rows per probe, and accumulates the
// squared Frobenius norm of the W_g tile it loaded; both go to a small fp32
// scratch with atomics.  A last one-CTA kernel forms the norms, means and the
// normalisation.  The pass reads W_O once: HBM-bound.
#include "gkv_internal.cuh"

namespace gkv {
namespace {

constexpr int kSeRows = 128;       // W_O rows (output features) per CTA
constexpr int kSeK = 64;           // K (head channels) per smem chunk
constexpr int kSePad = 8;          // row padding: ldmatrix / fragment reads hit distinct banks
constexpr int kSeMaxU = 64;

__device__ __forceinline__ void se_ldsm_x4(uint32_t addr, uint32_t a[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
                 : "r"(addr));
}

// Two stages: the copies of chunk k + 1 fly while chunk k is multiplied.
template <int NT8>
struct SeSmem {
    __nv_bfloat16 Ws[2][kSeRows][kSeK + kSePad];
    __nv_bfloat16 Xs[2][NT8 * 8][kSeK + kSePad];
    float red[8][NT8 * 8];
    float fred[8];
};

// grid (D / 128, G, L), 256 threads: warp w owns rows 16 w .. 16 w + 15 of the tile.
template <int NT8>
__global__ void __launch_bounds__(256) sens_tile_kernel(const __nv_bfloat16 *__restrict__ W,
                                                        const __nv_bfloat16 *__restrict__ o, int G, int Hq,
                                                        int d, int D, int U, float *sumsq, float *fro) {
    extern __shared__ __align__(16) unsigned char se_raw[];
    SeSmem<NT8> &sm = *reinterpret_cast<SeSmem<NT8> *>(se_raw);
    auto &Ws = sm.Ws;
    auto &Xs = sm.Xs;
    auto &red = sm.red;
    auto &fred = sm.fred;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int r0 = blockIdx.x * kSeRows, g = blockIdx.y, l = blockIdx.z;
    const int gq = Hq / G, Kg = gq * d;
    const size_t row = (size_t)Hq * d;
    const __nv_bfloat16 *Wl = W + (size_t)l * D * row + (size_t)g * Kg;   // the group's column block
    float acc[NT8][4];
#pragma unroll
    for (int n = 0; n < NT8; n++) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
    float fsq = 0.f;
    const int hq = lane >> 2, tq = lane & 3, mi = lane >> 3, ri = lane & 7;
    auto issue = [&](int k0, int st) {
        for (int e = tid; e < kSeRows * kSeK / 8; e += 256) {      // W tile [128][64]
            const int r = e / (kSeK / 8), c = e % (kSeK / 8);
            const bool in = r0 + r < D;
            cp_async16(&Ws[st][r][8 * c], in ? Wl + (size_t)(r0 + r) * row + k0 + 8 * c : Wl, in);
        }
        const int hh = k0 / d, i0 = k0 % d;                         // inside one head (d >= 64)
        for (int e = tid; e < NT8 * 8 * kSeK / 8; e += 256) {      // X chunk [probes][64]
            const int u = e / (kSeK / 8), c = e % (kSeK / 8);
            const bool in = u < U;
            cp_async16(&Xs[st][u][8 * c],
                       in ? o + (((size_t)l * Hq + g * gq + hh) * U + u) * d + i0 + 8 * c : o, in);
        }
        cp_async_commit();
    };
    issue(0, 0);
    for (int k0 = 0, st = 0; k0 < Kg; k0 += kSeK, st ^= 1) {
        if (k0 + kSeK < Kg) {
            issue(k0 + kSeK, st ^ 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        // squares of the W values this thread copied, for the Frobenius norm
        for (int e = tid; e < kSeRows * kSeK / 8; e += 256) {
            const int r = e / (kSeK / 8), c = e % (kSeK / 8);
            const uint4 v = *reinterpret_cast<const uint4 *>(&Ws[st][r][8 * c]);
            const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int q = 0; q < 4; q++) {
                const float lo = __uint_as_float(w4[q] << 16), hi = __uint_as_float(w4[q] & 0xffff0000u);
                fsq = fmaf(lo, lo, fsq);
                fsq = fmaf(hi, hi, fsq);
            }
        }
#pragma unroll
        for (int ks = 0; ks < kSeK / 16; ks++) {
            uint32_t a[4];
            se_ldsm_x4(static_cast<uint32_t>(__cvta_generic_to_shared(
                           &Ws[st][warp * 16 + ri + (mi & 1) * 8][ks * 16 + (mi >> 1) * 8])),
                       a);
#pragma unroll
            for (int n = 0; n < NT8; n++) {
                const uint32_t b0 = *reinterpret_cast<const uint32_t *>(&Xs[st][n * 8 + hq][ks * 16 + 2 * tq]);
                const uint32_t b1 = *reinterpret_cast<const uint32_t *>(&Xs[st][n * 8 + hq][ks * 16 + 8 + 2 * tq]);
                mma_bf16(acc[n], a, b0, b1);
            }
        }
        __syncthreads();    // the stage is refilled by the next issue
    }
    // squared 2-norm pieces per probe: rows hq and hq + 8 of the warp's 16
#pragma unroll
    for (int n = 0; n < NT8; n++) {
        float s0 = acc[n][0] * acc[n][0] + acc[n][2] * acc[n][2];   // probe 8 n + 2 tq
        float s1 = acc[n][1] * acc[n][1] + acc[n][3] * acc[n][3];   // probe 8 n + 2 tq + 1
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            s0 += __shfl_xor_sync(0xffffffffu, s0, off);
            s1 += __shfl_xor_sync(0xffffffffu, s1, off);
        }
        if (hq == 0) {
            red[warp][n * 8 + 2 * tq] = s0;
            red[warp][n * 8 + 2 * tq + 1] = s1;
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) fsq += __shfl_xor_sync(0xffffffffu, fsq, off);
    if (lane == 0) fred[warp] = fsq;
    __syncthreads();
    float *ss = sumsq + ((size_t)l * G + g) * kSeMaxU;
    for (int u = tid; u < U; u += 256) {
        float v = 0.f;
#pragma unroll
        for (int w = 0; w < 8; w++) v += red[w][u];
        atomicAdd(ss + u, v);
    }
    if (tid == 0) {
        float v = 0.f;
#pragma unroll
        for (int w = 0; w < 8; w++) v += fred[w];
        atomicAdd(fro + (size_t)l * G + g, v);
    }
}

// One CTA: norms, means over the probes, raw values, their mean, omega.
__global__ void __launch_bounds__(1024) sens_final_kernel(const float *sumsq, const float *fro, int LG, int U,
                                                          float eps, float *omega) {
    __shared__ float wsum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    float part = 0.f;
    for (int k = tid; k < LG; k += 1024) {
        float in = 0.f;
        for (int u = 0; u < U; u++) in += sqrtf(sumsq[(size_t)k * kSeMaxU + u]);
        in /= U;
        const float raw = sqrtf(sqrtf(fro[k]) * in);
        omega[k] = raw;
        part += raw;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
    if (lane == 0) wsum[warp] = part;
    __syncthreads();
    if (tid == 0) {
        float s = 0.f;
        for (int w = 0; w < 32; w++) s += wsum[w];
        wsum[0] = s / LG;
    }
    __syncthreads();
    const float mean = wsum[0];
    for (int k = tid; k < LG; k += 1024) omega[k] = omega[k] / (mean + eps);
}

template <int NT8>
cudaError_t launch_sens_tile(dim3 grid, cudaStream_t s, const __nv_bfloat16 *W, const __nv_bfloat16 *o, int G,
                             int Hq, int d, int D, int U, float *sumsq, float *fro) {
    constexpr size_t smem = sizeof(SeSmem<NT8>);
    static bool attr = false;     // the opt-in above 48 KB, once per instantiation
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(sens_tile_kernel<NT8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    sens_tile_kernel<NT8><<<grid, 256, smem, s>>>(W, o, G, Hq, d, D, U, sumsq, fro);
    return cudaGetLastError();
}

}  // namespace
}  // namespace gkv

extern "C" gkv_status gracekv_head_sensitivity(const void *W_O, const void *o, int32_t L, int32_t G, int32_t Hq,
                                               int32_t d, int32_t D, int32_t U, int32_t dtype, float *omega,
                                               float *scratch, void *stream) {
    if (!W_O || !o || !omega || !scratch) return GKV_EINVAL;
    if ((reinterpret_cast<uintptr_t>(W_O) & 15u) || (reinterpret_cast<uintptr_t>(o) & 15u) ||
        (reinterpret_cast<uintptr_t>(omega) & 3u) || (reinterpret_cast<uintptr_t>(scratch) & 3u))
        return GKV_EINVAL;
    if (L <= 0 || G <= 0 || Hq <= 0 || Hq % G || D <= 0 || U <= 0) return GKV_EINVAL;
    if (dtype != GKV_BF16 || (d != 64 && d != 128) || U > gkv::kSeMaxU || D % 8) return GKV_EUNSUPPORTED;
    const int LG = L * G;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float *sumsq = scratch, *fro = scratch + (size_t)LG * gkv::kSeMaxU;
    if (cudaMemsetAsync(scratch, 0, sizeof(float) * (size_t)LG * (gkv::kSeMaxU + 1), s) != cudaSuccess)
        return GKV_ECUDA;
    const dim3 grid((D + gkv::kSeRows - 1) / gkv::kSeRows, G, L);
    const auto *Wb = static_cast<const __nv_bfloat16 *>(W_O);
    const auto *ob = static_cast<const __nv_bfloat16 *>(o);
    cudaError_t e;
    if (U <= 16)
        e = gkv::launch_sens_tile<2>(grid, s, Wb, ob, G, Hq, d, D, U, sumsq, fro);
    else if (U <= 32)
        e = gkv::launch_sens_tile<4>(grid, s, Wb, ob, G, Hq, d, D, U, sumsq, fro);
    else
        e = gkv::launch_sens_tile<8>(grid, s, Wb, ob, G, Hq, d, D, U, sumsq, fro);
    if (e != cudaSuccess) return GKV_ECUDA;
    gkv::sens_final_kernel<<<1, 1024, 0, s>>>(sumsq, fro, LG, U, 1e-6f, omega);
    return cudaGetLastError() == cudaSuccess ? GKV_OK : GKV_ECUDA;
}
