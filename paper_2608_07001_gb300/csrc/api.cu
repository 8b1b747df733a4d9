// api.cu -- the C ABI of include/gracekv.h: parameter validation, budget
// resolution (App. A.1), workspace ownership and the stage state machine.
#include "gkv_internal.cuh"

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

using gkv::Ctx;

struct gracekv_ctx {
    Ctx c;
    std::vector<void *> allocs;
};

namespace {

// Device status bits (dev_int[1]).
enum : int { ST_NONFINITE_KAPPA = 1, ST_NONFINITE_ROWS = 2, ST_LONG_SLOT = 4, ST_NONFINITE_GAIN = 8,
             ST_BAD_SLOTS = 16, ST_PIPE_TIMEOUT = gkv::kStPipeTimeout, ST_LONG_CAP = gkv::kStLongCap };

gkv_status fail(gracekv_ctx *x, gkv_status s, const char *msg) {
    if (x) {
        if (x->c.err.empty()) x->c.err = msg;
        if (s == GKV_ECUDA) x->c.sticky = GKV_ECUDA;
    }
    return s;
}

gkv_status cuda_fail(gracekv_ctx *x, cudaError_t e, const char *where) {
    char buf[256];
    snprintf(buf, sizeof buf, "%s: %s", where, cudaGetErrorString(e));
    if (x && x->c.err.empty()) x->c.err = buf;
    if (x) x->c.sticky = GKV_ECUDA;
    return GKV_ECUDA;
}

template <typename T>
bool dalloc(gracekv_ctx *x, T **p, size_t n) {
    void *q = nullptr;
    if (n == 0) n = 1;
    if (cudaMalloc(&q, n * sizeof(T)) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    x->allocs.push_back(q);
    *p = static_cast<T *>(q);
    return true;
}

gkv_status check_status(gracekv_ctx *x, int st) {
    if (st & ST_PIPE_TIMEOUT) return fail(x, GKV_ECUDA, "a tensor-core pipeline wait timed out");
    if (st & ST_BAD_SLOTS) return fail(x, GKV_EINVAL, "supplied slot starts are not a partition of [c_s, c_e - r) into non-empty slots");
    if (st & ST_LONG_SLOT) return fail(x, GKV_EUNSUPPORTED, "a slot is longer than 16384 tokens");
    if (st & ST_LONG_CAP) return fail(x, GKV_ENOMEM, "long-unit work items exceeded their capacity");
    if (st & ST_NONFINITE_KAPPA) return fail(x, GKV_ENONFINITE, "non-finite curvature (NaN/Inf in the trajectory)");
    if (st & ST_NONFINITE_ROWS) return fail(x, GKV_ENONFINITE, "non-finite attention row statistics (NaN/Inf in K or Q)");
    if (st & ST_NONFINITE_GAIN) return fail(x, GKV_ENONFINITE, "non-finite gain (NaN/Inf in K, V, Q or omega)");
    return GKV_OK;
}

gkv_status ready(gracekv_ctx *x, int need_stage) {
    if (!x) return GKV_EINVAL;
    if (x->c.sticky != GKV_OK) return GKV_ESTATE;
    if (x->c.stage < need_stage) return fail(x, GKV_ESTATE, "call out of order");
    return GKV_OK;
}

__global__ void validate_slots_kernel(const int32_t *s, int J, int cs, int cend, int *status) {
    int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= J) return;
    int a = s[j], b = s[j + 1];
    bool bad = b - a < 1 || (j == 0 && a != cs) || (j == J - 1 && b != cend);
    if (bad) atomicOr(status, ST_BAD_SLOTS);
    else if (b - a > gkv::kMaxSlot) atomicOr(status, ST_LONG_SLOT);
}

}  // namespace

extern "C" {

gkv_status gracekv_default_params(gkv_params *p) {
    if (!p) return GKV_EINVAL;
    memset(p, 0, sizeof *p);
    p->dtype = GKV_BF16;
    p->recent = 32;                                    // App. A.1
    p->n_min = 16; p->n_max = 128; p->n0 = 64;         // App. B.3
    p->lambda_stab = 0.25; p->lambda_s = 0.15;         // App. B.2
    p->lambda_d = 0.25; p->lambda_n = 0.10; p->c_cut = 1.0;
    p->n_seg_layers = 0;                               // depths 0.33 / 0.50 / 0.67
    p->windows[0] = 4; p->windows[1] = 8; p->windows[2] = 16; p->n_windows = 3;
    p->k_cand = 16; p->lambda_kappa = 0.05;            // App. A.3, B.4
    p->lambda_Z = 0.25; p->lambda_M = 0.75;
    p->eps = 1e-6; p->base_frac = 0.1;
    p->lambda_graph = 0.0; p->alpha_floor = 0.0;
    p->floor_c = 0.5; p->floor_gamma = 1.2; p->floor_eta = 0.95; p->floor_half = 3;   // App. A.5 Stage I
    p->eta_seed = 0.9; p->rho_hop = 0.5; p->m_seed = 64; p->r_hop = 2;               // App. A.4
    p->ctx_start = 0; p->ctx_end = -1;                 // -1: T
    p->dp_warmup = 0;                                  // 512 tokens
    return GKV_OK;
}

int64_t gracekv_budget_for_ratio(int32_t L, int32_t G, int32_t n_ctx, double x) {
    if (L <= 0 || G <= 0 || n_ctx <= 0 || !(x >= 1.0)) return -1;
    double n = (double)L * G * n_ctx;
    if (x == std::floor(x) && x < 9.0e15) return (int64_t)L * G * n_ctx / (int64_t)x;
    return (int64_t)std::floor(n / x);
}

int32_t gracekv_graph_layers(int32_t L, int32_t *out) {
    if (L <= 0) return -1;
    int32_t gl[2];
    int32_t n = 0;
    for (double rho : {0.50, 0.75}) {   // relative depths of the graph layers (App. A.1)
        int32_t l = std::min((int32_t)std::floor(rho * L), L - 1);
        if (n == 0 || gl[n - 1] != l) gl[n++] = l;
    }
    if (out)
        for (int32_t k = 0; k < n; k++) out[k] = gl[k];
    return n;
}

const char *gracekv_status_string(gkv_status s) {
    switch (s) {
        case GKV_OK: return "ok";
        case GKV_EINVAL: return "invalid argument";
        case GKV_EBUDGET: return "budget too small";
        case GKV_ENOMEM: return "out of device memory";
        case GKV_ECUDA: return "CUDA error";
        case GKV_ETIMEOUT: return "device wait timed out";
        case GKV_ENONFINITE: return "non-finite value";
        case GKV_ESTATE: return "call out of order or context failed";
        case GKV_EUNSUPPORTED: return "unsupported configuration";
        case GKV_ECAPACITY: return "output capacity too small";
    }
    return "unknown status";
}

const char *gracekv_last_error(const gracekv_ctx *x) {
    if (!x) return "null context";
    return x->c.err.c_str();
}

void gracekv_destroy(gracekv_ctx *x) {
    if (!x) return;
    for (cudaEvent_t e : x->c.ev_pool) cudaEventDestroy(e);
    if (x->c.score_ev) cudaEventDestroy(x->c.score_ev);
    if (x->c.dp_ev) cudaEventDestroy(x->c.dp_ev);
    for (cudaEvent_t e : x->c.copy_ev) cudaEventDestroy(e);
    if (x->c.copy_stream) cudaStreamDestroy(x->c.copy_stream);
    for (void *p : x->allocs) cudaFree(p);
    delete x;
}

gkv_status gracekv_create(const gkv_params *pin, gracekv_ctx **out) {
    if (!pin || !out) return GKV_EINVAL;
    *out = nullptr;
    gkv_params p = *pin;
    if (p.ctx_end < 0) p.ctx_end = p.T;
    if (p.L <= 0 || p.G <= 0 || p.Hq <= 0 || p.T <= 0 || p.d <= 0 || p.W <= 0 || p.Hq % p.G)
        return GKV_EINVAL;
    if (p.dtype != GKV_F32 && p.dtype != GKV_BF16) return GKV_EINVAL;
    if (p.ctx_start < 0 || p.ctx_end > p.T || p.ctx_start >= p.ctx_end) return GKV_EINVAL;
    if (p.n_min < 1 || p.n_max < p.n_min || p.n0 < 1) return GKV_EINVAL;
    if (p.n_windows < 1 || p.n_windows > gkv::kMaxWindows) return GKV_EINVAL;
    for (int i = 0; i < p.n_windows; i++)
        if (p.windows[i] < 1 || p.windows[i] > 16) return GKV_EINVAL;
    if (p.n_seg_layers < 0 || p.n_seg_layers > gkv::kMaxSegLayers) return GKV_EINVAL;
    for (int i = 0; i < p.n_seg_layers; i++)
        if (p.seg_layers[i] < 0 || p.seg_layers[i] >= p.L) return GKV_EINVAL;
    if (p.k_cand < 0 || p.k_cand > 16) return GKV_EINVAL;
    if ((p.seg_mode != 0 && p.seg_mode != 1) || (p.quota_alloc != 0 && p.quota_alloc != 1)) return GKV_EINVAL;
    if (!(p.eps > 0) || !(p.base_frac >= 0)) return GKV_EINVAL;
    if (!(p.lambda_graph >= 0.0 && p.lambda_graph <= 1.0)) return GKV_EINVAL;
    if (p.lambda_graph > 0.0) {
        if (!(p.eta_seed > 0.0 && p.eta_seed <= 1.0) || p.m_seed < 1 || p.m_seed > 64 || p.r_hop < 1 ||
            p.r_hop > 8 || !(p.rho_hop >= 0.0))
            return GKV_EINVAL;
        if (p.dtype != GKV_BF16 || (p.d != 64 && p.d != 128)) return GKV_EUNSUPPORTED;
    }
    if (!(p.alpha_floor >= 0.0 && p.alpha_floor <= 1.0)) return GKV_EINVAL;
    if (p.alpha_floor > 0.0) {
        if (!(p.floor_c >= 0.0 && p.floor_c <= 1.0) || !(p.floor_gamma >= 0.0) ||
            !(p.floor_eta >= 0.0 && p.floor_eta <= 1.0) || p.floor_half < 0 || p.floor_half > 64)
            return GKV_EINVAL;
        if (p.quota_alloc) return GKV_EUNSUPPORTED;
    }
    if ((p.d != 64 && p.d != 128) || p.W > 64 || p.n_max > gkv::kMaxUnit ||
        (int64_t)p.G * p.d > 2048)
        return GKV_EUNSUPPORTED;
    // recent window (App. A.1): r = 32, shrunk to floor(B / (L G)) when it does
    // not fit, never below 4; the compressible region must stay non-empty.
    int64_t LG = (int64_t)p.L * p.G;
    int64_t r = p.recent;
    if (r < 0) return GKV_EINVAL;
    if (LG * r > p.budget) {
        r = p.budget / LG;
        if (r < 4) return GKV_EBUDGET;
    }
    int64_t Nc = (int64_t)p.ctx_end - r - p.ctx_start;
    if (Nc < 1) return GKV_EBUDGET;
    if (gkv::dp_smem_bytes(p, (int)std::min<int64_t>(Nc, 1 << 30)) > 227 * 1024 - 64)
        return GKV_EUNSUPPORTED;   // the DP's finish kernel keeps one exit table per chunk in shared memory
    if (p.lambda_graph > 0.0 && Nc > gkv::multihop_max_context()) return GKV_EUNSUPPORTED;

    gracekv_ctx *x = new (std::nothrow) gracekv_ctx();
    if (!x) return GKV_ENOMEM;
    Ctx &c = x->c;
    c.p = p;
    c.r = (int32_t)r;
    c.Nc = (int32_t)Nc;
    c.c_end = p.ctx_end - c.r;
    c.B_free = p.budget - LG * r;
    c.nwin = p.n_windows;
    if (p.n_seg_layers > 0) {
        c.nseg = p.n_seg_layers;
        for (int i = 0; i < c.nseg; i++) c.seg_layers[i] = p.seg_layers[i];
    } else {   // App. B.2 Eq. app_seg_layers
        const double rho[3] = {0.33, 0.50, 0.67};
        c.nseg = 0;
        for (double q : rho) {
            int l = (int)std::floor(q * p.L);
            if (l > p.L - 1) l = p.L - 1;
            bool dup = false;
            for (int i = 0; i < c.nseg; i++) dup |= c.seg_layers[i] == l;
            if (!dup) c.seg_layers[c.nseg++] = l;
        }
    }
    if (cudaGetDevice(&c.device) != cudaSuccess) {
        delete x;
        return GKV_ECUDA;
    }
    cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, c.device);
    const int Rg = (p.Hq / p.G) * p.W;
    const int64_t base = LG * ((Rg + 63) / 64);
    c.n_chunks = (int)std::max<int64_t>(1, std::min<int64_t>((4 * c.num_sms + base - 1) / base,
                                                             std::max(1, p.T / 256)));
    if (gkv::use_tc(c)) c.n_chunks = std::max(c.n_chunks, gkv::tc_row_chunks(c));
    c.node_cap = LG * 2 * Nc;
    if (c.node_cap >= (1LL << 31)) {   // node records are addressed with int32
        delete x;
        return GKV_EINVAL;
    }
    const int nb = p.n_max - p.n_min + 1;
    const int64_t nrow = (int64_t)p.L * p.Hq * p.W;
    int dp_S, dp_Wu, dp_nch;
    gkv::dp_chunking(p, (int)Nc, &dp_S, &dp_Wu, &dp_nch);
    gkv::Workspace &w = c.w;
    bool ok = dalloc(x, &w.rope, (size_t)p.T * (p.d / 2)) &&
              dalloc(x, &w.rope_rel, (size_t)(2 * gkv::kMaxSlot - 1) * (p.d / 2)) &&
              dalloc(x, &w.long_slots, (size_t)Nc + 2) && dalloc(x, &w.long_n, 4) &&
              dalloc(x, &w.ent, (size_t)p.budget + (size_t)p.L * p.G * (p.T - Nc)) &&
              dalloc(x, &w.inv_norm, (size_t)c.nseg * p.T) &&
              dalloc(x, &w.nrm2, (size_t)c.nseg * p.T) &&
              dalloc(x, &w.klw, (size_t)c.nseg * c.nwin * p.T) &&
              dalloc(x, &w.kappa, (size_t)p.T) && dalloc(x, &w.bscore, (size_t)p.T) &&
              dalloc(x, &w.zbuf, (size_t)p.T) && dalloc(x, &w.zdev, (size_t)p.T) &&
              dalloc(x, &w.sel_state, 4) && dalloc(x, &w.sel_hist, 2048) && dalloc(x, &w.p2, (size_t)Nc + 1) &&
              dalloc(x, &w.ew, (size_t)(Nc + 1) * ((nb + 3) & ~3)) && dalloc(x, &w.ewt, (size_t)p.n_max + 1) &&
              dalloc(x, &w.slots, (size_t)Nc + 2) && dalloc(x, &w.dp_len, (size_t)Nc + 16) &&
              dalloc(x, &w.dp_head, (size_t)dp_nch * 128) && dalloc(x, &w.dp_tail, (size_t)dp_nch * 256) &&
              dalloc(x, &w.dp_tab, (size_t)dp_nch * p.n_max) &&
              dalloc(x, &w.dev_int, 16) &&
              dalloc(x, &w.row_m, (size_t)nrow) && dalloc(x, &w.row_Z, (size_t)nrow) &&
              dalloc(x, &w.row_ZC, (size_t)nrow) && dalloc(x, &w.rowp, (size_t)3 * nrow * c.n_chunks) &&
              dalloc(x, &w.row_mneg, (size_t)nrow) && dalloc(x, &w.lg_scale, (size_t)LG) &&
              dalloc(x, &w.rtok, (size_t)LG * Nc) &&
              dalloc(x, &w.nd_a, (size_t)c.node_cap) && dalloc(x, &w.nd_b, (size_t)c.node_cap) &&
              dalloc(x, &w.nd_child0, (size_t)c.node_cap) && dalloc(x, &w.nd_parent, (size_t)c.node_cap) &&
              dalloc(x, &w.nd_unit, (size_t)c.node_cap) && dalloc(x, &w.nd_nchild, (size_t)c.node_cap) &&
              dalloc(x, &w.nd_cost, (size_t)c.node_cap) && dalloc(x, &w.nd_D, (size_t)c.node_cap) &&
              dalloc(x, &w.nd_R, (size_t)c.node_cap) && dalloc(x, &w.nd_U, (size_t)c.node_cap) &&
              dalloc(x, &w.nd_kappa, (size_t)c.node_cap) && dalloc(x, &w.nd_sel, (size_t)c.node_cap) &&
              dalloc(x, &w.ops, (size_t)c.node_cap / 2 + 1) && dalloc(x, &w.n_ops, 1) &&
              (!gkv::use_tc(c) || (dalloc(x, &w.Eg, (size_t)LG * Nc * 64) && dalloc(x, &w.qperm, (size_t)256))) &&
              (p.alpha_floor <= 0.0 || (dalloc(x, &w.fl_rbar, (size_t)Nc) && dalloc(x, &w.fl_f, (size_t)LG * Nc) &&
                                          dalloc(x, &w.fl_acc, (size_t)LG * Nc) &&
                                          dalloc(x, &w.fl_head, (size_t)LG * gkv::floor_head_words()) &&
                                          dalloc(x, &w.fl_glob, (size_t)4))) &&
              (p.lambda_graph <= 0.0 ||
               (dalloc(x, &w.mh_sc, (size_t)Nc) && dalloc(x, &w.mh_acc, (size_t)Nc) &&
                dalloc(x, &w.mh_dpart, (size_t)2 * p.Hq * Nc) &&
                dalloc(x, &w.mh_stat, (size_t)2 * p.Hq * gkv::multihop_chunks(p.T) * 64 * 2) &&
                dalloc(x, &w.mh_rowmz, (size_t)2 * p.Hq * 64 * 2) && dalloc(x, &w.mh_was, (size_t)Nc) &&
                dalloc(x, &w.mh_seeds, (size_t)64) && dalloc(x, &w.mh_nseed, (size_t)1) &&
                dalloc(x, &w.mh_graph_l, (size_t)2) && dalloc(x, &w.mh_w, (size_t)64) &&
                dalloc(x, &w.mh_red, (size_t)2) && dalloc(x, &w.mh_pkeys, (size_t)64 * 64) &&
                dalloc(x, &w.mh_psum, (size_t)64))) &&
              dalloc(x, &w.hist, (size_t)2048 * (p.quota_alloc ? LG : 1)) &&
              dalloc(x, &w.alloc_state, (size_t)16 * (p.quota_alloc ? (size_t)LG + 1 : 1)) && dalloc(x, &w.work, 4) &&
              dalloc(x, &w.pend_hist, 1 << 16) && dalloc(x, &w.pend_cut, 1) && dalloc(x, &w.pend_n, 1) &&
              dalloc(x, &w.pend_pot, 1);
    if (!ok) {
        gracekv_destroy(x);
        return GKV_ENOMEM;
    }
    cudaError_t e = cudaMemset(w.nd_cost, 0, (size_t)c.node_cap);
    if (e == cudaSuccess && w.qperm) {   // pass B's column order: probe u's row (u mod gq) W + u first
        const int gq = p.Hq / p.G;
        std::vector<short> perm;
        for (int u = 0; u < p.W; u++) perm.push_back((short)((u % gq) * p.W + u));
        for (int r = 0; r < gq * p.W; r++)
            if ((r % p.W) % gq != r / p.W) perm.push_back((short)r);
        perm.resize(256, 0);
        e = cudaMemcpy(w.qperm, perm.data(), 256 * sizeof(short), cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = cudaMemset(w.dev_int, 0, 16 * sizeof(int));
    if (e == cudaSuccess && w.mh_graph_l) {
        int32_t gl[2];
        int n = gracekv_graph_layers(p.L, gl);
        c.mh_ngraph = n;
        e = cudaMemcpy(w.mh_graph_l, gl, n * sizeof(int32_t), cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = gkv::launch_rope_table(c, 0);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        gracekv_destroy(x);
        return GKV_ECUDA;
    }
    *out = x;
    return GKV_OK;
}

gkv_status gracekv_query(const gracekv_ctx *x, int32_t *recent, int32_t *n_c, int64_t *b_free,
                         int32_t *n_slots) {
    if (!x) return GKV_EINVAL;
    if (recent) *recent = x->c.r;
    if (n_c) *n_c = x->c.Nc;
    if (b_free) *b_free = x->c.B_free;
    if (n_slots) *n_slots = x->c.J;
    return GKV_OK;
}

// Device tensors are read and written as 16-byte vectors (8-byte for the
// float2 tables), so their base addresses must be 16-byte aligned; index and
// scalar arrays need their natural alignment.
static bool al16(const void *p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
static bool al4(const void *p) { return !p || (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }
static bool al8(const void *p) { return !p || (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

static cudaError_t launch_score(Ctx &c, const void *K, const void *Q, cudaStream_t s);

gkv_status gracekv_segment(gracekv_ctx *x, const void *V, const float *hidden, int32_t Dh,
                           const float *surprisal, int32_t *slot_starts, int32_t cap,
                           int32_t *n_slots_host, float *kappa, void *stream) {
    gkv_status st = ready(x, 0);
    if (st) return st;
    Ctx &c = x->c;
    if (!V || !slot_starts || !n_slots_host || cap < 1) return fail(x, GKV_EINVAL, "segment: null argument");
    if (!al16(V) || (hidden && !al16(hidden)) || !al4(surprisal) || !al4(slot_starts) || !al4(kappa))
        return fail(x, GKV_EINVAL, "segment: misaligned pointer (V and hidden need 16 bytes, the others 4)");
    if (hidden && (Dh <= 0 || Dh > 2048 || Dh % 8))
        return fail(x, GKV_EINVAL, "segment: hidden dim must be a multiple of 8 in [8, 2048]");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    if (c.score_pending && !c.dp_ev) e = cudaEventCreateWithFlags(&c.dp_ev, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaMemsetAsync(c.w.dev_int, 0, 16 * sizeof(int), s);
    if (e == cudaSuccess && c.score_pending) {
        // requested score passes: they read no output of the segmentation, so
        // they run beside it, on the SMs its single-block kernels leave idle
        e = cudaEventRecord(c.dp_ev, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(c.score_stream, c.dp_ev, 0);
        if (e == cudaSuccess) e = launch_score(c, c.score_K, c.score_Q, c.score_stream);
    }
    if (c.p.seg_mode == 1) {
        // "w/o CS" ablation: uniform slots of target length n0, curvature 0
        const int N = c.Nc, J = std::max(1, (N + c.p.n0 / 2) / c.p.n0);
        std::vector<int32_t> hs(J + 1);
        for (int j = 0; j <= J; j++) hs[j] = c.p.ctx_start + (int32_t)(((int64_t)j * N) / J);
        if (e == cudaSuccess) {
            gkv::StageTimer tm(c, 0, s);
            e = cudaMemcpyAsync(c.w.slots, hs.data(), (size_t)(J + 1) * sizeof(int32_t), cudaMemcpyHostToDevice, s);
            if (e == cudaSuccess) e = cudaMemsetAsync(c.w.kappa, 0, (size_t)c.p.T * sizeof(double), s);
            if (e == cudaSuccess && kappa) e = cudaMemsetAsync(kappa, 0, (size_t)c.p.T * sizeof(float), s);
            if (e == cudaSuccess) e = cudaMemcpyAsync(c.w.dev_int, &J, sizeof(int), cudaMemcpyHostToDevice, s);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s);   // hs and J leave scope
        }
    } else if (e == cudaSuccess) {
        gkv::StageTimer tm(c, 0, s);
        e = gkv::launch_segment(c, V, hidden, hidden ? Dh : 0, surprisal, kappa, s);
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "segment launch");
    int h[gkv::kDpRerun + 1];
    e = cudaMemcpyAsync(h, c.w.dev_int, sizeof h, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(x, e, "segment");
    if (c.p.seg_mode == 0) {
        int S, Wu;
        gkv::dp_chunking(c.p, c.Nc, &S, &Wu, &c.dp_chunks);
        c.dp_rerun = h[gkv::kDpRerun];
    } else {
        c.dp_chunks = c.dp_rerun = 0;
    }
    st = check_status(x, h[1]);
    if (st) return st;
    if (h[0] <= 0) return fail(x, GKV_EINVAL, "segmentation found no partition");
    *n_slots_host = h[0];
    if (h[0] > cap) return fail(x, GKV_ECAPACITY, "segment: more slots than cap");
    e = cudaMemcpyAsync(slot_starts, c.w.slots, (size_t)(h[0] + 1) * sizeof(int32_t),
                        cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(x, e, "segment copy");
    c.J = h[0];
    c.stage = 1;
    return GKV_OK;
}

// The score passes on stream s, then the event the tree build waits for.
static cudaError_t launch_score(Ctx &c, const void *K, const void *Q, cudaStream_t s) {
    c.score_pending = false;
    cudaError_t e = cudaMemsetAsync(c.w.dev_int + gkv::kScoreStatus, 0, sizeof(int), s);
    if (e == cudaSuccess) {
        gkv::StageTimer tm(c, 1, s);
        e = gkv::launch_row_stats(c, K, Q, s);
    }
    if (e == cudaSuccess) {
        gkv::StageTimer tm(c, 2, s);
        e = gkv::launch_token_values(c, K, Q, s);
    }
    if (e == cudaSuccess && !c.score_ev) e = cudaEventCreateWithFlags(&c.score_ev, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventRecord(c.score_ev, s);
    if (e == cudaSuccess) c.scored = true;
    return e;
}

gkv_status gracekv_score(gracekv_ctx *x, const void *K, const void *Q, void *stream) {
    if (!x) return GKV_EINVAL;
    if (x->c.sticky != GKV_OK) return GKV_ESTATE;
    Ctx &c = x->c;
    if (!K || !Q) return fail(x, GKV_EINVAL, "score: null tensor");
    if (!al16(K) || !al16(Q)) return fail(x, GKV_EINVAL, "score: misaligned pointer (K, Q need 16 bytes)");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    c.scored = false;
    c.score_K = K;
    c.score_Q = Q;
    c.score_stream = s;
    if (c.stage != 1) {   // the next segmentation enqueues them when it starts
        c.score_pending = true;
        return GKV_OK;
    }
    cudaError_t e = launch_score(c, K, Q, s);
    if (e != cudaSuccess) return cuda_fail(x, e, "score");
    return GKV_OK;
}

// ---- tree building, in pieces (used by gracekv_build_trees and the host pipeline)

// Supplied slots (validated) or the segmentation's; unit arrays sized for them.
static gkv_status build_setup(gracekv_ctx *x, const int32_t *slot_starts, int32_t n_slots, cudaStream_t s) {
    Ctx &c = x->c;
    cudaError_t e;
    if (slot_starts) {
        if (n_slots < 1 || n_slots > c.Nc) return fail(x, GKV_EINVAL, "build_trees: bad n_slots");
        e = cudaMemcpyAsync(c.w.slots, slot_starts, (size_t)(n_slots + 1) * sizeof(int32_t),
                            cudaMemcpyDeviceToDevice, s);
        int h = 0;
        if (e == cudaSuccess) e = cudaMemsetAsync(c.w.dev_int + 1, 0, sizeof(int), s);
        if (e == cudaSuccess) {
            validate_slots_kernel<<<(n_slots + 255) / 256, 256, 0, s>>>(c.w.slots, n_slots, c.p.ctx_start,
                                                                          c.c_end, c.w.dev_int + 1);
            c.launches += 1;
            e = cudaGetLastError();
        }
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h, c.w.dev_int + 1, sizeof(int), cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(x, e, "build_trees slots");
        gkv_status st = check_status(x, h);
        if (st) return st;
        c.J = n_slots;
    }
    const int64_t nu = (int64_t)c.p.L * c.p.G * c.J;
    gkv::Workspace &w = c.w;
    if (nu > w.units_cap) {   // grows only when a partition has more slots than any before
        int64_t cap = std::max<int64_t>(nu, w.units_cap * 2);
        bool ok = dalloc(x, &w.u_nnodes, cap) && dalloc(x, &w.u_Uadd, cap) &&
                  dalloc(x, &w.u_Ddrop, cap) && dalloc(x, &w.u_sel, cap) &&
                  dalloc(x, &w.u_count, cap) && dalloc(x, &w.u_off, cap) &&
                  dalloc(x, &w.u_pend, cap) && dalloc(x, &w.u_list, cap) &&
                  (c.p.alpha_floor <= 0.0 || dalloc(x, &w.u_floor, cap)) &&
                  dalloc(x, &w.long_list, cap) &&
                  dalloc(x, &w.u_bsum, cap / 1024 + 2) &&
                  dalloc(x, &w.tie_bsum, cap / 1024 + (int64_t)c.p.L * c.p.G + 2);
        if (!ok) return fail(x, GKV_ENOMEM, "build_trees: unit arrays");
        w.units_cap = cap;
    }
    return GKV_OK;
}

// Work counters and the op list cleared; slots split into the short and long
// classes of the unit kernel and the long units (cnt: their sizes and the
// long units' tokens; synchronises s).
static cudaError_t build_classes(Ctx &c, int cnt[4], cudaStream_t s) {
    gkv::Workspace &w = c.w;
    const int64_t nu = (int64_t)c.p.L * c.p.G * c.J;
    static const float kNoCut = -INFINITY;
    cudaError_t e = cudaSuccess;
    if (!(c.B_free < nu)) e = cudaMemcpyAsync(w.pend_cut, &kNoCut, sizeof(float), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(w.work, 0, 4 * sizeof(unsigned long long), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(w.n_ops, 0, sizeof(unsigned int), s);
    cnt[0] = cnt[1] = cnt[2] = cnt[3] = 0;
    if (e == cudaSuccess) {
        gkv::StageTimer tm(c, 3, s);
        e = gkv::launch_slot_classes(c, w.slots, c.J, w.u_list, w.dev_int + 2, w.long_slots, s);
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(cnt, w.dev_int + 2, 4 * sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return e;
}

// The classes, and the work-item arrays of the long units sized for them: a
// level's items of one unit are disjoint intervals of >= 2 tokens, so at most
// n / 2 of them (or its root).
static gkv_status classes(gracekv_ctx *x, int cnt[4], cudaStream_t s) {
    Ctx &c = x->c;
    gkv::Workspace &w = c.w;
    cudaError_t e = build_classes(c, cnt, s);
    if (e != cudaSuccess) return cuda_fail(x, e, "build_trees classes");
    c.n_long = cnt[2];
    if (cnt[2] == 0) return GKV_OK;
    const int64_t LG = (int64_t)c.p.L * c.p.G;
    const int64_t items = LG * ((int64_t)cnt[3] / 2 + cnt[2]) + 16, units = LG * cnt[2];
    if (items > w.long_cap) {
        bool ok = dalloc(x, &w.long_gv, items) && dalloc(x, &w.long_uid, items) &&
                  dalloc(x, &w.long_kin, items) && dalloc(x, &w.long_ufl, items) &&
                  dalloc(x, &w.long_sub, 2 * items) &&
                  dalloc(x, reinterpret_cast<unsigned char **>(&w.long_res), items * gkv::long_res_bytes());
        if (!ok) return fail(x, GKV_ENOMEM, "build_trees: long-unit work items");
        w.long_cap = items;
    }
    if (units > w.long_units_cap) {
        if (!(dalloc(x, &w.long_start, units) && dalloc(x, &w.long_cnt, units)))
            return fail(x, GKV_ENOMEM, "build_trees: long-unit lists");
        w.long_units_cap = units;
    }
    return GKV_OK;
}

// Long units (build_long.cu): further levels of the listed units, every
// pending node at once, until none is left.
static cudaError_t long_to_leaves(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                                  const int32_t *units, int n_units, cudaStream_t s) {
    cudaError_t e = cudaSuccess;
    for (unsigned int items = 1; e == cudaSuccess && items > 0;)
        e = gkv::launch_long_level(c, K, V, Q, omega, c.w.slots, c.J, 0, 0, -INFINITY, units, n_units, 0, -1, s,
                                   &items);
    return e;
}

// The first tree-building launch of the units of (l, g) in [lg0, lg0 + nlg).
static cudaError_t build_fresh(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                               const int cnt[4], int lg0, int nlg, cudaStream_t s) {
    gkv::Workspace &w = c.w;
    const int64_t nu = (int64_t)c.p.L * c.p.G * c.J;
    // with per-(l, g) capacities ("w/o GA") the global threshold cannot prune:
    // the trees are built completely in this launch
    const bool full = c.p.quota_alloc != 0;
    const bool root_only = !full && c.B_free < nu;
    gkv::StageTimer tm(c, 3, s);
    cudaError_t e = gkv::launch_unit_build(c, K, V, Q, omega, w.slots, c.J, 0, root_only ? 1 : 0,
                                           full ? 4 * gkv::kMaxUnit : 1, 0.f, w.u_list, cnt[0],
                                           w.u_list + (c.J - cnt[1]), cnt[1], s, lg0, nlg);
    if (e != cudaSuccess || cnt[2] == 0) return e;
    e = gkv::launch_long_level(c, K, V, Q, omega, w.slots, c.J, 1, root_only ? 1 : 0, 0.f, w.long_slots, cnt[2],
                               lg0, nlg, s, nullptr);
    if (e != cudaSuccess || !full) return e;
    e = gkv::launch_long_units(c, w.long_slots, cnt[2], lg0, nlg, c.J, w.long_list, s);
    if (e != cudaSuccess) return e;
    return long_to_leaves(c, K, V, Q, omega, w.long_list, cnt[2] * nlg, s);
}

// Trees (build.cu).  Every op's key is bounded before it is built: a pending
// node's split key is at most min(creator key, omega R D).  Each pass derives
// the threshold tau of the ops built so far (a lower bound of the final one)
// and expands the pending nodes whose bound reaches it -- one level while tau
// still rises, up to four once it has settled (a child below tau stays
// pending) -- until none does; nodes left pending can never be selected.
// Several levels per launch save reloading the units that keep expanding.  When the budget is
// smaller than the number of units, the first launch evaluates only the
// roots' own distortion (their Add ops) and later passes expand the units
// with the largest bounds first, about 32768 at a time, so that tau rises
// before weaker units are considered; otherwise it evaluates every root's
// split at once.  When the budget left provably covers the complete
// expansion of every unit that reaches tau, those trees are built to the end.
static cudaError_t build_passes(Ctx &c, const void *K, const void *V, const void *Q, const float *omega,
                                cudaStream_t s) {
    if (c.p.quota_alloc) return cudaSuccess;     // complete trees: nothing is pending
    gkv::Workspace &w = c.w;
    const int J = c.J;
    const int64_t nu = (int64_t)c.p.L * c.p.G * J;
    const bool root_only = c.B_free < nu;
    const int pass_units = 32768;
    float tau_prev = -INFINITY;   // tau of the previous pass
    cudaError_t e = cudaSuccess;
    for (int it = 0; e == cudaSuccess; it++) {
        struct {
            int count[3];
            unsigned long long prefix, all, total, pot;
            float cut;
            unsigned int nqual;
        } h = {{0, 0, 0}, 0, 0, 0, 0, 0.f, 0};
        {
            gkv::StageTimer tm(c, 3, s);
            e = gkv::launch_threshold(c, J, s);
            if (e == cudaSuccess && root_only) e = gkv::launch_pend_cut(c, J, pass_units, w.pend_cut, w.pend_n, s);
            if (e == cudaSuccess) e = gkv::launch_prune_list(c, w.slots, J, w.u_list, w.dev_int + 2, w.long_list, s);
        }
        if (e == cudaSuccess) e = cudaMemcpyAsync(h.count, w.dev_int + 2, 3 * sizeof(int), cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.prefix, w.alloc_state, 2 * sizeof(unsigned long long),
                                                  cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.all, w.alloc_state + 2, sizeof(unsigned long long),
                                                  cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.cut, w.pend_cut, sizeof(float), cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.nqual, w.pend_n, sizeof(unsigned int), cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.total, w.alloc_state + 6, sizeof(unsigned long long),
                                                  cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&h.pot, w.pend_pot, sizeof(unsigned long long),
                                                  cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
        if (e != cudaSuccess || h.count[0] + h.count[1] + h.count[2] == 0) break;
        uint32_t bits = (uint32_t)h.prefix;
        float tau;
        memcpy(&tau, &bits, sizeof tau);
        if (h.all) tau = -INFINITY;
        const float tau_eff = fmaxf(tau, h.cut);
        // everything built so far fits and few units remain: expand them fully at once
        const bool fits = h.all && (long long)c.B_free - (long long)h.total >= (long long)h.pot;
        // several levels per launch once tau has settled (within 10 % of the
        // previous pass's): the children are then checked against a tau close to
        // the final one; while tau still rises, one level, so that a child it
        // would rule out next pass is not built.  With long units the passes
        // follow their levels anyway, and several levels per launch spare the
        // other units that many reloads.
        const bool settled = tau_prev > -INFINITY && tau <= tau_prev + 0.1f * fabsf(tau_prev);
        const int levels = fits ? 4 * gkv::kMaxUnit : ((settled || c.n_long > 0) ? 4 : 1);
        tau_prev = tau;
        gkv::StageTimer tm(c, 3, s);
        e = gkv::launch_unit_build(c, K, V, Q, omega, w.slots, J, 1, 0, levels, tau_eff, w.u_list,
                                   h.count[0], w.u_list + (nu - h.count[1]), h.count[1], s);
        if (e == cudaSuccess && h.count[2] > 0) {   // long units: one level, or all of them when they fit
            e = gkv::launch_long_level(c, K, V, Q, omega, w.slots, J, 0, 0, tau_eff, w.long_list, h.count[2], 0, -1,
                                       s, nullptr, tau);   // subtrees prune against tau itself, not the cut
            if (e == cudaSuccess && fits) e = long_to_leaves(c, K, V, Q, omega, w.long_list, h.count[2], s);
        }
        c.build_passes = it + 2;
    }
    return e;
}

gkv_status gracekv_build_trees(gracekv_ctx *x, const void *K, const void *V, const void *Q,
                               const float *omega, const int32_t *slot_starts, int32_t n_slots,
                               void *stream) {
    gkv_status st = ready(x, 1);
    if (st) return st;
    Ctx &c = x->c;
    if (!K || !V || !Q) return fail(x, GKV_EINVAL, "build_trees: null tensor");
    if (!al16(K) || !al16(V) || !al16(Q) || !al4(omega) || !al4(slot_starts))
        return fail(x, GKV_EINVAL, "build_trees: misaligned pointer (K, V, Q need 16 bytes)");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    st = build_setup(x, slot_starts, n_slots, s);
    if (st) return st;
    cudaError_t e = cudaSuccess;
    if (c.score_pending && c.score_K == K && c.score_Q == Q) {
        e = launch_score(c, K, Q, c.score_stream);
        if (e != cudaSuccess) return cuda_fail(x, e, "score");
    }
    c.score_pending = false;
    if (c.scored && c.score_K == K && c.score_Q == Q) {   // issued ahead by gracekv_score
        e = cudaStreamWaitEvent(s, c.score_ev, 0);
    } else {
        e = cudaMemsetAsync(c.w.dev_int + gkv::kScoreStatus, 0, sizeof(int), s);
        if (e == cudaSuccess) {
            gkv::StageTimer tm(c, 1, s);
            e = gkv::launch_row_stats(c, K, Q, s);
        }
        if (e == cudaSuccess) {
            gkv::StageTimer tm(c, 2, s);
            e = gkv::launch_token_values(c, K, Q, s);
        }
    }
    c.scored = false;
    int cnt[4];
    if (e == cudaSuccess && c.p.lambda_graph > 0.0) {   // R = (1 - lambda) s-hat + lambda d-hat
        if (!c.mh_Qg) return fail(x, GKV_EINVAL, "build_trees: multi-hop relevance needs gracekv_set_graph_queries");
        c.mh_K = K;
        gkv::StageTimer tm(c, 7, s);
        e = gkv::launch_multihop(c, s);
    }
    if (e == cudaSuccess && c.p.alpha_floor > 0.0) {   // Stage I: needs every (l, g)'s token values
        gkv::StageTimer tm(c, 6, s);
        e = gkv::launch_floor(c, c.J, s);
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "build_trees launch");
    st = classes(x, cnt, s);
    if (st) return st;
    e = build_fresh(c, K, V, Q, omega, cnt, 0, c.p.L * c.p.G, s);
    if (e == cudaSuccess) e = build_passes(c, K, V, Q, omega, s);
    if (e != cudaSuccess) return cuda_fail(x, e, "build_trees launch");
    c.stage = 2;
    return GKV_OK;
}

// ---- the whole pass from host buffers, copies overlapped with the work -------

gkv_status gracekv_compress_host(gracekv_ctx *x, const void *K, const void *V, const void *Q,
                                 const float *omega, void *K_out, void *V_out, int32_t *pos, float *log_m,
                                 int32_t *src_lo, int32_t *src_hi, int64_t *offsets, int64_t cap,
                                 int64_t *n_entries_host, void *stream) {
    if (x && x->c.p.lambda_graph > 0.0)
        return fail(x, GKV_EUNSUPPORTED, "compress_host: multi-hop relevance needs the device path");
    gkv_status st = ready(x, 0);
    if (st) return st;
    Ctx &c = x->c;
    const gkv_params &p = c.p;
    if (!K || !V || !Q || !K_out || !V_out || !pos || !log_m || !src_lo || !src_hi || !offsets || !n_entries_host)
        return fail(x, GKV_EINVAL, "compress_host: null argument");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t es = p.dtype == GKV_BF16 ? 2 : 4;
    const int LG = p.L * p.G;
    const size_t layer = (size_t)p.G * p.T * p.d * es;   // bytes of one layer of K (or V)
    const size_t qbytes = (size_t)p.L * p.Hq * p.W * p.d * es;
    const int ngrp = std::min(p.L, 4);
    // device buffers, allocated on the first call
    if (!c.hK) {
        const int64_t ecap = p.budget + (int64_t)LG * (p.T - c.Nc) + 8;
        bool ok = dalloc(x, reinterpret_cast<unsigned char **>(&c.hK), layer * p.L) &&
                  dalloc(x, reinterpret_cast<unsigned char **>(&c.hV), layer * p.L) &&
                  dalloc(x, reinterpret_cast<unsigned char **>(&c.hQ), qbytes) && dalloc(x, &c.hOm, (size_t)LG) &&
                  dalloc(x, &c.hSlots, (size_t)c.Nc + 2) &&
                  dalloc(x, reinterpret_cast<unsigned char **>(&c.oK), (size_t)ecap * p.d * es) &&
                  dalloc(x, reinterpret_cast<unsigned char **>(&c.oV), (size_t)ecap * p.d * es) &&
                  dalloc(x, &c.opos, (size_t)ecap) && dalloc(x, &c.olo, (size_t)ecap) &&
                  dalloc(x, &c.ohi, (size_t)ecap) && dalloc(x, &c.ologm, (size_t)ecap) &&
                  dalloc(x, &c.ooff, (size_t)LG + 1);
        if (!ok) {
            c.hK = nullptr;
            return fail(x, GKV_ENOMEM, "compress_host: device copies of the inputs");
        }
        c.ocap = ecap;
    }
    cudaError_t e = cudaSuccess;
    if (!c.copy_stream) e = cudaStreamCreateWithFlags(&c.copy_stream, cudaStreamNonBlocking);
    while (e == cudaSuccess && (int)c.copy_ev.size() < 2 + ngrp) {
        cudaEvent_t ev;
        e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e == cudaSuccess) c.copy_ev.push_back(ev);
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host setup");
    cudaStream_t cs = c.copy_stream;
    unsigned char *dK = static_cast<unsigned char *>(c.hK), *dV = static_cast<unsigned char *>(c.hV);
    const unsigned char *Kh = static_cast<const unsigned char *>(K), *Vh = static_cast<const unsigned char *>(V);
    auto is_seg = [&](int l) {
        for (int i = 0; i < c.nseg; i++)
            if (c.seg_layers[i] == l) return true;
        return false;
    };
    // copies: Q and the segmentation layers of V first, then the layer groups
    // (the copy stream starts after the work already on `stream`, which may
    // still read these buffers)
    e = cudaEventRecord(c.copy_ev[0], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, c.copy_ev[0], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(c.hQ, Q, qbytes, cudaMemcpyHostToDevice, cs);
    if (e == cudaSuccess && omega) e = cudaMemcpyAsync(c.hOm, omega, (size_t)LG * sizeof(float), cudaMemcpyHostToDevice, cs);
    for (int i = 0; e == cudaSuccess && i < c.nseg; i++) {
        const size_t off = (size_t)c.seg_layers[i] * layer;
        e = cudaMemcpyAsync(dV + off, Vh + off, layer, cudaMemcpyHostToDevice, cs);
    }
    if (e == cudaSuccess) e = cudaEventRecord(c.copy_ev[1], cs);
    for (int gi = 0; e == cudaSuccess && gi < ngrp; gi++) {
        const int l0 = gi * p.L / ngrp, l1 = (gi + 1) * p.L / ngrp;
        e = cudaMemcpyAsync(dK + l0 * layer, Kh + l0 * layer, (l1 - l0) * layer, cudaMemcpyHostToDevice, cs);
        for (int l = l0; e == cudaSuccess && l < l1; l++)
            if (!is_seg(l)) e = cudaMemcpyAsync(dV + l * layer, Vh + l * layer, layer, cudaMemcpyHostToDevice, cs);
        if (e == cudaSuccess) e = cudaEventRecord(c.copy_ev[2 + gi], cs);
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host copies");
    const float *om = omega ? c.hOm : nullptr;
    // segmentation as soon as its layers are in
    e = cudaStreamWaitEvent(s, c.copy_ev[1], 0);
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host");
    int32_t J = 0;
    c.score_pending = false;
    c.scored = false;
    st = gracekv_segment(x, c.hV, nullptr, 0, nullptr, c.hSlots, c.Nc + 1, &J, nullptr, stream);
    if (st) return st;
    st = build_setup(x, nullptr, 0, s);
    if (st) return st;
    int cnt[4];
    e = cudaMemsetAsync(c.w.dev_int + gkv::kScoreStatus, 0, sizeof(int), s);
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host");
    st = classes(x, cnt, s);
    if (st) return st;
    // per layer group, once it is in: score passes and the first tree-building launch
    const bool ranged = gkv::use_tc(c);
    const bool fl = p.alpha_floor > 0.0;   // the floor needs every (l, g)'s token values first
    for (int gi = 0; e == cudaSuccess && gi < ngrp; gi++) {
        const int l0 = gi * p.L / ngrp, l1 = (gi + 1) * p.L / ngrp;
        e = cudaStreamWaitEvent(s, c.copy_ev[2 + gi], 0);
        if (!ranged || e != cudaSuccess) continue;
        {
            gkv::StageTimer tm(c, 1, s);
            e = gkv::launch_row_stats(c, c.hK, c.hQ, s, l0, l1);
        }
        if (e == cudaSuccess) {
            gkv::StageTimer tm(c, 2, s);
            e = gkv::launch_token_values(c, c.hK, c.hQ, s, l0, l1);
        }
        if (e == cudaSuccess && !fl) e = build_fresh(c, c.hK, c.hV, c.hQ, om, cnt, l0 * p.G, (l1 - l0) * p.G, s);
    }
    if (e == cudaSuccess && fl) {
        if (ranged) {
            gkv::StageTimer tm(c, 6, s);
            e = gkv::launch_floor(c, c.J, s);
            if (e == cudaSuccess) e = build_fresh(c, c.hK, c.hV, c.hQ, om, cnt, 0, LG, s);
        }
    }
    if (e == cudaSuccess && !ranged) {   // other score paths: whole layers range at once
        {
            gkv::StageTimer tm(c, 1, s);
            e = gkv::launch_row_stats(c, c.hK, c.hQ, s);
        }
        if (e == cudaSuccess) {
            gkv::StageTimer tm(c, 2, s);
            e = gkv::launch_token_values(c, c.hK, c.hQ, s);
        }
        if (e == cudaSuccess && fl) {
            gkv::StageTimer tm(c, 6, s);
            e = gkv::launch_floor(c, c.J, s);
        }
        if (e == cudaSuccess) e = build_fresh(c, c.hK, c.hV, c.hQ, om, cnt, 0, LG, s);
    }
    if (e == cudaSuccess) e = build_passes(c, c.hK, c.hV, c.hQ, om, s);
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host trees");
    c.stage = 2;
    int64_t E = 0;
    st = gracekv_allocate(x, &E, stream);
    if (st) return st;
    *n_entries_host = E;
    if (E > cap) return fail(x, GKV_ECAPACITY, "compress_host: more cache entries than cap");
    st = gracekv_gather(x, c.hK, c.hV, c.oK, c.oV, c.opos, c.ologm, c.olo, c.ohi, c.ooff, c.ocap, stream);
    if (st) return st;
    const size_t row = (size_t)p.d * es;
    e = cudaMemcpyAsync(K_out, c.oK, (size_t)E * row, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(V_out, c.oV, (size_t)E * row, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(pos, c.opos, (size_t)E * 4, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(log_m, c.ologm, (size_t)E * 4, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(src_lo, c.olo, (size_t)E * 4, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(src_hi, c.ohi, (size_t)E * 4, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(offsets, c.ooff, (size_t)(LG + 1) * 8, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(x, e, "compress_host results");
    return GKV_OK;
}

gkv_status gracekv_allocate(gracekv_ctx *x, int64_t *n_entries_host, void *stream) {
    gkv_status st = ready(x, 2);
    if (st) return st;
    Ctx &c = x->c;
    if (!n_entries_host) return fail(x, GKV_EINVAL, "allocate: null argument");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e;
    {
        gkv::StageTimer tm(c, 4, s);
        e = gkv::launch_allocate(c, c.J, s);
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "allocate launch");
    unsigned long long used = 0;
    int h = 0;
    e = cudaMemcpyAsync(&used, c.w.alloc_state + 7, sizeof used, cudaMemcpyDeviceToHost, s);
    int hs = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&h, c.w.dev_int + 1, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&hs, c.w.dev_int + gkv::kScoreStatus, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(x, e, "allocate");
    st = check_status(x, h | hs);
    if (st) return st;
    const int64_t LG = (int64_t)c.p.L * c.p.G;
    c.used = (int64_t)used;
    *n_entries_host = LG * (c.p.T - c.Nc) + c.used;
    c.stage = 3;
    return GKV_OK;
}

gkv_status gracekv_set_graph_queries(gracekv_ctx *x, const void *Qg, int32_t n_graph) {
    if (!x) return GKV_EINVAL;
    if (x->c.sticky != GKV_OK) return GKV_ESTATE;
    Ctx &c = x->c;
    if (c.p.lambda_graph <= 0.0) return fail(x, GKV_ESTATE, "set_graph_queries: lambda_graph is 0");
    if (!Qg || !al16(Qg)) return fail(x, GKV_EINVAL, "set_graph_queries: null or misaligned Qg");
    if (n_graph != c.mh_ngraph) return fail(x, GKV_EINVAL, "set_graph_queries: wrong number of graph layers");
    c.mh_Qg = Qg;
    return GKV_OK;
}

gkv_status gracekv_export_floor(gracekv_ctx *x, uint8_t *accepted, float *f, int64_t *B_floor_host,
                                void *stream) {
    gkv_status st = ready(x, 2);
    if (st) return st;
    Ctx &c = x->c;
    if (c.p.alpha_floor <= 0.0) return fail(x, GKV_ESTATE, "export_floor: no floor was built");
    if (!accepted || !B_floor_host) return fail(x, GKV_EINVAL, "export_floor: null argument");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t n = (size_t)c.p.L * c.p.G * c.Nc;
    unsigned long long g[4] = {0, 0, 0, 0};
    cudaError_t e = cudaMemcpyAsync(accepted, c.w.fl_acc, n, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && f) e = cudaMemcpyAsync(f, c.w.fl_f, n * sizeof(float), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(g, c.w.fl_glob, sizeof g, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(x, e, "export_floor");
    *B_floor_host = (int64_t)g[2];
    return GKV_OK;
}

gkv_status gracekv_gather(gracekv_ctx *x, const void *K, const void *V, void *K_out, void *V_out,
                          int32_t *pos, float *log_m, int32_t *src_lo, int32_t *src_hi,
                          int64_t *offsets, int64_t cap, void *stream) {
    gkv_status st = ready(x, 3);
    if (st) return st;
    Ctx &c = x->c;
    if (!K || !V || !K_out || !V_out || !pos || !log_m || !src_lo || !src_hi || !offsets)
        return fail(x, GKV_EINVAL, "gather: null argument");
    if (!al16(K) || !al16(V) || !al16(K_out) || !al16(V_out) || !al4(pos) || !al4(log_m) ||
        !al4(src_lo) || !al4(src_hi) || !al8(offsets))
        return fail(x, GKV_EINVAL, "gather: misaligned pointer (K, V, K_out, V_out need 16 bytes)");
    const int64_t LG = (int64_t)c.p.L * c.p.G;
    if (cap < LG * (c.p.T - c.Nc) + c.used) return fail(x, GKV_ECAPACITY, "gather: cap below the entry count");
    cudaError_t e;
    {
        gkv::StageTimer tm(c, 5, static_cast<cudaStream_t>(stream));
        e = gkv::launch_gather(c, K, V, c.w.slots, c.J, K_out, V_out, pos, log_m, src_lo, src_hi,
                               offsets, static_cast<cudaStream_t>(stream));
    }
    if (e != cudaSuccess) return cuda_fail(x, e, "gather launch");
    return GKV_OK;
}

gkv_status gracekv_export(gracekv_ctx *x, int64_t node_cap, int64_t *n_nodes_host, int64_t *unit_first,
                          float *unit_Uadd, float *unit_Ddrop, uint8_t *add_sel, int32_t *a, int32_t *b,
                          int32_t *child0, int32_t *nchild, int32_t *cost, float *D, float *R, float *U,
                          float *kappa, uint8_t *split_sel, float *row_m, float *row_Z, float *row_ZC,
                          float *rtok, void *stream) {
    gkv_status st = ready(x, 2);
    if (st) return st;
    Ctx &c = x->c;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t LG = (int64_t)c.p.L * c.p.G, J = c.J, nu = LG * J;
    const gkv::Workspace &w = c.w;
    std::vector<int32_t> slots(J + 1), nn(nu);
    std::vector<int32_t> ha(c.node_cap), hb(c.node_cap), hc(c.node_cap);
    std::vector<int8_t> hn(c.node_cap), hk(c.node_cap);
    std::vector<float> hD(c.node_cap);
    std::vector<float> hR(c.node_cap), hU(c.node_cap), hK(c.node_cap);
    std::vector<uint8_t> hs(c.node_cap);
    cudaError_t e = cudaStreamSynchronize(s);
#define CP(dst, src, n) if (e == cudaSuccess) e = cudaMemcpy(dst, src, (n) * sizeof(*(dst)), cudaMemcpyDeviceToHost)
    CP(slots.data(), w.slots, J + 1);
    CP(nn.data(), w.u_nnodes, nu);
    CP(ha.data(), w.nd_a, c.node_cap); CP(hb.data(), w.nd_b, c.node_cap);
    CP(hc.data(), w.nd_child0, c.node_cap); CP(hn.data(), w.nd_nchild, c.node_cap);
    CP(hk.data(), w.nd_cost, c.node_cap); CP(hD.data(), w.nd_D, c.node_cap);
    CP(hR.data(), w.nd_R, c.node_cap); CP(hU.data(), w.nd_U, c.node_cap);
    CP(hK.data(), w.nd_kappa, c.node_cap); CP(hs.data(), w.nd_sel, c.node_cap);
    if (unit_Uadd) CP(unit_Uadd, w.u_Uadd, nu);
    if (unit_Ddrop) CP(unit_Ddrop, w.u_Ddrop, nu);
    if (add_sel) CP(add_sel, w.u_sel, nu);
    const int64_t nrow = (int64_t)c.p.L * c.p.Hq * c.p.W;
    if (row_m) CP(row_m, w.row_m, nrow);
    if (row_Z) CP(row_Z, w.row_Z, nrow);
    if (row_ZC) CP(row_ZC, w.row_ZC, nrow);
    if (rtok) CP(rtok, w.rtok, LG * c.Nc);
#undef CP
    if (e != cudaSuccess) return cuda_fail(x, e, "export");
    int64_t k = 0;
    for (int64_t uid = 0; uid < nu; uid++) {
        int lg = (int)(uid / J), j = (int)(uid % J);
        int64_t nb = gkv::node_base(lg, slots[j], c.p.ctx_start, c.Nc);
        if (unit_first) unit_first[uid] = k;
        for (int q = 0; q < nn[uid]; q++, k++) {
            if (k >= node_cap) continue;
            int64_t v = nb + q;
            if (a) a[k] = ha[v];
            if (b) b[k] = hb[v];
            if (child0) child0[k] = hc[v];
            if (nchild) nchild[k] = hn[v];
            if (cost) cost[k] = hk[v];
            if (D) D[k] = hD[v];
            if (R) R[k] = hR[v];
            if (U) U[k] = hU[v];
            if (kappa) kappa[k] = hK[v];
            if (split_sel) split_sel[k] = c.stage >= 3 ? hs[v] : 0;
        }
    }
    if (unit_first) unit_first[nu] = k;
    *n_nodes_host = k;
    if (k > node_cap) return fail(x, GKV_ECAPACITY, "export: node_cap too small");
    return GKV_OK;
}

gkv_status gracekv_profile(gracekv_ctx *x, int32_t enable) {
    if (!x) return GKV_EINVAL;
    x->c.profile = enable != 0;
    x->c.ev_used = 0;
    x->c.ev_stage.clear();
    return GKV_OK;
}

gkv_status gracekv_stats(gracekv_ctx *x, float *stage_ms, int32_t n_stages, int64_t *launches,
                         uint64_t *work, int32_t n_work) {
    if (!x) return GKV_EINVAL;
    Ctx &c = x->c;
    if (launches) *launches = c.launches;
    if (work && n_work > 0) {
        unsigned long long h[4] = {0, 0, 0, 0};
        cudaError_t e = cudaMemcpy(h, c.w.work, sizeof h, cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(x, e, "stats");
        for (int i = 0; i < n_work; i++)
            work[i] = i < 4 ? h[i] : i == 4 ? (uint64_t)c.dp_chunks : i == 5 ? (uint64_t)c.dp_rerun : 0;
    }
    if (stage_ms) {
        for (int i = 0; i < n_stages; i++) stage_ms[i] = 0.f;
        for (size_t k = 0; k < c.ev_stage.size(); k++) {
            cudaEvent_t e0 = c.ev_pool[2 * k], e1 = c.ev_pool[2 * k + 1];
            cudaError_t e = cudaEventSynchronize(e1);
            float ms = 0.f;
            if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
            if (e != cudaSuccess) return cuda_fail(x, e, "stats");
            int st = c.ev_stage[k];
            if (st >= 0 && st < n_stages) stage_ms[st] += ms;
        }
    }
    c.ev_used = 0;
    c.ev_stage.clear();
    return GKV_OK;
}

}  // extern "C"
