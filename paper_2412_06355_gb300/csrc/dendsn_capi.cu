// C ABI of libdendsn: argument validation, tiling plan, dispatch to the compiled
// kernel instances, and the deterministic parameter-gradient finalize kernel.
#include <algorithm>
#include <atomic>
#include <mutex>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "dendsn.h"
#include "dendsn_types.h"

namespace dendsn {

// Sums the block partials of every channel in a fixed order and writes the parameter
// gradients (grad_beta only when requested). One thread per (channel, gradient slot).
__global__ void param_grad_finalize_kernel(const FinArgs F) {
    pdl_wait();
    pdl_trigger();
    const Geometry &g = F.g;
    const int NP = 2 * g.K + 2 * g.Kb + 1;
    const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (w >= (int64_t)g.C * NP) return;
    const int c = (int)(w / NP);
    const int q = (int)(w % NP);
    float sum = 0.f;
    if (g.O > 0 && g.T > 0) {
        const int ct_lo = (int)(((int64_t)c * g.inner) / g.TXn);
        const int ct_hi = (int)((((int64_t)c + 1) * g.inner - 1) / g.TXn);
        for (int ct = ct_lo; ct <= ct_hi; ++ct) {
            const int lc = c - (int)(((int64_t)ct * g.TXn) / g.inner);
            const float *p = F.partials + ((int64_t)ct * g.nch_max + lc) * NP + q;
            const int64_t stride = (int64_t)g.nCT * g.nch_max * NP;   // between row groups
            // unrolled so that the loads of eight row groups are in flight together; the
            // additions keep their fixed order
            int rg = 0;
            for (; rg + 8 <= g.nRG; rg += 8) {
                float v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) v[u] = p[(int64_t)(rg + u) * stride];
#pragma unroll
                for (int u = 0; u < 8; ++u) sum = __fadd_rn(sum, v[u]);
            }
            for (; rg < g.nRG; ++rg) sum = __fadd_rn(sum, p[(int64_t)rg * stride]);
        }
    }
    if (q < g.K) F.g_alpha[(int64_t)c * g.K + q] = F.stateless ? 0.f : sum;
    else if (q < 2 * g.K) F.g_xi[(int64_t)c * g.K + (q - g.K)] = sum;
    else if (q < 2 * g.K + g.Kb) F.g_zeta[(int64_t)c * g.Kb + (q - 2 * g.K)] = sum;
    else if (q < 2 * g.K + 2 * g.Kb) F.g_kappa[(int64_t)c * g.Kb + (q - 2 * g.K - g.Kb)] = sum;
    else if (F.g_beta) F.g_beta[c] = sum;
}

cudaError_t launch_finalize(const FinArgs &a, cudaStream_t s) {
    const int64_t n = (int64_t)a.g.C * (2 * a.g.K + 2 * a.g.Kb + 1);
    const int threads = 256;
    const int blocks = (int)((n + threads - 1) / threads);
#if DENDSN_PDL
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, param_grad_finalize_kernel, a);
#else
    param_grad_finalize_kernel<<<blocks, threads, 0, s>>>(a);
    return cudaGetLastError();
#endif
}

namespace {
struct ResidentKey {
    const void *kernel;
    int threads;
    size_t bytes;
    int device;
    int blocks;
};
std::mutex g_resident_mutex;
ResidentKey g_resident[256];
int g_resident_n = 0;
}  // namespace

cudaError_t resident_blocks(const void *kernel, int threads, size_t bytes, int *out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_resident_mutex);
    for (int i = 0; i < g_resident_n; ++i) {
        const ResidentKey &k = g_resident[i];
        if (k.kernel == kernel && k.threads == threads && k.bytes == bytes && k.device == dev) {
            *out = k.blocks;
            return cudaSuccess;
        }
    }
    int n = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, bytes);
    if (e != cudaSuccess) return e;
    if (g_resident_n < (int)(sizeof g_resident / sizeof g_resident[0]))
        g_resident[g_resident_n++] = ResidentKey{kernel, threads, bytes, dev, n};
    *out = n;
    return cudaSuccess;
}

}  // namespace dendsn

using namespace dendsn;

namespace {

thread_local char g_last_error[512] = "";
std::atomic<uint64_t> g_launches{0};

dendsn_status fail(dendsn_status st, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return st;
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

struct Plan {
    Geometry gf, gb;   // forward and backward tilings (block sizes may differ)
    int blocks_f, blocks_b;
    size_t saved_bytes, scratch_bytes, ck_vd_bytes;
    bool keep_vs;      // saved holds V^s [T][BN] for the single-chunk (phased) backward
    int sx;            // bytes per x element
    int layout;        // 0 compartments innermost, 1 the paper's layer layout
    bool tp;           // the time-parallel kernels (one warp per neuron)
};

int sm_count() {
    static int cached = 0;
    if (cached == 0) {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0)
            cached = n;
        else
            cached = 152;   // GB300
    }
    return cached;
}

bool is01(int32_t v) { return v == 0 || v == 1; }

// Column tiling of the O x P neuron matrix for blocks of nt threads with lpn lanes per
// neuron: TXn columns x TY row lanes per block.
void tile_columns(Geometry &g, int nt, int lpn) {
    const int W = 32 / lpn;                     // columns per warp
    const int full = nt / lpn;                  // columns of a one-row tile
    g.TXn = (g.inner >= W && g.P % full == 0) ? full : W;
    g.TY = nt / (g.TXn * lpn);
    g.seg = (g.inner % W == 0) ? W : ((W % g.inner == 0) ? g.inner : 1);
    g.nCT = (int32_t)((g.P + g.TXn - 1) / g.TXn);
    // channels one column tile touches (tiles start at multiples of TXn)
    if (g.TXn % g.inner == 0) g.nch_max = g.TXn / g.inner;
    else if (g.inner % g.TXn == 0) g.nch_max = 1;
    else g.nch_max = std::min<int32_t>(g.C, (g.TXn - 1) / g.inner + 2);
}

// Row tiling: R rows per thread and nRG row groups, so that the grid is nCT * nRG blocks.
// The fixed sizing aims at about per_sm blocks per SM (measured best on the layer
// workloads when a wave is nearly full). With `resident` blocks of the kernel fitting on
// one SM the grid runs in waves of resident * sms blocks, and a last wave that is only
// partly filled leaves SMs idle while it finishes: the time is modelled as
// (waves) x (rows per thread + one row's worth of per-block set-up and reduction), and the
// row groups that minimise it (over up to four times the waves of the fixed sizing)
// replace the fixed sizing when the model predicts at least 8% less time. Below that the
// model is within its own error: on the layer workloads it predicted 4-6% that did not
// materialise, while its 11-20% predictions gave 7-13% (token layer forward and backward,
// event-stream layer backward).
dendsn_status tile_rows(Geometry &g, int64_t sms, int resident, int per_sm, int64_t *blocks) {
    const int64_t rows = std::max<int64_t>(1, (g.O + g.TY - 1) / g.TY);   // row slots per column
    auto rows_for = [&](int64_t nrg, int64_t *nrg_used) {
        const int64_t R = std::max<int64_t>(1, (rows + nrg - 1) / nrg);
        *nrg_used = (rows + R - 1) / R;
        return R;
    };
    // the fixed sizing: about per_sm blocks per SM in total, at least one row
    const int64_t target_blocks = (int64_t)per_sm * sms;
    const int64_t rg_target = std::max<int64_t>(1, (target_blocks + g.nCT - 1) / g.nCT);
    int64_t best_n = 0;
    int64_t best_R = rows_for(rg_target, &best_n);
    if (resident > 0) {
        const int64_t cap = (int64_t)resident * sms;
        auto cost = [&](int64_t nrg, int64_t R) {
            return (double)((g.nCT * nrg + cap - 1) / cap) * (double)(R + 1);
        };
        const double fixed_cost = cost(best_n, best_R);
        const int64_t wmax = std::min<int64_t>(64, 4 * std::max<int64_t>(1, (target_blocks + cap - 1) / cap));
        double best_cost = 0.0;
        int64_t cand_R = 0, cand_n = 0;
        for (int64_t w = 1; w <= wmax; ++w) {
            const int64_t top = std::max<int64_t>(1, std::min<int64_t>(rows, w * cap / g.nCT));
            for (int64_t nrg = std::max<int64_t>(1, top - 2); nrg <= top; ++nrg) {
                int64_t used = 0;
                const int64_t R = rows_for(nrg, &used);
                const double c = cost(used, R);
                if (cand_n == 0 || c < best_cost || (c == best_cost && used < cand_n)) {
                    best_cost = c;
                    cand_R = R;
                    cand_n = used;
                }
            }
        }
        if (cand_n > 0 && best_cost < 0.92 * fixed_cost) {
            best_R = cand_R;
            best_n = cand_n;
        }
    }
    g.R = (int32_t)best_R;
    g.nRG = (int32_t)((g.O + (int64_t)g.R * g.TY - 1) / ((int64_t)g.R * g.TY));
    *blocks = (int64_t)g.nCT * g.nRG;
    if (*blocks > INT32_MAX) return fail(DENDSN_ERR_UNSUPPORTED, "grid too large");
    return DENDSN_OK;
}

cudaError_t dispatch_forward(const dendsn_config &cfg, int layout, const FwdArgs &a, int blocks,
                             cudaStream_t s, int *resident = nullptr);
cudaError_t dispatch_backward(const dendsn_config &cfg, int layout, int L, const BwdArgs &a,
                              int blocks, cudaStream_t s, int *resident = nullptr);

dendsn_status make_plan(const dendsn_config *cfg, Plan *pl) {
    if (cfg == nullptr) return fail(DENDSN_ERR_INVALID_ARG, "cfg is NULL");
    const dendsn_config &c = *cfg;
    if (c.T < 0 || c.B < 0 || c.N < 0)
        return fail(DENDSN_ERR_INVALID_ARG, "negative size (T=%d B=%d N=%d)", c.T, c.B, c.N);
    if (c.C < 1 || c.inner < 1) return fail(DENDSN_ERR_INVALID_ARG, "C and inner must be >= 1");
    if (c.K < 1 || c.G < 1 || c.K % c.G != 0)
        return fail(DENDSN_ERR_INVALID_ARG, "need K >= 1, G >= 1 and G | K (K=%d G=%d)", c.K, c.G);
    if (!(c.x_dtype == DENDSN_F32 || c.x_dtype == DENDSN_BF16))
        return fail(DENDSN_ERR_INVALID_ARG, "bad x_dtype %d", c.x_dtype);
    if (!is01(c.psi) || !is01(c.reset) || !is01(c.detach_reset) || !is01(c.mask_per_neuron) ||
        !is01(c.stateless) || !is01(c.residual) || !is01(c.layout))
        return fail(DENDSN_ERR_INVALID_ARG, "enum/flag field out of range");
    if (c.surrogate != DENDSN_SG_ATAN)
        return fail(c.surrogate < 0 ? DENDSN_ERR_INVALID_ARG : DENDSN_ERR_UNSUPPORTED,
                    "surrogate %d not available (only the arctan surrogate)", c.surrogate);
    if (!std::isfinite(c.theta) || !std::isfinite(c.beta))
        return fail(DENDSN_ERR_INVALID_ARG, "theta and beta must be finite");
    const bool k_ok = c.K == 1 || c.K == 2 || c.K == 4 || c.K == 8 || c.K == 16;
    const int KT = lane_compartments(c.K);
    if (!k_ok || c.G > 4 || KT % c.G != 0)
        return fail(DENDSN_ERR_UNSUPPORTED, "K=%d G=%d not compiled in", c.K, c.G);
    const int64_t P = (int64_t)c.C * c.inner;
    if (P > INT32_MAX) return fail(DENDSN_ERR_UNSUPPORTED, "C*inner too large");
    if (c.N % P != 0)
        return fail(DENDSN_ERR_INVALID_ARG, "N=%d must be a multiple of C*inner=%lld", c.N,
                    (long long)P);
    const int64_t BN = (int64_t)c.B * c.N;
    const int64_t O = BN / P;
    if (O > INT32_MAX) return fail(DENDSN_ERR_UNSUPPORTED, "too many rows");

    Geometry g;
    std::memset(&g, 0, sizeof g);
    g.O = O;
    g.BN = BN;
    g.P = (int32_t)P;
    g.N = c.N;
    g.C = c.C;
    g.inner = c.inner;
    g.T = c.T;
    g.K = c.K;
    g.Kb = c.K / c.G;
    g.L = (c.T <= 4) ? 4 : 8;
    g.n_ck = (c.T > g.L) ? (c.T + g.L - 1) / g.L - 1 : 0;
    const int64_t sms = sm_count();
    int64_t bf = 0, bb = 0;
    pl->gf = g;
    pl->gb = g;
    const int KTB = bwd_lane_compartments(c.K, c.G, c.x_dtype, g.L);
    tile_columns(pl->gf, fwd_threads(c.K), c.K / KT);
    tile_columns(pl->gb, bwd_threads(KTB), c.K / KTB);
    pl->sx = (c.x_dtype == DENDSN_BF16) ? 2 : 4;
    pl->layout = (c.K > 1 && c.inner > 1) ? c.layout : 0;   // otherwise the layouts coincide
    // narrow layers with long horizons: one warp per neuron, time scanned in parallel
    pl->tp = c.T >= kTpMinT && BN <= kTpMaxNeurons && tp_smem_bytes(c.T, c.K, true) <= kTpMaxSmem;
    // blocks of the forward and backward kernels that fit on one SM. The backward's is taken
    // for the compartments-innermost layout and the build without dL/dbeta, so that both
    // layouts and both builds of a layer share one tiling (and sum the parameter gradients
    // in the same order).
    int res_f = 0, res_b = 0;
    if (!pl->tp && O > 0 && c.T > 0) {
        FwdArgs fa;
        std::memset(&fa, 0, sizeof fa);
        fa.g = pl->gf;
        fa.p.mask_mode = c.mask_per_neuron ? 2 : 0;
        BwdArgs ba;
        std::memset(&ba, 0, sizeof ba);
        ba.g = pl->gb;
        ba.p.mask_mode = fa.p.mask_mode;
        ba.p.residual = c.residual;
        // a failed query (no device) leaves the residency unknown: the fixed sizing applies
        if (dispatch_forward(c, pl->layout, fa, 0, nullptr, &res_f) != cudaSuccess) {
            res_f = 0;
            (void)cudaGetLastError();
        }
        if (dispatch_backward(c, 0, g.L, ba, 0, nullptr, &res_b) != cudaSuccess) {
            res_b = 0;
            (void)cudaGetLastError();
        }
    }
    dendsn_status st = tile_rows(pl->gf, sms, res_f, 16, &bf);
    if (st != DENDSN_OK) return st;
    // backward without the residency: when every column is its own channel (inner = 1)
    // each thread's parameter setup is heavier, and twice the rows per thread measured
    // faster (token layer 285 -> 272 us); elsewhere 16 blocks per SM measured best
    const int bwd_per_sm = (c.inner == 1) ? 8 : 16;
    if ((st = tile_rows(pl->gb, sms, res_b, bwd_per_sm, &bb)) != DENDSN_OK) return st;
    pl->blocks_f = (int)bf;
    pl->blocks_b = (int)bb;
    const size_t NP = 2 * (size_t)c.K + 2 * (size_t)g.Kb + 1;     // + the beta slot
    pl->scratch_bytes = (size_t)bb * pl->gb.nch_max * NP * sizeof(float);
    pl->scratch_bytes = (pl->scratch_bytes + 15) / 16 * 16;
    if (pl->tp) {
        pl->gf.n_ck = pl->gb.n_ck = 0;                 // the backward recomputes from x alone
        pl->scratch_bytes = ((size_t)BN * NP * sizeof(float) + 15) / 16 * 16;
        pl->ck_vd_bytes = pl->saved_bytes = 0;
        pl->keep_vs = false;
        return DENDSN_OK;
    }
    pl->ck_vd_bytes = (size_t)g.n_ck * (size_t)BN * c.K * sizeof(float);
    pl->saved_bytes = pl->ck_vd_bytes + (size_t)g.n_ck * (size_t)BN * sizeof(float);
    // bfloat16 rows of one chunk of whole 8-compartment neurons (the phased backward): the
    // forward keeps V^s, so that the backward recomputes only the compartment scan
    pl->keep_vs = c.x_dtype == DENDSN_BF16 &&
                  takes_phased_backward(c.K, c.G, KTB, pl->layout, c.T, g.L, c.residual != 0);
    if (pl->keep_vs) pl->saved_bytes = (size_t)c.T * (size_t)BN * sizeof(float);
    pl->saved_bytes = (pl->saved_bytes + 15) / 16 * 16;
    return DENDSN_OK;
}

Params make_params(const dendsn_config &c, const float *alpha, const float *xi,
                   const float *zeta, const float *kappa, const uint8_t *mask) {
    Params p;
    p.alpha = alpha;
    p.xi = xi;
    p.zeta = zeta;
    p.kappa = kappa;
    p.mask = mask;
    p.mask_mode = mask == nullptr ? 0 : (c.mask_per_neuron ? 2 : 1);
    p.theta = c.theta;
    p.beta = c.beta;
    p.soft = c.reset == DENDSN_RESET_SOFT;
    p.stateless = c.stateless;
    p.residual = c.residual;
    p.detach = c.detach_reset;
    return p;
}

dendsn_status check_params(const float *alpha, const float *xi, const float *zeta,
                           const float *kappa, const uint8_t *mask) {
    if (!alpha || !xi || !zeta || !kappa)
        return fail(DENDSN_ERR_INVALID_ARG, "parameter pointer is NULL");
    if (!aligned(alpha, 4) || !aligned(xi, 4) || !aligned(zeta, 4) || !aligned(kappa, 4))
        return fail(DENDSN_ERR_MISALIGNED, "parameters must be 4-byte aligned");
    if (mask && !aligned(mask, 4)) return fail(DENDSN_ERR_MISALIGNED, "mask must be 4-byte aligned");
    return DENDSN_OK;
}

#define DENDSN_FWD_CASE(KK, GG)                                                         \
    if (cfg.K == KK && cfg.G == GG) {                                                   \
        switch ((cfg.psi * 2 + cfg.x_dtype) * 2 + layout) {                             \
        case 0: return launch_forward<KK, GG, 0, 0, 0>(a, blocks, s, resident);         \
        case 1: return launch_forward<KK, GG, 0, 0, 1>(a, blocks, s, resident);         \
        case 2: return launch_forward<KK, GG, 0, 1, 0>(a, blocks, s, resident);         \
        case 3: return launch_forward<KK, GG, 0, 1, 1>(a, blocks, s, resident);         \
        case 4: return launch_forward<KK, GG, 1, 0, 0>(a, blocks, s, resident);         \
        case 5: return launch_forward<KK, GG, 1, 0, 1>(a, blocks, s, resident);         \
        case 6: return launch_forward<KK, GG, 1, 1, 0>(a, blocks, s, resident);         \
        default: return launch_forward<KK, GG, 1, 1, 1>(a, blocks, s, resident);        \
        }                                                                               \
    }

// layout: 0 compartments innermost, 1 the paper's layer layout (0 when K = 1 or inner = 1: the same)
cudaError_t dispatch_forward(const dendsn_config &cfg, int layout, const FwdArgs &a, int blocks,
                             cudaStream_t s, int *resident) {
    DENDSN_KG_LIST(DENDSN_FWD_CASE)
    return cudaErrorInvalidValue;
}

#define DENDSN_BWD_L(KK, GG, LL)                                                        \
    switch ((cfg.psi * 2 + cfg.x_dtype) * 2 + layout) {                                 \
    case 0: return launch_backward<KK, GG, 0, 0, LL, 0>(a, blocks, s, resident);        \
    case 1: return launch_backward<KK, GG, 0, 0, LL, 1>(a, blocks, s, resident);        \
    case 2: return launch_backward<KK, GG, 0, 1, LL, 0>(a, blocks, s, resident);        \
    case 3: return launch_backward<KK, GG, 0, 1, LL, 1>(a, blocks, s, resident);        \
    case 4: return launch_backward<KK, GG, 1, 0, LL, 0>(a, blocks, s, resident);        \
    case 5: return launch_backward<KK, GG, 1, 0, LL, 1>(a, blocks, s, resident);        \
    case 6: return launch_backward<KK, GG, 1, 1, LL, 0>(a, blocks, s, resident);        \
    default: return launch_backward<KK, GG, 1, 1, LL, 1>(a, blocks, s, resident);       \
    }

#define DENDSN_BWD_CASE(KK, GG)                                                         \
    if (cfg.K == KK && cfg.G == GG) {                                                   \
        if (L == 4) { DENDSN_BWD_L(KK, GG, 4) }                                         \
        DENDSN_BWD_L(KK, GG, 8)                                                         \
    }

cudaError_t dispatch_backward(const dendsn_config &cfg, int layout, int L, const BwdArgs &a,
                              int blocks, cudaStream_t s, int *resident) {
    DENDSN_KG_LIST(DENDSN_BWD_CASE)
    return cudaErrorInvalidValue;
}

#define DENDSN_TP_FWD_CASE(KK, GG)                                                      \
    if (cfg.K == KK && cfg.G == GG)                                                     \
        return cfg.x_dtype == DENDSN_BF16 ? launch_forward_tp<KK, GG, 1>(a, cfg.psi, layout, s) \
                                          : launch_forward_tp<KK, GG, 0>(a, cfg.psi, layout, s);
#define DENDSN_TP_BWD_CASE(KK, GG)                                                      \
    if (cfg.K == KK && cfg.G == GG)                                                     \
        return cfg.x_dtype == DENDSN_BF16 ? launch_backward_tp<KK, GG, 1>(a, cfg.psi, layout, s) \
                                          : launch_backward_tp<KK, GG, 0>(a, cfg.psi, layout, s);

cudaError_t dispatch_forward_tp(const dendsn_config &cfg, int layout, const FwdArgs &a, cudaStream_t s) {
    DENDSN_KG_LIST(DENDSN_TP_FWD_CASE)
    return cudaErrorInvalidValue;
}

cudaError_t dispatch_backward_tp(const dendsn_config &cfg, int layout, const BwdArgs &a, cudaStream_t s) {
    DENDSN_KG_LIST(DENDSN_TP_BWD_CASE)
    return cudaErrorInvalidValue;
}

}  // namespace

extern "C" {

dendsn_status dendsn_workspace_size(const dendsn_config *cfg, size_t *saved_bytes,
                                    size_t *scratch_bytes) {
    Plan pl;
    dendsn_status st = make_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (saved_bytes) *saved_bytes = pl.saved_bytes;
    if (scratch_bytes) *scratch_bytes = pl.scratch_bytes;
    return DENDSN_OK;
}

dendsn_status dendsn_forward(const dendsn_config *cfg, const void *x, const float *alpha,
                             const float *xi, const float *zeta, const float *kappa,
                             const uint8_t *mask, void *spikes, float *v_out, void *saved,
                             void *stream) {
    Plan pl;
    dendsn_status st = make_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (pl.gf.BN == 0 || pl.gf.T == 0) return DENDSN_OK;
    if (!x || !spikes) return fail(DENDSN_ERR_INVALID_ARG, "x or spikes is NULL");
    if ((st = check_params(alpha, xi, zeta, kappa, mask)) != DENDSN_OK) return st;
    if (!aligned(x, 16)) return fail(DENDSN_ERR_MISALIGNED, "x must be 16-byte aligned");
    if (!aligned(spikes, pl.sx)) return fail(DENDSN_ERR_MISALIGNED, "spikes misaligned");
    if (v_out && !aligned(v_out, 4)) return fail(DENDSN_ERR_MISALIGNED, "v_out misaligned");
    if (saved && !aligned(saved, 16)) return fail(DENDSN_ERR_MISALIGNED, "saved must be 16-byte aligned");
    FwdArgs a;
    a.g = pl.gf;
    a.p = make_params(*cfg, alpha, xi, zeta, kappa, mask);
    a.x = x;
    a.spikes = spikes;
    a.v_out = v_out;
    a.ck_vd = (saved && pl.gf.n_ck > 0) ? static_cast<float *>(saved) : nullptr;
    a.ck_vs = a.ck_vd ? reinterpret_cast<float *>(static_cast<char *>(saved) + pl.ck_vd_bytes)
                      : nullptr;
    a.vs_keep = (saved && pl.keep_vs) ? static_cast<float *>(saved) : nullptr;
    cudaError_t e = pl.tp ? dispatch_forward_tp(*cfg, pl.layout, a, static_cast<cudaStream_t>(stream))
                          : dispatch_forward(*cfg, pl.layout, a, pl.blocks_f, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess)
        return fail(DENDSN_ERR_CUDA, "forward launch failed: %s", cudaGetErrorString(e));
    g_launches.fetch_add(1, std::memory_order_relaxed);
    return DENDSN_OK;
}

}  // extern "C"

namespace {

dendsn_status backward_impl(const dendsn_config *cfg, const void *x, const float *alpha,
                            const float *xi, const float *zeta, const float *kappa,
                            const uint8_t *mask, const void *grad_spikes,
                            const float *grad_v, const void *saved, void *grad_x,
                            float *grad_alpha, float *grad_xi, float *grad_zeta,
                            float *grad_kappa, float *grad_beta, void *scratch, void *stream) {
    Plan pl;
    dendsn_status st = make_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (!grad_alpha || !grad_xi || !grad_zeta || !grad_kappa)
        return fail(DENDSN_ERR_INVALID_ARG, "parameter-gradient pointer is NULL");
    if (!aligned(grad_alpha, 4) || !aligned(grad_xi, 4) || !aligned(grad_zeta, 4) ||
        !aligned(grad_kappa, 4))
        return fail(DENDSN_ERR_MISALIGNED, "parameter gradients must be 4-byte aligned");
    const bool work = pl.gb.BN > 0 && pl.gb.T > 0;
    if (work) {
        if (!x || !grad_spikes || !grad_x)
            return fail(DENDSN_ERR_INVALID_ARG, "x, grad_spikes or grad_x is NULL");
        if ((st = check_params(alpha, xi, zeta, kappa, mask)) != DENDSN_OK) return st;
        if (!aligned(x, 16) || !aligned(grad_x, 16))
            return fail(DENDSN_ERR_MISALIGNED, "x and grad_x must be 16-byte aligned");
        if (!aligned(grad_spikes, pl.sx)) return fail(DENDSN_ERR_MISALIGNED, "grad_spikes misaligned");
        if (grad_v && !aligned(grad_v, 4)) return fail(DENDSN_ERR_MISALIGNED, "grad_v misaligned");
        if (pl.gb.n_ck > 0 && !saved)
            return fail(DENDSN_ERR_INVALID_ARG, "T=%d needs the forward's saved checkpoints", pl.gb.T);
        if (saved && !aligned(saved, 16)) return fail(DENDSN_ERR_MISALIGNED, "saved must be 16-byte aligned");
        if (!scratch) return fail(DENDSN_ERR_INVALID_ARG, "scratch is NULL");
        if (!aligned(scratch, 16)) return fail(DENDSN_ERR_MISALIGNED, "scratch must be 16-byte aligned");
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (work) {
        BwdArgs a;
        a.g = pl.gb;
        a.p = make_params(*cfg, alpha, xi, zeta, kappa, mask);
        a.x = x;
        a.gs = grad_spikes;
        a.gv = grad_v;
        a.ck_vd = pl.gb.n_ck > 0 ? static_cast<const float *>(saved) : nullptr;
        a.ck_vs = pl.gb.n_ck > 0 ? reinterpret_cast<const float *>(
                                      static_cast<const char *>(saved) + pl.ck_vd_bytes)
                                : nullptr;
        a.vs_saved = (saved && pl.keep_vs) ? static_cast<const float *>(saved) : nullptr;
        a.gx = grad_x;
        a.partials = static_cast<float *>(scratch);
        a.want_beta = grad_beta != nullptr;
        cudaError_t e = pl.tp ? dispatch_backward_tp(*cfg, pl.layout, a, s)
                              : dispatch_backward(*cfg, pl.layout, pl.gb.L, a, pl.blocks_b, s);
        if (e != cudaSuccess)
            return fail(DENDSN_ERR_CUDA, "backward launch failed: %s", cudaGetErrorString(e));
        g_launches.fetch_add(1, std::memory_order_relaxed);
    }
    FinArgs f;
    f.g = pl.gb;
    f.partials = static_cast<const float *>(scratch);
    f.g_alpha = grad_alpha;
    f.g_xi = grad_xi;
    f.g_zeta = grad_zeta;
    f.g_kappa = grad_kappa;
    f.g_beta = grad_beta;
    f.stateless = cfg->stateless;
    cudaError_t e = pl.tp ? launch_finalize_tp(f, s) : launch_finalize(f, s);
    if (e != cudaSuccess)
        return fail(DENDSN_ERR_CUDA, "finalize launch failed: %s", cudaGetErrorString(e));
    g_launches.fetch_add(1, std::memory_order_relaxed);
    return DENDSN_OK;
}

}  // namespace

extern "C" {

dendsn_status dendsn_backward(const dendsn_config *cfg, const void *x, const float *alpha,
                              const float *xi, const float *zeta, const float *kappa,
                              const uint8_t *mask, const void *grad_spikes,
                              const float *grad_v, const void *saved, void *grad_x,
                              float *grad_alpha, float *grad_xi, float *grad_zeta,
                              float *grad_kappa, void *scratch, void *stream) {
    return backward_impl(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                         grad_x, grad_alpha, grad_xi, grad_zeta, grad_kappa, nullptr, scratch,
                         stream);
}

dendsn_status dendsn_backward_plif(const dendsn_config *cfg, const void *x, const float *alpha,
                                   const float *xi, const float *zeta, const float *kappa,
                                   const uint8_t *mask, const void *grad_spikes,
                                   const float *grad_v, const void *saved, void *grad_x,
                                   float *grad_alpha, float *grad_xi, float *grad_zeta,
                                   float *grad_kappa, float *grad_beta, void *scratch,
                                   void *stream) {
    if (!grad_beta) return fail(DENDSN_ERR_INVALID_ARG, "grad_beta is NULL");
    if (!aligned(grad_beta, 4)) return fail(DENDSN_ERR_MISALIGNED, "grad_beta must be 4-byte aligned");
    return backward_impl(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                         grad_x, grad_alpha, grad_xi, grad_zeta, grad_kappa, grad_beta, scratch,
                         stream);
}

const char *dendsn_status_string(dendsn_status status) {
    switch (status) {
    case DENDSN_OK: return "ok";
    case DENDSN_ERR_INVALID_ARG: return "invalid argument";
    case DENDSN_ERR_UNSUPPORTED: return "unsupported configuration";
    case DENDSN_ERR_MISALIGNED: return "misaligned pointer";
    case DENDSN_ERR_CUDA: return "CUDA error";
    }
    return "unknown status";
}

const char *dendsn_last_error(void) { return g_last_error; }

uint64_t dendsn_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"

// ---------------------------------------------------------------- scratch-free backward
// A backward for callers that cannot hand the library a scratch buffer: for example a
// plain C host that only receives device pointers for the tensors and has no device
// allocator of its own, or a runtime whose device memory is budgeted up front and that
// must not allocate on each call. The per-block parameter-gradient partials go to a
// fixed buffer compiled into the library instead of caller memory.
namespace {

// Capacity of the built-in scratch buffer. Every GPU that loads the library keeps this
// much device memory reserved until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;   // 8 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 256;
std::mutex g_noalloc_mutex;
void *g_noalloc_ptr[kMaxDevices] = {};   // device address of g_noalloc_scratch, per device

// Device address of the built-in buffer on the current device. The first call on a
// device looks it up (cudaGetSymbolAddress, with that device current) and caches it.
dendsn_status noalloc_scratch(void **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return fail(DENDSN_ERR_CUDA, "cudaGetDevice failed: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return fail(DENDSN_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (g_noalloc_ptr[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr)
            return fail(DENDSN_ERR_CUDA, "cudaGetSymbolAddress of the built-in scratch failed: %s",
                        cudaGetErrorString(e));
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return DENDSN_OK;
}

}  // namespace

extern "C" dendsn_status dendsn_backward_noalloc(
    const dendsn_config *cfg, const void *x, const float *alpha, const float *xi,
    const float *zeta, const float *kappa, const uint8_t *mask, const void *grad_spikes,
    const float *grad_v, const void *saved, void *grad_x, float *grad_alpha, float *grad_xi,
    float *grad_zeta, float *grad_kappa, void *stream) {
    Plan pl;
    dendsn_status st = make_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (pl.scratch_bytes > kNoAllocScratchBytes)
        return fail(DENDSN_ERR_UNSUPPORTED,
                    "this layer needs %zu bytes of scratch, more than the %zu-byte built-in "
                    "buffer of dendsn_backward_noalloc; use dendsn_backward with a caller buffer",
                    pl.scratch_bytes, kNoAllocScratchBytes);
    void *scratch = nullptr;
    if ((st = noalloc_scratch(&scratch)) != DENDSN_OK) return st;
    // Nothing in the buffer needs to start at zero: the backward kernel writes every
    // partial sum that the finalize kernel then reads, in the same call.
    return dendsn_backward(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                           grad_x, grad_alpha, grad_xi, grad_zeta, grad_kappa, scratch, stream);
}

// ------------------------------------------------------------------ point-neuron LIF layer
namespace {

struct LifPlan {
    int64_t M;
    int n_ck;          // checkpoints (T > 8 only)
    int sx;
};

dendsn_status make_lif_plan(const dendsn_lif_config *cfg, LifPlan *pl) {
    if (cfg == nullptr) return fail(DENDSN_ERR_INVALID_ARG, "cfg is NULL");
    const dendsn_lif_config &c = *cfg;
    if (c.T < 0 || c.B < 0 || c.N < 0)
        return fail(DENDSN_ERR_INVALID_ARG, "negative size (T=%d B=%d N=%d)", c.T, c.B, c.N);
    if (c.x_dtype != DENDSN_F32 && c.x_dtype != DENDSN_BF16)
        return fail(DENDSN_ERR_INVALID_ARG, "bad x_dtype %d", c.x_dtype);
    if ((c.reset != 0 && c.reset != 1) || (c.detach_reset != 0 && c.detach_reset != 1))
        return fail(DENDSN_ERR_INVALID_ARG, "enum/flag field out of range");
    if (!std::isfinite(c.theta) || !std::isfinite(c.beta))
        return fail(DENDSN_ERR_INVALID_ARG, "theta and beta must be finite");
    pl->M = (int64_t)c.B * c.N;
    pl->n_ck = c.T > 8 ? (c.T + 7) / 8 - 1 : 0;
    pl->sx = c.x_dtype == DENDSN_BF16 ? 2 : 4;
    if ((pl->M + 3) / 4 > (int64_t)INT32_MAX * 256) return fail(DENDSN_ERR_UNSUPPORTED, "too many neurons");
    return DENDSN_OK;
}

template <int XT>
cudaError_t lif_dispatch(bool fwd, bool vec, const LifArgs &a, cudaStream_t s) {
    if (fwd) return vec ? launch_lif_forward<XT, 4>(a, s) : launch_lif_forward<XT, 1>(a, s);
    return vec ? launch_lif_backward<XT, 4>(a, s) : launch_lif_backward<XT, 1>(a, s);
}

}  // namespace

extern "C" {

dendsn_status dendsn_lif_workspace_size(const dendsn_lif_config *cfg, size_t *saved_bytes) {
    LifPlan pl;
    dendsn_status st = make_lif_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (saved_bytes) *saved_bytes = ((size_t)pl.n_ck * pl.M * 4 + 15) / 16 * 16;
    return DENDSN_OK;
}

dendsn_status dendsn_lif_forward(const dendsn_lif_config *cfg, const void *x, void *spikes,
                                 float *v_out, void *saved, void *stream) {
    LifPlan pl;
    dendsn_status st = make_lif_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (pl.M == 0 || cfg->T == 0) return DENDSN_OK;
    if (!x || !spikes) return fail(DENDSN_ERR_INVALID_ARG, "x or spikes is NULL");
    if (!aligned(x, pl.sx) || !aligned(spikes, pl.sx) || (v_out && !aligned(v_out, 4)))
        return fail(DENDSN_ERR_MISALIGNED, "x, spikes or v_out misaligned");
    if (saved && !aligned(saved, 16)) return fail(DENDSN_ERR_MISALIGNED, "saved must be 16-byte aligned");
    const bool vec = pl.M % 4 == 0 && aligned(x, 4 * pl.sx) && aligned(spikes, 4 * pl.sx) &&
                     (!v_out || aligned(v_out, 16));
    LifArgs a{};
    a.M = pl.M;
    a.T = cfg->T;
    a.theta = cfg->theta;
    a.beta = cfg->beta;
    a.soft = cfg->reset == DENDSN_RESET_SOFT;
    a.detach_reset = cfg->detach_reset;
    a.x = x;
    a.spikes = spikes;
    a.v_out = v_out;
    a.ck = (saved && pl.n_ck > 0) ? static_cast<float *>(saved) : nullptr;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cfg->x_dtype == DENDSN_BF16 ? lif_dispatch<1>(true, vec, a, s)
                                                : lif_dispatch<0>(true, vec, a, s);
    if (e != cudaSuccess) return fail(DENDSN_ERR_CUDA, "LIF forward launch failed: %s", cudaGetErrorString(e));
    g_launches.fetch_add(1, std::memory_order_relaxed);
    return DENDSN_OK;
}

dendsn_status dendsn_lif_backward(const dendsn_lif_config *cfg, const void *x,
                                  const void *grad_spikes, const float *grad_v,
                                  const void *saved, void *grad_x, void *stream) {
    LifPlan pl;
    dendsn_status st = make_lif_plan(cfg, &pl);
    if (st != DENDSN_OK) return st;
    if (pl.M == 0 || cfg->T == 0) return DENDSN_OK;
    if (!x || !grad_spikes || !grad_x) return fail(DENDSN_ERR_INVALID_ARG, "x, grad_spikes or grad_x is NULL");
    if (!aligned(x, pl.sx) || !aligned(grad_spikes, pl.sx) || !aligned(grad_x, pl.sx) ||
        (grad_v && !aligned(grad_v, 4)))
        return fail(DENDSN_ERR_MISALIGNED, "x, grad_spikes, grad_x or grad_v misaligned");
    if (pl.n_ck > 0 && !saved)
        return fail(DENDSN_ERR_INVALID_ARG, "T=%d needs the forward's saved checkpoints", cfg->T);
    if (saved && !aligned(saved, 16)) return fail(DENDSN_ERR_MISALIGNED, "saved must be 16-byte aligned");
    const bool vec = pl.M % 4 == 0 && aligned(x, 4 * pl.sx) && aligned(grad_spikes, 4 * pl.sx) &&
                     aligned(grad_x, 4 * pl.sx) && (!grad_v || aligned(grad_v, 16));
    LifArgs a{};
    a.M = pl.M;
    a.T = cfg->T;
    a.theta = cfg->theta;
    a.beta = cfg->beta;
    a.soft = cfg->reset == DENDSN_RESET_SOFT;
    a.detach_reset = cfg->detach_reset;
    a.x = x;
    a.ck = pl.n_ck > 0 ? static_cast<float *>(const_cast<void *>(saved)) : nullptr;
    a.gs = grad_spikes;
    a.gv = grad_v;
    a.gx = grad_x;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cfg->x_dtype == DENDSN_BF16 ? lif_dispatch<1>(false, vec, a, s)
                                                : lif_dispatch<0>(false, vec, a, s);
    if (e != cudaSuccess) return fail(DENDSN_ERR_CUDA, "LIF backward launch failed: %s", cudaGetErrorString(e));
    g_launches.fetch_add(1, std::memory_order_relaxed);
    return DENDSN_OK;
}

}  // extern "C"

