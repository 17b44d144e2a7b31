// Time-parallel DendSN kernels for narrow layers with long horizons (few neurons, large T,
// e.g. the L5PC fitting neuron: T = 2048, 16 neurons). One warp serves one neuron.
//
// The compartment recursion V^d_i[t] = alpha_i V^d_i[t-1] + X_i[t] (Eq. methods-compartment)
// is linear, so it is scanned in parallel over time: lane l owns the steps
// [l*TB, (l+1)*TB); it first scans its block from a zero state, keeping the end state e and
// alpha^len; a 5-step warp scan composes the blocks ((p2, e2) o (p1, e1) = (p2 p1, p2 e1 + e2))
// and gives every lane the state entering its block; a second pass over the block then
// produces V^d[t] and Z[t] (Eqs. methods-branch-aggregation .. methods-soma-input). Only the
// soma (Eq. methods-lif-reset-charge, -fire) is serial: one fused multiply-add, a compare
// and a select per step, run by every lane of the warp on Z[t] held in shared memory.
//
// The backward recomputes V^d and Z the same way (so spikes match the forward's bit for
// bit), runs the soma's reverse recursion serially (Eq. methods-sg), and then the
// compartment adjoint A_i[t] = direct_i[t] + alpha_i A_i[t+1] - again linear - with the
// same block scan in reverse time. Parameter-gradient partials are reduced over the warp in a
// fixed order and summed per channel by tp_finalize_kernel in neuron order: deterministic.
// Nothing is checkpointed: the forward leaves `saved` untouched.
#include "dendsn_kernels.cuh"

namespace dendsn {

namespace {

template <typename XT>
__device__ __forceinline__ float tp_load(const XT *p) {
    if constexpr (std::is_same<XT, float>::value) return __ldg(p);
    else return bf16_lo(__ldg(reinterpret_cast<const unsigned short *>(p)));
}

template <typename XT>
__device__ __forceinline__ void tp_store(XT *p, float v) {
    if constexpr (std::is_same<XT, float>::value) {
        *p = v;
    } else {
        const __nv_bfloat16 h = __float2bfloat16_rn(v);
        *reinterpret_cast<unsigned short *>(p) = *reinterpret_cast<const unsigned short *>(&h);
    }
}

// The neuron's parameters: every lane holds all K compartments.
template <int K, int G>
struct TpParams {
    static constexpr int Kb = K / G;
    float a[K], nxi[K], iz[Kb], km[Kb], mk[Kb];
    __device__ __forceinline__ void load(const Params &P, const Geometry &g, int64_t n, int chan) {
        load_param_arrays<K, G>(P, g, chan, 0, a, nxi, iz, km, mk);
        if (P.mask_mode == 2) {
            float kap[Kb];                       // km holds kappa itself here (mk = 1)
#pragma unroll
            for (int b = 0; b < Kb; ++b) kap[b] = km[b];
            apply_neuron_mask<Kb>(fetch_neuron_mask<Kb>(P, g, n, 0), kap, km, mk);
        }
    }
};

// Z[t] from V^d[t] (and X[t] for the residual term).
template <int K, int G>
__device__ __forceinline__ float tp_soma_input(const TpParams<K, G> &q, const float (&vd)[K],
                                               const float (&x)[K], int psi, bool residual) {
    constexpr int Kb = K / G;
    float z = 0.f;
#pragma unroll
    for (int b = 0; b < Kb; ++b) {
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < G; ++i) {
            const float u = __fmaf_rn(vd[b * G + i], q.iz[b], q.nxi[b * G + i]);
            ss = (i == 0) ? __fmul_rn(u, u) : __fmaf_rn(u, u, ss);
        }
        float y;
        if (psi == PSI_MEXHAT) {
            const float e = gauss_half(ss);
            y = __fmaf_rn(-ss, e, e);                          // (1 - r^2) e^{-r^2/2}
        } else {
            y = sqrtf(ss);                                     // r
        }
        z = (b == 0) ? __fmul_rn(q.km[b], y) : __fmaf_rn(q.km[b], y, z);
    }
    if (residual) {
        float xs = x[0];
#pragma unroll
        for (int i = 1; i < K; ++i) xs = __fadd_rn(xs, x[i]);
        z = __fmaf_rn(xs, 1.f / (float)K, z);
    }
    return z;
}

// Where a neuron's inputs live: element (t, k) at xn + t * sX + k * ks.
struct TpAddr {
    int64_t xo, sX, ks;
    __device__ __forceinline__ TpAddr(const Geometry &g, int64_t j, int layout) {
        sX = g.BN * g.K;
        if (layout == 0) {
            xo = j * g.K;
            ks = 1;
        } else {
            const int64_t s = j % g.inner;
            xo = (j - s) * g.K + s;
            ks = g.inner;
        }
    }
};

// x of the neuron into shared memory as float [T][K]: each lane fetches steps lane, lane+32,
// ..., a batch of independent loads before the batch's stores (in-order issue would
// otherwise wait on every load before the next).
template <int K, typename XT>
__device__ __forceinline__ void tp_stage_x(const XT *xn, const TpAddr &ad, int T, float *xs) {
    constexpr int NB = K >= 16 ? 2 : (K >= 8 ? 4 : (K >= 4 ? 8 : 16));
    const int lane = threadIdx.x & 31;
    for (int t0 = lane; t0 < T; t0 += 32 * NB) {
        float v[NB][K];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int t = t0 + 32 * b;
            if (t < T) {
                const XT *p = xn + (int64_t)t * ad.sX;
#pragma unroll
                for (int k = 0; k < K; ++k) v[b][k] = tp_load(p + k * ad.ks);
            }
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int t = t0 + 32 * b;
            if (t < T) {
#pragma unroll
                for (int k = 0; k < K; ++k) xs[(int64_t)t * K + k] = v[b][k];
            }
        }
    }
}

// A [T] series of the neuron (stride BN in global memory) into shared memory, batched.
template <typename LoadFn>
__device__ __forceinline__ void tp_stage_series(int T, float *dst, LoadFn load) {
    constexpr int NB = 16;
    const int lane = threadIdx.x & 31;
    for (int t0 = lane; t0 < T; t0 += 32 * NB) {
        float v[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int t = t0 + 32 * b;
            if (t < T) v[b] = load(t);
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int t = t0 + 32 * b;
            if (t < T) dst[t] = v[b];
        }
    }
}

// Passes 1 and 2 of the forward over x staged in `xv` ([T][K]): Z[t] to `zs`; with
// keep_vd, V^d[t] replaces x[t] in `xv` (each lane rewrites only its own steps).
template <int K, int G>
__device__ __forceinline__ void tp_dendrite(const Params &P, const TpParams<K, G> &q, int T,
                                            int psi, float *xv, float *zs, bool keep_vd) {
    const int lane = threadIdx.x & 31;
    const int TB = (T + 31) >> 5;
    const int t0 = min(T, lane * TB), t1 = min(T, t0 + TB);
    const bool stateless = P.stateless != 0;
    const bool residual = P.residual != 0;
    float vd[K];
#pragma unroll
    for (int k = 0; k < K; ++k) vd[k] = 0.f;
    if (!stateless) {
        // pass 1: the block from a zero state
        float e[K], pw[K];
#pragma unroll
        for (int k = 0; k < K; ++k) { e[k] = 0.f; pw[k] = 1.f; }
        for (int t = t0; t < t1; ++t) {
#pragma unroll
            for (int k = 0; k < K; ++k) {
                e[k] = __fmaf_rn(q.a[k], e[k], xv[(int64_t)t * K + k]);
                pw[k] = __fmul_rn(pw[k], q.a[k]);
            }
        }
        // compose the blocks over the lanes (inclusive scan), then shift by one lane
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
#pragma unroll
            for (int k = 0; k < K; ++k) {
                const float pa = __shfl_up_sync(0xffffffffu, pw[k], d);
                const float pe = __shfl_up_sync(0xffffffffu, e[k], d);
                if (lane >= d) {
                    e[k] = __fmaf_rn(pw[k], pe, e[k]);
                    pw[k] = __fmul_rn(pw[k], pa);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const float s = __shfl_up_sync(0xffffffffu, e[k], 1);
            vd[k] = (lane == 0) ? 0.f : s;
        }
    }
    // pass 2: V^d[t] and Z[t] of the block
    for (int t = t0; t < t1; ++t) {
        float x[K];
#pragma unroll
        for (int k = 0; k < K; ++k) {
            x[k] = xv[(int64_t)t * K + k];
            vd[k] = stateless ? x[k] : __fmaf_rn(q.a[k], vd[k], x[k]);
        }
        zs[t] = tp_soma_input<K, G>(q, vd, x, psi, residual);
        if (keep_vd) {
#pragma unroll
            for (int k = 0; k < K; ++k) xv[(int64_t)t * K + k] = vd[k];
        }
    }
}

// One soma step (Eq. methods-lif-reset-charge) shaped for a short dependency chain. Hard
// reset: keep = 1.0 while V < theta (PTX set.lt gives the float, no predicate), then
// V' = keep * (beta V) + Z, so the compare and beta V both start from V (measured 16% faster
// than a compare-and-select). Soft reset: V' = beta (V - theta S) + Z.
__device__ __forceinline__ float tp_keep(float v, float theta) {
    float k;
    asm("set.lt.f32.f32 %0, %1, %2;" : "=f"(k) : "f"(v), "f"(theta));
    return k;
}

template <bool SOFT>
__device__ __forceinline__ float tp_charge(float z, float v, float beta, float theta) {
    if constexpr (SOFT) return __fmaf_rn(beta, (v >= theta) ? __fsub_rn(v, theta) : v, z);
    return __fmaf_rn(tp_keep(v, theta), __fmul_rn(beta, v), z);
}

// Serial soma over Z[t] in `zs`, V^s[t] to `vs`. Every lane runs it and writes the same
// values; Z is read a block of 8 steps ahead and V written a block behind, so only the
// charge/threshold chain is on the critical path.
template <bool SOFT>
__device__ __forceinline__ void tp_soma_loop(const float beta, const float theta, const float *zs,
                                             float *vs, int T) {
    constexpr int U = 8;
    if (T <= 0) return;
    // V^s[0] = beta * 0 + Z[0] = Z[0] (no spike before the first step, whatever theta)
    float v = zs[0];
    vs[0] = v;
    const int Tu = 1 + (T - 1) / U * U;                // steps 1 .. Tu-1 in blocks of U
    float zn[U];
#pragma unroll
    for (int i = 0; i < U; ++i) zn[i] = (1 + i < Tu) ? zs[1 + i] : 0.f;
    for (int t = 1; t < Tu; t += U) {
        float z[U], out[U];
#pragma unroll
        for (int i = 0; i < U; ++i) z[i] = zn[i];
        if (t + U < Tu) {
#pragma unroll
            for (int i = 0; i < U; ++i) zn[i] = zs[t + U + i];
        }
#pragma unroll
        for (int i = 0; i < U; ++i) {
            v = tp_charge<SOFT>(z[i], v, beta, theta);
            out[i] = v;
        }
#pragma unroll
        for (int i = 0; i < U; ++i) vs[t + i] = out[i];
    }
    for (int t = Tu; t < T; ++t) {
        v = tp_charge<SOFT>(zs[t], v, beta, theta);
        vs[t] = v;
    }
}

__device__ __forceinline__ void tp_soma(const Params &P, const float *zs, float *vs, int T) {
    if (P.soft) tp_soma_loop<true>(P.beta, P.theta, zs, vs, T);
    else tp_soma_loop<false>(P.beta, P.theta, zs, vs, T);
    __syncwarp();
}

template <int K, int G, typename XT>
__global__ void __launch_bounds__(32) tp_forward_kernel(const FwdArgs A, int psi, int layout) {
    const Geometry &g = A.g;
    const Params &P = A.p;
    const int64_t j = blockIdx.x;                      // the neuron
    const int lane = threadIdx.x;
    const int64_t n = j % g.N;
    const int chan = (int)((n / g.inner) % g.C);
    TpParams<K, G> q;
    q.load(P, g, n, chan);
    const TpAddr ad(g, j, layout);
    extern __shared__ float tp_smem[];
    float *xv = tp_smem;                               // [T][K]: x, then V^s in [T]
    float *zs = xv + (int64_t)g.T * K;                 // [T]: Z
    tp_stage_x<K, XT>(static_cast<const XT *>(A.x) + ad.xo, ad, g.T, xv);
    __syncwarp();
    tp_dendrite<K, G>(P, q, g.T, psi, xv, zs, false);
    __syncwarp();
    tp_soma(P, zs, xv, g.T);
    XT *sp = static_cast<XT *>(A.spikes) + j;
    for (int t = lane; t < g.T; t += 32) {
        const float v = xv[t];
        Scalar<XT>::store_spike(sp + (int64_t)t * g.BN, v >= P.theta);   // Eq. methods-lif-fire
        if (A.v_out) A.v_out[(int64_t)t * g.BN + j] = v;
    }
}

template <int K, int G, typename XT, bool BETA>
__global__ void __launch_bounds__(32) tp_backward_kernel(const BwdArgs A, int psi, int layout) {
    constexpr int Kb = K / G;
    constexpr int NP = 2 * K + 2 * Kb + 1;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const int T = g.T;
    const int64_t j = blockIdx.x;
    const int lane = threadIdx.x;
    const int64_t n = j % g.N;
    const int chan = (int)((n / g.inner) % g.C);
    TpParams<K, G> q;
    q.load(P, g, n, chan);
    const TpAddr ad(g, j, layout);
    extern __shared__ float tp_smem[];
    float *vdh = tp_smem;                              // [T][K]: x, then V^d
    float *zsb = vdh + (int64_t)T * K;                 // [T] Z
    float *vs = zsb + T;                               // [T] V^s
    float *gsb = vs + T;                               // [T] dL/dS
    float *dz = gsb + T;                               // [T] dL/dZ
    float *gvb = dz + T;                               // [T] dL/dV^s (when given)
    const bool has_gv = A.gv != nullptr;
    tp_stage_x<K, XT>(static_cast<const XT *>(A.x) + ad.xo, ad, T, vdh);
    const XT *gsp = static_cast<const XT *>(A.gs) + j;
    tp_stage_series(T, gsb, [&](int t) {
        return Scalar<XT>::unpack(Scalar<XT>::load(gsp + (int64_t)t * g.BN));
    });
    if (has_gv) tp_stage_series(T, gvb, [&](int t) { return __ldg(A.gv + (int64_t)t * g.BN + j); });
    __syncwarp();
    tp_dendrite<K, G>(P, q, T, psi, vdh, zsb, true);
    __syncwarp();
    tp_soma(P, zsb, vs, T);
    // soma, reverse time (Eq. methods-sg). Given the forward trajectory the recursion is
    // linear in dL/dV: dv[t] = k1[t] + k2[t] dv[t+1] with k1 = sg (dL/dS) (+ dL/dV^s) and
    // k2 = sg dV[t+1]/dS[t] + dV[t+1]/dV[t], so it is scanned over time like the
    // compartments: per-step coefficients in parallel, block scans, a warp scan of the blocks.
    const float kv = (P.detach || P.soft) ? 0.f : -P.beta;
    const float cs = (P.detach || !P.soft) ? 0.f : -P.beta * P.theta;
    const float b_spike = P.soft ? P.beta : 0.f;
    const int TB = (T + 31) >> 5;
    const int t0 = min(T, lane * TB), t1 = min(T, t0 + TB);
    float *k1 = zsb;                                   // Z is no longer needed
    float *k2 = dz;
    for (int t = t0; t < t1; ++t) {
        const float v = vs[t];
        const float sg = surrogate(__fsub_rn(v, P.theta));
        const float dvds = __fmaf_rn(kv, v, cs);                         // dV[t+1]/dS[t]
        const float dvdv = (v >= P.theta) ? b_spike : P.beta;            // dV[t+1]/dV[t]
        k1[t] = has_gv ? __fmaf_rn(sg, gsb[t], gvb[t]) : __fmul_rn(sg, gsb[t]);
        k2[t] = __fmaf_rn(sg, dvds, dvdv);
    }
    {
        float e = 0.f, pw = 1.f;                       // the block from dv[t1] = 0
        for (int t = t1 - 1; t >= t0; --t) {
            e = __fmaf_rn(k2[t], e, k1[t]);
            pw = __fmul_rn(pw, k2[t]);
        }
#pragma unroll
        for (int dl = 1; dl < 32; dl <<= 1) {
            const float pa = __shfl_down_sync(0xffffffffu, pw, dl);
            const float pe = __shfl_down_sync(0xffffffffu, e, dl);
            if (lane + dl < 32) {
                e = __fmaf_rn(pw, pe, e);
                pw = __fmul_rn(pw, pa);
            }
        }
        const float nx = __shfl_down_sync(0xffffffffu, e, 1);
        float dvn = (lane == 31) ? 0.f : nx;           // dL/dV^s at the block's end
        __syncwarp();
        for (int t = t1 - 1; t >= t0; --t) {
            dvn = __fmaf_rn(k2[t], dvn, k1[t]);
            dz[t] = dvn;                               // k2[t] read before, own steps only
        }
    }
    __syncwarp();
    float gbeta = 0.f;                                 // sum of dL/dV[t+1] dV[t+1]/dbeta
    if constexpr (BETA) {
        for (int t = t0; t < t1; ++t) {
            if (t + 1 < T) {
                const float v = vs[t];
                const bool st = v >= P.theta;
                const float leak = st ? (P.soft ? __fsub_rn(v, P.theta) : 0.f) : v;
                gbeta = __fmaf_rn(dz[t + 1], leak, gbeta);
            }
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) gbeta = __fadd_rn(gbeta, __shfl_xor_sync(0xffffffffu, gbeta, d));
    }

    // dendrite, reverse time: direct_i[t] from V^d[t] and dL/dZ[t]; A_i[t] = direct_i[t] +
    // alpha_i A_i[t+1] scanned over the lanes' blocks like the forward
    const bool stateless = P.stateless != 0;
    const float inv_k = 1.f / (float)K;
    float gxi[K], gz[Kb], gk[Kb], ga[K];
#pragma unroll
    for (int k = 0; k < K; ++k) { gxi[k] = 0.f; ga[k] = 0.f; }
#pragma unroll
    for (int b = 0; b < Kb; ++b) { gz[b] = 0.f; gk[b] = 0.f; }
    // dL/dV^d[t] directly through Z[t] (and the parameter terms when `acc`)
    auto direct = [&](int t, float (&d)[K], bool acc) {
        const float dzt = dz[t];
#pragma unroll
        for (int b = 0; b < Kb; ++b) {
            float u[G];
            float ss = 0.f;
#pragma unroll
            for (int i = 0; i < G; ++i) {
                u[i] = __fmaf_rn(vdh[(int64_t)t * K + b * G + i], q.iz[b], q.nxi[b * G + i]);
                ss = (i == 0) ? __fmul_rn(u[i], u[i]) : __fmaf_rn(u[i], u[i], ss);
            }
            const float gy = __fmul_rn(q.km[b], dzt);
            float y, qq;                                    // Y_b; dL/du_i = qq u_i
            if (psi == PSI_MEXHAT) {
                const float e = gauss_half(ss);
                y = __fmaf_rn(-ss, e, e);
                qq = __fmul_rn(__fmul_rn(__fsub_rn(ss, 3.f), e), gy);   // psi'(r) / r
            } else {
                const float r = sqrtf(ss);
                y = r;
                qq = (r > 0.f) ? __fdiv_rn(gy, r) : 0.f;                // subgradient 0 at r = 0
            }
#pragma unroll
            for (int i = 0; i < G; ++i) d[b * G + i] = __fmul_rn(__fmul_rn(qq, u[i]), q.iz[b]);
            if (acc) {
#pragma unroll
                for (int i = 0; i < G; ++i) gxi[b * G + i] = __fsub_rn(gxi[b * G + i], d[b * G + i]);
                gz[b] = __fmaf_rn(-__fmul_rn(ss, qq), q.iz[b], gz[b]);  // -(dL/dr) r / zeta
                gk[b] = __fmaf_rn(__fmul_rn(q.mk[b], y), dzt, gk[b]);
            }
        }
    };
    float carry[K];
#pragma unroll
    for (int k = 0; k < K; ++k) carry[k] = 0.f;
    if (!stateless) {
        float e[K], pw[K];
#pragma unroll
        for (int k = 0; k < K; ++k) { e[k] = 0.f; pw[k] = 1.f; }
        for (int t = t1 - 1; t >= t0; --t) {
            float d[K];
            direct(t, d, false);
#pragma unroll
            for (int k = 0; k < K; ++k) {
                e[k] = __fmaf_rn(q.a[k], e[k], d[k]);
                pw[k] = __fmul_rn(pw[k], q.a[k]);
            }
        }
        // compose the blocks from the right: S_l = e_l + pw_l S_{l+1}
#pragma unroll
        for (int dl = 1; dl < 32; dl <<= 1) {
#pragma unroll
            for (int k = 0; k < K; ++k) {
                const float pa = __shfl_down_sync(0xffffffffu, pw[k], dl);
                const float pe = __shfl_down_sync(0xffffffffu, e[k], dl);
                if (lane + dl < 32) {
                    e[k] = __fmaf_rn(pw[k], pe, e[k]);
                    pw[k] = __fmul_rn(pw[k], pa);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const float s = __shfl_down_sync(0xffffffffu, e[k], 1);
            carry[k] = (lane == 31) ? 0.f : s;                         // A at the block's end
        }
    }
    XT *gxn = static_cast<XT *>(A.gx) + ad.xo;
    const bool residual = P.residual != 0;
    for (int t = t1 - 1; t >= t0; --t) {
        float d[K];
        direct(t, d, true);
        const float res = residual ? __fmul_rn(dz[t], inv_k) : 0.f;
        XT *p = gxn + (int64_t)t * ad.sX;
#pragma unroll
        for (int k = 0; k < K; ++k) {
            carry[k] = stateless ? d[k] : __fmaf_rn(q.a[k], carry[k], d[k]);
            tp_store(p + k * ad.ks, residual ? __fadd_rn(carry[k], res) : carry[k]);
            if (!stateless && t > 0) ga[k] = __fmaf_rn(carry[k], vdh[(int64_t)(t - 1) * K + k], ga[k]);
        }
    }
    // the warp's partial sums, in a fixed order, then one row per neuron
    float vals[NP];
#pragma unroll
    for (int k = 0; k < K; ++k) { vals[k] = ga[k]; vals[K + k] = gxi[k]; }
#pragma unroll
    for (int b = 0; b < Kb; ++b) { vals[2 * K + b] = gz[b]; vals[2 * K + Kb + b] = gk[b]; }
    vals[NP - 1] = 0.f;
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
#pragma unroll
        for (int v = 0; v < NP - 1; ++v) vals[v] = __fadd_rn(vals[v], __shfl_xor_sync(0xffffffffu, vals[v], d));
    }
    if (lane == 0) {
        vals[NP - 1] = BETA ? gbeta : 0.f;
        float *out = A.partials + j * NP;
#pragma unroll
        for (int v = 0; v < NP; ++v) out[v] = vals[v];
    }
}

// Per channel, the neurons' partials summed in neuron order.
__global__ void tp_finalize_kernel(const FinArgs F) {
    const Geometry &g = F.g;
    const int NP = 2 * g.K + 2 * g.Kb + 1;
    const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (w >= (int64_t)g.C * NP) return;
    const int c = (int)(w / NP);
    const int q = (int)(w % NP);
    float sum = 0.f;
    if (g.T > 0) {
        for (int64_t j = 0; j < g.BN; ++j) {
            const int64_t nn = j % g.N;
            if ((int)((nn / g.inner) % g.C) == c) sum = __fadd_rn(sum, F.partials[j * NP + q]);
        }
    }
    if (q < g.K) F.g_alpha[(int64_t)c * g.K + q] = F.stateless ? 0.f : sum;
    else if (q < 2 * g.K) F.g_xi[(int64_t)c * g.K + (q - g.K)] = sum;
    else if (q < 2 * g.K + g.Kb) F.g_zeta[(int64_t)c * g.Kb + (q - 2 * g.K)] = sum;
    else if (q < 2 * g.K + 2 * g.Kb) F.g_kappa[(int64_t)c * g.Kb + (q - 2 * g.K - g.Kb)] = sum;
    else if (F.g_beta) F.g_beta[c] = sum;
}

}  // namespace

size_t tp_smem_bytes(int T, int K, bool backward) {
    return sizeof(float) * (size_t)T * ((size_t)K + (backward ? 5 : 1));
}

template <int K, int G, int XT>
cudaError_t launch_forward_tp(const FwdArgs &a, int psi, int layout, cudaStream_t s) {
    using T = typename XType<XT>::type;
    const size_t smem = tp_smem_bytes(a.g.T, K, false);
    cudaError_t e = allow_smem(tp_forward_kernel<K, G, T>, smem);
    if (e != cudaSuccess) return e;
    tp_forward_kernel<K, G, T><<<(unsigned)a.g.BN, 32, smem, s>>>(a, psi, layout);
    return cudaGetLastError();
}

template <int K, int G, int XT>
cudaError_t launch_backward_tp(const BwdArgs &a, int psi, int layout, cudaStream_t s) {
    using T = typename XType<XT>::type;
    const size_t smem = tp_smem_bytes(a.g.T, K, true);
    if (a.want_beta) {
        cudaError_t e = allow_smem(tp_backward_kernel<K, G, T, true>, smem);
        if (e != cudaSuccess) return e;
        tp_backward_kernel<K, G, T, true><<<(unsigned)a.g.BN, 32, smem, s>>>(a, psi, layout);
    } else {
        cudaError_t e = allow_smem(tp_backward_kernel<K, G, T, false>, smem);
        if (e != cudaSuccess) return e;
        tp_backward_kernel<K, G, T, false><<<(unsigned)a.g.BN, 32, smem, s>>>(a, psi, layout);
    }
    return cudaGetLastError();
}

cudaError_t launch_finalize_tp(const FinArgs &a, cudaStream_t s) {
    const int64_t n = (int64_t)a.g.C * (2 * a.g.K + 2 * a.g.Kb + 1);
    tp_finalize_kernel<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(a);
    return cudaGetLastError();
}

#define DENDSN_TP_INST(K, G)                                                                    \
    template cudaError_t launch_forward_tp<K, G, 0>(const FwdArgs &, int, int, cudaStream_t);  \
    template cudaError_t launch_forward_tp<K, G, 1>(const FwdArgs &, int, int, cudaStream_t);  \
    template cudaError_t launch_backward_tp<K, G, 0>(const BwdArgs &, int, int, cudaStream_t); \
    template cudaError_t launch_backward_tp<K, G, 1>(const BwdArgs &, int, int, cudaStream_t);
DENDSN_KG_LIST(DENDSN_TP_INST)
#undef DENDSN_TP_INST

}  // namespace dendsn
