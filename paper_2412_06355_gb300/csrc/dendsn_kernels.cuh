// Fused DendSN layer kernels for sm_103a (GB300).
//
// Work decomposition. The B*N neurons of a layer are viewed as a matrix of
// O = B*N/P rows and P = C*inner columns: neuron j = o*P + p sits in row o,
// column p, and its parameter channel is c = p / inner, so every thread keeps
// one column, hence one parameter set, for its whole life. A block is a tile of
// TXn columns x TY row lanes; each neuron is served by LPN adjacent lanes of one
// warp that own KT = K / LPN compartments each (16 bytes of fp32 input per step,
// one 128-bit load). A thread walks R rows of its column; for each row it walks
// the T steps in chunks. The loads of the next chunk (or next row) are issued
// right after the current chunk's values are consumed, so loads stay in flight
// without a second register buffer.
//
// Forward (Eqs. methods-compartment .. methods-lif-fire): V^d, V^s and S stay in
// registers across all T steps; the HBM traffic per step is the K inputs read and
// the spike written (plus an optional V^s write and, when T > L, a checkpoint of
// (V^d, V^s) every L steps).
//
// Backward (BPTT with the arctan surrogate, Eq. methods-sg): chunks are visited
// in reverse; each is recomputed from its checkpoint (or from zero state) with the
// forward's step function, so recomputed potentials and spikes are bit-identical
// to the forward's; then the reverse-time recursion runs in registers and writes
// grad_x. Parameter-gradient partials stay in registers per thread, are reduced
// per channel inside the block in a fixed order (segmented warp shuffles, then
// shared memory), written to scratch, and summed over blocks in a fixed order by a
// finalize kernel: the parameter gradients are deterministic.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dendsn_types.h"

namespace dendsn {

// ---------------------------------------------------------------- element I/O
template <typename XT> struct IO;

template <> struct IO<float> {
    template <int KT>
    static __device__ __forceinline__ void load(const float *p, float (&v)[KT]) {
        if constexpr (KT == 4) {
            float4 q = __ldcs(reinterpret_cast<const float4 *>(p));
            v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
        } else if constexpr (KT == 2) {
            float2 q = __ldcs(reinterpret_cast<const float2 *>(p));
            v[0] = q.x; v[1] = q.y;
        } else {
            v[0] = __ldcs(p);
        }
    }
    template <int KT>
    static __device__ __forceinline__ void store(float *p, const float (&v)[KT]) {
        if constexpr (KT == 4) {
            __stcs(reinterpret_cast<float4 *>(p), make_float4(v[0], v[1], v[2], v[3]));
        } else if constexpr (KT == 2) {
            __stcs(reinterpret_cast<float2 *>(p), make_float2(v[0], v[1]));
        } else {
            __stcs(p, v[0]);
        }
    }
    static __device__ __forceinline__ float load1(const float *p) { return __ldcs(p); }
    static __device__ __forceinline__ void store1(float *p, float v) { __stcs(p, v); }
};

__device__ __forceinline__ float bf16_bits_to_float(uint32_t b16) {
    return __uint_as_float(b16 << 16);   // exact widening
}

template <> struct IO<__nv_bfloat16> {
    using T = __nv_bfloat16;
    template <int KT>
    static __device__ __forceinline__ void load(const T *p, float (&v)[KT]) {
        if constexpr (KT == 4) {
            uint2 q = __ldcs(reinterpret_cast<const uint2 *>(p));
            v[0] = bf16_bits_to_float(q.x & 0xffffu); v[1] = bf16_bits_to_float(q.x >> 16);
            v[2] = bf16_bits_to_float(q.y & 0xffffu); v[3] = bf16_bits_to_float(q.y >> 16);
        } else if constexpr (KT == 2) {
            uint32_t q = __ldcs(reinterpret_cast<const unsigned int *>(p));
            v[0] = bf16_bits_to_float(q & 0xffffu); v[1] = bf16_bits_to_float(q >> 16);
        } else {
            unsigned short q = __ldcs(reinterpret_cast<const unsigned short *>(p));
            v[0] = bf16_bits_to_float(q);
        }
    }
    static __device__ __forceinline__ uint32_t pack2(float a, float b) {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);   // .x = a, the low half
        return *reinterpret_cast<uint32_t *>(&h);
    }
    template <int KT>
    static __device__ __forceinline__ void store(T *p, const float (&v)[KT]) {
        if constexpr (KT == 4) {
            __stcs(reinterpret_cast<uint2 *>(p), make_uint2(pack2(v[0], v[1]), pack2(v[2], v[3])));
        } else if constexpr (KT == 2) {
            __stcs(reinterpret_cast<unsigned int *>(p), pack2(v[0], v[1]));
        } else {
            __nv_bfloat16 h = __float2bfloat16_rn(v[0]);
            __stcs(reinterpret_cast<unsigned short *>(p), *reinterpret_cast<unsigned short *>(&h));
        }
    }
    static __device__ __forceinline__ float load1(const T *p) {
        return bf16_bits_to_float(__ldcs(reinterpret_cast<const unsigned short *>(p)));
    }
    static __device__ __forceinline__ void store1(T *p, float v) {
        __nv_bfloat16 h = __float2bfloat16_rn(v);
        __stcs(reinterpret_cast<unsigned short *>(p), *reinterpret_cast<unsigned short *>(&h));
    }
};

template <int XT> struct XType;
template <> struct XType<0> { using type = float; };
template <> struct XType<1> { using type = __nv_bfloat16; };

// Mask bits of KTb branches of one lane, as 1.0f / 0.0f.
template <int KTb>
__device__ __forceinline__ void load_mask(const uint8_t *m, float (&mk)[KTb]) {
    if constexpr (KTb == 4) {
        const uint32_t q = __ldg(reinterpret_cast<const unsigned int *>(m));
#pragma unroll
        for (int b = 0; b < 4; ++b) mk[b] = ((q >> (8 * b)) & 0xffu) ? 1.f : 0.f;
    } else if constexpr (KTb == 2) {
        const uint32_t q = __ldg(reinterpret_cast<const unsigned short *>(m));
        mk[0] = (q & 0xffu) ? 1.f : 0.f;
        mk[1] = (q >> 8) ? 1.f : 0.f;
    } else {
        mk[0] = __ldg(m) ? 1.f : 0.f;
    }
}

// ---------------------------------------------------------------- the step
// Per-lane parameters of one neuron (KT compartments, KTb = KT/G branches).
template <int KT, int G>
struct LaneParams {
    static constexpr int KTb = KT / G;
    float a[KT];     // alpha (0 for a Stateless Dendrite)
    float xi[KT];
    float iz[KTb];   // 1 / zeta
    float km[KTb];   // kappa * mask
    float mk[KTb];   // mask (0/1)
};

// One compartment + branch step of one lane: advances V^d in place and returns the
// lane's share of Z[t] (Eqs. methods-compartment, -branch-aggregation,
// -mexican-hat, -soma-input, -residual). Explicit rounding intrinsics keep the
// forward kernel and the backward's recompute bit-identical.
template <int KT, int G, int PSI>
__device__ __forceinline__ float dendrite_step(const LaneParams<KT, G> &lp, float (&vd)[KT],
                                               const float (&x)[KT], bool residual,
                                               float inv_k) {
#pragma unroll
    for (int i = 0; i < KT; ++i) vd[i] = __fmaf_rn(lp.a[i], vd[i], x[i]);
    float zp = 0.f;
#pragma unroll
    for (int b = 0; b < KT / G; ++b) {
        float ss = 0.f, u0 = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
            const float u = __fmul_rn(__fsub_rn(vd[b * G + g], lp.xi[b * G + g]), lp.iz[b]);
            if (g == 0) u0 = u;
            ss = __fmaf_rn(u, u, ss);
        }
        float y;
        if constexpr (PSI == PSI_MEXHAT) {
            const float e = expf(__fmul_rn(-0.5f, ss));
            y = __fmaf_rn(-ss, e, e);                     // (1 - r^2) e^{-r^2/2}
        } else {
            y = (G == 1) ? fabsf(u0) : sqrtf(ss);         // r
        }
        zp = __fmaf_rn(lp.km[b], y, zp);
    }
    if (residual) {
        float xs = 0.f;
#pragma unroll
        for (int i = 0; i < KT; ++i) xs = __fadd_rn(xs, x[i]);
        zp = __fmaf_rn(xs, inv_k, zp);
    }
    return zp;
}

// Sum of the LPN lanes' shares (xor butterfly: every lane gets the same bits).
template <int LPN>
__device__ __forceinline__ float lanes_sum(float v) {
    if constexpr (LPN >= 2) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 1));
    if constexpr (LPN >= 4) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 2));
    if constexpr (LPN >= 8) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 4));
    return v;
}

// LIF soma charge with the reset folded in (Eq. methods-lif-reset-charge, or the
// soft variant V = beta (V - theta S) + Z).
__device__ __forceinline__ float soma_charge(float z, float v_prev, float s_prev,
                                             const Params &p) {
    const float leak = p.soft ? __fmaf_rn(-p.theta, s_prev, v_prev)
                              : __fmul_rn(__fsub_rn(1.f, s_prev), v_prev);
    return __fmaf_rn(p.beta, leak, z);
}

__device__ __forceinline__ float fire(float v, float theta) {   // Eq. methods-lif-fire
    return (v >= theta) ? 1.f : 0.f;
}

// Eq. methods-sg: 1 / (1 + pi^2 x^2).
__device__ __forceinline__ float surrogate(float x) {
    const float pi2 = 9.869604401089358f;
    return __frcp_rn(__fmaf_rn(__fmul_rn(pi2, x), x, 1.f));
}

// ---------------------------------------------------------------- thread setup
struct ThreadPos {
    int sub;        // lane within the neuron
    int p;          // column (clamped into range)
    bool active;    // the column exists
    int64_t row0;   // first row of this thread
    int rstride;    // row stride between this thread's rows
    int chan;
};

template <int LPN>
__device__ __forceinline__ ThreadPos thread_pos(const Geometry &g) {
    ThreadPos t;
    const int tid = threadIdx.x;
    t.sub = tid % LPN;
    const int cx = (tid / LPN) % g.TXn;
    const int ry = tid / (LPN * g.TXn);
    const int ct = blockIdx.x % g.nCT;
    const int rg = blockIdx.x / g.nCT;
    const int p = ct * g.TXn + cx;
    t.active = p < g.P;
    t.p = t.active ? p : g.P - 1;
    t.row0 = (int64_t)rg * g.R * g.TY + ry;
    t.rstride = g.TY;
    t.chan = t.p / g.inner;
    return t;
}

template <int KT, int G>
__device__ __forceinline__ void load_lane_params(const Params &P, const Geometry &g, int chan,
                                                 int sub, LaneParams<KT, G> &lp) {
    constexpr int KTb = KT / G;
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const int k = sub * KT + i;
        lp.a[i] = P.stateless ? 0.f : __ldg(P.alpha + (int64_t)chan * g.K + k);
        lp.xi[i] = __ldg(P.xi + (int64_t)chan * g.K + k);
    }
#pragma unroll
    for (int b = 0; b < KTb; ++b) {
        lp.iz[b] = __frcp_rn(__ldg(P.zeta + (int64_t)chan * g.Kb + sub * KTb + b));
        lp.mk[b] = 1.f;
    }
    if (P.mask_mode == 1) load_mask<KTb>(P.mask + (int64_t)chan * g.Kb + sub * KTb, lp.mk);
#pragma unroll
    for (int b = 0; b < KTb; ++b)
        lp.km[b] = __fmul_rn(__ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b), lp.mk[b]);
}

// Per-neuron mask (mask_mode 2): kappa * m for neuron j.
template <int KT, int G>
__device__ __forceinline__ void apply_neuron_mask(const Params &P, const Geometry &g,
                                                  int64_t j, int chan, int sub,
                                                  LaneParams<KT, G> &lp) {
    constexpr int KTb = KT / G;
    const int64_t n = j % g.N;
    load_mask<KTb>(P.mask + n * g.Kb + sub * KTb, lp.mk);
#pragma unroll
    for (int b = 0; b < KTb; ++b)
        lp.km[b] = __fmul_rn(__ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b), lp.mk[b]);
}

// ---------------------------------------------------------------- forward
// One load batch = kFwdBatch steps. Checkpoints every g.L steps (the backward's chunk).
template <int K, int G, int PSI, typename XT>
__global__ void __launch_bounds__(kThreads)
dendsn_forward_kernel(const FwdArgs A) {
    constexpr int KT = (K < 4) ? K : 4;
    constexpr int LPN = K / KT;
    constexpr int L = kFwdBatch;
    const Geometry &g = A.g;
    const ThreadPos pos = thread_pos<LPN>(g);
    LaneParams<KT, G> lp;
    load_lane_params<KT, G>(A.p, g, pos.chan, pos.sub, lp);
    const XT *__restrict__ x = static_cast<const XT *>(A.x);
    XT *__restrict__ spikes = static_cast<XT *>(A.spikes);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nb = (T + L - 1) / L;             // load batches per row (T >= 1 here)
    const int64_t stepX = g.BN * K;             // elements between steps of x
    const bool write_ck = (A.ck_vd != nullptr) && g.n_ck > 0;

    // unit u = (row u / nb, batch u % nb)
    const int64_t nunits = (int64_t)g.R * nb;
    auto unit_row = [&](int64_t u) -> int64_t { return pos.row0 + (u / nb) * pos.rstride; };

    float xb[L][KT];
    {
        const int64_t o = unit_row(0);
        if (o < g.O) {
            const XT *xp = x + (o * g.P + pos.p) * K + pos.sub * KT;
#pragma unroll
            for (int tt = 0; tt < L; ++tt)
                if (tt < T) IO<XT>::template load<KT>(xp + (int64_t)tt * stepX, xb[tt]);
        }
    }
    float vd[KT];
    float v = 0.f, s = 0.f;
    for (int64_t u = 0; u < nunits; ++u) {
        const int64_t o = unit_row(u);
        if (o >= g.O) break;                       // uniform per warp
        const int c = (int)(u % nb);
        const int t0 = c * L;
        const int64_t j = o * g.P + pos.p;
        if (c == 0) {
#pragma unroll
            for (int i = 0; i < KT; ++i) vd[i] = 0.f;
            v = 0.f;
            s = 0.f;
            if (A.p.mask_mode == 2) apply_neuron_mask<KT, G>(A.p, g, j, pos.chan, pos.sub, lp);
        }
        // next unit, for the rolling prefetch
        const int64_t un = u + 1;
        const int64_t on = unit_row(un);
        const bool has_next = (un < nunits) && (on < g.O);
        const int tn = (int)(un % nb) * L;
        const XT *xpn = x + (on * g.P + pos.p) * K + pos.sub * KT + (int64_t)tn * stepX;
#pragma unroll
        for (int tt = 0; tt < L; ++tt) {
            const int t = t0 + tt;
            if (t < T) {
                float xv[KT];
#pragma unroll
                for (int i = 0; i < KT; ++i) xv[i] = xb[tt][i];
                if (has_next && tn + tt < T)
                    IO<XT>::template load<KT>(xpn + (int64_t)tt * stepX, xb[tt]);
                const float z = lanes_sum<LPN>(
                    dendrite_step<KT, G, PSI>(lp, vd, xv, A.p.residual != 0, inv_k));
                v = soma_charge(z, v, s, A.p);
                s = fire(v, A.p.theta);
                if (pos.active) {
                    const int64_t so = (int64_t)t * g.BN + j;
                    if (pos.sub == 0) {
                        IO<XT>::store1(spikes + so, s);
                        if (A.v_out) __stcs(A.v_out + so, v);
                    }
                    if (write_ck && ((t + 1) % g.L) == 0 && t + 1 < T) {
                        const int ck = (t + 1) / g.L - 1;
                        IO<float>::template store<KT>(
                            A.ck_vd + ((int64_t)ck * g.BN + j) * K + pos.sub * KT, vd);
                        if (pos.sub == 0) __stcs(A.ck_vs + (int64_t)ck * g.BN + j, v);
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------- backward
template <int KT, int G>
struct GradAcc {
    static constexpr int KTb = KT / G;
    float ga[KT], gxi[KT], gz[KTb], gk[KTb];
};

// Gradients through the branches of one lane at one step, from V^d[t] (vd) and
// dL/dZ[t] (dz). direct[i] = dL/dV^d_i[t] through this step's branch only.
template <int KT, int G, int PSI>
__device__ __forceinline__ void branch_backward(const LaneParams<KT, G> &lp,
                                                const float (&vd)[KT], float dz,
                                                float (&direct)[KT], GradAcc<KT, G> &acc) {
#pragma unroll
    for (int b = 0; b < KT / G; ++b) {
        float u[G];
        float ss = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
            u[g] = __fmul_rn(__fsub_rn(vd[b * G + g], lp.xi[b * G + g]), lp.iz[b]);
            ss = __fmaf_rn(u[g], u[g], ss);
        }
        const float gy = __fmul_rn(lp.km[b], dz);       // dL/dY_b
        float y, grr;                                    // Y_b and (dL/dr_b) * r_b
        if constexpr (PSI == PSI_MEXHAT) {
            const float e = expf(__fmul_rn(-0.5f, ss));
            y = __fmaf_rn(-ss, e, e);
            // psi'(r) / r = (r^2 - 3) e^{-r^2/2}, so du_i = q u_i with no division
            const float q = __fmul_rn(__fmul_rn(__fsub_rn(ss, 3.f), e), gy);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const float d = __fmul_rn(__fmul_rn(q, u[g]), lp.iz[b]);
                direct[b * G + g] = d;
                acc.gxi[b * G + g] = __fsub_rn(acc.gxi[b * G + g], d);
            }
            grr = __fmul_rn(ss, q);
        } else {
            float r;
            if constexpr (G == 1) {
                r = fabsf(u[0]);
                const float gu = (u[0] > 0.f) ? gy : ((u[0] < 0.f) ? -gy : 0.f);
                const float d = __fmul_rn(gu, lp.iz[b]);
                direct[b] = d;
                acc.gxi[b] = __fsub_rn(acc.gxi[b], d);
            } else {
                r = sqrtf(ss);
                const float q = (r > 0.f) ? __fdiv_rn(gy, r) : 0.f;   // subgradient 0 at r = 0
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const float d = __fmul_rn(__fmul_rn(q, u[g]), lp.iz[b]);
                    direct[b * G + g] = d;
                    acc.gxi[b * G + g] = __fsub_rn(acc.gxi[b * G + g], d);
                }
            }
            y = r;
            grr = __fmul_rn(gy, r);
        }
        acc.gz[b] = __fsub_rn(acc.gz[b], __fmul_rn(grr, lp.iz[b]));
        acc.gk[b] = __fmaf_rn(__fmul_rn(lp.mk[b], y), dz, acc.gk[b]);
    }
}

template <int KT, int G>
constexpr int acc_count() { return 2 * KT + 2 * (KT / G); }

template <int K, int G, int PSI, typename XT, int L>
__global__ void __launch_bounds__(kThreads)
dendsn_backward_kernel(const BwdArgs A) {
    constexpr int KT = (K < 4) ? K : 4;
    constexpr int LPN = K / KT;
    constexpr int KTb = KT / G;
    constexpr int NA = acc_count<KT, G>();
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    LaneParams<KT, G> lp;
    load_lane_params<KT, G>(P, g, pos.chan, pos.sub, lp);
    const XT *__restrict__ x = static_cast<const XT *>(A.x);
    const XT *__restrict__ gsp = static_cast<const XT *>(A.gs);
    XT *__restrict__ gx = static_cast<XT *>(A.gx);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nc = (T + L - 1) / L;              // chunks per row (T >= 1 here)
    const int64_t stepX = g.BN * K;
    const float hard_dvds = -P.beta;             // dV[t+1]/dS[t] = -beta V[t]
    const float soft_dvds = -P.beta * P.theta;   // dV[t+1]/dS[t] = -beta theta

    GradAcc<KT, G> acc;
#pragma unroll
    for (int i = 0; i < KT; ++i) { acc.ga[i] = 0.f; acc.gxi[i] = 0.f; }
#pragma unroll
    for (int b = 0; b < KTb; ++b) { acc.gz[b] = 0.f; acc.gk[b] = 0.f; }

    // unit u = (row u / nc, chunk nc - 1 - u % nc): chunks are visited in reverse
    const int64_t nunits = (int64_t)g.R * nc;
    auto unit_row = [&](int64_t u) -> int64_t { return pos.row0 + (u / nc) * pos.rstride; };
    auto unit_chunk = [&](int64_t u) -> int { return nc - 1 - (int)(u % nc); };

    float xb[L][KT];     // inputs of the current unit (refilled with the next unit's)
    float gsb[L];        // grad_spikes of the current unit
    float ckd[KT];       // checkpoint V^d entering the current unit
    float ckv = 0.f;     // checkpoint V^s entering the current unit
    {
        const int64_t o = unit_row(0);
        if (o < g.O) {
            const int64_t j = o * g.P + pos.p;
            const int c = unit_chunk(0);
            const int t0 = c * L;
            const XT *xp = x + j * K + pos.sub * KT + (int64_t)t0 * stepX;
#pragma unroll
            for (int tt = 0; tt < L; ++tt)
                if (t0 + tt < T) {
                    IO<XT>::template load<KT>(xp + (int64_t)tt * stepX, xb[tt]);
                    gsb[tt] = IO<XT>::load1(gsp + (int64_t)(t0 + tt) * g.BN + j);
                }
            if (c > 0) {
                IO<float>::template load<KT>(A.ck_vd + ((int64_t)(c - 1) * g.BN + j) * K +
                                                 pos.sub * KT, ckd);
                ckv = __ldcs(A.ck_vs + (int64_t)(c - 1) * g.BN + j);
            }
        }
    }

    float Ad[KT];        // dL/dV^d[t+1], carried backwards
    float dvn = 0.f;     // dL/dV^s[t+1]
    for (int64_t u = 0; u < nunits; ++u) {
        const int64_t o = unit_row(u);
        if (o >= g.O) break;                       // uniform per warp
        const int c = unit_chunk(u);
        const int t0 = c * L;
        const int64_t j = o * g.P + pos.p;
        if (c == nc - 1) {                         // new row: adjoints start at zero
#pragma unroll
            for (int i = 0; i < KT; ++i) Ad[i] = 0.f;
            dvn = 0.f;
            if (P.mask_mode == 2) apply_neuron_mask<KT, G>(P, g, j, pos.chan, pos.sub, lp);
        }
        // state entering the chunk: zero at t = 0, else the forward's checkpoint
        float vd0[KT];
        float v0 = 0.f;
#pragma unroll
        for (int i = 0; i < KT; ++i) vd0[i] = (c == 0) ? 0.f : ckd[i];
        if (c > 0) v0 = ckv;
        const float s0 = (c == 0) ? 0.f : fire(v0, P.theta);

        // next unit (rolling prefetch)
        const int64_t un = u + 1;
        const int64_t on = unit_row(un);
        const bool has_next = (un < nunits) && (on < g.O);
        const int cn = unit_chunk(un);
        const int tn = cn * L;
        const int64_t jn = on * g.P + pos.p;
        const XT *xpn = x + jn * K + pos.sub * KT + (int64_t)tn * stepX;
        if (has_next && cn > 0) {
            IO<float>::template load<KT>(A.ck_vd + ((int64_t)(cn - 1) * g.BN + jn) * K +
                                             pos.sub * KT, ckd);
            ckv = __ldcs(A.ck_vs + (int64_t)(cn - 1) * g.BN + jn);
        }

        // recompute the chunk, keeping V^d, V^s and S of every step
        float vdh[L][KT];
        float vsh[L];
        float sh[L];
        float gsc[L];
        {
            float vd[KT];
#pragma unroll
            for (int i = 0; i < KT; ++i) vd[i] = vd0[i];
            float v = v0, s = s0;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                if (t0 + tt < T) {
                    float xv[KT];
#pragma unroll
                    for (int i = 0; i < KT; ++i) xv[i] = xb[tt][i];
                    gsc[tt] = gsb[tt];
                    if (has_next && tn + tt < T) {
                        IO<XT>::template load<KT>(xpn + (int64_t)tt * stepX, xb[tt]);
                        gsb[tt] = IO<XT>::load1(gsp + (int64_t)(tn + tt) * g.BN + jn);
                    }
                    const float z = lanes_sum<LPN>(
                        dendrite_step<KT, G, PSI>(lp, vd, xv, P.residual != 0, inv_k));
                    v = soma_charge(z, v, s, P);
                    s = fire(v, P.theta);
#pragma unroll
                    for (int i = 0; i < KT; ++i) vdh[tt][i] = vd[i];
                    vsh[tt] = v;
                    sh[tt] = s;
                }
            }
        }
        // reverse-time recursion over the chunk
#pragma unroll
        for (int tt = L - 1; tt >= 0; --tt) {
            const int t = t0 + tt;
            if (t < T) {
                const float vs = vsh[tt];
                const float dvds = P.detach ? 0.f : (P.soft ? soft_dvds : __fmul_rn(hard_dvds, vs));
                const float dvdv = P.soft ? P.beta : __fmul_rn(P.beta, __fsub_rn(1.f, sh[tt]));
                const float ds = __fmaf_rn(dvds, dvn, gsc[tt]);                    // dL/dS[t]
                float dv = __fmaf_rn(surrogate(__fsub_rn(vs, P.theta)), ds,
                                     __fmul_rn(dvdv, dvn));                        // dL/dV^s[t]
                if (A.gv) dv = __fadd_rn(dv, __ldcs(A.gv + (int64_t)t * g.BN + j));
                float direct[KT];
                branch_backward<KT, G, PSI>(lp, vdh[tt], dv, direct, acc);
                float gxv[KT];
                const float res = P.residual ? __fmul_rn(dv, inv_k) : 0.f;
#pragma unroll
                for (int i = 0; i < KT; ++i) {
                    Ad[i] = __fmaf_rn(lp.a[i], Ad[i], direct[i]);
                    gxv[i] = __fadd_rn(Ad[i], res);
                    const float vprev = (tt > 0) ? vdh[tt > 0 ? tt - 1 : 0][i] : vd0[i];
                    acc.ga[i] = __fmaf_rn(Ad[i], vprev, acc.ga[i]);
                }
                if (pos.active)
                    IO<XT>::template store<KT>(gx + ((int64_t)t * g.BN + j) * K + pos.sub * KT,
                                               gxv);
                dvn = dv;
            }
        }
    }

    // ---- parameter-gradient partials: per channel, fixed summation order
    float v[NA];
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        v[i] = (pos.active && !P.stateless) ? acc.ga[i] : 0.f;
        v[KT + i] = pos.active ? acc.gxi[i] : 0.f;
    }
#pragma unroll
    for (int b = 0; b < KTb; ++b) {
        v[2 * KT + b] = pos.active ? acc.gz[b] : 0.f;
        v[2 * KT + KTb + b] = pos.active ? acc.gk[b] : 0.f;
    }
    // stage 1: within a warp, columns of one channel come in aligned runs of g.seg
    for (int d = 1; d < g.seg; d <<= 1) {
#pragma unroll
        for (int a = 0; a < NA; ++a)
            v[a] = __fadd_rn(v[a], __shfl_xor_sync(0xffffffffu, v[a], d * LPN));
    }
    // stage 2: run leaders meet in shared memory; red[a][tid]
    extern __shared__ float red[];
#pragma unroll
    for (int a = 0; a < NA; ++a) red[a * kThreads + threadIdx.x] = v[a];
    __syncthreads();
    const int ct = blockIdx.x % g.nCT;
    const int p0 = ct * g.TXn;
    const int p1 = min(p0 + g.TXn, g.P);            // exclusive
    const int c_lo = p0 / g.inner;
    const int nch = (p1 - 1) / g.inner - c_lo + 1;
    const int NP = 2 * g.K + 2 * g.Kb;              // per-channel gradient vector
    float *out = A.partials + (int64_t)blockIdx.x * g.nch_max * NP;
    const int items = nch * LPN * NA;
    for (int w = threadIdx.x; w < items; w += kThreads) {
        const int a = w % NA;
        const int sub = (w / NA) % LPN;
        const int lc = w / (NA * LPN);
        const int c = c_lo + lc;
        const int cx_lo = max(c * g.inner, p0) - p0;
        const int cx_hi = min((c + 1) * g.inner, p1) - p0;
        float sum = 0.f;
        for (int ry = 0; ry < g.TY; ++ry)
            for (int cx = cx_lo; cx < cx_hi; cx += g.seg)
                sum = __fadd_rn(sum, red[a * kThreads + (ry * g.TXn + cx) * LPN + sub]);
        int slot;
        if (a < KT) slot = sub * KT + a;                                        // alpha
        else if (a < 2 * KT) slot = g.K + sub * KT + (a - KT);                  // xi
        else if (a < 2 * KT + KTb) slot = 2 * g.K + sub * KTb + (a - 2 * KT);   // zeta
        else slot = 2 * g.K + g.Kb + sub * KTb + (a - 2 * KT - KTb);            // kappa
        out[lc * NP + slot] = sum;
    }
}

// ---------------------------------------------------------------- launchers
template <int K, int G, int PSI, int XT>
cudaError_t launch_forward(const FwdArgs &a, int blocks, cudaStream_t s) {
    using T = typename XType<XT>::type;
    dendsn_forward_kernel<K, G, PSI, T><<<blocks, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <int K, int G, int PSI, int XT, int L>
cudaError_t launch_backward(const BwdArgs &a, int blocks, cudaStream_t s) {
    using T = typename XType<XT>::type;
    constexpr int KT = (K < 4) ? K : 4;
    const size_t smem = sizeof(float) * acc_count<KT, G>() * kThreads;
    dendsn_backward_kernel<K, G, PSI, T, L><<<blocks, kThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace dendsn
