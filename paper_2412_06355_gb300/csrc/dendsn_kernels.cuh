// Fused DendSN layer kernels for sm_103a (GB300).
//
// Work decomposition. The B*N neurons of a layer are viewed as a matrix of
// O = B*N/P rows and P = C*inner columns: neuron j = o*P + p sits in row o,
// column p, and its parameter channel is c = p / inner, so every thread keeps
// one column, hence one parameter set, for its whole life. A block is a tile of
// TXn columns x TY row lanes; each neuron is served by LPN adjacent lanes of one
// warp that own KT = K / LPN compartments each (16 bytes of fp32 input per step,
// one 128-bit load). A thread walks up to R rows of its column; for each row it
// walks the T steps in chunks. The loads of the next chunk (or next row) are
// issued right after the current chunk's values are taken, so loads stay in
// flight without a second register buffer.
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
//
// The loop nests use 32-bit counters and pointer increments; the only 64-bit
// divisions happen once per thread.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "dendsn_types.h"

namespace dendsn {

// ---------------------------------------------------------------- element I/O
// A lane's KT inputs of one step are kept in their stored form (Raw) until used.
template <typename XT, int KT> struct Vec;

template <int KT> struct Vec<float, KT> {
    using Raw = typename std::conditional<KT == 4, float4,
                typename std::conditional<KT == 2, float2, float>::type>::type;
    static __device__ __forceinline__ Raw load(const float *p) {
        return __ldcs(reinterpret_cast<const Raw *>(p));
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) {
        if constexpr (KT == 4) { v[0] = r.x; v[1] = r.y; v[2] = r.z; v[3] = r.w; }
        else if constexpr (KT == 2) { v[0] = r.x; v[1] = r.y; }
        else { v[0] = r; }
    }
    static __device__ __forceinline__ void store(float *p, const float (&v)[KT]) {
        if constexpr (KT == 4) __stcs(reinterpret_cast<float4 *>(p), make_float4(v[0], v[1], v[2], v[3]));
        else if constexpr (KT == 2) __stcs(reinterpret_cast<float2 *>(p), make_float2(v[0], v[1]));
        else __stcs(p, v[0]);
    }
};

__device__ __forceinline__ float bf16_lo(uint32_t q) { return __uint_as_float(q << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t q) { return __uint_as_float(q & 0xffff0000u); }
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);   // .x = lo, the low half
    return *reinterpret_cast<uint32_t *>(&h);
}

template <int KT> struct Vec<__nv_bfloat16, KT> {
    using T = __nv_bfloat16;
    using Raw = typename std::conditional<KT == 4, uint2,
                typename std::conditional<KT == 2, unsigned int, unsigned short>::type>::type;
    static __device__ __forceinline__ Raw load(const T *p) {
        return __ldcs(reinterpret_cast<const Raw *>(p));
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) {   // exact
        if constexpr (KT == 4) { v[0] = bf16_lo(r.x); v[1] = bf16_hi(r.x); v[2] = bf16_lo(r.y); v[3] = bf16_hi(r.y); }
        else if constexpr (KT == 2) { v[0] = bf16_lo(r); v[1] = bf16_hi(r); }
        else { v[0] = bf16_lo(r); }
    }
    static __device__ __forceinline__ void store(T *p, const float (&v)[KT]) {
        if constexpr (KT == 4) {
            __stcs(reinterpret_cast<uint2 *>(p), make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3])));
        } else if constexpr (KT == 2) {
            __stcs(reinterpret_cast<unsigned int *>(p), pack_bf16x2(v[0], v[1]));
        } else {
            __nv_bfloat16 h = __float2bfloat16_rn(v[0]);
            __stcs(reinterpret_cast<unsigned short *>(p), *reinterpret_cast<unsigned short *>(&h));
        }
    }
};

// Scalar (one value per neuron and step) elements: spikes, grad_spikes.
template <typename XT> struct Scalar;
template <> struct Scalar<float> {
    using Raw = float;
    static __device__ __forceinline__ Raw load(const float *p) { return __ldcs(p); }
    static __device__ __forceinline__ float unpack(Raw r) { return r; }
    static __device__ __forceinline__ void store_spike(float *p, bool s) { __stcs(p, s ? 1.f : 0.f); }
};
template <> struct Scalar<__nv_bfloat16> {
    using Raw = unsigned short;
    static __device__ __forceinline__ Raw load(const __nv_bfloat16 *p) {
        return __ldcs(reinterpret_cast<const unsigned short *>(p));
    }
    static __device__ __forceinline__ float unpack(Raw r) { return bf16_lo(r); }
    static __device__ __forceinline__ void store_spike(__nv_bfloat16 *p, bool s) {
        __stcs(reinterpret_cast<unsigned short *>(p), (unsigned short)(s ? 0x3f80u : 0u));
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

// ---------------------------------------------------------------- arithmetic
// 2^x with the hardware approximation (PTX ex2.approx.ftz.f32: relative error a
// few units in the last place; results below 2^-126 flush to zero).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// 1/x with the hardware approximation (PTX rcp.approx.ftz.f32, about 1 ulp).
__device__ __forceinline__ float fast_rcp(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// e^{-r^2/2} = 2^{r^2 * (-log2(e) / 2)}. The product's rounding perturbs the result
// by at most |r^2 log2(e) / 2| * 2^-24 relative, below 1e-6 wherever the Mexican hat
// is not negligibly small.
constexpr float kNegHalfLog2e = -0.72134752044448170368f;
__device__ __forceinline__ float gauss_half(float ss) { return fast_exp2(__fmul_rn(kNegHalfLog2e, ss)); }

// Eq. methods-sg: 1 / (1 + pi^2 x^2).
__device__ __forceinline__ float surrogate(float x) {
    const float pi2 = 9.869604401089358f;
    return fast_rcp(__fmaf_rn(__fmul_rn(pi2, x), x, 1.f));
}

// ---------------------------------------------------------------- the step
// Per-lane parameters of one neuron (KT compartments, KTb = KT/G branches).
template <int KT, int G>
struct LaneParams {
    static constexpr int KTb = KT / G;
    float a[KT];     // alpha (0 for a Stateless Dendrite)
    float nxi[KT];   // -xi / zeta
    float iz[KTb];   // 1 / zeta
    float km[KTb];   // kappa * mask
    float mk[KTb];   // mask (0/1)
};

// Affine input of compartment i: u = (V^d - xi) / zeta, evaluated as V^d/zeta - xi/zeta.
template <int KT, int G>
__device__ __forceinline__ float affine(const LaneParams<KT, G> &lp, float vd, int i) {
    return __fmaf_rn(vd, lp.iz[i / G], lp.nxi[i]);
}

// One compartment + branch step of one lane: advances V^d in place, stores the
// branch Gaussians e^{-r^2/2} (Mexican hat only) in eb, and returns the lane's share
// of Z[t] (Eqs. methods-compartment, -branch-aggregation, -mexican-hat,
// -soma-input, -residual). Explicit rounding intrinsics keep the forward kernel and
// the backward's recompute bit-identical.
template <int KT, int G, int PSI>
__device__ __forceinline__ float dendrite_step(const LaneParams<KT, G> &lp, float (&vd)[KT],
                                               const float (&x)[KT], bool residual, float inv_k,
                                               float (&eb)[KT / G]) {
#pragma unroll
    for (int i = 0; i < KT; ++i) vd[i] = __fmaf_rn(lp.a[i], vd[i], x[i]);
    float zp = 0.f;
#pragma unroll
    for (int b = 0; b < KT / G; ++b) {
        float ss = 0.f, u0 = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
            const float u = affine(lp, vd[b * G + g], b * G + g);
            if (g == 0) u0 = u;
            ss = (g == 0) ? __fmul_rn(u, u) : __fmaf_rn(u, u, ss);
        }
        float y;
        if constexpr (PSI == PSI_MEXHAT) {
            const float e = gauss_half(ss);
            eb[b] = e;
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

// LIF soma charge with the reset folded in: hard V = beta (1 - S) V + Z
// (Eq. methods-lif-reset-charge; (1 - S) V is exactly 0 or V), soft V = beta (V - theta S) + Z.
__device__ __forceinline__ float soma_charge(float z, float v_prev, bool s_prev, const Params &p) {
    const float leak = p.soft ? (s_prev ? __fsub_rn(v_prev, p.theta) : v_prev)
                              : (s_prev ? 0.f : v_prev);
    return __fmaf_rn(p.beta, leak, z);
}

// ---------------------------------------------------------------- thread setup
struct ThreadPos {
    int sub;        // lane within the neuron
    int p;          // column (clamped into range)
    bool active;    // the column exists
    int64_t row0;   // first row of this thread
    int rstride;    // row stride between this thread's rows
    int nrows;      // rows this thread walks (0 .. R)
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
    const int64_t left = g.O - t.row0;
    t.nrows = left <= 0 ? 0 : (int)min((int64_t)g.R, (left + g.TY - 1) / g.TY);
    t.chan = t.p / g.inner;
    return t;
}

template <int KT, int G>
__device__ __forceinline__ void load_lane_params(const Params &P, const Geometry &g, int chan,
                                                 int sub, LaneParams<KT, G> &lp) {
    constexpr int KTb = KT / G;
#pragma unroll
    for (int b = 0; b < KTb; ++b) {
        lp.iz[b] = __frcp_rn(__ldg(P.zeta + (int64_t)chan * g.Kb + sub * KTb + b));
        lp.mk[b] = 1.f;
    }
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const int k = sub * KT + i;
        lp.a[i] = P.stateless ? 0.f : __ldg(P.alpha + (int64_t)chan * g.K + k);
        lp.nxi[i] = -__fmul_rn(__ldg(P.xi + (int64_t)chan * g.K + k), lp.iz[i / G]);
    }
    if (P.mask_mode == 1) load_mask<KTb>(P.mask + (int64_t)chan * g.Kb + sub * KTb, lp.mk);
#pragma unroll
    for (int b = 0; b < KTb; ++b)
        lp.km[b] = __fmul_rn(__ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b), lp.mk[b]);
}

// Per-neuron mask (mask_mode 2): kappa * m for the neuron in column p of row o.
template <int KT, int G>
__device__ __forceinline__ void apply_neuron_mask(const Params &P, const Geometry &g,
                                                  int64_t o, int p, int chan, int sub,
                                                  LaneParams<KT, G> &lp) {
    constexpr int KTb = KT / G;
    const int64_t n = (o * g.P + p) % g.N;
    load_mask<KTb>(P.mask + n * g.Kb + sub * KTb, lp.mk);
#pragma unroll
    for (int b = 0; b < KTb; ++b)
        lp.km[b] = __fmul_rn(__ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b), lp.mk[b]);
}

// ---------------------------------------------------------------- forward
// One load batch = kFwdBatch steps; checkpoints every g.L steps (g.L is a power of
// two and a multiple of the batch, so they fall on batch ends).
template <int K, int G, int PSI, typename XT>
__global__ void __launch_bounds__(kThreads, 3)
dendsn_forward_kernel(const FwdArgs A) {
    constexpr int KT = (K < 4) ? K : 4;
    constexpr int LPN = K / KT;
    constexpr int KTb = KT / G;
    constexpr int L = kFwdBatch;
    using V = Vec<XT, KT>;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    if (pos.nrows == 0) return;                  // whole warps: rows are uniform per warp
    LaneParams<KT, G> lp;
    load_lane_params<KT, G>(P, g, pos.chan, pos.sub, lp);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nb = (T + L - 1) / L;              // load batches per row
    const int64_t stepX = g.BN * K;              // elements between steps of x
    const int64_t j0 = pos.row0 * g.P + pos.p;   // first neuron of this thread
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const XT *__restrict__ x0 = static_cast<const XT *>(A.x) + j0 * K + pos.sub * KT;
    XT *__restrict__ s0 = static_cast<XT *>(A.spikes) + j0;
    const bool write_ck = (A.ck_vd != nullptr) && g.n_ck > 0;
    const bool store = pos.active && pos.sub == 0;

    typename V::Raw xb[L];
#pragma unroll
    for (int tt = 0; tt < L; ++tt)
        if (tt < T) xb[tt] = V::load(x0 + tt * stepX);

    for (int i = 0; i < pos.nrows; ++i) {
        const XT *xr = x0 + i * jstep * K;
        const int64_t j = j0 + i * jstep;
        if (P.mask_mode == 2)
            apply_neuron_mask<KT, G>(P, g, pos.row0 + (int64_t)i * pos.rstride, pos.p, pos.chan,
                                     pos.sub, lp);
        float vd[KT];
#pragma unroll
        for (int k = 0; k < KT; ++k) vd[k] = 0.f;
        float v = 0.f;
        bool s = false;
        for (int c = 0; c < nb; ++c) {
            const int t0 = c * L;
            const bool same_row = c + 1 < nb;
            const bool has_next = same_row || (i + 1 < pos.nrows);
            const int tn = same_row ? t0 + L : 0;
            const XT *xn = same_row ? xr + tn * stepX : xr + jstep * K;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float xv[KT];
                V::unpack(xb[tt], xv);
                // refill slot tt for the next unit right after its value is taken
                if (has_next && tn + tt < T) xb[tt] = V::load(xn + tt * stepX);
                const int t = t0 + tt;
                if (t < T) {
                    float eb[KTb];
                    const float z = lanes_sum<LPN>(
                        dendrite_step<KT, G, PSI>(lp, vd, xv, P.residual != 0, inv_k, eb));
                    v = soma_charge(z, v, s, P);
                    s = v >= P.theta;                      // Eq. methods-lif-fire
                    if (store) {
                        Scalar<XT>::store_spike(s0 + t * g.BN + i * jstep, s);
                        if (A.v_out) __stcs(A.v_out + t * g.BN + j, v);
                    }
                }
            }
            if (write_ck && t0 + L < T && ((t0 + L) & (g.L - 1)) == 0 && pos.active) {
                const int ck = (t0 + L) / g.L - 1;
                Vec<float, KT>::store(A.ck_vd + ((int64_t)ck * g.BN + j) * K + pos.sub * KT, vd);
                if (pos.sub == 0) __stcs(A.ck_vs + (int64_t)ck * g.BN + j, v);
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

// Gradients through the branches of one lane at one step, from V^d[t] (vd), the
// branch Gaussians of the recompute (eb, Mexican hat) and dL/dZ[t] (dz).
// direct[i] = dL/dV^d_i[t] through this step's branch only.
template <int KT, int G, int PSI>
__device__ __forceinline__ void branch_backward(const LaneParams<KT, G> &lp,
                                                const float (&vd)[KT], const float (&eb)[KT / G],
                                                float dz, float (&direct)[KT],
                                                GradAcc<KT, G> &acc) {
#pragma unroll
    for (int b = 0; b < KT / G; ++b) {
        float u[G];
        float ss = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
            u[g] = affine(lp, vd[b * G + g], b * G + g);
            ss = (g == 0) ? __fmul_rn(u[g], u[g]) : __fmaf_rn(u[g], u[g], ss);
        }
        const float gy = __fmul_rn(lp.km[b], dz);       // dL/dY_b
        float y, grr;                                    // Y_b and (dL/dr_b) * r_b
        if constexpr (PSI == PSI_MEXHAT) {
            const float e = eb[b];
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
        acc.gz[b] = __fmaf_rn(-grr, lp.iz[b], acc.gz[b]);
        acc.gk[b] = __fmaf_rn(__fmul_rn(lp.mk[b], y), dz, acc.gk[b]);
    }
}

template <int KT, int G>
constexpr int acc_count() { return 2 * KT + 2 * (KT / G); }

template <int K, int G, int PSI, typename XT, int L>
__global__ void __launch_bounds__(kThreads, 2)
dendsn_backward_kernel(const BwdArgs A) {
    constexpr int KT = (K < 4) ? K : 4;
    constexpr int LPN = K / KT;
    constexpr int KTb = KT / G;
    constexpr int NA = acc_count<KT, G>();
    // L == 4 is only used for T <= 4: one chunk per row and never a checkpoint
    constexpr bool MULTI = L > 4;
    // keep the recompute's Gaussians for the reverse pass (costs L * KTb registers)
    constexpr bool KEEP_E = false;
    using V = Vec<XT, KT>;
    using S1 = Scalar<XT>;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    LaneParams<KT, G> lp;
    load_lane_params<KT, G>(P, g, pos.chan, pos.sub, lp);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nc = MULTI ? (T + L - 1) / L : 1;  // chunks per row
    const int64_t stepX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const XT *__restrict__ x0 = static_cast<const XT *>(A.x) + j0 * K + pos.sub * KT;
    const XT *__restrict__ gs0 = static_cast<const XT *>(A.gs) + j0;
    XT *__restrict__ gx0 = static_cast<XT *>(A.gx) + j0 * K + pos.sub * KT;
    const float hard_dvds = -P.beta;             // dV[t+1]/dS[t] = -beta V[t]
    const float soft_dvds = -P.beta * P.theta;   // dV[t+1]/dS[t] = -beta theta

    GradAcc<KT, G> acc;
#pragma unroll
    for (int i = 0; i < KT; ++i) { acc.ga[i] = 0.f; acc.gxi[i] = 0.f; }
#pragma unroll
    for (int b = 0; b < KTb; ++b) { acc.gz[b] = 0.f; acc.gk[b] = 0.f; }

    typename V::Raw xb[L];            // inputs of the current unit, refilled with the next unit's
    typename S1::Raw gsb[L];          // grad_spikes of the current unit
    float ckd[KT];                    // checkpoint V^d entering the current unit
    float ckv = 0.f;                  // checkpoint V^s entering the current unit
#pragma unroll
    for (int i = 0; i < KT; ++i) ckd[i] = 0.f;
    if (pos.nrows > 0) {
        const int c = nc - 1;
        const int t0 = c * L;
#pragma unroll
        for (int tt = 0; tt < L; ++tt)
            if (t0 + tt < T) {
                xb[tt] = V::load(x0 + (t0 + tt) * stepX);
                gsb[tt] = S1::load(gs0 + (t0 + tt) * BN);
            }
        if (MULTI && c > 0) {
            Vec<float, KT>::unpack(Vec<float, KT>::load(
                A.ck_vd + ((int64_t)(c - 1) * BN + j0) * K + pos.sub * KT), ckd);
            ckv = __ldcs(A.ck_vs + (int64_t)(c - 1) * BN + j0);
        }
    }

    for (int i = 0; i < pos.nrows; ++i) {
        const int64_t j = j0 + i * jstep;
        const XT *xr = x0 + i * jstep * K;
        const XT *gsr = gs0 + i * jstep;
        XT *gxr = gx0 + i * jstep * K;
        if (P.mask_mode == 2)
            apply_neuron_mask<KT, G>(P, g, pos.row0 + (int64_t)i * pos.rstride, pos.p, pos.chan,
                                     pos.sub, lp);
        float Ad[KT];        // dL/dV^d[t+1], carried backwards
#pragma unroll
        for (int k = 0; k < KT; ++k) Ad[k] = 0.f;
        float dvn = 0.f;     // dL/dV^s[t+1]
        for (int c = nc - 1; c >= 0; --c) {
            const int t0 = c * L;
            // state entering the chunk: zero at t = 0, else the forward's checkpoint
            float vd0[KT];
#pragma unroll
            for (int k = 0; k < KT; ++k) vd0[k] = (!MULTI || c == 0) ? 0.f : ckd[k];
            const float v0 = (!MULTI || c == 0) ? 0.f : ckv;
            // next unit: the previous chunk of this row, or the last chunk of the next row
            const bool same_row = MULTI && c > 0;
            const bool has_next = same_row || (i + 1 < pos.nrows);
            const int cn = same_row ? c - 1 : nc - 1;
            const int tn = cn * L;
            const int64_t jn = same_row ? j : j + jstep;
            const XT *xn = (same_row ? xr : xr + jstep * K) + tn * stepX;
            const XT *gsn = (same_row ? gsr : gsr + jstep) + tn * BN;
            if (MULTI && has_next && cn > 0) {
                Vec<float, KT>::unpack(Vec<float, KT>::load(
                    A.ck_vd + ((int64_t)(cn - 1) * BN + jn) * K + pos.sub * KT), ckd);
                ckv = __ldcs(A.ck_vs + (int64_t)(cn - 1) * BN + jn);
            }

            // recompute the chunk, keeping V^d and V^s of every step (and the Gaussians)
            float vdh[L][KT];
            float vsh[L];
            float gsc[L];
            float eh[KEEP_E ? L : 1][KTb];
            {
                float vd[KT];
#pragma unroll
                for (int k = 0; k < KT; ++k) vd[k] = vd0[k];
                float v = v0;
                bool s = (!MULTI || c == 0) ? false : (v0 >= P.theta);
#pragma unroll
                for (int tt = 0; tt < L; ++tt) {
                    float xv[KT];
                    V::unpack(xb[tt], xv);
                    gsc[tt] = S1::unpack(gsb[tt]);
                    // refill slot tt for the next unit right after its value is taken
                    if (has_next && tn + tt < T) {
                        xb[tt] = V::load(xn + tt * stepX);
                        gsb[tt] = S1::load(gsn + tt * BN);
                    }
                    if (t0 + tt < T) {
                        float eb[KTb];
                        const float z = lanes_sum<LPN>(
                            dendrite_step<KT, G, PSI>(lp, vd, xv, P.residual != 0, inv_k, eb));
                        v = soma_charge(z, v, s, P);
                        s = v >= P.theta;
#pragma unroll
                        for (int k = 0; k < KT; ++k) vdh[tt][k] = vd[k];
                        vsh[tt] = v;
                        if constexpr (KEEP_E) {
#pragma unroll
                            for (int b = 0; b < KTb; ++b) eh[KEEP_E ? tt : 0][b] = eb[b];
                        }
                    }
                }
            }
            // reverse-time recursion over the chunk
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const int t = t0 + tt;
                if (t < T) {
                    const float vs = vsh[tt];
                    const bool st = vs >= P.theta;
                    const float dvds = P.detach ? 0.f : (P.soft ? soft_dvds : __fmul_rn(hard_dvds, vs));
                    const float dvdv = (P.soft || !st) ? P.beta : 0.f;   // beta (1 - S[t]) when hard
                    const float ds = __fmaf_rn(dvds, dvn, gsc[tt]);                      // dL/dS[t]
                    float dv = __fmaf_rn(surrogate(__fsub_rn(vs, P.theta)), ds,
                                         __fmul_rn(dvdv, dvn));                          // dL/dV^s[t]
                    if (A.gv) dv = __fadd_rn(dv, __ldcs(A.gv + t * BN + j));
                    float eb[KTb];
                    if constexpr (KEEP_E) {
#pragma unroll
                        for (int b = 0; b < KTb; ++b) eb[b] = eh[KEEP_E ? tt : 0][b];
                    } else if constexpr (PSI == PSI_MEXHAT) {
#pragma unroll
                        for (int b = 0; b < KTb; ++b) {
                            float ss = 0.f;
#pragma unroll
                            for (int q = 0; q < G; ++q) {
                                const float u = affine(lp, vdh[tt][b * G + q], b * G + q);
                                ss = (q == 0) ? __fmul_rn(u, u) : __fmaf_rn(u, u, ss);
                            }
                            eb[b] = gauss_half(ss);
                        }
                    }
                    float direct[KT];
                    branch_backward<KT, G, PSI>(lp, vdh[tt], eb, dv, direct, acc);
                    float gxv[KT];
                    const float res = P.residual ? __fmul_rn(dv, inv_k) : 0.f;
#pragma unroll
                    for (int k = 0; k < KT; ++k) {
                        Ad[k] = __fmaf_rn(lp.a[k], Ad[k], direct[k]);
                        gxv[k] = __fadd_rn(Ad[k], res);
                        const float vprev = (tt > 0) ? vdh[tt > 0 ? tt - 1 : 0][k] : vd0[k];
                        acc.ga[k] = __fmaf_rn(Ad[k], vprev, acc.ga[k]);
                    }
                    if (pos.active) V::store(gxr + t * stepX, gxv);
                    dvn = dv;
                }
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
