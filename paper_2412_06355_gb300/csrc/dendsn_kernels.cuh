// Fused DendSN layer kernels for sm_103a (GB300).
//
// Work decomposition. The B*N neurons of a layer are viewed as a matrix of
// O = B*N/P rows and P = C*inner columns: neuron j = o*P + p sits in row o,
// column p, and its parameter channel is c = p / inner, so every thread keeps
// one column, hence one parameter set, for its whole life. A block is a tile of
// TXn columns x TY row lanes; each neuron is served by LPN adjacent lanes of one
// warp that own KT = K / LPN compartments each (16 bytes of fp32 input per step,
// one 128-bit load). A thread walks up to R rows of its column, and each row's T
// steps in order. Inputs are fetched a fixed number of steps ahead of use, across
// chunk and row boundaries: through a per-thread ring of shared-memory slots filled
// by cp.async (the forward; the backward of multi-chunk rows), or a ring of
// registers (the backward of rows of at most 4 steps). In the paper's (C_o, P, H, W)
// layout a lane's compartments are H*W apart; when H*W is a multiple of 32 the
// forward stages each warp's inputs together (dendsn_forward_staged_kernel).
//
// Forward (Eqs. methods-compartment .. methods-lif-fire): V^d, V^s and S stay in
// registers across all T steps; the HBM traffic per step is the K inputs read and
// the spike written (plus an optional V^s write and, when T > L, a checkpoint of
// (V^d, V^s) every L steps).
//
// Backward (BPTT with the arctan surrogate, Eq. methods-sg): chunks of L steps are
// visited in reverse; each is recomputed from its checkpoint (or from zero state)
// with the forward's step function, so recomputed potentials and spikes are
// bit-identical to the forward's; then the reverse-time recursion runs and writes
// grad_x. Parameter-gradient partials stay in registers per thread, are reduced per
// channel inside the block in a fixed order (segmented warp shuffles, then shared
// memory), written to scratch, and summed over blocks in a fixed order by a
// finalize kernel: the parameter gradients are deterministic. When T is a multiple
// of L a full-chunk build of the same kernel drops the step bounds tests. Rows of
// one full chunk of whole 8-compartment neurons take dendsn_backward_phased_kernel,
// which runs a row in phases (recompute into shared memory, soma in registers,
// dendritic reverse scan one compartment pair at a time) and gives bit-identical
// results with fewer live registers; for bfloat16 layers whose forward kept V^s in the
// saved buffer, dendsn_backward_phased_vs_kernel skips the recompute of the soma and
// rescans only V^d, per compartment pair, in registers. 4-step rows of 8-compartment
// float32 neurons on two lanes take dendsn_backward_rowpair_kernel: the same phases over
// two rows per thread, each paired instruction carrying one compartment of both rows.
//
// Arithmetic. With one compartment per branch (G = 1) the per-compartment work is
// done two compartments at a time with the paired fp32 instructions of sm_100+
// (__ffma2_rn and friends round each component exactly like __fmaf_rn), which
// halves the floating-point instruction count; G > 1 uses a scalar engine.
// Address arithmetic is pointer increments; 64-bit divisions happen once per thread.
//
// Waits. The kernels never spin: cp.async.wait_group waits on the thread's own copies,
// __syncwarp / __syncthreads on threads that always reach them, griddepcontrol.wait on
// the completion of the grid launched before this one in the stream.
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
    static __device__ __forceinline__ Raw pack(const float (&v)[KT]) {
        if constexpr (KT == 4) return make_float4(v[0], v[1], v[2], v[3]);
        else if constexpr (KT == 2) return make_float2(v[0], v[1]);
        else return v[0];
    }
    static __device__ __forceinline__ void store(float *p, const float (&v)[KT]) {
        __stcs(reinterpret_cast<Raw *>(p), pack(v));
    }
};

// Eight fp32 compartments of one lane: two 16-byte halves.
struct F8 { float4 a, b; };
template <> struct Vec<float, 8> {
    using Raw = F8;
    static __device__ __forceinline__ Raw load(const float *p) {
        F8 r;
        r.a = __ldcs(reinterpret_cast<const float4 *>(p));
        r.b = __ldcs(reinterpret_cast<const float4 *>(p) + 1);
        return r;
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[8]) {
        v[0] = r.a.x; v[1] = r.a.y; v[2] = r.a.z; v[3] = r.a.w;
        v[4] = r.b.x; v[5] = r.b.y; v[6] = r.b.z; v[7] = r.b.w;
    }
    static __device__ __forceinline__ Raw pack(const float (&v)[8]) {
        F8 r;
        r.a = make_float4(v[0], v[1], v[2], v[3]);
        r.b = make_float4(v[4], v[5], v[6], v[7]);
        return r;
    }
    static __device__ __forceinline__ void store(float *p, const float (&v)[8]) {
        const F8 r = pack(v);
        __stcs(reinterpret_cast<float4 *>(p), r.a);
        __stcs(reinterpret_cast<float4 *>(p) + 1, r.b);
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
    using Raw = typename std::conditional<KT == 8, uint4,
                typename std::conditional<KT == 4, uint2,
                typename std::conditional<KT == 2, unsigned int, unsigned short>::type>::type>::type;
    static __device__ __forceinline__ Raw load(const T *p) {
        return __ldcs(reinterpret_cast<const Raw *>(p));
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) {   // exact
        if constexpr (KT == 8) {
            v[0] = bf16_lo(r.x); v[1] = bf16_hi(r.x); v[2] = bf16_lo(r.y); v[3] = bf16_hi(r.y);
            v[4] = bf16_lo(r.z); v[5] = bf16_hi(r.z); v[6] = bf16_lo(r.w); v[7] = bf16_hi(r.w);
        }
        else if constexpr (KT == 4) { v[0] = bf16_lo(r.x); v[1] = bf16_hi(r.x); v[2] = bf16_lo(r.y); v[3] = bf16_hi(r.y); }
        else if constexpr (KT == 2) { v[0] = bf16_lo(r); v[1] = bf16_hi(r); }
        else { v[0] = bf16_lo(r); }
    }
    static __device__ __forceinline__ void store(T *p, const float (&v)[KT]) {
        if constexpr (KT == 8) {
            __stcs(reinterpret_cast<uint4 *>(p),
                   make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                              pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7])));
        } else if constexpr (KT == 4) {
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

template <typename XT> constexpr int xt_code() { return std::is_same<XT, float>::value ? 0 : 1; }

template <int XT> struct XType;
template <> struct XType<0> { using type = float; };
template <> struct XType<1> { using type = __nv_bfloat16; };

// Mask bits of KTb branches of one lane: fetched raw (one or two 32-bit loads, so a
// row's mask can be requested a row ahead of its use), then unpacked to 1.0f / 0.0f.
template <int KTb> struct MaskRaw { using T = typename std::conditional<KTb == 8, uint2, uint32_t>::type; };

template <int KTb>
__device__ __forceinline__ typename MaskRaw<KTb>::T fetch_mask(const uint8_t *m) {
    if constexpr (KTb == 8) {
        return make_uint2(__ldg(reinterpret_cast<const unsigned int *>(m)),
                          __ldg(reinterpret_cast<const unsigned int *>(m) + 1));
    } else if constexpr (KTb == 4) {
        return __ldg(reinterpret_cast<const unsigned int *>(m));
    } else if constexpr (KTb == 2) {
        return __ldg(reinterpret_cast<const unsigned short *>(m));
    } else {
        return __ldg(m);
    }
}

template <int KTb>
__device__ __forceinline__ void unpack_mask(const typename MaskRaw<KTb>::T &q, float (&mk)[KTb]) {
    if constexpr (KTb == 8) {
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            mk[b] = ((q.x >> (8 * b)) & 0xffu) ? 1.f : 0.f;
            mk[4 + b] = ((q.y >> (8 * b)) & 0xffu) ? 1.f : 0.f;
        }
    } else {
#pragma unroll
        for (int b = 0; b < KTb; ++b) mk[b] = ((q >> (8 * b)) & 0xffu) ? 1.f : 0.f;
    }
}

template <int KTb>
__device__ __forceinline__ void load_mask(const uint8_t *m, float (&mk)[KTb]) {
    unpack_mask<KTb>(fetch_mask<KTb>(m), mk);
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

__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 neg2(float2 a) { return make_float2(-a.x, -a.y); }

// Per-lane parameters as loaded (KT compartments, KTb = KT/G branches).
template <int KT, int G>
__device__ __forceinline__ void load_param_arrays(const Params &P, const Geometry &g, int chan,
                                                  int sub, float (&a)[KT], float (&nxi)[KT],
                                                  float (&iz)[KT / G], float (&km)[KT / G],
                                                  float (&mk)[KT / G]) {
    constexpr int KTb = KT / G;
#pragma unroll
    for (int b = 0; b < KTb; ++b) {
        iz[b] = __frcp_rn(__ldg(P.zeta + (int64_t)chan * g.Kb + sub * KTb + b));
        mk[b] = 1.f;
    }
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const int k = sub * KT + i;
        a[i] = P.stateless ? 0.f : __ldg(P.alpha + (int64_t)chan * g.K + k);
        nxi[i] = -__fmul_rn(__ldg(P.xi + (int64_t)chan * g.K + k), iz[i / G]);   // -xi / zeta
    }
    if (P.mask_mode == 1) load_mask<KTb>(P.mask + (int64_t)chan * g.Kb + sub * KTb, mk);
#pragma unroll
    for (int b = 0; b < KTb; ++b)
        km[b] = __fmul_rn(__ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b), mk[b]);
}

// The lane's unmasked kappa, read once for the parameter-gradient export.
template <int KTb>
__device__ __forceinline__ void lane_kappa(const Params &P, const Geometry &g, int chan, int sub,
                                           float (&kap)[KTb]) {
#pragma unroll
    for (int b = 0; b < KTb; ++b) kap[b] = __ldg(P.kappa + (int64_t)chan * g.Kb + sub * KTb + b);
}

// kappa * m and m for the neuron n of a per-neuron mask (mask_mode 2).
template <int KTb>
__device__ __forceinline__ typename MaskRaw<KTb>::T fetch_neuron_mask(const Params &P, const Geometry &g,
                                                                      int64_t n, int sub) {
    return fetch_mask<KTb>(P.mask + n * g.Kb + sub * KTb);
}

// kappa * m and m of a lane's KTb branches from their raw mask bytes (nonzero: kept) and
// kappa: a select, not a product (kappa * 1 = kappa, kappa * 0 = 0 up to the sign of zero).
template <int KTb>
__device__ __forceinline__ void apply_neuron_mask(const typename MaskRaw<KTb>::T &raw,
                                                  const float (&kap)[KTb],
                                                  float (&km)[KTb], float (&mk)[KTb]) {
#pragma unroll
    for (int b = 0; b < KTb; ++b) {
        uint32_t w;
        if constexpr (KTb == 8) w = b < 4 ? raw.x : raw.y;
        else w = raw;
        const bool on = (w & (0xffu << (8 * (b & 3)))) != 0u;
        km[b] = on ? kap[b] : 0.f;
        mk[b] = on ? 1.f : 0.f;
    }
}

// Bytes of dynamic shared memory in front of a kernel's other regions that hold each
// thread's KTb kappa values when masks are per neuron (else none).
__host__ __device__ constexpr size_t kappa_smem_bytes(int mask_mode, int KTb, int NT) {
    return mask_mode == 2 ? (size_t)KTb * NT * sizeof(float) : 0;
}

// ================================================================ paired engine, G = 1
// Compartment i is branch i. u = V^d/zeta - xi/zeta; r = |u|.
// In the backward the branch mask enters the Mexican hat through its exponent: lm = 0 for
// a kept branch and -inf for a masked one, so e^{-r^2/2} (and with it Y and psi') is
// exactly 0 where m = 0 at no extra instruction; for the identity lm holds m itself. (The
// forward needs no masked Y: kappa m = 0 already removes the branch from Z.)
// The backward carries the dendritic adjoint and three of its sums without the factor
// 1/zeta of Eq. methods-branch-aggregation (a per-lane constant): A = zeta Ad, and
// dL/dalpha, dL/dxi, dL/dzeta are scaled by 1/zeta once, in acc_export. Lanes of 8
// compartments (KAPPA_FREE) also leave out the factor kappa m of Eq. methods-soma-input:
// A = zeta Ad / (kappa m), so that dL/du / (kappa m) = -dL/dZ psi'(u) enters the scan with
// no product by kappa m; dL/dX = A (kappa m / zeta), and the three sums are scaled by
// kappa / zeta in acc_export (a masked branch's terms are 0: its e^{-r^2/2}, or for the
// identity its m, is 0; so the unmasked kappa scales every row, whatever the row's mask;
// a kappa of 0 gives A finite and every scaled result 0). The phased backward forms
// kappa m / zeta once per compartment pair and row, which saves one paired multiply per
// pair and step (kept-V^s deeper conv backward 428.4 -> 418.4 us); the chunked backward
// must form it every step, and with 4 compartments per lane that version spilled more
// (conv layer 216 -> 230 us), so 4-compartment lanes keep the product by kappa m in the
// step. Both layouts of a layer take lanes of the same width, so their bits still agree.
template <int KT, int PSI, bool TREE>
struct PairArith {
    static constexpr bool kTree = TREE;
    static constexpr bool KAPPA_FREE = KT == 8;
    static constexpr int N2 = KT / 2;
    static constexpr int KTb = KT;
    struct LP { float2 a[N2], nxi[N2], iz[N2], km[N2], lm[N2]; };
    struct St { float2 v[N2]; };
    struct Acc { float2 ga[N2], ngxi[N2], ngz[N2], ngk[N2]; };  // ngxi, ngz, ngk: negated sums
    // mask value as the engine keeps it (see above)
    static __device__ __forceinline__ float mask_term(float m) {
        if constexpr (PSI == PSI_MEXHAT) return m != 0.f ? 0.f : -INFINITY;
        else return m;
    }

    static __device__ __forceinline__ void load(const Params &P, const Geometry &g, int chan, int sub, LP &lp) {
        float a[KT], nxi[KT], iz[KT], km[KT], mk[KT];
        load_param_arrays<KT, 1>(P, g, chan, sub, a, nxi, iz, km, mk);
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            lp.a[m] = make_float2(a[2 * m], a[2 * m + 1]);
            lp.nxi[m] = make_float2(nxi[2 * m], nxi[2 * m + 1]);
            lp.iz[m] = make_float2(iz[2 * m], iz[2 * m + 1]);
            lp.km[m] = make_float2(km[2 * m], km[2 * m + 1]);
            lp.lm[m] = make_float2(mask_term(mk[2 * m]), mask_term(mk[2 * m + 1]));
        }
    }
    using MRaw = typename MaskRaw<KTb>::T;
    static __device__ __forceinline__ MRaw fetch_neuron_mask(const Params &P, const Geometry &g, int64_t n, int sub) {
        return dendsn::fetch_neuron_mask<KT>(P, g, n, sub);
    }
    static __device__ __forceinline__ void neuron_mask(const MRaw &raw, const float (&kap)[KT], LP &lp) {
        float km[KT], mk[KT];
        apply_neuron_mask<KT>(raw, kap, km, mk);
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            lp.km[m] = make_float2(km[2 * m], km[2 * m + 1]);
            lp.lm[m] = make_float2(mask_term(mk[2 * m]), mask_term(mk[2 * m + 1]));
        }
    }
    static __device__ __forceinline__ void zero(St &s) {
#pragma unroll
        for (int m = 0; m < N2; ++m) s.v[m] = f2(0.f);
    }
    static __device__ __forceinline__ void to_array(const St &s, float (&v)[KT]) {
#pragma unroll
        for (int m = 0; m < N2; ++m) { v[2 * m] = s.v[m].x; v[2 * m + 1] = s.v[m].y; }
    }
    static __device__ __forceinline__ void from_array(St &s, const float (&v)[KT]) {
#pragma unroll
        for (int m = 0; m < N2; ++m) s.v[m] = make_float2(v[2 * m], v[2 * m + 1]);
    }
    // Pair m of one forward step (Eqs. methods-compartment, -branch-aggregation,
    // -mexican-hat): advances its V^d by the input x2 and returns its branch outputs Y.
    static __device__ __forceinline__ float2 pair_y(const LP &lp, int m, float2 &vd, float2 x2) {
        vd = ffma2(lp.a[m], vd, x2);
        const float2 u = ffma2(vd, lp.iz[m], lp.nxi[m]);
        if constexpr (PSI == PSI_MEXHAT) {
            const float2 ss = fmul2(u, u);
            const float2 t = fmul2(f2(kNegHalfLog2e), ss);
            const float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
            return ffma2(neg2(ss), e, e);                        // (1 - r^2) e^{-r^2/2}
        } else {
            return make_float2(fabsf(u.x), fabsf(u.y));          // r
        }
    }
    // The lane's share of Z as one chain over the pairs (used when the forward and the
    // backward give a neuron the same lanes; see step for the tree order).
    static __device__ __forceinline__ float step_chain(const LP &lp, St &vd, const float (&x)[KT],
                                                       bool residual, float inv_k) {
        float2 zp = f2(0.f);
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            const float2 y = pair_y(lp, m, vd.v[m], make_float2(x[2 * m], x[2 * m + 1]));
            zp = (m == 0) ? fmul2(lp.km[m], y) : ffma2(lp.km[m], y, zp);
        }
        float z = __fadd_rn(zp.x, zp.y);
        if (residual) {
            float xs = x[0];
#pragma unroll
            for (int i = 1; i < KT; ++i) xs = __fadd_rn(xs, x[i]);
            z = __fmaf_rn(xs, inv_k, z);
        }
        return z;
    }
    // Eqs. methods-compartment, -branch-aggregation, -mexican-hat, -soma-input, -residual.
    // The lane's share of Z is summed in a fixed tree: compartments in groups of four
    // (two pairs, reduced with one paired multiply and one paired FMA, then the two
    // halves), plus the group's share of the residual, then the groups pairwise. The
    // cross-lane butterfly continues the same tree, so the result is bit-identical for
    // any split of a neuron over 1, 2 or 4 lanes.
    static __device__ __forceinline__ float step(const LP &lp, St &vd, const float (&x)[KT],
                                                 bool residual, float inv_k) {
        if constexpr (!TREE) return step_chain(lp, vd, x, residual, inv_k);
        constexpr int NG = (N2 + 1) / 2;                          // groups of two pairs
        float gv[NG];
#pragma unroll
        for (int q = 0; q < NG; ++q) {
            float2 acc = f2(0.f);
#pragma unroll
            for (int h = 0; h < 2 && 2 * q + h < N2; ++h) {
                const int m = 2 * q + h;
                const float2 y = pair_y(lp, m, vd.v[m], make_float2(x[2 * m], x[2 * m + 1]));
                acc = (h == 0) ? fmul2(lp.km[m], y) : ffma2(lp.km[m], y, acc);
            }
            gv[q] = __fadd_rn(acc.x, acc.y);
            if (residual) {
                float xs = x[4 * q];
#pragma unroll
                for (int i = 1; i < 4 && 4 * q + i < KT; ++i) xs = __fadd_rn(xs, x[4 * q + i]);
                gv[q] = __fmaf_rn(xs, inv_k, gv[q]);
            }
        }
        if constexpr (NG == 2) gv[0] = __fadd_rn(gv[0], gv[NG - 1]);
        return gv[0];
    }
    static __device__ __forceinline__ void acc_zero(Acc &c) {
#pragma unroll
        for (int m = 0; m < N2; ++m) { c.ga[m] = f2(0.f); c.ngxi[m] = f2(0.f); c.ngz[m] = f2(0.f); c.ngk[m] = f2(0.f); }
    }
    // Floats in Acc; acc_flush adds them into per-thread totals t[q * NT] and zeroes them,
    // acc_load reads them back.
    static constexpr int kAccFloats = 8 * N2;
    template <int NT>
    static __device__ __forceinline__ void acc_flush(Acc &c, float *t) {
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            const float2 *f[4] = {&c.ga[m], &c.ngxi[m], &c.ngz[m], &c.ngk[m]};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                t[(8 * m + 2 * q) * NT] = __fadd_rn(t[(8 * m + 2 * q) * NT], f[q]->x);
                t[(8 * m + 2 * q + 1) * NT] = __fadd_rn(t[(8 * m + 2 * q + 1) * NT], f[q]->y);
            }
        }
        acc_zero(c);
    }
    template <int NT>
    static __device__ __forceinline__ void acc_load(Acc &c, const float *t) {
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            float2 *f[4] = {&c.ga[m], &c.ngxi[m], &c.ngz[m], &c.ngk[m]};
#pragma unroll
            for (int q = 0; q < 4; ++q) *f[q] = make_float2(t[(8 * m + 2 * q) * NT], t[(8 * m + 2 * q + 1) * NT]);
        }
    }
    // [alpha KT | xi KT | zeta KTb | kappa KTb]; the first three carry the factor 1/zeta, or
    // kappa/zeta (KAPPA_FREE), here (kap: the lane's unmasked kappa)
    static __device__ __forceinline__ void acc_export(const LP &lp, const Acc &c, float *v,
                                                      const float (&kap)[KT]) {
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            const float2 kz = KAPPA_FREE ? fmul2(make_float2(kap[2 * m], kap[2 * m + 1]), lp.iz[m]) : lp.iz[m];
            const float2 ga = fmul2(c.ga[m], kz);
            const float2 gxi = fmul2(c.ngxi[m], kz);
            const float2 gz = fmul2(c.ngz[m], kz);
            v[2 * m] = ga.x;                     v[2 * m + 1] = ga.y;
            v[KT + 2 * m] = -gxi.x;              v[KT + 2 * m + 1] = -gxi.y;
            v[2 * KT + 2 * m] = -gz.x;           v[2 * KT + 2 * m + 1] = -gz.y;
            v[3 * KT + 2 * m] = -c.ngk[m].x;     v[3 * KT + 2 * m + 1] = -c.ngk[m].y;
        }
    }
    // One reverse step: V^d[t] (vdt), V^d[t-1] (vdp) and dL/dZ[t] (dz) update the scaled
    // dendritic adjoint A (reverse scan of Eq. methods-compartment), the parameter-gradient
    // partials, and give dL/dX[t] + res.
    // Per branch (G = 1): dL/du = kappa m dz psi'(u) with psi'(u) = u (u^2 - 3) e^{-u^2/2}
    // (the Mexican hat of |u| is smooth in u) or sign(u) (identity); the direct term of
    // dL/dV^d is dL/du / zeta; du/dxi = -1/zeta; du/dzeta = -u / zeta.
    static __device__ __forceinline__ void backward(const LP &lp, const St &vdt, const St &vdp, float dz,
                                                    St &Ad, Acc &acc, float res, float (&gx)[KT]) {
        const float2 ndz2 = f2(-dz);
        const float2 res2 = f2(res);
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            const float2 g = pair_back(lp, m, vdt.v[m], vdp.v[m], ndz2, res2, Ad.v[m], acc,
                                       KAPPA_FREE ? fmul2(lp.km[m], lp.iz[m]) : lp.iz[m]);
            gx[2 * m] = g.x;
            gx[2 * m + 1] = g.y;
        }
    }
    // Pair m of one reverse step (see backward), given ndz2 = -dL/dZ[t] and the pair's
    // kappa m / zeta (KAPPA_FREE) or 1 / zeta (kmz); returns dL/dX[t] of the pair.
    static __device__ __forceinline__ float2 pair_back(const LP &lp, int m, float2 vdt, float2 vdp,
                                                       float2 ndz2, float2 res2, float2 &Adm, Acc &acc,
                                                       float2 kmz) {
        {
            const float2 u = ffma2(vdt, lp.iz[m], lp.nxi[m]);
            // -dL/dY, or -m dL/dZ (KAPPA_FREE)
            const float2 ngy = fmul2(KAPPA_FREE ? lp.lm[m] : lp.km[m], ndz2);
            float2 y, du;                                        // m Y; dL/du, or / (kappa m)
            if constexpr (PSI == PSI_MEXHAT) {
                const float2 ss = fmul2(u, u);
                const float2 t = ffma2(f2(kNegHalfLog2e), ss, lp.lm[m]);
                const float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
                y = ffma2(neg2(ss), e, e);
                // psi'(r) / r = (r^2 - 3) e^{-r^2/2} = -(2 e^{-r^2/2} + psi(r)): one fused
                // multiply-add from y; its sign cancels against that of -dL/dZ
                const float2 nw = ffma2(f2(2.f), e, y);
                du = KAPPA_FREE ? fmul2(fmul2(nw, u), ndz2) : fmul2(nw, fmul2(u, ngy));
            } else {
                y = fmul2(lp.lm[m], make_float2(fabsf(u.x), fabsf(u.y)));
                du = make_float2(u.x > 0.f ? -ngy.x : (u.x < 0.f ? ngy.x : 0.f),
                                 u.y > 0.f ? -ngy.y : (u.y < 0.f ? ngy.y : 0.f));
            }
            // (KAPPA_FREE: each of ngxi, ngz, ga times kappa)
            acc.ngxi[m] = fadd2(acc.ngxi[m], du);                // zeta dxi = -sum du
            acc.ngz[m] = ffma2(u, du, acc.ngz[m]);               // zeta dzeta = -sum u du
            acc.ngk[m] = ffma2(y, ndz2, acc.ngk[m]);             // dkappa = sum m Y dz
            Adm = ffma2(lp.a[m], Adm, du);
            acc.ga[m] = ffma2(Adm, vdp, acc.ga[m]);              // zeta dalpha
            return ffma2(Adm, kmz, res2);
        }
    }
};

// ================================================================ scalar engine, any G
template <int KT, int G, int PSI>
struct ScalarArith {
    static constexpr int KTb = KT / G;
    static constexpr bool KAPPA_FREE = false;
    struct LP { float a[KT], nxi[KT], iz[KTb], km[KTb], mk[KTb]; };
    struct St { float v[KT]; };
    struct Acc { float ga[KT], gxi[KT], gz[KTb], gk[KTb]; };

    static __device__ __forceinline__ void load(const Params &P, const Geometry &g, int chan, int sub, LP &lp) {
        load_param_arrays<KT, G>(P, g, chan, sub, lp.a, lp.nxi, lp.iz, lp.km, lp.mk);
    }
    using MRaw = typename MaskRaw<KTb>::T;
    static __device__ __forceinline__ MRaw fetch_neuron_mask(const Params &P, const Geometry &g, int64_t n, int sub) {
        return dendsn::fetch_neuron_mask<KTb>(P, g, n, sub);
    }
    static __device__ __forceinline__ void neuron_mask(const MRaw &raw, const float (&kap)[KTb], LP &lp) {
        apply_neuron_mask<KTb>(raw, kap, lp.km, lp.mk);
    }
    static __device__ __forceinline__ void zero(St &s) {
#pragma unroll
        for (int i = 0; i < KT; ++i) s.v[i] = 0.f;
    }
    static __device__ __forceinline__ void to_array(const St &s, float (&v)[KT]) {
#pragma unroll
        for (int i = 0; i < KT; ++i) v[i] = s.v[i];
    }
    static __device__ __forceinline__ void from_array(St &s, const float (&v)[KT]) {
#pragma unroll
        for (int i = 0; i < KT; ++i) s.v[i] = v[i];
    }
    static __device__ __forceinline__ float affine(const LP &lp, float vd, int i) {
        return __fmaf_rn(vd, lp.iz[i / G], lp.nxi[i]);
    }
    // Eqs. methods-compartment, -branch-aggregation, -mexican-hat, -soma-input.
    static __device__ __forceinline__ float step(const LP &lp, St &vd, const float (&x)[KT],
                                                 bool residual, float inv_k) {
#pragma unroll
        for (int i = 0; i < KT; ++i) vd.v[i] = __fmaf_rn(lp.a[i], vd.v[i], x[i]);
        float zp = 0.f;
#pragma unroll
        for (int b = 0; b < KTb; ++b) {
            float ss = 0.f, u0 = 0.f;
#pragma unroll
            for (int q = 0; q < G; ++q) {
                const float u = affine(lp, vd.v[b * G + q], b * G + q);
                if (q == 0) u0 = u;
                ss = (q == 0) ? __fmul_rn(u, u) : __fmaf_rn(u, u, ss);
            }
            float y;
            if constexpr (PSI == PSI_MEXHAT) {
                const float e = gauss_half(ss);
                y = __fmaf_rn(-ss, e, e);                     // (1 - r^2) e^{-r^2/2}
            } else {
                y = (G == 1) ? fabsf(u0) : sqrtf(ss);         // r
            }
            zp = __fmaf_rn(lp.km[b], y, zp);
        }
        if (residual) {
            float xs = x[0];
#pragma unroll
            for (int i = 1; i < KT; ++i) xs = __fadd_rn(xs, x[i]);
            zp = __fmaf_rn(xs, inv_k, zp);
        }
        return zp;
    }
    static __device__ __forceinline__ void acc_zero(Acc &c) {
#pragma unroll
        for (int i = 0; i < KT; ++i) { c.ga[i] = 0.f; c.gxi[i] = 0.f; }
#pragma unroll
        for (int b = 0; b < KTb; ++b) { c.gz[b] = 0.f; c.gk[b] = 0.f; }
    }
    // Floats in Acc; acc_flush adds them into per-thread totals t[q * NT] and zeroes them,
    // acc_load reads them back.
    static constexpr int kAccFloats = 2 * KT + 2 * KTb;
    template <int NT>
    static __device__ __forceinline__ void acc_flush(Acc &c, float *t) {
#pragma unroll
        for (int i = 0; i < KT; ++i) {
            t[i * NT] = __fadd_rn(t[i * NT], c.ga[i]);
            t[(KT + i) * NT] = __fadd_rn(t[(KT + i) * NT], c.gxi[i]);
        }
#pragma unroll
        for (int b = 0; b < KTb; ++b) {
            t[(2 * KT + b) * NT] = __fadd_rn(t[(2 * KT + b) * NT], c.gz[b]);
            t[(2 * KT + KTb + b) * NT] = __fadd_rn(t[(2 * KT + KTb + b) * NT], c.gk[b]);
        }
        acc_zero(c);
    }
    template <int NT>
    static __device__ __forceinline__ void acc_load(Acc &c, const float *t) {
#pragma unroll
        for (int i = 0; i < KT; ++i) { c.ga[i] = t[i * NT]; c.gxi[i] = t[(KT + i) * NT]; }
#pragma unroll
        for (int b = 0; b < KTb; ++b) { c.gz[b] = t[(2 * KT + b) * NT]; c.gk[b] = t[(2 * KT + KTb + b) * NT]; }
    }
    template <int N>
    static __device__ __forceinline__ void acc_export(const LP &, const Acc &c, float *v, const float (&)[N]) {
#pragma unroll
        for (int i = 0; i < KT; ++i) { v[i] = c.ga[i]; v[KT + i] = c.gxi[i]; }
#pragma unroll
        for (int b = 0; b < KTb; ++b) { v[2 * KT + b] = c.gz[b]; v[2 * KT + KTb + b] = c.gk[b]; }
    }
    static __device__ __forceinline__ void backward(const LP &lp, const St &vdt, const St &vdp, float dz,
                                                    St &Ad, Acc &acc, float res, float (&gx)[KT]) {
        float direct[KT];
#pragma unroll
        for (int b = 0; b < KTb; ++b) {
            float u[G];
            float ss = 0.f;
#pragma unroll
            for (int q = 0; q < G; ++q) {
                u[q] = affine(lp, vdt.v[b * G + q], b * G + q);
                ss = (q == 0) ? __fmul_rn(u[q], u[q]) : __fmaf_rn(u[q], u[q], ss);
            }
            const float gy = __fmul_rn(lp.km[b], dz);       // dL/dY_b
            float y, grr;                                    // Y_b and (dL/dr_b) * r_b
            if constexpr (PSI == PSI_MEXHAT) {
                const float e = gauss_half(ss);
                y = __fmaf_rn(-ss, e, e);
                // psi'(r) / r = (r^2 - 3) e^{-r^2/2}, so du_i = q u_i with no division
                const float qq = __fmul_rn(__fmul_rn(__fsub_rn(ss, 3.f), e), gy);
#pragma unroll
                for (int q = 0; q < G; ++q) {
                    const float d = __fmul_rn(__fmul_rn(qq, u[q]), lp.iz[b]);
                    direct[b * G + q] = d;
                    acc.gxi[b * G + q] = __fsub_rn(acc.gxi[b * G + q], d);
                }
                grr = __fmul_rn(ss, qq);
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
                    const float qq = (r > 0.f) ? __fdiv_rn(gy, r) : 0.f;   // subgradient 0 at r = 0
#pragma unroll
                    for (int q = 0; q < G; ++q) {
                        const float d = __fmul_rn(__fmul_rn(qq, u[q]), lp.iz[b]);
                        direct[b * G + q] = d;
                        acc.gxi[b * G + q] = __fsub_rn(acc.gxi[b * G + q], d);
                    }
                }
                y = r;
                grr = __fmul_rn(gy, r);
            }
            acc.gz[b] = __fmaf_rn(-grr, lp.iz[b], acc.gz[b]);
            acc.gk[b] = __fmaf_rn(__fmul_rn(lp.mk[b], y), dz, acc.gk[b]);
        }
#pragma unroll
        for (int i = 0; i < KT; ++i) {
            Ad.v[i] = __fmaf_rn(lp.a[i], Ad.v[i], direct[i]);
            gx[i] = __fadd_rn(Ad.v[i], res);
            acc.ga[i] = __fmaf_rn(Ad.v[i], vdp.v[i], acc.ga[i]);
        }
    }
};

// fp32 layers sum Z in the group tree (their forward and backward may split a neuron
// over different lane counts); bf16 layers use the shorter chain.
template <int KT, int G, int PSI, typename XT>
using Arith = typename std::conditional<(G == 1 && KT % 2 == 0),
                                        PairArith<KT, PSI, std::is_same<XT, float>::value>,
                                        ScalarArith<KT, G, PSI>>::type;

// Per-neuron branch masks (mask_mode 2) of a thread's rows, each fetched one row ahead of
// its use so the row start does not wait on the load. kappa * m is rebuilt at each row
// from the lane's kappa, copied once into the front of the block's dynamic shared memory
// (kappa_smem_bytes: vectors of W values, vector v of thread i at [v * NT + i]) rather than
// re-read from global memory per row. n: the neuron (within a sample) of the next row;
// step: the thread's row stride in neurons, modulo N.
template <typename AR, int NT>
struct MaskAhead {
    static constexpr int KTb = AR::KTb;
    static constexpr int W = KTb % 4 == 0 ? 4 : (KTb % 2 == 0 ? 2 : 1);
    using KV = typename std::conditional<W == 4, float4,
                                         typename std::conditional<W == 2, float2, float>::type>::type;
    typename AR::MRaw next;
    KV *kap;
    int n, step;
    __device__ __forceinline__ void init(const Params &P, const Geometry &g, int64_t j0,
                                         int64_t jstep, int chan, int sub, int nrows,
                                         void *kbase) {
        n = (int)(j0 % g.N);
        step = (int)(jstep % g.N);
        kap = reinterpret_cast<KV *>(kbase) + threadIdx.x;
        if (P.mask_mode != 2) return;
        const float *src = P.kappa + (int64_t)chan * g.Kb + sub * KTb;
#pragma unroll
        for (int v = 0; v < KTb / W; ++v) {
            KV q;
#pragma unroll
            for (int w = 0; w < W; ++w) reinterpret_cast<float *>(&q)[w] = __ldg(src + v * W + w);
            kap[v * NT] = q;
        }
        if (nrows > 0) next = AR::fetch_neuron_mask(P, g, n, sub);
    }
    // applies the current row's mask, then requests the next row's (if `more`)
    __device__ __forceinline__ void advance(const Params &P, const Geometry &g, int sub,
                                            bool more, typename AR::LP &lp) {
        if (P.mask_mode != 2) return;
        float k[KTb];
#pragma unroll
        for (int v = 0; v < KTb / W; ++v) {
            const KV q = kap[v * NT];
#pragma unroll
            for (int w = 0; w < W; ++w) k[v * W + w] = reinterpret_cast<const float *>(&q)[w];
        }
        AR::neuron_mask(next, k, lp);
        n += step;
        if (n >= g.N) n -= g.N;
        if (more) next = AR::fetch_neuron_mask(P, g, n, sub);
    }
};

// Sum of the LPN lanes' shares (xor butterfly: every lane gets the same bits).
template <int LPN>
__device__ __forceinline__ float lanes_sum(float v) {
    if constexpr (LPN >= 2) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 1));
    if constexpr (LPN >= 4) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 2));
    if constexpr (LPN >= 8) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, 4));
    return v;
}

// Z[t] of the neuron: the lane's branch share (plus its residual share), summed over lanes.
template <typename AR, int KT, int LPN>
__device__ __forceinline__ float soma_input(const typename AR::LP &lp, typename AR::St &vd,
                                            const float (&x)[KT], bool residual, float inv_k) {
    return lanes_sum<LPN>(AR::step(lp, vd, x, residual, inv_k));
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

// ---------------------------------------------------------------- forward
// Tuning: the forward's minimum resident blocks per SM (register cap), and whether
// its inputs are staged through shared memory with cp.async (else a register ring).
#ifndef DENDSN_FWD_MINB
#define DENDSN_FWD_MINB 3
#endif
#ifndef DENDSN_FWD_ASYNC
#define DENDSN_FWD_ASYNC 1
#endif
constexpr int kFwdDepth = 8;   // steps of x in flight per thread on the cp.async path
// The forward's ring depth: 16 steps for float32 slots of up to 16 bytes (conv and event
// layers' forward 1-2% faster), else 8 (wider slots would halve the resident blocks; the
// bf16 8-compartment forward measured 1% slower with 16)
template <typename XT, typename Raw> constexpr int fwd_depth() {
    return (std::is_same<XT, float>::value && sizeof(Raw) <= 16) ? 16 : 8;
}
#ifndef DENDSN_BWD_ASYNC
#define DENDSN_BWD_ASYNC 1
#endif
constexpr int kBwdDepth = 8;   // steps of x in flight per thread in the backward's cp.async ring
#ifndef DENDSN_BWD_PHASED
#define DENDSN_BWD_PHASED 1
#endif
#ifndef DENDSN_BWD_ROWPAIR
#define DENDSN_BWD_ROWPAIR 1
#endif

// Asynchronous 4/8/16-byte global -> shared copy (PTX cp.async). `dep` is an unused
// operand that orders the copy after the computation producing it.
template <int BYTES>
__device__ __forceinline__ void cp_async(void *smem, const void *gmem, float dep) {
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem);
    if constexpr (BYTES == 16)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16; // %2\n" :: "r"(d), "l"(gmem), "f"(dep) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], %3; // %2\n" :: "r"(d), "l"(gmem), "f"(dep), "n"(BYTES) : "memory");
}
// Copies one lane's Raw element (4, 8, 16 or 32 bytes) with cp.async.
template <typename Raw>
__device__ __forceinline__ void cp_async_raw(Raw *smem, const void *gmem, float dep) {
    if constexpr (sizeof(Raw) == 32) {
        cp_async<16>(reinterpret_cast<char *>(smem), gmem, dep);
        cp_async<16>(reinterpret_cast<char *>(smem) + 16, static_cast<const char *>(gmem) + 16, dep);
    } else {
        cp_async<sizeof(Raw)>(smem, gmem, dep);
    }
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" :: "n"(N) : "memory"); }

// ---------------------------------------------------------------- lane input access
// LAYOUT 0: x is [T, B, N, K], a neuron's K compartments contiguous (one vector per lane).
// LAYOUT 1: the paper's layer layout [T, B, N / inner, K, inner] (channels C_o, then
//           compartments P, then the spatial positions), compartments `inner` apart; a
//           warp of consecutive neurons reads each compartment as one contiguous span.
template <typename XT, int KT, int LAYOUT> struct XIO;

template <typename XT, int KT> struct XIO<XT, KT, 0> {
    using Raw = typename Vec<XT, KT>::Raw;
    static constexpr bool kAsync = sizeof(Raw) >= 4;
    static __device__ __forceinline__ Raw load(const XT *p, int64_t) { return Vec<XT, KT>::load(p); }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) { Vec<XT, KT>::unpack(r, v); }
    static __device__ __forceinline__ void store(XT *p, int64_t, const float (&v)[KT]) { Vec<XT, KT>::store(p, v); }
    static __device__ __forceinline__ void copy_async(Raw *slot, const XT *p, int64_t, float dep) {
        cp_async_raw(slot, p, dep);
    }
};

template <int KT> struct XIO<float, KT, 1> {
    using Raw = typename Vec<float, KT>::Raw;
    static constexpr bool kAsync = true;
    static __device__ __forceinline__ Raw load(const float *p, int64_t ks) {
        float v[KT];
#pragma unroll
        for (int k = 0; k < KT; ++k) v[k] = __ldcs(p + k * ks);
        return Vec<float, KT>::pack(v);
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) { Vec<float, KT>::unpack(r, v); }
    static __device__ __forceinline__ void store(float *p, int64_t ks, const float (&v)[KT]) {
#pragma unroll
        for (int k = 0; k < KT; ++k) __stcs(p + k * ks, v[k]);
    }
    static __device__ __forceinline__ void copy_async(Raw *slot, const float *p, int64_t ks, float dep) {
#pragma unroll
        for (int k = 0; k < KT; ++k) cp_async<4>(reinterpret_cast<float *>(slot) + k, p + k * ks, dep);
    }
};

template <int KT> struct XIO<__nv_bfloat16, KT, 1> {
    using T = __nv_bfloat16;
    using Raw = typename Vec<T, KT>::Raw;        // kept packed, as in the contiguous layout
    static constexpr bool kAsync = false;        // 2-byte elements: no cp.async
    static __device__ __forceinline__ uint32_t ld16(const T *p) {
        return __ldcs(reinterpret_cast<const unsigned short *>(p));
    }
    static __device__ __forceinline__ uint32_t ld2(const T *p, int64_t ks) {
        return ld16(p) | (ld16(p + ks) << 16);
    }
    static __device__ __forceinline__ Raw load(const T *p, int64_t ks) {
        if constexpr (KT == 8)
            return make_uint4(ld2(p, ks), ld2(p + 2 * ks, ks), ld2(p + 4 * ks, ks), ld2(p + 6 * ks, ks));
        else if constexpr (KT == 4) return make_uint2(ld2(p, ks), ld2(p + 2 * ks, ks));
        else if constexpr (KT == 2) return ld2(p, ks);
        else return (unsigned short)ld16(p);
    }
    static __device__ __forceinline__ void unpack(const Raw &r, float (&v)[KT]) { Vec<T, KT>::unpack(r, v); }
    static __device__ __forceinline__ void store(T *p, int64_t ks, const float (&v)[KT]) {
#pragma unroll
        for (int k = 0; k < KT; ++k) {
            __nv_bfloat16 h = __float2bfloat16_rn(v[k]);
            __stcs(reinterpret_cast<unsigned short *>(p + k * ks), *reinterpret_cast<unsigned short *>(&h));
        }
    }
    static __device__ __forceinline__ void copy_async(Raw *, const T *, int64_t, float) {}
};

// Offset of lane `sub`'s first compartment of neuron j (steps add T-multiples of B*N*K).
template <int LAYOUT>
__device__ __forceinline__ int64_t lane_x_offset(int64_t j, int sub, int KT, int K, int inner) {
    if constexpr (LAYOUT == 0) return j * K + (int64_t)sub * KT;
    const int64_t s = j % inner;
    return (j - s) * K + s + (int64_t)sub * KT * inner;
}

// x is fetched fwd_depth() steps ahead of use through the cp.async ring (or, without it, a
// ring of kFwdBatch registers); checkpoints every g.L steps (g.L is a power of two and a
// multiple of the batch).
// Lanes of 8 compartments: 2 blocks per SM (the 3-block register cap spills: bf16 15%
// slower, float32 with per-neuron masks 4% slower, float32 without them 1% slower).
template <int K, int G, int PSI, typename XT, int LAYOUT>
__global__ void __launch_bounds__(fwd_threads(K), lane_compartments(K) >= 8 ? 2 : DENDSN_FWD_MINB)
dendsn_forward_kernel(const FwdArgs A) {
    pdl_wait();
    constexpr int NT = fwd_threads(K);
    constexpr int KT = lane_compartments(K);
    constexpr int LPN = K / KT;
    constexpr int L = kFwdBatch;
    using V = XIO<XT, KT, LAYOUT>;
    using AR = Arith<KT, G, PSI, XT>;
    constexpr bool ASYNC = DENDSN_FWD_ASYNC && V::kAsync;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    if (pos.nrows == 0) return;                  // whole warps: rows are uniform per warp
    typename AR::LP lp;
    AR::load(P, g, pos.chan, pos.sub, lp);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nb = (T + L - 1) / L;              // batches per row
    const int64_t sX = g.BN * K;                 // x elements between steps
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;   // first neuron of this thread
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;                // x elements between this thread's rows
    const int64_t ks = LAYOUT == 0 ? 1 : g.inner;   // distance between a lane's compartments
    const XT *__restrict__ xrow = static_cast<const XT *>(A.x) +
                                  lane_x_offset<LAYOUT>(j0, pos.sub, KT, K, g.inner);
    XT *__restrict__ srow = static_cast<XT *>(A.spikes) + j0;
    float *vrow = A.v_out ? A.v_out + j0 : nullptr;
    // the kept V^s arises only for layers of the phased backward (one 8-compartment lane per
    // neuron, compartments innermost); elsewhere krow is null at compile time
    constexpr bool can_keep = K == 8 && G == 1 && LAYOUT == 0 && std::is_same<XT, __nv_bfloat16>::value;
    float *krow = (can_keep && A.vs_keep) ? A.vs_keep + j0 : nullptr;
    const bool write_ck = (A.ck_vd != nullptr) && g.n_ck > 0 && pos.active;
    const bool store = pos.active && pos.sub == 0;
    const bool residual = P.residual != 0;

    if constexpr (ASYNC) {
        // Inputs are staged through a ring of D shared-memory slots per thread, filled by
        // cp.async D steps ahead of use along this thread's (row, step) sequence; each
        // thread reads only its own slots.
        constexpr int D = fwd_depth<XT, typename V::Raw>();
        using Raw = typename V::Raw;
        // dynamic shared memory: the lanes' kappa (per-neuron masks only), then the ring
        extern __shared__ float4 fwd_smem[];
        Raw *ring = reinterpret_cast<Raw *>(reinterpret_cast<char *>(fwd_smem) +
                                            kappa_smem_bytes(P.mask_mode, AR::KTb, NT)) +
                    threadIdx.x;                                          // slot k at ring[k * NT]
        const XT *ip = xrow;                    // next step to fetch
        int it = 0, ir = 0;                     // its step and row
        const int64_t row_jump = rX - (int64_t)T * sX;
#pragma unroll
        for (int k = 0; k < D; ++k) {
            if (ir < pos.nrows) V::copy_async(ring + k * NT, ip, ks, 0.f);
            cp_async_commit();
            ip += sX;
            if (++it == T) { it = 0; ++ir; ip += row_jump; }
        }
        // The step loop is specialised on whether V^s and checkpoints are written and on
        // whether T divides the ring depth (then the step fetched D steps ahead is the
        // same step D/T rows further on: no walker needed).
        auto rows = [&](auto extra, auto div, auto tc, auto keep) {
            // EXTRA: V^s output and/or checkpoints requested (each still tested inside);
            // TC > 0: T == TC known at compile time (the step loop unrolls; slots are the
            // row's first slot plus the step); KEEP: V^s kept for the backward (A.vs_keep
            // non-null; a separate build, so that the other loops carry no test for it)
            constexpr bool EXTRA = decltype(extra)::value, DIV = decltype(div)::value;
            constexpr int TC = decltype(tc)::value;
            constexpr bool KEEP = decltype(keep)::value;
            int slot = 0;
            int64_t j = j0;
            const int rows_ahead = DIV ? D / T : 0;
            const int64_t ahead = (int64_t)rows_ahead * rX;
            const XT *xr = xrow;
            XT *sr = srow;
            float *vr = vrow;
            float *kr = KEEP ? krow : nullptr;
            MaskAhead<AR, NT> mask;
            mask.init(P, g, j0, jstep, pos.chan, pos.sub, pos.nrows, fwd_smem);
            for (int i = 0; i < pos.nrows; ++i) {
                mask.advance(P, g, pos.sub, i + 1 < pos.nrows, lp);
                typename AR::St vd;
                AR::zero(vd);
                float v = 0.f;
                bool s = false;
                XT *sp = sr;
                float *vp = vr;
                float *kp = kr;
                const XT *cp = xr;                       // this step's x in global memory
                const bool fetch_row = i + rows_ahead < pos.nrows;
                auto step = [&](int t, int sl) {
                    cp_async_wait<D - 1>();
                    float xv[KT];
                    V::unpack(ring[sl * NT], xv);
                    const float z = soma_input<AR, KT, LPN>(lp, vd, xv, residual, inv_k);
                    // the slot's value has been used (z depends on it): refill it
                    if constexpr (DIV) {
                        if (fetch_row) V::copy_async(ring + sl * NT, cp + ahead, ks, z);
                        cp += sX;
                    } else {
                        if (ir < pos.nrows) V::copy_async(ring + sl * NT, ip, ks, z);
                        ip += sX;
                        if (++it == T) { it = 0; ++ir; ip += row_jump; }
                    }
                    cp_async_commit();
                    v = soma_charge(z, v, s, P);
                    s = v >= P.theta;                      // Eq. methods-lif-fire
                    if (store) {
                        Scalar<XT>::store_spike(sp, s);
                        if constexpr (EXTRA) {
                            if (vp) __stcs(vp, v);
                        }
                        if constexpr (KEEP) __stcs(kp, v);
                    }
                    sp += BN;
                    if constexpr (KEEP) kp += BN;
                    if constexpr (EXTRA) {
                        if (vp) vp += BN;
                        if (write_ck && ((t + 1) & (g.L - 1)) == 0 && t + 1 < T) {
                            const int ck = (t + 1) / g.L - 1;
                            float vda[KT];
                            AR::to_array(vd, vda);
                            Vec<float, KT>::store(A.ck_vd + ((int64_t)ck * BN + j) * K + pos.sub * KT, vda);
                            if (pos.sub == 0) __stcs(A.ck_vs + (int64_t)ck * BN + j, v);
                        }
                    }
                };
                if constexpr (TC > 0) {
#pragma unroll
                    for (int t = 0; t < TC; ++t) step(t, slot + t);
                    slot = (slot + TC == D) ? 0 : slot + TC;
                } else {
                    for (int t = 0; t < T; ++t) {
                        step(t, slot);
                        slot = (slot == D - 1) ? 0 : slot + 1;
                    }
                }
                xr += rX;
                sr += jstep;
                if constexpr (EXTRA) {
                    if (vr) vr += jstep;
                }
                if constexpr (KEEP) kr += jstep;
                j += jstep;
            }
        };
        using yes = std::true_type;
        using no = std::false_type;
        using tc0 = std::integral_constant<int, 0>;
        using tc4 = std::integral_constant<int, 4>;
        using tc8 = std::integral_constant<int, 8>;
        const bool div = (D % T) == 0;
        const bool keep = can_keep && krow != nullptr;
        if (vrow != nullptr || write_ck || (keep && !(div && (T == 4 || T == 8)))) {
            if constexpr (can_keep) {
                if (keep) {
                    if (div) rows(yes{}, yes{}, tc0{}, yes{}); else rows(yes{}, no{}, tc0{}, yes{});
                    cp_async_wait<0>();
                    return;
                }
            }
            if (div) rows(yes{}, yes{}, tc0{}, no{}); else rows(yes{}, no{}, tc0{}, no{});
        } else if (div) {
            if (T == 4) {
                if constexpr (can_keep) {
                    if (keep) rows(no{}, yes{}, tc4{}, yes{}); else rows(no{}, yes{}, tc4{}, no{});
                } else {
                    rows(no{}, yes{}, tc4{}, no{});
                }
            } else if (T == 8) {
                if constexpr (can_keep) {
                    if (keep) rows(no{}, yes{}, tc8{}, yes{}); else rows(no{}, yes{}, tc8{}, no{});
                } else {
                    rows(no{}, yes{}, tc8{}, no{});
                }
            } else {
                rows(no{}, yes{}, tc0{}, no{});
            }
        } else {
            rows(no{}, no{}, tc0{}, no{});
        }
        pdl_trigger();
        cp_async_wait<0>();
        return;
    }

    typename V::Raw xb[L];
    {
        const XT *p = xrow;
#pragma unroll
        for (int tt = 0; tt < L; ++tt) {
            if (tt < T) xb[tt] = V::load(p, ks);
            p += sX;
        }
    }
    int64_t j = j0;
    extern __shared__ float4 fwd_smem[];         // the lanes' kappa (per-neuron masks only)
    MaskAhead<AR, NT> mask;
    mask.init(P, g, j0, jstep, pos.chan, pos.sub, pos.nrows, fwd_smem);
    for (int i = 0; i < pos.nrows; ++i) {
        mask.advance(P, g, pos.sub, i + 1 < pos.nrows, lp);
        typename AR::St vd;
        AR::zero(vd);
        float v = 0.f;
        bool s = false;
        XT *sp = srow;
        float *vp = vrow;
        float *kp = krow;
        for (int c = 0; c < nb; ++c) {
            const int t0 = c * L;
            const int ncur = min(L, T - t0);                       // steps of this batch
            const bool same_row = c + 1 < nb;
            const bool has_next = same_row || (i + 1 < pos.nrows);
            // next batch: later in this row, or the start of the next row
            const XT *xn = same_row ? xrow + (int64_t)(t0 + L) * sX : xrow + rX;
            const int nnext = !has_next ? 0 : (same_row ? min(L, T - t0 - L) : min(L, T));
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float xv[KT];
                V::unpack(xb[tt], xv);
                // refill slot tt right after its value is taken
                if (tt < nnext) xb[tt] = V::load(xn, ks);
                xn += sX;
                if (tt < ncur) {
                    const float z = soma_input<AR, KT, LPN>(lp, vd, xv, residual, inv_k);
                    v = soma_charge(z, v, s, P);
                    s = v >= P.theta;                      // Eq. methods-lif-fire
                    if (store) {
                        Scalar<XT>::store_spike(sp, s);
                        if (vp) __stcs(vp, v);
                        if (kp) __stcs(kp, v);
                    }
                    sp += BN;
                    if (vp) vp += BN;
                    if (kp) kp += BN;
                }
            }
            if (write_ck && t0 + L < T && ((t0 + L) & (g.L - 1)) == 0) {
                const int ck = (t0 + L) / g.L - 1;
                float vda[KT];
                AR::to_array(vd, vda);
                Vec<float, KT>::store(A.ck_vd + ((int64_t)ck * BN + j) * K + pos.sub * KT, vda);
                if (pos.sub == 0) __stcs(A.ck_vs + (int64_t)ck * BN + j, v);
            }
        }
        xrow += rX;
        srow += jstep;
        if (vrow) vrow += jstep;
        if (krow) krow += jstep;
        j += jstep;
    }
}

// Forward in the paper's (C_o, P, H, W) layout with the inputs staged per warp. Used when a
// lane serves a whole neuron (K <= 8) and H*W and the column tile are multiples of 32: a
// warp's 32 neurons are then 32 consecutive positions of one channel group, so compartment k
// of all of them is one contiguous run of 32 elements. Each lane copies its share of the
// warp's K runs with 16-byte cp.async into the slot [k][32 lanes] (one copy per lane per
// step for 4 float32 compartments, as in the compartments-innermost layout) and reads back
// its own neuron's K values. Ordering: every lane waits for its own copy groups, then
// __syncwarp() makes all lanes' copies visible; a slot is refilled one step after it was
// read, behind that same barrier, so kFwdDepth - 1 steps are in flight.
template <int K, int G, int PSI, typename XT>
__global__ void __launch_bounds__(fwd_threads(K), K >= 8 ? 2 : DENDSN_FWD_MINB)
dendsn_forward_staged_kernel(const FwdArgs A) {
    pdl_wait();
    constexpr int NT = fwd_threads(K);
    constexpr int KT = K;                        // one lane per neuron
    constexpr int D = kFwdDepth;
    constexpr int SX = (int)sizeof(XT);
    constexpr int EPC = 16 / SX;                 // elements per 16-byte chunk
    constexpr int CPK = 32 / EPC;                // chunks per compartment run of a warp
    constexpr int NCH = K * CPK;                 // chunks per warp per step
    constexpr int CPL = (NCH + 31) / 32;         // chunks per lane
    using AR = Arith<KT, G, PSI, XT>;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<1>(g);
    // whole warps: rows are uniform per warp, and P % 32 == 0 makes activity uniform too
    if (pos.nrows == 0 || !pos.active) return;
    typename AR::LP lp;
    AR::load(P, g, pos.chan, 0, lp);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int64_t sX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;
    const int lane = threadIdx.x & 31;
    // the warp's first neuron: 32-aligned position, so every chunk is 16-byte aligned
    const XT *xw = static_cast<const XT *>(A.x) + lane_x_offset<1>(j0, 0, KT, K, g.inner) - lane;
    XT *sp = static_cast<XT *>(A.spikes) + j0;
    float *vp = A.v_out ? A.v_out + j0 : nullptr;
    const bool write_ck = (A.ck_vd != nullptr) && g.n_ck > 0;
    const bool residual = P.residual != 0;

    // dynamic shared memory: the lanes' kappa (per-neuron masks only), then the slots
    extern __shared__ float4 fwd_smem[];
    constexpr int kSlot = NT * K;                // elements of one slot (all warps)
    XT *wring = reinterpret_cast<XT *>(reinterpret_cast<char *>(fwd_smem) +
                                       kappa_smem_bytes(P.mask_mode, AR::KTb, NT)) +
                (threadIdx.x >> 5) * (32 * K);
    int64_t src[CPL];
    int dst[CPL];
#pragma unroll
    for (int m = 0; m < CPL; ++m) {
        const int c = lane + 32 * m;
        const int kc = c / CPK, pc = c % CPK;
        src[m] = (int64_t)kc * g.inner + pc * EPC;
        dst[m] = kc * 32 + pc * EPC;
    }
    auto fetch = [&](int slot, const XT *base) {
#pragma unroll
        for (int m = 0; m < CPL; ++m)
            if (lane + 32 * m < NCH) cp_async<16>(wring + slot * kSlot + dst[m], base + src[m], 0.f);
    };
    // fetch walker over this thread's (row, step) sequence
    const XT *ip = xw;
    int it = 0, ir = 0;
    const int64_t row_jump = rX - (int64_t)T * sX;
    auto walk = [&]() {
        ip += sX;
        if (++it == T) { it = 0; ++ir; ip += row_jump; }
    };
#pragma unroll
    for (int k = 0; k < D - 1; ++k) {
        if (ir < pos.nrows) fetch(k, ip);
        cp_async_commit();
        walk();
    }
    int slot = 0;
    int64_t j = j0;
    MaskAhead<AR, NT> mask;
    mask.init(P, g, j0, jstep, pos.chan, 0, pos.nrows, fwd_smem);
    for (int i = 0; i < pos.nrows; ++i) {
        mask.advance(P, g, 0, i + 1 < pos.nrows, lp);
        typename AR::St vd;
        AR::zero(vd);
        float v = 0.f;
        bool s = false;
        XT *spt = sp;
        float *vpt = vp;
        for (int t = 0; t < T; ++t) {
            cp_async_wait<D - 2>();
            __syncwarp();
            // refill the slot every lane read in the previous step
            if (ir < pos.nrows) fetch(slot == 0 ? D - 1 : slot - 1, ip);
            cp_async_commit();
            walk();
            float xv[KT];
#pragma unroll
            for (int k = 0; k < KT; ++k) {
                if constexpr (SX == 4) xv[k] = reinterpret_cast<const float *>(wring)[slot * kSlot + k * 32 + lane];
                else xv[k] = bf16_lo(reinterpret_cast<const unsigned short *>(wring)[slot * kSlot + k * 32 + lane]);
            }
            const float z = soma_input<AR, KT, 1>(lp, vd, xv, residual, inv_k);
            v = soma_charge(z, v, s, P);
            s = v >= P.theta;                    // Eq. methods-lif-fire
            Scalar<XT>::store_spike(spt, s);
            if (vpt) {
                __stcs(vpt, v);
                vpt += BN;
            }
            spt += BN;
            if (write_ck && ((t + 1) & (g.L - 1)) == 0 && t + 1 < T) {
                const int ck = (t + 1) / g.L - 1;
                float vda[KT];
                AR::to_array(vd, vda);
                Vec<float, KT>::store(A.ck_vd + ((int64_t)ck * BN + j) * K, vda);
                __stcs(A.ck_vs + (int64_t)ck * BN + j, v);
            }
            slot = (slot == D - 1) ? 0 : slot + 1;
        }
        sp += jstep;
        if (vp) vp += jstep;
        j += jstep;
    }
    cp_async_wait<0>();
}

// ---------------------------------------------------------------- backward
// Rows of the reduction buffer are NT + 1 floats apart, so that the threads of a warp that
// read one entry of consecutive gradient slots hit consecutive banks (rows NT apart would
// put all of them in one bank).
template <int NT> constexpr int red_stride() { return NT + 1; }
// Bytes of shared memory block_partials needs for NA1 gradient slots.
constexpr size_t red_bytes(int NA1, int NT) { return sizeof(float) * (size_t)NA1 * (NT + 1); }

// Per-channel partial sums of a block's parameter-gradient vectors v (one per thread,
// [alpha KT | xi KT | zeta KTb | kappa KTb | beta]) in a fixed order: segmented warp
// shuffles over the columns of one channel, then the run leaders in shared memory (red,
// red_bytes(NA1, NT)), one partial per (block, channel) to `partials`.
template <int KT, int G, int LPN, int NT, int NA1>
__device__ __forceinline__ void block_partials(const Geometry &g, const ThreadPos &pos,
                                               float (&v)[NA1], float *red, float *partials) {
    constexpr int KTb = KT / G;
    constexpr int NA = NA1 - 1;
    constexpr int RS = red_stride<NT>();
    // stage 1: within a warp, columns of one channel come in aligned runs of g.seg
    for (int d = 1; d < g.seg; d <<= 1) {
#pragma unroll
        for (int a = 0; a < NA1; ++a)
            v[a] = __fadd_rn(v[a], __shfl_xor_sync(0xffffffffu, v[a], d * LPN));
    }
    // stage 2: run leaders meet in shared memory; red[a][tid] (reuses the history space)
    __syncthreads();
#pragma unroll
    for (int a = 0; a < NA1; ++a) red[a * RS + threadIdx.x] = v[a];
    __syncthreads();
    const int ct = blockIdx.x % g.nCT;
    const int p0 = ct * g.TXn;
    const int p1 = min(p0 + g.TXn, g.P);            // exclusive
    const int c_lo = p0 / g.inner;
    const int nch = (p1 - 1) / g.inner - c_lo + 1;
    const int NP = 2 * g.K + 2 * g.Kb + 1;          // per-channel gradient vector
    float *out = partials + (int64_t)blockIdx.x * g.nch_max * NP;
    const int items = nch * LPN * NA1;
    for (int w = threadIdx.x; w < items; w += NT) {
        const int a = w % NA1;
        const int sub = (w / NA1) % LPN;
        const int lc = w / (NA1 * LPN);
        if (a == NA && sub > 0) continue;          // beta: one lane per neuron
        const int c = c_lo + lc;
        const int cx_lo = max(c * g.inner, p0) - p0;
        const int cx_hi = min((c + 1) * g.inner, p1) - p0;
        float sum = 0.f;
        for (int ry = 0; ry < g.TY; ++ry)
            for (int cx = cx_lo; cx < cx_hi; cx += g.seg)
                sum = __fadd_rn(sum, red[a * RS + (ry * g.TXn + cx) * LPN + sub]);
        int slot;
        if (a < KT) slot = sub * KT + a;                                        // alpha
        else if (a < 2 * KT) slot = g.K + sub * KT + (a - KT);                  // xi
        else if (a < 2 * KT + KTb) slot = 2 * g.K + sub * KTb + (a - 2 * KT);   // zeta
        else if (a < NA) slot = 2 * g.K + g.Kb + sub * KTb + (a - 2 * KT - KTb); // kappa
        else slot = NP - 1;                                                     // beta
        out[lc * NP + slot] = sum;
    }
}

template <int KT, int G>
constexpr int acc_count() { return 2 * KT + 2 * (KT / G); }

// Whether the chunked backward keeps two-level parameter-gradient sums for rows of several
// chunks (L == 8): all builds but eight float32 compartments per lane, whose totals would
// take the shared memory of one of their three resident blocks per SM.
template <int K, int G, typename XT, int L>
constexpr bool row_totals() {
    return L > 4 && !(bwd_lane_compartments(K, G, xt_code<XT>(), L) >= 8 && std::is_same<XT, float>::value);
}

// BETA: also accumulate dL/dbeta (a learnable somatic decay); a separate instance because
// even one more live accumulator slows the register-history path measurably.
// FULL: T is a multiple of L, so every chunk has exactly L steps; the step loops then carry
// no bounds tests, and when the x ring is one chunk deep (kBwdDepth == L) the slot of step
// tt is tt and the step it prefetches is step tt of the next chunk (no ring walker).
template <int K, int G, int PSI, typename XT, int L, int LAYOUT, bool BETA, bool FULL>
__global__ void __launch_bounds__(bwd_threads(bwd_lane_compartments(K, G, xt_code<XT>(), L)),
                                  bwd_threads(bwd_lane_compartments(K, G, xt_code<XT>(), L)) == 128 ? 3 : 2)
dendsn_backward_kernel(const BwdArgs A) {
    pdl_wait();
    constexpr int KT = bwd_lane_compartments(K, G, xt_code<XT>(), L);
    constexpr int NT = bwd_threads(KT);
    constexpr int LPN = K / KT;
    constexpr int KTb = KT / G;
    constexpr int NA = acc_count<KT, G>();
    // L == 4 is only used for T <= 4: one chunk per row and never a checkpoint
    constexpr bool MULTI = L > 4;
    // the recomputed history lives in shared memory for multi-chunk rows and for
    // 8-compartment lanes (registers), else in registers
    constexpr bool SHIST = MULTI || KT >= 8;
    constexpr int H = 4;                         // prefetch distance of x in steps
    using V = XIO<XT, KT, LAYOUT>;
    using S1 = Scalar<XT>;
    using AR = Arith<KT, G, PSI, XT>;
    using HistRaw = typename Vec<float, KT>::Raw;
    using XRaw = typename V::Raw;
    // x staged through a per-thread cp.async ring in shared memory when the history is
    // there too; otherwise (T <= 4, up to 4 compartments) a register ring, which
    // measured faster there
    constexpr bool BASYNC = DENDSN_BWD_ASYNC && SHIST && V::kAsync;
    constexpr int D = kBwdDepth;
    constexpr bool SLOTS = FULL && BASYNC && D == L;
    // float32 dL/dS of the next chunk reaches shared memory by cp.async as each slot of the
    // current chunk is taken (event-stream layer backward 1608 -> 1531 us; for the
    // register-history builds it measured slower: conv layer 217.6 -> 221.8 us)
    constexpr bool GSA = std::is_same<XT, float>::value && SLOTS;
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    typename AR::LP lp;
    AR::load(P, g, pos.chan, pos.sub, lp);
    const float inv_k = 1.f / (float)K;
    const int T = g.T;
    const int nc = MULTI ? (T + L - 1) / L : 1;  // chunks per row
    const int64_t sX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;
    const int64_t ks = LAYOUT == 0 ? 1 : g.inner;   // distance between a lane's compartments
    const int64_t xoff = lane_x_offset<LAYOUT>(j0, pos.sub, KT, K, g.inner);
    const XT *__restrict__ xrow = static_cast<const XT *>(A.x) + xoff;
    const XT *__restrict__ gsrow = static_cast<const XT *>(A.gs) + j0;
    XT *__restrict__ gxrow = static_cast<XT *>(A.gx) + xoff;
    const float *gvrow = A.gv ? A.gv + j0 : nullptr;
    // dV[t+1]/dS[t] = kv V[t] + cs: hard -beta V[t], soft -beta theta, 0 when detached;
    // dV[t+1]/dV[t] = beta, or b_spike after a spike (0 hard, beta soft)
    const float kv = (P.detach || P.soft) ? 0.f : -P.beta;
    const float cs = (P.detach || !P.soft) ? 0.f : -P.beta * P.theta;
    const float b_spike = P.soft ? P.beta : 0.f;
    const bool residual = P.residual != 0;
    const bool has_gv = A.gv != nullptr;

    // dynamic shared memory: the lanes' kappa (per-neuron masks only), then the history,
    // V^s history and x ring, or (at the end) the reduction
    extern __shared__ float4 smem_f4[];
    char *const sregion = reinterpret_cast<char *>(smem_f4) + kappa_smem_bytes(P.mask_mode, KTb, NT);
    HistRaw *hist = reinterpret_cast<HistRaw *>(sregion);                             // [L][NT]
    float *hist_vs = reinterpret_cast<float *>(hist + (SHIST ? L * NT : 0));   // [L][NT]
    XRaw *xring = reinterpret_cast<XRaw *>(hist_vs + (SHIST ? L * NT : 0)) + threadIdx.x;   // [D][NT]
    // rows of several chunks: the parameter-gradient terms of each row are summed on their
    // own and the row sums added into per-thread totals [kAccFloats + 1][NT] after the x ring
    // (a two-level sum: float32 rounding grows with the terms of one row, not of all rows)
    constexpr bool TOTALS = row_totals<K, G, XT, L>();
    float *const tot = reinterpret_cast<float *>(reinterpret_cast<char *>(hist_vs + (SHIST ? L * NT : 0)) +
                                                 (BASYNC ? sizeof(XRaw) * D * NT : 0)) + threadIdx.x;
    const bool use_tot = TOTALS && nc > 1;
    float *const gring = reinterpret_cast<float *>(reinterpret_cast<char *>(tot - threadIdx.x) +
                                                   (TOTALS ? sizeof(float) * (AR::kAccFloats + 1) * NT : 0)) +
                         threadIdx.x;                                                // [L][NT]
    if (use_tot) {
#pragma unroll
        for (int q = 0; q <= AR::kAccFloats; ++q) tot[q * NT] = 0.f;
    }
    // cp.async walker over this thread's sequence: rows, chunks in reverse, steps forward
    const XT *const xbase = xrow;
    int wr = 0, wc = nc - 1, wt = 0;
    int wlen = min(L, T - wc * L);
    const XT *wp = xbase + (int64_t)wc * L * sX;
    auto walk = [&]() {
        if (++wt == wlen) {
            wt = 0;
            if (--wc < 0) { wc = nc - 1; ++wr; }
            wlen = min(L, T - wc * L);
            wp = xbase + wr * rX + (int64_t)wc * L * sX;
        } else {
            wp += sX;
        }
    };
    int xslot = 0;
    if constexpr (BASYNC) {
#pragma unroll
        for (int k = 0; k < D; ++k) {
            if (wr < pos.nrows) V::copy_async(xring + k * NT, wp, ks, 0.f);
            cp_async_commit();
            walk();
        }
    }

    typename AR::Acc acc;
    AR::acc_zero(acc);
    float gbeta = 0.f;                // dL/dbeta (PLIF soma): sum of dL/dV^s[t+1] * leak[t]

    XRaw xb[BASYNC ? 1 : H];          // register ring: x of the next H steps to recompute
    typename S1::Raw gsb[L];          // grad_spikes of the current chunk
    float ckd[KT];                    // checkpoint V^d entering the current chunk
    float ckv = 0.f;                  // checkpoint V^s entering the current chunk
#pragma unroll
    for (int i = 0; i < KT; ++i) ckd[i] = 0.f;
    if (pos.nrows > 0) {
        const int t0 = (nc - 1) * L;
        const XT *p = xrow + (int64_t)t0 * sX;
        const XT *q = gsrow + (int64_t)t0 * BN;
#pragma unroll
        for (int tt = 0; tt < L; ++tt) {
            if (t0 + tt < T) {
                if (!BASYNC && tt < H) xb[(!BASYNC && tt < H) ? tt : 0] = V::load(p, ks);
                if constexpr (GSA) cp_async<4>(gring + tt * NT, q, 0.f);
                else gsb[tt] = S1::load(q);
            }
            p += sX;
            q += BN;
        }
        if (MULTI && nc > 1) {
            Vec<float, KT>::unpack(Vec<float, KT>::load(
                A.ck_vd + ((int64_t)(nc - 2) * BN + j0) * K + pos.sub * KT), ckd);
            ckv = __ldcs(A.ck_vs + (int64_t)(nc - 2) * BN + j0);
        }
    }
    if constexpr (GSA) cp_async_commit();

    int64_t j = j0;
    MaskAhead<AR, NT> mask;
    mask.init(P, g, j0, jstep, pos.chan, pos.sub, pos.nrows, smem_f4);
    for (int i = 0; i < pos.nrows; ++i) {
        mask.advance(P, g, pos.sub, i + 1 < pos.nrows, lp);
        typename AR::St Ad;           // dL/dV^d[t+1], carried backwards
        AR::zero(Ad);
        float dvn = 0.f;              // dL/dV^s[t+1]
        for (int c = nc - 1; c >= 0; --c) {
            const int t0 = c * L;
            const int ncur = FULL ? L : min(L, T - t0);
            // state entering the chunk: zero at t = 0, else the forward's checkpoint
            typename AR::St vd0;
            if (!MULTI || c == 0) {
                AR::zero(vd0);
            } else {
                AR::from_array(vd0, ckd);
            }
            const float v0 = (!MULTI || c == 0) ? 0.f : ckv;
            // next chunk: the previous chunk of this row, or the last chunk of the next row
            const bool same_row = MULTI && c > 0;
            const bool has_next = same_row || (i + 1 < pos.nrows);
            const int cn = same_row ? c - 1 : nc - 1;
            const int tn = cn * L;
            const int nnext = has_next ? (FULL ? L : min(L, T - tn)) : 0;
            const int64_t jn = same_row ? j : j + jstep;
            const XT *xn = (same_row ? xrow : xrow + rX) + (int64_t)tn * sX;
            const XT *gsn = (same_row ? gsrow : gsrow + jstep) + (int64_t)tn * BN;
            if (MULTI && has_next && cn > 0) {
                Vec<float, KT>::unpack(Vec<float, KT>::load(
                    A.ck_vd + ((int64_t)(cn - 1) * BN + jn) * K + pos.sub * KT), ckd);
                ckv = __ldcs(A.ck_vs + (int64_t)(cn - 1) * BN + jn);
            }

            // recompute the chunk, keeping V^d and V^s of every step (in registers for a
            // single chunk, in shared memory, one slot per thread and step, otherwise)
            typename AR::St vdh[SHIST ? 1 : L];
            float vsh[SHIST ? 1 : L];
            float gsc[SHIST ? 1 : L];     // register history: grad_spikes taken during the recompute
            {
                typename AR::St vd = vd0;
                float v = v0;
                bool s = (!MULTI || c == 0) ? false : (v0 >= P.theta);
                const XT *xa = xrow + (int64_t)(t0 + H) * sX;      // this chunk, H steps ahead
                const XT *xnn = xn;                                 // next chunk, from its start
                const XT *gq = gsn;                                 // next chunk's grad_spikes
#pragma unroll
                for (int tt = 0; tt < L; ++tt) {
                    float xv[KT];
                    if constexpr (!BASYNC) V::unpack(xb[BASYNC ? 0 : tt % H], xv);
                    if constexpr (!SHIST) {
                        gsc[SHIST ? 0 : tt] = S1::unpack(gsb[tt]);
                        if (tt < nnext) gsb[tt] = S1::load(gq);
                        gq += BN;
                    }
                    if constexpr (!BASYNC) {
                        // refill the slot with the step H ahead: later in this chunk, or
                        // the first steps of the next chunk
                        if (tt + H < L) {
                            if (tt + H < ncur) xb[BASYNC ? 0 : tt % H] = V::load(xa, ks);
                            xa += sX;
                        } else {
                            if (tt + H - L < nnext) xb[BASYNC ? 0 : tt % H] = V::load(xnn, ks);
                            xnn += sX;
                        }
                    }
                    if (tt < ncur) {
                        if constexpr (BASYNC) {
                            cp_async_wait<D - 1>();
                            V::unpack(xring[(SLOTS ? tt : xslot) * NT], xv);
                        }
                        const float z = soma_input<AR, KT, LPN>(lp, vd, xv, residual, inv_k);
                        if constexpr (SLOTS) {
                            // the slot's value has been used (z depends on it): refill it
                            // with the same step of the next chunk
                            if (has_next) V::copy_async(xring + tt * NT, xn + (int64_t)tt * sX, ks, z);
                            cp_async_commit();
                        } else if constexpr (BASYNC) {
                            if (wr < pos.nrows) V::copy_async(xring + xslot * NT, wp, ks, z);
                            cp_async_commit();
                            walk();
                            xslot = (xslot == D - 1) ? 0 : xslot + 1;
                        }
                        v = soma_charge(z, v, s, P);
                        s = v >= P.theta;
                        if constexpr (SHIST) {
                            float vda[KT];
                            AR::to_array(vd, vda);
                            hist[tt * NT + threadIdx.x] = Vec<float, KT>::pack(vda);
                            hist_vs[tt * NT + threadIdx.x] = v;
                        } else {
                            vdh[SHIST ? 0 : tt] = vd;
                            vsh[SHIST ? 0 : tt] = v;
                        }
                    }
                }
            }
            // reverse-time recursion over the chunk
            XT *gxp = gxrow + (int64_t)(t0 + L - 1) * sX;
            const float *gvp = has_gv ? gvrow + (int64_t)(t0 + L - 1) * BN : nullptr;
            const XT *gqr = gsn + (int64_t)(L - 1) * BN;            // next chunk's grad_spikes
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                float gs_t;
                if constexpr (GSA) {
                    gs_t = gring[tt * NT];
                    if (tt < nnext) cp_async<4>(gring + tt * NT, gqr, gs_t);
                    gqr -= BN;
                } else if constexpr (SHIST) {
                    gs_t = S1::unpack(gsb[tt]);
                    // refill slot tt with the next chunk's grad_spikes once this one is taken
                    if (tt < nnext) gsb[tt] = S1::load(gqr);
                    gqr -= BN;
                } else {
                    gs_t = gsc[SHIST ? 0 : tt];
                }
                if (tt < ncur) {
                    float vs;
                    typename AR::St vdt, vdp;                       // V^d[t], V^d[t-1]
                    if constexpr (SHIST) {
                        vs = hist_vs[tt * NT + threadIdx.x];
                        float a[KT];
                        Vec<float, KT>::unpack(hist[tt * NT + threadIdx.x], a);
                        AR::from_array(vdt, a);
                        if (tt > 0) {
                            Vec<float, KT>::unpack(hist[(tt > 0 ? tt - 1 : 0) * NT + threadIdx.x], a);
                            AR::from_array(vdp, a);
                        } else {
                            vdp = vd0;
                        }
                    } else {
                        vs = vsh[SHIST ? 0 : tt];
                        vdt = vdh[SHIST ? 0 : tt];
                        vdp = (tt > 0) ? vdh[SHIST ? 0 : (tt > 0 ? tt - 1 : 0)] : vd0;
                    }
                    const bool st = vs >= P.theta;
                    if constexpr (BETA) {
                        // dV[t+1]/dbeta: (1 - S[t]) V[t] (hard) or V[t] - theta S[t] (soft)
                        const float leak = st ? (P.soft ? __fsub_rn(vs, P.theta) : 0.f) : vs;
                        gbeta = __fmaf_rn(dvn, leak, gbeta);
                    }
                    const float dvds = __fmaf_rn(kv, vs, cs);               // dV[t+1]/dS[t]
                    const float dvdv = st ? b_spike : P.beta;               // dV[t+1]/dV[t]
                    const float ds = __fmaf_rn(dvds, dvn, gs_t);                          // dL/dS[t]
                    float dv = __fmaf_rn(surrogate(__fsub_rn(vs, P.theta)), ds,
                                         __fmul_rn(dvdv, dvn));                          // dL/dV^s[t]
                    if (has_gv) dv = __fadd_rn(dv, __ldcs(gvp));
                    float gxv[KT];
                    AR::backward(lp, vdt, vdp, dv, Ad, acc, residual ? __fmul_rn(dv, inv_k) : 0.f, gxv);
                    if (pos.active) V::store(gxp, ks, gxv);
                    dvn = dv;
                }
                gxp -= sX;
                if (has_gv) gvp -= BN;
            }
            if constexpr (GSA) cp_async_commit();
        }
        if (use_tot) {
            AR::template acc_flush<NT>(acc, tot);
            tot[AR::kAccFloats * NT] = __fadd_rn(tot[AR::kAccFloats * NT], gbeta);
            gbeta = 0.f;
        }
        xrow += rX;
        gsrow += jstep;
        gxrow += rX;
        if (has_gv) gvrow += jstep;
        j += jstep;
    }
    if (use_tot) {
        AR::template acc_load<NT>(acc, tot);
        gbeta = tot[AR::kAccFloats * NT];
    }

    // ---- parameter-gradient partials: per channel, fixed summation order
    // (slot NA: beta, counted once per neuron, by its first lane)
    constexpr int NA1 = NA + 1;
    float v[NA1];
    float kap[AR::KTb] = {};
    if constexpr (AR::KAPPA_FREE) lane_kappa<AR::KTb>(P, g, pos.chan, pos.sub, kap);
    AR::acc_export(lp, acc, v, kap);
    v[NA] = (BETA && pos.sub == 0) ? gbeta : 0.f;
#pragma unroll
    for (int a = 0; a < NA1; ++a)
        if (!pos.active || (a < KT && P.stateless)) v[a] = 0.f;
    if constexpr (BASYNC || GSA) cp_async_wait<0>();
    pdl_trigger();
    block_partials<KT, G, LPN, NT>(g, pos, v, reinterpret_cast<float *>(sregion), A.partials);
}

// ---------------------------------------------------------------- phased backward
// The backward for rows that are one full chunk (T == L) of neurons served whole by one
// lane of 8 compartments (paired engine, G = 1, compartments innermost, no residual term;
// the deeper bf16 conv layer). dendsn_backward_kernel walks each reverse step over all of
// a lane's compartment pairs at once, so the adjoints, temporaries and history of every
// pair are live together; here a row runs in phases so that the reverse scan holds one
// pair at a time:
//   1. recompute the chunk step by step (the forward's own step function, so Z and the
//      spikes are bit-identical), writing V^d of every step and pair to shared memory;
//      then fetch the next row's x into the freed ring;
//   2. the soma in registers: V^s forward, then its reverse recursion for dL/dZ[t]
//      (Eqs. methods-lif-reset-charge, methods-lif-fire, methods-sg); then fetch the next
//      row's dL/dS;
//   3. pair by pair, the dendritic reverse scan over the chunk (the same per-pair step as
//      dendsn_backward_kernel); dL/dX[t] of a pair overwrites its V^d[t] slot, which the
//      scan no longer needs;
//   4. gather each step's dL/dX from shared memory and store it as one vector.
// Every accumulator sees its terms in the same order as in dendsn_backward_kernel, so
// the two kernels give bit-identical results.
// Resident blocks of the phased backward: 3 (168 registers). 4 blocks at a 128-register cap
// measured 3% slower on the deeper conv layer (552.6 -> 569.5 us; 4 bytes of spill, and the
// compiler gives up instruction-level parallelism for the extra warps).
#ifndef DENDSN_PHASED_MINB
#define DENDSN_PHASED_MINB 3
#endif
// GSA: dL/dS reaches shared memory by cp.async, one row ahead, instead of registers
// loaded one row ahead (deeper conv backward 549.4 -> 516.6 us: the register loads
// still held up the soma phase; two rows ahead measured slower, 520.7 -> 525.6 us, and
// x two rows ahead too, 529 us). For bfloat16 each thread copies the aligned 4-byte word
// holding its element and its neighbour's; the launcher takes this build only when those
// words lie inside each step's row (gs 4-byte aligned, B*N even), else the register one.
template <int K, int PSI, typename XT, int L, bool BETA, bool GSA>
__global__ void __launch_bounds__(bwd_threads(K), bwd_threads(K) == 128 ? DENDSN_PHASED_MINB : 2)
dendsn_backward_phased_kernel(const BwdArgs A) {
    pdl_wait();
    constexpr int KT = K;
    constexpr int NT = bwd_threads(KT);
    constexpr int N2 = KT / 2;
    constexpr int NA = acc_count<KT, 1>();
    using V = XIO<XT, KT, 0>;
    using S1 = Scalar<XT>;
    using AR = Arith<KT, 1, PSI, XT>;
    using XRaw = typename V::Raw;
    static_assert(KT % 2 == 0 && AR::KTb == KT, "paired engine only");
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<1>(g);
    typename AR::LP lp;
    AR::load(P, g, pos.chan, 0, lp);
    const int64_t sX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;
    const XT *__restrict__ xrow = static_cast<const XT *>(A.x) + j0 * K;
    const XT *__restrict__ gsrow = static_cast<const XT *>(A.gs) + j0;
    XT *__restrict__ gxrow = static_cast<XT *>(A.gx) + j0 * K;
    const float *gvrow = A.gv ? A.gv + j0 : nullptr;
    const float kv = (P.detach || P.soft) ? 0.f : -P.beta;
    const float cs = (P.detach || !P.soft) ? 0.f : -P.beta * P.theta;
    const float b_spike = P.soft ? P.beta : 0.f;
    const bool has_gv = A.gv != nullptr;

    // dynamic shared memory: the lanes' kappa (per-neuron masks only), then the history
    // [L][N2][NT] float2, the x ring [L][NT] and (GSA) the dL/dS ring [L][NT], or (at the
    // end) the reduction
    extern __shared__ float4 smem_f4[];
    char *const sregion = reinterpret_cast<char *>(smem_f4) + kappa_smem_bytes(P.mask_mode, KT, NT);
    float2 *const hist = reinterpret_cast<float2 *>(sregion) + threadIdx.x;
    XRaw *const xring = reinterpret_cast<XRaw *>(reinterpret_cast<float2 *>(sregion) + L * N2 * NT) +
                        threadIdx.x;
    // dL/dS of a row as L 4-byte words (for bfloat16 the word holding the thread's element
    // and its neighbour's)
    uint32_t *const gring = reinterpret_cast<uint32_t *>(reinterpret_cast<char *>(sregion) +
                                                         sizeof(float2) * L * N2 * NT +
                                                         sizeof(XRaw) * L * NT) + threadIdx.x;
    auto gs_word = [&](const XT *p) {
        return reinterpret_cast<const uint32_t *>(reinterpret_cast<uintptr_t>(p) & ~(uintptr_t)3);
    };
    // byte selector that moves the thread's bfloat16 half of a word to the top (exact)
    auto gs_sel = [&](const XT *p) -> uint32_t {
        if constexpr (std::is_same<XT, float>::value) return 0x3210u;
        else return ((reinterpret_cast<uintptr_t>(p) >> 1) & 1) ? 0x3244u : 0x1044u;
    };
    if (pos.nrows > 0) {
#pragma unroll
        for (int tt = 0; tt < L; ++tt) V::copy_async(xring + tt * NT, xrow + (int64_t)tt * sX, 1, 0.f);
        if constexpr (GSA) {
#pragma unroll
            for (int tt = 0; tt < L; ++tt) cp_async<4>(gring + tt * NT, gs_word(gsrow + (int64_t)tt * BN), 0.f);
        }
    }
    cp_async_commit();

    typename AR::Acc acc;
    AR::acc_zero(acc);
    float gbeta = 0.f;
    MaskAhead<AR, NT> mask;
    mask.init(P, g, j0, jstep, pos.chan, 0, pos.nrows, smem_f4);
    // without GSA: grad_spikes of the row in registers, used in phase 2; the next row's are
    // requested right after it
    typename S1::Raw gsr[L];
    if (!GSA && pos.nrows > 0) {
#pragma unroll
        for (int tt = 0; tt < L; ++tt) gsr[tt] = S1::load(gsrow + (int64_t)tt * BN);
    }
    for (int i = 0; i < pos.nrows; ++i) {
        mask.advance(P, g, 0, i + 1 < pos.nrows, lp);

        // phase 1: recompute
        cp_async_wait<0>();
        float z[L];
        {
            typename AR::St vd;
            AR::zero(vd);
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float xv[KT];
                V::unpack(xring[tt * NT], xv);
                z[tt] = AR::step(lp, vd, xv, false, 0.f);
#pragma unroll
                for (int m = 0; m < N2; ++m) hist[(tt * N2 + m) * NT] = vd.v[m];
            }
        }
        if (i + 1 < pos.nrows) {
#pragma unroll
            for (int tt = 0; tt < L; ++tt)
                V::copy_async(xring + tt * NT, xrow + rX + (int64_t)tt * sX, 1, z[L - 1]);
        }
        cp_async_commit();

        // phase 2: the soma forward, then dL/dV^s backwards in time (dL/dZ = dL/dV^s)
        float dz[L];
        {
            float v = 0.f;
            bool s = false;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                v = soma_charge(z[tt], v, s, P);
                s = v >= P.theta;
                z[tt] = v;                       // z now holds V^s
            }
            float dvn = 0.f;                     // dL/dV^s[t+1]
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float vs = z[tt];
                const bool st = vs >= P.theta;
                if constexpr (BETA) {
                    const float leak = st ? (P.soft ? __fsub_rn(vs, P.theta) : 0.f) : vs;
                    gbeta = __fmaf_rn(dvn, leak, gbeta);
                }
                const float dvds = __fmaf_rn(kv, vs, cs);
                const float dvdv = st ? b_spike : P.beta;
                const float gst = GSA ? __uint_as_float(__byte_perm(gring[tt * NT], 0u, gs_sel(gsrow)))
                                      : S1::unpack(gsr[tt]);
                const float ds = __fmaf_rn(dvds, dvn, gst);
                float dv = __fmaf_rn(surrogate(__fsub_rn(vs, P.theta)), ds, __fmul_rn(dvdv, dvn));
                if (has_gv) dv = __fadd_rn(dv, __ldcs(gvrow + (int64_t)tt * BN));
                dz[tt] = dv;
                dvn = dv;
            }
        }
        // the next row's dL/dS: into the ring once phase 2 has read it (dz[0] depends on
        // every read), else into the registers
        if (i + 1 < pos.nrows) {
            if constexpr (GSA) {
#pragma unroll
                for (int tt = 0; tt < L; ++tt)
                    cp_async<4>(gring + tt * NT, gs_word(gsrow + jstep + (int64_t)tt * BN), dz[0]);
            } else {
#pragma unroll
                for (int tt = 0; tt < L; ++tt) gsr[tt] = S1::load(gsrow + jstep + (int64_t)tt * BN);
            }
        }
        if constexpr (GSA) cp_async_commit();

        // phase 3: the dendritic reverse scan, one pair at a time
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            const float2 kmz = fmul2(lp.km[m], lp.iz[m]);
            float2 Ad = f2(0.f);
            float2 vdt = hist[((L - 1) * N2 + m) * NT];
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float2 vdp = tt > 0 ? hist[((tt > 0 ? tt - 1 : 0) * N2 + m) * NT] : f2(0.f);
                hist[(tt * N2 + m) * NT] = AR::pair_back(lp, m, vdt, vdp, f2(-dz[tt]), f2(0.f), Ad, acc, kmz);
                vdt = vdp;
            }
        }

        // phase 4: dL/dX of each step as one vector
        if (pos.active) {
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float gxv[KT];
#pragma unroll
                for (int m = 0; m < N2; ++m) {
                    const float2 q = hist[(tt * N2 + m) * NT];
                    gxv[2 * m] = q.x;
                    gxv[2 * m + 1] = q.y;
                }
                V::store(gxrow + (int64_t)tt * sX, 1, gxv);
            }
        }
        xrow += rX;
        gsrow += jstep;
        gxrow += rX;
        if (has_gv) gvrow += jstep;
    }

    constexpr int NA1 = NA + 1;
    float v[NA1];
    float kap[AR::KTb] = {};
    if constexpr (AR::KAPPA_FREE) lane_kappa<AR::KTb>(P, g, pos.chan, 0, kap);
    AR::acc_export(lp, acc, v, kap);
    v[NA] = BETA ? gbeta : 0.f;
#pragma unroll
    for (int a = 0; a < NA1; ++a)
        if (!pos.active || (a < KT && P.stateless)) v[a] = 0.f;
    cp_async_wait<0>();
    pdl_trigger();
    block_partials<KT, 1, 1, NT>(g, pos, v, reinterpret_cast<float *>(sregion), A.partials);
}

// ---------------------------------------------------------------- phased backward, kept V^s
// dendsn_backward_phased_kernel for bfloat16 layers whose forward kept V^s (A.vs_saved).
// The soma needs no recompute, so a row runs in three phases and V^d never goes to shared
// memory:
//   2. the soma's reverse recursion from the kept V^s and dL/dS (both by cp.async, one row
//      ahead) gives dL/dZ[t] (Eqs. methods-lif-reset-charge, methods-lif-fire, methods-sg);
//   3. pair by pair: the pair's inputs of the row from the x ring, the compartment scan
//      forward into registers (Eq. methods-compartment), then the dendritic reverse scan
//      (the per-pair step of dendsn_backward_kernel), dL/dX of the pair to shared memory;
//   4. each step's dL/dX gathered and stored as one vector.
// x arrives two rows ahead (a row's x is read until its phase 3 ends, so the ring holds
// two rows). V^d, the accumulators and dL/dX see the same operations in the same order as
// in dendsn_backward_phased_kernel: both give the same bits. The forward pays 4 bytes per
// neuron-step for V^s (deeper conv forward 209 -> 230 us); the deeper conv backward went
// 516.5 -> 471.8 us with the kept V^s in the phased kernel's four phases, and to 442.9 us
// in these three. Reading x as 8-byte halves (two pairs) instead of each pair's 4-byte
// word (a 4-way bank conflict) measured slower: 442.8 -> 488.3 us (more live registers).
template <int K, int PSI, int L, bool BETA>
__global__ void __launch_bounds__(bwd_threads(K), 3)
dendsn_backward_phased_vs_kernel(const BwdArgs A) {
    pdl_wait();
    using XT = __nv_bfloat16;
    constexpr int KT = K;
    constexpr int NT = bwd_threads(KT);
    constexpr int N2 = KT / 2;
    constexpr int NA = acc_count<KT, 1>();
    using V = XIO<XT, KT, 0>;
    using AR = Arith<KT, 1, PSI, XT>;
    using XRaw = typename V::Raw;
    static_assert(KT == 8 && NT == 128 && sizeof(XRaw) == 16 && AR::KTb == KT,
                  "one lane of 8 bfloat16 compartments per neuron");
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<1>(g);
    typename AR::LP lp;
    AR::load(P, g, pos.chan, 0, lp);
    const int64_t sX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;
    const XT *__restrict__ xrow = static_cast<const XT *>(A.x) + j0 * K;
    const XT *__restrict__ gsrow = static_cast<const XT *>(A.gs) + j0;
    const float *__restrict__ vsrow = A.vs_saved + j0;
    XT *__restrict__ gxrow = static_cast<XT *>(A.gx) + j0 * K;
    const float *gvrow = A.gv ? A.gv + j0 : nullptr;
    const float kv = (P.detach || P.soft) ? 0.f : -P.beta;
    const float cs = (P.detach || !P.soft) ? 0.f : -P.beta * P.theta;
    const float b_spike = P.soft ? P.beta : 0.f;
    const bool has_gv = A.gv != nullptr;
    const int nrows = pos.nrows;

    // dynamic shared memory: the lanes' kappa (per-neuron masks only), then dL/dX as packed
    // bfloat16 pairs [L][N2][NT] (half the shared-memory traffic of float pairs: 442.6 ->
    // 428.8 us), the x ring [2][L][NT], dL/dS words [L][NT] and V^s [L][NT], or (at the end)
    // the reduction
    extern __shared__ float4 smem_f4[];
    char *const sregion = reinterpret_cast<char *>(smem_f4) + kappa_smem_bytes(P.mask_mode, KT, NT);
    uint32_t *const gxw = reinterpret_cast<uint32_t *>(sregion) + threadIdx.x;
    constexpr size_t GXB = sizeof(uint32_t) * L * N2 * NT;
    XRaw *const xring = reinterpret_cast<XRaw *>(sregion + GXB) + threadIdx.x;
    uint32_t *const gring = reinterpret_cast<uint32_t *>(sregion + GXB + sizeof(XRaw) * 2 * L * NT) +
                            threadIdx.x;
    float *const vring = reinterpret_cast<float *>(gring + L * NT);
    // the aligned 4-byte word of dL/dS holding the thread's element (the launcher checks
    // that it lies inside the step's row), and the byte selector that moves the element
    // to the top half (exact)
    auto gs_word = [&](const XT *p) {
        return reinterpret_cast<const uint32_t *>(reinterpret_cast<uintptr_t>(p) & ~(uintptr_t)3);
    };
    auto gs_sel = [&](const XT *p) -> uint32_t {
        return ((reinterpret_cast<uintptr_t>(p) >> 1) & 1) ? 0x3244u : 0x1044u;
    };
    auto fetch_x = [&](int slot, const XT *p, float dep) {
#pragma unroll
        for (int tt = 0; tt < L; ++tt) V::copy_async(xring + (slot * L + tt) * NT, p + (int64_t)tt * sX, 1, dep);
    };
    auto fetch_gv = [&](const XT *gp, const float *vp, float dep) {
#pragma unroll
        for (int tt = 0; tt < L; ++tt) {
            cp_async<4>(gring + tt * NT, gs_word(gp + (int64_t)tt * BN), dep);
            cp_async<4>(vring + tt * NT, vp + (int64_t)tt * BN, dep);
        }
    };
    // commit pattern: rows 0 (x, dL/dS, V^s) and 1 (x); then per row i, after phase 2 the
    // next row's dL/dS and V^s, after phase 3 the x of row i + 2. A row waits for all but the
    // newest group.
    if (nrows > 0) {
        fetch_x(0, xrow, 0.f);
        fetch_gv(gsrow, vsrow, 0.f);
    }
    cp_async_commit();
    if (nrows > 1) fetch_x(1, xrow + rX, 0.f);
    cp_async_commit();

    typename AR::Acc acc;
    AR::acc_zero(acc);
    float gbeta = 0.f;
    MaskAhead<AR, NT> mask;
    mask.init(P, g, j0, jstep, pos.chan, 0, nrows, smem_f4);
    for (int i = 0; i < nrows; ++i) {
        mask.advance(P, g, 0, i + 1 < nrows, lp);
        cp_async_wait<1>();

        // phase 2: dL/dV^s backwards in time from the kept V^s (dL/dZ = dL/dV^s)
        float dz[L];
        {
            const uint32_t sel = gs_sel(gsrow);
            float dvn = 0.f;                     // dL/dV^s[t+1]
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float vs = vring[tt * NT];
                const bool st = vs >= P.theta;
                if constexpr (BETA) {
                    const float leak = st ? (P.soft ? __fsub_rn(vs, P.theta) : 0.f) : vs;
                    gbeta = __fmaf_rn(dvn, leak, gbeta);
                }
                const float dvds = __fmaf_rn(kv, vs, cs);
                const float dvdv = st ? b_spike : P.beta;
                const float gst = __uint_as_float(__byte_perm(gring[tt * NT], 0u, sel));
                const float ds = __fmaf_rn(dvds, dvn, gst);
                float dv = __fmaf_rn(surrogate(__fsub_rn(vs, P.theta)), ds, __fmul_rn(dvdv, dvn));
                if (has_gv) dv = __fadd_rn(dv, __ldcs(gvrow + (int64_t)tt * BN));
                dz[tt] = dv;
                dvn = dv;
            }
        }
        // the next row's dL/dS and V^s, once phase 2 has read them (dz[0] depends on every read)
        if (i + 1 < nrows) fetch_gv(gsrow + jstep, vsrow + jstep, dz[0]);
        cp_async_commit();

        // phase 3: per compartment pair, V^d forward into registers, then the reverse scan
        const XRaw *xs = xring + (i & 1) * L * NT;
#pragma unroll
        for (int m = 0; m < N2; ++m) {
            float2 vd[L];
            float2 v = f2(0.f);
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                const uint32_t w = reinterpret_cast<const uint32_t *>(xs + tt * NT)[m];
                v = ffma2(lp.a[m], v, make_float2(bf16_lo(w), bf16_hi(w)));
                vd[tt] = v;
            }
            const float2 kmz = fmul2(lp.km[m], lp.iz[m]);
            float2 Ad = f2(0.f);
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float2 gq = AR::pair_back(lp, m, vd[tt], tt > 0 ? vd[tt > 0 ? tt - 1 : 0] : f2(0.f),
                                                f2(-dz[tt]), f2(0.f), Ad, acc, kmz);
                gxw[(tt * N2 + m) * NT] = pack_bf16x2(gq.x, gq.y);
            }
        }
        // x of row i + 2 into the slot just read (the sum depends on every pair's reads)
        if (i + 2 < nrows) {
            const float dep = __fadd_rn(__fadd_rn(acc.ga[0].x, acc.ga[1].x), __fadd_rn(acc.ga[2].x, acc.ga[3].x));
            fetch_x(i & 1, xrow + 2 * rX, dep);
        }
        cp_async_commit();

        // phase 4: dL/dX of each step as one vector
        if (pos.active) {
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                __stcs(reinterpret_cast<uint4 *>(gxrow + (int64_t)tt * sX),
                       make_uint4(gxw[(tt * N2 + 0) * NT], gxw[(tt * N2 + 1) * NT],
                                  gxw[(tt * N2 + 2) * NT], gxw[(tt * N2 + 3) * NT]));
            }
        }
        xrow += rX;
        gsrow += jstep;
        vsrow += jstep;
        gxrow += rX;
        if (has_gv) gvrow += jstep;
    }

    constexpr int NA1 = NA + 1;
    float v[NA1];
    float kap[AR::KTb] = {};
    if constexpr (AR::KAPPA_FREE) lane_kappa<AR::KTb>(P, g, pos.chan, 0, kap);
    AR::acc_export(lp, acc, v, kap);
    v[NA] = BETA ? gbeta : 0.f;
#pragma unroll
    for (int a = 0; a < NA1; ++a)
        if (!pos.active || (a < KT && P.stateless)) v[a] = 0.f;
    cp_async_wait<0>();
    pdl_trigger();
    block_partials<KT, 1, 1, NT>(g, pos, v, reinterpret_cast<float *>(sregion), A.partials);
}

// ---------------------------------------------------------------- row-pair backward
// The backward for 4-step rows (T == 4) of 8-compartment float32 neurons served by two
// lanes of four compartments (the transformer-token layer; no residual term). Each thread
// takes its half-neuron of two of its rows at once: a paired instruction carries the same
// compartment of the two neurons (both in the same column, so with the same parameters),
// and the soma recursions and the per-row bookkeeping are shared by the two rows. A row
// pair runs in the phases of dendsn_backward_phased_kernel:
//   1. recompute (Z of each row in the paired engine's tree order and the same lane
//      butterfly, so Z and the spikes are bit-identical to the forward's), V^d of every
//      step and compartment to shared memory; then x of the next row pair is requested;
//   2. the two somas forward, then their reverse recursions, in paired registers; then the
//      next pair's dL/dS (and per-neuron mask bytes) are requested;
//   3. the dendritic reverse scan one compartment at a time, dL/dX overwriting V^d[t];
//   4. each step's dL/dX of each row gathered and stored as one vector.
// x, dL/dS and the mask bytes of a row pair arrive by cp.async one pair ahead. A thread
// with an odd number of rows pairs its last row with a copy of itself whose dL/dS and
// dL/dV^s are zero (its contributions are exactly zero) and whose dL/dX is not stored.
template <int PSI, int LAYOUT, bool BETA>
__global__ void __launch_bounds__(256, 2)
dendsn_backward_rowpair_kernel(const BwdArgs A) {
    pdl_wait();
    constexpr int K = 8, KT = 4, LPN = 2, L = 4, NT = 256;
    constexpr int NA = acc_count<KT, 1>();
    using V = XIO<float, KT, LAYOUT>;
    using XRaw = typename V::Raw;
    static_assert(bwd_threads(KT) == NT, "the plan tiles this backward with bwd_threads(4)");
    const Geometry &g = A.g;
    const Params &P = A.p;
    const ThreadPos pos = thread_pos<LPN>(g);
    // the lane's compartments: alpha, -xi/zeta, 1/zeta, kappa * m (per channel) and m
    float a[KT], nxi[KT], iz[KT], kmc[KT], mkc[KT];
    load_param_arrays<KT, 1>(P, g, pos.chan, pos.sub, a, nxi, iz, kmc, mkc);
    const int64_t sX = g.BN * K;
    const int64_t BN = g.BN;
    const int64_t j0 = pos.row0 * g.P + pos.p;
    const int64_t jstep = (int64_t)pos.rstride * g.P;
    const int64_t rX = jstep * K;
    const int64_t ks = LAYOUT == 0 ? 1 : g.inner;
    const int64_t xoff = lane_x_offset<LAYOUT>(j0, pos.sub, KT, K, g.inner);
    const float *const x0 = static_cast<const float *>(A.x) + xoff;
    const float *const gs0 = static_cast<const float *>(A.gs) + j0;
    float *const gx0 = static_cast<float *>(A.gx) + xoff;
    const float kv = (P.detach || P.soft) ? 0.f : -P.beta;
    const float cs = (P.detach || !P.soft) ? 0.f : -P.beta * P.theta;
    const float b_spike = P.soft ? P.beta : 0.f;
    const bool has_gv = A.gv != nullptr;
    const int nrows = pos.nrows;
    const int nq = (nrows + 1) / 2;              // row pairs

    // dynamic shared memory: history [L][KT][NT] float2, x [2][L][NT], dL/dS [2][2][L][NT]
    // and mask bytes [2][2][NT] (two row pairs: the current one and the next); or (at the
    // end) the reduction
    extern __shared__ float4 smem_f4[];
    char *const sregion = reinterpret_cast<char *>(smem_f4);
    float2 *const hist = reinterpret_cast<float2 *>(sregion) + threadIdx.x;
    XRaw *const xring = reinterpret_cast<XRaw *>(sregion + sizeof(float2) * L * KT * NT) + threadIdx.x;
    float *const gring = reinterpret_cast<float *>(sregion + sizeof(float2) * L * KT * NT +
                                                   sizeof(XRaw) * 2 * L * NT) + threadIdx.x;
    uint32_t *const mring = reinterpret_cast<uint32_t *>(sregion + sizeof(float2) * L * KT * NT +
                                                         sizeof(XRaw) * 2 * L * NT +
                                                         sizeof(float) * 4 * L * NT) + threadIdx.x;
    // neuron (within a sample) of the first row of the pair being fetched, for the masks
    const int nstep = (int)(jstep % g.N);
    int nf = (int)(j0 % g.N);
    auto fetch_x = [&](int q, float dep) {
        const int k = 2 * q;
        if (k < nrows) {
            const float *p1 = x0 + (int64_t)k * rX;
            const float *p2 = (k + 1 < nrows) ? p1 + rX : p1;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                V::copy_async(xring + tt * NT, p1 + (int64_t)tt * sX, ks, dep);
                V::copy_async(xring + (L + tt) * NT, p2 + (int64_t)tt * sX, ks, dep);
            }
        }
        cp_async_commit();
    };
    // dL/dS and mask bytes of row pair q into buffer q & 1, one row pair ahead of their use
    auto fetch_gs = [&](int q, float dep) {
        const int k = 2 * q;
        float *const gbuf = gring + (q & 1) * 2 * L * NT;
        uint32_t *const mbuf = mring + (q & 1) * 2 * NT;
        if (k < nrows) {
            const bool two = k + 1 < nrows;
            const float *p1 = gs0 + (int64_t)k * jstep;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                cp_async<4>(gbuf + tt * NT, p1 + (int64_t)tt * BN, dep);
                if (two) cp_async<4>(gbuf + (L + tt) * NT, p1 + jstep + (int64_t)tt * BN, dep);
                else gbuf[(L + tt) * NT] = 0.f;
            }
            if (P.mask_mode == 2) {
                int n2 = nf + nstep;
                if (n2 >= g.N) n2 -= g.N;
                cp_async<4>(mbuf, P.mask + (int64_t)nf * g.Kb + pos.sub * KT, dep);
                cp_async<4>(mbuf + NT, P.mask + (int64_t)(two ? n2 : nf) * g.Kb + pos.sub * KT, dep);
                nf = n2 + nstep;
                if (nf >= g.N) nf -= g.N;
            }
        }
        cp_async_commit();
    };
    fetch_x(0, 0.f);
    fetch_gs(0, 0.f);
    float gdep = 0.f;   // a value computed from the last reads of the buffer fetch_gs refills

    float2 ga[KT], ngxi[KT], ngz[KT], ngk[KT];
#pragma unroll
    for (int c = 0; c < KT; ++c) { ga[c] = f2(0.f); ngxi[c] = f2(0.f); ngz[c] = f2(0.f); ngk[c] = f2(0.f); }
    float2 gb = f2(0.f);
    for (int q = 0; q < nq; ++q) {
        const int k = 2 * q;
        const bool two = k + 1 < nrows;
        cp_async_wait<0>();
        const float *const gcur = gring + (q & 1) * 2 * L * NT;
        const uint32_t *const mcur = mring + (q & 1) * 2 * NT;
        // the next pair's dL/dS and mask bytes go to the other buffer, read by the previous
        // pair (gdep depends on those reads)
        fetch_gs(q + 1, gdep);
        // the two rows' kappa * m and mask terms (exponent 0 / -inf, or m for the identity)
        float2 km2[KT], lm2[KT];
        if (P.mask_mode == 2) {
            const uint32_t m1 = mcur[0], m2 = mcur[NT];
#pragma unroll
            for (int c = 0; c < KT; ++c) {
                const bool on1 = ((m1 >> (8 * c)) & 0xffu) != 0u, on2 = ((m2 >> (8 * c)) & 0xffu) != 0u;
                km2[c] = make_float2(on1 ? kmc[c] : 0.f, on2 ? kmc[c] : 0.f);
                lm2[c] = make_float2(PairArith<KT, PSI, true>::mask_term(on1 ? 1.f : 0.f),
                                     PairArith<KT, PSI, true>::mask_term(on2 ? 1.f : 0.f));
            }
        } else {
#pragma unroll
            for (int c = 0; c < KT; ++c) {
                km2[c] = f2(kmc[c]);
                lm2[c] = f2(PairArith<KT, PSI, true>::mask_term(mkc[c]));
            }
        }

        // phase 1: recompute
        float2 z[L];
        {
            float2 vd[KT];
#pragma unroll
            for (int c = 0; c < KT; ++c) vd[c] = f2(0.f);
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float xa[KT], xb[KT];
                V::unpack(xring[tt * NT], xa);
                V::unpack(xring[(L + tt) * NT], xb);
                float2 y[KT];
#pragma unroll
                for (int c = 0; c < KT; ++c) {
                    vd[c] = ffma2(f2(a[c]), vd[c], make_float2(xa[c], xb[c]));
                    const float2 u = ffma2(vd[c], f2(iz[c]), f2(nxi[c]));
                    if constexpr (PSI == PSI_MEXHAT) {
                        const float2 ss = fmul2(u, u);
                        const float2 t = fmul2(f2(kNegHalfLog2e), ss);
                        const float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
                        y[c] = ffma2(neg2(ss), e, e);
                    } else {
                        y[c] = make_float2(fabsf(u.x), fabsf(u.y));
                    }
                    hist[(tt * KT + c) * NT] = vd[c];
                }
                // the paired engine's tree: compartments (0, 2) and (1, 3), then the halves
                float2 p = fmul2(km2[0], y[0]);
                p = ffma2(km2[2], y[2], p);
                float2 r = fmul2(km2[1], y[1]);
                r = ffma2(km2[3], y[3], r);
                float2 gv = fadd2(p, r);
                gv.x = __fadd_rn(gv.x, __shfl_xor_sync(0xffffffffu, gv.x, 1));
                gv.y = __fadd_rn(gv.y, __shfl_xor_sync(0xffffffffu, gv.y, 1));
                z[tt] = gv;
            }
        }
        fetch_x(q + 1, __fadd_rn(z[L - 1].x, z[L - 1].y));

        // phase 2: the somas forward, then dL/dV^s backwards in time (dL/dZ = dL/dV^s); ndz
        // keeps -dL/dZ
        float2 ndz[L];
        {
            float v1 = 0.f, v2 = 0.f;
            bool s1 = false, s2 = false;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                v1 = soma_charge(z[tt].x, v1, s1, P);
                v2 = soma_charge(z[tt].y, v2, s2, P);
                s1 = v1 >= P.theta;
                s2 = v2 >= P.theta;
                z[tt] = make_float2(v1, v2);      // z now holds V^s
            }
            const float pi2 = 9.869604401089358f;
            float2 dvn = f2(0.f);
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float2 vs = z[tt];
                const bool st1 = vs.x >= P.theta, st2 = vs.y >= P.theta;
                if constexpr (BETA) {
                    const float l1 = st1 ? (P.soft ? __fsub_rn(vs.x, P.theta) : 0.f) : vs.x;
                    const float l2 = st2 ? (P.soft ? __fsub_rn(vs.y, P.theta) : 0.f) : vs.y;
                    gb = ffma2(dvn, make_float2(l1, l2), gb);
                }
                const float2 dvds = ffma2(f2(kv), vs, f2(cs));
                const float2 dvdv = make_float2(st1 ? b_spike : P.beta, st2 ? b_spike : P.beta);
                const float2 ds = ffma2(dvds, dvn, make_float2(gcur[tt * NT], gcur[(L + tt) * NT]));
                const float2 xd = make_float2(__fsub_rn(vs.x, P.theta), __fsub_rn(vs.y, P.theta));
                const float2 qd = ffma2(fmul2(f2(pi2), xd), xd, f2(1.f));
                const float2 sg = make_float2(fast_rcp(qd.x), fast_rcp(qd.y));
                float2 dv = ffma2(sg, ds, fmul2(dvdv, dvn));
                if (has_gv) {
                    const float *gp = A.gv + j0 + (int64_t)k * jstep + (int64_t)tt * BN;
                    dv = make_float2(__fadd_rn(dv.x, __ldcs(gp)), __fadd_rn(dv.y, two ? __ldcs(gp + jstep) : 0.f));
                }
                ndz[tt] = neg2(dv);
                dvn = dv;
            }
        }
        gdep = __fadd_rn(ndz[0].x, ndz[0].y);

        // phase 3: the dendritic reverse scan, one compartment at a time. As in the paired
        // engine's 8-compartment lanes, the adjoint leaves out kappa m (formed with 1/zeta once
        // per compartment and row pair; the sums are scaled by kappa/zeta at the export):
        // token backward 216.3 -> 214.2 us
#pragma unroll
        for (int c = 0; c < KT; ++c) {
            float2 Ad = f2(0.f);
            float2 vdt = hist[((L - 1) * KT + c) * NT];
            const float2 kmz = fmul2(km2[c], f2(iz[c]));           // kappa m / zeta of each row
#pragma unroll
            for (int tt = L - 1; tt >= 0; --tt) {
                const float2 vdp = tt > 0 ? hist[((tt > 0 ? tt - 1 : 0) * KT + c) * NT] : f2(0.f);
                const float2 u = ffma2(vdt, f2(iz[c]), f2(nxi[c]));
                const float2 ngy = fmul2(lm2[c], ndz[tt]);          // -m dL/dZ (identity)
                float2 y, du;
                if constexpr (PSI == PSI_MEXHAT) {
                    const float2 ss = fmul2(u, u);
                    const float2 t = ffma2(f2(kNegHalfLog2e), ss, lm2[c]);
                    const float2 e = make_float2(fast_exp2(t.x), fast_exp2(t.y));
                    y = ffma2(neg2(ss), e, e);
                    const float2 nw = ffma2(f2(2.f), e, y);        // -psi'(r) / r
                    du = fmul2(fmul2(nw, u), ndz[tt]);
                } else {
                    y = fmul2(lm2[c], make_float2(fabsf(u.x), fabsf(u.y)));
                    du = make_float2(u.x > 0.f ? -ngy.x : (u.x < 0.f ? ngy.x : 0.f),
                                     u.y > 0.f ? -ngy.y : (u.y < 0.f ? ngy.y : 0.f));
                }
                ngxi[c] = fadd2(ngxi[c], du);
                ngz[c] = ffma2(u, du, ngz[c]);
                ngk[c] = ffma2(y, ndz[tt], ngk[c]);
                Ad = ffma2(f2(a[c]), Ad, du);
                ga[c] = ffma2(Ad, vdp, ga[c]);
                hist[(tt * KT + c) * NT] = fmul2(Ad, kmz);
                vdt = vdp;
            }
        }

        // phase 4: dL/dX of each step and row as one vector
        if (pos.active) {
            float *g1 = gx0 + (int64_t)k * rX;
#pragma unroll
            for (int tt = 0; tt < L; ++tt) {
                float ra[KT], rb[KT];
#pragma unroll
                for (int c = 0; c < KT; ++c) {
                    const float2 h = hist[(tt * KT + c) * NT];
                    ra[c] = h.x;
                    rb[c] = h.y;
                }
                V::store(g1 + (int64_t)tt * sX, ks, ra);
                if (two) V::store(g1 + rX + (int64_t)tt * sX, ks, rb);
            }
        }
    }

    // [alpha KT | xi KT | zeta KTb | kappa KTb | beta]; the first three carry 1/zeta here
    constexpr int NA1 = NA + 1;
    float v[NA1];
#pragma unroll
    for (int c = 0; c < KT; ++c) {
        const float kz = __fmul_rn(kmc[c], iz[c]);
        v[c] = __fmul_rn(__fadd_rn(ga[c].x, ga[c].y), kz);
        v[KT + c] = -__fmul_rn(__fadd_rn(ngxi[c].x, ngxi[c].y), kz);
        v[2 * KT + c] = -__fmul_rn(__fadd_rn(ngz[c].x, ngz[c].y), kz);
        v[3 * KT + c] = -__fadd_rn(ngk[c].x, ngk[c].y);
    }
    v[NA] = (BETA && pos.sub == 0) ? __fadd_rn(gb.x, gb.y) : 0.f;
#pragma unroll
    for (int i = 0; i < NA1; ++i)
        if (!pos.active || (i < KT && P.stateless)) v[i] = 0.f;
    cp_async_wait<0>();
    pdl_trigger();
    block_partials<KT, 1, LPN, NT>(g, pos, v, reinterpret_cast<float *>(sregion), A.partials);
}

// ---------------------------------------------------------------- launchers
// Dynamic shared memory above 48 KB needs an explicit opt-in per kernel.
template <typename Kern>
cudaError_t allow_smem(Kern kernel, size_t bytes) {
    if (bytes <= 48 * 1024) return cudaSuccess;
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// Blocks of `kernel` (threads, bytes of dynamic shared memory) that fit on one SM, cached
// per (kernel, threads, bytes) on the current device.
cudaError_t resident_blocks(const void *kernel, int threads, size_t bytes, int *out);

// Launches `kernel` on `blocks` blocks, or with `resident` non-null only reports how many of
// its blocks fit on one SM.
template <typename Kern, typename Args>
cudaError_t launch_or_query(Kern kernel, const Args &a, int blocks, int threads, size_t bytes,
                            cudaStream_t s, int *resident) {
    cudaError_t e = allow_smem(kernel, bytes);
    if (e != cudaSuccess) return e;
    if (resident) return resident_blocks(reinterpret_cast<const void *>(kernel), threads, bytes, resident);
#if DENDSN_PDL
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = bytes;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, a);
#else
    kernel<<<blocks, threads, bytes, s>>>(a);
    return cudaGetLastError();
#endif
}

template <int K, int G, int PSI, int XT, int LAYOUT>
cudaError_t launch_forward(const FwdArgs &a, int blocks, cudaStream_t s, int *resident) {
    using T = typename XType<XT>::type;
    constexpr int KT = lane_compartments(K);
    using XI = XIO<T, KT, LAYOUT>;
    constexpr size_t raw = sizeof(typename XI::Raw);
    constexpr int NT = fwd_threads(K);
    if constexpr (LAYOUT == 1 && K >= 2 && K <= 8 && DENDSN_FWD_ASYNC) {
        // the paper layout with warps of 32 consecutive positions: staged per warp
        if (a.g.inner % 32 == 0 && a.g.TXn % 32 == 0) {
            const size_t smem = (size_t)kFwdDepth * NT * K * sizeof(T) +
                                kappa_smem_bytes(a.p.mask_mode, K / G, NT);
            return launch_or_query(dendsn_forward_staged_kernel<K, G, PSI, T>, a, blocks, NT, smem,
                                   s, resident);
        }
    }
    const size_t smem = ((DENDSN_FWD_ASYNC && XI::kAsync) ? raw * fwd_depth<T, typename XI::Raw>() * NT : 0) +
                        kappa_smem_bytes(a.p.mask_mode, KT / G, NT);
    return launch_or_query(dendsn_forward_kernel<K, G, PSI, T, LAYOUT>, a, blocks, NT, smem, s,
                           resident);
}

template <int K, int G, int PSI, int XT, int L, int LAYOUT>
cudaError_t launch_backward(const BwdArgs &a, int blocks, cudaStream_t s, int *resident) {
    using T = typename XType<XT>::type;
    constexpr int KT = bwd_lane_compartments(K, G, XT, L);
    constexpr int NT = bwd_threads(KT);
    const size_t red = red_bytes(acc_count<KT, G>() + 1, NT);
    constexpr bool shist = (L > 4) || KT >= 8;
    const size_t hist = shist ? sizeof(float) * (KT + 1) * L * NT : 0;
    using XI = XIO<T, KT, LAYOUT>;
    constexpr size_t xraw = sizeof(typename XI::Raw);
    const size_t ring = (DENDSN_BWD_ASYNC && shist && XI::kAsync) ? xraw * kBwdDepth * NT : 0;
    const size_t totals = row_totals<K, G, T, L>() ? sizeof(float) * (acc_count<KT, G>() + 1) * NT : 0;
    constexpr bool bslots = (L == 8 || (K / KT == 1 && G == 1 && LAYOUT == 0)) && DENDSN_BWD_ASYNC &&
                            XI::kAsync && kBwdDepth == L;
    constexpr bool gsa = XT == 0 && bslots;
    const size_t gsb = gsa ? sizeof(float) * L * NT : 0;
    const size_t smem = (red > hist + ring + totals + gsb ? red : hist + ring + totals + gsb) +
                        kappa_smem_bytes(a.p.mask_mode, KT / G, NT);
    auto go_smem = [&](auto kernel, size_t bytes) {
        return launch_or_query(kernel, a, blocks, NT, bytes, s, resident);
    };
    auto go = [&](auto kernel) { return go_smem(kernel, smem); };
    // 4-step rows of 8-compartment float32 neurons on two lanes: two rows per thread
    constexpr bool kRowPair = DENDSN_BWD_ROWPAIR && K == 8 && G == 1 && XT == 0 && L == 4 && KT == 4;
    if constexpr (kRowPair) {
        if (a.g.T == 4 && !a.p.residual) {
            const size_t rp = sizeof(float2) * L * KT * NT + xraw * 2 * L * NT +
                              sizeof(float) * 4 * L * NT + sizeof(uint32_t) * 4 * NT;
            const size_t rsm = red > rp ? red : rp;
            return a.want_beta ? go_smem(dendsn_backward_rowpair_kernel<PSI, LAYOUT, true>, rsm)
                               : go_smem(dendsn_backward_rowpair_kernel<PSI, LAYOUT, false>, rsm);
        }
    }
    // rows of one full chunk, a whole 8-compartment neuron per lane: the phased kernel
    // (deeper conv layer 738 -> 556 us; for the 4-compartment conv layer and for the token
    // layer on one 8-compartment lane it measured slower: 217 -> 280 us, 261 -> 295 us)
    constexpr bool kPhased = DENDSN_BWD_PHASED && LAYOUT == 0 && G == 1 && K == 8 && KT == K &&
                             XI::kAsync;
    if constexpr (kPhased) {
        if (takes_phased_backward(K, G, KT, LAYOUT, a.g.T, L, a.p.residual != 0)) {
            // dL/dS by cp.async needs 4-byte words that stay inside each step's row; the
            // recompute build reserves its shared memory either way, so the residency query
            // (gs unknown) holds for both. (The kept-V^s kernel fits the same 3 blocks per SM.)
            const bool gsa = (reinterpret_cast<uintptr_t>(a.gs) & 3) == 0 && (XT == 0 || a.g.BN % 2 == 0);
            if constexpr (XT == 1) {
                if (gsa && a.vs_saved != nullptr) {
                    const size_t vb = sizeof(uint32_t) * (KT / 2) * L * NT + xraw * 2 * L * NT +
                                      2 * sizeof(uint32_t) * L * NT;
                    const size_t vsm = (red > vb ? red : vb) + kappa_smem_bytes(a.p.mask_mode, KT, NT);
                    return a.want_beta ? go_smem(dendsn_backward_phased_vs_kernel<K, PSI, L, true>, vsm)
                                       : go_smem(dendsn_backward_phased_vs_kernel<K, PSI, L, false>, vsm);
                }
            }
            const size_t ph = sizeof(float) * KT * L * NT + xraw * L * NT + sizeof(uint32_t) * L * NT;
            const size_t psm = (red > ph ? red : ph) + kappa_smem_bytes(a.p.mask_mode, KT, NT);
            if (gsa)
                return a.want_beta ? go_smem(dendsn_backward_phased_kernel<K, PSI, T, L, true, true>, psm)
                                   : go_smem(dendsn_backward_phased_kernel<K, PSI, T, L, false, true>, psm);
            return a.want_beta ? go_smem(dendsn_backward_phased_kernel<K, PSI, T, L, true, false>, psm)
                               : go_smem(dendsn_backward_phased_kernel<K, PSI, T, L, false, false>, psm);
        }
    }
    // full chunks: deeper conv layer 906 -> 738 us, event layer 1829 -> 1755 us, conv layer
    // 219.7 -> 217 us; with 4-step chunks only for whole neurons on one lane, one compartment
    // per branch and compartments innermost: the other 4-step full-chunk builds spill in
    // the loop (token layer 265 -> 314 us, conv layer in the paper layout with two
    // compartments per branch 230 -> 240 us)
    constexpr bool kFull = L == 8 || (K / KT == 1 && G == 1 && LAYOUT == 0);
    if constexpr (kFull) {
        if (a.g.T % L == 0)
            return a.want_beta ? go(dendsn_backward_kernel<K, G, PSI, T, L, LAYOUT, true, true>)
                               : go(dendsn_backward_kernel<K, G, PSI, T, L, LAYOUT, false, true>);
    }
    return a.want_beta ? go(dendsn_backward_kernel<K, G, PSI, T, L, LAYOUT, true, false>)
                       : go(dendsn_backward_kernel<K, G, PSI, T, L, LAYOUT, false, false>);
}

}  // namespace dendsn
