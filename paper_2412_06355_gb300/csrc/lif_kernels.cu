// Fused multi-step LIF layer (forward and BPTT backward): the point-neuron layer the
// paper compares the DendSN layer's speed against (Results, efficiency paragraph).
// The neuron is the DendSN soma (Eq. methods-lif-reset-charge, Eq. methods-lif-fire)
// driven directly by its input current, with the arctan surrogate of Eq. methods-sg.
//
// Same design rules as the DendSN kernels: every step of a neuron runs in one thread
// with the state in registers, the backward recomputes the forward from x (nothing is
// saved for T <= 8; V at the end of every 8-step chunk otherwise), and all tensors are
// streamed once with vector loads. A thread owns VEC consecutive neurons, so a warp
// moves 32 * VEC contiguous elements per step.
#include "dendsn_kernels.cuh"

namespace dendsn {

namespace {

// One LIF charge (hard or soft reset), as soma_charge but with plain arguments.
__device__ __forceinline__ float lif_charge(float x, float v_prev, bool s_prev, float beta,
                                            float theta, int soft) {
    const float leak = soft ? (s_prev ? __fsub_rn(v_prev, theta) : v_prev)
                            : (s_prev ? 0.f : v_prev);
    return __fmaf_rn(beta, leak, x);
}

// CH: steps per chunk (4 when T <= 4, else 8; checkpoints only with 8).
template <typename XT, int VEC, int CH>
__global__ void __launch_bounds__(256) lif_forward_kernel(const LifArgs A) {
    using V = Vec<XT, VEC>;
    const int64_t m0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * VEC;
    if (m0 >= A.M) return;
    const int64_t M = A.M;
    const int T = A.T;
    const XT *xp = static_cast<const XT *>(A.x) + m0;
    XT *sp = static_cast<XT *>(A.spikes) + m0;
    float v[VEC];
    bool s[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e) { v[e] = 0.f; s[e] = false; }
    for (int t0 = 0; t0 < T; t0 += CH) {
        const int n = min(CH, T - t0);
        typename V::Raw xr[CH];
#pragma unroll
        for (int tt = 0; tt < CH; ++tt)
            if (tt < n) xr[tt] = V::load(xp + (int64_t)(t0 + tt) * M);
#pragma unroll
        for (int tt = 0; tt < CH; ++tt) {
            if (tt < n) {
                float xv[VEC], sv[VEC];
                V::unpack(xr[tt], xv);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    v[e] = lif_charge(xv[e], v[e], s[e], A.beta, A.theta, A.soft);
                    s[e] = v[e] >= A.theta;                     // Eq. methods-lif-fire
                    sv[e] = s[e] ? 1.f : 0.f;
                }
                const int64_t off = (int64_t)(t0 + tt) * M;
                V::store(sp + off, sv);
                if (A.v_out) Vec<float, VEC>::store(A.v_out + m0 + off, v);
            }
        }
        if (CH == 8 && A.ck && t0 + CH < T)
            Vec<float, VEC>::store(A.ck + (int64_t)(t0 / CH) * M + m0, v);
    }
}

template <typename XT, int VEC, int CH>
__global__ void __launch_bounds__(256, 2) lif_backward_kernel(const LifArgs A) {
    using V = Vec<XT, VEC>;
    const int64_t m0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * VEC;
    if (m0 >= A.M) return;
    const int64_t M = A.M;
    const int T = A.T;
    const XT *xp = static_cast<const XT *>(A.x) + m0;
    const XT *gsp = static_cast<const XT *>(A.gs) + m0;
    XT *gxp = static_cast<XT *>(A.gx) + m0;
    const float *gvp = A.gv ? A.gv + m0 : nullptr;
    const float nbt = -A.beta * A.theta;                       // dV[t+1]/dS[t], soft reset
    float gn[VEC];                                             // dL/dV[t+1]
#pragma unroll
    for (int e = 0; e < VEC; ++e) gn[e] = 0.f;
    const int nch = (T + CH - 1) / CH;
    for (int c = nch - 1; c >= 0; --c) {
        const int t0 = c * CH;
        const int n = min(CH, T - t0);
        // 4-step chunks fetch grad_spikes together with x, before the recompute; 8-step
        // chunks fetch it step by step in the reverse loop (the whole chunk would spill)
        constexpr bool AHEAD = CH == 4;
        typename V::Raw xr[CH], gr[AHEAD ? CH : 1];
#pragma unroll
        for (int tt = 0; tt < CH; ++tt) {
            if (tt < n) {
                xr[tt] = V::load(xp + (int64_t)(t0 + tt) * M);
                if constexpr (AHEAD) gr[tt] = V::load(gsp + (int64_t)(t0 + tt) * M);
            }
        }
        // recompute the chunk's potentials from its starting state
        float v[VEC];
        bool s[VEC];
        if (c == 0) {
#pragma unroll
            for (int e = 0; e < VEC; ++e) { v[e] = 0.f; s[e] = false; }
        } else {
            Vec<float, VEC>::unpack(Vec<float, VEC>::load(A.ck + (int64_t)(c - 1) * M + m0), v);
#pragma unroll
            for (int e = 0; e < VEC; ++e) s[e] = v[e] >= A.theta;
        }
        float vh[CH][VEC];
#pragma unroll
        for (int tt = 0; tt < CH; ++tt) {
            if (tt < n) {
                float xv[VEC];
                V::unpack(xr[tt], xv);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    v[e] = lif_charge(xv[e], v[e], s[e], A.beta, A.theta, A.soft);
                    s[e] = v[e] >= A.theta;
                    vh[tt][e] = v[e];
                }
            }
        }
        // reverse time through the chunk
#pragma unroll
        for (int tt = CH - 1; tt >= 0; --tt) {
            if (tt < n) {
                const int64_t off = (int64_t)(t0 + tt) * M;
                float gsv[VEC], gv[VEC], gx[VEC];
                if constexpr (AHEAD) V::unpack(gr[tt], gsv);
                else V::unpack(V::load(gsp + off), gsv);
                if (gvp) Vec<float, VEC>::unpack(Vec<float, VEC>::load(gvp + off), gv);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float vt = vh[tt][e];
                    const bool st = vt >= A.theta;
                    const float dvdv = (A.soft || !st) ? A.beta : 0.f;
                    const float dvds = A.detach_reset ? 0.f : (A.soft ? nbt : -A.beta * vt);
                    const float ds = __fmaf_rn(dvds, gn[e], gsv[e]);
                    float dv = __fmaf_rn(surrogate(__fsub_rn(vt, A.theta)), ds,
                                         __fmul_rn(dvdv, gn[e]));
                    if (gvp) dv = __fadd_rn(dv, gv[e]);
                    gx[e] = dv;
                    gn[e] = dv;
                }
                V::store(gxp + off, gx);
            }
        }
    }
}

int lif_blocks(int64_t M, int vec) {
    const int64_t threads = (M + vec - 1) / vec;
    return (int)((threads + 255) / 256);
}

}  // namespace

template <int XT, int VEC>
cudaError_t launch_lif_forward(const LifArgs &a, cudaStream_t s) {
    using T = typename std::conditional<XT == 1, __nv_bfloat16, float>::type;
    const int blocks = lif_blocks(a.M, VEC);
    if (a.T <= 4) lif_forward_kernel<T, VEC, 4><<<blocks, 256, 0, s>>>(a);
    else lif_forward_kernel<T, VEC, 8><<<blocks, 256, 0, s>>>(a);
    return cudaGetLastError();
}

template <int XT, int VEC>
cudaError_t launch_lif_backward(const LifArgs &a, cudaStream_t s) {
    using T = typename std::conditional<XT == 1, __nv_bfloat16, float>::type;
    const int blocks = lif_blocks(a.M, VEC);
    if (a.T <= 4) lif_backward_kernel<T, VEC, 4><<<blocks, 256, 0, s>>>(a);
    else lif_backward_kernel<T, VEC, 8><<<blocks, 256, 0, s>>>(a);
    return cudaGetLastError();
}

template cudaError_t launch_lif_forward<0, 1>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_forward<0, 4>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_forward<1, 1>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_forward<1, 4>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_backward<0, 1>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_backward<0, 4>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_backward<1, 1>(const LifArgs &, cudaStream_t);
template cudaError_t launch_lif_backward<1, 4>(const LifArgs &, cudaStream_t);

}  // namespace dendsn
