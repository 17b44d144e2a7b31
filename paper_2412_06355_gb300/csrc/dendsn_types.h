// Host/device argument blocks and launcher declarations of the DendSN kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dendsn {

enum { PSI_IDENTITY = 0, PSI_MEXHAT = 1 };

constexpr int kFwdBatch = 4;      // time steps per load batch in the forward

// Compartments one lane owns in the forward (a neuron is served by K / that many lanes).
constexpr int lane_compartments(int K) { return K < 8 ? K : 8; }
// In the backward, 8 fp32 compartments per lane with T <= 4 measured slower than two
// lanes of 4 (their registers force the history into shared memory for a very short
// sequence), so that case splits. fp32 layers sum Z in an order that is the same for
// both splits (the paired engine's group tree).
constexpr int bwd_lane_compartments(int K, int G, int xt, int L) {
    return (K >= 8 && G == 1 && xt == 0 && L <= 4) ? 4 : lane_compartments(K);
}
#ifdef __CUDACC__
// Programmatic dependent launch.
// The library's kernels are launched with programmatic stream serialization: a kernel's
// launch overlaps the end of the one before it in the stream, and waits in pdl_wait for
// that one's completion and memory before touching global memory (whole steps 1-2% faster
// on the conv and token layers: the launch gaps between forward, backward and finalize).
#ifndef DENDSN_PDL
#define DENDSN_PDL 1
#endif
// Waits for the grid this one was launched after (and its memory) when launched with
// programmatic stream serialization; a no-op otherwise. Called before any global access.
__device__ __forceinline__ void pdl_wait() {
    if (DENDSN_PDL) asm volatile("griddepcontrol.wait;" ::: "memory");
}
// Lets the next grid in the stream begin launching once every block of this one has called
// it or exited (that grid still waits for this one's completion in pdl_wait).
__device__ __forceinline__ void pdl_trigger() {
    if (DENDSN_PDL) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
#endif

// Whether the backward takes the phased kernel: rows of one full chunk (T == L) of whole
// 8-compartment neurons (one lane each), one compartment per branch, compartments
// innermost, no residual term. The forward of such a layer keeps V^s for it when the
// caller provides the saved buffer.
constexpr bool takes_phased_backward(int K, int G, int KT_bwd, int layout, int T, int L,
                                     bool residual) {
    return K == 8 && G == 1 && KT_bwd == 8 && layout == 0 && T == L && !residual;
}
// Threads per block: the forward always 256; the backward 128 when a lane owns 8
// compartments (its ~165 registers allow three 128-thread blocks per SM).
constexpr int fwd_threads(int K) { return 256; }
constexpr int bwd_threads(int KT) { return KT >= 8 ? 128 : 256; }

// Tiling and sizes shared by every kernel of one call (computed on the host).
// Neuron j = o * P + p: row o in [0, O), column p in [0, P); channel = p / inner.
struct Geometry {
    int64_t O;        // rows
    int64_t BN;       // neurons = O * P
    int32_t P;        // columns = C * inner
    int32_t N, C, inner, T;
    int32_t K, Kb;
    int32_t TXn, TY;  // block tile: TXn columns x TY row lanes (x LPN lanes per neuron)
    int32_t R;        // rows per thread
    int32_t nCT;      // column tiles
    int32_t nRG;      // row groups (blocks along the rows)
    int32_t L;        // backward chunk length == checkpoint interval
    int32_t n_ck;     // checkpoints stored by the forward: ceil(T / L) - 1 when T > L, else 0
    int32_t nch_max;  // most channels one column tile can touch
    int32_t seg;      // columns of one warp that share a channel (power of 2)
};

struct Params {
    const float *alpha, *xi, *zeta, *kappa;
    const uint8_t *mask;
    int32_t mask_mode;   // 0 none, 1 per channel [C,Kb], 2 per neuron [N,Kb]
    float theta, beta;
    int32_t soft, stateless, residual, detach;
};

struct FwdArgs {
    Geometry g;
    Params p;
    const void *x;
    void *spikes;
    float *v_out;
    float *ck_vd;   // [n_ck][BN][K]  or NULL (no checkpoints written)
    float *ck_vs;   // [n_ck][BN]
    float *vs_keep; // [T][BN] V^s for a single-chunk backward (layers with keeps_vs), or NULL
};

struct BwdArgs {
    Geometry g;
    Params p;
    const void *x;
    const void *gs;
    const float *gv;
    const float *ck_vd;
    const float *ck_vs;
    const float *vs_saved;   // [T][BN] V^s the forward kept (vs_keep), or NULL: recomputed
    void *gx;
    float *partials;   // [nCT * nRG][nch_max][NP], NP = 2K + 2Kb + 1 (alpha, xi, zeta, kappa, beta)
    int32_t want_beta; // accumulate the beta slot (else it stays zero)
};

struct FinArgs {
    Geometry g;
    const float *partials;
    float *g_alpha, *g_xi, *g_zeta, *g_kappa;
    float *g_beta;     // [C] or null
    int32_t stateless;
};

// XT: 0 = float, 1 = bfloat16. LAYOUT: 0 = compartments innermost, 1 = the paper's
// (C_o, P, H, W) layer layout. Defined in the instantiation units. With `resident` non-null
// nothing is launched: *resident receives how many blocks of the kernel this call would
// launch fit on one SM (the planner sizes grids in whole waves of that many blocks per SM).
template <int K, int G, int PSI, int XT, int LAYOUT>
cudaError_t launch_forward(const FwdArgs &a, int blocks, cudaStream_t s, int *resident);
template <int K, int G, int PSI, int XT, int L, int LAYOUT>
cudaError_t launch_backward(const BwdArgs &a, int blocks, cudaStream_t s, int *resident);
cudaError_t launch_finalize(const FinArgs &a, cudaStream_t s);

// Time-parallel kernels (tp_kernels.cu): one warp per neuron, for layers with at least
// kTpMinT steps and at most kTpMaxNeurons neurons whose backward history fits in shared
// memory. XT: 0 = float, 1 = bfloat16; psi and layout are runtime arguments.
constexpr int kTpMinT = 256;
constexpr int64_t kTpMaxNeurons = 2048;
constexpr size_t kTpMaxSmem = 200 * 1024;
size_t tp_smem_bytes(int T, int K, bool backward);
template <int K, int G, int XT>
cudaError_t launch_forward_tp(const FwdArgs &a, int psi, int layout, cudaStream_t s);
template <int K, int G, int XT>
cudaError_t launch_backward_tp(const BwdArgs &a, int psi, int layout, cudaStream_t s);
cudaError_t launch_finalize_tp(const FinArgs &a, cudaStream_t s);

// Point-neuron LIF layer: x, spikes, gs, gx are [T, M] in the x dtype; v_out and gv
// [T, M] float32; ck [(T + 7) / 8 - 1, M] float32 somatic potentials at the ends of
// the 8-step chunks (T > 4 only).
struct LifArgs {
    int64_t M;         // neurons
    int32_t T;
    float theta, beta;
    int32_t soft, detach_reset;
    const void *x;
    void *spikes;
    float *v_out;      // or null
    float *ck;         // forward: written when not null; backward: read
    const void *gs;
    const float *gv;   // or null
    void *gx;
};

// XT: 0 = float, 1 = bfloat16; VEC: neurons per thread (4 needs M % 4 == 0 and
// 4-element-aligned tensors, else 1). Defined in lif_kernels.cu.
template <int XT, int VEC> cudaError_t launch_lif_forward(const LifArgs &a, cudaStream_t s);
template <int XT, int VEC> cudaError_t launch_lif_backward(const LifArgs &a, cudaStream_t s);

}  // namespace dendsn

// (K, G) pairs compiled into the library: K compartments per neuron, G per branch.
#define DENDSN_KG_LIST(X) \
    X(1, 1) X(2, 1) X(2, 2) X(4, 1) X(4, 2) X(4, 4) X(8, 1) X(8, 2) X(8, 4) X(16, 1) X(16, 2) X(16, 4)
