/*
 * dendsn.h - C ABI of libdendsn, the fused DendSN layer for NVIDIA GB300 (sm_103a).
 *
 * One DendSN layer (arXiv 2412.06355, Methods "Dendritic spiking neuron") maps the
 * branch input currents X[t, b, n, i] of B samples x N neurons x K compartments
 * over T time steps to somatic spikes S[t, b, n]:
 *
 *   V^d_i[t] = alpha_i V^d_i[t-1] + X_i[t]                 Eq. methods-compartment
 *   Y_j[t]   = psi( || (V^d_{C_j}[t] - xi_{C_j}) / zeta_j ||_2 )
 *                                                           Eq. methods-branch-aggregation
 *   psi(x)   = (1 - x^2) exp(-x^2 / 2)   or   psi(x) = x    Eq. methods-mexican-hat
 *   Z[t]     = sum_j kappa_j m_j Y_j[t]                     Eq. methods-soma-input,
 *                                                           Eq. methods-dbg-mask
 *   V^s[t]   = beta (1 - S[t-1]) V^s[t-1] + Z[t]            Eq. methods-lif-reset-charge
 *   S[t]     = Theta(V^s[t] - theta)                        Eq. methods-lif-fire
 *
 * and its backward is BPTT with the arctan surrogate dS/dV ~ 1/(1 + pi^2 (V - theta)^2)
 * (Eq. methods-sg). Branch j holds the G consecutive compartments j*G .. j*G+G-1
 * (G = P/B in the paper's notation); Kb = K / G branches.
 *
 * Conventions shared by every entry point
 *  - All tensor pointers are DEVICE pointers owned by the caller; the library never
 *    allocates, frees or copies between host and device.
 *  - Every call is asynchronous on the CUDA stream passed as `stream` (a
 *    cudaStream_t; NULL = legacy default stream). Argument errors are detected on
 *    the host before any launch and return a non-zero status with nothing enqueued.
 *    A failed launch returns DENDSN_ERR_CUDA. dendsn_last_error() describes the most
 *    recent failure of the calling thread.
 *  - Layouts are dense row-major:
 *      x, grad_x            [T, B, N, K] (or the PAPER layout, see dendsn_layout),
 *                           dtype x_dtype; base 16-byte aligned
 *      spikes, grad_spikes  [T, B, N]      dtype x_dtype (spikes are exactly 0 or 1)
 *      v_out, grad_v        [T, B, N]      float32
 *      alpha, xi            [C, K]         float32
 *      zeta, kappa          [C, Kb]        float32 (zeta > 0)
 *      mask                 [C, Kb] (mask_per_neuron = 0) or [N, Kb] (= 1), uint8 0/1,
 *                           base 4-byte aligned; NULL = all branches active
 *      grad_alpha, grad_xi  [C, K]         float32, OVERWRITTEN (not accumulated)
 *      grad_zeta, grad_kappa[C, Kb]        float32, OVERWRITTEN
 *    Neuron n of every sample uses parameter channel c(n) = (n / inner) % C, so the
 *    neurons at the spatial positions of a conv channel share parameters (Methods,
 *    "Dendritic spiking neural networks", constraint 3). N must be a multiple of
 *    C * inner. A layer-wide decay alpha (the paper's choice) is passed as a [C, K]
 *    array of equal values; its gradient is the sum of grad_alpha.
 *  - Supported: K in {1, 2, 4, 8, 16}; G in {1, 2, 4} with G dividing K;
 *    T >= 0; B * N < 2^31 * C * inner. Others return DENDSN_ERR_UNSUPPORTED.
 */
#ifndef DENDSN_H
#define DENDSN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DENDSN_OK = 0,
    DENDSN_ERR_INVALID_ARG = 1,   /* NULL pointer, bad size, bad enum value */
    DENDSN_ERR_UNSUPPORTED = 2,   /* valid but not compiled in (K, G, surrogate) */
    DENDSN_ERR_MISALIGNED = 3,    /* a pointer violates its alignment rule */
    DENDSN_ERR_CUDA = 4           /* a CUDA launch failed; see dendsn_last_error() */
} dendsn_status;

typedef enum { DENDSN_F32 = 0, DENDSN_BF16 = 1 } dendsn_dtype;
typedef enum { DENDSN_PSI_IDENTITY = 0, DENDSN_PSI_MEXHAT = 1 } dendsn_psi;
/* HARD: Eq. methods-lif-reset-charge. SOFT: V^s[t] = beta (V^s[t-1] - theta S[t-1]) + Z[t]. */
typedef enum { DENDSN_RESET_HARD = 0, DENDSN_RESET_SOFT = 1 } dendsn_reset;
/* ATAN: Eq. methods-sg, the only surrogate the paper uses. */
typedef enum { DENDSN_SG_ATAN = 0 } dendsn_surrogate;
/*
 * Layout of x and grad_x (spikes and the other [T, B, N] tensors are the same in both):
 *   KINNER: [T, B, N, K], a neuron's K compartments contiguous.
 *   PAPER : [T, B, N / inner, K, inner], i.e. a conv layer's output [T, B, C_o * P, H, W]
 *           read as (C_o, P, H, W) with inner = H * W (Methods, "Dendritic spiking neural
 *           networks"): compartment k of neuron n is (n / inner) * K * inner + k * inner
 *           + n % inner elements into the sample. No transpose is needed.
 */
typedef enum { DENDSN_LAYOUT_KINNER = 0, DENDSN_LAYOUT_PAPER = 1 } dendsn_layout;

typedef struct {
    int32_t T, B, N;        /* time steps, samples, neurons per sample */
    int32_t K, G;           /* compartments per neuron, compartments per branch */
    int32_t C, inner;       /* parameter channels; neurons per channel run */
    int32_t x_dtype;        /* dendsn_dtype of x, spikes, grad_spikes, grad_x */
    int32_t psi;            /* dendsn_psi */
    int32_t reset;          /* dendsn_reset */
    int32_t surrogate;      /* dendsn_surrogate */
    float theta;            /* firing threshold (1 in Eq. methods-lif-fire) */
    float beta;             /* somatic decay, 0 <= beta < 1 */
    int32_t detach_reset;   /* 1: no gradient through the reset term */
    int32_t mask_per_neuron;/* 0: mask is [C, Kb]; 1: mask is [N, Kb] */
    int32_t stateless;      /* 1: Stateless Dendrite, V^d = X (Methods, "Stateless compartment") */
    int32_t residual;       /* 1: Z += mean_i X_i (Eq. methods-residual) */
    int32_t layout;         /* dendsn_layout of x and grad_x */
} dendsn_config;

/*
 * Sizes of the two caller-owned device buffers a forward/backward pair needs.
 *   saved_bytes  : state the forward writes and the backward reads. For T > 8,
 *                  checkpoints of (V^d, V^s) every 8 steps (recompute with
 *                  checkpointing, Results "Constructing deep DendSNNs"). For layers
 *                  whose backward serves each 8-compartment neuron on one thread over
 *                  a single chunk (K = 8, G = 1, compartments innermost, no residual
 *                  term, T = 8, or T = 4 with bfloat16 x), V^s [T, B, N] float32, so
 *                  that the backward rescans only V^d; optional there (NULL in both
 *                  calls: the backward recomputes V^s from x, with the same bits).
 *                  Otherwise 0. 16-byte aligned. Must outlive the backward.
 *   scratch_bytes: per-block partial sums of the parameter gradients, used only by
 *                  dendsn_backward. 16-byte aligned. Contents need no initialisation.
 * Either output pointer may be NULL.
 */
dendsn_status dendsn_workspace_size(const dendsn_config *cfg, size_t *saved_bytes,
                                    size_t *scratch_bytes);

/*
 * Fused multi-step forward: compartment scan, L2 branch aggregation, psi, masked
 * kappa reduction and LIF soma, all T steps in one kernel with the state in
 * registers.
 *   x        [T,B,N,K] input currents (read)
 *   alpha..kappa, mask: parameters as above (read)
 *   spikes   [T,B,N] output (written)
 *   v_out    [T,B,N] float32 somatic potential V^s (written), or NULL
 *   saved    buffer of saved_bytes (written), or NULL when no backward will follow;
 *            ignored when saved_bytes == 0
 */
dendsn_status dendsn_forward(const dendsn_config *cfg, const void *x, const float *alpha,
                             const float *xi, const float *zeta, const float *kappa,
                             const uint8_t *mask, void *spikes, float *v_out, void *saved,
                             void *stream);

/*
 * Fused reverse-time backward (BPTT with the arctan surrogate, Eq. methods-sg). The
 * forward of each checkpoint interval is recomputed from x in registers.
 *   grad_spikes [T,B,N] dL/dS (read); grad_v [T,B,N] float32 dL/dV^s (read) or NULL
 *   saved       the buffer the forward of the same inputs filled (read); may be NULL
 *               when T <= 8 if it was NULL in the forward too (a buffer the forward did
 *               not fill gives wrong gradients, it is not detected)
 *   grad_x      [T,B,N,K] dL/dX (written)
 *   grad_alpha, grad_xi, grad_zeta, grad_kappa: parameter gradients summed over time,
 *               samples and the neurons of each channel (written, deterministic order).
 *               grad_alpha is all zero for a Stateless Dendrite. grad_kappa is the
 *               gradient w.r.t. the unmasked strength (zero where the mask is 0).
 *   scratch     scratch_bytes of device memory (contents are overwritten)
 */
dendsn_status dendsn_backward(const dendsn_config *cfg, const void *x, const float *alpha,
                              const float *xi, const float *zeta, const float *kappa,
                              const uint8_t *mask, const void *grad_spikes,
                              const float *grad_v, const void *saved, void *grad_x,
                              float *grad_alpha, float *grad_xi, float *grad_zeta,
                              float *grad_kappa, void *scratch, void *stream);

/*
 * dendsn_backward for a soma whose decay beta is learnable (the PLIF soma the paper cites
 * alongside LIF, read as Eq. methods-lif-reset-charge with beta a parameter). Same
 * arguments and outputs as dendsn_backward, plus
 *   grad_beta  [C] float32, OVERWRITTEN: dL/dbeta summed over time, samples and the
 *              neurons of each channel, where dV^s[t+1]/dbeta = (1 - S[t]) V^s[t] (hard
 *              reset) or V^s[t] - theta S[t] (soft). The gradient of the layer's single
 *              beta is the sum of the C entries (parameterisations such as
 *              beta = sigmoid(w) are applied by the caller).
 * Runs a separate build of the backward kernel that also accumulates dL/dbeta (one more
 * fused multiply-add per step); dendsn_backward does not pay for it.
 */
dendsn_status dendsn_backward_plif(const dendsn_config *cfg, const void *x, const float *alpha,
                                   const float *xi, const float *zeta, const float *kappa,
                                   const uint8_t *mask, const void *grad_spikes,
                                   const float *grad_v, const void *saved, void *grad_x,
                                   float *grad_alpha, float *grad_xi, float *grad_zeta,
                                   float *grad_kappa, float *grad_beta, void *scratch,
                                   void *stream);

/*
 * Same computation and outputs as dendsn_backward, without the caller's scratch buffer:
 * for callers that cannot allocate device memory for it, such as a C host that only
 * receives device pointers for the layer's tensors, or a runtime whose device memory is
 * budgeted in advance and that must not allocate per call. (The paper has no
 * counterpart; this is an interface convenience.)
 *   - The parameter-gradient partials go to a buffer compiled into the library:
 *     8 MiB of device memory on every GPU that loads the library, held until the
 *     process exits. A layer whose dendsn_workspace_size scratch_bytes exceeds 8 MiB
 *     is rejected with DENDSN_ERR_UNSUPPORTED before anything is enqueued.
 *   - The first call on a device looks up that buffer's device address (with that
 *     device current) and caches it; make that first call before any stream capture.
 *     The cached address belongs to the device's context at that time: after a
 *     cudaDeviceReset on that device (which unloads the library's device code) it is
 *     stale, so a process that resets a device must not call this entry point on it
 *     again.
 *   - All calls share the one buffer, which keeps the last call's contents. Nothing in
 *     it needs to start at zero. Calls whose executions overlap on the GPU (for example
 *     on two streams without ordering between them) race on it and give wrong results.
 *   - Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 * Arguments are those of dendsn_backward minus `scratch`.
 */
dendsn_status dendsn_backward_noalloc(const dendsn_config *cfg, const void *x,
                                      const float *alpha, const float *xi, const float *zeta,
                                      const float *kappa, const uint8_t *mask,
                                      const void *grad_spikes, const float *grad_v,
                                      const void *saved, void *grad_x, float *grad_alpha,
                                      float *grad_xi, float *grad_zeta, float *grad_kappa,
                                      void *stream);

/*
 * Point-neuron LIF layer: the baseline neuron the paper compares the DendSN layer's speed
 * with (Results, efficiency paragraph). It is the DendSN soma driven directly by one input
 * current per neuron (Eq. methods-lif-reset-charge with X[t] in place of Z[t],
 * Eq. methods-lif-fire; soft reset as above), trained with the same arctan surrogate
 * (Eq. methods-sg). Same conventions as the DendSN entry points (device pointers, async
 * on `stream`, host-side validation, dendsn_last_error()).
 *   x, grad_x, spikes, grad_spikes   [T, B, N]  dtype x_dtype, naturally aligned
 *   v_out, grad_v                    [T, B, N]  float32, 4-byte aligned; may be NULL
 *   saved   checkpoints (V at the end of every 8 steps), saved_bytes of 16-byte aligned
 *           device memory; needed (non-NULL) only when saved_bytes > 0, i.e. T > 8
 * Tensors whose neuron count B*N is a multiple of 4 and whose pointers are aligned to 4
 * elements (16 bytes for the float32 ones) take the vectorised kernels.
 */
typedef struct {
    int32_t T, B, N;        /* time steps, samples, neurons per sample */
    int32_t x_dtype;        /* dendsn_dtype of x, spikes, grad_spikes, grad_x */
    int32_t reset;          /* dendsn_reset */
    float theta, beta;      /* threshold, somatic decay (0 <= beta < 1) */
    int32_t detach_reset;   /* 1: no gradient through the reset term */
} dendsn_lif_config;

dendsn_status dendsn_lif_workspace_size(const dendsn_lif_config *cfg, size_t *saved_bytes);

/* Fused T-step LIF forward: writes spikes (and V if v_out), and the checkpoints to saved. */
dendsn_status dendsn_lif_forward(const dendsn_lif_config *cfg, const void *x, void *spikes,
                                 float *v_out, void *saved, void *stream);

/* Fused reverse-time LIF backward: dL/dX from dL/dS (and dL/dV if grad_v), recomputing V. */
dendsn_status dendsn_lif_backward(const dendsn_lif_config *cfg, const void *x,
                                  const void *grad_spikes, const float *grad_v,
                                  const void *saved, void *grad_x, void *stream);

/* Static description of a status code. */
const char *dendsn_status_string(dendsn_status status);

/* Message describing the calling thread's most recent failed call ("" if none). */
const char *dendsn_last_error(void);

/* Number of kernels the library enqueued since load (all threads). */
uint64_t dendsn_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* DENDSN_H */
