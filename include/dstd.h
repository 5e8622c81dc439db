/*
 * dstd.h -- C-ABI of libdstd: differentiable spike-time discretization (DSTD)
 * for time-to-first-spike LIF layers on one GB300 (sm_103a).
 *
 * Method (arxiv 2607.14672): a LIF neuron (Eq. LIF_model_TTFS)
 *     dv/dt = -v/tau_m + I,   dI/dt = -I/tau_s + sum_j w_ij delta(t - t_j)
 * fires once, when v first reaches v_th. DSTD (App. B, Alg. 2) replaces each
 * input spike t_j by weights s_jm on two neighbouring points of a fixed grid
 *     T_m = t_first + m dt - t_offset,  m = 0..M,  dt = (t_end - t_first)/M,
 * with s_jm = K_DSTD(t_j - T_m) (Eq. DSTD_kernel, Tab. DSTD_kernels), forms
 * w^_im = sum_j w_ij s_jm (Eq. DSTD), and takes as spike time the first root
 * of the discretised potential over the M intervals [T_q, T_{q+1})
 * (Tab. timing_DSTD, Eq. timing_DSTD). The backward pass is the analytic
 * gradient of that spike time (implicit function theorem).
 *
 * Conventions shared by every entry point
 *  - All array pointers are DEVICE memory owned by the caller, row-major,
 *    float32 unless stated, and must be 16-byte aligned. The library never
 *    allocates device memory; scratch comes from a caller workspace whose
 *    size the *_workspace_bytes queries return.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *    default stream). No call synchronises the device except
 *    dstd_device_status().
 *  - Silent neurons carry IEEE +INFINITY, in inputs and outputs.
 *  - Return 0 on success or a negative DSTD_E_* code; arguments are checked
 *    before anything is launched, so an error return launched nothing
 *    (DSTD_E_CUDA excepted: a launch was attempted and failed).
 *  - Device-side waits (TMA / tensor-core pipelines) are bounded; a wait
 *    that expires sets a device status word that dstd_device_status()
 *    returns as DSTD_E_TIMEOUT. No kernel traps.
 *  - Readings where the paper is silent (stated once here, used everywhere):
 *    candidates exist for q = 0..M-1 only and a neuron without a crossing by
 *    T_M is silent; a spike before T_{-1} = T_0 - dt gets no grid weight;
 *    a spike exactly on T_m uses the t >= 0 column of Tab. DSTD_kernels.
 */
#ifndef DSTD_H
#define DSTD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *dstd_stream_t; /* same type as cudaStream_t */

enum {
    DSTD_OK = 0,
    DSTD_E_INVALID = -1,     /* null pointer, non-positive size, bad constant */
    DSTD_E_UNSUPPORTED = -2, /* valid request outside what this build supports */
    DSTD_E_WORKSPACE = -3,   /* workspace smaller than the query returned */
    DSTD_E_CUDA = -4,        /* a CUDA runtime call or launch failed */
    DSTD_E_TIMEOUT = -5,     /* a bounded device-side wait expired */
    DSTD_E_NO_DEVICE = -6    /* no usable sm_103 device */
};

/* Arithmetic of the contractions (w^ = W s and its two transposes).
 *  F32   CUDA-core fp32 FMA GEMMs (reference precision).
 *  X3    tcgen05 tensor cores, each fp32 operand split into a 16-bit hi + lo
 *        pair and three products (hi*hi + hi*lo + lo*hi) accumulated in fp32
 *        TMEM, for fp32 workloads. Forward: fp16 pairs, W scaled per row by a
 *        power of two into fp16 range (~2^-21 relative operand error; spike
 *        times need it). Backward: bf16 pairs (~2^-17; gradients need 1e-3).
 *  BF16  tcgen05 tensor cores, bf16 operands, fp32 accumulation.
 * Scan, solve, binning and every epilogue run in fp32 in all modes. */
typedef enum { DSTD_MATH_F32 = 0, DSTD_MATH_X3 = 1, DSTD_MATH_BF16 = 2 } dstd_math;

/* One layer's constants (App. B.1 grid, App. C.1 synfire penalty).
 *  tau_m, tau_s    tau_v and tau_I of Eq. LIF_model_TTFS; > 0 or INFINITY.
 *  v_th            threshold, > 0.
 *  t_first, t_end  DSTD window (App. C.1), t_end > t_first; M >= 1 steps.
 *  t_offset        grid shift, in (-dt/2, dt/2] (Alg. 2 draws it per layer).
 *  t_head, t_tail  penalty edges t_head^(l), t_tail^(l) (Eq. temporal_penalty).
 *  gamma_head, gamma_tail, gamma_q   penalty weights (0 disables a term).
 *  penalty_norm    factor applied to T and gamma_Q Q and to their gradients:
 *                  1/B for dense layers (mini-batch mean, Eq. cost_function),
 *                  1/(B H W) for conv layers (App. C.1). */
typedef struct {
    float tau_m, tau_s;
    float v_th;
    float t_first, t_end;
    int32_t M;
    float t_offset;
    float t_head, t_tail;
    float gamma_head, gamma_tail, gamma_q;
    float penalty_norm;
} dstd_params;

/* Per-neuron state that dstd_dense_fwd saves for dstd_dense_bwd:
 * q (int32, interval index of the spike, M if silent), s (spike time minus
 * T_q), vdot (dv^/dt at the spike, floored at 1e-6 v_th/dt), each [B, N_out].
 * Opaque to the caller apart from its size. */
size_t dstd_dense_saved_bytes(int B, int N_out);

/* Workspace bytes needed by dstd_dense_fwd and dstd_dense_bwd (the max of the
 * two) for these sizes and math mode; 0 on invalid arguments. */
size_t dstd_dense_workspace_bytes(int B, int N_in, int N_out, const dstd_params *p, dstd_math math);

/* Binning alone (Eq. DSTD_kernel, Tab. DSTD_kernels): spike times -> grid
 * weights.
 *  t_in  [B, N]      input spike times (+inf = silent).
 *  s     [B, M, N]   out: s_jm for m = 0..M-1 (zero outside the support).
 *  ds    [B, M, N]   out (may be NULL): d s_jm / d t_j (one-sided at knots). */
int dstd_binning(const float *t_in, int B, int N, const dstd_params *p, float *s, float *ds,
                 dstd_stream_t stream);

/* Binning + contraction alone: w^_im = sum_j w_ij s_jm (Eq. DSTD).
 *  t_in [B, N_in], W [N_out, N_in]  ->  what [B, N_out, M]. */
int dstd_dense_what(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                    dstd_math math, float *what, void *workspace, size_t ws_bytes, dstd_stream_t stream);

/* Scan + threshold solve + first-spike select alone, from given w^
 * (Tab. timing_DSTD, Eq. timing_DSTD), plus the penalty terms.
 *  what    [B, N_out, M]  discretised inputs w^_im.
 *  t_out   [B, N_out]     out: spike times (+inf = silent).
 *  saved   dstd_dense_saved_bytes(B, N_out) bytes, out (may be NULL).
 *  penalty float[4] out (may be NULL): {norm * T, gamma_q * norm * Q,
 *          number of silent neurons, number of firing neurons}. Q needs
 *          the weight row sums: w_rowsum [N_out] (may be NULL = Q term 0). */
int dstd_scan_solve(const float *what, int B, int N_out, const dstd_params *p, const float *w_rowsum,
                    float *t_out, void *saved, float *penalty, dstd_stream_t stream);

/* Forward of one dense DSTD layer (Alg. 2 body): binning, contraction,
 * scan/solve/select, silent mask and penalty terms.
 *  t_in [B, N_in], W [N_out, N_in] (fp32; converted per call for tensor cores).
 *  t_out [B, N_out], saved, penalty[4] as in dstd_scan_solve. */
int dstd_dense_fwd(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                   dstd_math math, float *t_out, void *saved, float *penalty, void *workspace,
                   size_t ws_bytes, dstd_stream_t stream);

/* The layer forward of dstd_dense_fwd for callers that cannot allocate
 * device memory: code that runs where cudaMalloc is unavailable or
 * forbidden (inside a host callback, a real-time loop that may not touch the
 * allocator, a plugin whose host application owns every allocation) and has
 * no workspace to pass. It computes exactly what dstd_dense_fwd computes,
 * with the same arguments minus the workspace; the caller still provides
 * t_in, W, t_out, saved and penalty. (The paper has no counterpart: this is
 * a deployment convenience of this library.)
 * Scratch: a fixed 64 MiB array in device memory, part of the library's
 * image. With CUDA's lazy module loading it is taken on a device when the
 * library's module is first loaded there (the first launch of any of its
 * kernels, or this function's address lookup), by every process that uses
 * the library on that device whether or not it calls this function, and it
 * stays until the process exits. A call whose scratch need (dstd_dense_workspace_bytes' forward part)
 * exceeds 64 MiB returns DSTD_E_WORKSPACE and launches nothing; the 784-800
 * and 800-800 layers at B = 256, M = 32 fit. No call allocates or frees.
 * Every call uses the same array, which keeps whatever the previous call
 * left there (each call overwrites all the scratch it reads), so two calls
 * that can overlap on the GPU (different streams, or different host threads)
 * race; serialise them. The first call on each device looks up the array's
 * device address (cudaGetSymbolAddress) with that device current; make that
 * first call before starting any stream capture. The address is kept per
 * device for the life of the process: it belongs to the device's primary
 * context, so calls must come from that context (the runtime API's default),
 * and not after a cudaDeviceReset. */
int dstd_dense_fwd_noalloc(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                           dstd_math math, float *t_out, void *saved, float *penalty, dstd_stream_t stream);

/* Backward of one dense DSTD layer.
 *  g_t_out [B, N_out] dC/dt_out from above (the loss or the next layer); the
 *          layer adds its own temporal-penalty gradient (params) itself.
 *  g_t_in  [B, N_in]  out (may be NULL): dC/dt_in; 0 for silent inputs.
 *  g_W     [N_out, N_in] out (overwritten): dC/dW including the dead-neuron
 *          term -gamma_q * norm * (number of samples where neuron i is silent).
 * dt_i/dw^_im = -K(t_i - T_m)/v^'(t_i) for m <= q_i (IFT on v^(t_i) = v_th). */
int dstd_dense_bwd(const float *t_in, const float *W, const float *t_out, const void *saved,
                   const float *g_t_out, int B, int N_in, int N_out, const dstd_params *p, dstd_math math,
                   float *g_t_in, float *g_W, void *workspace, size_t ws_bytes, dstd_stream_t stream);

/* Convolutional DSTD layer (3x3 / k x k filters, stride, zero-spike padding),
 * the implicit-GEMM form of the same contraction: output position
 * (b, y, x) plays the role of a sample and filter tap (kh, kw, c) of an input.
 *  t_in   [B, H, W, C_in]     input spike times, NHWC (+inf = silent).
 *  W      [C_out, k, k, C_in] weights (tap-major rows).
 *  t_out  [B, Ho, Wo, C_out]  NHWC, Ho = (H + 2 pad - k)/stride + 1 (same Wo).
 *  saved  dstd_dense_saved_bytes(B*Ho*Wo, C_out) bytes.
 *  penalty as in dstd_dense_fwd; set p->penalty_norm = 1/(B*Ho*Wo) (App. C.1:
 *          T and Q of conv layers are divided by the spatial size).
 * Tensor-core math modes only (DSTD_MATH_F32 returns DSTD_E_UNSUPPORTED).
 * Padding taps read silent inputs.
 * In DSTD_MATH_BF16 with C_in below 64 (padded to 64 with silent inputs) or a
 * multiple of 64, C_out a multiple of 64 (at most 128 or a multiple of 128),
 * k <= 7 and M <= 64,
 * the layer runs as implicit GEMMs: each input spike becomes one 8-byte
 * record (its grid step and its two nonzero grid weights in bf16, the
 * compact support of Eq. DSTD_kernel); from those records the binned input
 * is either written out once per chunk ([images, H, W, Mp, C_in], no im2col
 * expansion) and read by the forward and dW through TMA boxes shifted per
 * filter tap, or generated tile by tap in shared memory
 * (dstd_conv_set_operand_policy); dS is the transposed
 * convolution of dw^ (TMA boxes shifted per tap, only the taps on the
 * stride grid) with the input-time gradient taken in its epilogue. Chunks
 * of whole images keep that scratch (w^ in fp32, dw^ and S in bf16) near 4 GiB
 * (dstd_conv_set_chunk_images). Other shapes and the three-product mode
 * gather the binned input per tap (im2col) in chunks of whole images near
 * 1 GiB. The workspace query accounts for either. */
size_t dstd_conv_workspace_bytes(int B, int H, int W, int C_in, int C_out, int k, int stride, int pad,
                                 const dstd_params *p, dstd_math math);
int dstd_conv_fwd(const float *t_in, const float *W, int B, int H, int Wd, int C_in, int C_out, int k, int stride,
                  int pad, const dstd_params *p, dstd_math math, float *t_out, void *saved, float *penalty,
                  void *workspace, size_t ws_bytes, dstd_stream_t stream);
/* Backward of the conv layer: g_t_out [B, Ho, Wo, C_out]; g_t_in [B, H, W, C_in]
 * (may be NULL; overwritten); g_W [C_out, k, k, C_in] (overwritten, with the
 * dead-neuron term -gamma_q * norm * silent count of the output channel). */
int dstd_conv_bwd(const float *t_in, const float *W, const float *t_out, const void *saved, const float *g_t_out,
                  int B, int H, int Wd, int C_in, int C_out, int k, int stride, int pad, const dstd_params *p,
                  dstd_math math, float *g_t_in, float *g_W, void *workspace, size_t ws_bytes,
                  dstd_stream_t stream);

/* The output layer's forward followed by the cross-entropy of its spike
 * times: the results of dstd_dense_fwd and then dstd_ce_loss(t_out, labels,
 * B, N_out, tau_soft, t_silent, loss, g_t_out). A layer on the few-output
 * path (at most 32 outputs, fp32 or three-product mode) computes the loss in
 * the same kernel, one block per sample, and the batch mean in sample order.
 *  loss: float[2], 8-byte aligned: loss[0] out; loss[1] is the kernel's
 *        scratch, zero before the first call (each call leaves it zero);
 *  labels [B] int32 in [0, N_out); g_t_out [B, N_out] out;
 *  the workspace also holds B floats of per-sample terms.
 * Errors as dstd_dense_fwd and dstd_ce_loss. */
int dstd_dense_fwd_ce(const float *t_in, const float *W, int B, int N_in, int N_out,
                      const dstd_params *p, dstd_math math, float *t_out, void *saved,
                      float *penalty, void *workspace, size_t ws_bytes, const int32_t *labels,
                      float tau_soft, float t_silent, float *loss, float *g_t_out,
                      dstd_stream_t stream);

/* Multi-spike layers (App. D, Eq. Vmem_multiSpikes): a neuron may fire up to
 * F_out times in the window; at each spike its membrane potential is reset to
 * 0 and its synaptic current kept. Each input spike is discretised on its
 * own and the grid weights of an input's spikes are summed, so w^ = W s is
 * the same contraction; the spikes of a neuron are found one after another
 * (after spike k the rest of its interval is tested again from v = 0).
 *  t_in  [B, N_in, F_in]   spike times of each input, +inf = none (any order);
 *  t_out [B, N_out, F_out] out: ascending, +inf after a neuron's last spike;
 *  saved dstd_ms_saved_bytes(B, N_out, F_out) bytes (bin, current and dv^/dt
 *        at every spike), written by the forward and read by the backward;
 *  g_t_out [B, N_out, F_out] dC/dt_out (entries after the last spike ignored);
 *  g_t_in  [B, N_in, F_in] out (may be NULL): dC/dt of every input spike, 0
 *        for +inf entries; g_W [N_out, N_in] out (overwritten).
 * Backward: the implicit function theorem per spike; spike k depends on w^
 * both directly and through the spike k - 1 it was reset at, and the
 * adjoints run from the last spike back to the first.
 * 1 <= F_in, F_out <= 8 (DSTD_E_UNSUPPORTED above); tensor-core modes only
 * (DSTD_MATH_F32 gives DSTD_E_UNSUPPORTED). The temporal and dead-neuron
 * penalties are not defined for this regime: the params' penalty fields are
 * not used. Other errors as dstd_dense_fwd / dstd_dense_bwd. */
size_t dstd_ms_saved_bytes(int B, int N_out, int F_out);
size_t dstd_ms_workspace_bytes(int B, int N_in, int N_out, int F_in, int F_out, const dstd_params *p,
                               dstd_math math);
int dstd_dense_fwd_ms(const float *t_in, const float *W, int B, int N_in, int N_out, int F_in, int F_out,
                      const dstd_params *p, dstd_math math, float *t_out, void *saved, void *workspace,
                      size_t ws_bytes, dstd_stream_t stream);
int dstd_dense_bwd_ms(const float *t_in, const float *W, const float *t_out, const void *saved,
                      const float *g_t_out, int B, int N_in, int N_out, int F_in, int F_out, const dstd_params *p,
                      dstd_math math, float *g_t_in, float *g_W, void *workspace, size_t ws_bytes,
                      dstd_stream_t stream);

/* Skip-and-delay input of the paper's 20-layer network (App. C.3, Fig.
 * skip_connection: the third layer of a block also receives the block's input,
 * delayed by 2 tau_shift). Spike tensors are NHWC, so this is a concatenation
 * along channels at each of `positions` = B*H*W positions:
 *   out[p, 0:C_a]       = a[p, :] + delay_a   (+inf stays +inf)
 *   out[p, C_a:C_a+C_b] = b[p, :]
 *  a [positions, C_a], b [positions, C_b], out [positions, C_a + C_b]: device
 *  fp32, caller-owned, out not overlapping a or b. DSTD_E_INVALID for null
 *  pointers, non-positive sizes or a non-finite delay. */
int dstd_concat_channels(const float *a, int C_a, float delay_a, const float *b, int C_b, int64_t positions,
                         float *out, dstd_stream_t stream);
/* Adjoint of dstd_concat_channels (the delay has unit derivative): from
 * g [positions, C_a + C_b], writes g_a [positions, C_a] and g_b
 * [positions, C_b]; either may be NULL (not both). With accumulate_x != 0
 * the part is added into g_x instead of overwriting it (the block input's
 * gradient also receives the block's first layer's). */
int dstd_split_channels(const float *g, int C_a, int C_b, int64_t positions, float *g_a, int accumulate_a,
                        float *g_b, int accumulate_b, dstd_stream_t stream);

/* Cross-entropy over softmax(-t/tau_soft) (Eqs. cost_function, L, S_i),
 * mini-batch mean; a silent output enters with the constant time t_silent
 * and passes no gradient.
 *  t_L [B, C], labels [B] int32 in [0, C); loss float[1] out; g_t_L [B, C] out. */
int dstd_ce_loss(const float *t_L, const int32_t *labels, int B, int C, float tau_soft, float t_silent,
                 float *loss, float *g_t_L, dstd_stream_t stream);

/* Loss = sum of the output spike times that fire; g = 1 where fired, else 0.
 *  t [n]; loss float[1] out; g [n] out. */
int dstd_sum_t_loss(const float *t, int64_t n, float *loss, float *g, dstd_stream_t stream);

/* AdamW step (App. C.1; decoupled weight decay), in place on w, m, v [n];
 * step is the 1-based update count. */
int dstd_adamw(float *w, const float *g, float *m, float *v, int64_t n, float lr, float beta1,
               float beta2, float eps, float weight_decay, int step, dstd_stream_t stream);

/* AdamW step (App. C.1) on up to 32 parameter tensors in one launch, with the
 * update count kept in device memory, so that a CUDA graph that captures the
 * call advances it on every replay.
 *  w[i], g[i], m[i], v[i]: host arrays of count device pointers, tensor i
 *      holding n[i] floats (w, m, v updated in place, g read);
 *  step: device int32[2], caller-owned, 8-byte aligned; step[0] = updates done
 *      so far (0 before the first), which the call uses plus one for the bias
 *      corrections and then stores; step[1] is the kernel's scratch and must
 *      be 0 before the first call (the call leaves it 0);
 *  lr_dev: optional device float read at run time in place of lr (a warm-up
 *      schedule under graph replay), or NULL.
 * Calls that share one step buffer must not overlap on the GPU. Returns
 * DSTD_E_INVALID for count outside [1, 32], a null pointer, n[i] < 1 or
 * invalid hyperparameters; nothing is launched then. */
int dstd_adamw_multi(int count, float *const *w, const float *const *g, float *const *m,
                     float *const *v, const int64_t *n, float lr, float beta1, float beta2,
                     float eps, float weight_decay, int32_t *step, const float *lr_dev,
                     dstd_stream_t stream);

/* The exact (event-driven) first-spike times of one dense layer, Alg. 1 /
 * Eq. timing_exact: the method DSTD replaces, on the same GPU, for timing
 * and accuracy comparisons. Per sample the finite input spike times before
 * p->t_end are sorted; the potential sum_{j<=k} w_ij K(t - t~_j) is walked
 * interval by interval and the first interval that reaches p->v_th holds
 * the spike. Spike times are exact up to fp32 (no grid); a neuron that does
 * not fire before p->t_end gets +inf. Only tau_m, tau_s, v_th and t_end of p
 * are used (t_first, M only for the root's tolerance); dstd_exact_bwd
 * gives its gradients.
 *  t_in [B, N_in] (+inf = silent), W [N_out, N_in] fp32, t_out [B, N_out] out;
 *  workspace of dstd_exact_workspace_bytes (16-byte aligned).
 * N_in up to 8192 (DSTD_E_UNSUPPORTED beyond). */
size_t dstd_exact_workspace_bytes(int B, int N_in, int N_out);
int dstd_exact_fwd(const float *t_in, const float *W, int B, int N_in, int N_out,
                   const dstd_params *p, float *t_out, void *workspace, size_t ws_bytes,
                   dstd_stream_t stream);
/* Backward of the exact layer: the implicit function theorem at each exact
 * spike time (Eq. timing_exact). A neuron i that fires at t_i (from
 * dstd_exact_fwd) has sum_j w_ij K(t_i - t_j) = v_th over its inputs with
 * t_j < t_i; with the slope V'_i = sum_j w_ij K'(t_i - t_j) there,
 *   g_W[i, j]    = -sum_b g_t_out[b, i] K(t_bi - t_bj) / V'_bi,
 *   g_t_in[b, j] =  sum_i g_t_out[b, i] w_ij K'(t_bi - t_bj) / V'_bi,
 * over the pairs with t_bj < t_bi; silent neurons and later inputs give 0.
 * K and K' are recomputed for every pair (nothing per candidate is stored):
 * O(B N_out N_in) exponentials. No penalty terms: add their dT/dt to
 * g_t_out. g_t_in may be NULL; g_W and g_t_in are overwritten. Same
 * workspace as dstd_exact_fwd. */
int dstd_exact_bwd(const float *t_in, const float *W, const float *t_out, const float *g_t_out,
                   int B, int N_in, int N_out, const dstd_params *p, float *g_t_in, float *g_W,
                   void *workspace, size_t ws_bytes, dstd_stream_t stream);

/* How the forward contraction of a wide dense layer is scheduled: on single
 * CTAs (128 x 128 tiles) or on SM pairs (tcgen05 cta_group::2, 256 x 128
 * tiles, half of B per SM). policy 0 (the default) lets a cost model choose
 * per layer; 1 takes SM pairs wherever they apply (x3 and bf16 forwards
 * without split-K); 2 never does. Results agree to fp32 rounding either
 * way. Returns the previous policy (0, 1 or 2), or DSTD_E_INVALID (negative)
 * for another value.
 * Process-wide; set it between calls, not while other threads launch. */
int dstd_set_pair_policy(int policy);

/* Images per chunk of the implicit-GEMM conv layers (bf16, channels in
 * multiples of 64): 0 (the default) takes as many as fit about 4 GiB of
 * per-image scratch; n > 0 caps a chunk at n images. It changes the
 * workspace size that dstd_conv_workspace_bytes returns, so query again
 * after setting it. Returns the previous value (max_images < 0 only reads
 * it). Process-wide; set it between calls, not while other threads launch. */
int dstd_conv_set_chunk_images(int max_images);

/* Operand of the implicit-GEMM conv forward and dW (bf16 layers above):
 * 1 generates the binned input tile by tile in shared memory from the
 * 8-byte records; 2 writes it out once per chunk, S [images, H, W, Mp, C_in]
 * in bf16 (the two nonzero grid weights of each input at grid steps k and
 * k + 1, zeros elsewhere), and the contractions read it through TMA boxes
 * shifted per filter tap; 0 (the default) writes S wherever its writer takes
 * the channel count (C_in <= 256, or a multiple of 256 up to 1024) and
 * generates elsewhere. Both compute the same products. It changes the workspace size, so query again after setting
 * it. Returns the previous value (a policy outside 0..2 only reads it).
 * Process-wide; set it between calls. */
int dstd_conv_set_operand_policy(int policy);

/* Kernel timing (tracing). While enabled, the library brackets every kernel
 * it launches with a CUDA event pair on the launching stream and files the
 * pair under the kernel's kind (dstd_kernel_kind_name). Kernels that
 * otherwise run beside each other on the library's side streams (the layer
 * backward's operand producers) then run one after another on the caller's
 * stream, so that each kind's time is that kernel's alone.
 * dstd_timing_enable(on) turns timing on/off and clears the counters.
 * dstd_timing_read(kind, total_ms, launches) synchronises the device and
 * returns the accumulated device time and launch count of one kind. */
int dstd_timing_enable(int on);
int dstd_timing_read(int kind, float *total_ms, int64_t *launches);
/* While timing is enabled, launches made on a stream that is being captured
 * into a CUDA graph are bracketed by event-record nodes of the graph instead
 * (the events stay with the graph: dstd_timing_enable drops them from the
 * library's lists without reusing them). After each replay of such a graph,
 * dstd_timing_collect() synchronises the device and adds that replay's
 * device time between every pair to its kind's totals. */
int dstd_timing_collect(void);
int dstd_kernel_kind_count(void);
const char *dstd_kernel_kind_name(int kind);

/* Self-test of the bounded device waits (failure detection without a fault):
 * launches one block whose thread waits on an mbarrier that nothing ever
 * completes, giving up after timeout_us microseconds (at most 10 s) and
 * setting the device status word, which dstd_device_status() then reports as
 * DSTD_E_TIMEOUT. The context stays usable. */
int dstd_selftest_wait_timeout(uint32_t timeout_us, dstd_stream_t stream);

/* Synchronises the current device and returns DSTD_OK, DSTD_E_TIMEOUT if a
 * bounded device wait expired since the last clear, or DSTD_E_CUDA.
 * clear != 0 resets the status word. */
int dstd_device_status(int clear);

/* Message for a DSTD_E_* code (static string). */
const char *dstd_error_string(int code);

/* Library version, major*10000 + minor*100 + patch. */
int dstd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DSTD_H */
