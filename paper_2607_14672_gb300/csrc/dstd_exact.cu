// The exact (event-driven) TTFS layer on the GPU: Alg. 1 of the paper, the
// method DSTD replaces, forward and backward, for an on-device comparison of
// the two.
//
// Per sample the finite input spike times before the window end are sorted,
// t~_1 <= ... <= t~_K; on each interval [t~_k, t~_{k+1}) (the last closed at
// the window end) the potential is sum_{j<=k} w_ij K(t - t~_j), and the first
// interval whose potential reaches v_th holds the spike (Eq. timing_exact).
// That potential is carried, as in the DSTD scan, as the exact decayed state
// (v, I) at the interval's start: I jumps by the weight of the input that
// opens it, and over an interval of length L, (v, I) <- (e^{-av L} v +
// K(L) I, e^{-aI L} I). The interval test and its root are those of the
// DSTD scan with the interval's length in place of the grid step.
//
//   k_exact_sort  one block per sample: a bitonic sort of (t, j) in shared
//                 memory (ties by input index, so the order is reproducible),
//                 then each interval's start, length and decay factors;
//   k_exact_walk  one thread per output neuron, 256 neurons of one sample
//                 per block (the sample's sorted intervals in shared
//                 memory): I += W_ij for the input opening each interval,
//                 read from W transposed so that a warp's 32 neurons load one
//                 128-byte row.
#include "dstd_internal.cuh"

namespace dstd {

constexpr int EXACT_SORT_THREADS = 512, EXACT_WALK_THREADS = 256;

__global__ void __launch_bounds__(EXACT_SORT_THREADS) k_exact_sort(const float *__restrict__ t_in, int N_in,
                                                                 LifConst c, float t_end, int P, int *perm,
                                                                 float *t_start, float4 *iv, int *count) {
    extern __shared__ __align__(16) unsigned char esm[];
    float *key = reinterpret_cast<float *>(esm);
    int *idx = reinterpret_cast<int *>(key + P);
    const int b = blockIdx.x;
    for (int e = threadIdx.x; e < P; e += EXACT_SORT_THREADS) {
        float x = e < N_in ? t_in[(long long)b * N_in + e] : INFINITY;
        if (!isfinite(x) || !(x < t_end)) x = INFINITY;  // silent, or after the window: no effect on it
        key[e] = x;
        idx[e] = e;
    }
    __syncthreads();
    // bitonic sort, ascending by (time, input index)
    for (int size = 2; size <= P; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int e = threadIdx.x; e < P; e += EXACT_SORT_THREADS) {
                const int f = e ^ stride;
                if (f > e) {
                    const bool up = (e & size) == 0;
                    const float ke = key[e], kf = key[f];
                    const int ie = idx[e], jf = idx[f];
                    const bool gt = ke > kf || (ke == kf && ie > jf);
                    if (gt == up) {
                        key[e] = kf;
                        key[f] = ke;
                        idx[e] = jf;
                        idx[f] = ie;
                    }
                }
            }
            __syncthreads();
        }
    }
    // the finite keys come first: count them, then the intervals they open
    for (int e = threadIdx.x; e < P; e += EXACT_SORT_THREADS)
        if (isfinite(key[e]) && (e + 1 == P || !isfinite(key[e + 1]))) count[b] = e + 1;
    if (threadIdx.x == 0 && !isfinite(key[0])) count[b] = 0;
    for (int e = threadIdx.x; e < N_in; e += EXACT_SORT_THREADS) {
        const float t0 = key[e];
        if (!isfinite(t0)) break;
        const float t1 = (e + 1 < P && isfinite(key[e + 1])) ? key[e + 1] : t_end;
        const float L = t1 - t0;
        const float rv = expf(-c.av * L);
        const long long o = (long long)b * N_in + e;
        perm[o] = idx[e];
        t_start[o] = t0;
        iv[o] = make_float4(rv, expf(-c.aI * L), rv * phi_f(c, L), L);
    }
}

__global__ void __launch_bounds__(EXACT_WALK_THREADS) k_exact_walk(const float *__restrict__ Wt, int N_in, int N_out,
                                                                 LifConst c, float kmax,
                                                                 const int *__restrict__ perm,
                                                                 const float *__restrict__ t_start,
                                                                 const float4 *__restrict__ iv,
                                                                 const int *__restrict__ count, float *t_out) {
    extern __shared__ __align__(16) unsigned char esm[];
    float4 *siv = reinterpret_cast<float4 *>(esm);
    float *st = reinterpret_cast<float *>(siv + N_in);
    int *sp = reinterpret_cast<int *>(st + N_in);
    const int b = blockIdx.y;
    const int n = count[b];
    for (int e = threadIdx.x; e < n; e += EXACT_WALK_THREADS) {
        const long long o = (long long)b * N_in + e;
        siv[e] = iv[o];
        st[e] = t_start[o];
        sp[e] = perm[o];
    }
    __syncthreads();
    const int i = blockIdx.x * EXACT_WALK_THREADS + threadIdx.x;
    if (i >= N_out) return;
    float v = 0.f, I = 0.f, t = INFINITY;
    for (int k = 0; k < n; ++k) {
        const float I0 = I + Wt[(long long)sp[k] * N_out + i];
        const float4 q = siv[k];  // e^{-av L}, e^{-aI L}, K(L), L
        const float ve = fmaf(q.z, I0, q.x * v);
        const float In = q.y * I0;
        const bool endp = ve >= c.vth;
        const bool peak = (fmaf(-c.av, v, I0) > 0.0f) & (fmaf(-c.av, ve, In) < 0.0f) &
                          (fmaf(fmaxf(I0, 0.0f), kmax, fmaxf(v, 0.0f)) >= c.vth);
        if (endp | peak) {
            const float hi = interval_test(c.av, c.aI, c.lam, c.lam_zero, q.y, q.w, c.vth, v, I0, ve);
            if (hi >= 0.0f) {
                t = st[k] + (hi > 0.0f ? interval_root(c, v, I0, hi) : 0.0f);
                break;
            }
        }
        v = ve;
        I = In;
    }
    t_out[(long long)b * N_out + i] = t;
}

cudaError_t launch_exact_fwd(const float *t_in, const float *W, int B, int N_in, int N_out, const LifConst &c,
                             float t_end, float kmax, const ExactWs &ws, float *t_out, cudaStream_t st) {
    if (N_in < 1 || N_in > kExactMaxIn) return cudaErrorInvalidValue;
    int P = 1;
    while (P < N_in) P <<= 1;
    cudaError_t e = launch_prep_weights(W, N_out, N_in, OpKind::F32, nullptr, nullptr, 0, nullptr, nullptr, 0, ws.Wt,
                                        N_out, nullptr, st);
    if (e != cudaSuccess) return e;
    const size_t smem_sort = (size_t)P * 8;
    if (smem_sort > 48 * 1024) {
        e = cudaFuncSetAttribute(k_exact_sort, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_sort);
        if (e != cudaSuccess) return e;
    }
    k_exact_sort<<<B, EXACT_SORT_THREADS, smem_sort, st>>>(t_in, N_in, c, t_end, P, ws.perm, ws.t_start, ws.iv,
                                                          ws.count);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const size_t smem_walk = (size_t)N_in * (sizeof(float4) + 8);
    if (smem_walk > 48 * 1024) {
        e = cudaFuncSetAttribute(k_exact_walk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_walk);
        if (e != cudaSuccess) return e;
    }
    dim3 grid((N_out + EXACT_WALK_THREADS - 1) / EXACT_WALK_THREADS, B);
    k_exact_walk<<<grid, EXACT_WALK_THREADS, smem_walk, st>>>(ws.Wt, N_in, N_out, c, kmax, ws.perm, ws.t_start,
                                                             ws.iv, ws.count, t_out);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Backward of the exact method: the implicit function theorem at each exact
// spike time. Neuron i fires at t_i with sum_j w_ij K(t_i - t_j) = v_th over
// its inputs before t_i; with the slope V'_i = sum_j w_ij K'(t_i - t_j),
//   dC/dw_ij = -g_i K(t_i - t_j) / V'_i,   dC/dt_j += g_i w_ij K'(t_i - t_j) / V'_i.
// K(x) = e^{-av x} phi(x) and K'(x) = e^{-aI x} - av K(x) are recomputed for
// every (sample, neuron, input) pair: nothing per candidate is kept, at the
// price of O(B N_out N_in) exponentials.
//   k_exact_slope  one thread per (sample, neuron): V'_i and g_i / V'_i
//   k_exact_gw     16 x 16 (neuron, input) tiles, samples staged in shared memory
//   k_exact_gt     one thread per (sample, input), neurons staged in shared memory
// ---------------------------------------------------------------------------
constexpr int EXACT_BWD_THREADS = 256, EXACT_BWD_CHUNK = 32;

__device__ __forceinline__ float exact_K(const LifConst &c, float x) { return __expf(-c.av * x) * phi_f(c, x); }
__device__ __forceinline__ float exact_dK(const LifConst &c, float x) {
    return __expf(-c.aI * x) - c.av * exact_K(c, x);
}

__global__ void __launch_bounds__(EXACT_BWD_THREADS) k_exact_slope(const float *__restrict__ t_in,
                                                                   const float *__restrict__ Wt,
                                                                   const float *__restrict__ t_out,
                                                                   const float *__restrict__ g_out, int N_in,
                                                                   int N_out, LifConst c, float *__restrict__ coef) {
    extern __shared__ float xs[];  // the sample's input times
    const int b = blockIdx.y;
    for (int j = threadIdx.x; j < N_in; j += EXACT_BWD_THREADS) xs[j] = t_in[(long long)b * N_in + j];
    __syncthreads();
    const int i = blockIdx.x * EXACT_BWD_THREADS + threadIdx.x;
    if (i >= N_out) return;
    const float ti = t_out[(long long)b * N_out + i];
    float cf = 0.f;
    if (isfinite(ti)) {
        float vp = 0.f;
        for (int j = 0; j < N_in; ++j) {
            const float x = ti - xs[j];  // +inf inputs give -inf
            if (x > 0.f) vp = fmaf(Wt[(long long)j * N_out + i], exact_dK(c, x), vp);
        }
        cf = g_out[(long long)b * N_out + i] / vp;
    }
    coef[(long long)b * N_out + i] = cf;
}

__global__ void __launch_bounds__(EXACT_BWD_THREADS) k_exact_gw(const float *__restrict__ t_in,
                                                                const float *__restrict__ t_out,
                                                                const float *__restrict__ coef, int B, int N_in,
                                                                int N_out, LifConst c, float *__restrict__ g_W) {
    __shared__ float so[EXACT_BWD_CHUNK][16], sc[EXACT_BWD_CHUNK][16], si[EXACT_BWD_CHUNK][16];
    const int tj = threadIdx.x & 15, ti = threadIdx.x >> 4;
    const int j = blockIdx.x * 16 + tj, i = blockIdx.y * 16 + ti;
    float acc = 0.f;
    for (int b0 = 0; b0 < B; b0 += EXACT_BWD_CHUNK) {
        for (int e = threadIdx.x; e < EXACT_BWD_CHUNK * 16; e += EXACT_BWD_THREADS) {
            const int bb = e >> 4, u = e & 15, b = b0 + bb;
            const int ii = blockIdx.y * 16 + u, jj = blockIdx.x * 16 + u;
            const bool okb = b < B;
            so[bb][u] = (okb && ii < N_out) ? t_out[(long long)b * N_out + ii] : INFINITY;
            sc[bb][u] = (okb && ii < N_out) ? coef[(long long)b * N_out + ii] : 0.f;
            si[bb][u] = (okb && jj < N_in) ? t_in[(long long)b * N_in + jj] : INFINITY;
        }
        __syncthreads();
        const int nb = B - b0 < EXACT_BWD_CHUNK ? B - b0 : EXACT_BWD_CHUNK;
        for (int bb = 0; bb < nb; ++bb) {
            const float cf = sc[bb][ti];
            const float x = so[bb][ti] - si[bb][tj];
            if (cf != 0.f && x > 0.f) acc = fmaf(cf, exact_K(c, x), acc);
        }
        __syncthreads();
    }
    if (i < N_out && j < N_in) g_W[(long long)i * N_in + j] = -acc;
}

__global__ void __launch_bounds__(EXACT_BWD_THREADS) k_exact_gt(const float *__restrict__ t_in,
                                                                const float *__restrict__ W,
                                                                const float *__restrict__ t_out,
                                                                const float *__restrict__ coef, int N_in, int N_out,
                                                                LifConst c, float *__restrict__ g_t_in) {
    __shared__ float so[EXACT_BWD_THREADS], sc[EXACT_BWD_THREADS];
    const int b = blockIdx.y;
    const int j = blockIdx.x * EXACT_BWD_THREADS + threadIdx.x;
    const float tj = j < N_in ? t_in[(long long)b * N_in + j] : INFINITY;
    float acc = 0.f;
    for (int i0 = 0; i0 < N_out; i0 += EXACT_BWD_THREADS) {
        const int ii = i0 + threadIdx.x;
        so[threadIdx.x] = ii < N_out ? t_out[(long long)b * N_out + ii] : INFINITY;
        sc[threadIdx.x] = ii < N_out ? coef[(long long)b * N_out + ii] : 0.f;
        __syncthreads();
        const int ni = N_out - i0 < EXACT_BWD_THREADS ? N_out - i0 : EXACT_BWD_THREADS;
        if (j < N_in && isfinite(tj)) {
            for (int u = 0; u < ni; ++u) {
                const float cf = sc[u];
                const float x = so[u] - tj;
                if (cf != 0.f && x > 0.f) acc = fmaf(cf * W[(long long)(i0 + u) * N_in + j], exact_dK(c, x), acc);
            }
        }
        __syncthreads();
    }
    if (j < N_in) g_t_in[(long long)b * N_in + j] = acc;
}

cudaError_t launch_exact_bwd(const float *t_in, const float *W, const float *t_out, const float *g_out, int B,
                             int N_in, int N_out, const LifConst &c, const ExactWs &ws, float *g_t_in, float *g_W,
                             cudaStream_t st) {
    if (N_in < 1 || N_in > kExactMaxIn) return cudaErrorInvalidValue;
    cudaError_t e = launch_prep_weights(W, N_out, N_in, OpKind::F32, nullptr, nullptr, 0, nullptr, nullptr, 0, ws.Wt,
                                        N_out, nullptr, st);
    if (e != cudaSuccess) return e;
    const size_t smem = (size_t)N_in * sizeof(float);
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(k_exact_slope, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    k_exact_slope<<<dim3((N_out + EXACT_BWD_THREADS - 1) / EXACT_BWD_THREADS, B), EXACT_BWD_THREADS, smem, st>>>(
        t_in, ws.Wt, t_out, g_out, N_in, N_out, c, ws.coef);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_exact_gw<<<dim3((N_in + 15) / 16, (N_out + 15) / 16), EXACT_BWD_THREADS, 0, st>>>(t_in, t_out, ws.coef, B, N_in,
                                                                                      N_out, c, g_W);
    e = cudaGetLastError();
    if (e != cudaSuccess || !g_t_in) return e;
    k_exact_gt<<<dim3((N_in + EXACT_BWD_THREADS - 1) / EXACT_BWD_THREADS, B), EXACT_BWD_THREADS, 0, st>>>(
        t_in, W, t_out, ws.coef, N_in, N_out, c, g_t_in);
    return cudaGetLastError();
}

}  // namespace dstd
