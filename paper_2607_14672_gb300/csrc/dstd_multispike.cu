// Multi-spike regime (App. D, "Extension to multi-spike regime"): a neuron
// may fire up to F times; at each spike v is reset to 0 and I is kept
// (Eq. Vmem_multiSpikes). Every input spike is discretised on its own and
// the grid weights of an input's spikes are summed (s_jm = sum_f s_jm^f), so
// the contraction w^ = W s is unchanged; the scan continues after each spike
// from the state (0, I(t_k)), and the spikes are found one after another.
//
//   k_binning_ms_rows  forward operand [B*Mp, ld]: row (b, m), column j
//   k_binning_ms_cols  dW operand      [N, ld]:    row j, column (b, m)
//   k_scan_ms          one thread per neuron: the walk over the M intervals
//                      with the decayed (v, I) state; on a spike, the reset
//                      and a new test of the rest of the same interval
//   k_dwhat_ms         dC/dw^ through the chain of spikes (implicit function
//                      theorem per spike, adjoints from the last spike back)
//   k_gt_ms            the input-time gradient of every input spike from dS
#include "dstd_internal.cuh"

namespace dstd {

namespace {

inline unsigned ms_blocks(long long n, int threads) { return (unsigned)((n + threads - 1) / threads); }

template <int OP>
__device__ __forceinline__ void ms_store(void *hi, void *lo, long long o, float v) {
    if (OP == 0) {
        static_cast<float *>(hi)[o] = v;
    } else if (OP == 3) {
        const __half h = __float2half_rn(v);
        static_cast<__half *>(hi)[o] = h;
        static_cast<__half *>(lo)[o] = __float2half_rn(v - __half2float(h));
    } else {
        const __nv_bfloat16 h = __float2bfloat16_rn(v);
        static_cast<__nv_bfloat16 *>(hi)[o] = h;
        if (OP == 1) static_cast<__nv_bfloat16 *>(lo)[o] = __float2bfloat16_rn(v - __bfloat162float(h));
    }
}

// the grid weights of the F spikes of one input: value at bin m
struct MsBins {
    int k[kMsMaxSpikes];
    float wR[kMsMaxSpikes], wL[kMsMaxSpikes];
    int n;
};
__device__ __forceinline__ void ms_bins(const LifConst &c, const float *t, int F, MsBins &b) {
    b.n = 0;
    for (int f = 0; f < F; ++f) {
        const float x = t[f];
        if (!isfinite(x)) continue;
        const BinW w = bin_weights(c, x, false);
        b.k[b.n] = w.k;
        b.wR[b.n] = w.wR;
        b.wL[b.n] = w.wL;
        ++b.n;
    }
}
__device__ __forceinline__ float ms_value(const LifConst &c, const MsBins &b, int m) {
    float v = 0.f;
    if (m >= c.M) return 0.f;
    for (int u = 0; u < b.n; ++u) {
        if (m == b.k[u]) v += b.wR[u];
        if (m == b.k[u] + 1) v += b.wL[u];
    }
    return v;
}

}  // namespace

template <int OP>
__global__ void k_binning_ms_rows(const float *__restrict__ t, int B, int N, int F, LifConst c, void *hi, void *lo,
                                  int ld) {
    const int b = blockIdx.y;
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= ld) return;
    MsBins bins;
    bins.n = 0;
    if (j < N) ms_bins(c, t + ((long long)b * N + j) * F, F, bins);
    for (int m = 0; m < c.Mp; ++m) ms_store<OP>(hi, lo, ((long long)b * c.Mp + m) * ld + j, ms_value(c, bins, m));
}

// a warp per (input j, sample b): lane f < F discretises spike f, the warp
// shares the results, and lane l writes bins l, l + 32, ... of the row
// segment (contiguous: column b*Mp + m)
template <int OP>
__global__ void __launch_bounds__(256) k_binning_ms_cols(const float *__restrict__ t, int B, int N, int F, LifConst c,
                                                         void *hi, void *lo, int ld) {
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x;
    const int b = blockIdx.y * 8 + (threadIdx.x >> 5);
    if (b >= B) return;
    int kf = -100;
    float wr = 0.f, wl = 0.f;
    if (lane < F) {
        const float x = t[((long long)b * N + j) * F + lane];
        if (isfinite(x)) {
            const BinW w = bin_weights(c, x, false);
            kf = w.k;
            wr = w.wR;
            wl = w.wL;
        }
    }
    MsBins bins;
    bins.n = 0;
    for (int f = 0; f < F; ++f) {
        const int k = __shfl_sync(0xffffffffu, kf, f);
        const float r = __shfl_sync(0xffffffffu, wr, f), l = __shfl_sync(0xffffffffu, wl, f);
        if (k != -100) {
            bins.k[bins.n] = k;
            bins.wR[bins.n] = r;
            bins.wL[bins.n] = l;
            ++bins.n;
        }
    }
    const long long o = (long long)j * ld + (long long)b * c.Mp;
    for (int m = lane; m < c.Mp; m += 32) ms_store<OP>(hi, lo, o + m, ms_value(c, bins, m));
}

cudaError_t launch_binning_ms(const float *t, int B, int N, int F, const LifConst &c, OpKind op, bool transposed,
                              void *hi, void *lo, int ld, cudaStream_t st) {
    if (F < 1 || F > kMsMaxSpikes) return cudaErrorInvalidValue;
#define DSTD_MS_BIN(OPV)                                                                                        \
    if (transposed)                                                                                             \
        k_binning_ms_cols<OPV><<<dim3((unsigned)N, (unsigned)((B + 7) / 8)), 256, 0, st>>>(t, B, N, F, c, hi,  \
                                                                                           lo, ld);             \
    else                                                                                                        \
        k_binning_ms_rows<OPV><<<dim3((unsigned)((ld + 127) / 128), (unsigned)B), 128, 0, st>>>(t, B, N, F, c, \
                                                                                                hi, lo, ld);
    switch (op) {
        case OpKind::F32: DSTD_MS_BIN(0) break;
        case OpKind::BF16X3: DSTD_MS_BIN(1) break;
        case OpKind::BF16: DSTD_MS_BIN(2) break;
        default: DSTD_MS_BIN(3) break;
    }
#undef DSTD_MS_BIN
    return cudaGetLastError();
}

// One thread per neuron (b, i): w^ of bin m at what[b*sb + i*si + m]. On
// interval m the state (v, I0) at its start is tested exactly (the same
// test and root as the first-spike scan, with the interval's remaining
// length); on a spike at s the state becomes (0, I0 e^{-aI s}) and the rest
// of the interval, of length L - s, is tested again. Outputs per spike k
// (index (b*N + i)*F + k): t, the bin q, I at the spike and dv^/dt there;
// t = +inf, q = M after the last spike.
__global__ void __launch_bounds__(256) k_scan_ms(const float *__restrict__ what, long long sb, long long si, int B,
                                                 int N, LifConst c, int F, float *t_out, int *q_out, float *I_out,
                                                 float *vd_out, int vec4) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N) return;
    const int b = (int)(idx / N), i = (int)(idx % N);
    const float *w = what + b * sb + i * si;
    float v = 0.f, I = 0.f;
    int nk = 0;
    const long long o = idx * F;
    float4 w4 = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int m = 0; m < c.M && nk < F; ++m) {
        if (vec4) {
            if ((m & 3) == 0) w4 = __ldg(reinterpret_cast<const float4 *>(w + m));
        }
        const float wm = vec4 ? ((m & 3) == 0 ? w4.x : (m & 3) == 1 ? w4.y : (m & 3) == 2 ? w4.z : w4.w) : w[m];
        float v0 = v, I0 = I + wm;
        // a whole interval with no spike in it yet: the cheap tests of the
        // first-spike scan decide whether the exact test is needed
        {
            const float ve = fmaf(c.KD, I0, c.rv * v0);
            const bool endp = ve >= c.vth;
            const bool peak = (fmaf(-c.av, v0, I0) > 0.0f) & (fmaf(-c.av, ve, c.rI * I0) < 0.0f) &
                              (fmaf(fmaxf(I0, 0.0f), c.Kmax, fmaxf(v0, 0.0f)) >= c.vth);
            if (!(endp | peak)) {
                v = ve;
                I = c.rI * I0;
                continue;
            }
        }
        float L = c.dt, start = c.T0 + (float)m * c.dt;
        // at most F spikes in all, so the inner loop ends
        while (nk < F) {
            const float rI = expf(-c.aI * L);
            const float ve = fmaf(expf(-c.av * L) * phi_f(c, L), I0, expf(-c.av * L) * v0);
            const float hi = interval_test(c.av, c.aI, c.lam, c.lam_zero, rI, L, c.vth, v0, I0, ve);
            if (hi < 0.0f) break;
            const float s = hi > 0.0f ? interval_root(c, v0, I0, hi) : 0.0f;
            const float Ik = I0 * expf(-c.aI * s);
            t_out[o + nk] = start + s;
            q_out[o + nk] = m;
            I_out[o + nk] = Ik;
            vd_out[o + nk] = fmaxf(fmaf(-c.av, c.vth, Ik), c.vdot_floor);
            ++nk;
            v0 = 0.f;
            I0 = Ik;
            start += s;
            L -= s;
            if (!(L > 1e-7f * c.dt)) break;  // the spike closed the interval
        }
        // the state at T_{m+1}
        const float e = expf(-c.av * L);
        v = fmaf(e * phi_f(c, L), I0, e * v0);
        I = I0 * expf(-c.aI * L);
    }
    for (int k = nk; k < F; ++k) {
        t_out[o + k] = INFINITY;
        q_out[o + k] = c.M;
        I_out[o + k] = 0.f;
        vd_out[o + k] = 0.f;
    }
}

cudaError_t launch_scan_ms(const float *what, long long sb, long long si, int B, int N, const LifConst &c, int F,
                           float *t_out, int *q, float *I, float *vd, cudaStream_t st) {
    if (F < 1 || F > kMsMaxSpikes) return cudaErrorInvalidValue;
    // 16-byte loads when every row of bins starts on a 16-byte boundary
    const int vec4 = (sb % 4 == 0) && (si % 4 == 0) && (reinterpret_cast<uintptr_t>(what) % 16 == 0) && (c.Mp % 4 == 0);
    k_scan_ms<<<ms_blocks((long long)B * N, 256), 256, 0, st>>>(what, sb, si, B, N, c, F, t_out, q, I, vd, vec4);
    return cudaGetLastError();
}

// dC/dw^_im of one neuron from dC/dt_k of its spikes. With v'_k the saved
// dv^/dt at spike k:
//   spike 0:  dt_0/dw^_m = -K(t_0 - T_m)/v'_0, m <= q_0;
//   spike k:  dt_k/dw^_m = -e^{-aI (t_{k-1} - T_m)} K(t_k - t_{k-1}) / v'_k  for m <= q_{k-1},
//                        = -K(t_k - T_m) / v'_k                             for q_{k-1} < m <= q_k,
//             dt_k/dt_{k-1} = -I_{k-1} [(av - aI) K(s) - e^{-aI s}] / v'_k, s = t_k - t_{k-1}
// (the current kept through the reset decays at aI; dK/ds = -av K + e^{-aI s}).
// The adjoints a_k = dC/dt_k + a_{k+1} dt_{k+1}/dt_k run from the last
// spike back; dC/dw^_m = sum_k a_k dt_k/dw^_m.
//
// A block takes 32 neurons of one sample: thread i < 32 runs neuron i's
// adjoints into shared memory, the block fills a [Mp][32] tile of dC/dw^
// (zero after a neuron's last spike), and writes it to both layouts with
// contiguous stores: the (i, (b, m)) rows (a warp per neuron, lanes over m)
// and, when b_hi is given, the ((b, m), i) rows (lanes over the 32 neurons).
constexpr int MS_DW_NEURONS = 32;
template <int OP>
__global__ void __launch_bounds__(256) k_dwhat_ms(const float *__restrict__ t_out, const int *__restrict__ qv,
                                                  const float *__restrict__ Iv, const float *__restrict__ vdv,
                                                  const float *__restrict__ g_up, int B, int N, int F, LifConst c,
                                                  void *a_hi, void *a_lo, int lda, void *b_hi, void *b_lo, int ldb) {
    extern __shared__ __align__(16) float dsm[];
    float *tile = dsm;                                        // [Mp][33]
    float *stk = tile + c.Mp * (MS_DW_NEURONS + 1);           // [32][F] spike times
    float *scf = stk + MS_DW_NEURONS * F;                     // [32][F] coefficients -a_k / v'_k
    float *sKk = scf + MS_DW_NEURONS * F;                     // [32][F] K(t_k - t_{k-1})
    int *sq = reinterpret_cast<int *>(sKk + MS_DW_NEURONS * F);  // [32][F] bins
    int *sn = sq + MS_DW_NEURONS * F;                         // [32] spike counts
    const int b = blockIdx.y;
    const int i0 = blockIdx.x * MS_DW_NEURONS;
    const int tid = threadIdx.x;
    if (tid < MS_DW_NEURONS) {
        const int i = i0 + tid;
        int n = 0;
        if (i < N) {
            const long long o = ((long long)b * N + i) * F;
            float tk[kMsMaxSpikes], Ik[kMsMaxSpikes], coef[kMsMaxSpikes];
            for (int k = 0; k < F; ++k) {
                if (qv[o + k] >= c.M) break;
                tk[k] = t_out[o + k];
                Ik[k] = Iv[o + k];
                coef[k] = g_up ? g_up[o + k] : 0.f;
                sq[tid * F + k] = qv[o + k];
                n = k + 1;
            }
            // adjoints, last spike first; coef_k = -a_k / v'_k
            for (int k = n - 1; k >= 0; --k) {
                coef[k] = -coef[k] / vdv[o + k];
                if (k > 0) {
                    const float s = tk[k] - tk[k - 1];
                    const float dv_dprev = Ik[k - 1] * fmaf(c.av - c.aI, kernel_K(c, s), -expf(-c.aI * s));
                    coef[k - 1] += coef[k] * dv_dprev;  // a_{k-1} += a_k (-dv_dprev / v'_k)
                }
            }
            for (int k = 0; k < n; ++k) {
                stk[tid * F + k] = tk[k];
                scf[tid * F + k] = coef[k];
                sKk[tid * F + k] = k > 0 ? kernel_K(c, tk[k] - tk[k - 1]) : 0.f;
            }
        }
        sn[tid] = n;
    }
    __syncthreads();
    // the tile: thread (neuron il, bins m = row, row + 8, ...)
    for (int e = tid; e < c.Mp * MS_DW_NEURONS; e += blockDim.x) {
        const int il = e % MS_DW_NEURONS, m = e / MS_DW_NEURONS;
        const int n = sn[il];
        float val = 0.f;
        if (n > 0 && m <= sq[il * F + n - 1]) {
            const float Tm = c.T0 + (float)m * c.dt;
            for (int k = 0; k < n; ++k) {
                const int qk = sq[il * F + k];
                if (m > qk) continue;
                float basis;
                if (k > 0 && m <= sq[il * F + k - 1])
                    basis = expf(-c.aI * (stk[il * F + k - 1] - Tm)) * sKk[il * F + k];
                else
                    basis = kernel_K(c, stk[il * F + k] - Tm);
                val = fmaf(scf[il * F + k], basis, val);
            }
        }
        tile[m * (MS_DW_NEURONS + 1) + il] = val;
    }
    __syncthreads();
    const int lane = tid & 31, warp = tid >> 5;
    for (int il = warp; il < MS_DW_NEURONS; il += blockDim.x / 32) {
        const int i = i0 + il;
        if (i >= N) break;
        const long long oa = (long long)i * lda + (long long)b * c.Mp;
        for (int m = lane; m < c.Mp; m += 32) ms_store<OP>(a_hi, a_lo, oa + m, tile[m * (MS_DW_NEURONS + 1) + il]);
    }
    if (b_hi) {
        const int i = i0 + lane;
        if (i < N)
            for (int m = warp; m < c.Mp; m += blockDim.x / 32)
                ms_store<OP>(b_hi, b_lo, ((long long)b * c.Mp + m) * ldb + i, tile[m * (MS_DW_NEURONS + 1) + lane]);
    }
}

cudaError_t launch_dwhat_ms(const float *t_out, const int *q, const float *I, const float *vd, const float *g_up,
                            int B, int N, int F, const LifConst &c, OpKind op, void *a_hi, void *a_lo, int lda,
                            void *b_hi, void *b_lo, int ldb, cudaStream_t st) {
    if (F < 1 || F > kMsMaxSpikes) return cudaErrorInvalidValue;
    const size_t smem = sizeof(float) * ((size_t)c.Mp * (MS_DW_NEURONS + 1) + 4 * MS_DW_NEURONS * F + MS_DW_NEURONS);
    const dim3 g((unsigned)((N + MS_DW_NEURONS - 1) / MS_DW_NEURONS), (unsigned)B);
    if (op == OpKind::F32)
        k_dwhat_ms<0><<<g, 256, smem, st>>>(t_out, q, I, vd, g_up, B, N, F, c, a_hi, a_lo, lda, b_hi, b_lo, ldb);
    else if (op == OpKind::BF16X3)
        k_dwhat_ms<1><<<g, 256, smem, st>>>(t_out, q, I, vd, g_up, B, N, F, c, a_hi, a_lo, lda, b_hi, b_lo, ldb);
    else
        k_dwhat_ms<2><<<g, 256, smem, st>>>(t_out, q, I, vd, g_up, B, N, F, c, a_hi, a_lo, lda, b_hi, b_lo, ldb);
    return cudaGetLastError();
}

// g_t of input spike f of input j in sample b: sum over its two bins of
// dS[j, (b, m)] ds_jm/dt (Tab. DSTD_kernels' derivative); 0 when silent.
__global__ void k_gt_ms(const float *__restrict__ D, long long ldd, const float *__restrict__ t_in, int B, int N,
                        int F, LifConst c, float *g_t_in) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N * F) return;
    const long long bj = idx / F;
    const int b = (int)(bj / N), j = (int)(bj % N);
    const float x = t_in[idx];
    float g = 0.f;
    if (isfinite(x)) {
        const BinW w = bin_weights(c, x, true);
        const float *row = D + (long long)j * ldd + (long long)b * c.Mp;
        if (w.k >= 0 && w.k < c.M) g += row[w.k] * w.dR;
        if (w.k + 1 >= 0 && w.k + 1 < c.M) g += row[w.k + 1] * w.dL;
    }
    g_t_in[idx] = g;
}

cudaError_t launch_gt_ms(const float *D, long long ldd, const float *t_in, int B, int N, int F, const LifConst &c,
                         float *g_t_in, cudaStream_t st) {
    const long long n = (long long)B * N * F;
    k_gt_ms<<<ms_blocks(n, 256), 256, 0, st>>>(D, ldd, t_in, B, N, F, c, g_t_in);
    return cudaGetLastError();
}

}  // namespace dstd
