// Memory-bound kernels of the DSTD layer: weight preparation, binning (the
// prologue of Eq. DSTD), the scan/solve/select of Tab. timing_DSTD on a
// materialised w^, the backward's dw^ generation and input-time gradient,
// split-K reduction, losses and AdamW.
#include "dstd_internal.cuh"

#include <math.h>

namespace dstd {

int padded_M(int M) {
    int p = 8;
    while (p < M) p <<= 1;
    return p;
}

LifConst make_const(const dstd_params &p, int Mp) {
    LifConst c{};
    const double tv = p.tau_m, ti = p.tau_s;
    const double av = isinf(tv) ? 0.0 : 1.0 / tv;
    const double aI = isinf(ti) ? 0.0 : 1.0 / ti;
    const double lam = aI - av;
    const double dt = ((double)p.t_end - (double)p.t_first) / p.M;
    const double phi_dt = lam == 0.0 ? dt : -expm1(-lam * dt) / lam;
    c.av = (float)av;
    c.aI = (float)aI;
    c.lam = (float)lam;
    c.lam_zero = (lam == 0.0);
    c.inv_lam = lam == 0.0 ? 0.0f : (float)(1.0 / lam);
    c.T0 = (float)((double)p.t_first - (double)p.t_offset);
    c.dt = (float)dt;
    c.inv_dt = (float)(1.0 / dt);
    c.rv = (float)exp(-av * dt);
    c.rI = (float)exp(-aI * dt);
    c.KD = (float)(exp(-av * dt) * phi_dt);
    c.inv_phi_dt = (float)(1.0 / phi_dt);
    c.vth = p.v_th;
    c.M = p.M;
    c.Mp = Mp;
    c.vdot_floor = (float)(1e-6 * p.v_th / dt);
    {
        // K(s) = e^{-av s} phi(s) rises to a single maximum (or keeps rising
        // when av = 0 or aI = 0); take it at min(dt, peak time)
        double tp = INFINITY;  // keeps rising: the end of the window
        if (av > 0.0 && aI > 0.0) tp = (lam == 0.0) ? 1.0 / av : log(aI / av) / lam;
        const double s_ = tp < dt ? tp : dt;
        const double phis = lam == 0.0 ? s_ : -expm1(-lam * s_) / lam;
        c.Kmax = (float)(exp(-av * s_) * phis * (1.0 + 1e-6));
        const double s4 = tp < 4.0 * dt ? tp : 4.0 * dt;
        const double phi4 = lam == 0.0 ? s4 : -expm1(-lam * s4) / lam;
        c.Kmax4 = (float)(exp(-av * s4) * phi4 * (1.0 + 1e-6));
    }
    c.t_head = p.t_head;
    c.t_tail = p.t_tail;
    c.g_head = p.gamma_head;
    c.g_tail = p.gamma_tail;
    c.g_q = p.gamma_q;
    c.norm = p.penalty_norm;
    return c;
}

static inline unsigned blocks_for(long long n, int threads) {
    return (unsigned)((n + threads - 1) / threads);
}

static int num_sms_cached() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            sms <= 0)
            sms = 148;
    }
    return sms;
}

// blocks_for capped at 8 blocks per SM, for grid-stride kernels that end in
// one atomic per block
static unsigned grid_cap(long long n, int threads) {
    const int sms = num_sms_cached();
    const unsigned b = blocks_for(n, threads), cap = 8u * (unsigned)sms;
    return b < 1 ? 1 : (b < cap ? b : cap);
}

__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16 &hi, __nv_bfloat16 &lo) {
    hi = __float2bfloat16_rn(x);
    lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// ---------------------------------------------------------------------------
// Weights: fp32 [R, C] -> bf16 hi/lo [R, ldo] (zero pad), transposed copies
// [C, ldt] (bf16 hi/lo) or [C, ldf] (fp32), row sums.
// ---------------------------------------------------------------------------
__global__ void k_prep_weights(const float *__restrict__ W, int R, int C, int op, __nv_bfloat16 *hi,
                               __nv_bfloat16 *lo, int ldo, __nv_bfloat16 *hiT, __nv_bfloat16 *loT, int ldt,
                               float *f32T, int ldf, float *rowsum) {
    __shared__ float tile[32][33];
    const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
    const int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
    for (int yy = ty; yy < 32; yy += 8) {
        int r = by + yy, cc = bx + tx;
        float x = (r < R && cc < C) ? W[(long long)r * C + cc] : 0.0f;
        tile[yy][tx] = x;
        if (hi && r < R && cc < ldo) {
            __nv_bfloat16 h, l;
            split_bf16(x, h, l);
            hi[(long long)r * ldo + cc] = h;
            if (lo) lo[(long long)r * ldo + cc] = l;
        }
    }
    __syncthreads();
    // transposed writes: row = column index of W
    for (int yy = ty; yy < 32; yy += 8) {
        int cc = bx + yy, r = by + tx;
        float x = tile[tx][yy];
        if (hiT && cc < C && r < ldt) {
            __nv_bfloat16 h, l;
            split_bf16(x, h, l);
            hiT[(long long)cc * ldt + r] = h;
            if (loT) loT[(long long)cc * ldt + r] = l;
        }
        if (f32T && cc < C && r < ldf) f32T[(long long)cc * ldf + r] = x;
    }
    if (rowsum && ty == 0) {
        // one warp per 32 rows of this tile column block: accumulate partial sums
        int r = by + tx;
        if (r < R) {
            float sum = 0.0f;
            for (int k = 0; k < 32; ++k) sum += tile[tx][k];
            atomicAdd(&rowsum[r], sum);
        }
    }
    (void)op;
}

__device__ __forceinline__ void split_f16(float x, __half &hi, __half &lo) {
    hi = __float2half_rn(x);
    lo = __float2half_rn(x - __half2float(hi));
}

// One block per row: every load of the row is in flight at once (the row
// is read once into registers, up to PREP_PER_THREAD values per thread, and
// re-read from memory only for longer rows).
constexpr int PREP_THREADS = 256, PREP_PER_THREAD = 8;

// Row r of the forward weight operand (one block of PREP_THREADS threads).
__device__ __forceinline__ void prep_row_f16(const float *__restrict__ W, int R, int C, __half *hi, __half *lo, int ldo,
                                             float *inv_scale, float *rowsum, int r) {
    __shared__ float red_max[PREP_THREADS / 32], red_sum[PREP_THREADS / 32];
    __shared__ float sc_sh;
    if (r >= R) return;
    const float *w = W + (long long)r * C;
    float x[PREP_PER_THREAD];
    float amax = 0.f, sum = 0.f;
#pragma unroll
    for (int u = 0; u < PREP_PER_THREAD; ++u) {
        const int j = threadIdx.x + u * PREP_THREADS;
        x[u] = j < C ? w[j] : 0.f;
        amax = fmaxf(amax, fabsf(x[u]));
        sum += x[u];
    }
    for (int j = threadIdx.x + PREP_PER_THREAD * PREP_THREADS; j < C; j += PREP_THREADS) {
        const float y = w[j];
        amax = fmaxf(amax, fabsf(y));
        sum += y;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        sum += __shfl_xor_sync(0xffffffffu, sum, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        red_max[warp] = amax;
        red_sum[warp] = sum;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float m = 0.f, t = 0.f;
        for (int k = 0; k < PREP_THREADS / 32; ++k) {
            m = fmaxf(m, red_max[k]);
            t += red_sum[k];
        }
        // power of two bringing the row's largest |w| into [2^13, 2^14]
        int k = 0;
        if (m > 0.f && isfinite(m)) {
            int e;
            frexpf(m, &e);  // m = f 2^e, f in [0.5, 1)
            k = 14 - e;
            k = k > 100 ? 100 : (k < -100 ? -100 : k);
        }
        sc_sh = ldexpf(1.0f, k);
        inv_scale[r] = ldexpf(1.0f, -k);
        if (rowsum) rowsum[r] = t;
    }
    __syncthreads();
    const float sc = sc_sh;
#pragma unroll
    for (int u = 0; u < PREP_PER_THREAD; ++u) {
        const int j = threadIdx.x + u * PREP_THREADS;
        if (j < ldo) {
            __half h, l;
            split_f16(x[u] * sc, h, l);
            hi[(long long)r * ldo + j] = h;
            lo[(long long)r * ldo + j] = l;
        }
    }
    for (int j = threadIdx.x + PREP_PER_THREAD * PREP_THREADS; j < ldo; j += PREP_THREADS) {
        __half h, l;
        split_f16(j < C ? w[j] * sc : 0.f, h, l);
        hi[(long long)r * ldo + j] = h;
        lo[(long long)r * ldo + j] = l;
    }
}

__global__ void __launch_bounds__(PREP_THREADS) k_prep_weights_f16(const float *__restrict__ W, int R, int C,
                                                                 __half *hi, __half *lo, int ldo, float *inv_scale,
                                                                 float *rowsum) {
    prep_row_f16(W, R, C, hi, lo, ldo, inv_scale, rowsum, blockIdx.x);
}

cudaError_t launch_prep_weights_f16(const float *W, int R, int C, __half *hi, __half *lo, int ldo, float *inv_scale,
                                    float *rowsum, cudaStream_t st) {
    k_prep_weights_f16<<<R, PREP_THREADS, 0, st>>>(W, R, C, hi, lo, ldo, inv_scale, rowsum);
    return cudaGetLastError();
}

// The forward operand in the bf16 modes: row r of W split into bf16 hi (and
// lo), padded with zeros to ldo columns, and the row's sum; one block per
// row, two adjacent columns per thread and step (one 4-byte store of a bf16
// pair per array), the sum reduced in a fixed order.
__global__ void __launch_bounds__(PREP_THREADS) k_split_rows_bf16(const float *__restrict__ W, int C,
                                                                  __nv_bfloat16 *hi, __nv_bfloat16 *lo, int ldo,
                                                                  float *rowsum) {
    __shared__ float red[PREP_THREADS / 32];
    const int r = blockIdx.x;
    const float *w = W + (long long)r * C;
    float sum = 0.f;
    for (int j = 2 * threadIdx.x; j < ldo; j += 2 * PREP_THREADS) {
        const float x0 = j < C ? w[j] : 0.f, x1 = j + 1 < C ? w[j + 1] : 0.f;
        sum += x0 + x1;
        __nv_bfloat16 h0, l0, h1, l1;
        split_bf16(x0, h0, l0);
        split_bf16(x1, h1, l1);
        const long long o = (long long)r * ldo + j;
        *reinterpret_cast<__nv_bfloat162 *>(hi + o) = __halves2bfloat162(h0, h1);
        if (lo) *reinterpret_cast<__nv_bfloat162 *>(lo + o) = __halves2bfloat162(l0, l1);
    }
    for (int j = ldo + threadIdx.x; j < C; j += PREP_THREADS) sum += w[j];  // columns past ldo (none in practice)
    if (!rowsum) return;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int k = 0; k < PREP_THREADS / 32; ++k) t += red[k];
        rowsum[r] = t;
    }
}

// Transposed copies only (W^T split into bf16 hi/lo, or W^T in fp32): one
// 64 x 64 tile per block, read row by row (two 128-byte rows per warp
// instruction pair), written as 64 output rows of 64 elements, two elements
// per lane (one 4-byte store of a bf16 pair), so that a warp writes 128
// contiguous bytes per instruction and array.
constexpr int SPLIT_T_TILE = 64;
__global__ void __launch_bounds__(256) k_split_T(const float *__restrict__ W, int R, int C,
                                                 __nv_bfloat16 *hiT, __nv_bfloat16 *loT, int ldt, float *f32T,
                                                 int ldf, int pairs) {
    __shared__ float tile[SPLIT_T_TILE][SPLIT_T_TILE + 1];
    const int c0 = blockIdx.x * SPLIT_T_TILE, r0 = blockIdx.y * SPLIT_T_TILE;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int k = 0; k < SPLIT_T_TILE / 8; ++k) {
        const int rr = w + 8 * k, r = r0 + rr;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int cc = c0 + lane + 32 * hh;
            tile[rr][lane + 32 * hh] = (r < R && cc < C) ? W[(long long)r * C + cc] : 0.0f;
        }
    }
    __syncthreads();
    const int r = r0 + 2 * lane;
#pragma unroll
    for (int k = 0; k < SPLIT_T_TILE / 8; ++k) {
        const int cl = w + 8 * k, cc = c0 + cl;
        if (cc >= C) break;
        const float x0 = tile[2 * lane][cl], x1 = tile[2 * lane + 1][cl];
        if (hiT && r < ldt) {
            __nv_bfloat16 h0, l0, h1, l1;
            split_bf16(x0, h0, l0);
            split_bf16(x1, h1, l1);
            const long long o = (long long)cc * ldt + r;
            if (pairs && r + 1 < ldt) {
                *reinterpret_cast<__nv_bfloat162 *>(hiT + o) = __halves2bfloat162(h0, h1);
                if (loT) *reinterpret_cast<__nv_bfloat162 *>(loT + o) = __halves2bfloat162(l0, l1);
            } else {
                hiT[o] = h0;
                if (loT) loT[o] = l0;
                if (r + 1 < ldt) {
                    hiT[o + 1] = h1;
                    if (loT) loT[o + 1] = l1;
                }
            }
        }
        if (f32T && r < ldf) {
            const long long o = (long long)cc * ldf + r;
            f32T[o] = x0;
            if (r + 1 < ldf) f32T[o + 1] = x1;
        }
    }
}

cudaError_t launch_prep_weights(const float *W, int R, int C, OpKind op, __nv_bfloat16 *hi, __nv_bfloat16 *lo,
                                int ldo, __nv_bfloat16 *hiT, __nv_bfloat16 *loT, int ldt, float *f32T, int ldf,
                                float *rowsum, cudaStream_t st) {
    if (hi && !hiT && !f32T && ldo >= C && ldo % 2 == 0 && ((uintptr_t)hi % 4 == 0) && (!lo || (uintptr_t)lo % 4 == 0)) {
        k_split_rows_bf16<<<R, PREP_THREADS, 0, st>>>(W, C, hi, lo, ldo, rowsum);
        return cudaGetLastError();
    }
    if (!hi && !rowsum && (hiT || f32T)) {
        int rr = R;  // output columns to write, padding included
        if (hiT && ldt > rr) rr = ldt;
        if (f32T && ldf > rr) rr = ldf;
        // bf16 pair stores need every output row to start on a 4-byte boundary
        const int pairs = hiT && (ldt % 2 == 0) && ((uintptr_t)hiT % 4 == 0) && (!loT || (uintptr_t)loT % 4 == 0);
        dim3 grid((unsigned)((C + SPLIT_T_TILE - 1) / SPLIT_T_TILE), (unsigned)((rr + SPLIT_T_TILE - 1) / SPLIT_T_TILE));
        k_split_T<<<grid, 256, 0, st>>>(W, R, C, hiT, loT, ldt, f32T, ldf, pairs);
        return cudaGetLastError();
    }
    if (rowsum) {
        cudaError_t e = cudaMemsetAsync(rowsum, 0, sizeof(float) * R, st);
        if (e != cudaSuccess) return e;
    }
    int cmax = C > ldo ? C : ldo;
    int rmax = R > ldt ? R : ldt;
    if (ldf > rmax) rmax = ldf;
    dim3 grid((cmax + 31) / 32, (rmax + 31) / 32);
    k_prep_weights<<<grid, dim3(32, 8), 0, st>>>(W, R, C, (int)op, hi, lo, ldo, hiT, loT, ldt, f32T, ldf, rowsum);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Binning (Eq. DSTD_kernel): one thread per (sample, pair of inputs) writes
// the Mp rows of its two columns; rows m >= M and padding columns are zero.
// ---------------------------------------------------------------------------
template <int OP>
__global__ void k_binning_rows(const float *__restrict__ t, int B, int N, LifConst c, void *hi, void *lo,
                               int ld) {
    const int b = blockIdx.y;
    const int j0 = 2 * (blockIdx.x * blockDim.x + threadIdx.x);
    if (j0 >= ld) return;
    BinW w0{-100, 0.f, 0.f, 0.f, 0.f}, w1{-100, 0.f, 0.f, 0.f, 0.f};
    if (j0 < N) {
        float x = t[(long long)b * N + j0];
        if (isfinite(x)) w0 = bin_weights(c, x, false);
    }
    if (j0 + 1 < N) {
        float x = t[(long long)b * N + j0 + 1];
        if (isfinite(x)) w1 = bin_weights(c, x, false);
    }
    for (int m = 0; m < c.Mp; ++m) {
        float v0 = 0.f, v1 = 0.f;
        if (m < c.M) {
            v0 = (m == w0.k) ? w0.wR : ((m == w0.k + 1) ? w0.wL : 0.f);
            v1 = (m == w1.k) ? w1.wR : ((m == w1.k + 1) ? w1.wL : 0.f);
        }
        long long off = ((long long)b * c.Mp + m) * ld + j0;
        if (OP == 0) {
            *reinterpret_cast<float2 *>((float *)hi + off) = make_float2(v0, v1);
        } else if (OP == 3) {
            __half h0, l0, h1, l1;
            split_f16(v0, h0, l0);
            split_f16(v1, h1, l1);
            *reinterpret_cast<__half2 *>((__half *)hi + off) = __halves2half2(h0, h1);
            *reinterpret_cast<__half2 *>((__half *)lo + off) = __halves2half2(l0, l1);
        } else {
            __nv_bfloat16 h0, l0, h1, l1;
            split_bf16(v0, h0, l0);
            split_bf16(v1, h1, l1);
            *reinterpret_cast<__nv_bfloat162 *>((__nv_bfloat16 *)hi + off) = __halves2bfloat162(h0, h1);
            if (OP == 1) *reinterpret_cast<__nv_bfloat162 *>((__nv_bfloat16 *)lo + off) = __halves2bfloat162(l0, l1);
        }
    }
}

// transposed: row j, columns (b, m). A warp takes 32 consecutive samples of
// one input j: each lane evaluates the grid weights of its own sample, then
// the warp writes the 32 samples' Mp bins as consecutive 16-byte chunks
// (lane l writes chunk l of each round, taking the weights of the chunk's
// sample by shuffle), so every store instruction fills whole sectors. With
// bw != null each lane also writes (k, ds/dt at T_k, ds/dt at T_{k+1}) of
// its sample to bw[b*N + j] (k = -100 for a silent input) for the input-time
// gradient.
template <int OP>
__global__ void k_binning_cols(const float *__restrict__ t, int B, int N, LifConst c, void *hi, void *lo, int ld,
                               float4 *bw) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int b0 = (blockIdx.x * (blockDim.x >> 5) + warp) * 32;
    if (b0 >= B) return;
    const int cps = c.Mp / 8;  // 8-bin chunks per sample
    for (int j = blockIdx.y; j < N; j += gridDim.y) {
        const int b = b0 + lane;
        BinW w{-100, 0.f, 0.f, 0.f, 0.f};
        if (b < B) {
            const float x = t[(long long)b * N + j];
            if (isfinite(x)) w = bin_weights(c, x, bw != nullptr);
            if (bw) bw[(long long)b * N + j] = make_float4(__int_as_float(w.k), w.dR, w.dL, 0.f);
        }
        const long long rowbase = (long long)j * ld + (long long)b0 * c.Mp;
        for (int r = 0; r < cps; ++r) {
            const int gc = r * 32 + lane;  // chunk of the warp's 32 samples
            const int sl = gc / cps, ch = gc - sl * cps;
            const int kk = __shfl_sync(0xffffffffu, w.k, sl);
            const float wR = __shfl_sync(0xffffffffu, w.wR, sl);
            const float wL = __shfl_sync(0xffffffffu, w.wL, sl);
            if (b0 + sl >= B) continue;
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int m = ch * 8 + u;
                v[u] = (m < c.M) ? ((m == kk) ? wR : ((m == kk + 1) ? wL : 0.f)) : 0.f;
            }
            const long long off = rowbase + (long long)gc * 8;
            if (OP == 0) {
                float4 *p = reinterpret_cast<float4 *>((float *)hi + off);
                p[0] = make_float4(v[0], v[1], v[2], v[3]);
                p[1] = make_float4(v[4], v[5], v[6], v[7]);
            } else {
                __align__(16) __nv_bfloat16 h[8], l[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) split_bf16(v[u], h[u], l[u]);
                *reinterpret_cast<uint4 *>((__nv_bfloat16 *)hi + off) = *reinterpret_cast<uint4 *>(h);
                if (OP == 1) *reinterpret_cast<uint4 *>((__nv_bfloat16 *)lo + off) = *reinterpret_cast<uint4 *>(l);
            }
        }
    }
}

// 16-bit operands, written sparse: of the Mp bins of an input only two are
// nonzero, so the operand is first zero-filled with 16-byte stores and the
// two weights (hi and lo parts) are then stored element-wise by the same
// thread (program order makes the later store win). OP 1: bf16 hi + lo,
// 2: bf16, 3: fp16 hi + lo.
template <int OP>
__device__ __forceinline__ void split16(float x, uint16_t &h, uint16_t &l) {
    if (OP == 3) {
        __half hh, ll;
        split_f16(x, hh, ll);
        h = __half_as_ushort(hh);
        l = __half_as_ushort(ll);
    } else {
        __nv_bfloat16 hh, ll;
        split_bf16(x, hh, ll);
        h = __bfloat16_as_ushort(hh);
        l = __bfloat16_as_ushort(ll);
    }
}

// rows (b, m), columns j: a block of ROWS8_THREADS takes one sample and as
// many consecutive columns; it zero-fills that Mp x columns patch with
// 16-byte stores, synchronises (which orders the block's global stores), and
// then each thread stores the two weights of its own column (rows m >= M and
// columns >= N stay zero).
constexpr int ROWS8_THREADS = 128;
template <int OP, int NT>
__device__ __forceinline__ void binning_rows8_block(const float *__restrict__ t, int N, const LifConst &c, uint16_t *hi,
                                                    uint16_t *lo, int ld, int b, int col0) {
    const int nch = ((ld - col0) < NT ? (ld - col0) : NT) / 8;  // 16-byte chunks per row
    const long long base = (long long)b * c.Mp * ld + col0;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (int idx = threadIdx.x; idx < c.Mp * nch; idx += NT) {
        const int m = idx / nch, cc = idx - m * nch;
        const long long o = base + (long long)m * ld + 8 * cc;
        *reinterpret_cast<uint4 *>(hi + o) = z;
        if (OP != 2) *reinterpret_cast<uint4 *>(lo + o) = z;
    }
    __syncthreads();
    const int j = col0 + threadIdx.x;
    if (j >= N) return;
    const float x = t[(long long)b * N + j];
    if (!isfinite(x)) return;
    const BinW w = bin_weights(c, x, false);
    uint16_t h, l;
    if (w.k >= 0 && w.k < c.M) {
        split16<OP>(w.wR, h, l);
        const long long o = base + (long long)w.k * ld + threadIdx.x;
        hi[o] = h;
        if (OP != 2) lo[o] = l;
    }
    if (w.k + 1 >= 0 && w.k + 1 < c.M) {
        split16<OP>(w.wL, h, l);
        const long long o = base + (long long)(w.k + 1) * ld + threadIdx.x;
        hi[o] = h;
        if (OP != 2) lo[o] = l;
    }
}

template <int OP>
__global__ void __launch_bounds__(ROWS8_THREADS) k_binning_rows8(const float *__restrict__ t, int B, int N,
                                                                 LifConst c, uint16_t *hi, uint16_t *lo, int ld) {
    binning_rows8_block<OP, ROWS8_THREADS>(t, N, c, hi, lo, ld, blockIdx.y, blockIdx.x * ROWS8_THREADS);
}

// The two operands of the x3 forward contraction in one launch (they do not
// depend on each other): blocks [0, nbin) bin the spike times (sample
// blockIdx / nbx, columns of chunk blockIdx % nbx), the rest split weight
// rows into fp16 hi + lo.
__global__ void __launch_bounds__(PREP_THREADS) k_fwd_operands_f16(const float *__restrict__ t, int N, LifConst c,
                                                                 uint16_t *s_hi, uint16_t *s_lo, int ld, int nbx,
                                                                 int nbin, const float *__restrict__ W, int R,
                                                                 __half *w_hi, __half *w_lo, float *inv_scale,
                                                                 float *rowsum) {
    if ((int)blockIdx.x < nbin) {
        const int b = blockIdx.x / nbx, cb = blockIdx.x - b * nbx;
        binning_rows8_block<3, PREP_THREADS>(t, N, c, s_hi, s_lo, ld, b, cb * PREP_THREADS);
    } else {
        prep_row_f16(W, R, N, w_hi, w_lo, ld, inv_scale, rowsum, blockIdx.x - nbin);
    }
}

cudaError_t launch_fwd_operands_f16(const float *t, int B, int N, const LifConst &c, void *s_hi, void *s_lo, int ld,
                                    const float *W, int R, __half *w_hi, __half *w_lo, float *inv_scale,
                                    float *rowsum, cudaStream_t st) {
    if ((ld % 8) != 0 || ((reinterpret_cast<uintptr_t>(s_hi) | reinterpret_cast<uintptr_t>(s_lo)) & 15) != 0)
        return cudaErrorInvalidValue;
    const int nbx = (ld + PREP_THREADS - 1) / PREP_THREADS;
    const long long nbin = (long long)nbx * B;
    if (nbin + R > 0x7fffffffLL) return cudaErrorInvalidValue;
    k_fwd_operands_f16<<<(unsigned)(nbin + R), PREP_THREADS, 0, st>>>(
        t, N, c, static_cast<uint16_t *>(s_hi), static_cast<uint16_t *>(s_lo), ld, nbx, (int)nbin, W, R, w_hi, w_lo,
        inv_scale, rowsum);
    return cudaGetLastError();
}

// row j, columns (b, m), for a tile of 32 inputs x 32 samples per block (4
// warps): first the tile's spike times are read along j (coalesced), binned,
// and with bw != null the per-input records (k, ds/dt at T_k, at T_{k+1}; k =
// -100 for a silent input) written along j to bw[b*N + j]; the bin and the
// two weights (hi and lo halves packed in pairs) go to shared memory. Then
// each warp writes 8 of the tile's rows: the 32 samples' Mp bins of row j are
// consecutive, and lane g of a round builds 16-byte chunk g of them from the
// bin and weights of its sample (at most two nonzero halves), so a store
// instruction covers 512 contiguous bytes.
template <int OP>
__global__ void __launch_bounds__(128) k_binning_cols8(const float *__restrict__ t, int B, int N, LifConst c,
                                                       uint16_t *hi, uint16_t *lo, int ld, float4 *bw) {
    __shared__ int sk[32][33];
    __shared__ uint32_t swh[32][33], swl[32][33];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j0 = blockIdx.x * 32, b0 = blockIdx.y * 32;
    const int j = j0 + lane;
    for (int bb = warp; bb < 32; bb += 4) {
        const int b = b0 + bb;
        BinW w{-100, 0.f, 0.f, 0.f, 0.f};
        if (b < B && j < N) {
            const float x = __ldg(t + (long long)b * N + j);
            if (isfinite(x)) w = bin_weights(c, x, bw != nullptr);
            if (bw) bw[(long long)b * N + j] = make_float4(__int_as_float(w.k), w.dR, w.dL, 0.f);
        }
        uint16_t hR = 0, lR = 0, hL = 0, lL = 0;
        if (w.k >= 0 && w.k < c.M) split16<OP>(w.wR, hR, lR);
        if (w.k + 1 >= 0 && w.k + 1 < c.M) split16<OP>(w.wL, hL, lL);
        sk[lane][bb] = w.k;
        swh[lane][bb] = (uint32_t)hR | ((uint32_t)hL << 16);
        swl[lane][bb] = (uint32_t)lR | ((uint32_t)lL << 16);
    }
    __syncthreads();
    const int ns = (B - b0) < 32 ? (B - b0) : 32;
    const int cps = c.Mp >> 3;  // 16-byte chunks per sample
    const int nch = ns * cps;
    for (int jj = warp; jj < 32; jj += 4) {
        const int jr = j0 + jj;
        if (jr >= N) break;
        const long long rowbase = (long long)jr * ld + (long long)b0 * c.Mp;
        for (int g = lane; g < nch; g += 32) {
            const int bb = g / cps, q = g - bb * cps;
            const int k = sk[jj][bb];
            // the sample's weight at T_k sits at half e1 of the chunk, at T_{k+1} at e1 + 1
            const int e1 = k - 8 * q;
            const uint32_t ph = swh[jj][bb], pl = swl[jj][bb];
            uint32_t h[4] = {0u, 0u, 0u, 0u}, l[4] = {0u, 0u, 0u, 0u};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                // halves 2i and 2i + 1 of the chunk
                if (e1 == 2 * i) {
                    h[i] = ph;
                    l[i] = pl;
                } else if (e1 == 2 * i - 1) {
                    h[i] = ph >> 16;
                    l[i] = pl >> 16;
                } else if (e1 == 2 * i + 1) {
                    h[i] = ph << 16;
                    l[i] = pl << 16;
                }
            }
            *reinterpret_cast<uint4 *>(hi + rowbase + 8 * g) = make_uint4(h[0], h[1], h[2], h[3]);
            if (OP != 2) *reinterpret_cast<uint4 *>(lo + rowbase + 8 * g) = make_uint4(l[0], l[1], l[2], l[3]);
        }
    }
}

cudaError_t launch_binning(const float *t, int B, int N, const LifConst &c, OpKind op, bool transposed, void *hi,
                           void *lo, int ld, cudaStream_t st, float4 *bw) {
    uint16_t *h16 = static_cast<uint16_t *>(hi), *l16 = static_cast<uint16_t *>(lo);
    // the sparse writers need 16-byte aligned rows of 8-element multiples
    const bool sparse = op != OpKind::F32 && (ld % 8) == 0 && ((reinterpret_cast<uintptr_t>(hi) |
                                                                 reinterpret_cast<uintptr_t>(lo)) & 15) == 0;
    if (!transposed) {
        if (sparse) {
            dim3 grid(blocks_for(ld, ROWS8_THREADS), B);
            if (op == OpKind::BF16X3) k_binning_rows8<1><<<grid, ROWS8_THREADS, 0, st>>>(t, B, N, c, h16, l16, ld);
            else if (op == OpKind::F16X3) k_binning_rows8<3><<<grid, ROWS8_THREADS, 0, st>>>(t, B, N, c, h16, l16, ld);
            else k_binning_rows8<2><<<grid, ROWS8_THREADS, 0, st>>>(t, B, N, c, h16, l16, ld);
            return cudaGetLastError();
        }
        int pairs = (ld + 1) / 2;
        dim3 grid(blocks_for(pairs, 128), B);
        if (op == OpKind::F32) k_binning_rows<0><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld);
        else if (op == OpKind::BF16X3) k_binning_rows<1><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld);
        else if (op == OpKind::F16X3) k_binning_rows<3><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld);
        else k_binning_rows<2><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld);
    } else {
        if (sparse && op != OpKind::F16X3) {
            if ((N + 31) / 32 > 0x7fffffff || (B + 31) / 32 > 65535) return cudaErrorInvalidValue;
            dim3 g8((unsigned)((N + 31) / 32), (unsigned)((B + 31) / 32));
            if (op == OpKind::BF16X3) k_binning_cols8<1><<<g8, 128, 0, st>>>(t, B, N, c, h16, l16, ld, bw);
            else k_binning_cols8<2><<<g8, 128, 0, st>>>(t, B, N, c, h16, l16, ld, bw);
            return cudaGetLastError();
        }
        dim3 grid(blocks_for(B, 128), N < 65535 ? N : 65535);
        if (op == OpKind::F32) k_binning_cols<0><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld, bw);
        else if (op == OpKind::BF16X3) k_binning_cols<1><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld, bw);
        else k_binning_cols<2><<<grid, 128, 0, st>>>(t, B, N, c, hi, lo, ld, bw);
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// im2col binning for convolutions: the grid weights of the input spike that
// filter tap kidx = (kh*k + kw)*C + c reads at output position pos
// (out-of-image taps read a silent input, i.e. zero weights).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float im2col_time(const float *__restrict__ t, const ConvGeom &g, int pos, int kidx) {
    const int c = kidx % g.C;
    const int kw = (kidx / g.C) % g.k;
    const int kh = kidx / (g.C * g.k);
    const int x = pos % g.Wo;
    const int y = (pos / g.Wo) % g.Ho;
    const int b = pos / (g.Wo * g.Ho);
    const int iy = y * g.s + kh - g.p, ix = x * g.s + kw - g.p;
    if (iy < 0 || iy >= g.H || ix < 0 || ix >= g.W) return INFINITY;
    return t[(((long long)b * g.H + iy) * g.W + ix) * g.C + c];
}

template <int OP>
__global__ void k_binning_im2col_rows(const float *__restrict__ t, ConvGeom g, int pos0, int npos, LifConst c,
                                      void *hi, void *lo, int ld) {
    const int K = g.k * g.k * g.C;
    const int j0 = 2 * (blockIdx.x * blockDim.x + threadIdx.x);
    if (j0 >= ld) return;
    for (int pl = blockIdx.y; pl < npos; pl += gridDim.y) {
        BinW w0{-100, 0.f, 0.f, 0.f, 0.f}, w1{-100, 0.f, 0.f, 0.f, 0.f};
        if (j0 < K) {
            float x = im2col_time(t, g, pos0 + pl, j0);
            if (isfinite(x)) w0 = bin_weights(c, x, false);
        }
        if (j0 + 1 < K) {
            float x = im2col_time(t, g, pos0 + pl, j0 + 1);
            if (isfinite(x)) w1 = bin_weights(c, x, false);
        }
        for (int m = 0; m < c.Mp; ++m) {
            float v0 = 0.f, v1 = 0.f;
            if (m < c.M) {
                v0 = (m == w0.k) ? w0.wR : ((m == w0.k + 1) ? w0.wL : 0.f);
                v1 = (m == w1.k) ? w1.wR : ((m == w1.k + 1) ? w1.wL : 0.f);
            }
            long long off = ((long long)pl * c.Mp + m) * ld + j0;
            if (OP == 3) {
                __half h0, l0, h1, l1;
                split_f16(v0, h0, l0);
                split_f16(v1, h1, l1);
                *reinterpret_cast<__half2 *>((__half *)hi + off) = __halves2half2(h0, h1);
                *reinterpret_cast<__half2 *>((__half *)lo + off) = __halves2half2(l0, l1);
            } else {
                __nv_bfloat16 h0, l0, h1, l1;
                split_bf16(v0, h0, l0);
                split_bf16(v1, h1, l1);
                *reinterpret_cast<__nv_bfloat162 *>((__nv_bfloat16 *)hi + off) = __halves2bfloat162(h0, h1);
                if (OP == 1)
                    *reinterpret_cast<__nv_bfloat162 *>((__nv_bfloat16 *)lo + off) = __halves2bfloat162(l0, l1);
            }
        }
    }
}

template <int OP>
__global__ void k_binning_im2col_cols(const float *__restrict__ t, ConvGeom g, int pos0, int npos, LifConst c,
                                      void *hi, void *lo, int ld) {
    const int K = g.k * g.k * g.C;
    const int pl = blockIdx.x * blockDim.x + threadIdx.x;
    if (pl >= npos) return;
    for (int kidx = blockIdx.y; kidx < K; kidx += gridDim.y) {
        BinW w{-100, 0.f, 0.f, 0.f, 0.f};
        float x = im2col_time(t, g, pos0 + pl, kidx);
        if (isfinite(x)) w = bin_weights(c, x, false);
        const long long base = (long long)kidx * ld + (long long)pl * c.Mp;
        for (int m0 = 0; m0 < c.Mp; m0 += 8) {
            __align__(16) __nv_bfloat16 h[8], l[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                int m = m0 + u;
                float v = (m < c.M) ? ((m == w.k) ? w.wR : ((m == w.k + 1) ? w.wL : 0.f)) : 0.f;
                split_bf16(v, h[u], l[u]);
            }
            *reinterpret_cast<uint4 *>((__nv_bfloat16 *)hi + base + m0) = *reinterpret_cast<uint4 *>(h);
            if (OP == 1) *reinterpret_cast<uint4 *>((__nv_bfloat16 *)lo + base + m0) = *reinterpret_cast<uint4 *>(l);
        }
    }
}

// Sparse writers of the im2col operands (as the dense ones): a block zero-
// fills the Mp rows of one output position over 256 tap columns, or a warp
// the Mp bins of 32 consecutive positions of one tap, with 16-byte stores,
// synchronises, and each thread then stores the two weights of its own
// (position, tap).
template <int OP>
__global__ void __launch_bounds__(256) k_binning_im2col_rows8(const float *__restrict__ t, ConvGeom g, int pos0,
                                                              int npos, LifConst c, uint16_t *hi, uint16_t *lo,
                                                              int ld) {
    const int K = g.k * g.k * g.C;
    const int col0 = blockIdx.x * 256;
    const int nch = ((ld - col0) < 256 ? (ld - col0) : 256) / 8;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (int pl = blockIdx.y; pl < npos; pl += gridDim.y) {
        const long long base = (long long)pl * c.Mp * ld + col0;
        for (int idx = threadIdx.x; idx < c.Mp * nch; idx += 256) {
            const int m = idx / nch, cc = idx - m * nch;
            const long long o = base + (long long)m * ld + 8 * cc;
            *reinterpret_cast<uint4 *>(hi + o) = z;
            if (OP != 2) *reinterpret_cast<uint4 *>(lo + o) = z;
        }
        __syncthreads();
        const int kidx = col0 + threadIdx.x;
        if (kidx < K) {
            const float x = im2col_time(t, g, pos0 + pl, kidx);
            if (isfinite(x)) {
                const BinW w = bin_weights(c, x, false);
                uint16_t h, l;
                if (w.k >= 0 && w.k < c.M) {
                    split16<OP>(w.wR, h, l);
                    const long long o = base + (long long)w.k * ld + threadIdx.x;
                    hi[o] = h;
                    if (OP != 2) lo[o] = l;
                }
                if (w.k + 1 >= 0 && w.k + 1 < c.M) {
                    split16<OP>(w.wL, h, l);
                    const long long o = base + (long long)(w.k + 1) * ld + threadIdx.x;
                    hi[o] = h;
                    if (OP != 2) lo[o] = l;
                }
            }
        }
        __syncthreads();  // the next position's zero fill may touch no column before this one's weights are out
    }
}

template <int OP>
__global__ void __launch_bounds__(128) k_binning_im2col_cols8(const float *__restrict__ t, ConvGeom g, int pos0,
                                                              int npos, LifConst c, uint16_t *hi, uint16_t *lo,
                                                              int ld) {
    const int K = g.k * g.k * g.C;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int p0 = (blockIdx.x * 4 + warp) * 32;
    if (p0 >= npos) return;
    const int ns = (npos - p0) < 32 ? (npos - p0) : 32;
    const int nch = ns * c.Mp / 8;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (int kidx = blockIdx.y; kidx < K; kidx += gridDim.y) {
        const long long rowbase = (long long)kidx * ld + (long long)p0 * c.Mp;
        for (int gq = lane; gq < nch; gq += 32) {
            *reinterpret_cast<uint4 *>(hi + rowbase + 8 * gq) = z;
            if (OP != 2) *reinterpret_cast<uint4 *>(lo + rowbase + 8 * gq) = z;
        }
        __syncwarp();
        if (lane < ns) {
            const float x = im2col_time(t, g, pos0 + p0 + lane, kidx);
            if (isfinite(x)) {
                const BinW w = bin_weights(c, x, false);
                const long long o = rowbase + (long long)lane * c.Mp;
                uint16_t h, l;
                if (w.k >= 0 && w.k < c.M) {
                    split16<OP>(w.wR, h, l);
                    hi[o + w.k] = h;
                    if (OP != 2) lo[o + w.k] = l;
                }
                if (w.k + 1 >= 0 && w.k + 1 < c.M) {
                    split16<OP>(w.wL, h, l);
                    hi[o + w.k + 1] = h;
                    if (OP != 2) lo[o + w.k + 1] = l;
                }
            }
        }
        __syncwarp();
    }
}

cudaError_t launch_binning_im2col(const float *t, const ConvGeom &g, int pos0, int npos, const LifConst &c,
                                  OpKind op, bool transposed, void *hi, void *lo, int ld, cudaStream_t st) {
    const int K = g.k * g.k * g.C;
    uint16_t *h16 = static_cast<uint16_t *>(hi), *l16 = static_cast<uint16_t *>(lo);
    const bool sparse = (ld % 8) == 0 && ((reinterpret_cast<uintptr_t>(hi) | reinterpret_cast<uintptr_t>(lo)) & 15) == 0;
    if (sparse && !transposed) {
        dim3 grid((ld + 255) / 256, npos < 65535 ? npos : 65535);
        if (op == OpKind::F16X3) k_binning_im2col_rows8<3><<<grid, 256, 0, st>>>(t, g, pos0, npos, c, h16, l16, ld);
        else if (op == OpKind::BF16X3) k_binning_im2col_rows8<1><<<grid, 256, 0, st>>>(t, g, pos0, npos, c, h16, l16, ld);
        else if (op == OpKind::BF16) k_binning_im2col_rows8<2><<<grid, 256, 0, st>>>(t, g, pos0, npos, c, h16, l16, ld);
        else return cudaErrorInvalidValue;
        return cudaGetLastError();
    }
    if (sparse && transposed && (op == OpKind::BF16X3 || op == OpKind::BF16)) {
        dim3 grid((npos + 127) / 128, K < 65535 ? K : 65535);
        if (op == OpKind::BF16X3) k_binning_im2col_cols8<1><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, h16, l16, ld);
        else k_binning_im2col_cols8<2><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, h16, l16, ld);
        return cudaGetLastError();
    }
    if (!transposed) {
        dim3 grid(blocks_for((ld + 1) / 2, 128), npos < 65535 ? npos : 65535);
        if (op == OpKind::F16X3) k_binning_im2col_rows<3><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, hi, lo, ld);
        else if (op == OpKind::BF16X3) k_binning_im2col_rows<1><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, hi, lo, ld);
        else if (op == OpKind::BF16) k_binning_im2col_rows<2><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, hi, lo, ld);
        else return cudaErrorInvalidValue;
    } else {
        dim3 grid(blocks_for(npos, 128), K < 65535 ? K : 65535);
        if (op == OpKind::BF16X3) k_binning_im2col_cols<1><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, hi, lo, ld);
        else if (op == OpKind::BF16) k_binning_im2col_cols<2><<<grid, 128, 0, st>>>(t, g, pos0, npos, c, hi, lo, ld);
        else return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

__global__ void k_binning_public(const float *__restrict__ t, int B, int N, LifConst c, float *s, float *ds) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N) return;
    int b = (int)(idx / N), j = (int)(idx % N);
    BinW w{-100, 0.f, 0.f, 0.f, 0.f};
    float x = t[idx];
    if (isfinite(x)) w = bin_weights(c, x, ds != nullptr);
    for (int m = 0; m < c.M; ++m) {
        long long o = ((long long)b * c.M + m) * N + j;
        s[o] = (m == w.k) ? w.wR : ((m == w.k + 1) ? w.wL : 0.f);
        if (ds) ds[o] = (m == w.k) ? w.dR : ((m == w.k + 1) ? w.dL : 0.f);
    }
}

cudaError_t launch_binning_public(const float *t, int B, int N, const LifConst &c, float *s, float *ds,
                                  cudaStream_t st) {
    long long n = (long long)B * N;
    k_binning_public<<<blocks_for(n, 256), 256, 0, st>>>(t, B, N, c, s, ds);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Scan/solve/select from a materialised w^ (one thread per neuron), with the
// temporal penalty and dead-neuron sums (warp-reduced, one atomic per warp).
// ---------------------------------------------------------------------------
// Block-wide sums of the four penalty terms, one atomic per term per block
// (blockDim.x a multiple of 32, at most 1024; every thread of the block calls).
__device__ __forceinline__ void flush_penalty(float acc[4], float *penalty) {
    __shared__ float part[32][4];
    if (!penalty) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float v = warp_sum(acc[k]);
        if (lane == 0) part[warp][k] = v;
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            float v = lane < nw ? part[lane][k] : 0.0f;
            v = warp_sum(v);
            if (lane == 0 && v != 0.0f) atomicAdd(&penalty[k], v);
        }
    }
}

// One thread per neuron (b, i); element (b, i, m) of w^ at
// what[b*sb + i*si + m*sm], times scale[i] when given. SUB bins at a time
// are loaded together (16-byte loads when sm = 1 and rows are 16-byte
// aligned) into the thread's own row of shared memory (stride SUB + 4
// floats: 16-byte accesses of 8 consecutive lanes hit distinct banks).
// Each block of SUB bins takes two passes:
//   fast  all SUB bins, four per 16-byte read, branch-free: the recurrence,
//         and bit u of a mask for "v^ may reach v_th in bin u" (end point at
//         v_th, or an interior maximum that the cheap bound does not
//         exclude); the state at every eighth bin is kept in registers;
//   exact the flagged bins in order: from the nearest kept state, walk to
//         the bin and test it exactly (interior_test out of line). The first
//         bin that passes holds the spike.
// A lane whose candidate fails goes straight to its next flagged bin, so no
// lane walks a block twice.
constexpr int SCAN_THREADS = 256;

template <int SUB, bool VEC, bool WIDE>
__global__ void __launch_bounds__(SCAN_THREADS, 4) k_scan_solve(const float *__restrict__ what, long long sb,
                                                                long long si, long long sm, int B, int N, LifConst c,
                                                                const float *__restrict__ scale,
                                                                const float *__restrict__ rowsum, float *t_out,
                                                                int *q, float *s, float *vdot, float *penalty) {
    constexpr int LD = SUB + 4;
    __shared__ __align__(16) float sw[SCAN_THREADS * LD];
    float *row = sw + threadIdx.x * LD;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    const long long n = (long long)B * N;
    for (long long idx = (long long)blockIdx.x * SCAN_THREADS + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * SCAN_THREADS) {
        int b, i;
        if (WIDE) {
            b = (int)(idx / N);
            i = (int)(idx % N);
        } else {
            b = (int)((unsigned)idx / (unsigned)N);
            i = (int)((unsigned)idx - (unsigned)b * (unsigned)N);
        }
        const float *w = what + b * sb + i * si;
        const float sc = scale ? scale[i] : 1.0f;
        ScanState st;
        scan_reset(st, c.M);
        float v = 0.f, I = 0.f;
        for (int m0 = 0; m0 < c.M && st.q == c.M; m0 += SUB) {
            const int mend = (c.M - m0) < SUB ? (c.M - m0) : SUB;
            if (VEC && mend == SUB) {
#pragma unroll
                for (int j = 0; j < SUB; j += 4) {
                    const float4 u = __ldg(reinterpret_cast<const float4 *>(w + m0 + j));
                    *reinterpret_cast<float4 *>(row + j) = make_float4(u.x * sc, u.y * sc, u.z * sc, u.w * sc);
                }
            } else {
#pragma unroll
                for (int j = 0; j < SUB; ++j) row[j] = (j < mend) ? __ldg(w + (m0 + j) * sm) * sc : 0.0f;
            }
            if (scan_walk<SUB>(c, row, m0, mend, v, I, st)) break;
        }
        scan_finish(c, st);
        finish_neuron(c, st, b, i, N, rowsum, t_out, q, s, vdot, acc);
    }
    flush_penalty(acc, penalty);
}

cudaError_t launch_scan_solve(const float *what, long long sb, long long si, long long sm, int B, int N,
                              const LifConst &c, const float *scale, const float *rowsum, float *t_out, int *q,
                              float *s, float *vdot, float *penalty, cudaStream_t st) {
    long long n = (long long)B * N;
    const unsigned g = grid_cap(n, SCAN_THREADS);
    const bool vec = sm == 1 && (si % 4) == 0 && (sb % 4) == 0 && (reinterpret_cast<uintptr_t>(what) % 16) == 0;
    const bool wide = n >= (1ll << 31);
#define DSTD_SCAN_L(SUB, V, W) \
    k_scan_solve<SUB, V, W><<<g, SCAN_THREADS, 0, st>>>(what, sb, si, sm, B, N, c, scale, rowsum, t_out, q, s, vdot, penalty)
#define DSTD_SCAN(SUB)                          \
    if (wide) DSTD_SCAN_L(SUB, false, true);    \
    else if (vec) DSTD_SCAN_L(SUB, true, false); \
    else DSTD_SCAN_L(SUB, false, false);
    if (c.M <= 8) {
        DSTD_SCAN(8)
    } else if (c.M <= 16) {
        DSTD_SCAN(16)
    } else {
        DSTD_SCAN(32)
    }
#undef DSTD_SCAN
#undef DSTD_SCAN_L
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Layers with few outputs (N_out <= kNarrowMaxOut) on CUDA cores, in fp32.
// A 128-row tensor-core tile would be mostly padding here, and each input
// spike touches only two grid points, so the contraction is done sparse.
// ---------------------------------------------------------------------------
constexpr int NARROW_FWD_THREADS = 512, NARROW_BWD_THREADS = 1024;

// Forward, one block per sample b: w^_im = sum_j W_ij s_jm (Eq. DSTD) from
// the two grid weights of each input spike (wR at T_k, wL at T_{k+1}), then
// the scan/solve/select of the sample's N_out neurons (one thread each) and
// the penalty sums. The inputs are first put in a stable order by grid step
// (a counting sort whose within-step order is the input order, so the sums
// below have a fixed order and the forward is bitwise reproducible): warp w
// ranks its own contiguous slice of inputs by key k + 1 in [0, M] (M + 1 = no
// grid weight) with __match_any_sync, the per-warp counts give every (warp,
// key) its offset, and a second pass places (j, wR, wL). Then one warp per
// grid point m sums, for every output at once (registers), the inputs of
// step m - 1 (their wL) and of step m (their wR): the lanes stride over
// those inputs, reading W_.j as one row of the transposed copy of W in
// shared memory, and a fixed butterfly of shuffles adds the lanes.
template <int SUB, int NOUT>
__global__ void __launch_bounds__(NARROW_FWD_THREADS) k_narrow_fwd(const float *__restrict__ t,
                                                                 const float *__restrict__ W, int N_in, int N_out,
                                                                 LifConst c, float *t_out, int *q, float *s,
                                                                 float *vdot, float *penalty, NarrowCe ce) {
    constexpr int NW = NARROW_FWD_THREADS / 32;
    extern __shared__ __align__(16) unsigned char nsm[];
    const int NK = c.M + 2;  // keys 0 .. M, and M + 1 for "no weight"
    // w^ first: its rows (Mp floats, Mp a power of two >= 8) stay 32-byte
    // aligned for the scan's 16-byte reads, and so does W^T after it
    float *acc = reinterpret_cast<float *>(nsm);        // [N_out][Mp]
    float *ws = acc + N_out * c.Mp;                      // [N_out][N_in]: W
    float *rsum = ws + (size_t)N_in * N_out;             // [N_out]
    int *hist = reinterpret_cast<int *>(rsum + N_out);   // [NW][NK]: counts, then offsets
    int *start = hist + NW * NK;                         // [NK + 1]
    int *upos = start + NK + 1;                          // [N_in]: rank within (warp, key)
    int *sj = upos + N_in;                               // [N_in]: inputs sorted by key
    float2 *sw = reinterpret_cast<float2 *>((reinterpret_cast<uintptr_t>(sj + N_in) + 7) & ~uintptr_t(7));  // (wR, wL)
    const int b = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float *tb = t + (long long)b * N_in;
    auto key_of = [&](float x) {
        if (!isfinite(x)) return c.M + 1;
        const int k = bin_index(c, x);
        return (k >= -1 && k < c.M) ? k + 1 : c.M + 1;
    };
    // warp w owns inputs [j_lo, j_hi), whole rounds of 32 (at most NR rounds);
    // the spike times are loaded once, first, and kept for both passes
    constexpr int NR = (kNarrowMaxIn + NW * 32 - 1) / (NW * 32);
    const int C = (((N_in + NW - 1) / NW) + 31) & ~31;
    const int j_lo = warp * C, j_hi = (j_lo + C) < N_in ? (j_lo + C) : N_in;
    float xr[NR];
#pragma unroll
    for (int r = 0; r < NR; ++r) {
        const int j = j_lo + 32 * r + lane;
        xr[r] = (32 * r < C && j < j_hi) ? tb[j] : INFINITY;
    }
    for (int e = threadIdx.x; e < N_out * c.Mp; e += NARROW_FWD_THREADS) acc[e] = 0.f;
    for (int e = threadIdx.x; e < NW * NK; e += NARROW_FWD_THREADS) hist[e] = 0;
    // W as it is: 16-byte copies when the sizes allow (consecutive threads,
    // consecutive addresses: no bank conflicts)
    if (((N_in * N_out) & 3) == 0 && (reinterpret_cast<uintptr_t>(W) & 15) == 0 &&
        (reinterpret_cast<uintptr_t>(ws) & 15) == 0) {
        const int nq = (N_in * N_out) >> 2;
        for (int e0 = threadIdx.x; e0 < nq; e0 += 4 * NARROW_FWD_THREADS) {
            float4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int e = e0 + u * NARROW_FWD_THREADS;
                if (e < nq) v[u] = reinterpret_cast<const float4 *>(W)[e];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int e = e0 + u * NARROW_FWD_THREADS;
                if (e < nq) reinterpret_cast<float4 *>(ws)[e] = v[u];
            }
        }
    } else {
        for (int e = threadIdx.x; e < N_in * N_out; e += NARROW_FWD_THREADS) ws[e] = W[e];
    }
    __syncthreads();
    // pass 1: ranks within (warp, key)
#pragma unroll
    for (int r = 0; r < NR; ++r) {
        if (32 * r >= C) break;
        const int j = j_lo + 32 * r + lane;
        const int key = (j < j_hi) ? key_of(xr[r]) : c.M + 1;
        const unsigned match = __match_any_sync(0xffffffffu, key);
        const unsigned lt = match & ((1u << lane) - 1u);
        const int base = hist[warp * NK + key];
        if (j < j_hi) upos[j] = base + __popc(lt);
        __syncwarp();
        if (lt == 0) hist[warp * NK + key] = base + __popc(match);
        __syncwarp();
    }
    // row sums of W (dead-neuron term), warp w taking rows w, w + NW, ...
    for (int i = warp; i < N_out; i += NW) {
        float r = 0.f;
        for (int j = lane; j < N_in; j += 32) r += ws[i * N_in + j];
        r = warp_sum(r);
        if (lane == 0) rsum[i] = r;
    }
    __syncthreads();
    // offsets: the start of each key (an exclusive scan over keys by warp 0,
    // up to 96 keys), then of each (warp, key) in warp order
    if (warp == 0) {
        int tot[3], run = 0;
#pragma unroll
        for (int r = 0; r < 3; ++r) {
            const int k = lane * 3 + r;
            int n = 0;
            if (k < NK)
                for (int w = 0; w < NW; ++w) n += hist[w * NK + k];
            tot[r] = n;
            run += n;
        }
        int incl = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        int ex = incl - run;
#pragma unroll
        for (int r = 0; r < 3; ++r) {
            const int k = lane * 3 + r;
            if (k < NK) start[k] = ex;
            ex += tot[r];
        }
        if (lane == 31) start[NK] = incl;
    }
    __syncthreads();
    if (threadIdx.x < NK) {
        const int k = threadIdx.x;
        int run = start[k];
        for (int w = 0; w < NW; ++w) {
            const int n = hist[w * NK + k];
            hist[w * NK + k] = run;
            run += n;
        }
    }
    __syncthreads();
    // pass 2: place (j, wR, wL) of every input with a weight
#pragma unroll
    for (int r = 0; r < NR; ++r) {
        if (32 * r >= C) break;
        const int j = j_lo + 32 * r + lane;
        if (j >= j_hi) continue;
        const float x = xr[r];
        const int key = key_of(x);
        if (key > c.M) continue;
        const BinW w = bin_weights(c, x, false);
        const int pos = hist[warp * NK + key] + upos[j];
        sj[pos] = j;
        sw[pos] = make_float2(w.wR, w.wL);
    }
    __syncthreads();
    // w^_.m: warp per grid point m; step m - 1 (key m) gives wL, step m
    // (key m + 1) gives wR
    for (int m = warp; m < c.M; m += NW) {
        float a[NOUT];
#pragma unroll
        for (int i = 0; i < NOUT; ++i) a[i] = 0.f;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int p0 = start[m + h], p1 = start[m + h + 1];
            for (int p = p0 + lane; p < p1; p += 32) {
                const float2 ww = sw[p];
                const float wv = h ? ww.x : ww.y;
                const float *col = ws + sj[p];
#pragma unroll
                for (int i = 0; i < NOUT; ++i)
                    if (i < N_out) a[i] = fmaf(col[i * N_in], wv, a[i]);
            }
        }
#pragma unroll
        for (int i = 0; i < NOUT; ++i) {
            if (i >= N_out) break;
            const float r = warp_sum(a[i]);
            if (lane == 0) acc[i * c.Mp + m] = r;
        }
    }
    __syncthreads();
    float pacc[4] = {0.f, 0.f, 0.f, 0.f};
    if (threadIdx.x < N_out) {
        const int i = threadIdx.x;
        ScanState st;
        scan_reset(st, c.M);
        float v = 0.f, I = 0.f;
        for (int m0 = 0; m0 < c.M; m0 += SUB) {
            const int mend = (c.M - m0) < SUB ? (c.M - m0) : SUB;
            if (scan_walk<SUB>(c, acc + i * c.Mp + m0, m0, mend, v, I, st)) break;
        }
        scan_finish(c, st);
        finish_neuron(c, st, b, i, N_out, rsum, t_out, q, s, vdot, pacc);
    }
    flush_penalty(pacc, penalty);
    if (ce.loss == nullptr) return;
    // cross-entropy over softmax(-t / tau_soft) of this sample (Eqs.
    // cost_function, L, S_i), one lane per output: a silent output enters
    // with t_silent and passes no gradient; the batch mean of the per-sample
    // terms is taken by the block that finishes last, in sample order
    __syncthreads();  // the sample's t_out (written above) visible to warp 0
    if (warp != 0) return;
    const float inv_tau = 1.0f / ce.tau_soft;
    const int B = gridDim.x, y = ce.labels[b];
    const float x = lane < N_out ? t_out[(long long)b * N_out + lane] : INFINITY;
    const bool fin = isfinite(x);
    const float z = lane < N_out ? -(fin ? x : ce.t_silent) * inv_tau : -INFINITY;
    float zmax = z;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) zmax = fmaxf(zmax, __shfl_xor_sync(0xffffffffu, zmax, o));
    const float e = lane < N_out ? expf(z - zmax) : 0.f;
    const float den = warp_sum(e);
    const float zy = __shfl_sync(0xffffffffu, z, y & 31);
    if (lane < N_out)
        ce.g[(long long)b * N_out + lane] = fin ? (-inv_tau / (float)B) * (e / den - (lane == y ? 1.f : 0.f)) : 0.f;
    unsigned ticket = 0u;
    if (lane == 0) {
        ce.scratch[b] = -(zy - zmax - logf(den)) / (float)B;
        __threadfence();
        ticket = atomicAdd(reinterpret_cast<unsigned int *>(ce.loss + 1), 1u);
    }
    ticket = __shfl_sync(0xffffffffu, ticket, 0);
    if (ticket != (unsigned)(B - 1)) return;
    __threadfence();
    float sum = 0.f;
    for (int k = lane; k < B; k += 32) sum += __ldcg(ce.scratch + k);
    sum = warp_sum(sum);
    if (lane == 0) {
        ce.loss[0] = sum;
        reinterpret_cast<unsigned int *>(ce.loss)[1] = 0u;
    }
}

size_t narrow_fwd_smem(int N_in, int N_out, int M, int Mp) {
    const int NW = NARROW_FWD_THREADS / 32, NK = M + 2;
    return sizeof(float) * ((size_t)N_in * N_out + (size_t)N_out * Mp + N_out) +
           sizeof(int) * ((size_t)NW * NK + NK + 1 + 2 * N_in + 1) + sizeof(float2) * (size_t)N_in + 16;
}

cudaError_t launch_narrow_fwd(const float *t, const float *W, int B, int N_in, int N_out, const LifConst &c,
                              float *t_out, int *q, float *s, float *vdot, float *penalty, cudaStream_t st,
                              const NarrowCe &ce) {
    if (N_out < 1 || N_out > kNarrowMaxOut || N_in > kNarrowMaxIn || c.M + 2 > 96) return cudaErrorInvalidValue;
    const size_t smem = narrow_fwd_smem(N_in, N_out, c.M, c.Mp);
    if (smem > kNarrowMaxSmem) return cudaErrorInvalidValue;
    cudaError_t e = cudaSuccess;
#define DSTD_NARROW_FWD(S, NO)                                                                                    \
    e = cudaFuncSetAttribute(k_narrow_fwd<S, NO>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);        \
    if (e != cudaSuccess) return e;                                                                                \
    k_narrow_fwd<S, NO><<<B, NARROW_FWD_THREADS, smem, st>>>(t, W, N_in, N_out, c, t_out, q, s, vdot, penalty, ce);
#define DSTD_NARROW_FWD_NO(S) \
    if (N_out <= 8) {         \
        DSTD_NARROW_FWD(S, 8) \
    } else if (N_out <= 16) { \
        DSTD_NARROW_FWD(S, 16) \
    } else {                  \
        DSTD_NARROW_FWD(S, 32) \
    }
    if (c.Mp <= 8) {
        DSTD_NARROW_FWD_NO(8)
    } else if (c.Mp <= 16) {
        DSTD_NARROW_FWD_NO(16)
    } else {
        DSTD_NARROW_FWD_NO(32)
    }
#undef DSTD_NARROW_FWD_NO
#undef DSTD_NARROW_FWD
    return cudaGetLastError();
}

// Backward, one block per NARROW_SAMPLES samples:
//   dw^_im = -g_i K(t_i - T_m) / v^'(t_i) for m <= q_i (as k_dwhat, in fp32,
//            in shared memory), and the count of silent neurons per output;
//   per input j and sample: its grid point k and the weights and their
//            t-derivatives (Tab. DSTD_kernels), the input-time gradient
//            g_t_j = sum_i W_ij (dw^_ik ds_k/dt + dw^_i,k+1 ds_k+1/dt), and
//            dW_ij += dw^_ik wR + dw^_i,k+1 wL;
// the block adds its dW (and the dead-neuron term qcoef * silent count) into
// g_W, which the caller zeroes.
constexpr int NARROW_SAMPLES = 2;
template <int NOUT>  // a bound on N_out: 8, 16 or 32
__global__ void __launch_bounds__(NARROW_BWD_THREADS) k_narrow_bwd(const float *__restrict__ t_in,
                                                             const float *__restrict__ W,
                                                             const float *__restrict__ t_out,
                                                             const int *__restrict__ qv, const float *__restrict__ sv,
                                                             const float *__restrict__ vd,
                                                             const float *__restrict__ g_up, int B, int N_in,
                                                             int N_out, LifConst c, float qcoef, float *g_t_in,
                                                             float *g_W) {
    extern __shared__ __align__(16) float nsh[];
    const int b0 = blockIdx.x * NARROW_SAMPLES;
    const int nb = (B - b0) < NARROW_SAMPLES ? (B - b0) : NARROW_SAMPLES;
    float *dw = nsh;                                     // [nb][N_out][Mp]
    float *cnt = nsh + NARROW_SAMPLES * N_out * c.Mp;    // [N_out]
    for (int e = threadIdx.x; e < N_out; e += NARROW_BWD_THREADS) cnt[e] = 0.f;
    __syncthreads();
    for (int e = threadIdx.x; e < nb * N_out * c.Mp; e += NARROW_BWD_THREADS) {
        const int m = e % c.Mp, r = e / c.Mp;
        const int i = r % N_out, sb = r / N_out;
        const long long idx = (long long)(b0 + sb) * N_out + i;
        const int q = qv[idx];
        float val = 0.f;
        if (q < c.M) {
            if (m <= q) {
                float pv, pg;
                penalty_T(c, t_out[idx], pv, pg);
                const float g = (g_up ? g_up[idx] : 0.f) + pg;
                val = -g / vd[idx] * kernel_K(c, sv[idx] + (float)(q - m) * c.dt);
            }
        } else if (m == 0) {
            atomicAdd(&cnt[i], 1.0f);
        }
        dw[e] = val;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < N_in; j += NARROW_BWD_THREADS) {
        float wcol[NOUT], dacc[NOUT];
#pragma unroll
        for (int i = 0; i < NOUT; ++i) {
            wcol[i] = (i < N_out) ? W[(long long)i * N_in + j] : 0.f;
            dacc[i] = 0.f;
        }
        for (int sb = 0; sb < nb; ++sb) {
            const float x = t_in[(long long)(b0 + sb) * N_in + j];
            BinW w{-100, 0.f, 0.f, 0.f, 0.f};
            if (isfinite(x)) w = bin_weights(c, x, g_t_in != nullptr);
            const bool in0 = w.k >= 0 && w.k < c.M, in1 = w.k + 1 >= 0 && w.k + 1 < c.M;
            const float *d = dw + sb * N_out * c.Mp;
            float gt = 0.f;
#pragma unroll
            for (int i = 0; i < NOUT; ++i) {
                if (i < N_out) {
                    const float d0 = in0 ? d[i * c.Mp + w.k] : 0.f;
                    const float d1 = in1 ? d[i * c.Mp + w.k + 1] : 0.f;
                    gt = fmaf(wcol[i], fmaf(d0, w.dR, d1 * w.dL), gt);
                    dacc[i] = fmaf(d0, w.wR, fmaf(d1, w.wL, dacc[i]));
                }
            }
            if (g_t_in) g_t_in[(long long)(b0 + sb) * N_in + j] = gt;
        }
#pragma unroll
        for (int i = 0; i < NOUT; ++i)
            if (i < N_out) atomicAdd(&g_W[(long long)i * N_in + j], fmaf(qcoef, cnt[i], dacc[i]));
    }
}

cudaError_t launch_narrow_bwd(const float *t_in, const float *W, const float *t_out, const int *q, const float *s,
                              const float *vdot, const float *g_up, int B, int N_in, int N_out, const LifConst &c,
                              float qcoef, float *g_t_in, float *g_W, cudaStream_t st) {
    if (N_out < 1 || N_out > kNarrowMaxOut) return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(g_W, 0, sizeof(float) * (size_t)N_out * N_in, st);
    if (e != cudaSuccess) return e;
    const size_t smem = sizeof(float) * ((size_t)NARROW_SAMPLES * N_out * c.Mp + N_out);
    const unsigned g = (unsigned)((B + NARROW_SAMPLES - 1) / NARROW_SAMPLES);
#define DSTD_NARROW_BWD(NO)                                                                                    \
    k_narrow_bwd<NO><<<g, NARROW_BWD_THREADS, smem, st>>>(t_in, W, t_out, q, s, vdot, g_up, B, N_in, N_out, c, qcoef, \
                                                     g_t_in, g_W);
    if (N_out <= 8) {
        DSTD_NARROW_BWD(8)
    } else if (N_out <= 16) {
        DSTD_NARROW_BWD(16)
    } else {
        DSTD_NARROW_BWD(32)
    }
#undef DSTD_NARROW_BWD
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Backward, step 1: dC/dw^_im = -g_i K(t_i - T_m) / v^'(t_i) for m <= q_i
// (implicit function theorem on v^(t_i) = v_th), g_i = upstream + dT/dt_i.
// Writes it in the layout
//   A [N, lda]: row i, columns (b, m)
// which dW = dw^T . s reads as its K-major A operand and the tensor-core dS =
// dw^ . W reads transposed (MN-major B). The fp32 mode's CUDA-core dS wants
// the transposed copy too, when b is given:
//   B [B*Mp, ldb]: row (b, m), column i
// ---------------------------------------------------------------------------
// Two adjacent lanes share one neuron (b, i): lane h = 0, 1 takes the
// 16-byte chunks h, h+2, h+4, ... of its Mp bins, so that every 16-byte
// store of the (i, (b, m)) layout is half of a sector the other lane fills in
// the same instruction; the ((b, m), i) layout is written element-wise, 16
// consecutive neurons per row and instruction.
template <int OP>
__global__ void k_dwhat(const float *__restrict__ t_out, const int *__restrict__ qv, const float *__restrict__ sv,
                        const float *__restrict__ vd, const float *__restrict__ g_up, int B, int N, LifConst c,
                        void *a_hi, void *a_lo, int lda, void *b_hi, void *b_lo, int ldb, float *count) {
    constexpr int EB = OP == 0 ? 4 : 2;  // bytes per element
    constexpr int BPC = 16 / EB;         // bins per 16-byte chunk
    const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long idx = tid >> 1;
    const int h = (int)(tid & 1);
    if (idx >= (long long)B * N) return;
    const int b = (int)(idx / N), i = (int)(idx % N);
    const int q = qv[idx];
    float coef = 0.f, s0 = 0.f;
    if (q < c.M) {
        float pv, pg;
        penalty_T(c, t_out[idx], pv, pg);
        const float g = (g_up ? g_up[idx] : 0.f) + pg;
        coef = -g / vd[idx];
        s0 = sv[idx];
    } else if (count && h == 0) {
        atomicAdd(&count[i], 1.0f);
    }
    const long long abase = (long long)i * lda + (long long)b * c.Mp;
    // K(x) at x = s0 + (q - m) dt. Away from the spike K = (e^{-av x} -
    // e^{-aI x}) / lam (x e^{-av x} when lam = 0): both exponentials are taken
    // at the first bin of a chunk and advance by the factors e^{av dt},
    // e^{aI dt} per bin (x falls by dt); the spike's own bin and the one
    // before it (x < 2 dt, where that difference cancels) take the expm1
    // form. Chunks after the spike's bin, and every chunk of a silent
    // neuron, are zero.
    const bool fired = q < c.M;
    const float Kq = fired ? kernel_K(c, s0) : 0.f;
    const float Kq1 = fired ? kernel_K(c, s0 + c.dt) : 0.f;
    const float fv = __expf(c.av * c.dt), fI = __expf(c.aI * c.dt);
    const int nch = c.Mp / BPC;
    for (int ch = h; ch < nch; ch += 2) {
        const int m0 = ch * BPC;
        float v[BPC];
        if (!fired || m0 > q) {
#pragma unroll
            for (int u = 0; u < BPC; ++u) v[u] = 0.f;
        } else {
            float x = s0 + (float)(q - m0) * c.dt;
            float ev = __expf(-c.av * x), eI = __expf(-c.aI * x);
#pragma unroll
            for (int u = 0; u < BPC; ++u) {
                const int m = m0 + u;
                const float Kf = c.lam_zero ? x * ev : (ev - eI) * c.inv_lam;
                const float K = (m == q) ? Kq : ((m == q - 1) ? Kq1 : Kf);
                v[u] = (m <= q) ? coef * K : 0.f;
                ev *= fv;
                eI *= fI;
                x -= c.dt;
            }
        }
        if (OP == 0) {
            *reinterpret_cast<float4 *>((float *)a_hi + abase + m0) = make_float4(v[0], v[1], v[2], v[3]);
            if (b_hi) {
#pragma unroll
                for (int u = 0; u < BPC; ++u) ((float *)b_hi)[((long long)b * c.Mp + m0 + u) * ldb + i] = v[u];
            }
        } else {
            __align__(16) __nv_bfloat16 hh[BPC], ll[BPC];
#pragma unroll
            for (int u = 0; u < BPC; ++u) split_bf16(v[u], hh[u], ll[u]);
            *reinterpret_cast<uint4 *>((__nv_bfloat16 *)a_hi + abase + m0) = *reinterpret_cast<uint4 *>(hh);
            if (OP == 1) *reinterpret_cast<uint4 *>((__nv_bfloat16 *)a_lo + abase + m0) = *reinterpret_cast<uint4 *>(ll);
            if (b_hi) {
#pragma unroll
                for (int u = 0; u < BPC; ++u) {
                    const long long o = ((long long)b * c.Mp + m0 + u) * ldb + i;
                    ((__nv_bfloat16 *)b_hi)[o] = hh[u];
                    if (OP == 1) ((__nv_bfloat16 *)b_lo)[o] = ll[u];
                }
            }
        }
    }
}

// The same values in the (i, (b, m)) layout only, written row-contiguously,
// a block per 32 neurons x spb (<= 32) samples. First the block reads the
// per-(sample, neuron) inputs along the neurons (coalesced) and keeps each
// neuron's bin q, the coefficient -g/v^' folded into the two exponential
// terms of K at T_0, and the two accurate kernel values next to the spike
// in shared memory. Then each warp writes the rows of 4 neurons: lane f of a
// row's (sample, 16-byte chunk) sequence writes chunk f, so every store
// instruction covers up to 512 contiguous bytes (column b Mp + m). A chunk
// wholly before the spike's last two bins is the bare geometric recurrence
// in m (factors e^{av dt}, e^{aI dt}), a chunk after the spike is zero, and
// only the chunk holding bins q - 1, q selects per bin. Silent neurons are
// counted per block column and added with one atomic each.
template <int OP>
__global__ void __launch_bounds__(256) k_dwhat_rows(const float *__restrict__ t_out, const int *__restrict__ qv,
                                                    const float *__restrict__ sv, const float *__restrict__ vd,
                                                    const float *__restrict__ g_up, int B, int N, LifConst c,
                                                    void *a_hi, void *a_lo, int lda, float *count, int spb) {
    constexpr int EB = OP == 0 ? 4 : 2;
    constexpr int BPC = 16 / EB;
    __shared__ int sq[32][33];
    __shared__ float sa[32][33], sb[32][33], sk0[32][33], sk1[32][33];
    __shared__ int scount[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int i0 = blockIdx.x * 32, b0 = blockIdx.y * spb;
    const int nb = (B - b0) < spb ? (B - b0) : spb;
    if (threadIdx.x < 32) scount[threadIdx.x] = 0;
    __syncthreads();
    {
        const int i = i0 + lane;
        int silent = 0;
        for (int bl = warp; bl < nb; bl += 8) {
            int q = c.M;
            float A = 0.f, Bt = 0.f, K0 = 0.f, K1 = 0.f;
            if (i < N) {
                const long long idx = (long long)(b0 + bl) * N + i;
                q = __ldg(qv + idx);
                const float to = __ldg(t_out + idx), gu = g_up ? __ldg(g_up + idx) : 0.f, vdi = __ldg(vd + idx),
                            s0 = __ldg(sv + idx);
                if (q < c.M) {
                    float pv, pg;
                    penalty_T(c, to, pv, pg);
                    const float coef = -(gu + pg) / vdi;
                    const float x = s0 + (float)q * c.dt;  // t - T_0
                    K0 = coef * kernel_K(c, s0);
                    K1 = coef * kernel_K(c, s0 + c.dt);
                    if (c.lam_zero) {
                        A = coef * __expf(-c.av * x);
                        Bt = x;
                    } else {
                        A = coef * c.inv_lam * __expf(-c.av * x);
                        Bt = coef * c.inv_lam * __expf(-c.aI * x);
                    }
                } else {
                    ++silent;
                }
            }
            sq[lane][bl] = q;
            sa[lane][bl] = A;
            sb[lane][bl] = Bt;
            sk0[lane][bl] = K0;
            sk1[lane][bl] = K1;
        }
        if (silent) atomicAdd(&scount[lane], silent);
    }
    __syncthreads();
    if (count && threadIdx.x < 32 && i0 + threadIdx.x < N && scount[threadIdx.x])
        atomicAdd(&count[i0 + threadIdx.x], (float)scount[threadIdx.x]);
    const int cps = c.Mp / BPC;
    const int total = nb * cps;
    const float fv = __expf(c.av * c.dt), fI = __expf(c.aI * c.dt);
    for (int il = warp; il < 32; il += 8) {
        const int i = i0 + il;
        if (i >= N) break;
        for (int f = lane; f < total; f += 32) {
            const int bl = f / cps, ch = f - bl * cps;
            const int q = sq[il][bl];
            const int m0 = ch * BPC;
            float v[BPC];
#pragma unroll
            for (int u = 0; u < BPC; ++u) v[u] = 0.f;
            if (q < c.M && m0 <= q) {
                // the terms at T_m0: e^{av m0 dt}, e^{aI m0 dt} times those at T_0
                const float gv = __expf(c.av * c.dt * (float)m0), gI = __expf(c.aI * c.dt * (float)m0);
                float A = sa[il][bl] * gv, Bt = c.lam_zero ? sb[il][bl] - (float)m0 * c.dt : sb[il][bl] * gI;
                if (m0 + BPC - 1 < q - 1) {
#pragma unroll
                    for (int u = 0; u < BPC; ++u) {
                        v[u] = c.lam_zero ? A * Bt : A - Bt;
                        A *= fv;
                        Bt = c.lam_zero ? Bt - c.dt : Bt * fI;
                    }
                } else {
                    const float K0 = sk0[il][bl], K1 = sk1[il][bl];
#pragma unroll
                    for (int u = 0; u < BPC; ++u) {
                        const int m = m0 + u;
                        const float d = c.lam_zero ? A * Bt : A - Bt;
                        v[u] = m < q - 1 ? d : (m == q - 1 ? K1 : (m == q ? K0 : 0.f));
                        A *= fv;
                        Bt = c.lam_zero ? Bt - c.dt : Bt * fI;
                    }
                }
            }
            const long long o = (long long)i * lda + (long long)(b0 + bl) * c.Mp + m0;
            if (OP == 0) {
                *reinterpret_cast<float4 *>((float *)a_hi + o) = make_float4(v[0], v[1], v[2], v[3]);
            } else {
                __align__(16) __nv_bfloat16 hh[BPC], ll[BPC];
#pragma unroll
                for (int u = 0; u < BPC; ++u) split_bf16(v[u], hh[u], ll[u]);
                *reinterpret_cast<uint4 *>((__nv_bfloat16 *)a_hi + o) = *reinterpret_cast<uint4 *>(hh);
                if (OP == 1) *reinterpret_cast<uint4 *>((__nv_bfloat16 *)a_lo + o) = *reinterpret_cast<uint4 *>(ll);
            }
        }
    }
}

cudaError_t launch_dwhat(const float *t_out, const int *q, const float *s, const float *vdot, const float *g_up,
                         int B, int N, const LifConst &c, OpKind op, void *a_hi, void *a_lo, int lda, void *b_hi,
                         void *b_lo, int ldb, float *silent_count, cudaStream_t st, bool accumulate_count) {
    if (silent_count && !accumulate_count) {
        cudaError_t e = cudaMemsetAsync(silent_count, 0, sizeof(float) * N, st);
        if (e != cudaSuccess) return e;
    }
    // samples per block: 64 chunks per warp (two stores per lane and array), at most 32
    const int cps = c.Mp / (op == OpKind::F32 ? 4 : 8);
    const int spb = cps >= 32 ? 2 : (64 / cps > 32 ? 32 : 64 / cps);
    const long long gy = ((long long)B + spb - 1) / spb;
    if (!b_hi && gy <= 65535) {
        dim3 grid((unsigned)((N + 31) / 32), (unsigned)gy);
        if (op == OpKind::F32)
            k_dwhat_rows<0><<<grid, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, silent_count, spb);
        else if (op == OpKind::BF16X3)
            k_dwhat_rows<1><<<grid, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, silent_count, spb);
        else
            k_dwhat_rows<2><<<grid, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, silent_count, spb);
        return cudaGetLastError();
    }
    long long n = 2ll * B * N;  // two lanes per neuron
    unsigned g = blocks_for(n, 256);
    if (op == OpKind::F32)
        k_dwhat<0><<<g, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, b_hi, b_lo, ldb, silent_count);
    else if (op == OpKind::BF16X3)
        k_dwhat<1><<<g, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, b_hi, b_lo, ldb, silent_count);
    else
        k_dwhat<2><<<g, 256, 0, st>>>(t_out, q, s, vdot, g_up, B, N, c, a_hi, a_lo, lda, b_hi, b_lo, ldb, silent_count);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Backward, input times: g_t_j = sum_{m in {k, k+1}} dS[j, (b, m)] ds_jm/dt_j.
// ---------------------------------------------------------------------------
__global__ void k_gt_from_ds(const float *__restrict__ D, long long ldd, const float *__restrict__ t_in, int B,
                             int N, LifConst c, float *g_t_in) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N) return;
    const int b = (int)(idx / N), j = (int)(idx % N);
    float x = t_in[idx];
    float g = 0.f;
    if (isfinite(x)) {
        BinW w = bin_weights(c, x, true);
        const float *row = D + (long long)j * ldd + (long long)b * c.Mp;
        if (w.k >= 0 && w.k < c.M) g += row[w.k] * w.dR;
        if (w.k + 1 >= 0 && w.k + 1 < c.M) g += row[w.k + 1] * w.dL;
    }
    g_t_in[idx] = g;
}

cudaError_t launch_gt_from_ds(const float *D, long long ldd, const float *t_in, int B, int N, const LifConst &c,
                              float *g_t_in, cudaStream_t st) {
    long long n = (long long)B * N;
    k_gt_from_ds<<<blocks_for(n, 256), 256, 0, st>>>(D, ldd, t_in, B, N, c, g_t_in);
    return cudaGetLastError();
}

// Input-time gradient of a layer with few outputs, straight from its
// definition: g_t[b, j] = sum_n W[n, j] (dw^[b, n, k] ds_k/dt + dw^[b, n, k+1]
// ds_{k+1}/dt) over the two grid points k, k+1 of input j (the derivative of
// Tab. DSTD_kernels), with k and the derivatives from the transposed binning
// (bw) and dw^ from its (n, (b, m)) operand layout, fp32 = hi + lo. One
// thread per (b, j); 2 N_out multiply-adds each.
__global__ void k_gradt_small(const float *__restrict__ W, int N_out, int N_in, int B, LifConst c,
                              const float4 *__restrict__ bw, const __nv_bfloat16 *__restrict__ d_hi,
                              const __nv_bfloat16 *__restrict__ d_lo, int ld, float *g_t_in) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N_in) return;
    const int b = (int)(idx / N_in), j = (int)(idx % N_in);
    const float4 q = bw[idx];
    const int k = __float_as_int(q.x);
    const bool in0 = k >= 0 && k < c.M, in1 = k + 1 >= 0 && k + 1 < c.M;
    float g = 0.f;
    if (in0 || in1) {
        for (int n = 0; n < N_out; ++n) {
            const long long base = (long long)n * ld + (long long)b * c.Mp + k;
            float d0 = 0.f, d1 = 0.f;
            if (in0) d0 = __bfloat162float(d_hi[base]) + (d_lo ? __bfloat162float(d_lo[base]) : 0.f);
            if (in1) d1 = __bfloat162float(d_hi[base + 1]) + (d_lo ? __bfloat162float(d_lo[base + 1]) : 0.f);
            g = fmaf(W[(long long)n * N_in + j], fmaf(d0, q.y, d1 * q.z), g);
        }
    }
    g_t_in[idx] = g;
}

cudaError_t launch_gradt_small(const float *W, int N_out, int N_in, int B, const LifConst &c, const float4 *bw,
                               const __nv_bfloat16 *d_hi, const __nv_bfloat16 *d_lo, int ld, float *g_t_in,
                               cudaStream_t st) {
    long long n = (long long)B * N_in;
    k_gradt_small<<<blocks_for(n, 256), 256, 0, st>>>(W, N_out, N_in, B, c, bw, d_hi, d_lo, ld, g_t_in);
    return cudaGetLastError();
}

__global__ void k_dw_reduce(const float *__restrict__ part, int splits, long long zstride, int ldp, int R, int C,
                            const float *__restrict__ count, float qcoef, float *g_W, int accumulate) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)R * C) return;
    int i = (int)(idx / C), j = (int)(idx % C);
    float s = 0.f;
    for (int z = 0; z < splits; ++z) s += part[z * zstride + (long long)i * ldp + j];
    if (count) s += qcoef * count[i];
    g_W[idx] = accumulate ? g_W[idx] + s : s;
}

cudaError_t launch_dw_reduce(const float *part, int splits, long long zstride, int ldp, int R, int C,
                             const float *count, float qcoef, float *g_W, cudaStream_t st, bool accumulate) {
    long long n = (long long)R * C;
    k_dw_reduce<<<blocks_for(n, 256), 256, 0, st>>>(part, splits, zstride, ldp, R, C, count, qcoef, g_W,
                                                    accumulate ? 1 : 0);
    return cudaGetLastError();
}

__global__ void k_what_to_public(const float *__restrict__ D, long long ld, int B, int N, int M, int Mp,
                                 float *out) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N * M) return;
    int m = (int)(idx % M);
    long long r = idx / M;
    int i = (int)(r % N), b = (int)(r / N);
    out[idx] = D[(long long)i * ld + (long long)b * Mp + m];
}

cudaError_t launch_what_to_public(const float *D, long long ld, int B, int N, int M, int Mp, float *out,
                                  cudaStream_t st) {
    long long n = (long long)B * N * M;
    k_what_to_public<<<blocks_for(n, 256), 256, 0, st>>>(D, ld, B, N, M, Mp, out);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Losses and optimizer.
// ---------------------------------------------------------------------------
__global__ void k_ce_loss(const float *__restrict__ t, const int32_t *__restrict__ lab, int B, int C, float tau_soft,
                          float t_silent, float *loss, float *g) {
    int b = blockIdx.x * blockDim.x + threadIdx.x;
    float contrib = 0.f;
    if (b < B) {
        const float *tb = t + (long long)b * C;
        float zmax = -INFINITY;
        for (int k = 0; k < C; ++k) {
            float x = isfinite(tb[k]) ? tb[k] : t_silent;
            zmax = fmaxf(zmax, -x / tau_soft);
        }
        float den = 0.f;
        for (int k = 0; k < C; ++k) {
            float x = isfinite(tb[k]) ? tb[k] : t_silent;
            den += expf(-x / tau_soft - zmax);
        }
        int y = lab[b];
        for (int k = 0; k < C; ++k) {
            bool fin = isfinite(tb[k]);
            float x = fin ? tb[k] : t_silent;
            float p = expf(-x / tau_soft - zmax) / den;
            if (k == y) contrib = -(-x / tau_soft - zmax - logf(den));
            float gg = -(p - (k == y ? 1.f : 0.f)) / tau_soft / (float)B;
            g[(long long)b * C + k] = fin ? gg : 0.f;
        }
    }
    float v = warp_sum(contrib / (float)B);
    if ((threadIdx.x & 31) == 0 && v != 0.f) atomicAdd(loss, v);
}

// Batches of up to 1024 samples and up to 32 classes: one block, one thread
// per sample with its row in registers, a block reduction, the loss written
// directly (no zeroing launch, no atomics).
constexpr int CE_MAX_C = 32;
__global__ void __launch_bounds__(1024) k_ce_loss_block(const float *__restrict__ t, const int32_t *__restrict__ lab,
                                                        int B, int C, float tau_soft, float t_silent, float *loss,
                                                        float *g) {
    __shared__ float part[32];
    const int b = threadIdx.x;
    const float inv_tau = 1.0f / tau_soft;
    float contrib = 0.f;
    if (b < B) {
        const float *tb = t + (long long)b * C;
        float z[CE_MAX_C];
        bool fin[CE_MAX_C];
        const int y = lab[b];
        float zmax = -INFINITY, zy = 0.f;
#pragma unroll
        for (int k = 0; k < CE_MAX_C; ++k) {
            if (k < C) {
                const float x = tb[k];
                fin[k] = isfinite(x);
                z[k] = -(fin[k] ? x : t_silent) * inv_tau;
                zmax = fmaxf(zmax, z[k]);
                if (k == y) zy = z[k];
            }
        }
        float den = 0.f;
#pragma unroll
        for (int k = 0; k < CE_MAX_C; ++k) {
            if (k < C) {
                z[k] = expf(z[k] - zmax);  // e_k = exp(z_k - zmax)
                den += z[k];
            }
        }
        const float inv_den = 1.0f / den;
        const float scale = -inv_tau / (float)B;
#pragma unroll
        for (int k = 0; k < CE_MAX_C; ++k) {
            if (k < C) {
                const float p = z[k] * inv_den;
                g[(long long)b * C + k] = fin[k] ? scale * (p - (k == y ? 1.f : 0.f)) : 0.f;
            }
        }
        contrib = -(zy - zmax - logf(den)) / (float)B;
    }
    const float v = warp_sum(contrib);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x < 32) {
        float u = threadIdx.x < (int)((blockDim.x + 31) >> 5) ? part[threadIdx.x] : 0.f;
        u = warp_sum(u);
        if (threadIdx.x == 0) loss[0] = u;
    }
}

cudaError_t launch_ce_loss(const float *t, const int32_t *lab, int B, int C, float tau_soft, float t_silent,
                           float *loss, float *g, cudaStream_t st) {
    if (B <= 1024 && C <= CE_MAX_C) {
        k_ce_loss_block<<<1, (B + 31) / 32 * 32, 0, st>>>(t, lab, B, C, tau_soft, t_silent, loss, g);
        return cudaGetLastError();
    }
    cudaError_t e = cudaMemsetAsync(loss, 0, sizeof(float), st);
    if (e != cudaSuccess) return e;
    k_ce_loss<<<blocks_for(B, 128), 128, 0, st>>>(t, lab, B, C, tau_soft, t_silent, loss, g);
    return cudaGetLastError();
}

__global__ void k_sum_t(const float *__restrict__ t, long long n, float *loss, float *g) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    float c = 0.f;
    if (idx < n) {
        float x = t[idx];
        bool f = isfinite(x);
        g[idx] = f ? 1.f : 0.f;
        c = f ? x : 0.f;
    }
    float v = warp_sum(c);
    if ((threadIdx.x & 31) == 0 && v != 0.f) atomicAdd(loss, v);
}

// ---------------------------------------------------------------------------
// Skip-and-delay input (App. C.3, Fig. skip_connection): the third layer of
// a block sees the block's input, delayed by a fixed time, beside the second
// layer's output. With NHWC spike tensors (channels innermost) that is a
// concatenation along channels per position p:
//   out[p, 0:Ca] = a[p, :] + delay,   out[p, Ca:Ca+Cb] = b[p, :]
// (+inf stays +inf: a silent input stays silent). Its adjoint splits the
// gradient back, overwriting or adding into each part.
// ---------------------------------------------------------------------------
__global__ void k_concat_channels(const float *__restrict__ a, int Ca, float delay, const float *__restrict__ b,
                                  int Cb, long long n, float *out) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n) return;
    const int Ct = Ca + Cb;
    const long long p = idx / Ct;
    const int ch = (int)(idx - p * Ct);
    out[idx] = ch < Ca ? a[p * Ca + ch] + delay : b[p * Cb + (ch - Ca)];
}

__global__ void k_split_channels(const float *__restrict__ g, int Ca, int Cb, long long n, float *ga, int acc_a,
                                 float *gb, int acc_b) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n) return;
    const int Ct = Ca + Cb;
    const long long p = idx / Ct;
    const int ch = (int)(idx - p * Ct);
    const float v = g[idx];
    if (ch < Ca) {
        if (ga) {
            float *d = ga + p * Ca + ch;
            *d = acc_a ? *d + v : v;
        }
    } else if (gb) {
        float *d = gb + p * Cb + (ch - Ca);
        *d = acc_b ? *d + v : v;
    }
}

cudaError_t launch_concat_channels(const float *a, int Ca, float delay, const float *b, int Cb, long long P, float *out,
                                   cudaStream_t st) {
    const long long n = P * (Ca + Cb);
    k_concat_channels<<<blocks_for(n, 256), 256, 0, st>>>(a, Ca, delay, b, Cb, n, out);
    return cudaGetLastError();
}

cudaError_t launch_split_channels(const float *g, int Ca, int Cb, long long P, float *ga, bool acc_a, float *gb,
                                  bool acc_b, cudaStream_t st) {
    const long long n = P * (Ca + Cb);
    k_split_channels<<<blocks_for(n, 256), 256, 0, st>>>(g, Ca, Cb, n, ga, acc_a ? 1 : 0, gb, acc_b ? 1 : 0);
    return cudaGetLastError();
}

cudaError_t launch_sum_t(const float *t, long long n, float *loss, float *g, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(loss, 0, sizeof(float), st);
    if (e != cudaSuccess) return e;
    k_sum_t<<<blocks_for(n, 256), 256, 0, st>>>(t, n, loss, g);
    return cudaGetLastError();
}

__global__ void k_adamw(float *w, const float *__restrict__ g, float *m, float *v, long long n, float lr, float b1,
                        float b2, float eps, float wd, float bc1, float bc2) {
    long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n) return;
    float gi = g[idx];
    float wi = w[idx] * (1.f - lr * wd);
    float mi = b1 * m[idx] + (1.f - b1) * gi;
    float vi = b2 * v[idx] + (1.f - b2) * gi * gi;
    m[idx] = mi;
    v[idx] = vi;
    w[idx] = wi - lr * (mi / bc1) / (sqrtf(vi / bc2) + eps);
}

cudaError_t launch_adamw(float *w, const float *g, float *m, float *v, long long n, float lr, float b1, float b2,
                         float eps, float wd, int step, cudaStream_t st) {
    float bc1 = (float)(1.0 - pow((double)b1, step));
    float bc2 = (float)(1.0 - pow((double)b2, step));
    k_adamw<<<blocks_for(n, 256), 256, 0, st>>>(w, g, m, v, n, lr, b1, b2, eps, wd, bc1, bc2);
    return cudaGetLastError();
}

// All parameter tensors of a network in one launch, with the update count in
// device memory (so a captured CUDA graph advances it on every replay).
// step[0] holds the count and step[1] a ticket; read together as one 64-bit
// word, each block adds one to the ticket at its start and so learns the
// count, and the block that draws the last ticket (every other block has then
// drawn its own) stores count + 1 with the ticket reset. Element e of the
// concatenation belongs to the segment whose offset range holds it; with VEC
// the offsets and sizes are in units of 4 floats. One unit per thread: its
// loads are issued before the count arrives.
template <int VEC>
__global__ void __launch_bounds__(256) k_adamw_multi(const AdamMultiArgs a) {
    __shared__ unsigned long long s_old;
    unsigned long long *word = reinterpret_cast<unsigned long long *>(a.step);
    if (threadIdx.x == 0) s_old = atomicAdd(word, 1ull << 32);
    const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const bool live = u < a.total;
    int k = 0;
    while (k + 1 < a.count && u >= a.seg[k + 1].off) ++k;
    const AdamSeg &sg = a.seg[k];
    const long long e = live ? u - sg.off : 0;
    float4 gi = make_float4(0.f, 0.f, 0.f, 0.f), wi = gi, mi = gi, vi = gi;
    if (live) {
        if (VEC) {
            gi = reinterpret_cast<const float4 *>(sg.g)[e];
            wi = reinterpret_cast<const float4 *>(sg.w)[e];
            mi = reinterpret_cast<const float4 *>(sg.m)[e];
            vi = reinterpret_cast<const float4 *>(sg.v)[e];
        } else {
            gi.x = sg.g[e];
            wi.x = sg.w[e];
            mi.x = sg.m[e];
            vi.x = sg.v[e];
        }
    }
    __syncthreads();
    const unsigned long long old = s_old;
    const int step = (int)(unsigned)(old & 0xffffffffull) + 1;
    if (threadIdx.x == 0 && (old >> 32) == (unsigned long long)(gridDim.x - 1))
        *word = (unsigned long long)(unsigned)step;  // count + 1, ticket 0
    if (!live) return;
    // fp32 (FP64 is slow on this part): 1 - beta^t to within a few ulp
    const float bc1 = 1.f - powf(a.b1, (float)step);
    const float bc2 = 1.f - powf(a.b2, (float)step);
    const float lr = a.lr_dev ? *a.lr_dev : a.lr;
    const float decay = 1.f - lr * a.wd;
    float *wp = &wi.x, *mp = &mi.x, *vp = &vi.x;
    const float *gp = &gi.x;
#pragma unroll
    for (int j = 0; j < (VEC ? 4 : 1); ++j) {
        mp[j] = a.b1 * mp[j] + (1.f - a.b1) * gp[j];
        vp[j] = a.b2 * vp[j] + (1.f - a.b2) * gp[j] * gp[j];
        wp[j] = wp[j] * decay - lr * (mp[j] / bc1) / (sqrtf(vp[j] / bc2) + a.eps);
    }
    if (VEC) {
        reinterpret_cast<float4 *>(sg.m)[e] = mi;
        reinterpret_cast<float4 *>(sg.v)[e] = vi;
        reinterpret_cast<float4 *>(sg.w)[e] = wi;
    } else {
        sg.m[e] = mi.x;
        sg.v[e] = vi.x;
        sg.w[e] = wi.x;
    }
}

cudaError_t launch_adamw_multi(const AdamMultiArgs &args, cudaStream_t st) {
    AdamMultiArgs a = args;
    bool vec = true;
    for (int i = 0; i < a.count; ++i) {
        const AdamSeg &sg = a.seg[i];
        vec = vec && (sg.n % 4) == 0 && ((reinterpret_cast<uintptr_t>(sg.w) | reinterpret_cast<uintptr_t>(sg.g) |
                                          reinterpret_cast<uintptr_t>(sg.m) | reinterpret_cast<uintptr_t>(sg.v)) &
                                         15) == 0;
    }
    long long off = 0;
    for (int i = 0; i < a.count; ++i) {
        a.seg[i].off = off;
        off += vec ? a.seg[i].n / 4 : a.seg[i].n;
    }
    a.total = off;
    const unsigned g = blocks_for(off > 0 ? off : 1, 256);
    if (vec) k_adamw_multi<1><<<g, 256, 0, st>>>(a);
    else k_adamw_multi<0><<<g, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace dstd
