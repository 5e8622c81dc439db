// Convolutional DSTD layer as implicit GEMMs on sm_103a (bf16 operands,
// tcgen05 + TMA), with no im2col operand.
//
// Layouts (a chunk of whole images, NHWC positions p = (b*H + y)*W + x):
//   S     [P_in][Mp][C_in]   bf16  grid weights of the input spikes (Eq.
//                                  DSTD_kernel): row (p, m), channel innermost
//   w^    [P_out][Mp][C_out] fp32  the forward contraction (Eq. DSTD)
//   dw^   [P_out][Mp][C_out] bf16  dC/dw^ (implicit-function theorem)
//   Wf    [C_out][k k C_in]  bf16  filters, taps (kh, kw) then channels
//   Wt    [C_in][k k C_out]  bf16  the same filters transposed
// A row (p, m) holds 64 channels per 128-byte swizzled line, so one TMA box
// of a 5-D tensor map (channel, m, x, y, b) = (64, Mp, 1, 1, 1) is the
// K-major operand slice of one position for one filter tap: the tap shifts
// the (x, y) coordinates, and coordinates outside the image read zeros,
// which is the silent padding. Nothing is gathered or expanded in memory.
//
//   forward  w^[(p, m), o]  = sum_{tap, c} S[(p + tap), m, c] Wf[o, tap, c]
//   dS       dS[(p', m), c] = sum_{tap, o} dw^[(p' - tap) / s, m, o] Wt[c, tap, o]
//            (the transposed convolution; taps whose output position is not
//            on the stride grid read zeros), consumed in the epilogue:
//            dC/dt_j = sum_{m in {k, k+1}} dS[(p', m), c] ds_jm/dt_j
//   dW       dW[o, tap, c]  = sum_{(p, m)} dw^[(p, m), o] S[(p + tap), m, c]
//            (both operands MN-major, K = positions x grid steps, split-K)
//
// One thread issues tcgen05.mma (M = 128, N = BN <= 256, K = 16) into one of
// two TMEM accumulators, so the epilogue of a tile overlaps the MMAs of the
// next. Every mbarrier wait is bounded; an expired wait sets this unit's
// status word, the role stops, and the CTA still frees its TMEM.
#include "dstd_internal.cuh"
#include "dstd_tc_ptx.cuh"

#include <cuda.h>
#include <mutex>

namespace dstd {

// status word of this unit (bit STATUS_TIMEOUT: an expired bounded wait)
__device__ unsigned int g_status_conv = 0;

static __device__ __forceinline__ void conv_set_status(unsigned int code) { atomicOr(&g_status_conv, code); }

cudaError_t conv_status_read(unsigned int *out, int clear) {
    cudaError_t e = cudaMemcpyFromSymbol(out, g_status_conv, sizeof(unsigned int));
    if (e != cudaSuccess || !clear) return e;
    unsigned int z = 0;
    return cudaMemcpyToSymbol(g_status_conv, &z, sizeof(z));
}

namespace {

static int conv_num_sms() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
    }
    return n;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// ---------------------------------------------------------------------------
// Binning (Eq. DSTD_kernel) into S [P][Mp][C]: a thread takes 8 channels of
// one position, computes their grid step and two weights, then writes the
// position's Mp rows of those channels (16 bytes per row, zeros away from the
// two grid points; a warp's store covers whole 128-byte lines).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_bin_pmc(const float *__restrict__ t, long long P, int C, LifConst c,
                                                 __nv_bfloat16 *__restrict__ S) {
    const int groups = C >> 3;
    const long long n = P * groups;
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long p = idx / groups;
        const int c0 = (int)(idx - p * groups) * 8;
        int k[8];
        float wR[8], wL[8];
        const float4 a = __ldg(reinterpret_cast<const float4 *>(t + p * C + c0));
        const float4 b = __ldg(reinterpret_cast<const float4 *>(t + p * C + c0 + 4));
        const float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            k[u] = -100;
            wR[u] = wL[u] = 0.f;
            if (isfinite(x[u])) {
                const BinW w = bin_weights(c, x[u], false);
                k[u] = w.k;
                wR[u] = w.wR;
                wL[u] = w.wL;
            }
        }
        uint4 *dst = reinterpret_cast<uint4 *>(S + p * (long long)c.Mp * C + c0);
        const int step = C >> 3;  // uint4 per row
        for (int m = 0; m < c.Mp; ++m) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                v[u] = (m < c.M) ? ((m == k[u]) ? wR[u] : ((m == k[u] + 1) ? wL[u] : 0.f)) : 0.f;
            dst[(long long)m * step] =
                make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                           pack_bf16x2(v[6], v[7]));
        }
    }
}

// ---------------------------------------------------------------------------
// dC/dw^_{p,m,o} = -g K(t - T_m) / v^'(t) for m <= q (0 after the spike's
// interval and for silent neurons), g = upstream + dT/dt, into [P][Mp][C_out]
// bf16. A thread takes 8 consecutive neurons of one position (16 bytes per
// row). K(x), x = t - T_m, falls along m by the factors e^{av dt}, e^{aI dt}
// from its value at m = 0; the spike's own bin and the one before it (x <
// 2 dt, where (e^{-av x} - e^{-aI x}) / lam cancels) take the accurate form.
// Silent neurons are counted per output channel (grid-stride loop, a fixed
// channel group per thread, one atomic per thread and channel at the end).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_dwhat_pmc(const float *__restrict__ t_out, const int *__restrict__ qv,
                                                   const float *__restrict__ sv, const float *__restrict__ vd,
                                                   const float *__restrict__ g_up, long long P, int C, LifConst c,
                                                   __nv_bfloat16 *__restrict__ D, float *count) {
    const int groups = C >> 3;
    const int tpb = blockDim.x;
    const int per_blk = tpb / groups;  // positions per block iteration (blockDim a multiple of groups)
    const int g = threadIdx.x % groups, pl = threadIdx.x / groups;
    const int c0 = g * 8;
    float cnt[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) cnt[u] = 0.f;
    const float fv = __expf(c.av * c.dt), fI = __expf(c.aI * c.dt);
    if (pl < per_blk) {
        for (long long p = (long long)blockIdx.x * per_blk + pl; p < P; p += (long long)gridDim.x * per_blk) {
            int q[8];
            float coef[8], ev[8], eI[8], x[8], Kq[8], Kq1[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const long long idx = p * C + c0 + u;
                q[u] = qv[idx];
                coef[u] = 0.f;
                x[u] = 0.f;
                Kq[u] = Kq1[u] = 0.f;
                if (q[u] < c.M) {
                    float pv, pg;
                    penalty_T(c, t_out[idx], pv, pg);
                    coef[u] = -((g_up ? g_up[idx] : 0.f) + pg) / vd[idx];
                    const float s0 = sv[idx];
                    x[u] = s0 + (float)q[u] * c.dt;  // t - T_0
                    Kq[u] = kernel_K(c, s0);
                    Kq1[u] = kernel_K(c, s0 + c.dt);
                } else {
                    cnt[u] += 1.f;
                }
                ev[u] = __expf(-c.av * x[u]);
                eI[u] = __expf(-c.aI * x[u]);
            }
            uint4 *dst = reinterpret_cast<uint4 *>(D + p * (long long)c.Mp * C + c0);
            const int step = C >> 3;
            for (int m = 0; m < c.Mp; ++m) {
                float v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const float Kf = c.lam_zero ? x[u] * ev[u] : (ev[u] - eI[u]) * c.inv_lam;
                    const float K = (m == q[u]) ? Kq[u] : ((m == q[u] - 1) ? Kq1[u] : Kf);
                    v[u] = (m <= q[u] && q[u] < c.M) ? coef[u] * K : 0.f;
                    ev[u] *= fv;
                    eI[u] *= fI;
                    x[u] -= c.dt;
                }
                dst[(long long)m * step] = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                                      pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
            }
        }
    }
    if (count) {
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (cnt[u] != 0.f) atomicAdd(&count[c0 + u], cnt[u]);
    }
}

// Filters [C_out][T][C_in] fp32 -> Wt [C_in][T][C_out] bf16 (T = k k taps).
__global__ void k_filters_t(const float *__restrict__ W, int C_out, int T, int C_in, __nv_bfloat16 *__restrict__ Wt) {
    const long long n = (long long)C_out * T * C_in;
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int o = (int)(idx % C_out);
        const long long r = idx / C_out;
        const int tap = (int)(r % T), ci = (int)(r / T);
        Wt[idx] = __float2bfloat16_rn(W[((long long)o * T + tap) * C_in + ci]);
    }
}


// ---------------------------------------------------------------------------
// TMA loads of 5-D boxes (channel, m, x, y, b) into this CTA's shared memory
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int c, int m, int x,
                                            int y, int b) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c), "r"(m), "r"(x), "r"(y), "r"(b), "r"(tc::smem_u32(bar))
        : "memory");
}

// Instruction descriptor, kind::f16 with bf16 A and B and fp32 D; a_mn / b_mn
// select MN-major operands (transpose bits 15 and 16).
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

constexpr int CONV_NEPI = 8;                          // epilogue warps
constexpr int CONV_THREADS = (2 + CONV_NEPI) * 32;    // + TMA producer warp + MMA warp
constexpr int CONV_SMEM_BUDGET = 200 * 1024;
constexpr int EPI_LD = 33;                            // per-warp transpose buffer row stride (floats)

// Geometry of one implicit-GEMM launch over a chunk of ni images.
struct ConvGemmArgs {
    int ni;              // images in the chunk
    int H, W, C_in;      // layer input grid
    int Ho, Wo, C_out;   // layer output grid
    int k, stride, pad;
    int Mp;
    int P_rows;          // row positions (forward: ni Ho Wo; dS: ni H W; dW: K positions ni Ho Wo)
    int n_row, n_col, n_split, kt_per_split, ktiles;
    float *what;         // forward: w^ [P_out][Mp][C_out]
    const float *t_in;   // dS: layer input spike times [P_in][C_in]
    float *g_t_in;       // dS: [P_in][C_in], zeroed, accumulated
    float *g_W;          // dW: [C_out][k k C_in], accumulated
    const float *count;  // dW: silent neurons per output channel (dead-neuron term), or null
    float qcoef;         // dW: -gamma_Q norm
    int nst;             // generated-operand kernels: pipeline stages
    int res_bytes;       // generated-operand forward: resident filter bytes (0: streamed)
    int groups;          // generated-operand dW: row tiles per CTA
    LifConst c;
};

template <int BN, int MODE>  // MODE 0 forward, 1 dS, 2 dW
struct ConvCfg {
    static constexpr int A_BYTES = 128 * 128;          // 128 rows (or MN) x 64 k of bf16
    static constexpr int B_BYTES = BN * 128;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int EPI_BYTES = MODE == 1 ? CONV_NEPI * 32 * EPI_LD * 4 : 0;
    static constexpr int STAGES_RAW = (CONV_SMEM_BUDGET - EPI_BYTES) / STAGE;
    static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
    static constexpr int SMEM = STAGES * STAGE + EPI_BYTES + 1024 + 256;
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static_assert(STAGES >= 2, "at least two stages");
    static_assert(BN == 64 || BN == 128 || BN == 256, "BN");
};

// position p of an (ni, h, w) grid -> (b, y, x)
__device__ __forceinline__ void pos_decode(int p, int h, int w, int &b, int &y, int &x) {
    const int hw = h * w;
    b = p / hw;
    const int r = p - b * hw;
    y = r / w;
    x = r - y * w;
}

// Source coordinates (x, y, b) of the A box of row position p and tap
// (kh, kw). Forward: the input position the tap reads. dS: the output
// position whose tap reads p, when p - tap is on the stride grid. Anything
// out of range is left outside the tensor, where TMA reads zeros.
template <int MODE>
__device__ __forceinline__ void conv_src(const ConvGemmArgs &a, int p, int kh, int kw, int &sx, int &sy, int &sb) {
    if (p >= a.P_rows) {
        sx = 0;
        sy = 0;
        sb = a.ni;
        return;
    }
    int b, y, x;
    if (MODE == 1) {
        pos_decode(p, a.H, a.W, b, y, x);
        const int ny = y + a.pad - kh, nx = x + a.pad - kw;
        sb = b;
        if (ny % a.stride != 0 || nx % a.stride != 0) {
            sx = 0;
            sy = -1;
        } else {
            sy = ny / a.stride;
            sx = nx / a.stride;
        }
    } else {
        pos_decode(p, a.Ho, a.Wo, b, y, x);
        sb = b;
        sy = y * a.stride + kh - a.pad;
        sx = x * a.stride + kw - a.pad;
    }
}

// ---------------------------------------------------------------------------
// Forward and dS: rows (position, m) of 128 per tile (128 / Mp positions),
// columns BN of the n_total channels; K = k k taps x blocks of 64 channels of
// the source activation. Persistent: CTA b takes tiles b, b + grid, ...
//   warp 0  TMA producer (one lane): the 128/Mp position boxes of A, B's box
//   warp 1  TMEM allocation and MMA issue (one lane)
//   warps 2-9  epilogue: warp w reads TMEM lane quarter w % 4, 32-column
//              chunks (w - 2) / 4, +2, ... of the tile
// Barriers: full/empty per stage; acc_full/acc_empty per accumulator (two).
// ---------------------------------------------------------------------------
template <int BN, int MODE>
__global__ void __launch_bounds__(CONV_THREADS, 1)
    k_conv_gemm(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, ConvGemmArgs a) {
    using Cfg = ConvCfg<BN, MODE>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    float *epi = reinterpret_cast<float *>(smem + Cfg::STAGES * Cfg::STAGE);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + Cfg::STAGES * Cfg::STAGE + Cfg::EPI_BYTES);
    uint64_t *empty = full + Cfg::STAGES;
    uint64_t *acc_full = empty + Cfg::STAGES;  // [2]
    uint64_t *acc_empty = acc_full + 2;       // [2]
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 2);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = a.n_row * a.n_col;
    const int Mp = a.Mp;
    const int ppt = 128 / Mp;  // positions per tile
    const int c_red = MODE == 0 ? a.C_in : a.C_out;
    const int ncb = c_red >> 6;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&acc_full[u], 1);
            tc::mbar_init(&acc_empty[u], CONV_NEPI);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                const int rt = t / a.n_col, ct = t - rt * a.n_col;
                for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                    const int s = it % Cfg::STAGES;
                    const uint32_t ph = (it / Cfg::STAGES) & 1u;
                    if (!tc::mbar_wait(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full[s], (uint32_t)Cfg::STAGE);
                    const int tap = kt / ncb, cb = kt - tap * ncb;
                    const int kh = tap / a.k, kw = tap - kh * a.k;
                    const uint32_t st = tc::smem_u32(smem + s * Cfg::STAGE);
                    for (int pp = 0; pp < ppt; ++pp) {
                        int sx, sy, sb;
                        conv_src<MODE>(a, rt * ppt + pp, kh, kw, sx, sy, sb);
                        tma_load_5d(st + pp * Mp * 128, &mapA, &full[s], cb * 64, 0, sx, sy, sb);
                    }
                    tc::tma_load_2d(st + Cfg::A_BYTES, &mapB, &full[s], tap * c_red + cb * 64, ct * BN);
                }
            }
            // loads still in flight (after an expired wait) land before the CTA exits
            const uint32_t n_drain = it < (uint32_t)Cfg::STAGES ? it : (uint32_t)Cfg::STAGES;
            for (uint32_t i = it - n_drain; i < it; ++i)
                tc::mbar_wait(&full[i % Cfg::STAGES], (i / Cfg::STAGES) & 1u);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, false, false);
            uint32_t it = 0, j = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                const uint32_t buf = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait(&acc_empty[buf], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc = tmem + buf * BN;
                for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                    const int s = it % Cfg::STAGES;
                    const uint32_t ph = (it / Cfg::STAGES) & 1u;
                    if (!tc::mbar_wait(&full[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * Cfg::STAGE);
                    const uint32_t sbb = sa + Cfg::A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc::mma_bf16(acc, tc::sdesc_sw128(sa + kk * 32), tc::sdesc_sw128(sbb + kk * 32), idesc,
                                     (kt > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_commit(&empty[s]);
                }
                if (ok) tc::mma_commit(&acc_full[buf]);
            }
        }
        __syncwarp();
    } else {
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        float *tb = epi + (warp - 2) * 32 * EPI_LD;
        const int r = quarter * 32 + lane;       // tile row of this lane
        const int pp = (quarter * 32) / Mp;      // position of this warp's rows (Mp >= 32)
        const int m_base = (quarter * 32) % Mp;  // first grid step of this warp's rows
        uint32_t j = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
            const int rt = t / a.n_col, ct = t - rt * a.n_col;
            const uint32_t buf = j & 1u;
            if (!tc::mbar_wait_sleep(&acc_full[buf], (j >> 1) & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            const int p = rt * ppt + pp;
            for (int cc = group; cc < BN / 32; cc += 2) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + buf * BN + cc * 32, v);
                const int col0 = ct * BN + cc * 32;
                if (MODE == 0) {
                    if (p < a.P_rows) {
                        float *dst = a.what + ((long long)p * Mp + (r % Mp)) * a.C_out + col0;
#pragma unroll
                        for (int u = 0; u < 32; u += 4)
                            *reinterpret_cast<float4 *>(dst + u) = make_float4(v[u], v[u + 1], v[u + 2], v[u + 3]);
                    }
                } else {
                    // dS: lane m of the warp holds grid step m_base + m of 32
                    // channels; transpose through shared memory so that lane
                    // u owns channel col0 + u and reads its two grid steps
#pragma unroll
                    for (int u = 0; u < 32; ++u) tb[lane * EPI_LD + u] = v[u];
                    __syncwarp();
                    if (p < a.P_rows) {
                        const long long e = (long long)p * a.C_in + col0 + lane;
                        const float x = __ldg(a.t_in + e);
                        if (isfinite(x)) {
                            const BinW w = bin_weights(a.c, x, true);
                            float g = 0.f;
                            const int k0 = w.k - m_base, k1 = w.k + 1 - m_base;
                            if (k0 >= 0 && k0 < 32 && w.k < a.c.M) g = fmaf(tb[k0 * EPI_LD + lane], w.dR, g);
                            if (k1 >= 0 && k1 < 32 && w.k + 1 < a.c.M) g = fmaf(tb[k1 * EPI_LD + lane], w.dL, g);
                            if (g != 0.f) atomicAdd(a.g_t_in + e, g);
                        }
                    }
                    __syncwarp();
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// dW: rows = (tap, channel) of the filters in blocks of 64 (two per tile),
// columns = BN output channels, K = (output position, m) in steps of 64
// (64 / Mp positions). Both operands MN-major, straight from S and dw^:
//   A  S at the input position each row block's tap reads (two boxes of 64
//      channels), 64 k-rows each;
//   B  dw^ at the output positions (BN / 64 boxes of 64 channels).
// Split-K over positions; every split adds its tile into g_W atomically
// (split 0 also adds the dead-neuron term qcoef * count[o]).
// ---------------------------------------------------------------------------
template <int BN>
__global__ void __launch_bounds__(CONV_THREADS, 1)
    k_conv_dw(const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapD, ConvGemmArgs a) {
    using Cfg = ConvCfg<BN, 2>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + Cfg::STAGES * Cfg::STAGE);
    uint64_t *empty = full + Cfg::STAGES;
    uint64_t *acc_full = empty + Cfg::STAGES;
    uint64_t *acc_empty = acc_full + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 2);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = a.n_row * a.n_col * a.n_split;
    const int Mp = a.Mp;
    const int kpos = 64 / Mp;        // positions per K step
    const int ncb = a.C_in >> 6;     // channel blocks per tap
    const int nrb = a.k * a.k * ncb; // row blocks of 64
    const int Ktot = a.k * a.k * a.C_in;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&acc_full[u], 1);
            tc::mbar_init(&acc_empty[u], CONV_NEPI);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // tile t -> (split, row tile, column tile); K steps [kt0, kt0 + nkt)
    auto decode = [&](int t, int &rt, int &ct, int &kt0, int &nkt) {
        const int per = a.n_row * a.n_col;
        const int sp = t / per, rem = t - sp * per;
        rt = rem / a.n_col;
        ct = rem - rt * a.n_col;
        kt0 = sp * a.kt_per_split;
        nkt = a.ktiles - kt0;
        if (nkt > a.kt_per_split) nkt = a.kt_per_split;
    };

    if (warp == 0) {
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                int rt, ct, kt0, nkt;
                decode(t, rt, ct, kt0, nkt);
                for (int i = 0; i < nkt; ++i, ++it) {
                    const int s = it % Cfg::STAGES;
                    const uint32_t ph = (it / Cfg::STAGES) & 1u;
                    if (!tc::mbar_wait(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full[s], (uint32_t)Cfg::STAGE);
                    const uint32_t st = tc::smem_u32(smem + s * Cfg::STAGE);
                    const int kt = kt0 + i;
                    for (int kp = 0; kp < kpos; ++kp) {
                        const int p = kt * kpos + kp;  // output position of these k-rows
                        int b, y, x;
                        const bool in = p < a.P_rows;
                        if (in) pos_decode(p, a.Ho, a.Wo, b, y, x);
                        // A: the two row blocks' taps at input positions
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int rb = 2 * rt + h;
                            int sx = 0, sy = 0, sbi = a.ni, cb = 0;
                            if (in && rb < nrb) {
                                const int tap = rb / ncb;
                                cb = rb - tap * ncb;
                                const int kh = tap / a.k, kw = tap - kh * a.k;
                                sx = x * a.stride + kw - a.pad;
                                sy = y * a.stride + kh - a.pad;
                                sbi = b;
                            }
                            tma_load_5d(st + h * 8192 + kp * Mp * 128, &mapS, &full[s], cb * 64, 0, sx, sy, sbi);
                        }
                        // B: dw^ of the output position, BN / 64 channel boxes
                        for (int g = 0; g < BN / 64; ++g)
                            tma_load_5d(st + Cfg::A_BYTES + g * 8192 + kp * Mp * 128, &mapD, &full[s],
                                        ct * BN + g * 64, 0, in ? x : 0, in ? y : 0, in ? b : a.ni);
                    }
                }
            }
            const uint32_t n_drain = it < (uint32_t)Cfg::STAGES ? it : (uint32_t)Cfg::STAGES;
            for (uint32_t i = it - n_drain; i < it; ++i)
                tc::mbar_wait(&full[i % Cfg::STAGES], (i / Cfg::STAGES) & 1u);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, true, true);
            uint32_t it = 0, j = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                int rt, ct, kt0, nkt;
                decode(t, rt, ct, kt0, nkt);
                const uint32_t buf = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait(&acc_empty[buf], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc = tmem + buf * BN;
                for (int i = 0; i < nkt; ++i, ++it) {
                    const int s = it % Cfg::STAGES;
                    const uint32_t ph = (it / Cfg::STAGES) & 1u;
                    if (!tc::mbar_wait(&full[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * Cfg::STAGE);
                    const uint32_t sbb = sa + Cfg::A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc::mma_bf16(acc, tc::sdesc_sw128_mn(sa + kk * 2048, 8192), tc::sdesc_sw128_mn(sbb + kk * 2048, 8192),
                                     idesc, (i > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_commit(&empty[s]);
                }
                if (ok) tc::mma_commit(&acc_full[buf]);
            }
        }
        __syncwarp();
    } else {
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const int r = quarter * 32 + lane;
        uint32_t j = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
            int rt, ct, kt0, nkt;
            decode(t, rt, ct, kt0, nkt);
            const uint32_t buf = j & 1u;
            if (!tc::mbar_wait_sleep(&acc_full[buf], (j >> 1) & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            const int kidx = rt * 128 + r;  // (tap, channel) of this lane
            const bool first = kt0 == 0;
            for (int cc = group; cc < BN / 32; cc += 2) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + buf * BN + cc * 32, v);
                if (kidx < Ktot) {
                    const int o0 = ct * BN + cc * 32;
#pragma unroll
                    for (int u = 0; u < 32; ++u) {
                        const float add = (first && a.count) ? a.qcoef * a.count[o0 + u] : 0.f;
                        atomicAdd(a.g_W + (long long)(o0 + u) * Ktot + kidx, v[u] + add);
                    }
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Binned operand generated on chip (the compact support of K_DSTD: each
// input spike has two nonzero grid weights among Mp). The binning writes
// one 8-byte record per input, rec[p][c] = (grid step k, bf16 pair (w at
// T_k, w at T_{k+1})), k = -128 when silent. Per K step the TMA producer
// copies the records the tile needs (64 per position and tap) into the stage;
// four generator warps then write each record's two nonzeros into the
// swizzled A tile that the tensor core reads. Each thread owns fixed columns
// of the tile, so before writing it erases the two entries it wrote the last
// time it used that stage (all stages start zeroed): 4 two-byte shared
// stores per input instead of 16 KB of operand per K step from L2.
// ---------------------------------------------------------------------------
constexpr int REC_SILENT = -128;

__global__ void __launch_bounds__(256) k_bin_rec(const float *__restrict__ t, long long n, LifConst c,
                                                 uint2 *__restrict__ rec) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const float x = __ldg(t + i);
        uint2 r = make_uint2((uint32_t)REC_SILENT, 0u);
        if (isfinite(x)) {
            const BinW w = bin_weights(c, x, false);
            if (w.k >= -1 && w.k < c.M) r = make_uint2((uint32_t)w.k, pack_bf16x2(w.wR, w.wL));
        }
        rec[i] = r;
    }
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int c, int x, int y,
                                            int b) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c), "r"(x), "r"(y), "r"(b), "r"(tc::smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void sts_u16(uint32_t addr, uint16_t v) {
    asm volatile("st.shared.u16 [%0], %1;" ::"r"(addr), "h"(v) : "memory");
}

// byte offset of element (row r, column c) of a 128-byte-swizzled tile of
// 128-byte rows (K-major: r = M/N row, c = k; MN-major: r = k, c = M/N)
__device__ __forceinline__ uint32_t sw128_off(int r, int c) {
    return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((((c >> 3) ^ (r & 7)) & 7) << 4) + (c & 7) * 2);
}

// Write one record's two grid weights into column c of the rows of one
// position (rows row0 + k, row0 + k + 1, grid steps below M), after erasing
// the two this thread wrote there before (old step kold).
__device__ __forceinline__ void gen_put(uint32_t tile, int row0, int c, int kold, uint2 r, int M) {
    if (kold != REC_SILENT) {
        if (kold >= 0) sts_u16(tile + sw128_off(row0 + kold, c), 0);
        if (kold + 1 < M) sts_u16(tile + sw128_off(row0 + kold + 1, c), 0);
    }
    const int k = (int)r.x;
    if (k != REC_SILENT) {
        if (k >= 0) sts_u16(tile + sw128_off(row0 + k, c), (uint16_t)(r.y & 0xffffu));
        if (k + 1 < M) sts_u16(tile + sw128_off(row0 + k + 1, c), (uint16_t)(r.y >> 16));
    }
}

// the same for an MN-major tile: the record's column c of atom h, k-rows
// kr0 + k and kr0 + k + 1
__device__ __forceinline__ void gen_put_mn(uint32_t tile, int kr0, int c, int kold, uint2 r, int M) {
    if (kold != REC_SILENT) {
        if (kold >= 0) sts_u16(tile + sw128_off(kr0 + kold, c), 0);
        if (kold + 1 < M) sts_u16(tile + sw128_off(kr0 + kold + 1, c), 0);
    }
    const int k = (int)r.x;
    if (k != REC_SILENT) {
        if (k >= 0) sts_u16(tile + sw128_off(kr0 + k, c), (uint16_t)(r.y & 0xffffu));
        if (k + 1 < M) sts_u16(tile + sw128_off(kr0 + k + 1, c), (uint16_t)(r.y >> 16));
    }
}

constexpr int GEN_WARPS = 4;
constexpr int GEN_THREADS = (2 + CONV_NEPI + GEN_WARPS) * 32;  // 448

// shared-memory plan of the generated-operand kernels: per stage the A tile,
// the B tile (unless resident) and the records; the stage count and the
// resident bytes are chosen on the host (ConvGemmArgs::nst, ::res_bytes)
template <int BN, bool RES>
struct GenFwdCfg {
    static constexpr int A_BYTES = 128 * 128;
    static constexpr int B_BYTES = RES ? 0 : BN * 128;
    static constexpr int R_BYTES = 2048;            // up to 4 positions x 64 records x 8 B
    static constexpr int STAGE = A_BYTES + B_BYTES + R_BYTES;
    static constexpr int MAX_STAGES = 8;
    static constexpr int PREV_BYTES = MAX_STAGES * 256 * 2;  // last grid step written, per stage and slot
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static __host__ __device__ int smem(int nst, int res_bytes) { return nst * STAGE + res_bytes + PREV_BYTES + 1024 + 256; }
};
constexpr int GEN_SMEM_MAX = 225 * 1024;

// Forward with the binned operand generated on chip. Warps: 0 TMA (records,
// and the filter tiles unless RES: then all of them once, resident), 1 MMA,
// 2-9 epilogue (w^ rows as k_conv_gemm), 10-13 generators.
template <int BN, bool RES>
__global__ void __launch_bounds__(GEN_THREADS, 1)
    k_conv_fwd_gen(const __grid_constant__ CUtensorMap mapR, const __grid_constant__ CUtensorMap mapB, ConvGemmArgs a) {
    using Cfg = GenFwdCfg<BN, RES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int NST = a.nst;
    uint8_t *bres = smem + NST * Cfg::STAGE;                           // resident filters (RES)
    int16_t *prevk = reinterpret_cast<int16_t *>(bres + a.res_bytes);
    uint64_t *full_t = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(prevk) + Cfg::PREV_BYTES);
    uint64_t *full_a = full_t + Cfg::MAX_STAGES;
    uint64_t *empty = full_a + Cfg::MAX_STAGES;
    uint64_t *acc_full = empty + Cfg::MAX_STAGES;
    uint64_t *acc_empty = acc_full + 2;
    uint64_t *bres_full = acc_empty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bres_full + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = a.n_row * a.n_col;
    const int Mp = a.Mp;
    const int ppt = 128 / Mp;
    const int ncb = a.C_in >> 6;

    // zero every stage's A tile and mark every slot unwritten
    for (int i = threadIdx.x; i < NST * (Cfg::A_BYTES / 16); i += blockDim.x) {
        const int st = i / (Cfg::A_BYTES / 16), off = i - st * (Cfg::A_BYTES / 16);
        reinterpret_cast<uint4 *>(smem + st * Cfg::STAGE)[off] = make_uint4(0u, 0u, 0u, 0u);
    }
    for (int i = threadIdx.x; i < Cfg::PREV_BYTES / 2; i += blockDim.x) prevk[i] = (int16_t)REC_SILENT;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            tc::mbar_init(&full_t[s], 1);
            tc::mbar_init(&full_a[s], GEN_WARPS);
            tc::mbar_init(&empty[s], 1);
        }
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&acc_full[u], 1);
            tc::mbar_init(&acc_empty[u], CONV_NEPI);
        }
        tc::mbar_init(bres_full, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the zeroed tiles, for the tensor core
    if (warp == 1) tc::tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            if (RES) {
                // every K slice of the filters of the single column tile, once
                tc::mbar_expect_tx(bres_full, (uint32_t)(a.ktiles * BN * 128));
                for (int kt = 0; kt < a.ktiles; ++kt) {
                    const int tap = kt / ncb, cb = kt - tap * ncb;
                    tc::tma_load_2d(tc::smem_u32(bres + kt * BN * 128), &mapB, bres_full, tap * a.C_in + cb * 64, 0);
                }
            }
            uint32_t it = 0;
            bool ok = true;
            const uint32_t tx = (uint32_t)(ppt * 512 + Cfg::B_BYTES);
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                const int rt = t / a.n_col, ct = t - rt * a.n_col;
                for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                    const int s = it % NST;
                    const uint32_t ph = (it / NST) & 1u;
                    if (!tc::mbar_wait(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full_t[s], tx);
                    const int tap = kt / ncb, cb = kt - tap * ncb;
                    const int kh = tap / a.k, kw = tap - kh * a.k;
                    const uint32_t st = tc::smem_u32(smem + s * Cfg::STAGE);
                    const uint32_t sr = st + Cfg::A_BYTES + Cfg::B_BYTES;
                    for (int pp = 0; pp < ppt; ++pp) {
                        int sx, sy, sb;
                        conv_src<0>(a, rt * ppt + pp, kh, kw, sx, sy, sb);
                        tma_load_4d(sr + pp * 512, &mapR, &full_t[s], 2 * cb * 64, sx, sy, sb);
                    }
                    if (!RES) tc::tma_load_2d(st + Cfg::A_BYTES, &mapB, &full_t[s], tap * a.C_in + cb * 64, ct * BN);
                }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i)
                tc::mbar_wait(&full_t[i % NST], (i / NST) & 1u);
            if (RES) tc::mbar_wait(bres_full, 0);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, false, false);
            uint32_t it = 0, j = 0;
            bool ok = true;
            if (RES && !tc::mbar_wait(bres_full, 0)) {
                conv_set_status(STATUS_TIMEOUT);
                ok = false;
            }
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                const uint32_t buf = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait(&acc_empty[buf], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc = tmem + buf * BN;
                for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                    const int s = it % NST;
                    const uint32_t ph = (it / NST) & 1u;
                    if (!tc::mbar_wait(&full_t[s], ph) || !tc::mbar_wait(&full_a[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * Cfg::STAGE);
                    const uint32_t sbb = RES ? tc::smem_u32(bres + kt * BN * 128) : sa + Cfg::A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc::mma_bf16(acc, tc::sdesc_sw128(sa + kk * 32), tc::sdesc_sw128(sbb + kk * 32), idesc,
                                     (kt > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_commit(&empty[s]);
                }
                if (ok) tc::mma_commit(&acc_full[buf]);
            }
        }
        __syncwarp();
    } else if (warp < 2 + CONV_NEPI) {
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const int r = quarter * 32 + lane;
        const int pp = (quarter * 32) / Mp;
        uint32_t j = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
            const int rt = t / a.n_col, ct = t - rt * a.n_col;
            const uint32_t buf = j & 1u;
            if (!tc::mbar_wait_sleep(&acc_full[buf], (j >> 1) & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            const int p = rt * ppt + pp;
            for (int cc = group; cc < BN / 32; cc += 2) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + buf * BN + cc * 32, v);
                if (p < a.P_rows) {
                    float *dst = a.what + ((long long)p * Mp + (r % Mp)) * a.C_out + ct * BN + cc * 32;
#pragma unroll
                    for (int u = 0; u < 32; u += 4)
                        *reinterpret_cast<float4 *>(dst + u) = make_float4(v[u], v[u + 1], v[u + 2], v[u + 3]);
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
        }
    } else {
        // generators: thread g owns slots g, g + 128, ... (slot = position
        // pp x 64 + channel c of the tile) in every stage
        const int g = threadIdx.x - (2 + CONV_NEPI) * 32;
        const int nslots = ppt * 64;
        uint32_t it = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
            for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                const int s = it % NST;
                const uint32_t ph = (it / NST) & 1u;
                if (!tc::mbar_wait(&full_t[s], ph)) {
                    conv_set_status(STATUS_TIMEOUT);
                    ok = false;
                    break;
                }
                uint8_t *st = smem + s * Cfg::STAGE;
                const uint32_t tile = tc::smem_u32(st);
                const uint2 *rec = reinterpret_cast<const uint2 *>(st + Cfg::A_BYTES + Cfg::B_BYTES);
                for (int slot = g; slot < nslots; slot += GEN_WARPS * 32) {
                    const int pp = slot >> 6, c = slot & 63;
                    const uint2 r = rec[slot];
                    int16_t *pk = prevk + s * 256 + slot;
                    gen_put(tile, pp * Mp, c, (int)*pk, r, a.c.M);
                    *pk = (int16_t)(int)r.x;
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&full_a[s]);
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// dW with the binned operand generated on chip: a CTA tile is G row tiles
// (128 filter rows (tap, channel) each, two 64-channel row blocks) by BN
// output channels over a range of K = (output position, m). Per K step it
// stages one dw^ tile (MN-major, by TMA) and the records of the G row
// tiles' inputs, the generators write the G MN-major A tiles, and G MMAs
// (one TMEM accumulator each) reuse the dw^ tile. Split-K over positions;
// each split adds its tiles into g_W atomically (split 0 also the
// dead-neuron term).
// ---------------------------------------------------------------------------
constexpr int DWG_MAX_G = 8;
constexpr int DWG_MAX_STAGES = 4;

template <int BN>
struct GenDwCfg {
    static constexpr int B_BYTES = BN * 128;
    static __host__ __device__ int stage(int G, int kpos) { return G * (128 * 128 + 2 * kpos * 512) + B_BYTES; }
    static __host__ __device__ int prev_bytes(int nst, int G, int kpos) { return nst * G * 128 * kpos * 2; }
    static __host__ __device__ int smem(int nst, int G, int kpos) {
        return nst * stage(G, kpos) + prev_bytes(nst, G, kpos) + 1024 + 256;
    }
};

template <int BN>
__global__ void __launch_bounds__(GEN_THREADS, 1)
    k_conv_dw_gen(const __grid_constant__ CUtensorMap mapR, const __grid_constant__ CUtensorMap mapD, ConvGemmArgs a) {
    using Cfg = GenDwCfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int G = a.groups, NST = a.nst;
    const int Mp = a.Mp;
    const int kpos = 64 / Mp;
    const int STG = Cfg::stage(G, kpos);
    const int a_bytes = G * 128 * 128;
    const int slots = G * 128 * kpos;                 // (row tile, row block, position, channel)
    int16_t *prevk = reinterpret_cast<int16_t *>(smem + NST * STG);
    uint64_t *full_t = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(prevk) + Cfg::prev_bytes(NST, G, kpos));
    uint64_t *full_a = full_t + DWG_MAX_STAGES;
    uint64_t *empty = full_a + DWG_MAX_STAGES;
    uint64_t *acc_full = empty + DWG_MAX_STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_grp = a.n_row;                        // row groups of G row tiles
    const int ntiles = n_grp * a.n_col * a.n_split;
    const int ncb = a.C_in >> 6;
    const int nrb = a.k * a.k * ncb;
    const int Ktot = a.k * a.k * a.C_in;
    uint32_t tcols = 32;
    while ((int)tcols < G * BN) tcols <<= 1;

    for (int i = threadIdx.x; i < NST * (a_bytes / 16); i += blockDim.x) {
        const int st = i / (a_bytes / 16), off = i - st * (a_bytes / 16);
        reinterpret_cast<uint4 *>(smem + st * STG)[off] = make_uint4(0u, 0u, 0u, 0u);
    }
    for (int i = threadIdx.x; i < NST * slots; i += blockDim.x) prevk[i] = (int16_t)REC_SILENT;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            tc::mbar_init(&full_t[s], 1);
            tc::mbar_init(&full_a[s], GEN_WARPS);
            tc::mbar_init(&empty[s], 1);
        }
        tc::mbar_init(acc_full, 1);
        tc::mbar_init(acc_empty, CONV_NEPI);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (warp == 1) tc::tmem_alloc(tmem_slot, tcols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    auto decode = [&](int t, int &rg, int &ct, int &kt0, int &nkt) {
        const int per = n_grp * a.n_col;
        const int sp = t / per, rem = t - sp * per;
        rg = rem / a.n_col;
        ct = rem - rg * a.n_col;
        kt0 = sp * a.kt_per_split;
        nkt = a.ktiles - kt0;
        if (nkt > a.kt_per_split) nkt = a.kt_per_split;
    };

    if (warp == 0) {
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            const uint32_t tx = (uint32_t)(G * 2 * kpos * 512 + Cfg::B_BYTES);
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                for (int i = 0; i < nkt; ++i, ++it) {
                    const int s = it % NST;
                    const uint32_t ph = (it / NST) & 1u;
                    if (!tc::mbar_wait(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full_t[s], tx);
                    const uint32_t st = tc::smem_u32(smem + s * STG);
                    const uint32_t sr = st + a_bytes + Cfg::B_BYTES;
                    const int kt = kt0 + i;
                    for (int kp = 0; kp < kpos; ++kp) {
                        const int p = kt * kpos + kp;
                        const bool in = p < a.P_rows;
                        int b = 0, y = 0, x = 0;
                        if (in) pos_decode(p, a.Ho, a.Wo, b, y, x);
                        for (int u = 0; u < 2 * G; ++u) {
                            const int rb = rg * 2 * G + u;
                            int sx = 0, sy = 0, sbi = a.ni, cb = 0;
                            if (in && rb < nrb) {
                                const int tap = rb / ncb;
                                cb = rb - tap * ncb;
                                const int kh = tap / a.k, kw = tap - kh * a.k;
                                sx = x * a.stride + kw - a.pad;
                                sy = y * a.stride + kh - a.pad;
                                sbi = b;
                            }
                            tma_load_4d(sr + (u * kpos + kp) * 512, &mapR, &full_t[s], 2 * cb * 64, sx, sy, sbi);
                        }
                        for (int gq = 0; gq < BN / 64; ++gq)
                            tma_load_5d(st + a_bytes + gq * 8192 + kp * Mp * 128, &mapD, &full_t[s], ct * BN + gq * 64,
                                        0, in ? x : 0, in ? y : 0, in ? b : a.ni);
                    }
                }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i) tc::mbar_wait(&full_t[i % NST], (i / NST) & 1u);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, true, true);
            uint32_t it = 0, j = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                if (j >= 1) {
                    if (!tc::mbar_wait(acc_empty, (j - 1) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                for (int i = 0; i < nkt; ++i, ++it) {
                    const int s = it % NST;
                    const uint32_t ph = (it / NST) & 1u;
                    if (!tc::mbar_wait(&full_t[s], ph) || !tc::mbar_wait(&full_a[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * STG);
                    const uint32_t sbb = sa + a_bytes;
                    for (int gi = 0; gi < G; ++gi) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc::mma_bf16(tmem + gi * BN, tc::sdesc_sw128_mn(sa + gi * 16384 + kk * 2048, 8192),
                                         tc::sdesc_sw128_mn(sbb + kk * 2048, 8192), idesc, (i > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(&empty[s]);
                }
                if (ok) tc::mma_commit(acc_full);
            }
        }
        __syncwarp();
    } else if (warp < 2 + CONV_NEPI) {
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const int r = quarter * 32 + lane;
        uint32_t j = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
            int rg, ct, kt0, nkt;
            decode(t, rg, ct, kt0, nkt);
            if (!tc::mbar_wait_sleep(acc_full, j & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            const bool first = kt0 == 0;
            for (int gi = 0; gi < G; ++gi) {
                const int kidx = (rg * G + gi) * 128 + r;
                for (int cc = group; cc < BN / 32; cc += 2) {
                    float v[32];
                    tc::tmem_ld32(tmem + lane_base + gi * BN + cc * 32, v);
                    if (kidx < Ktot) {
                        const int o0 = ct * BN + cc * 32;
#pragma unroll
                        for (int u = 0; u < 32; ++u) {
                            const float add = (first && a.count) ? a.qcoef * a.count[o0 + u] : 0.f;
                            atomicAdd(a.g_W + (long long)(o0 + u) * Ktot + kidx, v[u] + add);
                        }
                    }
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(acc_empty);
        }
    } else {
        const int g = threadIdx.x - (2 + CONV_NEPI) * 32;
        uint32_t it = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
            int rg, ct, kt0, nkt;
            decode(t, rg, ct, kt0, nkt);
            for (int i = 0; i < nkt; ++i, ++it) {
                const int s = it % NST;
                const uint32_t ph = (it / NST) & 1u;
                if (!tc::mbar_wait(&full_t[s], ph)) {
                    conv_set_status(STATUS_TIMEOUT);
                    ok = false;
                    break;
                }
                uint8_t *st = smem + s * STG;
                const uint32_t tile0 = tc::smem_u32(st);
                const uint2 *rec = reinterpret_cast<const uint2 *>(st + a_bytes + Cfg::B_BYTES);
                for (int slot = g; slot < slots; slot += GEN_WARPS * 32) {
                    // slot = ((u = 2 row tile + block) kpos + kp) 64 + c
                    const int c = slot & 63, q = slot >> 6;
                    const int kp = q % kpos, u = q / kpos;
                    const uint2 r = rec[slot];
                    int16_t *pk = prevk + s * slots + slot;
                    gen_put_mn(tile0 + (u >> 1) * 16384 + (u & 1) * 8192, kp * Mp, c, (int)*pk, r, a.c.M);
                    *pk = (int16_t)(int)r.x;
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&full_a[s]);
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, tcols);
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                             const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                             CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeFn conv_encode() {
    static EncodeFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeFn>(p);
    });
    return fn;
}

// activation [ni][h][w][Mp][C] bf16 as a 5-D map (C, Mp, w, h, ni), boxes of
// (64, Mp, 1, 1, 1), 128-byte swizzle, zeros outside
static bool map_act(CUtensorMap *m, const void *ptr, int ni, int h, int w, int Mp, int C) {
    EncodeFn enc = conv_encode();
    if (!enc) return false;
    cuuint64_t dims[5] = {(cuuint64_t)C, (cuuint64_t)Mp, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)ni};
    cuuint64_t strides[4] = {(cuuint64_t)C * 2, (cuuint64_t)Mp * C * 2, (cuuint64_t)w * Mp * C * 2,
                             (cuuint64_t)h * w * Mp * C * 2};
    cuuint32_t box[5] = {64, (cuuint32_t)Mp, 1, 1, 1};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// rows x cols bf16 matrix, boxes of box_rows x 64
static bool map_mat(CUtensorMap *m, const void *ptr, int rows, int cols, int box_rows) {
    EncodeFn enc = conv_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static int pick_bn(int n) { return (n % 256 == 0) ? 256 : ((n % 128 == 0) ? 128 : 64); }

// records [ni][h][w][C] of 8 bytes as a 4-D map of 32-bit words (2C, w, h,
// ni), boxes of 64 records of one position, no swizzle, zeros outside
static bool map_rec(CUtensorMap *m, const void *ptr, int ni, int h, int w, int C) {
    EncodeFn enc = conv_encode();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)2 * C, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)ni};
    cuuint64_t strides[3] = {(cuuint64_t)C * 8, (cuuint64_t)w * C * 8, (cuuint64_t)h * w * C * 8};
    cuuint32_t box[4] = {128, 1, 1, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, bool RES>
static cudaError_t launch_fwd_gen_bn(const CUtensorMap &mR, const CUtensorMap &mB, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = GenFwdCfg<BN, RES>;
    const int fixed = a.res_bytes + Cfg::PREV_BYTES + 1024 + 256;
    int nst = (GEN_SMEM_MAX - fixed) / Cfg::STAGE;
    if (nst > Cfg::MAX_STAGES) nst = Cfg::MAX_STAGES;
    if (nst < 2) return cudaErrorInvalidConfiguration;
    a.nst = nst;
    const int smem = Cfg::smem(nst, a.res_bytes);
    cudaError_t e = cudaFuncSetAttribute(k_conv_fwd_gen<BN, RES>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_fwd_gen<BN, RES><<<grid, GEN_THREADS, smem, st>>>(mR, mB, a);
    return cudaGetLastError();
}

template <int BN>
static cudaError_t launch_dw_gen_bn(const CUtensorMap &mR, const CUtensorMap &mD, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = GenDwCfg<BN>;
    const int kpos = 64 / a.Mp;
    int nst = DWG_MAX_STAGES;
    while (nst > 2 && Cfg::smem(nst, a.groups, kpos) > GEN_SMEM_MAX) --nst;
    if (Cfg::smem(nst, a.groups, kpos) > GEN_SMEM_MAX) return cudaErrorInvalidConfiguration;
    a.nst = nst;
    const int smem = Cfg::smem(nst, a.groups, kpos);
    cudaError_t e = cudaFuncSetAttribute(k_conv_dw_gen<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col * a.n_split;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_dw_gen<BN><<<grid, GEN_THREADS, smem, st>>>(mR, mD, a);
    return cudaGetLastError();
}

template <int BN, int MODE>
static cudaError_t launch_gemm_bn(const CUtensorMap &mA, const CUtensorMap &mB, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = ConvCfg<BN, MODE>;
    cudaError_t e = cudaFuncSetAttribute(k_conv_gemm<BN, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_gemm<BN, MODE><<<grid, CONV_THREADS, Cfg::SMEM, st>>>(mA, mB, a);
    return cudaGetLastError();
}

template <int BN>
static cudaError_t launch_dw_bn(const CUtensorMap &mS, const CUtensorMap &mD, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = ConvCfg<BN, 2>;
    cudaError_t e = cudaFuncSetAttribute(k_conv_dw<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col * a.n_split;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_dw<BN><<<grid, CONV_THREADS, Cfg::SMEM, st>>>(mS, mD, a);
    return cudaGetLastError();
}

static ConvGemmArgs base_args(const ConvGeom &g, int ni, const LifConst &c) {
    ConvGemmArgs a{};
    a.ni = ni;
    a.H = g.H;
    a.W = g.W;
    a.C_in = g.C;
    a.Ho = g.Ho;
    a.Wo = g.Wo;
    a.k = g.k;
    a.stride = g.s;
    a.pad = g.p;
    a.Mp = c.Mp;
    a.c = c;
    return a;
}

}  // namespace

bool conv_implicit_supported(const ConvGeom &g, int C_out, int Mp) {
    return g.C % 64 == 0 && C_out % 64 == 0 && (Mp == 32 || Mp == 64 || Mp == 128) && g.k <= 7 &&
           g.C * g.k * g.k <= 65535 && C_out * g.k * g.k <= 65535;
}

cudaError_t launch_bin_pmc(const float *t, long long P, int C, const LifConst &c, __nv_bfloat16 *S, cudaStream_t st) {
    if (C % 8 != 0) return cudaErrorInvalidValue;
    const long long n = P * (C / 8);
    long long blocks = (n + 255) / 256;
    const long long cap = 8ll * conv_num_sms();
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    k_bin_pmc<<<(unsigned)blocks, 256, 0, st>>>(t, P, C, c, S);
    return cudaGetLastError();
}

cudaError_t launch_dwhat_pmc(const float *t_out, const int *q, const float *s, const float *vdot, const float *g_up,
                             long long P, int C, const LifConst &c, __nv_bfloat16 *D, float *count,
                             cudaStream_t st) {
    if (C % 8 != 0 || C / 8 > 256) return cudaErrorInvalidValue;
    const int groups = C / 8;
    const int per_blk = 256 / groups;
    long long blocks = (P + per_blk - 1) / per_blk;
    const long long cap = 8ll * conv_num_sms();
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    k_dwhat_pmc<<<(unsigned)blocks, 256, 0, st>>>(t_out, q, s, vdot, g_up, P, C, c, D, count);
    return cudaGetLastError();
}

cudaError_t launch_filters_t(const float *W, int C_out, int T, int C_in, __nv_bfloat16 *Wt, cudaStream_t st) {
    const long long n = (long long)C_out * T * C_in;
    long long blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    k_filters_t<<<(unsigned)blocks, 256, 0, st>>>(W, C_out, T, C_in, Wt);
    return cudaGetLastError();
}

// forward contraction of ni images: S [ni H W][Mp][C_in], Wf [C_out][k k C_in]
// -> w^ [ni Ho Wo][Mp][C_out]
cudaError_t launch_conv_fwd_gemm(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                                 const __nv_bfloat16 *Wf, float *what, cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    const int BN = pick_bn(C_out);
    a.n_row = (a.P_rows + (128 / c.Mp) - 1) / (128 / c.Mp);
    a.n_col = C_out / BN;
    a.ktiles = g.k * g.k * (g.C / 64);
    a.what = what;
    CUtensorMap mA, mB;
    if (!map_act(&mA, S, ni, g.H, g.W, c.Mp, g.C) || !map_mat(&mB, Wf, C_out, g.k * g.k * g.C, BN))
        return cudaErrorInvalidValue;
    switch (BN) {
        case 256: return launch_gemm_bn<256, 0>(mA, mB, a, st);
        case 128: return launch_gemm_bn<128, 0>(mA, mB, a, st);
        default: return launch_gemm_bn<64, 0>(mA, mB, a, st);
    }
}

// dS of ni images with the input-time gradient: dw^ [ni Ho Wo][Mp][C_out],
// Wt [C_in][k k C_out], t_in [ni H W][C_in] -> g_t_in (zeroed first)
cudaError_t launch_conv_ds_gemm(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *dW_hat,
                                const __nv_bfloat16 *Wt, const float *t_in, float *g_t_in, cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.H * g.W;
    const int BN = pick_bn(g.C);
    a.n_row = (a.P_rows + (128 / c.Mp) - 1) / (128 / c.Mp);
    a.n_col = g.C / BN;
    a.ktiles = g.k * g.k * (C_out / 64);
    a.t_in = t_in;
    a.g_t_in = g_t_in;
    cudaError_t e = cudaMemsetAsync(g_t_in, 0, sizeof(float) * (size_t)a.P_rows * g.C, st);
    if (e != cudaSuccess) return e;
    CUtensorMap mA, mB;
    if (!map_act(&mA, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out) || !map_mat(&mB, Wt, g.C, g.k * g.k * C_out, BN))
        return cudaErrorInvalidValue;
    switch (BN) {
        case 256: return launch_gemm_bn<256, 1>(mA, mB, a, st);
        case 128: return launch_gemm_bn<128, 1>(mA, mB, a, st);
        default: return launch_gemm_bn<64, 1>(mA, mB, a, st);
    }
}

// dW over ni images added into g_W [C_out][k k C_in] (zeroed by the caller
// before the first chunk); count (may be null) adds qcoef * count[o] once
cudaError_t launch_conv_dw_gemm(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                                const __nv_bfloat16 *dW_hat, const float *count, float qcoef, float *g_W,
                                cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    const int BN = pick_bn(C_out);
    const int Ktot = g.k * g.k * g.C;
    a.n_row = (Ktot / 64 + 1) / 2;
    a.n_col = C_out / BN;
    const int kpos = 64 / c.Mp;
    a.ktiles = (a.P_rows + kpos - 1) / kpos;
    // split-K: about two tiles per SM, at least 16 K steps each
    const int tiles = a.n_row * a.n_col;
    int splits = (2 * conv_num_sms() + tiles - 1) / tiles;
    const int max_splits = (a.ktiles + 15) / 16;
    if (splits > max_splits) splits = max_splits;
    if (splits < 1) splits = 1;
    a.kt_per_split = (a.ktiles + splits - 1) / splits;
    a.n_split = (a.ktiles + a.kt_per_split - 1) / a.kt_per_split;
    a.g_W = g_W;
    a.count = count;
    a.qcoef = qcoef;
    CUtensorMap mS, mD;
    if (!map_act(&mS, S, ni, g.H, g.W, c.Mp, g.C) || !map_act(&mD, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out))
        return cudaErrorInvalidValue;
    switch (BN) {
        case 256: return launch_dw_bn<256>(mS, mD, a, st);
        case 128: return launch_dw_bn<128>(mS, mD, a, st);
        default: return launch_dw_bn<64>(mS, mD, a, st);
    }
}

cudaError_t launch_bin_rec(const float *t, long long n, const LifConst &c, uint2 *rec, cudaStream_t st) {
    long long blocks = (n + 255) / 256;
    const long long cap = 8ll * conv_num_sms();
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    k_bin_rec<<<(unsigned)blocks, 256, 0, st>>>(t, n, c, rec);
    return cudaGetLastError();
}

// forward contraction with the binned operand generated on chip from the
// records rec [ni H W][C_in]; filters resident in shared memory when all of
// them fit (one column tile, at most 144 KB)
cudaError_t launch_conv_fwd_gen(const ConvGeom &g, int ni, int C_out, const LifConst &c, const uint2 *rec,
                                const __nv_bfloat16 *Wf, float *what, cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    const int BN = pick_bn(C_out);
    a.n_row = (a.P_rows + (128 / c.Mp) - 1) / (128 / c.Mp);
    a.n_col = C_out / BN;
    a.ktiles = g.k * g.k * (g.C / 64);
    a.what = what;
    const long long res = (long long)a.ktiles * BN * 128;
    const bool resident = a.n_col == 1 && res <= 144 * 1024;
    a.res_bytes = resident ? (int)res : 0;
    CUtensorMap mR, mB;
    if (!map_rec(&mR, rec, ni, g.H, g.W, g.C) || !map_mat(&mB, Wf, C_out, g.k * g.k * g.C, BN))
        return cudaErrorInvalidValue;
    if (resident) {
        switch (BN) {
            case 256: return launch_fwd_gen_bn<256, true>(mR, mB, a, st);
            case 128: return launch_fwd_gen_bn<128, true>(mR, mB, a, st);
            default: return launch_fwd_gen_bn<64, true>(mR, mB, a, st);
        }
    }
    switch (BN) {
        case 256: return launch_fwd_gen_bn<256, false>(mR, mB, a, st);
        case 128: return launch_fwd_gen_bn<128, false>(mR, mB, a, st);
        default: return launch_fwd_gen_bn<64, false>(mR, mB, a, st);
    }
}

// dW over ni images with the binned operand generated on chip from rec,
// added into g_W (zeroed by the caller before the first chunk)
cudaError_t launch_conv_dw_gen(const ConvGeom &g, int ni, int C_out, const LifConst &c, const uint2 *rec,
                               const __nv_bfloat16 *dW_hat, const float *count, float qcoef, float *g_W,
                               cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    const int BN = pick_bn(C_out);
    const int Ktot = g.k * g.k * g.C;
    const int row_tiles = (Ktot / 64 + 1) / 2;
    int gmax = 512 / BN;
    if (gmax > DWG_MAX_G) gmax = DWG_MAX_G;
    const int kpos = 64 / c.Mp;
    // shared memory: at least two stages of G tiles
    auto smem2 = [&](int G) {
        return BN == 256 ? GenDwCfg<256>::smem(2, G, kpos)
                         : (BN == 128 ? GenDwCfg<128>::smem(2, G, kpos) : GenDwCfg<64>::smem(2, G, kpos));
    };
    while (gmax > 1 && smem2(gmax) > GEN_SMEM_MAX) --gmax;
    const int ngrp = (row_tiles + gmax - 1) / gmax;
    a.groups = (row_tiles + ngrp - 1) / ngrp;     // balanced groups
    a.n_row = (row_tiles + a.groups - 1) / a.groups;
    a.n_col = C_out / BN;
    a.ktiles = (a.P_rows + kpos - 1) / kpos;
    const int tiles = a.n_row * a.n_col;
    int splits = (2 * conv_num_sms() + tiles - 1) / tiles;
    const int max_splits = (a.ktiles + 15) / 16;
    if (splits > max_splits) splits = max_splits;
    if (splits < 1) splits = 1;
    a.kt_per_split = (a.ktiles + splits - 1) / splits;
    a.n_split = (a.ktiles + a.kt_per_split - 1) / a.kt_per_split;
    a.g_W = g_W;
    a.count = count;
    a.qcoef = qcoef;
    CUtensorMap mR, mD;
    if (!map_rec(&mR, rec, ni, g.H, g.W, g.C) || !map_act(&mD, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out))
        return cudaErrorInvalidValue;
    switch (BN) {
        case 256: return launch_dw_gen_bn<256>(mR, mD, a, st);
        case 128: return launch_dw_gen_bn<128>(mR, mD, a, st);
        default: return launch_dw_gen_bn<64>(mR, mD, a, st);
    }
}

}  // namespace dstd
