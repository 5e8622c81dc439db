// Convolutional DSTD layer as implicit GEMMs on sm_103a (bf16 operands,
// tcgen05), with no im2col operand and no binned array in memory.
//
// Layouts (a chunk of whole images, NHWC positions p = (b*H + y)*W + x):
//   rec   [P_in][C_in]       8 B   per input spike: grid step k and the bf16
//                                  pair of its two weights (Eq. DSTD_kernel)
//   w^    [P_out][C_out][Mp] fp32  the forward contraction (Eq. DSTD), the
//                                  Mp grid steps of a neuron contiguous
//   dw^   [P_out][Mp][C_out] bf16  dC/dw^ (implicit-function theorem)
//   Wf    [C_out][k k C_in]  bf16  filters, taps (kh, kw) then channels
//   Wt    [C_in][k k C_out]  bf16  the same filters transposed
//
//   forward  w^[(p, m), o]  = sum_{tap, c} S[(p + tap), m, c] Wf[o, tap, c]:
//            the binned operand S is generated in shared memory from the
//            records of the inputs each tap reads (two nonzeros per input)
//   dS       dS[(p', m), c] = sum_{tap, o} dw^[(p' - tap) / s, m, o] Wt[c, tap, o]
//            (the transposed convolution; one TMA box of a 5-D tensor map
//            (channel, m, x, y, b) per position and tap, coordinates outside
//            the image or off the stride grid read zeros), consumed in the
//            epilogue: dC/dt_j = sum_{m in {k, k+1}} dS[(p', m), c] ds_jm/dt_j
//   dW       dW[o, tap, c]  = sum_{(p, m)} dw^[(p, m), o] S[(p + tap), m, c]
//            (both operands MN-major, S generated on chip, split-K)
//
// One thread issues tcgen05.mma (M = 128, N = BN <= 256, K = 16) into TMEM
// accumulators. Every mbarrier wait is bounded; an expired wait sets this
// unit's status word, the role stops, and the CTA still frees its TMEM.
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
// dC/dw^_{p,m,o} = -g K(t - T_m) / v^'(t) for m <= q (0 after the spike's
// interval and for silent neurons), g = upstream + dT/dt, into [P][Mp][C_out]
// bf16. A warp writes one position (or one 128-channel segment of it) at a
// time, a contiguous block of its rows: a thread takes 4 consecutive neurons
// and every R-th grid step (R = 32 / (channels / 4)). C_out is at most 128 or
// a multiple of 128. With C_out = 64 the block is built in the warp's shared
// buffer and written with one bulk copy; otherwise every store instruction
// writes whole lines (streaming stores).
// K(x), x = t - T_m, falls along m by the factors e^{av dt}, e^{aI dt}; a
// thread steps R grid steps at a time. The spike's own
// bin and the one before it (x < 2 dt, where (e^{-av x} - e^{-aI x}) / lam
// cancels) take the accurate form. Silent neurons are counted per output
// channel (the thread of row phase 0 of a channel group adds its counts).
// ---------------------------------------------------------------------------
#ifndef DWHAT_NPT
#define DWHAT_NPT 4
#endif
// NPT consecutive bf16 of one row, streamed (evict-first)
// (SHARED: p is in shared memory, a plain store; else a streaming global store)
template <int NPT, bool SHARED>
__device__ __forceinline__ void dwhat_store(__nv_bfloat16 *p, const float (&v)[NPT]) {
    if constexpr (NPT == 8) {
        const uint4 x = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                                   pack_bf16x2(v[6], v[7]));
        if constexpr (SHARED) *reinterpret_cast<uint4 *>(p) = x;
        else __stcs(reinterpret_cast<uint4 *>(p), x);
    } else {
        const uint2 x = make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
        if constexpr (SHARED) *reinterpret_cast<uint2 *>(p) = x;
        else __stcs(reinterpret_cast<uint2 *>(p), x);
    }
}

template <int NPT, bool BULK>
__global__ void __launch_bounds__(256) k_dwhat_pmc(const float *__restrict__ t_out, const int *__restrict__ qv,
                                                   const float *__restrict__ sv, const float *__restrict__ vd,
                                                   const float *__restrict__ g_up, long long P, int C, LifConst c,
                                                   __nv_bfloat16 *__restrict__ D, float *count) {
    const int nseg = (C + 32 * NPT - 1) / (32 * NPT);  // segments of a position
    constexpr int SEGC = 32 * NPT;                    // channels of a segment: one per lane x NPT
    const int groups = (C < SEGC ? C : SEGC) / NPT;   // NPT-neuron groups of a segment (<= 32)
    const int R = 32 / groups;                        // rows of a warp store
    const int lane = threadIdx.x & 31;
    if (lane >= R * groups) return;                   // idle lanes (C = 192)
    const int g = lane % groups, r = lane / groups;
    const int wpb = blockDim.x >> 5;
    // BULK (C <= 32 NPT, one segment): a position's Mp x C block is built in
    // this warp's shared buffer and written with one bulk copy
    extern __shared__ __align__(128) uint8_t dw_smem[];
    __nv_bfloat16 *wbuf = reinterpret_cast<__nv_bfloat16 *>(dw_smem) + (threadIdx.x >> 5) * c.Mp * C;
    bool pending = false;
    const long long wid = (long long)blockIdx.x * wpb + (threadIdx.x >> 5), nw = (long long)gridDim.x * wpb;
    float cnt[NPT];
#pragma unroll
    for (int u = 0; u < NPT; ++u) cnt[u] = 0.f;
    const float fv = __expf(c.av * c.dt * R), fI = __expf(c.aI * c.dt * R);
    int c0 = g * NPT;
    for (long long item = wid; item < P * nseg; item += nw) {
        long long p = item;
        if (nseg > 1) {
            p = item / nseg;
            const int seg = (int)(item - p * nseg);
            // counts of the previous segment's channels
            if (r == 0) {
#pragma unroll
                for (int u = 0; u < NPT; ++u)
                    if (cnt[u] != 0.f) {
                        if (count) atomicAdd(&count[c0 + u], cnt[u]);
                        cnt[u] = 0.f;
                    }
            }
            c0 = seg * SEGC + g * NPT;
        }
        // every input of the 8 neurons first, without branches
        int q[NPT];
        float tt[NPT], gu[NPT], vv[NPT], ss[NPT];
        const long long idx0 = p * C + c0;
#pragma unroll
        for (int u = 0; u < NPT; ++u) {
            q[u] = __ldg(qv + idx0 + u);
            tt[u] = __ldg(t_out + idx0 + u);
            gu[u] = g_up ? __ldg(g_up + idx0 + u) : 0.f;
            vv[u] = __ldg(vd + idx0 + u);
            ss[u] = __ldg(sv + idx0 + u);
        }
        // per neuron: the recurrence terms at this thread's first row r, the
        // two accurate rows, and the band [m_lo, m_hi] holding them
        float a[NPT], b[NPT], K1[NPT], K0[NPT];
        int m_lo = c.Mp, m_hi = -1;
#pragma unroll
        for (int u = 0; u < NPT; ++u) {
            a[u] = b[u] = K1[u] = K0[u] = 0.f;
            if (q[u] < c.M) {
                float pv, pg;
                penalty_T(c, tt[u], pv, pg);
                const float coef = -(gu[u] + pg) / vv[u];
                const float s0 = ss[u];
                const float x = s0 + (float)(q[u] - r) * c.dt;  // t - T_r
                K0[u] = coef * kernel_K(c, s0);
                K1[u] = coef * kernel_K(c, s0 + c.dt);
                if (c.lam_zero) {
                    a[u] = coef * __expf(-c.av * x);
                    b[u] = x;
                } else {
                    a[u] = coef * c.inv_lam * __expf(-c.av * x);
                    b[u] = coef * c.inv_lam * __expf(-c.aI * x);
                }
                m_lo = min(m_lo, q[u] - 1);
                m_hi = max(m_hi, q[u]);
            } else {
                if (r == 0) cnt[u] += 1.f;
                q[u] = -1;
            }
        }
        if (BULK && pending) {  // the previous position's copy has read the buffer
            if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
            __syncwarp();
        }
        __nv_bfloat16 *dst = (BULK ? wbuf : D + p * (long long)c.Mp * C) + c0;
        const int step = C;
        const float dtR = c.dt * R;
        int m = r;
        if (c.lam_zero) {
            for (; m < m_lo; m += R) {
                float v[NPT];
#pragma unroll
                for (int u = 0; u < NPT; ++u) {
                    v[u] = a[u] * b[u];
                    a[u] *= fv;
                    b[u] -= dtR;
                }
                dwhat_store<NPT, BULK>(dst + (long long)m * step, v);
            }
            for (; m <= m_hi; m += R) {
                float v[NPT];
#pragma unroll
                for (int u = 0; u < NPT; ++u) {
                    const float d = a[u] * b[u];
                    v[u] = m < q[u] - 1 ? d : (m == q[u] - 1 ? K1[u] : (m == q[u] ? K0[u] : 0.f));
                    a[u] *= fv;
                    b[u] -= dtR;
                }
                dwhat_store<NPT, BULK>(dst + (long long)m * step, v);
            }
        } else {
            for (; m < m_lo; m += R) {
                float v[NPT];
#pragma unroll
                for (int u = 0; u < NPT; ++u) {
                    v[u] = a[u] - b[u];
                    a[u] *= fv;
                    b[u] *= fI;
                }
                dwhat_store<NPT, BULK>(dst + (long long)m * step, v);
            }
            for (; m <= m_hi; m += R) {
                float v[NPT];
#pragma unroll
                for (int u = 0; u < NPT; ++u) {
                    const float d = a[u] - b[u];
                    v[u] = m < q[u] - 1 ? d : (m == q[u] - 1 ? K1[u] : (m == q[u] ? K0[u] : 0.f));
                    a[u] *= fv;
                    b[u] *= fI;
                }
                dwhat_store<NPT, BULK>(dst + (long long)m * step, v);
            }
        }
        if (m < c.Mp) {
            float z[NPT];
#pragma unroll
            for (int u = 0; u < NPT; ++u) z[u] = 0.f;
            for (; m < c.Mp; m += R) dwhat_store<NPT, BULK>(dst + (long long)m * step, z);
        }
        if (BULK) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
                asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                                 D + p * (long long)c.Mp * C),
                             "r"(tc::smem_u32(wbuf)), "r"((uint32_t)(c.Mp * C * 2))
                             : "memory");
                asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            }
            pending = true;
        }
    }
    if (BULK && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    if (count && r == 0) {
#pragma unroll
        for (int u = 0; u < NPT; ++u)
            if (cnt[u] != 0.f) atomicAdd(&count[c0 + u], cnt[u]);
    }
}

// Filters [C_out][T][C_in] fp32 -> Wt [C_pad][T][C_out] bf16 (T = k k taps;
// rows C_in .. C_pad - 1 zero).
__global__ void k_filters_t(const float *__restrict__ W, int C_out, int T, int C_in, int C_pad,
                            __nv_bfloat16 *__restrict__ Wt) {
    const long long n = (long long)C_out * T * C_pad;
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int o = (int)(idx % C_out);
        const long long r = idx / C_out;
        const int tap = (int)(r % T), ci = (int)(r / T);
        Wt[idx] = __float2bfloat16_rn(ci < C_in ? W[((long long)o * T + tap) * C_in + ci] : 0.f);
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
constexpr int EPI_LD = 33;                            // per-warp transpose buffer row stride (floats)

// Geometry of one implicit-GEMM launch over a chunk of ni images.
struct ConvGemmArgs {
    int ni;              // images in the chunk
    int H, W, C_in;      // layer input grid
    int Ho, Wo, C_out;   // layer output grid
    int k, stride, pad;
    int Mp;
    int P_rows;          // row positions (forward: ni Ho Wo; dS: ni H W; dW: K positions ni Ho Wo)
    int C_t;             // the layer's input channels (C_in is that rounded up to 64 when smaller)
    int n_row, n_col, n_split, kt_per_split, ktiles;
    float *what;         // forward: w^ [P_out][C_out][Mp]
    const float *t_in;   // dS: layer input spike times [P_in][C_in]
    float *g_t_in;       // dS: [P_in][C_in], zeroed, accumulated
    float *g_W;          // dW: [C_out][k k C_in], accumulated
    const float *count;  // dW: silent neurons per output channel (dead-neuron term), or null
    float qcoef;         // dW: -gamma_Q norm
    int nst;             // generated-operand kernels: pipeline stages
    int res_bytes;       // generated-operand forward: resident filter bytes (0: streamed)
    int groups;          // generated-operand dW: row tiles per CTA
    // forward with the scan in its epilogue: per output neuron [P_out][C_out]
    float *t_out;
    int *q_out;
    float *s_out, *vdot_out;
    const float *rowsum;  // dead-neuron term per output channel
    float *penalty;       // [4] sums, or null
    LifConst c;
};

// position p of an (ni, h, w) grid -> (b, y, x)
__device__ __forceinline__ void pos_decode(int p, int h, int w, int &b, int &y, int &x) {
    const int hw = h * w;
    b = p / hw;
    const int r = p - b * hw;
    y = r / w;
    x = r - y * w;
}

// dS row tiles group the input positions by stride class (y mod s, x mod s):
// every position of a class is reached by the same taps, those whose offset
// lands on the stride grid, so a tile multiplies only those. Class c holds
// the positions y = py + ps yy, x = px + ps xx of every image, in image-major
// order; with stride 1 the one class is the identity order.
constexpr int DS_MAX_CLS = 4;
struct DsClass {
    int py, px;    // class offsets
    int Hc, Wc;    // class grid of one image
    int count;     // positions of the class over all images
    int tile0;     // first row tile of the class
    int kh0, kw0;  // first tap row / column that reaches the class
    int nkh, nkw;  // taps reaching it: rows kh0, kh0 + ts, ..., columns alike
};
struct DsPlan {
    int a_bytes, b_bytes, stage, res_bytes, nst, units, taps_per_unit;
    int epi_bytes;     // the epilogue's shared memory
    int run_ok;        // the map of ppt-position boxes is valid
    int ncls, ps, ts;  // classes, position step within a class, tap step
    DsClass cls[DS_MAX_CLS];
};

__device__ __forceinline__ int ds_class(const DsPlan &pl, int rt) {
    int c = 0;
    while (c + 1 < pl.ncls && rt >= pl.cls[c + 1].tile0) ++c;
    return c;
}

// position held by row slot pp of row tile rt (of class c) in a grid of
// gh x gw positions per image (dS: the input grid; forward: the output
// grid), or -1
__device__ __forceinline__ int ds_pos(const DsPlan &pl, int gh, int gw, int c, int rt, int pp, int ppt) {
    const DsClass &q = pl.cls[c];
    const int j = (rt - q.tile0) * ppt + pp;
    if (j >= q.count) return -1;
    const int per = q.Hc * q.Wc;
    const int b = j / per, r = j - b * per;
    const int yy = r / q.Wc, xx = r - yy * q.Wc;
    return (b * gh + q.py + pl.ps * yy) * gw + q.px + pl.ps * xx;
}

constexpr int DS_MAX_STAGES = 8;
constexpr int DS_EPI_BYTES = CONV_NEPI * 32 * EPI_LD * 4;
// forward epilogue: per (epilogue group, position of the tile) the w^ rows
// of Mp / 32 chunks of 32 neurons, Mp + pad floats each (Mp = 64: 2 x 2 x 2
// x 32 x (64 + pad) floats; Mp = 32: 2 x 4 x 1 x 32 x (32 + pad)). Rows are
// read as float4 with pad 4; the 128-channel forward on row boxes reads them
// one float at a time with pad 1 (still free of bank conflicts), which
// leaves room for two row-box stages
__host__ __device__ constexpr int fwd_epi_pad(bool tight) { return tight ? 1 : 4; }
__host__ __device__ constexpr int fwd_epi_bytes(bool tight) { return 2 * 2 * 2 * 32 * (64 + fwd_epi_pad(tight)) * 4; }

// ---------------------------------------------------------------------------
// Tap-shifted contraction over a [positions][Mp][channels] bf16 operand read
// through TMA boxes, in two modes:
//  FWD  the forward w^ of Eq. DSTD: rows (output position, m), columns BN of
//       the C_out channels, K = k k taps x blocks of 64 input channels of the
//       binned input S; the epilogue runs the scan/solve/select of each
//       neuron on its w^ column (Eq. LIF_Vmem_DSTD, the first threshold
//       crossing) and writes the spike outputs: w^ never leaves the chip.
//  !FWD dS with the input-time gradient: rows (input position, m), columns BN
//       of the C_in channels; K = k k taps x blocks of 64 output channels of
//       dw^ (the transposed convolution); the epilogue takes dC/dt_in.
// 128 / Mp positions per tile. Persistent: CTA b takes tiles b, b + grid, ...
//   warp 0  TMA producer (one lane): A boxes and the B tiles (or, with RES,
//           every B tile once)
//   warp 1  TMEM allocation and MMA issue (one lane)
//   warps 2-9  epilogue: warp w reads TMEM lane quarter w % 4, 32-column
//              chunks (w - 2) / 4, +2, ... of the tile
// ROWBOX (stride 1, tiles within one image row): one box of 128/Mp + k - 1
// positions per (kh, channel block) serves all k taps kw of that filter row;
// tap kw's A tile starts kw (FWD) or k - 1 - kw (dS) positions into it.
// Barriers: full/empty per unit; acc_full/acc_empty per accumulator (two).
// ---------------------------------------------------------------------------
template <int BN, bool ROWBOX, bool RES, bool FWD>
__global__ void __launch_bounds__(CONV_THREADS, 1)
    k_conv_tap_gemm(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                    const __grid_constant__ CUtensorMap mapR, ConvGemmArgs a, const __grid_constant__ DsPlan pl) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int NST = pl.nst;
    uint8_t *bres = smem + NST * pl.stage;
    float *epi = reinterpret_cast<float *>(bres + pl.res_bytes);
    uint64_t *full = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(epi) + pl.epi_bytes);
    uint64_t *empty = full + DS_MAX_STAGES;
    uint64_t *acc_full = empty + DS_MAX_STAGES;  // [2]
    uint64_t *acc_empty = acc_full + 2;          // [2]
    uint64_t *bres_full = acc_empty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bres_full + 1);
    constexpr uint32_t TMEM_COLS = 2 * BN;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = a.n_row * a.n_col;
    const int Mp = a.Mp;
    const int ppt = 128 / Mp;  // positions per tile
    const int kc = FWD ? a.C_in : a.C_out;  // channels contracted per tap
    const int ncb = kc >> 6;
    const int k = a.k;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&acc_full[u], 1);
            // the epilogue groups take alternate tiles (one per accumulator)
            tc::mbar_init(&acc_empty[u], CONV_NEPI / 2);
        }
        tc::mbar_init(bres_full, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, TMEM_COLS);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            if (RES) {
                // every (tap, channel block) B tile of the single column tile, once
                const int nslices = k * k * ncb;
                tc::mbar_expect_tx(bres_full, (uint32_t)(nslices * BN * 128));
                for (int q = 0; q < nslices; ++q) {
                    const int tap = q / ncb, cb = q - tap * ncb;
                    tc::tma_load_2d(tc::smem_u32(bres + q * BN * 128), &mapB, bres_full, tap * kc + cb * 64, 0);
                }
            }
            // one thread issues every copy: the loops below keep its work per
            // unit to a few additions (positions decoded once per tile, stage
            // and phase counted, taps stepped)
            uint32_t it = 0;  // units issued
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                const int rt = t / a.n_col, ct = t - rt * a.n_col;
                const DsClass &q = pl.cls[ds_class(pl, rt)];
                int b0 = 0, y0 = 0, x0 = 0;
                int pb[4], pyy[4], pxx[4];  // image and class coordinates of the tile's positions
                if (ROWBOX) {
                    if (FWD) pos_decode(rt * ppt, a.Ho, a.Wo, b0, y0, x0);
                    else pos_decode(rt * ppt, a.H, a.W, b0, y0, x0);
                } else {
#pragma unroll
                    for (int pp = 0; pp < 4; ++pp) {
                        pb[pp] = a.ni;  // padding row: a box outside the tensor (zeros)
                        pyy[pp] = pxx[pp] = 0;
                        const int jj = (rt - q.tile0) * ppt + pp;
                        if (pp < ppt && jj < q.count) {
                            const int per = q.Hc * q.Wc;
                            pb[pp] = jj / per;
                            const int r = jj - pb[pp] * per;
                            pyy[pp] = r / q.Wc;
                            pxx[pp] = r - pyy[pp] * q.Wc;
                            if (FWD) {  // input origin of the output position's receptive field
                                pyy[pp] = pyy[pp] * a.stride - a.pad;
                                pxx[pp] = pxx[pp] * a.stride - a.pad;
                            }
                        }
                    }
                }
                // class coordinates: tap (kh0 + ih ts, kw0 + iw ts) reads output
                // position (yy + by0 - ih, xx + bx0 - iw)
                const bool cls_order = pl.ps == a.stride;
                // the tile's positions read one run of consecutive positions of
                // a row for every tap (stride 1 forward; dS in stride classes):
                // one box of ppt positions (mapR) instead of ppt boxes
                bool run = !ROWBOX && pl.run_ok && ppt > 1 && (FWD ? a.stride == 1 : cls_order);
#pragma unroll
                for (int pp = 1; pp < 4; ++pp)
                    if (pp < ppt) run = run && pb[pp] == pb[0] && pyy[pp] == pyy[0] && pxx[pp] == pxx[0] + pp;
                const int by0 = cls_order ? (q.py + a.pad - q.kh0) / pl.ts : 0;
                const int bx0 = cls_order ? (q.px + a.pad - q.kw0) / pl.ts : 0;
                const int nkh = ROWBOX ? k : q.nkh, nkw = ROWBOX ? 1 : q.nkw;
                for (int ih = 0; ih < nkh && ok; ++ih)
                    for (int iw = 0; iw < nkw && ok; ++iw)
                        for (int cb = 0; cb < ncb; ++cb, ++it) {
                            if (!tc::mbar_wait_spin(&empty[s], ph ^ 1u)) {
                                conv_set_status(STATUS_TIMEOUT);
                                ok = false;
                                break;
                            }
                            tc::mbar_expect_tx(&full[s], (uint32_t)(pl.a_bytes + pl.b_bytes));
                            const uint32_t st = tc::smem_u32(smem + s * pl.stage);
                            if (ROWBOX) {
                                // unit (kh, cb): FWD input positions x0 - pad .. of row y0 - pad + kh;
                                // dS output positions x0 + pad - (k - 1) .. of row y0 + pad - kh
                                if (FWD)
                                    tma_load_5d(st, &mapA, &full[s], cb * 64, 0, x0 - a.pad, y0 - a.pad + ih, b0);
                                else
                                    tma_load_5d(st, &mapA, &full[s], cb * 64, 0, x0 + a.pad - (k - 1), y0 + a.pad - ih,
                                                b0);
                                if (!RES)
                                    for (int kw = 0; kw < k; ++kw)
                                        tc::tma_load_2d(st + pl.a_bytes + kw * BN * 128, &mapB, &full[s],
                                                        (ih * k + kw) * kc + cb * 64, ct * BN);
                            } else {
                                const int kh = q.kh0 + ih * pl.ts, kw = q.kw0 + iw * pl.ts;
#pragma unroll
                                for (int pp = 0; pp < 4; ++pp) {
                                    if (pp >= (run ? 1 : ppt)) break;
                                    int sx, sy;
                                    if (FWD) {
                                        sy = pyy[pp] + kh;
                                        sx = pxx[pp] + kw;
                                    } else if (cls_order) {
                                        sy = pyy[pp] + by0 - ih;
                                        sx = pxx[pp] + bx0 - iw;
                                    } else {  // identity order (stride above 2): off-grid taps read zeros
                                        const int ny = pyy[pp] + a.pad - kh, nx = pxx[pp] + a.pad - kw;
                                        const bool on = ny % a.stride == 0 && nx % a.stride == 0;
                                        sy = on ? ny / a.stride : -1;
                                        sx = on ? nx / a.stride : 0;
                                    }
                                    tma_load_5d(st + pp * Mp * 128, run ? &mapR : &mapA, &full[s], cb * 64, 0, sx, sy,
                                                pb[pp]);
                                }
                                if (!RES)
                                    tc::tma_load_2d(st + pl.a_bytes, &mapB, &full[s], (kh * k + kw) * kc + cb * 64,
                                                    ct * BN);
                            }
                            if (++s == NST) {
                                s = 0;
                                ph ^= 1u;
                            }
                        }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i) tc::mbar_wait_spin(&full[i % NST], (i / NST) & 1u);
            if (RES) tc::mbar_wait_spin(bres_full, 0);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, false, false);
            uint32_t j = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            if (RES && !tc::mbar_wait_spin(bres_full, 0)) {
                conv_set_status(STATUS_TIMEOUT);
                ok = false;
            }
            const int tpu = ROWBOX ? k : 1;  // taps per unit
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                const uint32_t buf = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait_spin(&acc_empty[buf], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc = tmem + buf * BN;
                const DsClass &q = pl.cls[ds_class(pl, t / a.n_col)];
                const int nkh = ROWBOX ? k : q.nkh, nkw = ROWBOX ? 1 : q.nkw;
                bool first = true;
                for (int ih = 0; ih < nkh && ok; ++ih)
                    for (int iw = 0; iw < nkw && ok; ++iw)
                        for (int cb = 0; cb < ncb; ++cb) {
                            if (!tc::mbar_wait_spin(&full[s], ph)) {
                                conv_set_status(STATUS_TIMEOUT);
                                ok = false;
                                break;
                            }
                            tc::tc_fence_after();
                            const uint32_t sa = tc::smem_u32(smem + s * pl.stage);
                            for (int v = 0; v < tpu; ++v) {
                                int tap;
                                uint32_t abase;
                                if (ROWBOX) {
                                    tap = ih * k + v;
                                    abase = sa + (uint32_t)((FWD ? v : k - 1 - v) * Mp * 128);
                                } else {
                                    tap = (q.kh0 + ih * pl.ts) * k + q.kw0 + iw * pl.ts;
                                    abase = sa;
                                }
                                const uint32_t bbase = RES ? tc::smem_u32(bres + (tap * ncb + cb) * BN * 128)
                                                           : sa + (uint32_t)(pl.a_bytes + v * BN * 128);
                                // descriptors built once; each 16-deep slice is 32 bytes on (+2)
                                const uint64_t ad = tc::sdesc_sw128(abase), bd = tc::sdesc_sw128(bbase);
                                tc::mma_bf16(acc, ad, bd, idesc, (!first || v > 0) ? 1u : 0u);
#pragma unroll
                                for (int kk = 1; kk < 4; ++kk) tc::mma_bf16(acc, ad + 2 * kk, bd + 2 * kk, idesc, 1u);
                            }
                            first = false;
                            tc::mma_commit(&empty[s]);
                            if (++s == NST) {
                                s = 0;
                                ph ^= 1u;
                            }
                        }
                if (ok) tc::mma_commit(&acc_full[buf]);
            }
        }
        __syncwarp();
    } else if (FWD) {
        // Scan in the epilogue. Epilogue group g takes the tiles of
        // accumulator g (every other tile). Warp w of the group reads TMEM
        // lane quarter w % 4 (grid steps mq .. mq + 31 of position pp); per
        // round the qpp = Mp / 32 warps of a position write qpp chunks of 32
        // channels as neuron-major rows of their buffers, then, after a
        // barrier over those warps, each walks one chunk's 32 neurons, one per
        // lane, as the scan kernel does.
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const int qpp = Mp >> 5;  // lane quarters per position
        const int pp = quarter / qpp, wip = quarter - pp * qpp, mq = wip * 32;
        constexpr bool TIGHT = FWD && BN == 128 && ROWBOX;
        const int LDB = Mp + fwd_epi_pad(TIGHT);
        float *pbuf = epi + (group * ppt + pp) * qpp * 32 * LDB;
        const int bar_id = 1 + group * ppt + pp;  // named barrier of the position's warps
        auto sync_pos = [&]() {
            if (qpp == 1) __syncwarp();
            else asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "r"(qpp * 32) : "memory");
        };
        auto any_pos = [&](bool x) -> bool {
            if (qpp == 1) return __any_sync(0xffffffffu, x);
            uint32_t r;
            asm volatile(
                "{\n"
                ".reg .pred pi, po;\n"
                "setp.ne.u32 pi, %1, 0;\n"
                "barrier.cta.red.or.pred po, %2, %3, pi;\n"
                "selp.u32 %0, 1, 0, po;\n"
                "}\n"
                : "=r"(r)
                : "r"((uint32_t)x), "r"(bar_id), "r"(qpp * 32)
                : "memory");
            return r != 0;
        };
        const int rounds = (BN / 32) / qpp;
        float pacc[4] = {0.f, 0.f, 0.f, 0.f};
        for (int j = group, t = blockIdx.x + group * gridDim.x; t < ntiles; j += 2, t += 2 * gridDim.x) {
            const int rt = t / a.n_col, ct = t - rt * a.n_col;
            const uint32_t buf = (uint32_t)group;
            const int p = ds_pos(pl, a.Ho, a.Wo, ds_class(pl, rt), rt, pp, ppt);
            // an expired wait ends the role of every warp of the position
            // together, so that none is left at their barrier
            const bool fail = !tc::mbar_wait_sleep(&acc_full[buf], (uint32_t)(j >> 1) & 1u);
            if (any_pos(fail)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            for (int r = 0; r < rounds; ++r) {
                for (int k = 0; k < qpp; ++k) {
                    float v[32];
                    tc::tmem_ld32(tmem + lane_base + buf * BN + (r * qpp + k) * 32, v);
                    float *tb = pbuf + k * 32 * LDB;
#pragma unroll
                    for (int u = 0; u < 32; ++u) tb[u * LDB + mq + lane] = v[u];
                }
                if (r == rounds - 1) {  // the tile's last TMEM read of this warp
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
                }
                sync_pos();
                if (p >= 0) {
                    const float *row = pbuf + (wip * 32 + lane) * LDB;
                    ScanState st;
                    scan_reset(st, a.c.M);
                    float vv = 0.f, I = 0.f;
                    for (int m0 = 0; m0 < a.c.M; m0 += 32) {
                        const int mend = (a.c.M - m0) < 32 ? (a.c.M - m0) : 32;
                        if (scan_walk<32, !TIGHT>(a.c, row + m0, m0, mend, vv, I, st)) break;
                    }
                    scan_finish(a.c, st);
                    finish_neuron(a.c, st, p, ct * BN + (r * qpp + wip) * 32 + lane, a.C_out, a.rowsum, a.t_out,
                                  a.q_out, a.s_out, a.vdot_out, pacc);
                }
                sync_pos();
            }
        }
        if (a.penalty) {
#pragma unroll
            for (int k2 = 0; k2 < 4; ++k2) {
                const float sum = warp_sum(pacc[k2]);
                if (lane == 0 && sum != 0.f) atomicAdd(&a.penalty[k2], sum);
            }
        }
    } else {
        // dS: epilogue group g takes the tiles of accumulator g (every other
        // tile), all BN columns of them; warp w reads TMEM lane quarter w % 4
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        float *tb = epi + (warp - 2) * 32 * EPI_LD;
        const int pp = (quarter * 32) / Mp;      // position of this warp's rows (Mp >= 32)
        const int m_base = (quarter * 32) % Mp;  // first grid step of this warp's rows
        constexpr int NCH = BN / 32;             // 32-column chunks of the tile
        for (int j = group, t = blockIdx.x + group * gridDim.x; t < ntiles; j += 2, t += 2 * gridDim.x) {
            const int rt = t / a.n_col, ct = t - rt * a.n_col;
            const uint32_t buf = (uint32_t)group;
            const int p = ds_pos(pl, a.H, a.W, ds_class(pl, rt), rt, pp, ppt);
            // the grid step and the two kernel derivatives of the input each
            // lane will own, loaded while the tile's MMAs run
            int wk[NCH];
            float wdR[NCH], wdL[NCH];
#pragma unroll
            for (int h = 0; h < NCH; ++h) {
                wk[h] = -1000;
                wdR[h] = wdL[h] = 0.f;
                const int col0 = ct * BN + h * 32;
                if (p >= 0 && col0 + lane < a.C_t) {
                    const float x = __ldg(a.t_in + (long long)p * a.C_t + col0 + lane);
                    if (isfinite(x)) {
                        const BinW w = bin_weights(a.c, x, true);
                        wk[h] = w.k;
                        wdR[h] = w.dR;
                        wdL[h] = w.dL;
                    }
                }
            }
            if (!tc::mbar_wait_sleep(&acc_full[buf], (uint32_t)(j >> 1) & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
#pragma unroll
            for (int h = 0; h < NCH; ++h) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + buf * BN + h * 32, v);
                if (h == NCH - 1) {  // the tile's last TMEM read of this warp
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
                }
                // lane m of the warp holds grid step m_base + m of 32 channels;
                // transpose through shared memory so that lane u owns channel
                // col0 + u and reads its two grid steps
#pragma unroll
                for (int u = 0; u < 32; ++u) tb[lane * EPI_LD + u] = v[u];
                __syncwarp();
                if (p >= 0 && wk[h] > -1000) {
                    float g = 0.f;
                    const int k0 = wk[h] - m_base, k1 = wk[h] + 1 - m_base;
                    if (k0 >= 0 && k0 < 32 && wk[h] < a.c.M) g = fmaf(tb[k0 * EPI_LD + lane], wdR[h], g);
                    if (k1 >= 0 && k1 < 32 && wk[h] + 1 < a.c.M) g = fmaf(tb[k1 * EPI_LD + lane], wdL[h], g);
                    if (g != 0.f) atomicAdd(a.g_t_in + (long long)p * a.C_t + ct * BN + h * 32 + lane, g);
                }
                __syncwarp();
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, TMEM_COLS);
}

// ---------------------------------------------------------------------------
// dS of two row tiles at once (stride 1, image rows a multiple of 2 ppt
// positions wide). The pair's 2 ppt input positions are consecutive in one
// row, so one box of 2 ppt + k - 1 positions of dw^ per (filter row,
// channel block) serves both tiles and all k taps of the row, and every
// filter slice feeds two MMAs back to back (one per tile, each into its own
// accumulator): consecutive MMAs on the same B operand issue faster than
// MMAs that each fetch new operands. TMEM: two pair slots x two tiles x BN
// columns. Epilogue group g takes tile g of every pair (the same work per
// warp as the single-tile kernel's epilogue); acc_empty counts all eight
// epilogue warps. Warps and barriers otherwise as in k_conv_tap_gemm.
// ---------------------------------------------------------------------------
template <int BN, bool RES>
__global__ void __launch_bounds__(CONV_THREADS, 1)
    k_conv_ds_pair(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, ConvGemmArgs a,
                   const __grid_constant__ DsPlan pl) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int NST = pl.nst;
    uint8_t *bres = smem + NST * pl.stage;
    float *epi = reinterpret_cast<float *>(bres + pl.res_bytes);
    uint64_t *full = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(epi) + pl.epi_bytes);
    uint64_t *empty = full + DS_MAX_STAGES;
    uint64_t *acc_full = empty + DS_MAX_STAGES;  // [2] pair slots
    uint64_t *acc_empty = acc_full + 2;          // [2]
    uint64_t *bres_full = acc_empty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bres_full + 1);
    constexpr uint32_t TMEM_COLS = 4 * BN;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int npairs = (a.n_row >> 1) * a.n_col;
    const int Mp = a.Mp;
    const int ppt = 128 / Mp;  // positions per tile
    const int kc = a.C_out;    // channels contracted per tap
    const int ncb = kc >> 6;
    const int k = a.k;
    const uint32_t tile_bytes = (uint32_t)(ppt * Mp * 128);  // the second tile's rows in the box

    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int u = 0; u < 2; ++u) {
            tc::mbar_init(&acc_full[u], 1);
            tc::mbar_init(&acc_empty[u], CONV_NEPI);  // both groups read every pair slot
        }
        tc::mbar_init(bres_full, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, TMEM_COLS);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            if (RES) {
                const int nslices = k * k * ncb;
                tc::mbar_expect_tx(bres_full, (uint32_t)(nslices * BN * 128));
                for (int q = 0; q < nslices; ++q) {
                    const int tap = q / ncb, cb = q - tap * ncb;
                    tc::tma_load_2d(tc::smem_u32(bres + q * BN * 128), &mapB, bres_full, tap * kc + cb * 64, 0);
                }
            }
            uint32_t it = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int pr = blockIdx.x; pr < npairs && ok; pr += gridDim.x) {
                const int rp = pr / a.n_col, ct = pr - rp * a.n_col;
                int b0, y0, x0;
                pos_decode(rp * 2 * ppt, a.H, a.W, b0, y0, x0);
                for (int ih = 0; ih < k && ok; ++ih)
                    for (int cb = 0; cb < ncb; ++cb, ++it) {
                        if (!tc::mbar_wait_spin(&empty[s], ph ^ 1u)) {
                            conv_set_status(STATUS_TIMEOUT);
                            ok = false;
                            break;
                        }
                        tc::mbar_expect_tx(&full[s], (uint32_t)(pl.a_bytes + pl.b_bytes));
                        const uint32_t st = tc::smem_u32(smem + s * pl.stage);
                        // output positions x0 + pad - (k - 1) .. of row y0 + pad - kh
                        tma_load_5d(st, &mapA, &full[s], cb * 64, 0, x0 + a.pad - (k - 1), y0 + a.pad - ih, b0);
                        if (!RES)
                            for (int kw = 0; kw < k; ++kw)
                                tc::tma_load_2d(st + pl.a_bytes + kw * BN * 128, &mapB, &full[s],
                                                (ih * k + kw) * kc + cb * 64, ct * BN);
                        if (++s == NST) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i) tc::mbar_wait_spin(&full[i % NST], (i / NST) & 1u);
            if (RES) tc::mbar_wait_spin(bres_full, 0);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, false, false);
            uint32_t j = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            if (RES && !tc::mbar_wait_spin(bres_full, 0)) {
                conv_set_status(STATUS_TIMEOUT);
                ok = false;
            }
            for (int pr = blockIdx.x; pr < npairs && ok; pr += gridDim.x, ++j) {
                const uint32_t slot = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait_spin(&acc_empty[slot], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc0 = tmem + slot * 2 * BN, acc1 = acc0 + BN;
                bool first = true;
                for (int ih = 0; ih < k && ok; ++ih)
                    for (int cb = 0; cb < ncb; ++cb) {
                        if (!tc::mbar_wait_spin(&full[s], ph)) {
                            conv_set_status(STATUS_TIMEOUT);
                            ok = false;
                            break;
                        }
                        tc::tc_fence_after();
                        const uint32_t sa = tc::smem_u32(smem + s * pl.stage);
                        for (int v = 0; v < k; ++v) {
                            const int tap = ih * k + v;
                            const uint32_t abase = sa + (uint32_t)((k - 1 - v) * Mp * 128);
                            const uint32_t bbase = RES ? tc::smem_u32(bres + (tap * ncb + cb) * BN * 128)
                                                       : sa + (uint32_t)(pl.a_bytes + v * BN * 128);
                            const uint64_t ad0 = tc::sdesc_sw128(abase), ad1 = tc::sdesc_sw128(abase + tile_bytes);
                            const uint64_t bd = tc::sdesc_sw128(bbase);
                            const uint32_t acc_in = (!first || v > 0) ? 1u : 0u;
                            tc::mma_bf16(acc0, ad0, bd, idesc, acc_in);
                            tc::mma_bf16(acc1, ad1, bd, idesc, acc_in);
#pragma unroll
                            for (int kk = 1; kk < 4; ++kk) {
                                tc::mma_bf16(acc0, ad0 + 2 * kk, bd + 2 * kk, idesc, 1u);
                                tc::mma_bf16(acc1, ad1 + 2 * kk, bd + 2 * kk, idesc, 1u);
                            }
                        }
                        first = false;
                        tc::mma_commit(&empty[s]);
                        if (++s == NST) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                if (ok) tc::mma_commit(&acc_full[slot]);
            }
        }
        __syncwarp();
    } else {
        // group g reads tile g of every pair, all BN columns; warp w reads
        // TMEM lane quarter w % 4
        const int quarter = warp & 3, group = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        float *tb = epi + (warp - 2) * 32 * EPI_LD;
        const int pp = (quarter * 32) / Mp;      // position of this warp's rows (Mp >= 32)
        const int m_base = (quarter * 32) % Mp;  // first grid step of this warp's rows
        constexpr int NCH = BN / 32;
        uint32_t j = 0;
        for (int pr = blockIdx.x; pr < npairs; pr += gridDim.x, ++j) {
            const int rp = pr / a.n_col, ct = pr - rp * a.n_col;
            const int rt = rp * 2 + group;
            const uint32_t slot = j & 1u;
            const int p = ds_pos(pl, a.H, a.W, 0, rt, pp, ppt);
            int wk[NCH];
            float wdR[NCH], wdL[NCH];
#pragma unroll
            for (int h = 0; h < NCH; ++h) {
                wk[h] = -1000;
                wdR[h] = wdL[h] = 0.f;
                const int col0 = ct * BN + h * 32;
                if (p >= 0 && col0 + lane < a.C_t) {
                    const float x = __ldg(a.t_in + (long long)p * a.C_t + col0 + lane);
                    if (isfinite(x)) {
                        const BinW w = bin_weights(a.c, x, true);
                        wk[h] = w.k;
                        wdR[h] = w.dR;
                        wdL[h] = w.dL;
                    }
                }
            }
            if (!tc::mbar_wait_sleep(&acc_full[slot], (j >> 1) & 1u)) {
                conv_set_status(STATUS_TIMEOUT);
                break;
            }
            tc::tc_fence_after();
            const uint32_t acc = tmem + (slot * 2 + (uint32_t)group) * BN;
#pragma unroll
            for (int h = 0; h < NCH; ++h) {
                float v[32];
                tc::tmem_ld32(acc + lane_base + h * 32, v);
                if (h == NCH - 1) {  // the pair slot's last TMEM read of this warp
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(&acc_empty[slot]);
                }
#pragma unroll
                for (int u = 0; u < 32; ++u) tb[lane * EPI_LD + u] = v[u];
                __syncwarp();
                if (p >= 0 && wk[h] > -1000) {
                    float g = 0.f;
                    const int k0 = wk[h] - m_base, k1 = wk[h] + 1 - m_base;
                    if (k0 >= 0 && k0 < 32 && wk[h] < a.c.M) g = fmaf(tb[k0 * EPI_LD + lane], wdR[h], g);
                    if (k1 >= 0 && k1 < 32 && wk[h] + 1 < a.c.M) g = fmaf(tb[k1 * EPI_LD + lane], wdL[h], g);
                    if (g != 0.f) atomicAdd(a.g_t_in + (long long)p * a.C_t + ct * BN + h * 32 + lane, g);
                }
                __syncwarp();
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Binned operand generated on chip (the compact support of K_DSTD: each
// input spike has two nonzero grid weights among Mp). The binning writes
// one 8-byte record per input, rec[p][c] = (grid step k, bf16 pair (w at
// T_k, w at T_{k+1})), k = -128 when silent. Generator warps load the
// records a K step needs (64 consecutive per position and tap: a warp reads
// 256 contiguous bytes) several K steps ahead and write each record's two
// nonzeros into the swizzled A tile that the tensor core reads. Each thread
// owns fixed columns of the tile, so before writing it erases the two
// entries it wrote the last time it used that stage (all stages start
// zeroed): 4 two-byte shared stores per input instead of 16 KB of operand
// per K step from L2.
// ---------------------------------------------------------------------------
constexpr int REC_SILENT = -128;

// the record of one input spike time x (+inf: silent)
__device__ __forceinline__ uint2 bin_record(const LifConst &c, float x) {
    uint2 r = make_uint2((uint32_t)REC_SILENT, 0u);
    if (isfinite(x)) {
        const BinW w = bin_weights(c, x, false);
        if (w.k >= -1 && w.k < c.M) r = make_uint2((uint32_t)w.k, pack_bf16x2(w.wR, w.wL));
    }
    return r;
}

__global__ void __launch_bounds__(256) k_bin_rec(const float *__restrict__ t, long long n, LifConst c,
                                                 uint2 *__restrict__ rec) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
        rec[i] = bin_record(c, __ldg(t + i));
}

// The binned input written out for the TMA-fed contractions: S [P][Mp][C]
// bf16, row (p, m) holding grid step m of the C channels, from the spike
// times t [P][C] (each input's record, as k_bin_rec forms it: the two
// nonzeros of input (p, c) at m = k and k + 1 < M, zeros elsewhere). A block builds R = 256 / C consecutive positions (one for
// C >= 256) in shared memory and writes them with one bulk copy; two
// buffers alternate, and a thread, which owns fixed (position, channel)
// slots of the buffers, erases the two entries it wrote in a buffer before
// writing the new ones, so the zeros are written to shared memory once.
constexpr int BINS_THREADS = 256;
constexpr int BINS_MAXSPT = 4;  // channels per thread: C <= 1024

__device__ __forceinline__ void bins_put(uint16_t *T, int row0, int C, int c, int kold, uint2 q, int M) {
    if (kold != REC_SILENT) {
        if (kold >= 0) T[(row0 + kold) * C + c] = 0;
        if (kold + 1 < M) T[(row0 + kold + 1) * C + c] = 0;
    }
    const int k = (int)q.x;
    if (k != REC_SILENT) {
        if (k >= 0) T[(row0 + k) * C + c] = (uint16_t)(q.y & 0xffffu);
        if (k + 1 < M) T[(row0 + k + 1) * C + c] = (uint16_t)(q.y >> 16);
    }
}

__global__ void __launch_bounds__(BINS_THREADS) k_bin_S(const float *__restrict__ t, int P, int C, int Ct,
                                                        LifConst lc, __nv_bfloat16 *__restrict__ S) {
    const int Mp = lc.Mp, M = lc.M;
    extern __shared__ __align__(128) uint8_t bins_smem[];
    const int R = C >= BINS_THREADS ? 1 : BINS_THREADS / C;  // positions per group
    const int tile = R * Mp * C;                            // elements per buffer
    uint16_t *buf0 = reinterpret_cast<uint16_t *>(bins_smem), *buf1 = buf0 + tile;
    const int spt = C > BINS_THREADS ? C / BINS_THREADS : (threadIdx.x < R * C ? 1 : 0);
    const int r = C >= BINS_THREADS ? 0 : threadIdx.x / C;
    const int c0 = C >= BINS_THREADS ? threadIdx.x : threadIdx.x - r * C;
    for (int i = threadIdx.x; i < tile / 4; i += blockDim.x) reinterpret_cast<uint4 *>(buf0)[i] = make_uint4(0, 0, 0, 0);
    int kold0[BINS_MAXSPT], kold1[BINS_MAXSPT];
#pragma unroll
    for (int j = 0; j < BINS_MAXSPT; ++j) kold0[j] = kold1[j] = REC_SILENT;
    const int ngroups = (P + R - 1) / R;
    int it = 0;
    for (int gi = blockIdx.x; gi < ngroups; gi += gridDim.x, ++it) {
        const bool odd = it & 1;
        uint16_t *T = odd ? buf1 : buf0;
        // the bulk copy that read this buffer two groups ago is done with it
        if (threadIdx.x == 0 && it >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
        __syncthreads();
        const int p = gi * R + r;
#pragma unroll
        for (int j = 0; j < BINS_MAXSPT; ++j) {
            if (j < spt) {
                const int c = c0 + j * BINS_THREADS;
                // channels past the layer's Ct (padding up to C) are silent
                const uint2 q = p < P && c < Ct ? bin_record(lc, __ldg(t + (long long)p * Ct + c))
                                                : make_uint2((uint32_t)REC_SILENT, 0u);
                bins_put(T, r * Mp, C, c, odd ? kold1[j] : kold0[j], q, M);
                if (odd) kold1[j] = (int)q.x;
                else kold0[j] = (int)q.x;
            }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (threadIdx.x == 0) {
            const int np = P - gi * R < R ? P - gi * R : R;
            const uint32_t bytes = (uint32_t)np * Mp * C * 2;
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                             S + (long long)gi * R * Mp * C),
                         "r"(tc::smem_u32(T)), "r"(bytes)
                         : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        }
    }
    if (threadIdx.x == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int c, int m, int p) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c), "r"(m), "r"(p), "r"(tc::smem_u32(bar))
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

constexpr int GEN_WARPS = 4;                                    // per generator group (one K step)
constexpr int FWD_GEN_GROUPS = 4;                               // forward: K steps generated at once
constexpr int FWD_THREADS = (2 + CONV_NEPI + GEN_WARPS * FWD_GEN_GROUPS) * 32;  // 832

// shared-memory plan of the generated-operand forward: per stage the A tile
// and the B tile (unless the filters are resident); the stage count and the
// resident bytes are chosen on the host (ConvGemmArgs::nst, ::res_bytes)
template <int BN, bool RES>
struct GenFwdCfg {
    static constexpr int A_BYTES = 128 * 128;
    static constexpr int B_BYTES = RES ? 0 : BN * 128;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int MAX_STAGES = 8;
    static constexpr int PREV_BYTES = MAX_STAGES * 256 * 2;  // last grid step written, per stage and slot
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static __host__ __device__ int smem(int nst, int res_bytes) {
        return nst * STAGE + res_bytes + PREV_BYTES + 1024 + 256;
    }
};
constexpr int GEN_SMEM_MAX = 225 * 1024;
constexpr int GEN_AHEAD = 8;  // K steps of records a generator thread loads ahead

// Forward with the binned operand generated on chip. Warps: 0 TMA (the
// filter tiles per K step, or all of them once when RES), 1 MMA, 2-9
// epilogue (w^ rows), 10-13 generators. A generator thread owns slots
// (position pp, channel c) g and g + 128 of the tile; it loads their records
// GEN_AHEAD K steps ahead (a warp reads 32 consecutive records), waits until
// the stage's previous MMAs are done, writes the A tile, and arrives.
template <int BN, bool RES>
__global__ void __launch_bounds__(FWD_THREADS, 1)
    k_conv_fwd_gen(const uint2 *__restrict__ rec, const __grid_constant__ CUtensorMap mapB, ConvGemmArgs a) {
    using Cfg = GenFwdCfg<BN, RES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int NST = a.nst;
    uint8_t *bres = smem + NST * Cfg::STAGE;  // resident filters (RES)
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
                tc::mbar_wait_spin(bres_full, 0);
            } else {
                uint32_t it = 0;
                int s = 0;
                uint32_t ph = 0;
                bool ok = true;
                for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                    const int ct = t % a.n_col;
                    int tap = 0, cb = 0;
                    for (int kt = 0; kt < a.ktiles; ++kt, ++it) {
                        if (!tc::mbar_wait_spin(&empty[s], ph ^ 1u)) {
                            conv_set_status(STATUS_TIMEOUT);
                            ok = false;
                            break;
                        }
                        tc::mbar_expect_tx(&full_t[s], (uint32_t)Cfg::B_BYTES);
                        tc::tma_load_2d(tc::smem_u32(smem + s * Cfg::STAGE + Cfg::A_BYTES), &mapB, &full_t[s],
                                        tap * a.C_in + cb * 64, ct * BN);
                        if (++cb == ncb) {
                            cb = 0;
                            ++tap;
                        }
                        if (++s == NST) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                }
                const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
                for (uint32_t i = it - n_drain; i < it; ++i)
                    tc::mbar_wait_spin(&full_t[i % NST], (i / NST) & 1u);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, false, false);
            uint32_t j = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            if (RES && !tc::mbar_wait_spin(bres_full, 0)) {
                conv_set_status(STATUS_TIMEOUT);
                ok = false;
            }
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                const uint32_t buf = j & 1u;
                if (j >= 2) {
                    if (!tc::mbar_wait_spin(&acc_empty[buf], ((j >> 1) + 1u) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                const uint32_t acc = tmem + buf * BN;
                for (int kt = 0; kt < a.ktiles; ++kt) {
                    if ((!RES && !tc::mbar_wait_spin(&full_t[s], ph)) || !tc::mbar_wait_spin(&full_a[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * Cfg::STAGE);
                    const uint32_t sbb = RES ? tc::smem_u32(bres + kt * BN * 128) : sa + Cfg::A_BYTES;
                    const uint64_t sad = tc::sdesc_sw128(sa), sbd = tc::sdesc_sw128(sbb);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc::mma_bf16(acc, sad + 2 * kk, sbd + 2 * kk, idesc, (kt > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_commit(&empty[s]);
                    if (++s == NST) {
                        s = 0;
                        ph ^= 1u;
                    }
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
                    // w^ [p][o][m]: for each neuron o the warp's 32 lanes hold 32
                    // consecutive grid steps, one 128-byte line per store
                    float *dst = a.what + ((long long)p * a.C_out + ct * BN + cc * 32) * Mp + (r % Mp);
#pragma unroll
                    for (int u = 0; u < 32; ++u) __stcs(dst + (long long)u * Mp, v[u]);
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
        }
    } else {
        // generator group grp (4 warps) takes K steps it = grp, grp + 4, ...;
        // the stage count is a multiple of 4, so a stage always belongs to the
        // same group and each of its slots to the same thread
        const int gw = warp - (2 + CONV_NEPI);
        const int grp = gw / GEN_WARPS;
        const int g = (gw % GEN_WARPS) * 32 + lane;
        const int nslots = ppt * 64;
        uint2 q[GEN_AHEAD][2];
        // the K step whose records load next (tile la_t, step la_kt), and the
        // decoded positions of this thread's two slots in tile la_t
        int la_t = blockIdx.x, la_kt = grp;
        while (la_kt >= a.ktiles && la_t < ntiles) {
            la_kt -= a.ktiles;
            la_t += gridDim.x;
        }
        // per slot of tile la_t: the receptive-field origin (ys, xs) and the
        // record index of its tap (0, 0) channel block 0; the tap (la_kh,
        // la_kw) and channel block la_cb of step la_kt advance by counting
        int pc_t = -1, ys[2] = {0, 0}, xs[2] = {0, 0};
        long long base[2] = {0, 0};
        bool pv[2] = {false, false};
        int la_kh = 0, la_kw = 0, la_cb = 0;
        auto set_tap = [&]() {
            const int tap = la_kt / ncb;
            la_cb = la_kt - tap * ncb;
            la_kh = tap / a.k;
            la_kw = tap - la_kh * a.k;
        };
        set_tap();
        auto load_next = [&](uint2(&dst)[2]) {
            if (la_t < ntiles && la_t != pc_t) {
                pc_t = la_t;
                const int p0 = (la_t / a.n_col) * ppt;
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int slot = g + u * 128, p = p0 + (slot >> 6);
                    pv[u] = slot < nslots && p < a.P_rows;
                    if (pv[u]) {
                        int b, y, x;
                        pos_decode(p, a.Ho, a.Wo, b, y, x);
                        ys[u] = y * a.stride - a.pad;
                        xs[u] = x * a.stride - a.pad;
                        base[u] = (((long long)b * a.H + ys[u]) * a.W + xs[u]) * a.C_in + (slot & 63);
                    }
                }
            }
            const int off = (la_kh * a.W + la_kw) * a.C_in + la_cb * 64;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                dst[u] = make_uint2((uint32_t)REC_SILENT, 0u);
                if (la_t < ntiles && pv[u] && (unsigned)(ys[u] + la_kh) < (unsigned)a.H &&
                    (unsigned)(xs[u] + la_kw) < (unsigned)a.W)
                    dst[u] = __ldg(rec + base[u] + off);
            }
            la_kt += FWD_GEN_GROUPS;
            if (la_kt >= a.ktiles) {
                while (la_kt >= a.ktiles && la_t < ntiles) {
                    la_kt -= a.ktiles;
                    la_t += gridDim.x;
                }
                set_tap();
            } else {
#pragma unroll
                for (int i = 0; i < FWD_GEN_GROUPS; ++i)
                    if (++la_cb == ncb) {
                        la_cb = 0;
                        if (++la_kw == a.k) {
                            la_kw = 0;
                            ++la_kh;
                        }
                    }
            }
        };
#pragma unroll
        for (int d = 0; d < GEN_AHEAD; ++d) load_next(q[d]);
        int s = grp;  // stage of this group's next K step, and its phase
        uint32_t ph = 0;
        int cur_t = blockIdx.x, cur_kt = grp;
        while (cur_kt >= a.ktiles && cur_t < ntiles) {
            cur_kt -= a.ktiles;
            cur_t += gridDim.x;
        }
        bool ok = true;
        while (cur_t < ntiles && ok) {
#pragma unroll
            for (int d = 0; d < GEN_AHEAD; ++d) {
                if (cur_t < ntiles && ok) {
                    int w_ok = 1;
                    // generators run ahead of the MMAs: park (suspend hint) rather
                    // than poll, which would take shared-memory cycles from the
                    // tensor core's operand reads
                    if (lane == 0) w_ok = tc::mbar_wait(&empty[s], ph ^ 1u) ? 1 : 0;
                    w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
                    if (!w_ok) {
                        if (lane == 0) conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                    } else {
                        const uint32_t tile = tc::smem_u32(smem + s * Cfg::STAGE);
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            const int slot = g + u * 128;
                            if (slot < nslots) {
                                int16_t *pk = prevk + s * 256 + slot;
                                gen_put(tile, (slot >> 6) * Mp, slot & 63, (int)*pk, q[d][u], a.c.M);
                                *pk = (int16_t)(int)q[d][u].x;
                            }
                        }
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(&full_a[s]);
                        load_next(q[d]);
                        s += FWD_GEN_GROUPS;
                        if (s >= NST) {
                            s -= NST;
                            ph ^= 1u;
                        }
                        cur_kt += FWD_GEN_GROUPS;
                        while (cur_kt >= a.ktiles && cur_t < ntiles) {
                            cur_kt -= a.ktiles;
                            cur_t += gridDim.x;
                        }
                    }
                }
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
// output channels over a range of K = (output position, m). Per K step the
// TMA producer stages one dw^ tile (MN-major: BN / 64 boxes of a 3-D view
// (channel, m, position), 64 k-rows each); the generators write the G
// MN-major A tiles from the records of the G row tiles' inputs (loaded
// DW_AHEAD K steps ahead), and G MMAs (one TMEM accumulator each) reuse the
// dw^ tile. Split-K over positions; each split adds its tiles into g_W
// atomically (split 0 also the dead-neuron term).
// ---------------------------------------------------------------------------
constexpr int DWG_MAX_G = 8;
constexpr int DWG_MAX_STAGES = 4;
constexpr int DW_AHEAD = 2;
constexpr int DW_MAX_SPT = 8;   // slots per generator thread: G kpos <= 8
constexpr int DW_GEN_GROUPS = 2;  // K steps generated at once
constexpr int DW_THREADS = (2 + CONV_NEPI + GEN_WARPS * DW_GEN_GROUPS) * 32;  // 576

template <int BN>
struct GenDwCfg {
    static constexpr int B_BYTES = BN * 128;
    static __host__ __device__ int stage(int G) { return G * 128 * 128 + B_BYTES; }
    static __host__ __device__ int prev_bytes(int nst, int G, int kpos) { return nst * G * 128 * kpos * 2; }
    static __host__ __device__ int smem(int nst, int G, int kpos) {
        return nst * stage(G) + prev_bytes(nst, G, kpos) + 1024 + 256;
    }
};

template <int BN>
__global__ void __launch_bounds__(DW_THREADS, 1)
    k_conv_dw_gen(const uint2 *__restrict__ rec, const __grid_constant__ CUtensorMap mapD, ConvGemmArgs a) {
    using Cfg = GenDwCfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int G = a.groups, NST = a.nst;
    const int Mp = a.Mp;
    const int kpos = 64 / Mp;
    const int STG = Cfg::stage(G);
    const int a_bytes = G * 128 * 128;
    const int slots = G * 128 * kpos;  // (row block u of the group, position kp, channel c)
    int16_t *prevk = reinterpret_cast<int16_t *>(smem + NST * STG);
    uint64_t *full_t = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(prevk) + Cfg::prev_bytes(NST, G, kpos));
    uint64_t *full_a = full_t + DWG_MAX_STAGES;
    uint64_t *empty = full_a + DWG_MAX_STAGES;
    uint64_t *acc_full = empty + DWG_MAX_STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_grp = a.n_row;  // row groups of G row tiles
    const int ntiles = n_grp * a.n_col * a.n_split;
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
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                for (int i = 0; i < nkt; ++i, ++it) {
                    if (!tc::mbar_wait_spin(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full_t[s], (uint32_t)Cfg::B_BYTES);
                    const uint32_t sb = tc::smem_u32(smem + s * STG + a_bytes);
                    for (int gq = 0; gq < BN / 64; ++gq)
                        tma_load_3d(sb + gq * 8192, &mapD, &full_t[s], ct * BN + gq * 64, 0, (kt0 + i) * kpos);
                    if (++s == NST) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i) tc::mbar_wait_spin(&full_t[i % NST], (i / NST) & 1u);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, true, true);
            uint32_t j = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                if (j >= 1) {
                    if (!tc::mbar_wait_spin(acc_empty, (j - 1) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                for (int i = 0; i < nkt; ++i) {
                    if (!tc::mbar_wait_spin(&full_t[s], ph) || !tc::mbar_wait_spin(&full_a[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * STG);
                    const uint32_t sbb = sa + a_bytes;
                    // descriptors built once: a row tile is 16 KB on (+1024), a
                    // 16-deep slice 2 KB (+128)
                    const uint64_t ad0 = tc::sdesc_sw128_mn(sa, 8192), bd0 = tc::sdesc_sw128_mn(sbb, 8192);
                    for (int gi = 0; gi < G; ++gi) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc::mma_bf16(tmem + gi * BN, ad0 + (uint64_t)(gi * 1024 + kk * 128), bd0 + (uint64_t)(kk * 128),
                                         idesc, (i > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(&empty[s]);
                    if (++s == NST) {
                        s = 0;
                        ph ^= 1u;
                    }
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
        // generator group grp (4 warps) takes K steps it = grp, grp + 2, ...
        // (the stage count is even: a stage and its slots keep their owners)
        const int gw = warp - (2 + CONV_NEPI);
        const int grp = gw / GEN_WARPS;
        const int g = (gw % GEN_WARPS) * 32 + lane;
        // K steps of tile t (split-K tiles have kt_per_split but the last)
        auto tile_nkt = [&](int t) {
            int rg, ct, kt0, nkt;
            decode(t, rg, ct, kt0, nkt);
            return nkt;
        };
        // advance a (tile t, step i of its nkt) cursor by n K steps of this CTA's sequence
        auto advance = [&](int &t, int &i, int &nkt, int n) {
            i += n;
            while (t < ntiles && i >= nkt) {
                i -= nkt;
                t += gridDim.x;
                if (t < ntiles) nkt = tile_nkt(t);
            }
        };
        // this thread's slots v: (row block u, position kp, channel c = g & 63),
        // fixed per tile: packed channel cb 64 + c (bits 0-15), kh (16-19),
        // kw (20-23), kp (24), u (25-29), valid (31)
        uint32_t spk[DW_MAX_SPT];
        int pk_t = -1, la_rg = 0, la_kt0 = 0;
        auto slot_consts = [&](int t) {
            pk_t = t;
            int ct, nkt;
            decode(t, la_rg, ct, la_kt0, nkt);
            const int ncb = a.C_in >> 6, nrb = a.k * a.k * ncb;
#pragma unroll
            for (int v = 0; v < DW_MAX_SPT; ++v) {
                const int slot = g + v * 128, qq = slot >> 6;
                const int u = qq / kpos, kp = qq - u * kpos;
                const int rb = la_rg * 2 * G + u;
                spk[v] = 0u;
                if (slot < slots && rb < nrb) {
                    const int tap = rb / ncb, cb = rb - tap * ncb;
                    const int kh = tap / a.k, kw = tap - kh * a.k;
                    spk[v] = (uint32_t)(cb * 64 + (g & 63)) | ((uint32_t)kh << 16) | ((uint32_t)kw << 20) |
                             ((uint32_t)kp << 24) | ((uint32_t)u << 25) | 0x80000000u;
                }
            }
        };
        uint2 q[DW_AHEAD][DW_MAX_SPT];
        int la_t = blockIdx.x, la_i = 0, la_nkt = la_t < ntiles ? tile_nkt(la_t) : 0;  // next K step to load
        advance(la_t, la_i, la_nkt, grp);
        auto load_next = [&](uint2(&dst)[DW_MAX_SPT]) {
            int ys[2] = {0, 0}, xs[2] = {0, 0};
            long long base[2] = {0, 0};
            bool pv[2] = {false, false};
            if (la_t < ntiles) {
                if (la_t != pk_t) slot_consts(la_t);
                // the step's kpos (<= 2) output positions
#pragma unroll
                for (int kp = 0; kp < 2; ++kp) {
                    const int p = (la_kt0 + la_i) * kpos + kp;
                    pv[kp] = kp < kpos && p < a.P_rows;
                    if (pv[kp]) {
                        int b, y, x;
                        pos_decode(p, a.Ho, a.Wo, b, y, x);
                        ys[kp] = y * a.stride - a.pad;
                        xs[kp] = x * a.stride - a.pad;
                        base[kp] = (((long long)b * a.H + ys[kp]) * a.W + xs[kp]) * a.C_in;
                    }
                }
            }
#pragma unroll
            for (int v = 0; v < DW_MAX_SPT; ++v) {
                dst[v] = make_uint2((uint32_t)REC_SILENT, 0u);
                const uint32_t w = spk[v];
                const int kh = (w >> 16) & 15, kw = (w >> 20) & 15, kp = (w >> 24) & 1;
                const int ysk = kp ? ys[1] : ys[0], xsk = kp ? xs[1] : xs[0];
                if ((w >> 31) && (kp ? pv[1] : pv[0]) && (unsigned)(ysk + kh) < (unsigned)a.H &&
                    (unsigned)(xsk + kw) < (unsigned)a.W)
                    dst[v] = __ldg(rec + (kp ? base[1] : base[0]) + (kh * a.W + kw) * a.C_in + (w & 0xffffu));
            }
            advance(la_t, la_i, la_nkt, DW_GEN_GROUPS);
        };
#pragma unroll
        for (int d = 0; d < DW_AHEAD; ++d) load_next(q[d]);
        int s = grp;  // stage of this group's next K step, and its phase
        uint32_t ph = 0;
        int cur_t = blockIdx.x, cur_i = 0, cur_nkt = cur_t < ntiles ? tile_nkt(cur_t) : 0;
        advance(cur_t, cur_i, cur_nkt, grp);
        bool ok = true;
        while (cur_t < ntiles && ok) {
#pragma unroll
            for (int d = 0; d < DW_AHEAD; ++d) {
                if (cur_t < ntiles && ok) {
                    int w_ok = 1;
                    if (lane == 0) w_ok = tc::mbar_wait(&empty[s], ph ^ 1u) ? 1 : 0;
                    w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
                    if (!w_ok) {
                        if (lane == 0) conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                    } else {
                        const uint32_t tile0 = tc::smem_u32(smem + s * STG);
#pragma unroll
                        for (int v = 0; v < DW_MAX_SPT; ++v) {
                            const int slot = g + v * 128;
                            if (slot < slots) {
                                // slot geometry from the index alone (the packed constants
                                // may already belong to the next tile)
                                const int qq = slot >> 6, u = kpos == 1 ? qq : qq >> 1, kp = qq - u * kpos;
                                int16_t *pk = prevk + s * slots + slot;
                                gen_put_mn(tile0 + (u >> 1) * 16384 + (u & 1) * 8192, kp * Mp, g & 63, (int)*pk,
                                           q[d][v], a.c.M);
                                *pk = (int16_t)(int)q[d][v].x;
                            }
                        }
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(&full_a[s]);
                        load_next(q[d]);
                        s += DW_GEN_GROUPS;
                        if (s >= NST) {
                            s -= NST;
                            ph ^= 1u;
                        }
                        advance(cur_t, cur_i, cur_nkt, DW_GEN_GROUPS);
                    }
                }
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) tc::tmem_dealloc(tmem, tcols);
}

// ---------------------------------------------------------------------------
// dW from the binned input S [P_in][Mp][C_in] read through TMA: the same CTA
// tiles as k_conv_dw_gen (G row tiles of 128 filter rows (tap, channel) by
// BN output channels over a range of K = (output position, m), split-K),
// with the A tiles loaded instead of generated: per K step and row block
// (tap, 64 channels) one box (64 channels, Mp grid steps) of S per output
// position of the step, at the input position the tap reads (outside the
// image: zeros), and BN / 64 boxes of dw^. Warps: 0 TMA (one lane), 1 MMA,
// 2-9 epilogue (fp32 atomics into g_W, dead-neuron term on the first split).
// ---------------------------------------------------------------------------
constexpr int DWT_MAX_STAGES = 8;

template <int BN>
__global__ void __launch_bounds__(CONV_THREADS, 1)
    k_conv_dw_tma(const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapD, ConvGemmArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int G = a.groups, NST = a.nst;
    const int Mp = a.Mp;
    const int kpos = 64 / Mp;
    const int a_bytes = G * 128 * 128;
    const int STG = a_bytes + BN * 128;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + NST * STG);
    uint64_t *empty = full + DWT_MAX_STAGES;
    uint64_t *acc_full = empty + DWT_MAX_STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_grp = a.n_row;
    const int ntiles = n_grp * a.n_col * a.n_split;
    const int ncb = a.C_in >> 6;
    const int nrb = a.k * a.k * ncb;  // row blocks (tap, 64 channels)
    const int Ktot = a.k * a.k * a.C_in;
    uint32_t tcols = 32;
    while ((int)tcols < G * BN) tcols <<= 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        tc::mbar_init(acc_full, 1);
        tc::mbar_init(acc_empty, CONV_NEPI);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
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
            const uint32_t tx = (uint32_t)(STG);  // 2G row blocks x kpos boxes of Mp x 128 B, and the dw^ tile
            uint32_t it = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                // the tile's row blocks: (kh, kw, channel block), or none
                int rkh[2 * DWG_MAX_G], rkw[2 * DWG_MAX_G], rcb[2 * DWG_MAX_G];
#pragma unroll
                for (int u = 0; u < 2 * DWG_MAX_G; ++u) {
                    const int rb = rg * 2 * G + u;
                    rkh[u] = -1;
                    rkw[u] = rcb[u] = 0;
                    if (u < 2 * G && rb < nrb) {
                        const int tap = rb / ncb;
                        rcb[u] = rb - tap * ncb;
                        rkh[u] = tap / a.k;
                        rkw[u] = tap - rkh[u] * a.k;
                    }
                }
                // first output position of the first K step, stepped by one
                int p = kt0 * kpos, b, y, x;
                pos_decode(p, a.Ho, a.Wo, b, y, x);
                for (int i = 0; i < nkt; ++i, ++it) {
                    if (!tc::mbar_wait_spin(&empty[s], ph ^ 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full[s], tx);
                    const uint32_t st = tc::smem_u32(smem + s * STG);
                    for (int kp = 0; kp < kpos; ++kp) {
                        const bool pv = p < a.P_rows;
                        const int ys = y * a.stride - a.pad, xs = x * a.stride - a.pad;
#pragma unroll
                        for (int u = 0; u < 2 * DWG_MAX_G; ++u) {
                            if (u < 2 * G) {
                                // a row block past the filter rows or a position past the
                                // chunk reads a box outside the tensor (zeros)
                                const bool on = pv && rkh[u] >= 0;
                                tma_load_5d(st + (u >> 1) * 16384 + (u & 1) * 8192 + kp * Mp * 128, &mapS, &full[s],
                                            rcb[u] * 64, 0, on ? xs + rkw[u] : 0, on ? ys + rkh[u] : 0, on ? b : a.ni);
                            }
                        }
                        ++p;
                        if (++x == a.Wo) {
                            x = 0;
                            if (++y == a.Ho) {
                                y = 0;
                                ++b;
                            }
                        }
                    }
                    const uint32_t sb = st + a_bytes;
                    for (int gq = 0; gq < BN / 64; ++gq)
                        tma_load_3d(sb + gq * 8192, &mapD, &full[s], ct * BN + gq * 64, 0, (kt0 + i) * kpos);
                    if (++s == NST) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            const uint32_t n_drain = it < (uint32_t)NST ? it : (uint32_t)NST;
            for (uint32_t i = it - n_drain; i < it; ++i) tc::mbar_wait_spin(&full[i % NST], (i / NST) & 1u);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, true, true);
            uint32_t j = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                int rg, ct, kt0, nkt;
                decode(t, rg, ct, kt0, nkt);
                if (j >= 1) {
                    if (!tc::mbar_wait_spin(acc_empty, (j - 1) & 1u)) {
                        conv_set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc::tc_fence_after();
                }
                for (int i = 0; i < nkt; ++i) {
                    if (!tc::mbar_wait_spin(&full[s], ph)) {
                        conv_set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t sa = tc::smem_u32(smem + s * STG);
                    const uint32_t sbb = sa + a_bytes;
                    // descriptors built once: a row tile is 16 KB on (+1024), a
                    // 16-deep slice 2 KB (+128)
                    const uint64_t ad0 = tc::sdesc_sw128_mn(sa, 8192), bd0 = tc::sdesc_sw128_mn(sbb, 8192);
                    for (int gi = 0; gi < G; ++gi) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc::mma_bf16(tmem + gi * BN, ad0 + (uint64_t)(gi * 1024 + kk * 128), bd0 + (uint64_t)(kk * 128),
                                         idesc, (i > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(&empty[s]);
                    if (++s == NST) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (ok) tc::mma_commit(acc_full);
            }
        }
        __syncwarp();
    } else {
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
                    // filter row kidx = (tap, channel) of the padded K; its place in
                    // g_W [C_out][k k C_t] (rows of padding channels are dropped)
                    int kreal = kidx, Kreal = Ktot;
                    if (a.C_t != a.C_in) {
                        const int tap = kidx / a.C_in, ch = kidx - tap * a.C_in;
                        kreal = ch < a.C_t ? tap * a.C_t + ch : -1;
                        Kreal = a.k * a.k * a.C_t;
                    }
                    if (kidx < Ktot && kreal >= 0) {
                        const int o0 = ct * BN + cc * 32;
#pragma unroll
                        for (int u = 0; u < 32; ++u) {
                            const float add = (first && a.count) ? a.qcoef * a.count[o0 + u] : 0.f;
                            atomicAdd(a.g_W + (long long)(o0 + u) * Kreal + kreal, v[u] + add);
                        }
                    }
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(acc_empty);
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
// (64, Mp, box_x, 1, 1), 128-byte swizzle, zeros outside
static bool map_act(CUtensorMap *m, const void *ptr, int ni, int h, int w, int Mp, int C, int box_x = 1) {
    EncodeFn enc = conv_encode();
    if (!enc) return false;
    cuuint64_t dims[5] = {(cuuint64_t)C, (cuuint64_t)Mp, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)ni};
    cuuint64_t strides[4] = {(cuuint64_t)C * 2, (cuuint64_t)Mp * C * 2, (cuuint64_t)w * Mp * C * 2,
                             (cuuint64_t)h * w * Mp * C * 2};
    cuuint32_t box[5] = {64, (cuuint32_t)Mp, (cuuint32_t)box_x, 1, 1};
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

template <int BN, bool RES>
static cudaError_t launch_fwd_gen_bn(const uint2 *rec, const CUtensorMap &mB, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = GenFwdCfg<BN, RES>;
    const int fixed = a.res_bytes + Cfg::PREV_BYTES + 1024 + 256;
    int nst = (GEN_SMEM_MAX - fixed) / Cfg::STAGE;
    if (nst > Cfg::MAX_STAGES) nst = Cfg::MAX_STAGES;
    nst -= nst % FWD_GEN_GROUPS;  // each stage belongs to one generator group
    if (nst < FWD_GEN_GROUPS) return cudaErrorInvalidConfiguration;
    a.nst = nst;
    const int smem = Cfg::smem(nst, a.res_bytes);
    cudaError_t e = cudaFuncSetAttribute(k_conv_fwd_gen<BN, RES>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_fwd_gen<BN, RES><<<grid, FWD_THREADS, smem, st>>>(rec, mB, a);
    return cudaGetLastError();
}

// dw^ [P][Mp][C] bf16 as a 3-D map (C, Mp, P), boxes of (64, Mp, 64 / Mp):
// the 64 k-rows (position, m) of one K step of dW, 128-byte swizzle
static bool map_act3(CUtensorMap *m, const void *ptr, long long P, int Mp, int C) {
    EncodeFn enc = conv_encode();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)C, (cuuint64_t)Mp, (cuuint64_t)P};
    cuuint64_t strides[2] = {(cuuint64_t)C * 2, (cuuint64_t)Mp * C * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)Mp, (cuuint32_t)(64 / Mp)};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN>
static cudaError_t launch_dw_gen_bn(const uint2 *rec, const CUtensorMap &mD, ConvGemmArgs a, cudaStream_t st) {
    using Cfg = GenDwCfg<BN>;
    const int kpos = 64 / a.Mp;
    int nst = DWG_MAX_STAGES;
    while (nst > DW_GEN_GROUPS && Cfg::smem(nst, a.groups, kpos) > GEN_SMEM_MAX) nst -= DW_GEN_GROUPS;
    if (Cfg::smem(nst, a.groups, kpos) > GEN_SMEM_MAX) return cudaErrorInvalidConfiguration;
    a.nst = nst;
    const int smem = Cfg::smem(nst, a.groups, kpos);
    cudaError_t e = cudaFuncSetAttribute(k_conv_dw_gen<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col * a.n_split;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_dw_gen<BN><<<grid, DW_THREADS, smem, st>>>(rec, mD, a);
    return cudaGetLastError();
}

template <int BN, bool ROWBOX, bool RES, bool FWD>
static cudaError_t launch_tap_bn(const CUtensorMap &mA, const CUtensorMap &mB, const CUtensorMap &mR, ConvGemmArgs a,
                                 DsPlan pl, cudaStream_t st) {
    const int smem = pl.nst * pl.stage + pl.res_bytes + pl.epi_bytes + 1024 + 256;
    cudaError_t e = cudaFuncSetAttribute(k_conv_tap_gemm<BN, ROWBOX, RES, FWD>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int ntiles = a.n_row * a.n_col;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
    k_conv_tap_gemm<BN, ROWBOX, RES, FWD><<<grid, CONV_THREADS, smem, st>>>(mA, mB, mR, a, pl);
    return cudaGetLastError();
}

template <int BN, bool RES>
static cudaError_t launch_ds_pair_bn(const CUtensorMap &mA, const CUtensorMap &mB, ConvGemmArgs a, DsPlan pl,
                                     cudaStream_t st) {
    const int smem = pl.nst * pl.stage + pl.res_bytes + pl.epi_bytes + 1024 + 256;
    cudaError_t e =
        cudaFuncSetAttribute(k_conv_ds_pair<BN, RES>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int npairs = (a.n_row / 2) * a.n_col;
    const int grid = npairs < conv_num_sms() ? npairs : conv_num_sms();
    k_conv_ds_pair<BN, RES><<<grid, CONV_THREADS, smem, st>>>(mA, mB, a, pl);
    return cudaGetLastError();
}

static ConvGemmArgs base_args(const ConvGeom &g, int ni, const LifConst &c) {
    ConvGemmArgs a{};
    a.ni = ni;
    a.H = g.H;
    a.W = g.W;
    a.C_in = g.C;
    a.C_t = g.C;
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
    const int Cp = conv_padded_channels(g.C);
    return Cp % 64 == 0 && C_out % 64 == 0 && (C_out <= 128 || C_out % 128 == 0) && (Mp == 32 || Mp == 64) &&
           g.k <= 7 && Cp * g.k * g.k <= 65535 && C_out * g.k * g.k <= 65535;
}

int conv_padded_channels(int C) { return C < 64 ? 64 : C; }

cudaError_t launch_dwhat_pmc(const float *t_out, const int *q, const float *s, const float *vdot, const float *g_up,
                             long long P, int C, const LifConst &c, __nv_bfloat16 *D, float *count,
                             cudaStream_t st) {
    // a warp covers one position or one segment of 32 NPT channels of it
    constexpr int NPT = DWHAT_NPT;
    if (C % 64 != 0 || (C > 32 * NPT && C % (32 * NPT) != 0)) return cudaErrorInvalidValue;
    long long blocks = (P * ((C + 32 * NPT - 1) / (32 * NPT)) + 7) / 8;  // 8 warps per block
    // 64-channel positions: each warp builds the position's block in shared
    // memory (8 KB; at 128 channels the 16 KB buffers leave one block per SM,
    // and direct stores are faster)
    const bool bulk = C <= 64;
    const int smem = bulk ? 8 * c.Mp * C * 2 : 0;
    const long long cap = (long long)(bulk ? (227 * 1024) / smem : 8) * conv_num_sms();
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (bulk) {
        cudaError_t e = cudaFuncSetAttribute(k_dwhat_pmc<NPT, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        k_dwhat_pmc<NPT, true><<<(unsigned)blocks, 256, smem, st>>>(t_out, q, s, vdot, g_up, P, C, c, D, count);
    } else {
        k_dwhat_pmc<NPT, false><<<(unsigned)blocks, 256, 0, st>>>(t_out, q, s, vdot, g_up, P, C, c, D, count);
    }
    return cudaGetLastError();
}

cudaError_t launch_filters_t(const float *W, int C_out, int T, int C_in, int C_pad, __nv_bfloat16 *Wt,
                             cudaStream_t st) {
    const long long n = (long long)C_out * T * C_pad;
    long long blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    k_filters_t<<<(unsigned)blocks, 256, 0, st>>>(W, C_out, T, C_in, C_pad, Wt);
    return cudaGetLastError();
}

// shared-memory plan of the tap-shifted contraction (see DsPlan)
static DsPlan tap_plan(int k, int ppt, int Mp, int BN, bool resident, long long res, bool rowbox, int epi_bytes, int ncb,
                       int smem_max = GEN_SMEM_MAX) {
    DsPlan pl{};
    pl.taps_per_unit = rowbox ? k : 1;
    pl.a_bytes = rowbox ? (ppt + k - 1) * Mp * 128 : 128 * 128;
    pl.b_bytes = resident ? 0 : pl.taps_per_unit * BN * 128;
    pl.stage = (pl.a_bytes + pl.b_bytes + 1023) & ~1023;
    pl.res_bytes = resident ? (int)res : 0;
    pl.units = (rowbox ? k : k * k) * ncb;
    pl.epi_bytes = epi_bytes;
    const int nst = (smem_max - pl.res_bytes - epi_bytes - 1280) / pl.stage;
    pl.nst = nst > DS_MAX_STAGES ? DS_MAX_STAGES : nst;
    return pl;
}

// dS of ni images with the input-time gradient: dw^ [ni Ho Wo][Mp][C_out],
// Wt [C_in][k k C_out], t_in [ni H W][C_in] -> g_t_in (zeroed first)
cudaError_t launch_conv_ds_gemm(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *dW_hat,
                                const __nv_bfloat16 *Wt, const float *t_in, float *g_t_in, int C_t, cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.H * g.W;
    const int BN = pick_bn(g.C);
    const int ppt = 128 / c.Mp;
    const int ncb = C_out / 64;
    a.n_col = g.C / BN;
    a.t_in = t_in;
    a.g_t_in = g_t_in;
    a.C_t = C_t;
    cudaError_t e = cudaMemsetAsync(g_t_in, 0, sizeof(float) * (size_t)a.P_rows * C_t, st);
    if (e != cudaSuccess) return e;
    // resident transposed filters when they are small; one box per filter row
    // at stride 1 when every tile lies within one image row
    const long long res = (long long)g.k * g.k * ncb * BN * 128;
    const bool resident = a.n_col == 1 && res <= 80 * 1024;
    auto plan = [&](bool rowbox) { return tap_plan(g.k, ppt, c.Mp, BN, resident, res, rowbox, DS_EPI_BYTES, ncb); };
    const bool row_ok = g.s == 1 && g.W % ppt == 0 && ppt + g.k - 1 <= 256;
    DsPlan pl = plan(row_ok);
    bool rowbox = row_ok && pl.nst >= 2;
    if (!rowbox) pl = plan(false);
    if (pl.nst < 2) return cudaErrorInvalidConfiguration;
    // stride classes (one for stride 1); a stride whose s x s classes do not
    // fit runs every tap in the identity order, off-grid taps reading zeros
    const bool classes = g.s * g.s <= DS_MAX_CLS;
    pl.ps = classes ? g.s : 1;
    pl.ts = classes ? g.s : 1;
    pl.ncls = 0;
    a.n_row = 0;
    for (int py = 0; py < pl.ps; ++py)
        for (int px = 0; px < pl.ps; ++px) {
            DsClass q{};
            q.py = py;
            q.px = px;
            q.Hc = g.H > py ? (g.H - py + pl.ps - 1) / pl.ps : 0;
            q.Wc = g.W > px ? (g.W - px + pl.ps - 1) / pl.ps : 0;
            q.count = ni * q.Hc * q.Wc;
            q.kh0 = (py + g.p) % pl.ts;
            q.kw0 = (px + g.p) % pl.ts;
            q.nkh = q.kh0 < g.k ? (g.k - q.kh0 + pl.ts - 1) / pl.ts : 0;
            q.nkw = q.kw0 < g.k ? (g.k - q.kw0 + pl.ts - 1) / pl.ts : 0;
            if (q.count == 0 || q.nkh * q.nkw == 0) continue;  // no tap reaches it: its gradient stays zero
            pl.cls[pl.ncls++] = q;
        }
    // most taps first, so that the persistent CTAs' last tiles are the light ones
    for (int i = 1; i < pl.ncls; ++i)
        for (int j = i; j > 0 && pl.cls[j].nkh * pl.cls[j].nkw > pl.cls[j - 1].nkh * pl.cls[j - 1].nkw; --j) {
            const DsClass q = pl.cls[j];
            pl.cls[j] = pl.cls[j - 1];
            pl.cls[j - 1] = q;
        }
    for (int i = 0; i < pl.ncls; ++i) {
        pl.cls[i].tile0 = a.n_row;
        a.n_row += (pl.cls[i].count + ppt - 1) / ppt;
    }
    if (a.n_row == 0) return cudaSuccess;
    CUtensorMap mA, mB, mR;
    if (!map_mat(&mB, Wt, g.C, g.k * g.k * C_out, BN)) return cudaErrorInvalidValue;
    // two row tiles at once when image rows hold whole pairs (one class,
    // an even number of row tiles), for 64-wide column tiles
    if (rowbox && g.W % (2 * ppt) == 0 && 2 * ppt + g.k - 1 <= 256 && BN == 64 && pl.ncls == 1 &&
        a.n_row % 2 == 0) {
        DsPlan pq = pl;
        pq.a_bytes = (2 * ppt + g.k - 1) * c.Mp * 128;
        pq.b_bytes = resident ? 0 : g.k * BN * 128;
        pq.stage = (pq.a_bytes + pq.b_bytes + 1023) & ~1023;
        const int nst = (GEN_SMEM_MAX - pq.res_bytes - pq.epi_bytes - 1280) / pq.stage;
        pq.nst = nst > DS_MAX_STAGES ? DS_MAX_STAGES : nst;
        if (pq.nst >= 2 && map_act(&mA, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out, 2 * ppt + g.k - 1))
            return resident ? launch_ds_pair_bn<64, true>(mA, mB, a, pq, st)
                            : launch_ds_pair_bn<64, false>(mA, mB, a, pq, st);
    }
    if (!map_act(&mA, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out, rowbox ? ppt + g.k - 1 : 1)) return cudaErrorInvalidValue;
    pl.run_ok = map_act(&mR, dW_hat, ni, g.Ho, g.Wo, c.Mp, C_out, ppt) ? 1 : 0;
    if (!pl.run_ok) mR = mA;
#define DSTD_DS(BNV)                                                                                   \
    if (rowbox) return resident ? launch_tap_bn<BNV, true, true, false>(mA, mB, mR, a, pl, st)         \
                                : launch_tap_bn<BNV, true, false, false>(mA, mB, mR, a, pl, st);       \
    return resident ? launch_tap_bn<BNV, false, true, false>(mA, mB, mR, a, pl, st)                    \
                    : launch_tap_bn<BNV, false, false, false>(mA, mB, mR, a, pl, st);
    switch (BN) {
        case 256: { DSTD_DS(256) }
        case 128: { DSTD_DS(128) }
        default: { DSTD_DS(64) }
    }
#undef DSTD_DS
}

// forward of ni images from the binned input S [ni H W][Mp][C_in] and the
// filters Wf [C_out][k k C_in], with the scan/solve/select in the epilogue:
// spike outputs [ni Ho Wo][C_out], penalty sums added into penalty[4]
cudaError_t launch_conv_fwd_tma(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                                const __nv_bfloat16 *Wf, const float *rowsum, float *t_out, int *q, float *s,
                                float *vdot, float *penalty, cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    a.t_out = t_out;
    a.q_out = q;
    a.s_out = s;
    a.vdot_out = vdot;
    a.rowsum = rowsum;
    a.penalty = penalty;
    const int BN = pick_bn(C_out);
    const int ppt = 128 / c.Mp;
    const int ncb = g.C / 64;
    a.n_col = C_out / BN;
    a.n_row = (a.P_rows + ppt - 1) / ppt;
    if (a.n_row == 0) return cudaSuccess;
    const long long res = (long long)g.k * g.k * ncb * BN * 128;
    const bool resident = a.n_col == 1 && res <= 80 * 1024;
    const bool row_ok = g.s == 1 && g.Wo % ppt == 0 && ppt + g.k - 1 <= 256;
    DsPlan pl = tap_plan(g.k, ppt, c.Mp, BN, resident, res, row_ok, fwd_epi_bytes(false), ncb);
    if (row_ok && pl.nst < 2 && BN == 128) {
        // the tight epilogue rows and the device's whole opt-in shared memory
        int dev = 0, optin = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) == cudaSuccess)
            pl = tap_plan(g.k, ppt, c.Mp, BN, resident, res, true, fwd_epi_bytes(true), ncb, optin);
    }
    const bool rowbox = row_ok && pl.nst >= 2;
    if (!rowbox) pl = tap_plan(g.k, ppt, c.Mp, BN, resident, res, false, fwd_epi_bytes(false), ncb);
    if (pl.nst < 2) return cudaErrorInvalidConfiguration;
    // every tap of every output position, in position order
    pl.ncls = 1;
    pl.ps = pl.ts = 1;
    DsClass &cl = pl.cls[0];
    cl.py = cl.px = 0;
    cl.Hc = g.Ho;
    cl.Wc = g.Wo;
    cl.count = a.P_rows;
    cl.tile0 = 0;
    cl.kh0 = cl.kw0 = 0;
    cl.nkh = cl.nkw = g.k;
    CUtensorMap mA, mB, mR;
    if (!map_act(&mA, S, ni, g.H, g.W, c.Mp, g.C, rowbox ? ppt + g.k - 1 : 1) ||
        !map_mat(&mB, Wf, C_out, g.k * g.k * g.C, BN))
        return cudaErrorInvalidValue;
    pl.run_ok = map_act(&mR, S, ni, g.H, g.W, c.Mp, g.C, ppt) ? 1 : 0;
    if (!pl.run_ok) mR = mA;
#define DSTD_FT(BNV)                                                                                   \
    if (rowbox) return resident ? launch_tap_bn<BNV, true, true, true>(mA, mB, mR, a, pl, st)          \
                                : launch_tap_bn<BNV, true, false, true>(mA, mB, mR, a, pl, st);        \
    return resident ? launch_tap_bn<BNV, false, true, true>(mA, mB, mR, a, pl, st)                     \
                    : launch_tap_bn<BNV, false, false, true>(mA, mB, mR, a, pl, st);
    switch (BN) {
        case 256: { DSTD_FT(256) }
        case 128: { DSTD_FT(128) }
        default: { DSTD_FT(64) }
    }
#undef DSTD_FT
}

// dW of ni images from the binned input S [ni H W][Mp][C_in] and dw^
// [ni Ho Wo][Mp][C_out], added into g_W (zeroed by the caller before the
// first chunk)
cudaError_t launch_conv_dw_tma(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                               const __nv_bfloat16 *dW_hat, const float *count, float qcoef, float *g_W, int C_t,
                               cudaStream_t st) {
    ConvGemmArgs a = base_args(g, ni, c);
    a.C_t = C_t;
    a.C_out = C_out;
    a.P_rows = ni * g.Ho * g.Wo;
    if (a.P_rows == 0) return cudaSuccess;
    const int BN = pick_bn(C_out);
    const int Ktot = g.k * g.k * g.C;
    const int row_tiles = (Ktot / 64 + 1) / 2;
    const int kpos = 64 / c.Mp;
    const int extra = 1024 + 256;  // alignment and barriers
    auto stg = [&](int G) { return G * 16384 + BN * 128; };
    // the most row tiles per CTA (one dw^ tile feeds them all) that TMEM
    // holds and that leave three stages
    int gmax = 512 / BN;
    if (gmax > DWG_MAX_G) gmax = DWG_MAX_G;
    while (gmax > 1 && 3 * stg(gmax) + extra > GEN_SMEM_MAX) --gmax;
    const int ngrp = (row_tiles + gmax - 1) / gmax;
    a.groups = (row_tiles + ngrp - 1) / ngrp;
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
    int nst = (GEN_SMEM_MAX - extra) / stg(a.groups);
    if (nst > DWT_MAX_STAGES) nst = DWT_MAX_STAGES;
    if (nst < 2) return cudaErrorInvalidConfiguration;
    a.nst = nst;
    a.g_W = g_W;
    a.count = count;
    a.qcoef = qcoef;
    CUtensorMap mS, mD;
    if (!map_act(&mS, S, ni, g.H, g.W, c.Mp, g.C, 1) || !map_act3(&mD, dW_hat, (long long)a.P_rows, c.Mp, C_out))
        return cudaErrorInvalidValue;
    const int smem = nst * stg(a.groups) + extra;
    const int ntiles = tiles * a.n_split;
    const int grid = ntiles < conv_num_sms() ? ntiles : conv_num_sms();
#define DSTD_DWT(BNV)                                                                                            \
    {                                                                                                            \
        cudaError_t e = cudaFuncSetAttribute(k_conv_dw_tma<BNV>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem); \
        if (e != cudaSuccess) return e;                                                                          \
        k_conv_dw_tma<BNV><<<grid, CONV_THREADS, smem, st>>>(mS, mD, a);                                         \
        return cudaGetLastError();                                                                               \
    }
    switch (BN) {
        case 256: DSTD_DWT(256)
        case 128: DSTD_DWT(128)
        default: DSTD_DWT(64)
    }
#undef DSTD_DWT
}

bool conv_bin_S_supported(int C) {
    return C % 64 == 0 && C <= BINS_THREADS * BINS_MAXSPT && (C <= BINS_THREADS || C % BINS_THREADS == 0);
}

cudaError_t launch_bin_S(const float *t, long long P, int C, int Ct, const LifConst &c, __nv_bfloat16 *S,
                         cudaStream_t st) {
    const int Mp = c.Mp;
    if (!conv_bin_S_supported(C) || Ct < 1 || Ct > C || P >= (1ll << 31) || P * Mp * C >= (1ll << 31))
        return cudaErrorInvalidValue;
    if (P == 0) return cudaSuccess;
    const int R = C >= BINS_THREADS ? 1 : BINS_THREADS / C;
    const int smem = 2 * R * Mp * C * 2;
    if (smem > 227 * 1024) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_bin_S, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const long long ngroups = (P + R - 1) / R;
    int per_sm = (227 * 1024) / smem;
    if (per_sm > 8) per_sm = 8;
    long long blocks = (long long)per_sm * conv_num_sms();
    if (blocks > ngroups) blocks = ngroups;
    k_bin_S<<<(unsigned)blocks, BINS_THREADS, smem, st>>>(t, (int)P, C, Ct, c, S);
    return cudaGetLastError();
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
    CUtensorMap mB;
    if (!map_mat(&mB, Wf, C_out, g.k * g.k * g.C, BN)) return cudaErrorInvalidValue;
    if (resident) {
        switch (BN) {
            case 256: return launch_fwd_gen_bn<256, true>(rec, mB, a, st);
            case 128: return launch_fwd_gen_bn<128, true>(rec, mB, a, st);
            default: return launch_fwd_gen_bn<64, true>(rec, mB, a, st);
        }
    }
    switch (BN) {
        case 256: return launch_fwd_gen_bn<256, false>(rec, mB, a, st);
        case 128: return launch_fwd_gen_bn<128, false>(rec, mB, a, st);
        default: return launch_fwd_gen_bn<64, false>(rec, mB, a, st);
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
    if (gmax * kpos > DW_MAX_SPT) gmax = DW_MAX_SPT / kpos;
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
    CUtensorMap mD;
    if (!map_act3(&mD, dW_hat, (long long)a.P_rows, c.Mp, C_out)) return cudaErrorInvalidValue;
    switch (BN) {
        case 256: return launch_dw_gen_bn<256>(rec, mD, a, st);
        case 128: return launch_dw_gen_bn<128>(rec, mD, a, st);
        default: return launch_dw_gen_bn<64>(rec, mD, a, st);
    }
}

}  // namespace dstd
