// Tensor-core contraction of the DSTD layer on sm_103a (tcgen05 + TMA).
//
// D[r, c] = sum_k A[r, k] B[c, k] with A and B 16-bit, staged by TMA
// (128-byte swizzle, no multicast) through a STAGES-deep mbarrier ring. A is
// K-major; B is K-major ([C, K] rows) or, with BMN, MN-major ([K, C] rows:
// the tensor core reads it transposed, so an operand written for one
// contraction serves the transposed one without a second copy). One
// thread issues tcgen05.mma (cta_group::1, M = 128, N = BN, K = 16 per
// instruction) into fp32 accumulators in TMEM; eight warps read them back
// with tcgen05.ld (lane = row) and run the epilogue:
//   Store  plain fp32 tile (w^ of the forward, rows = (sample, grid step),
//          columns = neurons; split-K partials of the weight gradient),
//   GradT  rows = inputs, columns = (sample, grid step): the input-time
//          gradient sum_m dS ds/dt, so dS never reaches HBM.
// The three-product split (fp32 operand = 16-bit hi + lo) accumulates
// hi*hi + hi*lo + lo*hi (three MMAs per K step). The tensor core's fp32
// accumulation error grows with the number of MMAs summed into one
// accumulator, so the main hi*hi products of successive k-tiles go round-robin
// into P_MAIN separate TMEM accumulators and the small corrections into one
// more; the epilogue adds them in fp32 registers.
//
// Every mbarrier wait is bounded (about 2 s of %globaltimer); an expired wait
// sets the device status word, skips the epilogue and frees TMEM.
#include "dstd_internal.cuh"
#include "dstd_tc_ptx.cuh"

#include <cuda.h>
#include <atomic>
#include <mutex>

namespace dstd {

// device status word: bit STATUS_TIMEOUT is set by an expired bounded wait
__device__ unsigned int g_status = 0;

__device__ __forceinline__ void set_status(unsigned int code) { atomicOr(&g_status, code); }

cudaError_t status_read(unsigned int *out, int clear) {
    cudaError_t e = cudaMemcpyFromSymbol(out, g_status, sizeof(unsigned int));
    if (e != cudaSuccess || !clear) return e;
    unsigned int z = 0;
    return cudaMemcpyToSymbol(g_status, &z, sizeof(z));
}

namespace tc {

// One thread waits on a barrier phase that never completes; the bounded wait
// expires and records a timeout in the status word.
__global__ void k_wait_selftest(unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (!mbar_wait(&bar, 0, limit_ns)) set_status(STATUS_TIMEOUT);
    }
}

// The tile's value at columns [cc, cc+32) of this lane: the sum of the n_main
// main accumulators (columns p*BN + cc) and, with corr, the correction one.
template <int BN>
__device__ __forceinline__ void tmem_ld_acc(uint32_t tbase, int cc, int n_main, bool corr, float (&v)[32]) {
    tmem_ld32(tbase + cc, v);
    for (int p = 1; p < n_main; ++p) {
        float u[32];
        tmem_ld32(tbase + p * BN + cc, u);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] += u[j];
    }
    if (corr) {
        float u[32];
        tmem_ld32(tbase + 3 * BN + cc, u);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] += u[j];
    }
}

template <int NPASS, int BN>
struct Cfg {
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int NOP = (NPASS == 3) ? 2 : 1;
    static constexpr int STAGE = NOP * (A_BYTES + B_BYTES);
    static constexpr int STAGES = (200 * 1024) / STAGE > 8 ? 8 : (200 * 1024) / STAGE;
    static constexpr int SMEM = STAGES * STAGE + 1024 + 256;
    // accumulators: P_MAIN round-robin copies of the tile for the main
    // products (plus one for the hi*lo + lo*hi corrections when NPASS = 3)
    static constexpr int P_MAIN = (NPASS == 3) ? 3 : 4;
    static constexpr uint32_t TMEM_COLS = 4 * BN;  // 512 for BN = 128
    static_assert(TMEM_COLS <= 512, "TMEM holds 512 columns");
};

// ---------------------------------------------------------------------------
// Epilogues. Each thread owns one accumulator row (its TMEM lane).
// ---------------------------------------------------------------------------
// ---------------------------------------------------------------------------
// Epilogues. Each epilogue warp owns one TMEM lane quarter (rows 32q..32q+31)
// and one column group; a thread owns one accumulator row. The work on a
// chunk of 32 columns is written against registers, so a tile whose group
// chunk is a single one can be drained from TMEM first (and TMEM handed back
// to the MMA warp) before the chunk is processed.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void store_chunk(const float (&v)[32], int row, int col0, int cc, int R, int Cn,
                                            const TcEpiArgs &a, int split) {
    if (row >= R) return;
    const float rs = a.row_scale ? a.row_scale[row] : 1.0f;
    if (a.atomic) {
        const float add = (a.qcount && split == 0) ? a.qcoef * a.qcount[row] : 0.0f;
        float *dst = a.D + (long long)row * a.ldd + col0 + cc;
        if (col0 + cc + 32 <= Cn && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
            for (int j = 0; j < 32; j += 4)
                atomicAdd(reinterpret_cast<float4 *>(dst + j), make_float4(fmaf(v[j], rs, add), fmaf(v[j + 1], rs, add),
                                                                           fmaf(v[j + 2], rs, add),
                                                                           fmaf(v[j + 3], rs, add)));
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (col0 + cc + j < Cn) atomicAdd(dst + j, fmaf(v[j], rs, add));
        }
        return;
    }
    float *D = a.D + (long long)split * a.zstride;
    float *dst = D + (long long)row * a.ldd + col0 + cc;
    if (col0 + cc + 32 <= Cn && (a.ldd % 4) == 0) {
#pragma unroll
        for (int j = 0; j < 32; j += 4)
            *reinterpret_cast<float4 *>(dst + j) =
                make_float4(v[j] * rs, v[j + 1] * rs, v[j + 2] * rs, v[j + 3] * rs);
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (col0 + cc + j < Cn) dst[j] = v[j] * rs;
    }
}

// Input-time gradient over one chunk (dense: row = input j; conv: row = tap).
template <int SUB>
__device__ __forceinline__ void gradt_chunk(const float (&v)[32], int row, int colbase, BinW &w, float &g,
                                            const TcEpiArgs &a) {
    const LifConst &c = a.c;
    const int Mp = c.Mp;
#pragma unroll
    for (int sb = 0; sb < 32; sb += SUB) {
        const int col = colbase + sb;
        const int m0 = col & (Mp - 1);
        const int b = col / Mp;
        long long e = -1;  // input element this (row, sample) reads; -1 = none
        if (row < a.N && b < a.B) {
            if (!a.conv) {
                e = (long long)b * a.N + row;
            } else {
                const ConvGeom &geo = a.g;
                const int pos = a.pos0 + b;
                const int cch = row % geo.C, kw = (row / geo.C) % geo.k, kh = row / (geo.C * geo.k);
                const int x = pos % geo.Wo, y = (pos / geo.Wo) % geo.Ho, bb = pos / (geo.Wo * geo.Ho);
                const int iy = y * geo.s + kh - geo.p, ix = x * geo.s + kw - geo.p;
                if (iy >= 0 && iy < geo.H && ix >= 0 && ix < geo.W)
                    e = (((long long)bb * geo.H + iy) * geo.W + ix) * geo.C + cch;
            }
        }
        if (m0 == 0) {
            g = 0.f;
            w.k = -100;
            if (e >= 0) {
                if (a.bw) {
                    const float4 q = a.bw[e];
                    w.k = __float_as_int(q.x);
                    w.dR = q.y;
                    w.dL = q.z;
                } else {
                    const float x = a.t_in[e];
                    if (isfinite(x)) w = bin_weights(c, x, true);
                }
            }
        }
        // the two grid points of the spike (m = k, k + 1), if in this block
#pragma unroll
        for (int j = 0; j < SUB; ++j) {
            const int m = m0 + j;
            g += (m == w.k && m < c.M) ? v[sb + j] * w.dR : 0.f;
            g += (m == w.k + 1 && m < c.M) ? v[sb + j] * w.dL : 0.f;
        }
        if (m0 + SUB == Mp && e >= 0) {
            if (a.conv) atomicAdd(&a.g_t_in[e], g);
            else a.g_t_in[e] = g;
        }
    }
}

// ---------------------------------------------------------------------------
// The kernel: persistent, one CTA per SM looping over output tiles.
//   warp 0      TMA producer (one lane)
//   warp 1      TMEM allocation, MMA issuer (one lane)
//   warps 2-9   epilogue (warp w: lane quarter w % 4, column group (w-2)/4 of
//               64 columns; a thread owns one accumulator row of its group)
// Barriers: full/empty per smem stage; acc_full (MMA -> epilogue, per tile);
// acc_empty (epilogue -> MMA: the accumulator may be overwritten), 8 warps.
// ---------------------------------------------------------------------------
constexpr int NEPI = 8;
constexpr int NTHREADS = (2 + NEPI) * 32;
constexpr int GCOLS = 64;  // accumulator columns per epilogue warp group (BN / (NEPI / 4))

struct TileInfo {
    int row0, col0, kt0, nkt, split;
};

__device__ __forceinline__ TileInfo tile_info(int t, int n_row, int n_col, int ktiles, int kt_per_split, int BNv) {
    TileInfo ti;
    const int per_split = n_row * n_col;
    ti.split = t / per_split;
    const int rem = t % per_split;
    ti.row0 = (rem % n_row) * BM;
    ti.col0 = (rem / n_row) * BNv;
    ti.kt0 = ti.split * kt_per_split;
    ti.nkt = ktiles - ti.kt0;
    if (ti.nkt > kt_per_split) ti.nkt = kt_per_split;
    return ti;
}

template <int NPASS, int BN, int EPI, bool F16, bool BMN>
__global__ void __launch_bounds__(NTHREADS, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap mA_hi, const __grid_constant__ CUtensorMap mA_lo,
              const __grid_constant__ CUtensorMap mB_hi, const __grid_constant__ CUtensorMap mB_lo, int R, int Cn,
              int ktiles, int kt_per_split, int n_row, int n_col, int n_split, TcEpiArgs args) {
    using C = Cfg<NPASS, BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + C::STAGES * C::STAGE);
    uint64_t *empty = full + C::STAGES;
    uint64_t *acc_full = empty + C::STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = n_row * n_col * n_split;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(acc_empty, NEPI);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // TMA producer: stage ring shared by all tiles of this CTA
            uint32_t it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                const TileInfo ti = tile_info(t, n_row, n_col, ktiles, kt_per_split, BN);
                for (int i = 0; i < ti.nkt; ++i, ++it) {
                    const int s = it % C::STAGES;
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait(&empty[s], ph ^ 1u)) {
                        set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(&full[s], (uint32_t)C::STAGE);
                    const int kx = (ti.kt0 + i) * BK;
                    const uint32_t st = smem_u32(smem + s * C::STAGE);
                    tma_load_2d(st, &mA_hi, &full[s], kx, ti.row0);
                    if (NPASS == 3) tma_load_2d(st + C::A_BYTES, &mA_lo, &full[s], kx, ti.row0);
                    const uint32_t sb = st + C::NOP * C::A_BYTES;
                    if (!BMN) {
                        tma_load_2d(sb, &mB_hi, &full[s], kx, ti.col0);
                        if (NPASS == 3) tma_load_2d(sb + C::B_BYTES, &mB_lo, &full[s], kx, ti.col0);
                    } else {
                        // BK rows of k, each 64 columns wide per box
#pragma unroll
                        for (int h = 0; h < BN / 64; ++h) {
                            tma_load_2d(sb + h * (BK * 128), &mB_hi, &full[s], ti.col0 + 64 * h, kx);
                            if (NPASS == 3)
                                tma_load_2d(sb + C::B_BYTES + h * (BK * 128), &mB_lo, &full[s], ti.col0 + 64 * h, kx);
                        }
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            // MMA issuer
            constexpr uint32_t idesc = idesc_16bit(BM, BN, F16, BMN);
            uint32_t it = 0, j = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++j) {
                const TileInfo ti = tile_info(t, n_row, n_col, ktiles, kt_per_split, BN);
                if (j > 0) {
                    // the epilogue of the previous tile has taken the accumulator
                    if (!mbar_wait(acc_empty, (j - 1) & 1u)) {
                        set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc_fence_after();
                }
                for (int i = 0; i < ti.nkt; ++i, ++it) {
                    const int s = it % C::STAGES;
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait(&full[s], ph)) {
                        set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_hi = smem_u32(smem + s * C::STAGE);
                    const uint32_t a_lo = a_hi + C::A_BYTES;
                    const uint32_t b_hi = a_hi + C::NOP * C::A_BYTES;
                    const uint32_t b_lo = b_hi + C::B_BYTES;
                    const uint32_t acc_main = tmem + (uint32_t)((i % C::P_MAIN) * BN);
                    const uint32_t acc_corr = tmem + (uint32_t)(3 * BN);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint64_t da = sdesc_sw128(a_hi + kk * 32);
                        // K step of 16: 32 bytes along a K-major row, or 16
                        // rows (two 1024-byte atoms) of an MN-major tile
                        const uint64_t db = BMN ? sdesc_sw128_mn(b_hi + kk * 2048, BK * 128) : sdesc_sw128(b_hi + kk * 32);
                        mma_bf16(acc_main, da, db, idesc, (i >= C::P_MAIN || kk > 0) ? 1u : 0u);
                        if (NPASS == 3) {
                            const uint64_t dbl =
                                BMN ? sdesc_sw128_mn(b_lo + kk * 2048, BK * 128) : sdesc_sw128(b_lo + kk * 32);
                            mma_bf16(acc_corr, da, dbl, idesc, (i > 0 || kk > 0) ? 1u : 0u);
                            mma_bf16(acc_corr, sdesc_sw128(a_lo + kk * 32), db, idesc, 1u);
                        }
                    }
                    mma_commit(&empty[s]);
                }
                if (ok) mma_commit(acc_full);
            }
        }
        __syncwarp();
    } else {
        // epilogue warps
        const int ew = warp - 2;
        const int quarter = warp & 3, group = ew >> 2;
        const uint32_t tbase = tmem + ((uint32_t)(quarter * 32) << 16);
        // columns of a group: GCOLS, or a whole sample when one spans more
        const int span = (EPI != (int)Epi::Store && args.c.Mp > GCOLS) ? args.c.Mp : GCOLS;
        int c_lo = group * span, c_hi = c_lo + span;
        if (c_lo >= BN) c_lo = c_hi = BN;
        if (c_hi > BN) c_hi = BN;
        uint32_t j = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++j) {
            const TileInfo ti = tile_info(t, n_row, n_col, ktiles, kt_per_split, BN);
            if (!mbar_wait_sleep(acc_full, j & 1u)) {
                set_status(STATUS_TIMEOUT);
                break;
            }
            tc_fence_after();
            const int row = ti.row0 + quarter * 32 + lane;
            const int n_main = ti.nkt < C::P_MAIN ? ti.nkt : C::P_MAIN;
            const bool corr = (NPASS == 3);
            if (c_hi - c_lo == GCOLS) {
                // drain the group's chunks, hand the accumulator back, then work
                float v[GCOLS / 32][32];
#pragma unroll
                for (int h = 0; h < GCOLS / 32; ++h) tmem_ld_acc<BN>(tbase, c_lo + 32 * h, n_main, corr, v[h]);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(acc_empty);
                if (EPI == (int)Epi::Store) {
#pragma unroll
                    for (int h = 0; h < GCOLS / 32; ++h) store_chunk(v[h], row, ti.col0, c_lo + 32 * h, R, Cn, args, ti.split);
                } else {
                    BinW w{-100, 0.f, 0.f, 0.f, 0.f};
                    float g = 0.f;
                    if (args.c.Mp == 8) {
#pragma unroll
                        for (int h = 0; h < GCOLS / 32; ++h) gradt_chunk<8>(v[h], row, ti.col0 + c_lo + 32 * h, w, g, args);
                    } else if (args.c.Mp == 16) {
#pragma unroll
                        for (int h = 0; h < GCOLS / 32; ++h) gradt_chunk<16>(v[h], row, ti.col0 + c_lo + 32 * h, w, g, args);
                    } else {
#pragma unroll
                        for (int h = 0; h < GCOLS / 32; ++h) gradt_chunk<32>(v[h], row, ti.col0 + c_lo + 32 * h, w, g, args);
                    }
                }
            } else {
                // a sample spans more than GCOLS columns (Mp > GCOLS) or the
                // group is idle: work chunk by chunk out of TMEM, then hand it back
                BinW w{-100, 0.f, 0.f, 0.f, 0.f};
                float g = 0.f;
                for (int cc = c_lo; cc < c_hi; cc += 32) {
                    float v[32];
                    tmem_ld_acc<BN>(tbase, cc, n_main, corr, v);
                    if (EPI == (int)Epi::GradT) gradt_chunk<32>(v, row, ti.col0 + cc, w, g, args);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(acc_empty);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, C::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Two-SM variant (tcgen05 cta_group::2). Clusters of two CTAs compute output
// tiles of 256 rows x 128 columns, the MMA's M = 256 spanning the pair: each
// CTA holds its own 128 rows of A and half (64 rows) of the tile's B in
// shared memory, and the MMA issued by the even CTA reads B from both. Per
// 64-deep K step of x3 an SM so takes in 48 KB of operands instead of 64 KB
// for the same tensor work. D rows 0..127 of a tile land in the even CTA's
// TMEM, rows 128..255 in the odd CTA's.
//   full[s]    the even CTA's collects both CTAs' TMA bytes (the odd CTA's
//              loads signal it remotely; the even CTA's producer arms it);
//   empty[s]   in both CTAs, released by the even CTA's MMA commit (multicast);
//   acc_full   in both CTAs, by the same commit after a tile's last MMA;
//   acc_empty  the even CTA's, arrived on by the epilogue warps of both.
// Epilogue StoreT: D^T[c][r] = acc[r][c] * col_scale[c], the transposed
// store (the forward computes w^ as S W^T: rows (b, m), columns i, written
// as w^[i][(b, m)]; consecutive lanes, consecutive addresses).
// Every wait is bounded; neither CTA leaves before the other (cluster
// barrier), and the pair frees its TMEM together.
// ---------------------------------------------------------------------------
constexpr int BM2 = 128;  // A rows per CTA (256 per pair)
constexpr int BNH = 64;   // B rows per CTA (128 per pair: the MMA's N)

template <int NPASS>
struct Cfg2 {
    static constexpr int A_BYTES = BM2 * BK * 2;
    static constexpr int B_BYTES = BNH * BK * 2;
    static constexpr int NOP = (NPASS == 3) ? 2 : 1;
    static constexpr int STAGE = NOP * (A_BYTES + B_BYTES);
    static constexpr int STAGES = (200 * 1024) / STAGE > 8 ? 8 : (200 * 1024) / STAGE;
    static constexpr int SMEM = STAGES * STAGE + 1024 + 256;
    static constexpr int P_MAIN = (NPASS == 3) ? 3 : 4;
    static constexpr int BNP = 2 * BNH;               // accumulator columns
    static constexpr uint32_t TMEM_COLS = 4 * BNP;    // 512
};

__device__ __forceinline__ uint32_t mapa_rank(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}

// TMA load into this CTA's shared memory whose completion is signalled on an
// mbarrier of either CTA of the pair (a shared::cluster address)
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void mma_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n"
        ".reg .pred p;\n"
        "setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n"
        "}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit_pair(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            smem_u32(bar)),
        "h"((uint16_t)3)
        : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t *slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n"
        ".reg .pred p;\n"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n"
        "selp.u32 %0, 1, 0, p;\n"
        "}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
        : "memory");
    return ok != 0;
}

// bounded wait at cluster scope (barriers that a peer CTA arrives on)
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t *bar, uint32_t parity, bool sleep) {
    const uint64_t t0 = globaltimer();
    for (;;) {
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if (globaltimer() - t0 > WAIT_NS) return false;
        if (sleep) __nanosleep(256);
    }
}

template <int NPASS, bool F16>
__global__ void __launch_bounds__(NTHREADS, 1)
    k_tc_gemm_pair(const __grid_constant__ CUtensorMap mA_hi, const __grid_constant__ CUtensorMap mA_lo,
                   const __grid_constant__ CUtensorMap mB_hi, const __grid_constant__ CUtensorMap mB_lo, int R,
                   int Cn, int ktiles, int n_row, int n_col, TcEpiArgs args) {
    using C = Cfg2<NPASS>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + C::STAGES * C::STAGE);
    uint64_t *empty = full + C::STAGES;
    uint64_t *acc_full = empty + C::STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = (int)cluster_ctarank();
    const int cid = (int)cluster_id_x(), ncl = (int)cluster_count_x();
    const bool leader = rank == 0;
    const int ntiles = n_row * n_col;  // tiles of 256 x 128

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(acc_empty, 2 * NEPI);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) tmem_alloc_pair(tmem_slot, C::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers exist before any remote signal
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // TMA producer of this CTA's half of every stage
            const uint32_t full0 = mapa_rank(smem_u32(&full[0]), 0);
            uint32_t it = 0;
            bool ok = true;
            for (int t = cid; t < ntiles && ok; t += ncl) {
                const int row0 = (t % n_row) * (2 * BM2) + rank * BM2;
                const int brow0 = (t / n_row) * (2 * BNH) + rank * BNH;
                for (int i = 0; i < ktiles; ++i, ++it) {
                    const int s = it % C::STAGES;
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait_cluster(&empty[s], ph ^ 1u, false)) {
                        set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    if (leader) mbar_expect_tx(&full[s], (uint32_t)(2 * C::STAGE));
                    const uint32_t fb = full0 + (uint32_t)(s * sizeof(uint64_t));
                    const int kx = i * BK;
                    const uint32_t st = smem_u32(smem + s * C::STAGE);
                    tma_load_2d_pair(st, &mA_hi, fb, kx, row0);
                    if (NPASS == 3) tma_load_2d_pair(st + C::A_BYTES, &mA_lo, fb, kx, row0);
                    const uint32_t sb = st + C::NOP * C::A_BYTES;
                    tma_load_2d_pair(sb, &mB_hi, fb, kx, brow0);
                    if (NPASS == 3) tma_load_2d_pair(sb + C::B_BYTES, &mB_lo, fb, kx, brow0);
                }
            }
            if (ok) {
                // every stage released by the pair's MMAs: no commit targets this CTA afterwards
                for (int i = 0; i < C::STAGES; ++i, ++it) {
                    const int s = it % C::STAGES;
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait_cluster(&empty[s], ph ^ 1u, false)) {
                        set_status(STATUS_TIMEOUT);
                        break;
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0 && leader) {
            // MMA issuer of the pair
            constexpr uint32_t idesc = idesc_16bit(2 * BM2, C::BNP, F16);
            uint32_t it = 0, j = 0;
            bool ok = true;
            for (int t = cid; t < ntiles && ok; t += ncl, ++j) {
                if (j > 0) {
                    // both CTAs' epilogues have taken the previous tile
                    if (!mbar_wait_cluster(acc_empty, (j - 1) & 1u, false)) {
                        set_status(STATUS_TIMEOUT);
                        break;
                    }
                    tc_fence_after();
                }
                for (int i = 0; i < ktiles; ++i, ++it) {
                    const int s = it % C::STAGES;
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait_cluster(&full[s], ph, false)) {
                        set_status(STATUS_TIMEOUT);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_hi = smem_u32(smem + s * C::STAGE);
                    const uint32_t a_lo = a_hi + C::A_BYTES;
                    const uint32_t b_hi = a_hi + C::NOP * C::A_BYTES;
                    const uint32_t b_lo = b_hi + C::B_BYTES;
                    const uint32_t acc_main = tmem + (uint32_t)((i % C::P_MAIN) * C::BNP);
                    const uint32_t acc_corr = tmem + (uint32_t)(3 * C::BNP);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint64_t da = sdesc_sw128(a_hi + kk * 32);
                        const uint64_t db = sdesc_sw128(b_hi + kk * 32);
                        mma_pair(acc_main, da, db, idesc, (i >= C::P_MAIN || kk > 0) ? 1u : 0u);
                        if (NPASS == 3) {
                            mma_pair(acc_corr, da, sdesc_sw128(b_lo + kk * 32), idesc, (i > 0 || kk > 0) ? 1u : 0u);
                            mma_pair(acc_corr, sdesc_sw128(a_lo + kk * 32), db, idesc, 1u);
                        }
                    }
                    mma_commit_pair(&empty[s]);
                }
                if (ok) mma_commit_pair(acc_full);
            }
        }
        __syncwarp();
    } else {
        // epilogue warps of both CTAs: this CTA's 128 rows of the tile
        const int ew = warp - 2;
        const int quarter = warp & 3, group = ew >> 2;
        const uint32_t tbase = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t acc_empty0 = mapa_rank(smem_u32(acc_empty), 0);
        const int c_lo = group * GCOLS;
        const int n_main = ktiles < C::P_MAIN ? ktiles : C::P_MAIN;
        uint32_t j = 0;
        for (int t = cid; t < ntiles; t += ncl, ++j) {
            const int row = (t % n_row) * (2 * BM2) + rank * BM2 + quarter * 32 + lane;
            const int col0 = (t / n_row) * C::BNP + c_lo;
            if (!mbar_wait_cluster(acc_full, j & 1u, true)) {
                set_status(STATUS_TIMEOUT);
                break;
            }
            tc_fence_after();
            float v[GCOLS / 32][32];
#pragma unroll
            for (int h = 0; h < GCOLS / 32; ++h) tmem_ld_acc<C::BNP>(tbase, c_lo + 32 * h, n_main, NPASS == 3, v[h]);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acc_empty0);
            if (row < R) {
#pragma unroll
                for (int h = 0; h < GCOLS / 32; ++h) {
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) {
                        const int col = col0 + 32 * h + jj;
                        if (col < Cn) {
                            const float cs = args.row_scale ? args.row_scale[col] : 1.0f;
                            args.D[(long long)col * args.ldd + row] = v[h][jj] * cs;
                        }
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // both epilogues done with TMEM, every remote arrive landed
    if (warp == 1) tmem_dealloc_pair(tmem, C::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Host side: tensor maps and launch.
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// rows x cols 16-bit matrix with row stride ld elements; box = box_rows x 64
static bool make_map(CUtensorMap *m, const void *ptr, int rows, int cols, int ld, int box_rows, bool f16) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t gstride[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(m, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                     const_cast<void *>(ptr), gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static int num_sms() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
    }
    return n;
}

template <int NPASS, int BN, int EPI, bool F16, bool BMN>
static cudaError_t launch_one(const CUtensorMap &a_hi, const CUtensorMap &a_lo, const CUtensorMap &b_hi,
                              const CUtensorMap &b_lo, int R, int Cn, int K, int splits, const TcEpiArgs &args,
                              cudaStream_t st) {
    using C = Cfg<NPASS, BN>;
    cudaError_t e = cudaFuncSetAttribute(k_tc_gemm<NPASS, BN, EPI, F16, BMN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    const int ktiles = (K + BK - 1) / BK;
    const int per = (ktiles + splits - 1) / splits;
    const int n_row = (R + BM - 1) / BM, n_col = (Cn + BN - 1) / BN;
    const long long ntiles = (long long)n_row * n_col * splits;
    const int grid = (int)(ntiles < num_sms() ? ntiles : num_sms());
    k_tc_gemm<NPASS, BN, EPI, F16, BMN><<<grid, NTHREADS, C::SMEM, st>>>(a_hi, a_lo, b_hi, b_lo, R, Cn, ktiles, per,
                                                                            n_row, n_col, splits, args);
    return cudaGetLastError();
}

}  // namespace tc

cudaError_t launch_wait_selftest(unsigned long long limit_ns, cudaStream_t st) {
    tc::k_wait_selftest<<<1, 32, 0, st>>>(limit_ns);
    return cudaGetLastError();
}

namespace tc {
// SM pairs that can hold a pair kernel's clusters at once (a pair must sit in
// one GPC: a GPC with an odd number of usable SMs leaves one out)
template <int NPASS, bool F16>
static int resident_pairs() {
    static int resident = 0;
    if (resident == 0) {
        using C = Cfg2<NPASS>;
        auto kern = k_tc_gemm_pair<NPASS, F16>;
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) != cudaSuccess) return 0;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cfg.blockDim = dim3(NTHREADS);
        cfg.dynamicSmemBytes = C::SMEM;
        cfg.gridDim = dim3((num_sms() / 2) * 2);
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) return 0;
        resident = n;
    }
    return resident;
}

template <int NPASS, bool F16>
static cudaError_t launch_pair(const CUtensorMap &a_hi, const CUtensorMap &a_lo, const CUtensorMap &b_hi,
                               const CUtensorMap &b_lo, int R, int Cn, int K, const TcEpiArgs &args,
                               cudaStream_t st) {
    using C = Cfg2<NPASS>;
    auto kern = k_tc_gemm_pair<NPASS, F16>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    const int ktiles = (K + BK - 1) / BK;
    const int n_row = (R + 2 * BM2 - 1) / (2 * BM2), n_col = (Cn + C::BNP - 1) / C::BNP;
    const long long ntiles = (long long)n_row * n_col;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.blockDim = dim3(NTHREADS);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = st;
    // persistent: as many pairs as can be resident at once
    const int resident = resident_pairs<NPASS, F16>();
    if (resident < 1) return cudaErrorInvalidConfiguration;
    const int pairs = (int)(ntiles < resident ? ntiles : resident);
    cfg.gridDim = dim3(2 * pairs);
    return cudaLaunchKernelEx(&cfg, kern, a_hi, a_lo, b_hi, b_lo, R, Cn, ktiles, n_row, n_col, args);
}
}  // namespace tc

// Work on the busiest SM, in units of one K step of a single-CTA tile: rounds
// of 128 x 128 tiles on single CTAs, (K steps + 2) each, against rounds of
// 256 x 128 tiles on resident SM pairs, (0.92 K steps + 4) each. A pair's K
// step is cheaper (each SM takes in 48 KB instead of 64 KB of operands), its
// tile boundary dearer (the handshakes between the two SMs); fitted to the
// 784-wide forward of the MLP (13 K steps: single CTAs faster) and 4096- and
// 8192-wide layers (64 and 128 K steps: pairs faster, 85-90% against 83% of
// the bf16 peak).
static std::atomic<int> g_pair_policy{0};

int tc_gemm_pair_policy(int policy) {
    if (policy < 0 || policy > 2) return g_pair_policy.load();
    return g_pair_policy.exchange(policy);
}

bool tc_gemm_pair_preferred(int R, int Cn, int K, OpKind op) {
    if (op != OpKind::F16X3 && op != OpKind::BF16) return false;
    const int policy = g_pair_policy.load();
    if (policy != 0) return policy == 1;
    const int pairs = tc_gemm_resident_pairs(op);
    if (pairs < 1) return false;
    const long long t1 = (long long)((R + 127) / 128) * ((Cn + 127) / 128);
    const long long t2 = (long long)((R + 255) / 256) * ((Cn + 127) / 128);
    const long long r1 = (t1 + tc::num_sms() - 1) / tc::num_sms(), r2 = (t2 + pairs - 1) / pairs;
    const double kt = (double)((K + tc::BK - 1) / tc::BK);
    return (double)r2 * (0.92 * kt + 4.0) < (double)r1 * (kt + 2.0);
}

int tc_gemm_resident_pairs(OpKind op) {
    return op == OpKind::F16X3    ? tc::resident_pairs<3, true>()
           : op == OpKind::BF16X3 ? tc::resident_pairs<3, false>()
                                  : tc::resident_pairs<1, false>();
}

cudaError_t launch_tc_gemm_pair_storeT(const void *A_hi, const void *A_lo, int lda, const void *B_hi, const void *B_lo,
                                       int ldb, int R, int Cn, int K, OpKind op, const TcEpiArgs &args,
                                       cudaStream_t st) {
    CUtensorMap a_hi, a_lo, b_hi, b_lo;
    const bool three = (op == OpKind::BF16X3 || op == OpKind::F16X3);
    const bool f16 = (op == OpKind::F16X3);
    if (op == OpKind::F32) return cudaErrorInvalidValue;
    if (!tc::make_map(&a_hi, A_hi, R, K, lda, tc::BM2, f16) || !tc::make_map(&b_hi, B_hi, Cn, K, ldb, tc::BNH, f16))
        return cudaErrorInvalidValue;
    if (three) {
        if (!tc::make_map(&a_lo, A_lo, R, K, lda, tc::BM2, f16) || !tc::make_map(&b_lo, B_lo, Cn, K, ldb, tc::BNH, f16))
            return cudaErrorInvalidValue;
        return f16 ? tc::launch_pair<3, true>(a_hi, a_lo, b_hi, b_lo, R, Cn, K, args, st)
                   : tc::launch_pair<3, false>(a_hi, a_lo, b_hi, b_lo, R, Cn, K, args, st);
    }
    a_lo = a_hi;
    b_lo = b_hi;
    return tc::launch_pair<1, false>(a_hi, a_lo, b_hi, b_lo, R, Cn, K, args, st);
}

int tc_gemm_splits_valid(int K, int splits) {
    const int ktiles = (K + tc::BK - 1) / tc::BK;
    const int per = (ktiles + splits - 1) / splits;
    return per * (splits - 1) < ktiles;
}

cudaError_t launch_tc_gemm(const void *A_hi, const void *A_lo, int lda, const void *B_hi, const void *B_lo, int ldb,
                           int R, int Cn, int K, int splits, OpKind op, Epi epi, const TcEpiArgs &args,
                           cudaStream_t st, bool b_mn) {
    constexpr int BN = 128;
    CUtensorMap a_hi, a_lo, b_hi, b_lo;
    const bool three = (op == OpKind::BF16X3 || op == OpKind::F16X3);
    const bool f16 = (op == OpKind::F16X3);
    if (op == OpKind::F32) return cudaErrorInvalidValue;
    // the Store epilogue runs with a K-major B, the GradT one with an MN-major B
    if (b_mn != (epi == Epi::GradT)) return cudaErrorInvalidValue;
    // K-major B: [Cn, K] rows, boxes of BN rows x 64 k; MN-major B: [K, Cn]
    // rows, boxes of 64 k-rows x 64 columns
    auto map_b = [&](CUtensorMap *m, const void *p) {
        return b_mn ? tc::make_map(m, p, K, Cn, ldb, tc::BK, f16) : tc::make_map(m, p, Cn, K, ldb, BN, f16);
    };
    if (!tc::make_map(&a_hi, A_hi, R, K, lda, tc::BM, f16) || !map_b(&b_hi, B_hi)) return cudaErrorInvalidValue;
    if (three) {
        if (!tc::make_map(&a_lo, A_lo, R, K, lda, tc::BM, f16) || !map_b(&b_lo, B_lo)) return cudaErrorInvalidValue;
    } else {
        a_lo = a_hi;
        b_lo = b_hi;
    }
    if (splits < 1) splits = 1;
#define DSTD_TC_LAUNCH(NP, F)                                                                                      \
    switch (epi) {                                                                                                 \
        case Epi::Store: return tc::launch_one<NP, BN, 0, F, false>(a_hi, a_lo, b_hi, b_lo, R, Cn, K, splits, args, st); \
        default: return tc::launch_one<NP, BN, 1, F, true>(a_hi, a_lo, b_hi, b_lo, R, Cn, K, splits, args, st);          \
    }
    if (f16) {
        DSTD_TC_LAUNCH(3, true)
    } else if (three) {
        DSTD_TC_LAUNCH(3, false)
    } else {
        DSTD_TC_LAUNCH(1, false)
    }
#undef DSTD_TC_LAUNCH
}

}  // namespace dstd
