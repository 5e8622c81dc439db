// Internal declarations of libdstd: per-layer constants, LIF device math,
// launch helpers. Not part of the public ABI (include/dstd.h).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/dstd.h"

namespace dstd {

// ---------------------------------------------------------------------------
// Per-layer constants, computed on the host in double and rounded once.
//
// With rates av = 1/tau_m, aI = 1/tau_s (0 for an infinite constant) and
// lam = aI - av, the spike kernel of Tab. kernel is, for every row,
//     K(s) = e^{-av s} phi(s),  phi(s) = (1 - e^{-lam s}) / lam  (= s if lam = 0),
// the response of v to a unit impulse in I. The DSTD kernel of
// Tab. DSTD_kernels becomes, with r = t - T_k in [0, dt) for a spike in bin k,
//     weight at T_k     : e^{av r} phi(dt - r) / phi(dt)        (t >= 0 column)
//     weight at T_{k+1} : e^{aI (r - dt)} phi(r) / phi(dt)       (t < 0 column)
// which is the table's expression rewritten with expm1 so that no difference
// of nearly equal exponentials is formed.
// ---------------------------------------------------------------------------
struct LifConst {
    float av, aI, lam;     // rates; lam = aI - av
    int lam_zero;          // lam == 0 exactly (tau_m == tau_s, incl. both inf)
    float inv_lam;         // 1 / lam (0 when lam_zero)
    float T0, dt, inv_dt;  // T_0 = t_first - t_offset, step
    float rv, rI, KD;      // e^{-av dt}, e^{-aI dt}, K(dt)
    float inv_phi_dt;      // 1 / phi(dt)
    float vth;
    int M, Mp;             // steps, padded bin axis of the internal layouts
    float vdot_floor;      // lower bound on dv^/dt at a spike (1e-6 v_th / dt)
    float Kmax;            // max of K(s) over s in [0, dt] (with a 1e-6 relative margin)
    float Kmax4;           // the same over [0, 4 dt]
    float t_head, t_tail, g_head, g_tail, g_q, norm;
};

LifConst make_const(const dstd_params &p, int Mp);
int padded_M(int M);       // next power of two >= max(M, 8)

__device__ __forceinline__ float phi_f(const LifConst &c, float x) {
    return c.lam_zero ? x : -expm1f(-c.lam * x) / c.lam;
}
// inverse of phi: the s with phi(s) = y (needs 1 - lam y > 0)
__device__ __forceinline__ float phi_inv_f(const LifConst &c, float y) {
    return c.lam_zero ? y : -log1pf(-c.lam * y) / c.lam;
}
// K(s) = e^{-av s} phi(s), s >= 0
__device__ __forceinline__ float kernel_K(const LifConst &c, float s) {
    return __expf(-c.av * s) * phi_f(c, s);
}

// DSTD grid weights of one finite spike t: bin k (= floor((t - T0)/dt)), the
// weights wR at T_k and wL at T_{k+1}, and optionally their t-derivatives.
struct BinW {
    int k;
    float wR, wL, dR, dL;
};
// the grid step k of a finite spike t (clamped far outside the grid)
__device__ __forceinline__ float bin_floor(const LifConst &c, float t) { return floorf((t - c.T0) * c.inv_dt); }
__device__ __forceinline__ int bin_index(const LifConst &c, float t) {
    return (int)fmaxf(fminf(bin_floor(c, t), 1e9f), -1e9f);
}
__device__ __forceinline__ BinW bin_weights(const LifConst &c, float t, bool deriv) {
    BinW b;
    const float kf = bin_floor(c, t);
    b.k = bin_index(c, t);
    float r = t - (c.T0 + kf * c.dt);
    r = fminf(fmaxf(r, 0.0f), c.dt);
    float pR = phi_f(c, c.dt - r), pL = phi_f(c, r);
    float eR = expf(c.av * r), eL = expf(c.aI * (r - c.dt));
    b.wR = eR * pR * c.inv_phi_dt;
    b.wL = eL * pL * c.inv_phi_dt;
    if (deriv) {
        // d/dr of the two columns: phi'(x) = e^{-lam x}
        float dpR = c.lam_zero ? 1.0f : expf(-c.lam * (c.dt - r));
        float dpL = c.lam_zero ? 1.0f : expf(-c.lam * r);
        b.dR = eR * (c.av * pR - dpR) * c.inv_phi_dt;
        b.dL = eL * (c.aI * pL + dpL) * c.inv_phi_dt;
    } else {
        b.dR = b.dL = 0.0f;
    }
    return b;
}

// ---------------------------------------------------------------------------
// Scan over the M intervals of one neuron (Tab. timing_DSTD via state).
//
// The prefix sums a_iq, b_iq of Tab. timing_DSTD are carried as the exact
// state (v, I) at T_q: at each grid point I jumps by w^_q, and over one step
// (v, I) <- (rv v + KD I, rI I). On interval q the potential is
//     v^(s) = e^{-av s} (v_q + phi(s) I_q),  s = t - T_q in [0, dt),
// with at most one interior extremum. The first interval whose maximum
// reaches v_th holds the spike. The scan only finds that interval (a cheap
// bound, max(v_q, 0) + max(I_q, 0) Kmax >= v_th, gates the exact checks);
// its root is solved once afterwards (scan_finish), by safeguarded Newton,
// so the lanes of a warp solve together instead of once per interval.
// ---------------------------------------------------------------------------
struct ScanState {
    float v, I;
    int q;       // M while silent
    float v0, I0, hi;  // state at T_q and bracket end of the firing interval
    float s, vdot;
};

__device__ __forceinline__ void scan_reset(ScanState &st, int M) {
    st.v = 0.f; st.I = 0.f; st.q = M; st.v0 = 0.f; st.I0 = 0.f; st.hi = 0.f; st.s = 0.f; st.vdot = 0.f;
}

__device__ __forceinline__ float vhat_at(const LifConst &c, float v0, float I0, float s) {
    return __expf(-c.av * s) * (v0 + phi_f(c, s) * I0);
}

// first root of v^(s) = v_th on [0, hi] given v^(0) < v_th <= v^(hi):
// Newton from the secant guess inside the shrinking bracket (bisection when a
// step leaves it). v^ - v_th is formed with one rounding (fma, accurate
// exponentials), so its fp32 noise is about 1e-7 v_th. The iteration ends
// with the Newton step taken from a point where |v^ - v_th| <= 4e-7 v_th
// (which lands within the noise of the root), or when the step or the
// bracket is below 1e-6 dt: two or three steps from the secant guess; a
// nearly tangential crossing can fall back to bisection, hence up to 24.
__device__ __forceinline__ float interval_root(const LifConst &c, float v0, float I0, float hi) {
    if (c.av == 0.0f) {
        // v^ = v0 + phi(s) I0 is monotone here: invert phi in closed form
        float s = phi_inv_f(c, (c.vth - v0) / I0);
        return fminf(fmaxf(s, 0.0f), hi);
    }
    const float tol = 1e-6f * c.dt;
    const float ftol = 4e-7f * fabsf(c.vth);
    float lo = 0.0f;
    const float vhi = vhat_at(c, v0, I0, hi);
    float s = (vhi > v0) ? hi * __fdividef(c.vth - v0, vhi - v0) : 0.5f * hi;
    s = fminf(fmaxf(s, 0.0f), hi);
    for (int it = 0; it < 24; ++it) {
        const float em = expf(-c.av * s);
        const float ph = c.lam_zero ? s : -expm1f(-c.lam * s) * c.inv_lam;
        const float f = fmaf(em, fmaf(ph, I0, v0), -c.vth);
        if (f > 0.0f) hi = s; else lo = s;
        // dv^/ds = -av v^ + I0 e^{-aI s}, with e^{-aI s} = e^{-av s} (1 - lam phi(s))
        const float df = fmaf(I0 * em, 1.0f - c.lam * ph, -c.av * (f + c.vth));
        // (the step is self-correcting: a fast quotient is enough)
        float sn = s - __fdividef(f, df);
        if (!(df > 0.0f) || !(sn >= lo) || !(sn <= hi)) sn = 0.5f * (lo + hi);
        const bool done = fabsf(f) <= ftol || fabsf(sn - s) <= tol || hi - lo <= tol;
        s = sn;
        if (done) break;
    }
    return fminf(fmaxf(s, 0.0f), hi);
}

// Exact firing test of one interval whose cheap bound reached v_th: the
// bracket end for the root (0 if v^ is already at v_th at T_q, dt if v^(dt)
// >= v_th, the interior maximum if only that reaches v_th), or -1. Out of
// line where it runs once per interval (scan_step), inline where it runs
// once per block of intervals (scan_block).
__device__ __forceinline__ float interval_test(float av, float aI, float lam, int lam_zero, float rI, float dt,
                                               float vth, float v0, float I0, float ve) {
    if (v0 >= vth) return 0.0f;
    if (ve >= vth) return dt;
    if (av > 0.0f && aI > 0.0f && I0 > 0.0f) {
        // interior maximum: dv^/ds > 0 at s = 0 and < 0 at s = dt
        const float d0 = -av * v0 + I0;
        const float dE = -av * ve + rI * I0;
        if (d0 > 0.0f && dE < 0.0f) {
            // e^{-lam s*} = 1 + lam y with y = (av v0 - I0)/(I0 aI)
            const float y = (av * v0 - I0) / (I0 * aI);
            float sp = lam_zero ? -y : -log1pf(lam * y) / lam;
            sp = fminf(fmaxf(sp, 0.0f), dt);
            const float ph = lam_zero ? sp : -expm1f(-lam * sp) / lam;
            if (__expf(-av * sp) * (v0 + ph * I0) >= vth) return sp;
        }
    }
    return -1.0f;
}
// Consume w^_m for the SUB intervals m0 .. m0+SUB-1 of one neuron at once,
// with the grid weights in registers (w[off + j] * rs for interval m0 + j).
// Same result as SUB calls of scan_step, in two phases so that the lanes of
// a warp stay together: a branch-free pass runs the recurrence and picks the
// first interval where v^ reaches v_th at an end point, or has an interior
// maximum that the cheap bound does not exclude; the exact test then runs
// once, for all lanes at their own candidate. Only an interior maximum that
// stays below v_th fails it; the pass then restarts after that interval.
template <int SUB>
__device__ __forceinline__ void scan_block(const LifConst &c, ScanState &st, const float (&w)[32], int off, float rs,
                                           int m0) {
    if (st.q < c.M) return;
    const int nvalid = c.M - m0;  // intervals of the block below M
    if (nvalid <= 0) return;
    const float v_in = st.v, I_in = st.I;
    int j0 = 0;
    for (int pass = 0; pass < SUB; ++pass) {
        float v = v_in, I = I_in;
        int cand = SUB;
        float cv0 = 0.f, cI0 = 0.f, cve = 0.f;
#pragma unroll
        for (int j = 0; j < SUB; ++j) {
            const float I0 = I + w[off + j] * rs;
            const float ve = c.rv * v + c.KD * I0;
            // v^ reaches v_th at an end of the interval, or may at an
            // interior maximum (rising at s = 0, falling at s = dt, bound met)
            const float d0 = -c.av * v + I0;
            const float dE = -c.av * ve + c.rI * I0;
            const bool endp = (v >= c.vth) | (ve >= c.vth);
            const bool peak = (d0 > 0.0f) & (dE < 0.0f) & (fmaxf(v, 0.0f) + fmaxf(I0, 0.0f) * c.Kmax >= c.vth);
            const bool take = (cand == SUB) & (j >= j0) & (j < nvalid) & (endp | peak);
            cand = take ? j : cand;
            cv0 = take ? v : cv0;
            cI0 = take ? I0 : cI0;
            cve = take ? ve : cve;
            v = ve;
            I = c.rI * I0;
        }
        if (pass == 0) {
            st.v = v;
            st.I = I;
        }
        if (cand == SUB) return;
        const float hi = interval_test(c.av, c.aI, c.lam, c.lam_zero, c.rI, c.dt, c.vth, cv0, cI0, cve);
        if (hi >= 0.0f) {
            st.q = m0 + cand;
            st.v0 = cv0;
            st.I0 = cI0;
            st.hi = hi;
            return;
        }
        j0 = cand + 1;
    }
}

// Root of the firing interval and dv^/dt there (once per neuron).
__device__ __forceinline__ void scan_finish(const LifConst &c, ScanState &st) {
    if (st.q >= c.M) return;
    const float s = st.hi > 0.0f ? interval_root(c, st.v0, st.I0, st.hi) : 0.0f;
    st.s = s;
    // dv^/dt at the spike, -av v_th + I(t), formed with one rounding: when
    // it is small the two terms nearly cancel
    st.vdot = fmaxf(fmaf(st.I0, expf(-c.aI * s), -c.av * c.vth), c.vdot_floor);
}

// Temporal penalty of one firing neuron (Eq. temporal_penalty) and dT/dt,
// both times norm.
__device__ __forceinline__ void penalty_T(const LifConst &c, float t, float &val, float &grad) {
    val = 0.f; grad = 0.f;
    if (t < c.t_head) { float d = t - c.t_head; val += c.g_head * d * d; grad += 2.f * c.g_head * d; }
    if (t > c.t_tail) { float d = t - c.t_tail; val += c.g_tail * d * d; grad += 2.f * c.g_tail * d; }
    val *= c.norm; grad *= c.norm;
}

// ---------------------------------------------------------------------------
// The walk over the bins of one neuron from w^ held in shared memory, shared
// by the scan kernel and the conv forward's fused epilogue, and the per-neuron
// outputs with the penalty sums.
// ---------------------------------------------------------------------------
// Exact test of an interval whose v^ has an interior maximum (dv^/ds > 0 at
// s = 0, < 0 at s = dt) and whose cheap bound reached v_th: the bracket end
// for the root, or -1. Before the exact maximum (a log and two exponentials)
// it tries a tighter bound: on [0, s*] v^ >= v0 and e^{-aI s} <= 1 give
//   v^(s*) <= v0 + max_s [ -av v0 s + I0 (1 - e^{-aI s}) / aI ],
// whose maximiser has e^{-aI s} = av v0 / I0. Out of line: it runs rarely.
static __device__ __noinline__ float interior_test(float av, float aI, float lam, int lam_zero, float rI, float dt,
                                                   float vth, float v0, float I0, float ve) {
    if (!(av > 0.0f && aI > 0.0f && I0 > 0.0f)) return -1.0f;
    float g;
    const float inv_aI = 1.0f / aI;
    if (v0 > 0.0f) {
        const float sm = logf(I0 / (av * v0)) * inv_aI;
        g = sm < dt ? -av * v0 * sm + (I0 - av * v0) * inv_aI : -av * v0 * dt + I0 * (1.0f - rI) * inv_aI;
    } else {
        g = -av * v0 * dt + I0 * (1.0f - rI) * inv_aI;
    }
    // margin: rounding of the bound's own terms
    if (v0 + g + 1e-6f * (fabsf(v0) + fabsf(g)) < vth) return -1.0f;
    return interval_test(av, aI, lam, lam_zero, rI, dt, vth, v0, I0, ve);
}

// One interval of the walk, with explicit fma so that the fast pass and the
// exact pass round alike: the end state and the two flags.
struct BinStep {
    float ve, In;
    bool endp, peak;
};
__device__ __forceinline__ BinStep bin_step(const LifConst &c, float v, float I0) {
    BinStep r;
    r.ve = fmaf(c.KD, I0, c.rv * v);
    r.In = c.rI * I0;
    r.endp = r.ve >= c.vth;
    r.peak = (fmaf(-c.av, v, I0) > 0.0f) & (fmaf(-c.av, r.ve, r.In) < 0.0f) &
             (fmaf(fmaxf(I0, 0.0f), c.Kmax, fmaxf(v, 0.0f)) >= c.vth);
    return r;
}

// The two passes over SUB bins m0 .. m0+SUB-1 of one neuron, whose w^
// values sit in row[0 .. SUB) (shared memory, zero past mend; 16-byte
// aligned when VEC, read as float4), starting from the state (v, I) at T_m0.
// On a spike, fills st (bin, state at its start, bracket end) and returns
// true; otherwise leaves (v, I) at the end of the block.
template <int SUB, bool VEC = true>
__device__ __forceinline__ bool scan_walk(const LifConst &c, const float *row, int m0, int mend, float &v, float &I,
                                          ScanState &st) {
    static_assert(SUB % 8 == 0 && SUB <= 32, "blocks of 8, 16 or 32 bins");
    constexpr int NCK = SUB / 8;  // kept states per block
    float kv[NCK], kI[NCK];
    uint32_t mask = 0u;
    const unsigned lanes = __activemask();
#pragma unroll
    for (int g = 0; g < SUB; g += 4) {
        if ((g & 7) == 0) {
            kv[g >> 3] = v;
            kI[g >> 3] = I;
        }
        float xs[4];
        if (VEC) {
            const float4 x = *reinterpret_cast<const float4 *>(row + g);
            xs[0] = x.x; xs[1] = x.y; xs[2] = x.z; xs[3] = x.w;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) xs[u] = row[g + u];
        }
        // over these four bins the potential is at most max(v, 0) + Kmax4
        // (max(I, 0) + the positive inputs), Kmax4 the largest K(s) over four
        // steps (K >= 0, and the current only decays between inputs); well
        // below v_th no bin can hold the spike and its flags are not needed
        const float ipos = fmaxf(I, 0.0f) + fmaxf(xs[0], 0.0f) + fmaxf(xs[1], 0.0f) + fmaxf(xs[2], 0.0f) +
                           fmaxf(xs[3], 0.0f);
        const bool quiet = fmaf(ipos, c.Kmax4, fmaxf(v, 0.0f)) < c.vth * 0.99999f;
        // one path per group for the whole warp: the flagged pass (its flags
        // kept only where the bound is not met) unless every lane is quiet;
        // both passes round alike, so the state does not depend on the path
        if (__all_sync(lanes, quiet)) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float I0 = I + xs[u];
                v = fmaf(c.KD, I0, c.rv * v);
                I = c.rI * I0;
            }
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const BinStep r = bin_step(c, v, I + xs[u]);
                if (!quiet && (r.endp | r.peak)) mask |= 1u << (g + u);
                v = r.ve;
                I = r.In;
            }
        }
    }
    if (mend < 32) mask &= (1u << mend) - 1u;
    while (mask) {
        const int m = __ffs(mask) - 1;
        mask &= mask - 1u;
        const int gk = m >> 3;
        float vw = kv[0], Iw = kI[0];
#pragma unroll
        for (int k = 1; k < NCK; ++k) {
            vw = (gk == k) ? kv[k] : vw;
            Iw = (gk == k) ? kI[k] : Iw;
        }
        for (int k = gk * 8; k < m; ++k) {
            const BinStep r = bin_step(c, vw, Iw + row[k]);
            vw = r.ve;
            Iw = r.In;
        }
        const float I0 = Iw + row[m];
        const BinStep r = bin_step(c, vw, I0);
        float hi = -1.0f;
        if (r.endp) hi = c.dt;
        else if (r.peak) hi = interior_test(c.av, c.aI, c.lam, c.lam_zero, c.rI, c.dt, c.vth, vw, I0, r.ve);
        if (hi >= 0.0f) {
            st.q = m0 + m;
            st.v0 = vw;
            st.I0 = I0;
            st.hi = hi;
            return true;
        }
    }
    return false;
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ void finish_neuron(const LifConst &c, const ScanState &st, int b, int i, int N,
                                              const float *rowsum, float *t_out, int *q, float *s, float *vdot,
                                              float acc[4]) {
    long long o = (long long)b * N + i;
    bool fired = st.q < c.M;
    float t = fired ? c.T0 + (float)st.q * c.dt + st.s : INFINITY;
    t_out[o] = t;
    if (q) q[o] = st.q;
    if (s) s[o] = st.s;
    if (vdot) vdot[o] = st.vdot;
    if (fired) {
        float pv, pg;
        penalty_T(c, t, pv, pg);
        acc[0] += pv;
        acc[3] += 1.0f;
    } else {
        if (rowsum) acc[1] += -c.g_q * c.norm * rowsum[i];
        acc[2] += 1.0f;
    }
}

// ---------------------------------------------------------------------------
// Device status word (bounded waits that expire set it); it lives in the
// tensor-core translation unit, the only device code that waits.
// ---------------------------------------------------------------------------
constexpr unsigned int STATUS_TIMEOUT = 1u;
cudaError_t status_read(unsigned int *out, int clear);
cudaError_t launch_wait_selftest(unsigned long long limit_ns, cudaStream_t st);

// ---------------------------------------------------------------------------
// Kernel launch entry points (host functions that launch on a stream).
// Layouts: "internal" bin axis padded to Mp (power of two), rows of 16-bit
// operands padded to a multiple of 8 elements (TMA needs 16-byte strides).
// ---------------------------------------------------------------------------
// Operand formats of a contraction: fp32 (CUDA cores), bf16 hi+lo, bf16,
// fp16 hi+lo (values pre-scaled into fp16 range by the producer).
enum class OpKind { F32 = 0, BF16X3 = 1, BF16 = 2, F16X3 = 3 };

inline int pad8(int x) { return (x + 7) & ~7; }

// W fp32 [R, C] -> fp16 hi/lo [R, ldo] of W * 2^k_i with one power of two
// per row (largest |w| of the row near 2^14), inv_scale [R] = 2^-k_i, and
// row sums [R]. One warp per row.
cudaError_t launch_prep_weights_f16(const float *W, int R, int C, __half *hi, __half *lo, int ldo, float *inv_scale,
                                    float *rowsum, cudaStream_t st);
// the x3 forward's two operands (binned spike times, fp16 weight split) in
// one launch: same results as launch_binning (F16X3) and launch_prep_weights_f16
// with ldo = ld
cudaError_t launch_fwd_operands_f16(const float *t, int B, int N, const LifConst &c, void *s_hi, void *s_lo, int ld,
                                    const float *W, int R, __half *w_hi, __half *w_lo, float *inv_scale,
                                    float *rowsum, cudaStream_t st);
// W fp32 [R, C] -> hi/lo bf16 [R, ldo] (and optional transpose [C, ldt]),
// fp32 copy (F32 path), row sums [R].
cudaError_t launch_prep_weights(const float *W, int R, int C, OpKind op, __nv_bfloat16 *hi, __nv_bfloat16 *lo,
                                int ldo, __nv_bfloat16 *hiT, __nv_bfloat16 *loT, int ldt, float *f32T,
                                int ldf, float *rowsum, cudaStream_t st);
// t [B, N] -> grid weights in the layout chosen by `transposed`:
//  !transposed: [B*Mp, ldk] (row (b,m), column j)    (contraction operand)
//   transposed: [N, ldk'] with ldk' >= B*Mp (row j, column (b,m))
// as bf16 hi/lo (BF16X3), bf16 hi (BF16) or fp32 (F32). Pad entries are 0.
// With transposed and bw != null, also bw[b*N + j] = (k as int bits, ds/dt at
// T_k, ds/dt at T_{k+1}, 0) per input (k = -100 when silent).
cudaError_t launch_binning(const float *t, int B, int N, const LifConst &c, OpKind op, bool transposed,
                           void *hi, void *lo, int ld, cudaStream_t st, float4 *bw = nullptr);
// Convolution geometry: input [B, H, W, C] (NHWC), filter k x k, stride s,
// zero-spike padding p, output [B, Ho, Wo, Cout]. An output position
// pos = (b*Ho + y)*Wo + x plays the role of a sample; the contraction axis is
// kidx = (kh*k + kw)*C + c (filter layout [Cout, k, k, C]).
struct ConvGeom {
    int B, H, W, C, Ho, Wo, k, s, p;
};
// Implicit-GEMM conv layer in bf16 (dstd_conv_tc.cu), for C_in and C_out
// multiples of 64 and Mp in {32, 64}: no im2col operand. ni = images of the
// chunk; positions NHWC.
bool conv_implicit_supported(const ConvGeom &g, int C_out, int Mp);
// input channels of the implicit path: C_in below 64 is padded to 64 (silent
// inputs, zero filter rows)
int conv_padded_channels(int C);
// dw^ [P][Mp][C] bf16 from the saved state [P][C]; silent counts per channel
// added into count (zeroed by the caller)
cudaError_t launch_dwhat_pmc(const float *t_out, const int *q, const float *s, const float *vdot, const float *g_up,
                             long long P, int C, const LifConst &c, __nv_bfloat16 *D, float *count, cudaStream_t st);
// filters [C_out][T][C_in] fp32 -> [C_pad][T][C_out] bf16 (padding rows zero)
cudaError_t launch_filters_t(const float *W, int C_out, int T, int C_in, int C_pad, __nv_bfloat16 *Wt,
                             cudaStream_t st);
// dS of ni images (the transposed convolution of dw^ [ni Ho Wo][Mp][C_out]
// with Wt [C_in][k k C_out]) with the input-time gradient in the epilogue:
// g_t_in [ni H W][C_in] (zeroed first) from t_in [ni H W][C_in]
// (g.C may be the padded channel count; t_in and g_t_in have C_t channels)
cudaError_t launch_conv_ds_gemm(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *dW_hat,
                                const __nv_bfloat16 *Wt, const float *t_in, float *g_t_in, int C_t, cudaStream_t st);
// the binned operand generated on chip: one 8-byte record per input
// (grid step, bf16 pair of its two weights), then the forward (w^ [ni Ho
// Wo][C_out][Mp] fp32) and dW (added into g_W [C_out][k k C_in], zeroed by
// the caller before the first chunk) contractions write their operand
// tiles in shared memory from the records
cudaError_t launch_bin_rec(const float *t, long long n, const LifConst &c, uint2 *rec, cudaStream_t st);
cudaError_t launch_conv_fwd_gen(const ConvGeom &g, int ni, int C_out, const LifConst &c, const uint2 *rec,
                                const __nv_bfloat16 *Wf, float *what, cudaStream_t st);
cudaError_t launch_conv_dw_gen(const ConvGeom &g, int ni, int C_out, const LifConst &c, const uint2 *rec,
                               const __nv_bfloat16 *dW_hat, const float *count, float qcoef, float *g_W,
                               cudaStream_t st);
// the binned input written out, S [P][Mp][C] bf16, from the spike times, and the
// forward contraction that reads it through tap-shifted TMA boxes, with the
// scan/solve/select of each neuron in its epilogue (outputs as from
// launch_scan_solve: spike times, q, s, dv^/dt, penalty sums)
bool conv_bin_S_supported(int C);  // channel counts the S writer takes
// t has Ct <= C channels; channels Ct .. C - 1 of S are silent
cudaError_t launch_bin_S(const float *t, long long P, int C, int Ct, const LifConst &c, __nv_bfloat16 *S,
                         cudaStream_t st);
cudaError_t launch_conv_fwd_tma(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                                const __nv_bfloat16 *Wf, const float *rowsum, float *t_out, int *q, float *s,
                                float *vdot, float *penalty, cudaStream_t st);
// dW from S and dw^ (added into g_W as for launch_conv_dw_gen)
// (g.C may be the padded channel count; g_W is [C_out][k k C_t])
cudaError_t launch_conv_dw_tma(const ConvGeom &g, int ni, int C_out, const LifConst &c, const __nv_bfloat16 *S,
                               const __nv_bfloat16 *dW_hat, const float *count, float qcoef, float *g_W, int C_t,
                               cudaStream_t st);
cudaError_t conv_status_read(unsigned int *out, int clear);
// im2col binning of positions [pos0, pos0 + npos): the grid weights of the
// input spike under each filter tap. !transposed: [npos*Mp, ld] (row (pos, m),
// column kidx); transposed: [K, ld] (row kidx, column (pos, m)).
cudaError_t launch_binning_im2col(const float *t, const ConvGeom &g, int pos0, int npos, const LifConst &c,
                                  OpKind op, bool transposed, void *hi, void *lo, int ld, cudaStream_t st);
// public-layout binning: s, ds [B, M, N] fp32
cudaError_t launch_binning_public(const float *t, int B, int N, const LifConst &c, float *s, float *ds,
                                  cudaStream_t st);
// scan/solve from w^ with element (b, i, m) at what[b*sb + i*si + m*sm],
// scaled by scale[i] when scale is not null
cudaError_t launch_scan_solve(const float *what, long long sb, long long si, long long sm, int B, int N,
                              const LifConst &c, const float *scale, const float *rowsum, float *t_out, int *q,
                              float *s, float *vdot, float *penalty, cudaStream_t st);
// dw^ from saved state; writes [B*Mp, ldn] (row (b,m), col i) and [N, ldbm]
// (row i, col (b,m)) in the operand format; silent counts per neuron.
// (silent_count is zeroed first unless accumulate_count)
cudaError_t launch_dwhat(const float *t_out, const int *q, const float *s, const float *vdot, const float *g_up,
                         int B, int N, const LifConst &c, OpKind op, void *a_hi, void *a_lo, int lda,
                         void *b_hi, void *b_lo, int ldb, float *silent_count, cudaStream_t st,
                         bool accumulate_count = false);
// g_t_in of a layer with few outputs (N_out <= kGradtSmallMaxOut) directly
// from W, dw^ (operand layout [N_out, ld] over (b, m), hi/lo or hi only) and
// the per-input bin index / kernel derivatives bw.
constexpr int kGradtSmallMaxOut = 32;
// The exact (event-driven) forward, Alg. 1, for comparison with DSTD: W^T,
// the sorted inputs and their intervals in the workspace (exact_layout).
// multi-spike regime (App. D): at most this many spikes per neuron, in and out
constexpr int kMsMaxSpikes = 8;
cudaError_t launch_binning_ms(const float *t, int B, int N, int F, const LifConst &c, OpKind op, bool transposed,
                              void *hi, void *lo, int ld, cudaStream_t st);
cudaError_t launch_scan_ms(const float *what, long long sb, long long si, int B, int N, const LifConst &c, int F,
                           float *t_out, int *q, float *I, float *vd, cudaStream_t st);
cudaError_t launch_dwhat_ms(const float *t_out, const int *q, const float *I, const float *vd, const float *g_up,
                            int B, int N, int F, const LifConst &c, OpKind op, void *a_hi, void *a_lo, int lda,
                            void *b_hi, void *b_lo, int ldb, cudaStream_t st);
cudaError_t launch_gt_ms(const float *D, long long ldd, const float *t_in, int B, int N, int F, const LifConst &c,
                         float *g_t_in, cudaStream_t st);

constexpr int kExactMaxIn = 8192;  // a sample's inputs are sorted in shared memory
struct ExactWs {
    float *Wt = nullptr;       // [N_in][N_out]
    int *perm = nullptr;       // [B][N_in]: input of the k-th interval
    float *t_start = nullptr;  // [B][N_in]: its start
    float4 *iv = nullptr;      // [B][N_in]: e^{-av L}, e^{-aI L}, K(L), L
    int *count = nullptr;      // [B]: intervals (finite inputs before the window end)
    float *coef = nullptr;     // [B][N_out]: dC/dt_i / V'_i (backward)
    size_t bytes = 0;
};
cudaError_t launch_exact_fwd(const float *t_in, const float *W, int B, int N_in, int N_out, const LifConst &c,
                             float t_end, float kmax, const ExactWs &ws, float *t_out, cudaStream_t st);
// the exact method's backward: g_W [N_out][N_in] (overwritten) and, when
// g_t_in is not null, g_t_in [B][N_in] (overwritten) from g_out [B][N_out]
cudaError_t launch_exact_bwd(const float *t_in, const float *W, const float *t_out, const float *g_out, int B,
                             int N_in, int N_out, const LifConst &c, const ExactWs &ws, float *g_t_in, float *g_W,
                             cudaStream_t st);

// Layers with at most kNarrowMaxOut outputs run forward and backward on CUDA
// cores in fp32 (sparse over the two grid points of each input spike).
constexpr int kNarrowMaxOut = 32;
constexpr int kNarrowMaxIn = 4096;       // the forward sorts a sample's inputs in shared memory
constexpr size_t kNarrowMaxSmem = 200 * 1024;  // and holds W there: its shared memory, at most this
size_t narrow_fwd_smem(int N_in, int N_out, int M, int Mp);
// Cross-entropy of the output layer fused into its few-output forward:
// loss float[2] (loss[1] a ticket: zero before the first call, left zero),
// g [B, N_out], scratch float[B] (per-sample terms, summed in order by the
// last block); loss == nullptr: no loss.
struct NarrowCe {
    const int32_t *labels = nullptr;
    float tau_soft = 1.f, t_silent = 0.f;
    float *loss = nullptr, *g = nullptr, *scratch = nullptr;
};
cudaError_t launch_narrow_fwd(const float *t, const float *W, int B, int N_in, int N_out, const LifConst &c,
                              float *t_out, int *q, float *s, float *vdot, float *penalty, cudaStream_t st,
                              const NarrowCe &ce = NarrowCe());
// zeroes g_W, then adds every block's share
cudaError_t launch_narrow_bwd(const float *t_in, const float *W, const float *t_out, const int *q, const float *s,
                              const float *vdot, const float *g_up, int B, int N_in, int N_out, const LifConst &c,
                              float qcoef, float *g_t_in, float *g_W, cudaStream_t st);
cudaError_t launch_gradt_small(const float *W, int N_out, int N_in, int B, const LifConst &c, const float4 *bw,
                               const __nv_bfloat16 *d_hi, const __nv_bfloat16 *d_lo, int ld, float *g_t_in,
                               cudaStream_t st);
// g_t_in from dS stored as D[j, (b,m)] (row stride ldd)
cudaError_t launch_gt_from_ds(const float *D, long long ldd, const float *t_in, int B, int N, const LifConst &c,
                              float *g_t_in, cudaStream_t st);
// g_W[i, j] (+)= sum_z part[z][i, j] + qcoef*count[i] (count may be null)
cudaError_t launch_dw_reduce(const float *part, int splits, long long zstride, int ldp, int R, int C,
                             const float *count, float qcoef, float *g_W, cudaStream_t st, bool accumulate = false);
// copy internal w^ D[i, (b, m)] (ld) -> public [B, N, M]
cudaError_t launch_what_to_public(const float *D, long long ld, int B, int N, int M, int Mp, float *out,
                                  cudaStream_t st);

// D = A B^T, fp32 CUDA cores. A [R, K] (lda), B [Cn, K] (ldb), D [R, Cn] (ldd);
// split-K over `splits` writes D + z*zstride.
cudaError_t launch_sgemm_tn(const float *A, int lda, const float *Bm, int ldb, float *D, int ldd, int R, int Cn,
                            int K, int splits, long long zstride, cudaStream_t st);

// tcgen05 GEMM D = A B^T on bf16 operands (hi/lo for BF16X3), fp32 TMEM
// accumulation, with a fused epilogue.
enum class Epi { Store = 0, GradT = 1 };
struct TcEpiArgs {
    const float *row_scale;  // per-row factor applied to the accumulator (Store, Scan), may be null
    // Store: split z writes D + z*zstride, or with atomic != 0 every split
    // adds into D (zeroed by the caller) and split 0 also adds
    // qcoef * qcount[row] when qcount is given (the Q term of dW)
    float *D; long long ldd; long long zstride;
    int atomic; const float *qcount; float qcoef;
    // GradT: layer constants and sizes (rows N, samples B)
    LifConst c; int B; int N;
    // GradT (rows = inputs j, columns = (b, m)); with conv != 0 the rows are
    // filter taps kidx, the columns (output position, m), and each result is
    // added atomically into the input element the tap reads (col2im)
    const float *t_in; float *g_t_in;
    const float4 *bw;  // dense GradT: per-input (k, ds/dt at T_k, at T_{k+1}) from the binning, or null
    int conv; int pos0; ConvGeom g;
};
// A, B: 16-bit operands (bf16 for BF16X3 / BF16, fp16 for F16X3). A is
// [R, K] rows (stride lda). B is [Cn, K] rows (stride ldb) for Epi::Store and
// [K, Cn] rows (b_mn: read transposed by the tensor core) for Epi::GradT.
cudaError_t launch_tc_gemm(const void *A_hi, const void *A_lo, int lda, const void *B_hi, const void *B_lo, int ldb,
                           int R, int Cn, int K, int splits, OpKind op, Epi epi, const TcEpiArgs &args,
                           cudaStream_t st, bool b_mn = false);
// The same product on SM pairs (tcgen05 cta_group::2, 256 x 128 tiles), with
// the transposed store D[c * ldd + r] = (A B^T)[r][c] * row_scale[c]
// (args.D, args.ldd, args.row_scale): A [R, K] rows, B [Cn, K] rows. For the
// F16X3 and BF16 forward operands.
cudaError_t launch_tc_gemm_pair_storeT(const void *A_hi, const void *A_lo, int lda, const void *B_hi, const void *B_lo,
                                       int ldb, int R, int Cn, int K, OpKind op, const TcEpiArgs &args,
                                       cudaStream_t st);
// whether the pair kernel is expected to beat the single-CTA one for an
// R x Cn x K product (resident pairs counted once per process)
bool tc_gemm_pair_preferred(int R, int Cn, int K, OpKind op);
int tc_gemm_resident_pairs(OpKind op);
// 0 the cost model, 1 pairs wherever they apply, 2 never pairs; returns the previous setting
int tc_gemm_pair_policy(int policy);

cudaError_t launch_ce_loss(const float *t, const int32_t *lab, int B, int C, float tau_soft, float t_silent,
                           float *loss, float *g, cudaStream_t st);
cudaError_t launch_sum_t(const float *t, long long n, float *loss, float *g, cudaStream_t st);
cudaError_t launch_concat_channels(const float *a, int Ca, float delay, const float *b, int Cb, long long P, float *out,
                                   cudaStream_t st);
cudaError_t launch_split_channels(const float *g, int Ca, int Cb, long long P, float *ga, bool acc_a, float *gb,
                                  bool acc_b, cudaStream_t st);
cudaError_t launch_adamw(float *w, const float *g, float *m, float *v, long long n, float lr, float b1, float b2,
                         float eps, float wd, int step, cudaStream_t st);

// one parameter tensor of a multi-tensor AdamW launch (off: set by the launcher)
struct AdamSeg {
    float *w;
    const float *g;
    float *m;
    float *v;
    long long n, off;
};
constexpr int kAdamMaxTensors = 32;
struct AdamMultiArgs {
    AdamSeg seg[kAdamMaxTensors];
    int count;
    long long total;
    float lr, b1, b2, eps, wd;
    int32_t *step;        // device: [0] updates done so far, [1] block ticket (0 between calls)
    const float *lr_dev;  // device learning rate, or null for lr
};
cudaError_t launch_adamw_multi(const AdamMultiArgs &args, cudaStream_t st);

}  // namespace dstd
