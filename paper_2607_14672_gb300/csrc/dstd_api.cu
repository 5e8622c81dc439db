// C-ABI entry points of libdstd (include/dstd.h): argument checks, workspace
// layout and the order of kernel launches for one dense DSTD layer.
#include "dstd_internal.cuh"

#include <math.h>
#include <string.h>

#include <mutex>
#include <utility>
#include <vector>

namespace dstd {
int tc_gemm_splits_valid(int K, int splits);
}

using namespace dstd;

namespace {

constexpr int kVersion = 100;  // 0.1.0

// 256-byte bump allocator over a caller workspace (nullptr base = size query)
struct Bump {
    char *base;
    size_t off = 0;
    explicit Bump(void *b) : base(static_cast<char *>(b)) {}
    template <class T>
    T *take(size_t count) {
        off = (off + 255) & ~(size_t)255;
        T *p = base ? reinterpret_cast<T *>(base + off) : nullptr;
        off += count * sizeof(T);
        return p;
    }
};

bool finite_pos_or_inf(float x) { return (x > 0.0f && isfinite(x)) || (isinf(x) && x > 0.0f); }

int check_params(const dstd_params *p) {
    if (!p) return DSTD_E_INVALID;
    if (!finite_pos_or_inf(p->tau_m) || !finite_pos_or_inf(p->tau_s)) return DSTD_E_INVALID;
    if (!(p->v_th > 0.0f) || !isfinite(p->v_th)) return DSTD_E_INVALID;
    if (!isfinite(p->t_first) || !isfinite(p->t_end) || !(p->t_end > p->t_first)) return DSTD_E_INVALID;
    if (p->M < 1) return DSTD_E_INVALID;
    if (p->M > 256) return DSTD_E_UNSUPPORTED;
    const double dt = ((double)p->t_end - (double)p->t_first) / p->M;
    if (!isfinite(p->t_offset) || !(p->t_offset > -dt / 2) || !(p->t_offset <= dt / 2 * (1 + 1e-6)))
        return DSTD_E_INVALID;
    if (!isfinite(p->gamma_head) || !isfinite(p->gamma_tail) || !isfinite(p->gamma_q) ||
        !isfinite(p->penalty_norm) || isnan(p->t_head) || isnan(p->t_tail))
        return DSTD_E_INVALID;
    return DSTD_OK;
}

int check_math(dstd_math m, int Mp) {
    if (m != DSTD_MATH_F32 && m != DSTD_MATH_X3 && m != DSTD_MATH_BF16) return DSTD_E_INVALID;
    if (m != DSTD_MATH_F32 && Mp > 128) return DSTD_E_UNSUPPORTED;  // one sample per tensor-core tile
    return DSTD_OK;
}

// operand format of the forward contraction and of the two backward ones
OpKind op_of(dstd_math m) {
    return m == DSTD_MATH_F32 ? OpKind::F32 : (m == DSTD_MATH_X3 ? OpKind::F16X3 : OpKind::BF16);
}
OpKind bwd_op_of(dstd_math m) {
    return m == DSTD_MATH_F32 ? OpKind::F32 : (m == DSTD_MATH_X3 ? OpKind::BF16X3 : OpKind::BF16);
}
bool two_part(OpKind op) { return op == OpKind::BF16X3 || op == OpKind::F16X3; }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int device_ok() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DSTD_E_NO_DEVICE;
    static int cached_dev = -1, cached_ok = 0;
    if (dev == cached_dev) return cached_ok ? DSTD_OK : DSTD_E_NO_DEVICE;
    int maj = 0, min = 0;
    if (cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&min, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
        return DSTD_E_NO_DEVICE;
    cached_dev = dev;
    cached_ok = (maj == 10 && min == 3);
    return cached_ok ? DSTD_OK : DSTD_E_NO_DEVICE;
}

inline int cu(cudaError_t e) { return e == cudaSuccess ? DSTD_OK : DSTD_E_CUDA; }

// ---------------------------------------------------------------------------
// Kernel timing: an event pair per launch, filed by kernel kind.
// ---------------------------------------------------------------------------
enum Kind {
    KK_PREP = 0, KK_BIN, KK_BIN_T, KK_GEMM_FWD, KK_SCAN, KK_DWHAT, KK_GEMM_DS, KK_GT, KK_GEMM_DW, KK_REDUCE,
    KK_LOSS, KK_ADAMW, KK_BIN_PUB, KK_WHAT_PUB, KK_SELFTEST, KK_NARROW_FWD, KK_NARROW_BWD, KK_EXACT_FWD, KK_SKIP,
    KK_EXACT_BWD, KK_COUNT
};
const char *const kKindNames[KK_COUNT] = {
    "prep_weights", "binning", "binning_T", "gemm_fwd_scan", "scan_solve", "dwhat", "gemm_dS_gradt",
    "gradt_gather", "gemm_dW", "dw_reduce", "loss", "adamw", "binning_public", "what_public", "selftest", "narrow_fwd",
    "narrow_bwd", "exact_fwd", "skip_channels", "exact_bwd"};

struct Timing {
    std::mutex mu;
    bool on = false;
    std::vector<cudaEvent_t> pool;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending[KK_COUNT];
    // pairs captured into a CUDA graph as event-record nodes: every replay
    // records them again; dstd_timing_collect adds one replay's worth
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> graph[KK_COUNT];
    double ms[KK_COUNT] = {};
    long long n[KK_COUNT] = {};
};
Timing g_timing;

cudaEvent_t take_event() {
    cudaEvent_t e = nullptr;
    if (!g_timing.pool.empty()) {
        e = g_timing.pool.back();
        g_timing.pool.pop_back();
    } else if (cudaEventCreate(&e) != cudaSuccess) {
        e = nullptr;
    }
    return e;
}

// drain pending pairs into the totals (caller holds the lock, device synced)
void drain_pending() {
    for (int k = 0; k < KK_COUNT; ++k) {
        for (auto &pr : g_timing.pending[k]) {
            float ms = 0.f;
            if (cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess) {
                g_timing.ms[k] += ms;
                g_timing.n[k] += 1;
            }
            g_timing.pool.push_back(pr.first);
            g_timing.pool.push_back(pr.second);
        }
        g_timing.pending[k].clear();
    }
}

// Brackets the launches of one scope with an event pair: recorded directly
// in eager mode, or, on a stream being captured, as external event-record
// nodes of the graph (read back per replay by dstd_timing_collect).
struct Timed {
    int kind;
    cudaStream_t st;
    cudaEvent_t a = nullptr;
    bool captured = false;
    Timed(int k, cudaStream_t s) : kind(k), st(s) {
        if (!g_timing.on) return;
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) return;
        captured = cs == cudaStreamCaptureStatusActive;
        if (cs != cudaStreamCaptureStatusNone && !captured) return;
        std::lock_guard<std::mutex> lk(g_timing.mu);
        a = take_event();
        const cudaError_t e = captured ? cudaEventRecordWithFlags(a, s, cudaEventRecordExternal) : cudaEventRecord(a, s);
        if (a && e != cudaSuccess) {
            g_timing.pool.push_back(a);
            a = nullptr;
        }
    }
    ~Timed() {
        if (!a) return;
        std::lock_guard<std::mutex> lk(g_timing.mu);
        cudaEvent_t b = take_event();
        const cudaError_t e =
            !b ? cudaErrorUnknown : (captured ? cudaEventRecordWithFlags(b, st, cudaEventRecordExternal) : cudaEventRecord(b, st));
        if (e == cudaSuccess) (captured ? g_timing.graph : g_timing.pending)[kind].push_back({a, b});
        else {
            g_timing.pool.push_back(a);
            if (b) g_timing.pool.push_back(b);
        }
    }
};
#define TRY(x)                       \
    do {                             \
        int _r = (x);                \
        if (_r != DSTD_OK) return _r; \
    } while (0)

// ---------------------------------------------------------------------------
// Side streams. Launches of one call that do not depend on each other (in
// the backward: dw^ beside the transposed binning and the weight transpose)
// run on two library-owned streams: Fork makes both wait for
// the work already enqueued on the caller's stream, and join() (or the
// destructor) makes the caller's stream wait for both again. Under stream
// capture this becomes a fork and a join in the graph. The side streams are
// per device and shared; a Fork holds a lock from fork to join, so calls from
// several host threads enqueue one after the other. If a stream or event
// cannot be had, every launch stays on the caller's stream.
// ---------------------------------------------------------------------------
struct SideSet {
    cudaStream_t s[2] = {nullptr, nullptr};
    cudaEvent_t fork = nullptr, join[2] = {nullptr, nullptr};
    int state = 0;  // 0 not made, 1 ready, -1 unavailable
};
constexpr int kMaxDevices = 64;
SideSet g_side[kMaxDevices];
std::mutex g_side_mu;

struct Fork {
    cudaStream_t main, side[2];
    SideSet *ss = nullptr;
    std::unique_lock<std::mutex> lk;
    explicit Fork(cudaStream_t st) : main(st), side{st, st}, lk(g_side_mu) {
        // with kernel timing on, everything runs on the caller's stream, one
        // kernel after another, so that each kind's time is its own (and not
        // that of kernels sharing the GPU with it)
        if (g_timing.on) return;
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return;
        SideSet &q = g_side[dev];
        if (q.state == 0) {
            bool good = cudaEventCreateWithFlags(&q.fork, cudaEventDisableTiming) == cudaSuccess;
            for (int i = 0; i < 2 && good; ++i)
                good = cudaStreamCreateWithFlags(&q.s[i], cudaStreamNonBlocking) == cudaSuccess &&
                       cudaEventCreateWithFlags(&q.join[i], cudaEventDisableTiming) == cudaSuccess;
            q.state = good ? 1 : -1;
        }
        if (q.state != 1 || cudaEventRecord(q.fork, st) != cudaSuccess) return;
        for (int i = 0; i < 2; ++i)
            if (cudaStreamWaitEvent(q.s[i], q.fork, 0) == cudaSuccess) side[i] = q.s[i];
        ss = &q;
    }
    int join() {
        if (!ss) return DSTD_OK;
        int r = DSTD_OK;
        for (int i = 0; i < 2; ++i) {
            if (side[i] == main) continue;
            if (cudaEventRecord(ss->join[i], side[i]) != cudaSuccess ||
                cudaStreamWaitEvent(main, ss->join[i], 0) != cudaSuccess)
                r = DSTD_E_CUDA;
            side[i] = main;
        }
        ss = nullptr;
        return r;
    }
    ~Fork() { join(); }
};

// ---------------------------------------------------------------------------
// Workspace layouts (one for the forward, one for the backward; both start at
// the workspace base).
// ---------------------------------------------------------------------------
struct FwdWs {
    uint16_t *w_hi = nullptr, *w_lo = nullptr, *s_hi = nullptr, *s_lo = nullptr;  // 16-bit operands
    float *s32 = nullptr, *D = nullptr, *rowsum = nullptr, *row_scale = nullptr;
    size_t bytes = 0;
    int kpad = 0, ldD = 0;
};

FwdWs fwd_layout(void *base, int B, int N_in, int N_out, int Mp, OpKind op, bool need_D) {
    FwdWs w;
    Bump b(base);
    w.kpad = pad8(N_in);
    const long long cols = (long long)B * Mp;
    w.rowsum = b.take<float>(N_out);
    if (op == OpKind::F32) {
        w.s32 = b.take<float>((size_t)cols * w.kpad);
        w.D = b.take<float>((size_t)N_out * cols);
    } else {
        w.w_hi = b.take<uint16_t>((size_t)N_out * w.kpad);
        if (two_part(op)) w.w_lo = b.take<uint16_t>((size_t)N_out * w.kpad);
        w.s_hi = b.take<uint16_t>((size_t)cols * w.kpad);
        if (two_part(op)) w.s_lo = b.take<uint16_t>((size_t)cols * w.kpad);
        if (op == OpKind::F16X3) w.row_scale = b.take<float>(N_out);
        // w^ in fp32: [N_out, B*Mp] for the public copy (need_D), else the
        // scan's layout [B*Mp, ldD] (row (b, m), column i)
        w.ldD = (N_out + 3) & ~3;
        w.D = b.take<float>((size_t)cols * w.ldD);  // >= N_out * cols
        (void)need_D;
    }
    w.bytes = b.off;
    return w;
}

struct BwdWs {
    __nv_bfloat16 *wt_hi = nullptr, *wt_lo = nullptr, *dA_hi = nullptr, *dA_lo = nullptr, *sT_hi = nullptr,
                  *sT_lo = nullptr;
    float *wt32 = nullptr, *dA32 = nullptr, *dB32 = nullptr, *sT32 = nullptr, *DS = nullptr, *part = nullptr,
          *count = nullptr;
    float4 *bw = nullptr;  // per-input bin index and kernel derivatives (input-time gradient)
    int ldt = 0, ldn = 0, ldbm = 0, ldp = 0, splits = 1;
    size_t bytes = 0;
};

// split-K factor of the forward contraction: enough splits to give every SM
// a tile when the output has fewer tiles than SMs, each split at least two
// 64-deep K slices
int fwd_splits(int N_out, long long cols, int N_in) {
    const long long tiles = (long long)((N_out + 127) / 128) * ((cols + 127) / 128);
    const int ktiles = (N_in + 63) / 64;
    long long s = tiles >= 152 ? 1 : 152 / tiles;
    if (s > ktiles / 2) s = ktiles / 2;
    if (s < 1) s = 1;
    while (s > 1 && !tc_gemm_splits_valid(N_in, (int)s)) --s;
    return (int)s;
}

int dw_splits(int N_in, int N_out, int K, OpKind op) {
    const int tm = op == OpKind::F32 ? 64 : 128, tn = op == OpKind::F32 ? 64 : 128;
    const long long tiles = (long long)((N_out + tm - 1) / tm) * ((N_in + tn - 1) / tn);
    const int kunit = op == OpKind::F32 ? 16 : 64;
    const int ktiles = (K + kunit - 1) / kunit;
    if (op == OpKind::F32) {
        long long want = (2 * 152 + tiles - 1) / tiles;
        int s = (int)(want < 1 ? 1 : (want > ktiles ? ktiles : want));
        return s < 1 ? 1 : (s > 64 ? 64 : s);
    }
    // persistent tensor-core contraction on 152 SMs: the busiest CTA runs
    // ceil(items / 152) work items of ceil(ktiles / s) K slices each, plus
    // about two slices of pipeline fill and epilogue per item
    int best = 1;
    long long best_cost = -1;
    for (int s = 1; s <= 64 && s <= ktiles; ++s) {
        if (!tc_gemm_splits_valid(K, s)) continue;
        const long long rounds = (tiles * s + 151) / 152;
        const long long cost = rounds * ((ktiles + s - 1) / s + 2);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = s;
        }
    }
    return best;
}

// whether dW runs on SM pairs (transposed, no split-K) rather than on
// single CTAs with the split-K factor of dw_splits: the same cost units as
// both (rounds of work x K slices per item, plus fill and drain), with the
// pair's 256 x 128 tiles, resident pairs and a pair K slice at 0.92 of a
// single CTA's (measured); the scheduling policy can force either
bool dw_on_pairs(int N_in, int N_out, int K, OpKind op) {
    const int policy = tc_gemm_pair_policy(-1);
    if (policy == 1) return true;
    if (policy == 2) return false;
    if (N_in < 256 || N_out < 256) return false;  // a narrow side leaves the pair's 256 x 128 tiles mostly padding
    const int s = dw_splits(N_in, N_out, K, op);
    const long long kt = (K + 63) / 64;
    const long long tiles = (long long)((N_out + 127) / 128) * ((N_in + 127) / 128);
    const double single = (double)((tiles * s + 151) / 152) * (double)((kt + s - 1) / s + 2);
    const long long pairs = tc_gemm_resident_pairs(op);
    if (pairs < 1) return false;
    const long long t2 = (long long)((N_in + 255) / 256) * ((N_out + 127) / 128);
    const double pair = (double)((t2 + pairs - 1) / pairs) * (0.92 * (double)kt + 4.0);
    return pair < single;
}

BwdWs bwd_layout(void *base, int B, int N_in, int N_out, int Mp, OpKind op, bool need_gt) {
    BwdWs w;
    Bump b(base);
    const long long cols = (long long)B * Mp;
    w.ldt = pad8(N_out);
    w.ldn = pad8(N_out);
    w.ldbm = pad8((int)cols);
    w.ldp = (N_in + 3) & ~3;
    w.splits = dw_splits(N_in, N_out, (int)cols, op);
    w.count = b.take<float>(N_out);
    if (op == OpKind::F32) {
        w.part = b.take<float>((size_t)w.splits * N_out * w.ldp);  // split-K partials (the tensor-core path adds atomically)
        w.dA32 = b.take<float>((size_t)N_out * w.ldbm);
        w.dB32 = b.take<float>((size_t)cols * w.ldn);
        w.sT32 = b.take<float>((size_t)N_in * w.ldbm);
        if (need_gt) {
            w.wt32 = b.take<float>((size_t)N_in * w.ldt);
            w.DS = b.take<float>((size_t)N_in * cols);
        }
    } else {
        const bool three = op == OpKind::BF16X3;
        // dw^ once, [N_out, B*Mp]: the A operand of dW and, read transposed,
        // the B operand of dS
        w.dA_hi = b.take<__nv_bfloat16>((size_t)N_out * w.ldbm);
        if (three) w.dA_lo = b.take<__nv_bfloat16>((size_t)N_out * w.ldbm);
        w.sT_hi = b.take<__nv_bfloat16>((size_t)N_in * w.ldbm);
        if (three) w.sT_lo = b.take<__nv_bfloat16>((size_t)N_in * w.ldbm);
        if (need_gt) {
            w.wt_hi = b.take<__nv_bfloat16>((size_t)N_in * w.ldt);
            if (three) w.wt_lo = b.take<__nv_bfloat16>((size_t)N_in * w.ldt);
            w.bw = b.take<float4>((size_t)B * N_in);
        }
    }
    w.bytes = b.off;
    return w;
}

ExactWs exact_layout(void *base, int B, int N_in, int N_out) {
    ExactWs w;
    Bump bp(base);
    w.Wt = bp.take<float>((size_t)N_in * N_out);
    w.perm = bp.take<int>((size_t)B * N_in);
    w.t_start = bp.take<float>((size_t)B * N_in);
    w.iv = bp.take<float4>((size_t)B * N_in);
    w.count = bp.take<int>((size_t)B);
    w.coef = bp.take<float>((size_t)B * N_out);
    w.bytes = bp.off;
    return w;
}

// sup over s >= 0 of K(s) = e^{-av s} phi(s) (+inf when both rates are 0)
double kernel_sup(double av, double aI) {
    if (av > 0.0 && aI > 0.0) {
        const double lam = aI - av;
        const double tp = lam == 0.0 ? 1.0 / av : log(aI / av) / lam;
        const double ph = lam == 0.0 ? tp : -expm1(-lam * tp) / lam;
        return exp(-av * tp) * ph;
    }
    if (av > 0.0) return 1.0 / av;
    if (aI > 0.0) return 1.0 / aI;
    return INFINITY;
}

struct Saved {
    int *q;
    float *s, *vdot;
};
Saved saved_view(void *saved, int B, int N_out) {
    Bump b(saved);
    Saved v;
    v.q = b.take<int>((size_t)B * N_out);
    v.s = b.take<float>((size_t)B * N_out);
    v.vdot = b.take<float>((size_t)B * N_out);
    return v;
}

int check_sizes(int B, int N_in, int N_out) {
    if (B < 1 || N_in < 1 || N_out < 1) return DSTD_E_INVALID;
    // grid limits: B is a grid y extent (<= 65535); row tiles of 32 for N
    if (B > 65535 || N_in > (1 << 20) || N_out > (1 << 20)) return DSTD_E_UNSUPPORTED;
    return DSTD_OK;
}

// forward up to w^: binning + contraction; Scan epilogue fused (TC) unless
// `store_D` (then the fp32 w^ lands in ws.D, layout [N_out, B*Mp]).
// A layer with few outputs runs on CUDA cores in fp32 (fp32 and three-product
// modes; the bf16 mode keeps its bf16 operands on the tensor cores).
bool narrow_layer(int N_in, int N_out, int M, OpKind op) {
    return N_out <= kNarrowMaxOut && N_in <= kNarrowMaxIn && M <= 94 &&
           narrow_fwd_smem(N_in, N_out, M, padded_M(M)) <= kNarrowMaxSmem &&
           (op == OpKind::F32 || op == OpKind::F16X3 || op == OpKind::BF16X3);
}

int dense_forward_core(const float *t_in, const float *W, int B, int N_in, int N_out, const LifConst &c, OpKind op,
                       const FwdWs &ws, bool store_D, const Saved *sv, float *t_out, float *penalty,
                       cudaStream_t st) {
    const long long cols = (long long)B * c.Mp;
    if (!store_D && narrow_layer(N_in, N_out, c.M, op)) {
        Timed tm(KK_NARROW_FWD, st);
        return cu(launch_narrow_fwd(t_in, W, B, N_in, N_out, c, t_out, sv->q, sv->s, sv->vdot, penalty, st));
    }
    if (op == OpKind::F32) {
        {
            Timed tm(KK_PREP, st);
            TRY(cu(launch_prep_weights(W, N_out, N_in, op, nullptr, nullptr, 0, nullptr, nullptr, 0, nullptr, 0,
                                       ws.rowsum, st)));
        }
        {
            Timed tm(KK_BIN, st);
            TRY(cu(launch_binning(t_in, B, N_in, c, op, false, ws.s32, nullptr, ws.kpad, st)));
        }
        {
            Timed tm(KK_GEMM_FWD, st);
            TRY(cu(launch_sgemm_tn(W, N_in, ws.s32, ws.kpad, ws.D, (int)cols, N_out, (int)cols, N_in, 1, 0, st)));
        }
        if (!store_D) {
            Timed tm(KK_SCAN, st);
            TRY(cu(launch_scan_solve(ws.D, c.Mp, cols, 1, B, N_out, c, nullptr, ws.rowsum, t_out, sv->q, sv->s,
                                     sv->vdot, penalty, st)));
        }
        return DSTD_OK;
    }
    // the weight split and the binning are independent: one launch does both
    // for the x3 forward (a fork/join around two kernels this short costs
    // more than their overlap gains)
    if (op == OpKind::F16X3 && (ws.kpad % 8) == 0) {
        Timed tm(KK_BIN, st);
        TRY(cu(launch_fwd_operands_f16(t_in, B, N_in, c, ws.s_hi, ws.s_lo, ws.kpad, W, N_out, (__half *)ws.w_hi,
                                       (__half *)ws.w_lo, ws.row_scale, ws.rowsum, st)));
    } else {
        {
            Timed tm(KK_PREP, st);
            if (op == OpKind::F16X3)
                TRY(cu(launch_prep_weights_f16(W, N_out, N_in, (__half *)ws.w_hi, (__half *)ws.w_lo, ws.kpad,
                                               ws.row_scale, ws.rowsum, st)));
            else
                TRY(cu(launch_prep_weights(W, N_out, N_in, op, (__nv_bfloat16 *)ws.w_hi, (__nv_bfloat16 *)ws.w_lo,
                                           ws.kpad, nullptr, nullptr, 0, nullptr, 0, ws.rowsum, st)));
        }
        {
            Timed tm(KK_BIN, st);
            TRY(cu(launch_binning(t_in, B, N_in, c, op, false, ws.s_hi, ws.s_lo, ws.kpad, st)));
        }
    }
    TcEpiArgs a{};
    a.c = c;
    a.B = B;
    a.N = N_out;
    a.row_scale = ws.row_scale;
    if (store_D) {
        Timed tm(KK_GEMM_FWD, st);
        a.D = ws.D;
        a.ldd = cols;
        a.zstride = 0;
        return cu(launch_tc_gemm(ws.w_hi, ws.w_lo, ws.kpad, ws.s_hi, ws.s_lo, ws.kpad, N_out, (int)cols, N_in, 1, op,
                                 Epi::Store, a, st));
    }
    // w^ with rows i and columns (b, m): the Mp bins of a neuron are 128
    // contiguous bytes (Mp = 32) that the scan reads with 16-byte loads. With
    // fewer output tiles than SMs (a narrow layer) K is split across CTAs
    // whose partial sums add into w^ (zeroed first).
    {
        const int splits = fwd_splits(N_out, cols, N_in);
        if (splits == 1 && tc_gemm_pair_preferred((int)cols, N_out, N_in, op)) {
            // on SM pairs, computed transposed: (S W^T)[(b, m), i], stored as w^[i][(b, m)]
            {
                Timed tm(KK_GEMM_FWD, st);
                a.D = ws.D;
                a.ldd = cols;
                TRY(cu(launch_tc_gemm_pair_storeT(ws.s_hi, ws.s_lo, ws.kpad, ws.w_hi, ws.w_lo, ws.kpad, (int)cols,
                                                  N_out, N_in, op, a, st)));
            }
            Timed ts(KK_SCAN, st);
            return cu(launch_scan_solve(ws.D, c.Mp, cols, 1, B, N_out, c, nullptr, ws.rowsum, t_out, sv->q, sv->s,
                                        sv->vdot, penalty, st));
        }
        if (splits > 1) TRY(cu(cudaMemsetAsync(ws.D, 0, sizeof(float) * (size_t)N_out * cols, st)));
        Timed tm(KK_GEMM_FWD, st);
        a.D = ws.D;
        a.ldd = cols;
        a.zstride = 0;
        a.atomic = splits > 1;
        TRY(cu(launch_tc_gemm(ws.w_hi, ws.w_lo, ws.kpad, ws.s_hi, ws.s_lo, ws.kpad, N_out, (int)cols, N_in, splits,
                              op, Epi::Store, a, st)));
    }
    Timed tm(KK_SCAN, st);
    return cu(launch_scan_solve(ws.D, c.Mp, cols, 1, B, N_out, c, nullptr, ws.rowsum, t_out, sv->q, sv->s,
                                sv->vdot, penalty, st));
}

// ---------------------------------------------------------------------------
// Convolution layers: output positions act as samples, filter taps as the
// contraction axis; the binned inputs are gathered per filter tap (im2col)
// for a chunk of whole images at a time, so the scratch stays bounded.
// ---------------------------------------------------------------------------
constexpr size_t kConvChunkBudget = 1ull << 30;  // bytes of im2col operands per chunk

struct ConvPlan {
    ConvGeom g;
    int K, kpad, npos, chunk, nchunks;
};

int conv_plan(int B, int H, int W, int C, int k, int stride, int pad, int Mp, bool two, int Cout, ConvPlan *pl) {
    if (B < 1 || H < 1 || W < 1 || C < 1 || k < 1 || stride < 1 || pad < 0 || pad >= k) return DSTD_E_INVALID;
    const int Ho = (H + 2 * pad - k) / stride + 1, Wo = (W + 2 * pad - k) / stride + 1;
    if (Ho < 1 || Wo < 1) return DSTD_E_INVALID;
    const long long K = (long long)k * k * C;
    const long long npos = (long long)B * Ho * Wo;
    if (K > 65535 || npos * Mp > (1ll << 31) - 1 || B > 65535) return DSTD_E_UNSUPPORTED;
    pl->g = ConvGeom{B, H, W, C, Ho, Wo, k, stride, pad};
    pl->K = (int)K;
    pl->kpad = pad8((int)K);
    pl->npos = (int)npos;
    const long long img = (long long)Ho * Wo;
    // per image: the im2col operands and the fp32 w^ of its positions
    const long long per_img = img * Mp * ((long long)pl->kpad * 2 * (two ? 2 : 1) + (long long)((Cout + 3) & ~3) * 4);
    long long imgs = (long long)(kConvChunkBudget / (size_t)(per_img > 0 ? per_img : 1));
    if (imgs < 1) imgs = 1;
    if (imgs > B) imgs = B;
    pl->chunk = (int)(imgs * img);
    pl->nchunks = (int)((npos + pl->chunk - 1) / pl->chunk);
    return DSTD_OK;
}

struct ConvFwdWs {
    uint16_t *w_hi = nullptr, *w_lo = nullptr, *s_hi = nullptr, *s_lo = nullptr;
    float *rowsum = nullptr, *row_scale = nullptr, *D = nullptr;
    int ldD = 0;
    size_t bytes = 0;
};

ConvFwdWs conv_fwd_layout(void *base, const ConvPlan &pl, int Cout, int Mp, OpKind op) {
    ConvFwdWs w;
    Bump b(base);
    const bool two = two_part(op);
    w.rowsum = b.take<float>(Cout);
    w.row_scale = b.take<float>(Cout);
    w.w_hi = b.take<uint16_t>((size_t)Cout * pl.kpad);
    if (two) w.w_lo = b.take<uint16_t>((size_t)Cout * pl.kpad);
    w.s_hi = b.take<uint16_t>((size_t)pl.chunk * Mp * pl.kpad);
    if (two) w.s_lo = b.take<uint16_t>((size_t)pl.chunk * Mp * pl.kpad);
    w.ldD = (Cout + 3) & ~3;
    w.D = b.take<float>((size_t)pl.chunk * Mp * w.ldD);  // w^ of a chunk: row (pos, m), column o
    w.bytes = b.off;
    return w;
}

struct ConvBwdWs {
    __nv_bfloat16 *wt_hi = nullptr, *wt_lo = nullptr, *dA_hi = nullptr, *dA_lo = nullptr, *sT_hi = nullptr,
                  *sT_lo = nullptr;
    float *part = nullptr, *count = nullptr;
    int ldt = 0, ldn = 0, ldbm = 0, ldp = 0, splits = 1;
    size_t bytes = 0;
};

ConvBwdWs conv_bwd_layout(void *base, const ConvPlan &pl, int Cout, int Mp, OpKind op, bool need_gt) {
    ConvBwdWs w;
    Bump b(base);
    const bool two = two_part(op);
    const long long cols = (long long)pl.chunk * Mp;
    w.ldt = pad8(Cout);
    w.ldn = pad8(Cout);
    w.ldbm = pad8((int)cols);
    w.ldp = (pl.K + 3) & ~3;
    w.splits = dw_splits(pl.K, Cout, (int)cols, op);
    w.count = b.take<float>(Cout);
    // (dW adds into g_W atomically: no split-K partials)
    // dw^ of a chunk once, [Cout, positions*Mp]: dW's A operand and, read
    // transposed, the B operand of dS
    w.dA_hi = b.take<__nv_bfloat16>((size_t)Cout * w.ldbm);
    if (two) w.dA_lo = b.take<__nv_bfloat16>((size_t)Cout * w.ldbm);
    w.sT_hi = b.take<__nv_bfloat16>((size_t)pl.K * w.ldbm);
    if (two) w.sT_lo = b.take<__nv_bfloat16>((size_t)pl.K * w.ldbm);
    if (need_gt) {
        w.wt_hi = b.take<__nv_bfloat16>((size_t)pl.K * w.ldt);
        if (two) w.wt_lo = b.take<__nv_bfloat16>((size_t)pl.K * w.ldt);
    }
    w.bytes = b.off;
    return w;
}

// Implicit-GEMM path (bf16, C_in and C_out multiples of 64): the binned
// input is one 8-byte record per input spike (grid step and its two
// weights), from which the forward and dW contractions generate their
// operand tiles in shared memory (no binned or im2col array in memory); w^
// is [positions][C_out][Mp] and dw^ [positions][Mp][C_out]. Chunks of whole images bound the
// scratch.
constexpr size_t kConvImplBudget = 4ull << 30;  // bytes of per-image operands per chunk
static int g_conv_chunk_images = 0;             // 0: from the budget; else at most this many images per chunk
// operand of the implicit-GEMM forward and dW: 0 by layer shape, 1 generated
// on chip from the records everywhere, 2 the binned input S written out and
// read through TMA everywhere
static int g_conv_operand_policy = 0;

// By default both contractions read S wherever its writer takes the
// channel count: writing S costs one pass at HBM speed per chunk and
// direction, and the TMA-fed tiles keep the tensor core fed, where the
// generator warps (one stage per group when the filters stream) do not.
// (A layer with fewer than 64 input channels is padded to 64 and always
// reads S: the generated path takes multiples of 64 only.)
static bool conv_fwd_tma(const ConvGeom &g, int C_out) {
    (void)C_out;
    const int Cp = conv_padded_channels(g.C);
    return conv_bin_S_supported(Cp) && (g_conv_operand_policy != 1 || Cp != g.C);
}
static bool conv_dw_tma(const ConvGeom &g, int C_out) {
    (void)C_out;
    const int Cp = conv_padded_channels(g.C);
    return conv_bin_S_supported(Cp) && (g_conv_operand_policy != 1 || Cp != g.C);
}
// the geometry the implicit kernels see: input channels padded to 64
static ConvGeom conv_padded(const ConvGeom &g) {
    ConvGeom gp = g;
    gp.C = conv_padded_channels(g.C);
    return gp;
}

struct ConvImplWs {
    __nv_bfloat16 *Wf = nullptr, *Wt = nullptr, *dwh = nullptr, *S = nullptr;
    uint2 *rec = nullptr;
    float *rowsum = nullptr, *count = nullptr, *what = nullptr;
    int imgs = 1;
    size_t bytes = 0;
};

int conv_impl_images(const ConvGeom &g, int C_out, int Mp) {
    // per image, the larger of the forward's and the backward's scratch:
    // S (bf16) or the 8-byte records, and w^ (fp32, generated forward only)
    // or dw^ (bf16)
    const long long outs = (long long)g.Ho * g.Wo * Mp * C_out;
    const int Cp = conv_padded_channels(g.C);
    const long long S = (long long)g.H * g.W * Mp * Cp * 2, rec = (long long)g.H * g.W * g.C * 8;
    const long long fwd = conv_fwd_tma(g, C_out) ? S : rec + outs * 4;
    const long long bwd = (conv_dw_tma(g, C_out) ? S : rec) + outs * 2;
    const long long per_img = fwd > bwd ? fwd : bwd;
    long long imgs = (long long)(kConvImplBudget / (size_t)per_img);
    if (g_conv_chunk_images > 0 && imgs > g_conv_chunk_images) imgs = g_conv_chunk_images;
    if (imgs < 1) imgs = 1;
    if (imgs > g.B) imgs = g.B;
    return (int)imgs;
}

ConvImplWs conv_impl_layout(void *base, const ConvGeom &g, int C_out, int Mp, bool fwd) {
    ConvImplWs w;
    Bump b(base);
    const int Cp = conv_padded_channels(g.C);
    const long long K = (long long)g.k * g.k * Cp;
    w.imgs = conv_impl_images(g, C_out, Mp);
    w.rowsum = b.take<float>(C_out);
    w.count = b.take<float>(C_out);
    w.Wf = b.take<__nv_bfloat16>((size_t)C_out * K);
    w.Wt = b.take<__nv_bfloat16>((size_t)C_out * K);
    if (fwd ? conv_fwd_tma(g, C_out) : conv_dw_tma(g, C_out))
        w.S = b.take<__nv_bfloat16>((size_t)w.imgs * g.H * g.W * Mp * Cp);
    else
        w.rec = b.take<uint2>((size_t)w.imgs * g.H * g.W * g.C);
    if (fwd && !w.S)
        w.what = b.take<float>((size_t)w.imgs * g.Ho * g.Wo * Mp * C_out);
    else
        w.dwh = b.take<__nv_bfloat16>((size_t)w.imgs * g.Ho * g.Wo * Mp * C_out);
    w.bytes = b.off;
    return w;
}

bool conv_use_implicit(dstd_math math, const ConvGeom &g, int C_out, int Mp) {
    return math == DSTD_MATH_BF16 && conv_implicit_supported(g, C_out, Mp);
}

int conv_fwd_implicit(const float *t_in, const float *W, const ConvGeom &g, int C_out, const dstd_params *p, int Mp,
                      float *t_out, void *saved, float *penalty, void *workspace, size_t ws_bytes, cudaStream_t st) {
    const ConvImplWs ws = conv_impl_layout(workspace, g, C_out, Mp, true);
    if (ws_bytes < ws.bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    const long long npos = (long long)g.B * g.Ho * g.Wo;
    const int K = g.k * g.k * g.C;
    const ConvGeom gp = conv_padded(g);
    Saved sv = saved_view(saved, npos, C_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    {
        Timed tm(KK_PREP, st);
        if (gp.C == g.C) {
            TRY(cu(launch_prep_weights(W, C_out, K, OpKind::BF16, ws.Wf, nullptr, K, nullptr, nullptr, 0, nullptr, 0,
                                       ws.rowsum, st)));
        } else {  // rows (o, tap) of C channels into rows of gp.C (zero padding), row sums per o
            TRY(cu(launch_prep_weights(W, C_out * g.k * g.k, g.C, OpKind::BF16, ws.Wf, nullptr, gp.C, nullptr,
                                       nullptr, 0, nullptr, 0, nullptr, st)));
            TRY(cu(launch_prep_weights(W, C_out, K, OpKind::BF16, nullptr, nullptr, K, nullptr, nullptr, 0, nullptr, 0,
                                       ws.rowsum, st)));
        }
    }
    for (int img0 = 0; img0 < g.B; img0 += ws.imgs) {
        const int ni = (g.B - img0) < ws.imgs ? (g.B - img0) : ws.imgs;
        const long long in_off = (long long)img0 * g.H * g.W * g.C;
        const long long out_off = (long long)img0 * g.Ho * g.Wo * C_out;
        const long long P_out = (long long)ni * g.Ho * g.Wo;
        {
            Timed tm(KK_BIN, st);
            if (ws.S)
                TRY(cu(launch_bin_S(t_in + in_off, (long long)ni * g.H * g.W, gp.C, g.C, c, ws.S, st)));
            else
                TRY(cu(launch_bin_rec(t_in + in_off, (long long)ni * g.H * g.W * g.C, c, ws.rec, st)));
        }
        if (ws.S) {  // the scan runs in the contraction's epilogue
            Timed tm(KK_GEMM_FWD, st);
            TRY(cu(launch_conv_fwd_tma(gp, ni, C_out, c, ws.S, ws.Wf, ws.rowsum, t_out + out_off, sv.q + out_off,
                                       sv.s + out_off, sv.vdot + out_off, penalty, st)));
            continue;
        }
        {
            Timed tm(KK_GEMM_FWD, st);
            TRY(cu(launch_conv_fwd_gen(g, ni, C_out, c, ws.rec, ws.Wf, ws.what, st)));
        }
        Timed tm(KK_SCAN, st);
        TRY(cu(launch_scan_solve(ws.what, (long long)Mp * C_out, Mp, 1, (int)P_out, C_out, c, nullptr, ws.rowsum,
                                 t_out + out_off, sv.q + out_off, sv.s + out_off, sv.vdot + out_off, penalty, st)));
    }
    return DSTD_OK;
}

int conv_bwd_implicit(const float *t_in, const float *W, const ConvGeom &g, int C_out, const dstd_params *p, int Mp,
                      const float *t_out, const void *saved, const float *g_t_out, float *g_t_in, float *g_W,
                      void *workspace, size_t ws_bytes, cudaStream_t st) {
    const ConvImplWs ws = conv_impl_layout(workspace, g, C_out, Mp, false);
    if (ws_bytes < ws.bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    const long long npos = (long long)g.B * g.Ho * g.Wo;
    const int T = g.k * g.k;
    Saved sv = saved_view(const_cast<void *>(saved), npos, C_out);
    const float qcoef = -p->gamma_q * p->penalty_norm;
    TRY(cu(cudaMemsetAsync(g_W, 0, sizeof(float) * (size_t)C_out * T * g.C, st)));
    TRY(cu(cudaMemsetAsync(ws.count, 0, sizeof(float) * (size_t)C_out, st)));
    const ConvGeom gp = conv_padded(g);
    if (g_t_in) {
        Timed tm(KK_PREP, st);
        TRY(cu(launch_filters_t(W, C_out, T, g.C, gp.C, ws.Wt, st)));
    }
    for (int img0 = 0; img0 < g.B; img0 += ws.imgs) {
        const int ni = (g.B - img0) < ws.imgs ? (g.B - img0) : ws.imgs;
        const bool last = img0 + ni >= g.B;
        const long long in_off = (long long)img0 * g.H * g.W * g.C;
        const long long out_off = (long long)img0 * g.Ho * g.Wo * C_out;
        const long long P_out = (long long)ni * g.Ho * g.Wo;
        {
            Timed tm(KK_DWHAT, st);
            TRY(cu(launch_dwhat_pmc(t_out + out_off, sv.q + out_off, sv.s + out_off, sv.vdot + out_off,
                                    g_t_out ? g_t_out + out_off : nullptr, P_out, C_out, c, ws.dwh, ws.count, st)));
        }
        if (g_t_in) {
            Timed tm(KK_GEMM_DS, st);
            TRY(cu(launch_conv_ds_gemm(gp, ni, C_out, c, ws.dwh, ws.Wt, t_in + in_off, g_t_in + in_off, g.C, st)));
        }
        {
            Timed tm(KK_BIN_T, st);
            if (ws.S)
                TRY(cu(launch_bin_S(t_in + in_off, (long long)ni * g.H * g.W, gp.C, g.C, c, ws.S, st)));
            else
                TRY(cu(launch_bin_rec(t_in + in_off, (long long)ni * g.H * g.W * g.C, c, ws.rec, st)));
        }
        Timed tm(KK_GEMM_DW, st);
        if (ws.S)
            TRY(cu(launch_conv_dw_tma(gp, ni, C_out, c, ws.S, ws.dwh, last ? ws.count : nullptr, qcoef, g_W, g.C,
                                      st)));
        else
            TRY(cu(launch_conv_dw_gen(g, ni, C_out, c, ws.rec, ws.dwh, last ? ws.count : nullptr, qcoef, g_W, st)));
    }
    return DSTD_OK;
}

}  // namespace

extern "C" {

int dstd_version(void) { return kVersion; }

const char *dstd_error_string(int code) {
    switch (code) {
        case DSTD_OK: return "ok";
        case DSTD_E_INVALID: return "invalid argument";
        case DSTD_E_UNSUPPORTED: return "unsupported size or mode";
        case DSTD_E_WORKSPACE: return "workspace too small";
        case DSTD_E_CUDA: return "CUDA call or kernel launch failed";
        case DSTD_E_TIMEOUT: return "a bounded device-side wait expired";
        case DSTD_E_NO_DEVICE: return "no usable sm_103 device";
        default: return "unknown error code";
    }
}

size_t dstd_dense_saved_bytes(int B, int N_out) {
    if (B < 1 || N_out < 1) return 0;
    Bump b(nullptr);
    b.take<int>((size_t)B * N_out);
    b.take<float>((size_t)B * N_out);
    b.take<float>((size_t)B * N_out);
    return b.off;
}

size_t dstd_dense_workspace_bytes(int B, int N_in, int N_out, const dstd_params *p, dstd_math math) {
    if (check_sizes(B, N_in, N_out) != DSTD_OK || check_params(p) != DSTD_OK) return 0;
    const int Mp = padded_M(p->M);
    if (check_math(math, Mp) != DSTD_OK) return 0;
    const OpKind op = op_of(math);
    size_t f = fwd_layout(nullptr, B, N_in, N_out, Mp, op, true).bytes;
    size_t g = bwd_layout(nullptr, B, N_in, N_out, Mp, bwd_op_of(math), true).bytes;
    return f > g ? f : g;
}

int dstd_binning(const float *t_in, int B, int N, const dstd_params *p, float *s, float *ds,
                 dstd_stream_t stream) {
    if (!t_in || !s || B < 1 || N < 1) return DSTD_E_INVALID;
    TRY(check_params(p));
    TRY(device_ok());
    LifConst c = make_const(*p, padded_M(p->M));
    Timed tm(KK_BIN_PUB, (cudaStream_t)stream);
    return cu(launch_binning_public(t_in, B, N, c, s, ds, (cudaStream_t)stream));
}

int dstd_dense_what(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                    dstd_math math, float *what, void *workspace, size_t ws_bytes, dstd_stream_t stream) {
    if (!t_in || !W || !what || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace)) return DSTD_E_INVALID;
    const OpKind op = op_of(math);
    if (ws_bytes < fwd_layout(nullptr, B, N_in, N_out, Mp, op, true).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs ws = fwd_layout(workspace, B, N_in, N_out, Mp, op, true);
    TRY(dense_forward_core(t_in, W, B, N_in, N_out, c, op, ws, true, nullptr, nullptr, nullptr, st));
    Timed tm(KK_WHAT_PUB, st);
    return cu(launch_what_to_public(ws.D, (long long)B * Mp, B, N_out, p->M, Mp, what, st));
}

int dstd_scan_solve(const float *what, int B, int N_out, const dstd_params *p, const float *w_rowsum, float *t_out,
                    void *saved, float *penalty, dstd_stream_t stream) {
    if (!what || !t_out || B < 1 || N_out < 1) return DSTD_E_INVALID;
    TRY(check_params(p));
    TRY(device_ok());
    cudaStream_t st = (cudaStream_t)stream;
    LifConst c = make_const(*p, padded_M(p->M));
    Saved sv{nullptr, nullptr, nullptr};
    if (saved) sv = saved_view(saved, B, N_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    Timed tm(KK_SCAN, st);
    return cu(launch_scan_solve(what, (long long)N_out * p->M, p->M, 1, B, N_out, c, nullptr, w_rowsum, t_out, sv.q,
                                sv.s, sv.vdot, penalty, st));
}

int dstd_dense_fwd(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                   dstd_math math, float *t_out, void *saved, float *penalty, void *workspace, size_t ws_bytes,
                   dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    const OpKind op = op_of(math);
    if (ws_bytes < fwd_layout(nullptr, B, N_in, N_out, Mp, op, false).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs ws = fwd_layout(workspace, B, N_in, N_out, Mp, op, false);
    Saved sv = saved_view(saved, B, N_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    return dense_forward_core(t_in, W, B, N_in, N_out, c, op, ws, false, &sv, t_out, penalty, st);
}

int dstd_dense_fwd_ce(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                      dstd_math math, float *t_out, void *saved, float *penalty, void *workspace, size_t ws_bytes,
                      const int32_t *labels, float tau_soft, float t_silent, float *loss, float *g_t_out,
                      dstd_stream_t stream) {
    if (!labels || !loss || !g_t_out) return DSTD_E_INVALID;
    if (!(tau_soft > 0.0f) || !isfinite(tau_soft) || !isfinite(t_silent)) return DSTD_E_INVALID;
    if (!t_in || !W || !t_out || !saved || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    if ((reinterpret_cast<uintptr_t>(loss) & 7) != 0) return DSTD_E_INVALID;
    const OpKind op = op_of(math);
    if (ws_bytes < fwd_layout(nullptr, B, N_in, N_out, Mp, op, false).bytes || ws_bytes < sizeof(float) * (size_t)B)
        return DSTD_E_WORKSPACE;
    TRY(device_ok());
    cudaStream_t st = (cudaStream_t)stream;
    if (!narrow_layer(N_in, N_out, p->M, op)) {
        TRY(dstd_dense_fwd(t_in, W, B, N_in, N_out, p, math, t_out, saved, penalty, workspace, ws_bytes, stream));
        return dstd_ce_loss(t_out, labels, B, N_out, tau_soft, t_silent, loss, g_t_out, stream);
    }
    LifConst c = make_const(*p, Mp);
    Saved sv = saved_view(saved, B, N_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    NarrowCe ce;
    ce.labels = labels;
    ce.tau_soft = tau_soft;
    ce.t_silent = t_silent;
    ce.loss = loss;
    ce.g = g_t_out;
    ce.scratch = static_cast<float *>(workspace);
    Timed tm(KK_NARROW_FWD, st);
    return cu(launch_narrow_fwd(t_in, W, B, N_in, N_out, c, t_out, sv.q, sv.s, sv.vdot, penalty, st, ce));
}

int dstd_dense_bwd(const float *t_in, const float *W, const float *t_out, const void *saved, const float *g_t_out,
                   int B, int N_in, int N_out, const dstd_params *p, dstd_math math, float *g_t_in, float *g_W,
                   void *workspace, size_t ws_bytes, dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !g_W || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    const OpKind bop = bwd_op_of(math);
    const OpKind op = bop;
    const bool need_gt = g_t_in != nullptr;
    if (ws_bytes < bwd_layout(nullptr, B, N_in, N_out, Mp, bop, need_gt).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    BwdWs ws = bwd_layout(workspace, B, N_in, N_out, Mp, bop, need_gt);
    Saved sv = saved_view(const_cast<void *>(saved), B, N_out);
    const long long cols = (long long)B * Mp;
    const float qcoef = -p->gamma_q * p->penalty_norm;
    if (narrow_layer(N_in, N_out, c.M, op)) {
        Timed tm(KK_NARROW_BWD, st);
        return cu(launch_narrow_bwd(t_in, W, t_out, sv.q, sv.s, sv.vdot, g_t_out, B, N_in, N_out, c, qcoef, g_t_in,
                                    g_W, st));
    }
    if (op == OpKind::F32) {
        {
            Timed tm(KK_DWHAT, st);
            TRY(cu(launch_dwhat(t_out, sv.q, sv.s, sv.vdot, g_t_out, B, N_out, c, op, ws.dA32, nullptr, ws.ldbm,
                                ws.dB32, nullptr, ws.ldn, ws.count, st)));
        }
        if (need_gt) {
            {
                Timed tm(KK_PREP, st);
                TRY(cu(launch_prep_weights(W, N_out, N_in, op, nullptr, nullptr, 0, nullptr, nullptr, 0, ws.wt32,
                                           ws.ldt, nullptr, st)));
            }
            {
                Timed tm(KK_GEMM_DS, st);
                TRY(cu(launch_sgemm_tn(ws.wt32, ws.ldt, ws.dB32, ws.ldn, ws.DS, (int)cols, N_in, (int)cols, N_out, 1,
                                       0, st)));
            }
            {
                Timed tm(KK_GT, st);
                TRY(cu(launch_gt_from_ds(ws.DS, cols, t_in, B, N_in, c, g_t_in, st)));
            }
        }
        {
            Timed tm(KK_BIN_T, st);
            TRY(cu(launch_binning(t_in, B, N_in, c, op, true, ws.sT32, nullptr, ws.ldbm, st)));
        }
        const long long zs = (long long)N_out * ws.ldp;
        {
            Timed tm(KK_GEMM_DW, st);
            TRY(cu(launch_sgemm_tn(ws.dA32, ws.ldbm, ws.sT32, ws.ldbm, ws.part, ws.ldp, N_out, N_in, (int)cols,
                                   ws.splits, zs, st)));
        }
        Timed tm(KK_REDUCE, st);
        return cu(launch_dw_reduce(ws.part, ws.splits, zs, ws.ldp, N_out, N_in, ws.count, qcoef, g_W, st));
    }
    const bool small_gt = need_gt && N_out <= kGradtSmallMaxOut;
    {
        // three independent producers: dw^ (caller's stream), s^T with the
        // per-input kernel derivatives (side 0), and W^T for dS plus the
        // zeroing of dW (side 1)
        Fork f(st);
        {
            Timed tm(KK_BIN_T, f.side[0]);
            TRY(cu(launch_binning(t_in, B, N_in, c, op, true, ws.sT_hi, ws.sT_lo, ws.ldbm, f.side[0], ws.bw)));
        }
        if (need_gt && !small_gt) {
            Timed tm(KK_PREP, f.side[1]);
            TRY(cu(launch_prep_weights(W, N_out, N_in, op, nullptr, nullptr, 0, ws.wt_hi, ws.wt_lo, ws.ldt, nullptr,
                                       0, nullptr, f.side[1])));
        }
        TRY(cu(cudaMemsetAsync(g_W, 0, sizeof(float) * (size_t)N_out * N_in, f.side[1])));
        {
            Timed tm(KK_DWHAT, st);
            TRY(cu(launch_dwhat(t_out, sv.q, sv.s, sv.vdot, g_t_out, B, N_out, c, op, ws.dA_hi, ws.dA_lo, ws.ldbm,
                                nullptr, nullptr, 0, ws.count, st)));
        }
        TRY(f.join());
    }
    if (small_gt) {
        // few outputs: the input-time gradient by its definition, no contraction
        Timed tm(KK_GT, st);
        TRY(cu(launch_gradt_small(W, N_out, N_in, B, c, ws.bw, ws.dA_hi, ws.dA_lo, ws.ldbm, g_t_in, st)));
    } else if (need_gt) {
        TcEpiArgs a{};
        a.c = c;
        a.B = B;
        a.N = N_in;
        a.t_in = t_in;
        a.g_t_in = g_t_in;
        a.bw = ws.bw;
        Timed tm(KK_GEMM_DS, st);
        // dw^ read transposed from its dW layout [N_out, B*Mp]
        TRY(cu(launch_tc_gemm(ws.wt_hi, ws.wt_lo, ws.ldt, ws.dA_hi, ws.dA_lo, ws.ldbm, N_in, (int)cols, N_out, 1, op,
                              Epi::GradT, a, st, true)));
    }
    if (dw_on_pairs(N_in, N_out, (int)cols, op)) {
        // on SM pairs, computed transposed: (s^T dw^)[j, i] stored as dW[i][j];
        // then the dead-neuron term qcoef * count_i added in place
        TcEpiArgs a{};
        a.D = g_W;
        a.ldd = N_in;
        {
            Timed tm(KK_GEMM_DW, st);
            TRY(cu(launch_tc_gemm_pair_storeT(ws.sT_hi, ws.sT_lo, ws.ldbm, ws.dA_hi, ws.dA_lo, ws.ldbm, N_in, N_out,
                                              (int)cols, op, a, st)));
        }
        if (qcoef == 0.0f) return DSTD_OK;
        Timed tm(KK_REDUCE, st);
        return cu(launch_dw_reduce(g_W, 1, 0, N_in, N_out, N_in, ws.count, qcoef, g_W, st, false));
    }
    // dW = dw^T s: the split-K slices add into g_W (zeroed above); split 0
    // also adds the dead-neuron term qcoef * count_i
    TcEpiArgs a{};
    a.D = g_W;
    a.ldd = N_in;
    a.atomic = 1;
    a.qcount = ws.count;
    a.qcoef = qcoef;
    Timed tm(KK_GEMM_DW, st);
    return cu(launch_tc_gemm(ws.dA_hi, ws.dA_lo, ws.ldbm, ws.sT_hi, ws.sT_lo, ws.ldbm, N_out, N_in, (int)cols,
                             ws.splits, op, Epi::Store, a, st));
}

int dstd_ce_loss(const float *t_L, const int32_t *labels, int B, int C, float tau_soft, float t_silent, float *loss,
                 float *g_t_L, dstd_stream_t stream) {
    if (!t_L || !labels || !loss || !g_t_L || B < 1 || C < 1) return DSTD_E_INVALID;
    if (!(tau_soft > 0.0f) || !isfinite(tau_soft) || !isfinite(t_silent)) return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_LOSS, (cudaStream_t)stream);
    return cu(launch_ce_loss(t_L, labels, B, C, tau_soft, t_silent, loss, g_t_L, (cudaStream_t)stream));
}

int dstd_concat_channels(const float *a, int C_a, float delay_a, const float *b, int C_b, int64_t positions,
                         float *out, dstd_stream_t stream) {
    if (!a || !b || !out || C_a < 1 || C_b < 1 || positions < 1 || !isfinite(delay_a)) return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_SKIP, (cudaStream_t)stream);
    return cu(launch_concat_channels(a, C_a, delay_a, b, C_b, positions, out, (cudaStream_t)stream));
}

int dstd_split_channels(const float *g, int C_a, int C_b, int64_t positions, float *g_a, int accumulate_a,
                        float *g_b, int accumulate_b, dstd_stream_t stream) {
    if (!g || (!g_a && !g_b) || C_a < 1 || C_b < 1 || positions < 1) return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_SKIP, (cudaStream_t)stream);
    return cu(launch_split_channels(g, C_a, C_b, positions, g_a, accumulate_a != 0, g_b, accumulate_b != 0,
                                    (cudaStream_t)stream));
}

int dstd_sum_t_loss(const float *t, int64_t n, float *loss, float *g, dstd_stream_t stream) {
    if (!t || !loss || !g || n < 1) return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_LOSS, (cudaStream_t)stream);
    return cu(launch_sum_t(t, n, loss, g, (cudaStream_t)stream));
}

int dstd_adamw(float *w, const float *g, float *m, float *v, int64_t n, float lr, float beta1, float beta2, float eps,
               float weight_decay, int step, dstd_stream_t stream) {
    if (!w || !g || !m || !v || n < 1 || step < 1) return DSTD_E_INVALID;
    if (!(lr >= 0.0f) || !(beta1 >= 0.0f && beta1 < 1.0f) || !(beta2 >= 0.0f && beta2 < 1.0f) || !(eps > 0.0f))
        return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_ADAMW, (cudaStream_t)stream);
    return cu(launch_adamw(w, g, m, v, n, lr, beta1, beta2, eps, weight_decay, step, (cudaStream_t)stream));
}

int dstd_adamw_multi(int count, float *const *w, const float *const *g, float *const *m, float *const *v,
                     const int64_t *n, float lr, float beta1, float beta2, float eps, float weight_decay,
                     int32_t *step, const float *lr_dev, dstd_stream_t stream) {
    if (count < 1 || count > kAdamMaxTensors || !w || !g || !m || !v || !n || !step) return DSTD_E_INVALID;
    if ((reinterpret_cast<uintptr_t>(step) & 7) != 0) return DSTD_E_INVALID;
    if (!(lr >= 0.0f) || !(beta1 >= 0.0f && beta1 < 1.0f) || !(beta2 >= 0.0f && beta2 < 1.0f) || !(eps > 0.0f))
        return DSTD_E_INVALID;
    AdamMultiArgs a{};
    for (int i = 0; i < count; ++i) {
        if (!w[i] || !g[i] || !m[i] || !v[i] || n[i] < 1) return DSTD_E_INVALID;
        a.seg[i] = AdamSeg{w[i], g[i], m[i], v[i], (long long)n[i], 0};
    }
    a.count = count;
    a.lr = lr;
    a.b1 = beta1;
    a.b2 = beta2;
    a.eps = eps;
    a.wd = weight_decay;
    a.step = step;
    a.lr_dev = lr_dev;
    TRY(device_ok());
    Timed tm(KK_ADAMW, (cudaStream_t)stream);
    return cu(launch_adamw_multi(a, (cudaStream_t)stream));
}

size_t dstd_conv_workspace_bytes(int B, int H, int W, int C_in, int C_out, int k, int stride, int pad,
                                 const dstd_params *p, dstd_math math) {
    if (check_params(p) != DSTD_OK || C_out < 1) return 0;
    const int Mp = padded_M(p->M);
    if (math == DSTD_MATH_F32 || check_math(math, Mp) != DSTD_OK) return 0;
    ConvPlan pl;
    if (conv_plan(B, H, W, C_in, k, stride, pad, Mp, true, C_out, &pl) != DSTD_OK) return 0;
    if (conv_use_implicit(math, pl.g, C_out, Mp)) {
        size_t f = conv_impl_layout(nullptr, pl.g, C_out, Mp, true).bytes;
        size_t g = conv_impl_layout(nullptr, pl.g, C_out, Mp, false).bytes;
        return f > g ? f : g;
    }
    size_t f = conv_fwd_layout(nullptr, pl, C_out, Mp, op_of(math)).bytes;
    size_t g = conv_bwd_layout(nullptr, pl, C_out, Mp, bwd_op_of(math), true).bytes;
    return f > g ? f : g;
}

int dstd_conv_fwd(const float *t_in, const float *W, int B, int H, int Wd, int C_in, int C_out, int k, int stride,
                  int pad, const dstd_params *p, dstd_math math, float *t_out, void *saved, float *penalty,
                  void *workspace, size_t ws_bytes, dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !workspace || C_out < 1) return DSTD_E_INVALID;
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    if (math == DSTD_MATH_F32) return DSTD_E_UNSUPPORTED;
    TRY(check_math(math, Mp));
    if (C_out > (1 << 20)) return DSTD_E_UNSUPPORTED;
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    ConvPlan pl;
    TRY(conv_plan(B, H, Wd, C_in, k, stride, pad, Mp, true, C_out, &pl));
    if (conv_use_implicit(math, pl.g, C_out, Mp))
        return conv_fwd_implicit(t_in, W, pl.g, C_out, p, Mp, t_out, saved, penalty, workspace, ws_bytes,
                                 (cudaStream_t)stream);
    const OpKind op = op_of(math);
    if (ws_bytes < conv_fwd_layout(nullptr, pl, C_out, Mp, op).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    ConvFwdWs ws = conv_fwd_layout(workspace, pl, C_out, Mp, op);
    Saved sv = saved_view(saved, pl.npos, C_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    {
        Timed tm(KK_PREP, st);
        if (op == OpKind::F16X3)
            TRY(cu(launch_prep_weights_f16(W, C_out, pl.K, (__half *)ws.w_hi, (__half *)ws.w_lo, pl.kpad,
                                           ws.row_scale, ws.rowsum, st)));
        else
            TRY(cu(launch_prep_weights(W, C_out, pl.K, op, (__nv_bfloat16 *)ws.w_hi, (__nv_bfloat16 *)ws.w_lo,
                                       pl.kpad, nullptr, nullptr, 0, nullptr, 0, ws.rowsum, st)));
    }
    for (int ch = 0; ch < pl.nchunks; ++ch) {
        const int pos0 = ch * pl.chunk;
        const int npos = (pl.npos - pos0) < pl.chunk ? (pl.npos - pos0) : pl.chunk;
        {
            Timed tm(KK_BIN, st);
            TRY(cu(launch_binning_im2col(t_in, pl.g, pos0, npos, c, op, false, ws.s_hi, ws.s_lo, pl.kpad, st)));
        }
        const long long cols = (long long)npos * Mp;
        TcEpiArgs a{};
        a.D = ws.D;
        a.ldd = cols;
        a.zstride = 0;
        a.row_scale = op == OpKind::F16X3 ? ws.row_scale : nullptr;
        {
            Timed tm(KK_GEMM_FWD, st);
            TRY(cu(launch_tc_gemm(ws.w_hi, ws.w_lo, pl.kpad, ws.s_hi, ws.s_lo, pl.kpad, C_out, (int)cols, pl.K, 1, op,
                                  Epi::Store, a, st)));
        }
        const long long off = (long long)pos0 * C_out;
        Timed tr(KK_SCAN, st);
        TRY(cu(launch_scan_solve(ws.D, Mp, cols, 1, npos, C_out, c, nullptr, ws.rowsum, t_out + off, sv.q + off,
                                 sv.s + off, sv.vdot + off, penalty, st)));
    }
    return DSTD_OK;
}

int dstd_conv_bwd(const float *t_in, const float *W, const float *t_out, const void *saved, const float *g_t_out,
                  int B, int H, int Wd, int C_in, int C_out, int k, int stride, int pad, const dstd_params *p,
                  dstd_math math, float *g_t_in, float *g_W, void *workspace, size_t ws_bytes,
                  dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !g_W || !workspace || C_out < 1) return DSTD_E_INVALID;
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    if (math == DSTD_MATH_F32) return DSTD_E_UNSUPPORTED;
    TRY(check_math(math, Mp));
    if (C_out > (1 << 20)) return DSTD_E_UNSUPPORTED;
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    ConvPlan pl;
    TRY(conv_plan(B, H, Wd, C_in, k, stride, pad, Mp, true, C_out, &pl));
    if (conv_use_implicit(math, pl.g, C_out, Mp))
        return conv_bwd_implicit(t_in, W, pl.g, C_out, p, Mp, t_out, saved, g_t_out, g_t_in, g_W, workspace,
                                 ws_bytes, (cudaStream_t)stream);
    const OpKind bop = bwd_op_of(math);
    const bool need_gt = g_t_in != nullptr;
    if (ws_bytes < conv_bwd_layout(nullptr, pl, C_out, Mp, bop, need_gt).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    ConvBwdWs ws = conv_bwd_layout(workspace, pl, C_out, Mp, bop, need_gt);
    Saved sv = saved_view(const_cast<void *>(saved), pl.npos, C_out);
    const float qcoef = -p->gamma_q * p->penalty_norm;
    if (need_gt) {
        TRY(cu(cudaMemsetAsync(g_t_in, 0, sizeof(float) * (size_t)B * H * Wd * C_in, st)));
        Timed tm(KK_PREP, st);
        TRY(cu(launch_prep_weights(W, C_out, pl.K, bop, nullptr, nullptr, 0, ws.wt_hi, ws.wt_lo, ws.ldt, nullptr, 0,
                                   nullptr, st)));
    }
    for (int ch = 0; ch < pl.nchunks; ++ch) {
        const int pos0 = ch * pl.chunk;
        const int npos = (pl.npos - pos0) < pl.chunk ? (pl.npos - pos0) : pl.chunk;
        const long long off = (long long)pos0 * C_out;
        const long long cols = (long long)npos * Mp;
        const bool last = (ch == pl.nchunks - 1);
        {
            Timed tm(KK_DWHAT, st);
            TRY(cu(launch_dwhat(t_out + off, sv.q + off, sv.s + off, sv.vdot + off, g_t_out ? g_t_out + off : nullptr,
                                npos, C_out, c, bop, ws.dA_hi, ws.dA_lo, ws.ldbm, nullptr, nullptr, 0, ws.count, st,
                                ch > 0)));
        }
        if (need_gt) {
            TcEpiArgs a{};
            a.c = c;
            a.B = npos;
            a.N = pl.K;
            a.t_in = t_in;
            a.g_t_in = g_t_in;
            a.conv = 1;
            a.pos0 = pos0;
            a.g = pl.g;
            Timed tm(KK_GEMM_DS, st);
            TRY(cu(launch_tc_gemm(ws.wt_hi, ws.wt_lo, ws.ldt, ws.dA_hi, ws.dA_lo, ws.ldbm, pl.K, (int)cols, C_out, 1,
                                  bop, Epi::GradT, a, st, true)));
        }
        {
            Timed tm(KK_BIN_T, st);
            TRY(cu(launch_binning_im2col(t_in, pl.g, pos0, npos, c, bop, true, ws.sT_hi, ws.sT_lo, ws.ldbm, st)));
        }
        // dW over all chunks and split-K slices adds into g_W (zeroed before
        // the first chunk); the last chunk's split 0 adds the dead-neuron term
        if (ch == 0) TRY(cu(cudaMemsetAsync(g_W, 0, sizeof(float) * (size_t)C_out * pl.K, st)));
        TcEpiArgs a{};
        a.D = g_W;
        a.ldd = pl.K;
        a.atomic = 1;
        a.qcount = last ? ws.count : nullptr;
        a.qcoef = qcoef;
        Timed tm(KK_GEMM_DW, st);
        TRY(cu(launch_tc_gemm(ws.dA_hi, ws.dA_lo, ws.ldbm, ws.sT_hi, ws.sT_lo, ws.ldbm, C_out, pl.K, (int)cols,
                              ws.splits, bop, Epi::Store, a, st)));
    }
    return DSTD_OK;
}

int dstd_timing_enable(int on) {
    if (cudaDeviceSynchronize() != cudaSuccess) return DSTD_E_CUDA;
    std::lock_guard<std::mutex> lk(g_timing.mu);
    drain_pending();
    for (int k = 0; k < KK_COUNT; ++k) {
        g_timing.ms[k] = 0.0;
        g_timing.n[k] = 0;
        // a graph may still record these: they are dropped from the list, not reused
        g_timing.graph[k].clear();
    }
    g_timing.on = on != 0;
    return DSTD_OK;
}

size_t dstd_exact_workspace_bytes(int B, int N_in, int N_out) {
    if (check_sizes(B, N_in, N_out) != DSTD_OK || N_in > kExactMaxIn) return 0;
    return exact_layout(nullptr, B, N_in, N_out).bytes;
}

int dstd_exact_fwd(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p, float *t_out,
                   void *workspace, size_t ws_bytes, dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    if (N_in > kExactMaxIn) return DSTD_E_UNSUPPORTED;
    if (!aligned16(workspace)) return DSTD_E_INVALID;
    if (ws_bytes < exact_layout(nullptr, B, N_in, N_out).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, padded_M(p->M));
    const double kmax = kernel_sup(c.av, c.aI) * (1.0 + 1e-6);
    ExactWs ws = exact_layout(workspace, B, N_in, N_out);
    Timed tm(KK_EXACT_FWD, (cudaStream_t)stream);
    return cu(launch_exact_fwd(t_in, W, B, N_in, N_out, c, p->t_end, (float)kmax, ws, t_out, (cudaStream_t)stream));
}

int dstd_exact_bwd(const float *t_in, const float *W, const float *t_out, const float *g_t_out, int B, int N_in,
                   int N_out, const dstd_params *p, float *g_t_in, float *g_W, void *workspace, size_t ws_bytes,
                   dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !g_t_out || !g_W || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    if (N_in > kExactMaxIn) return DSTD_E_UNSUPPORTED;
    if (!aligned16(workspace)) return DSTD_E_INVALID;
    if (ws_bytes < exact_layout(nullptr, B, N_in, N_out).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, padded_M(p->M));
    ExactWs ws = exact_layout(workspace, B, N_in, N_out);
    Timed tm(KK_EXACT_BWD, (cudaStream_t)stream);
    return cu(launch_exact_bwd(t_in, W, t_out, g_t_out, B, N_in, N_out, c, ws, g_t_in, g_W, (cudaStream_t)stream));
}

// ---------------------------------------------------------------------------
// Multi-spike layers (App. D): the forward operands and the contraction of
// the tensor-core modes, the scan with reset, and a backward whose dS is
// stored (each input spike gathers its own two bins).
// ---------------------------------------------------------------------------
struct MsSaved {
    int *q;
    float *I, *vdot;
};
MsSaved ms_saved_view(void *saved, int B, int N_out, int F) {
    Bump b(saved);
    MsSaved v;
    v.q = b.take<int>((size_t)B * N_out * F);
    v.I = b.take<float>((size_t)B * N_out * F);
    v.vdot = b.take<float>((size_t)B * N_out * F);
    return v;
}

struct MsBwdWs {
    __nv_bfloat16 *wt_hi = nullptr, *wt_lo = nullptr, *dA_hi = nullptr, *dA_lo = nullptr, *dB_hi = nullptr,
                  *dB_lo = nullptr, *sT_hi = nullptr, *sT_lo = nullptr;
    float *DS = nullptr;
    int ldt = 0, ldn = 0, ldbm = 0, splits = 1;
    size_t bytes = 0;
};
MsBwdWs ms_bwd_layout(void *base, int B, int N_in, int N_out, int Mp, OpKind op, bool need_gt) {
    MsBwdWs w;
    Bump b(base);
    const long long cols = (long long)B * Mp;
    const bool three = op == OpKind::BF16X3;
    w.ldt = pad8(N_out);
    w.ldn = pad8(N_out);
    w.ldbm = pad8((int)cols);
    w.splits = dw_splits(N_in, N_out, (int)cols, op);
    w.dA_hi = b.take<__nv_bfloat16>((size_t)N_out * w.ldbm);
    if (three) w.dA_lo = b.take<__nv_bfloat16>((size_t)N_out * w.ldbm);
    w.sT_hi = b.take<__nv_bfloat16>((size_t)N_in * w.ldbm);
    if (three) w.sT_lo = b.take<__nv_bfloat16>((size_t)N_in * w.ldbm);
    if (need_gt) {
        w.dB_hi = b.take<__nv_bfloat16>((size_t)cols * w.ldn);
        if (three) w.dB_lo = b.take<__nv_bfloat16>((size_t)cols * w.ldn);
        w.wt_hi = b.take<__nv_bfloat16>((size_t)N_in * w.ldt);
        if (three) w.wt_lo = b.take<__nv_bfloat16>((size_t)N_in * w.ldt);
        w.DS = b.take<float>((size_t)N_in * cols);
    }
    w.bytes = b.off;
    return w;
}

int check_ms(int F_in, int F_out, dstd_math math) {
    if (F_in < 1 || F_out < 1) return DSTD_E_INVALID;
    if (F_in > kMsMaxSpikes || F_out > kMsMaxSpikes) return DSTD_E_UNSUPPORTED;
    if (math == DSTD_MATH_F32) return DSTD_E_UNSUPPORTED;
    return DSTD_OK;
}

size_t dstd_ms_saved_bytes(int B, int N_out, int F_out) {
    if (B < 1 || N_out < 1 || F_out < 1 || F_out > kMsMaxSpikes) return 0;
    Bump b(nullptr);
    b.take<int>((size_t)B * N_out * F_out);
    b.take<float>((size_t)B * N_out * F_out);
    b.take<float>((size_t)B * N_out * F_out);
    return b.off;
}

size_t dstd_ms_workspace_bytes(int B, int N_in, int N_out, int F_in, int F_out, const dstd_params *p,
                               dstd_math math) {
    if (check_sizes(B, N_in, N_out) != DSTD_OK || check_params(p) != DSTD_OK) return 0;
    if (check_ms(F_in, F_out, math) != DSTD_OK) return 0;
    const int Mp = padded_M(p->M);
    if (check_math(math, Mp) != DSTD_OK) return 0;
    const size_t f = fwd_layout(nullptr, B, N_in, N_out, Mp, op_of(math), true).bytes;
    const size_t g = ms_bwd_layout(nullptr, B, N_in, N_out, Mp, bwd_op_of(math), true).bytes;
    return f > g ? f : g;
}

int dstd_dense_fwd_ms(const float *t_in, const float *W, int B, int N_in, int N_out, int F_in, int F_out,
                      const dstd_params *p, dstd_math math, float *t_out, void *saved, void *workspace,
                      size_t ws_bytes, dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    TRY(check_ms(F_in, F_out, math));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    const OpKind op = op_of(math);
    if (ws_bytes < fwd_layout(nullptr, B, N_in, N_out, Mp, op, true).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs ws = fwd_layout(workspace, B, N_in, N_out, Mp, op, true);
    MsSaved sv = ms_saved_view(saved, B, N_out, F_out);
    const long long cols = (long long)B * Mp;
    {
        Timed tm(KK_PREP, st);
        if (op == OpKind::F16X3)
            TRY(cu(launch_prep_weights_f16(W, N_out, N_in, (__half *)ws.w_hi, (__half *)ws.w_lo, ws.kpad,
                                           ws.row_scale, ws.rowsum, st)));
        else
            TRY(cu(launch_prep_weights(W, N_out, N_in, op, (__nv_bfloat16 *)ws.w_hi, (__nv_bfloat16 *)ws.w_lo,
                                       ws.kpad, nullptr, nullptr, 0, nullptr, 0, ws.rowsum, st)));
    }
    {
        Timed tm(KK_BIN, st);
        TRY(cu(launch_binning_ms(t_in, B, N_in, F_in, c, op, false, ws.s_hi, ws.s_lo, ws.kpad, st)));
    }
    {
        const int splits = fwd_splits(N_out, cols, N_in);
        if (splits > 1) TRY(cu(cudaMemsetAsync(ws.D, 0, sizeof(float) * (size_t)N_out * cols, st)));
        TcEpiArgs a{};
        a.row_scale = ws.row_scale;
        a.D = ws.D;
        a.ldd = cols;
        a.atomic = splits > 1;
        Timed tm(KK_GEMM_FWD, st);
        TRY(cu(launch_tc_gemm(ws.w_hi, ws.w_lo, ws.kpad, ws.s_hi, ws.s_lo, ws.kpad, N_out, (int)cols, N_in, splits,
                              op, Epi::Store, a, st)));
    }
    Timed tm(KK_SCAN, st);
    return cu(launch_scan_ms(ws.D, Mp, cols, B, N_out, c, F_out, t_out, sv.q, sv.I, sv.vdot, st));
}

int dstd_dense_bwd_ms(const float *t_in, const float *W, const float *t_out, const void *saved,
                      const float *g_t_out, int B, int N_in, int N_out, int F_in, int F_out, const dstd_params *p,
                      dstd_math math, float *g_t_in, float *g_W, void *workspace, size_t ws_bytes,
                      dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved || !g_W || !workspace) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    TRY(check_ms(F_in, F_out, math));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(workspace) || !aligned16(saved)) return DSTD_E_INVALID;
    const OpKind op = bwd_op_of(math);
    const bool need_gt = g_t_in != nullptr;
    if (ws_bytes < ms_bwd_layout(nullptr, B, N_in, N_out, Mp, op, need_gt).bytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    const LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    MsBwdWs ws = ms_bwd_layout(workspace, B, N_in, N_out, Mp, op, need_gt);
    MsSaved sv = ms_saved_view(const_cast<void *>(saved), B, N_out, F_out);
    const long long cols = (long long)B * Mp;
    {
        Timed tm(KK_DWHAT, st);
        TRY(cu(launch_dwhat_ms(t_out, sv.q, sv.I, sv.vdot, g_t_out, B, N_out, F_out, c, op, ws.dA_hi, ws.dA_lo,
                               ws.ldbm, ws.dB_hi, ws.dB_lo, ws.ldn, st)));
    }
    if (need_gt) {
        {
            Timed tm(KK_PREP, st);
            TRY(cu(launch_prep_weights(W, N_out, N_in, op, nullptr, nullptr, 0, ws.wt_hi, ws.wt_lo, ws.ldt, nullptr,
                                       0, nullptr, st)));
        }
        {
            // dS[j, (b, m)] = sum_i W_ij dw^_i(b, m), stored in fp32
            TcEpiArgs a{};
            a.D = ws.DS;
            a.ldd = cols;
            Timed tm(KK_GEMM_DS, st);
            TRY(cu(launch_tc_gemm(ws.wt_hi, ws.wt_lo, ws.ldt, ws.dB_hi, ws.dB_lo, ws.ldn, N_in, (int)cols, N_out, 1,
                                  op, Epi::Store, a, st)));
        }
        Timed tm(KK_GT, st);
        TRY(cu(launch_gt_ms(ws.DS, cols, t_in, B, N_in, F_in, c, g_t_in, st)));
    }
    {
        Timed tm(KK_BIN_T, st);
        TRY(cu(launch_binning_ms(t_in, B, N_in, F_in, c, op, true, ws.sT_hi, ws.sT_lo, ws.ldbm, st)));
    }
    TRY(cu(cudaMemsetAsync(g_W, 0, sizeof(float) * (size_t)N_out * N_in, st)));
    TcEpiArgs a{};
    a.D = g_W;
    a.ldd = N_in;
    a.atomic = 1;
    Timed tm(KK_GEMM_DW, st);
    return cu(launch_tc_gemm(ws.dA_hi, ws.dA_lo, ws.ldbm, ws.sT_hi, ws.sT_lo, ws.ldbm, N_out, N_in, (int)cols,
                             ws.splits, op, Epi::Store, a, st));
}

int dstd_set_pair_policy(int policy) {
    if (policy < 0 || policy > 2) return DSTD_E_INVALID;
    return tc_gemm_pair_policy(policy);
}

int dstd_timing_collect(void) {
    if (cudaDeviceSynchronize() != cudaSuccess) return DSTD_E_CUDA;
    std::lock_guard<std::mutex> lk(g_timing.mu);
    for (int k = 0; k < KK_COUNT; ++k) {
        for (auto &pr : g_timing.graph[k]) {
            float ms = 0.f;
            if (cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess) {
                g_timing.ms[k] += ms;
                g_timing.n[k] += 1;
            }
        }
    }
    return DSTD_OK;
}

int dstd_timing_read(int kind, float *total_ms, int64_t *launches) {
    if (kind < 0 || kind >= KK_COUNT || !total_ms || !launches) return DSTD_E_INVALID;
    if (cudaDeviceSynchronize() != cudaSuccess) return DSTD_E_CUDA;
    std::lock_guard<std::mutex> lk(g_timing.mu);
    drain_pending();
    *total_ms = (float)g_timing.ms[kind];
    *launches = g_timing.n[kind];
    return DSTD_OK;
}

int dstd_kernel_kind_count(void) { return KK_COUNT; }

const char *dstd_kernel_kind_name(int kind) {
    return (kind >= 0 && kind < KK_COUNT) ? kKindNames[kind] : "unknown";
}

int dstd_selftest_wait_timeout(uint32_t timeout_us, dstd_stream_t stream) {
    if (timeout_us == 0 || timeout_us > 10000000u) return DSTD_E_INVALID;
    TRY(device_ok());
    Timed tm(KK_SELFTEST, (cudaStream_t)stream);
    return cu(launch_wait_selftest(1000ull * timeout_us, (cudaStream_t)stream));
}

// ---------------------------------------------------------------------------
// Layer forward that allocates nothing (scratch in a static device array).
// ---------------------------------------------------------------------------
}  // extern "C"

namespace {

// Fixed scratch for dstd_dense_fwd_noalloc: 64 MiB, resident on every GPU
// that loads this library, for as long as the process runs.
constexpr size_t kNoAllocScratchBytes = 64ull << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void *g_noalloc_ptr[128] = {};

// Device address of the scratch array on the current device. The array's
// name is only a host-side stand-in, so its address is looked up (once per
// device, with that device current) and cached.
int noalloc_scratch(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DSTD_E_NO_DEVICE;
    if (dev < 0 || dev >= 128) return DSTD_E_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return DSTD_E_CUDA;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return DSTD_OK;
}

}  // namespace

extern "C" {

int dstd_dense_fwd_noalloc(const float *t_in, const float *W, int B, int N_in, int N_out, const dstd_params *p,
                           dstd_math math, float *t_out, void *saved, float *penalty, dstd_stream_t stream) {
    if (!t_in || !W || !t_out || !saved) return DSTD_E_INVALID;
    TRY(check_sizes(B, N_in, N_out));
    TRY(check_params(p));
    const int Mp = padded_M(p->M);
    TRY(check_math(math, Mp));
    if (!aligned16(t_in) || !aligned16(W) || !aligned16(saved)) return DSTD_E_INVALID;
    const OpKind op = op_of(math);
    if (fwd_layout(nullptr, B, N_in, N_out, Mp, op, false).bytes > kNoAllocScratchBytes) return DSTD_E_WORKSPACE;
    TRY(device_ok());
    void *scratch = nullptr;
    TRY(noalloc_scratch(&scratch));
    LifConst c = make_const(*p, Mp);
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs ws = fwd_layout(scratch, B, N_in, N_out, Mp, op, false);
    Saved sv = saved_view(saved, B, N_out);
    if (penalty) TRY(cu(cudaMemsetAsync(penalty, 0, 4 * sizeof(float), st)));
    return dense_forward_core(t_in, W, B, N_in, N_out, c, op, ws, false, &sv, t_out, penalty, st);
}

int dstd_device_status(int clear) {
    if (cudaDeviceSynchronize() != cudaSuccess) return DSTD_E_CUDA;
    unsigned int s = 0, s2 = 0;
    if (status_read(&s, clear) != cudaSuccess) return DSTD_E_CUDA;
    if (conv_status_read(&s2, clear) != cudaSuccess) return DSTD_E_CUDA;
    return ((s | s2) & STATUS_TIMEOUT) ? DSTD_E_TIMEOUT : DSTD_OK;
}

int dstd_conv_set_chunk_images(int max_images) {
    if (max_images < 0) return g_conv_chunk_images;
    const int prev = g_conv_chunk_images;
    g_conv_chunk_images = max_images;
    return prev;
}

int dstd_conv_set_operand_policy(int policy) {
    if (policy < 0 || policy > 2) return g_conv_operand_policy;
    const int prev = g_conv_operand_policy;
    g_conv_operand_policy = policy;
    return prev;
}

}  // extern "C"
