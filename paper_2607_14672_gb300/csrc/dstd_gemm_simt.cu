// fp32 CUDA-core GEMM D = A B^T (both operands K-major), the reference-
// precision contraction of the F32 math mode. 64x64 output tile per block,
// 256 threads with a 4x4 register tile each, k-slices of 16 staged in shared
// memory; split-K over gridDim.z writes separate partial outputs.
#include "dstd_internal.cuh"

namespace dstd {

namespace {
constexpr int TM = 64, TN = 64, TK = 16;

__global__ void __launch_bounds__(256) k_sgemm_tn(const float *__restrict__ A, int lda, const float *__restrict__ Bm,
                                                  int ldb, float *D, int ldd, int R, int Cn, int K, int kchunk,
                                                  long long zstride) {
    __shared__ float As[TK][TM + 4];
    __shared__ float Bs[TK][TN + 4];
    const int tid = threadIdx.x;
    const int tx = tid % 16, ty = tid / 16;
    const int r0 = blockIdx.y * TM, c0 = blockIdx.x * TN;
    const int kbeg = blockIdx.z * kchunk;
    const int kend = min(K, kbeg + kchunk);
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
    for (int k0 = kbeg; k0 < kend; k0 += TK) {
#pragma unroll
        for (int e = tid; e < TM * TK; e += 256) {
            int rr = e / TK, kk = e % TK;
            int gr = r0 + rr, gk = k0 + kk;
            As[kk][rr] = (gr < R && gk < kend) ? A[(long long)gr * lda + gk] : 0.f;
            int gc = c0 + rr;
            Bs[kk][rr] = (gc < Cn && gk < kend) ? Bm[(long long)gc * ldb + gk] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < TK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                a[u] = As[kk][ty * 4 + u];
                b[u] = Bs[kk][tx * 4 + u];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
        }
        __syncthreads();
    }
    float *Dz = D + blockIdx.z * zstride;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        int r = r0 + ty * 4 + u;
        if (r >= R) continue;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            int cc = c0 + tx * 4 + v;
            if (cc < Cn) Dz[(long long)r * ldd + cc] = acc[u][v];
        }
    }
}
}  // namespace

cudaError_t launch_sgemm_tn(const float *A, int lda, const float *Bm, int ldb, float *D, int ldd, int R, int Cn,
                            int K, int splits, long long zstride, cudaStream_t st) {
    if (splits < 1) splits = 1;
    int kchunk = (K + splits - 1) / splits;
    kchunk = (kchunk + TK - 1) / TK * TK;
    dim3 grid((Cn + TN - 1) / TN, (R + TM - 1) / TM, splits);
    k_sgemm_tn<<<grid, 256, 0, st>>>(A, lda, Bm, ldb, D, ldd, R, Cn, K, kchunk, zstride);
    return cudaGetLastError();
}

}  // namespace dstd
