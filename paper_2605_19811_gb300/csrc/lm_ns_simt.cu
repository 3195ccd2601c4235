// fp32 CUDA-core Newton-Schulz phases (the "fp32 mode" of the msign
// approximation; Section 2 names the odd-polynomial iteration).  Per
// iteration, for every matrix X (s x l, wide orientation) of every group:
//   GRAM : A = X X^T          (upper-triangle tiles, mirrored store)
//   POLY : B = b A + c A A    (upper-triangle tiles, mirrored store)
//   APPLY: X' = a X + B X
// Iteration 0 folds the normalisation X / (||G_hat||_F + eps) into GRAM
// (scale 1/(n+eps)^2) and APPLY (scale 1/(n+eps)).  Tensor cores have no
// full-fp32 mode, so this path runs fp32 FMA on the CUDA cores.
#include "lm_internal.h"

namespace lm {
namespace {

constexpr int BM = kSimtBM, BN = kSimtBN, BK = 16;
constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
    ns_simt_kernel(int phase, int iter, const NsGroup* __restrict__ groups,
                   const NsTile* __restrict__ tiles, int ntiles, const double* __restrict__ norm2,
                   NsCoeffs co) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;

  for (int w = blockIdx.x; w < ntiles; w += gridDim.x) {
    const NsTile t = tiles[w];
    const NsGroup g = groups[t.group];
    const int cur = iter & 1;
    const float* X = static_cast<const float*>(g.X[cur]) + (size_t)t.mat * g.s_pad * g.l_pad;
    const float* Am = static_cast<const float*>(g.A) + (size_t)t.mat * g.s_pad * g.s_pad;
    const float* Bm = static_cast<const float*>(g.B) + (size_t)t.mat * g.s_pad * g.s_pad;
    const float* opA;   // row-major, K contiguous
    const float* opB;   // GRAM/POLY: row-major rows j, K contiguous; APPLY: X[k][j]
    int lda, ldb, K;
    if (phase == NS_GRAM) {
      opA = X; opB = X; lda = ldb = g.l_pad; K = g.l_pad;
    } else if (phase == NS_POLY) {
      opA = Am; opB = Am; lda = ldb = g.s_pad; K = g.s_pad;
    } else {
      opA = Bm; opB = X; lda = g.s_pad; ldb = g.l_pad; K = g.s_pad;
    }
    const int i0 = t.tm * BM, j0 = t.tn * BN;
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

    for (int k0 = 0; k0 < K; k0 += BK) {
      {  // A tile: rows i0.., k0..k0+15 -> As[k][i]
        const int row = threadIdx.x >> 2, kq = (threadIdx.x & 3) * 4;
        const float4 v = *reinterpret_cast<const float4*>(opA + (size_t)(i0 + row) * lda + k0 + kq);
        As[kq + 0][row] = v.x; As[kq + 1][row] = v.y; As[kq + 2][row] = v.z; As[kq + 3][row] = v.w;
      }
      if (phase != NS_APPLY) {
        const int row = threadIdx.x >> 2, kq = (threadIdx.x & 3) * 4;
        const float4 v = *reinterpret_cast<const float4*>(opB + (size_t)(j0 + row) * ldb + k0 + kq);
        Bs[kq + 0][row] = v.x; Bs[kq + 1][row] = v.y; Bs[kq + 2][row] = v.z; Bs[kq + 3][row] = v.w;
      } else {
        const int kk = threadIdx.x >> 4, jq = (threadIdx.x & 15) * 4;
        const float4 v = *reinterpret_cast<const float4*>(opB + (size_t)(k0 + kk) * ldb + j0 + jq);
        Bs[kk][jq + 0] = v.x; Bs[kk][jq + 1] = v.y; Bs[kk][jq + 2] = v.z; Bs[kk][jq + 3] = v.w;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < BK; ++kk) {
        float av[4], bv[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) av[a] = As[kk][ty * 4 + a];
#pragma unroll
        for (int b = 0; b < 4; ++b) bv[b] = Bs[kk][tx * 4 + b];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(av[a], bv[b], acc[a][b]);
      }
      __syncthreads();
    }

    // epilogue
    float nscale = 1.f;
    if (iter == 0) {
      const float n = (float)sqrt(norm2[g.first_mat + t.mat]) + co.eps;
      nscale = (phase == NS_GRAM) ? 1.f / (n * n) : (phase == NS_APPLY ? 1.f / n : 1.f);
    }
    const int ncols = (phase == NS_APPLY) ? g.l : g.s;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + ty * 4 + a;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int j = j0 + tx * 4 + b;
        const bool valid = i < g.s && j < ncols;
        if (phase == NS_GRAM) {
          if (j < i) continue;
          const float v = valid ? acc[a][b] * nscale : 0.f;
          float* A = const_cast<float*>(Am);
          A[(size_t)i * g.s_pad + j] = v;
          A[(size_t)j * g.s_pad + i] = v;
        } else if (phase == NS_POLY) {
          if (j < i) continue;
          const float v = valid ? co.b * Am[(size_t)i * g.s_pad + j] + co.c * acc[a][b] : 0.f;
          float* B = const_cast<float*>(Bm);
          B[(size_t)i * g.s_pad + j] = v;
          B[(size_t)j * g.s_pad + i] = v;
        } else {
          float* Xn = static_cast<float*>(g.X[cur ^ 1]) + (size_t)t.mat * g.s_pad * g.l_pad;
          const float v = valid ? (co.a * X[(size_t)i * g.l_pad + j] + acc[a][b]) * nscale : 0.f;
          Xn[(size_t)i * g.l_pad + j] = v;
        }
      }
    }
  }
}

}  // namespace

int simt_pad(int x) { return (x + 63) / 64 * 64; }

cudaError_t launch_ns_simt(NsPhase ph, int iter, int ngroups, const NsGroup* dgroups,
                           const NsTile* tiles, int ntiles, const double* norm2, NsCoeffs co,
                           cudaStream_t st) {
  (void)ngroups;
  if (ntiles <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int grid = sms * 4;
  if (grid > ntiles) grid = ntiles;
  count_launch();
  ns_simt_kernel<<<grid, kThreads, 0, st>>>((int)ph, iter, dgroups, tiles, ntiles, norm2, co);
  return cudaGetLastError();
}

}  // namespace lm
