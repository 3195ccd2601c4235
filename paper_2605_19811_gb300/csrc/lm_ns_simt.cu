// fp32 CUDA-core Newton-Schulz phases (the "fp32 mode" of the msign
// approximation; Section 2 names the odd-polynomial iteration).  Per
// iteration, for every matrix X of every group (s x l, or l x s for a tall
// parameter, which iterates on X^T X and X B instead):
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

// Operand tile of 64 (i) x 16 (k) into S[k][i]: K-major (element (i, k) at
// op[i * ld + k]) or MN-major (at op[k * ld + i]).
__device__ __forceinline__ void load_tile(float (*S)[BM + 4], const float* op, int ld, bool mn,
                                          int i0, int k0) {
  if (!mn) {
    const int row = threadIdx.x >> 2, kq = (threadIdx.x & 3) * 4;
    const float4 v = *reinterpret_cast<const float4*>(op + (size_t)(i0 + row) * ld + k0 + kq);
    S[kq + 0][row] = v.x; S[kq + 1][row] = v.y; S[kq + 2][row] = v.z; S[kq + 3][row] = v.w;
  } else {
    const int kk = threadIdx.x >> 4, iq = (threadIdx.x & 15) * 4;
    const float4 v = *reinterpret_cast<const float4*>(op + (size_t)(k0 + kk) * ld + i0 + iq);
    S[kk][iq + 0] = v.x; S[kk][iq + 1] = v.y; S[kk][iq + 2] = v.z; S[kk][iq + 3] = v.w;
  }
}

// Wide groups hold X as s x l, tall groups as l x s:
//   GRAM  wide A = X X^T (rows of X), tall A = X^T X (columns of X)
//   POLY  B = b A + c A A
//   APPLY wide X' = a X + B X, tall X' = a X + X B
__global__ void __launch_bounds__(kThreads)
    ns_simt_kernel(int phase, int iter, const NsGroup* __restrict__ groups,
                   const NsTile* __restrict__ tiles, int ntiles, const double* __restrict__ norm2,
                   NsCoeffs co, const unsigned char* __restrict__ active) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;

  for (int w = blockIdx.x; w < ntiles; w += gridDim.x) {
    const NsTile t = tiles[w];
    const NsGroup g = groups[t.group];
    if (active != nullptr && !active[g.first_mat + t.mat]) continue;   // block-uniform
    const int cur = iter & 1;
    const bool tall = g.tall != 0;
    const int ldx = tall ? g.s_pad : g.l_pad;
    const float* X = static_cast<const float*>(g.X[cur]) + (size_t)t.mat * g.s_pad * g.l_pad;
    const float* Am = static_cast<const float*>(g.A) + (size_t)t.mat * g.s_pad * g.s_pad;
    const float* Bm = static_cast<const float*>(g.B) + (size_t)t.mat * g.s_pad * g.s_pad;
    const float* opA;
    const float* opB;
    int lda, ldb, K;
    bool amn, bmn;
    if (phase == NS_GRAM) {
      opA = X; opB = X; lda = ldb = ldx; K = g.l_pad; amn = bmn = tall;
    } else if (phase == NS_POLY) {
      opA = Am; opB = Am; lda = ldb = g.s_pad; K = g.s_pad; amn = bmn = false;
    } else if (tall) {
      opA = X; opB = Bm; lda = ldx; ldb = g.s_pad; K = g.s_pad; amn = false; bmn = true;
    } else {
      opA = Bm; opB = X; lda = g.s_pad; ldb = ldx; K = g.s_pad; amn = false; bmn = true;
    }
    const int i0 = t.tm * BM, j0 = t.tn * BN;
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

    for (int k0 = 0; k0 < K; k0 += BK) {
      load_tile(As, opA, lda, amn, i0, k0);
      load_tile(Bs, opB, ldb, bmn, j0, k0);
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
    const int nrows = (phase == NS_APPLY && tall) ? g.l : g.s;
    const int ncols = (phase == NS_APPLY) ? (tall ? g.s : g.l) : g.s;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + ty * 4 + a;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int j = j0 + tx * 4 + b;
        const bool valid = i < nrows && j < ncols;
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
          const float v = valid ? (co.a * X[(size_t)i * ldx + j] + acc[a][b]) * nscale : 0.f;
          Xn[(size_t)i * ldx + j] = v;
        }
      }
    }
  }
}

}  // namespace

int simt_pad(int x) { return (x + 63) / 64 * 64; }

cudaError_t launch_ns_simt(NsPhase ph, int iter, int ngroups, const NsGroup* dgroups,
                           const NsTile* tiles, int ntiles, const double* norm2, NsCoeffs co,
                           cudaStream_t st, const unsigned char* active) {
  (void)ngroups;
  if (ntiles <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int grid = sms * 4;
  if (grid > ntiles) grid = ntiles;
  count_launch();
  ns_simt_kernel<<<grid, kThreads, 0, st>>>((int)ph, iter, dgroups, tiles, ntiles, norm2, co, active);
  return cudaGetLastError();
}

}  // namespace lm
