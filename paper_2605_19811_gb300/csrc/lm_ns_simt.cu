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
//
// Block tile 128 x 128, 256 threads, 8 x 8 outputs per thread held as two
// 4 x 4 quadrants 64 apart in each direction (so that a warp's shared-memory
// reads are contiguous), K in slices of 16 double-buffered in shared memory:
// the global loads of slice k+1 are in flight while slice k is multiplied.
#include "lm_internal.h"

namespace lm {
namespace {

constexpr int BM = kSimtBM, BN = kSimtBN, BK = 16;
constexpr int kThreads = 256;
constexpr int kPadS = 4;   // row padding of the shared tiles (floats)

// One 128 (i) x 16 (k) operand slice, two float4 per thread, from a K-major
// (element (i, k) at op[i * ld + k]) or MN-major (at op[k * ld + i]) matrix.
struct SliceRegs {
  float4 v[2];
};
__device__ __forceinline__ void load_slice(SliceRegs& R, const float* op, int ld, bool mn, int i0, int k0) {
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int f = threadIdx.x + u * kThreads;   // float4 index 0 .. 511
    if (!mn) {
      const int i = f >> 2, kq = (f & 3) * 4;
      R.v[u] = *reinterpret_cast<const float4*>(op + (size_t)(i0 + i) * ld + k0 + kq);
    } else {
      const int kk = f >> 5, iq = (f & 31) * 4;
      R.v[u] = *reinterpret_cast<const float4*>(op + (size_t)(k0 + kk) * ld + i0 + iq);
    }
  }
}
__device__ __forceinline__ void store_slice(float (*S)[BM + kPadS], const SliceRegs& R, bool mn) {
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int f = threadIdx.x + u * kThreads;
    if (!mn) {
      const int i = f >> 2, kq = (f & 3) * 4;
      S[kq + 0][i] = R.v[u].x; S[kq + 1][i] = R.v[u].y; S[kq + 2][i] = R.v[u].z; S[kq + 3][i] = R.v[u].w;
    } else {
      const int kk = f >> 5, iq = (f & 31) * 4;
      *reinterpret_cast<float4*>(&S[kk][iq]) = R.v[u];
    }
  }
}

// Wide groups hold X as s x l, tall groups as l x s:
//   GRAM  wide A = X X^T (rows of X), tall A = X^T X (columns of X)
//   POLY  B = b A + c A A
//   APPLY wide X' = a X + B X, tall X' = a X + X B
__global__ void __launch_bounds__(kThreads, 2)   // two blocks per SM: at most 128 registers
    ns_simt_kernel(int phase, int iter, const NsGroup* __restrict__ groups,
                   const NsTile* __restrict__ tiles, int ntiles, const double* __restrict__ norm2,
                   NsCoeffs co, const unsigned char* __restrict__ active, float* __restrict__ split_ws,
                   const unsigned* flags) {
  if (lm_stopped(flags)) return;
  __shared__ __align__(16) float As[2][BK][BM + kPadS];
  __shared__ __align__(16) float Bs[2][BK][BN + kPadS];
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
    // split Gram tiles: K slices [kb0, kb1), the partial tile to its own workspace tile
    const bool split = phase == NS_GRAM && t.slot != 0;
    const int kbeg = split ? (int)t.kb0 * BK : 0;
    const int kend = split ? (int)t.kb1 * BK : K;
    float acc[8][8];
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
      for (int b = 0; b < 8; ++b) acc[a][b] = 0.f;

    SliceRegs ra, rb;
    load_slice(ra, opA, lda, amn, i0, kbeg);
    load_slice(rb, opB, ldb, bmn, j0, kbeg);
    __syncthreads();   // the previous tile's last reads of the buffers are done
    store_slice(As[0], ra, amn);
    store_slice(Bs[0], rb, bmn);
    __syncthreads();
    int buf = 0;
    for (int k0 = kbeg; k0 < kend; k0 += BK) {
      const bool more = k0 + BK < kend;
      if (more) {   // next slice in flight while this one is multiplied
        load_slice(ra, opA, lda, amn, i0, k0 + BK);
        load_slice(rb, opB, ldb, bmn, j0, k0 + BK);
      }
#pragma unroll
      for (int kk = 0; kk < BK; ++kk) {
        const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * 4]);
        const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][kk][64 + ty * 4]);
        const float4 b0 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * 4]);
        const float4 b1 = *reinterpret_cast<const float4*>(&Bs[buf][kk][64 + tx * 4]);
        const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
        for (int a = 0; a < 8; ++a)
#pragma unroll
          for (int b = 0; b < 8; ++b) acc[a][b] = fmaf(av[a], bv[b], acc[a][b]);
      }
      if (more) {
        store_slice(As[buf ^ 1], ra, amn);
        store_slice(Bs[buf ^ 1], rb, bmn);
        __syncthreads();
        buf ^= 1;
      }
    }

    // epilogue: rows i0 + ty*4 + a (+64), columns j0 + tx*4 + b (+64)
    float nscale = 1.f;
    if (iter == 0) {
      const float n = (float)sqrt(norm2[g.first_mat + t.mat]) + co.eps;
      nscale = (phase == NS_GRAM) ? 1.f / (n * n) : (phase == NS_APPLY ? 1.f / n : 1.f);
    }
    const int nrows = (phase == NS_APPLY && tall) ? g.l : g.s;
    const int ncols = (phase == NS_APPLY) ? (tall ? g.s : g.l) : g.s;
#pragma unroll
    for (int a = 0; a < 8; ++a) {
      const int i = i0 + (a >> 2) * 64 + ty * 4 + (a & 3);
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        const int j = j0 + (b >> 2) * 64 + tx * 4 + (b & 3);
        const bool valid = i < nrows && j < ncols;
        if (phase == NS_GRAM) {
          if (j < i && !split) continue;
          const float v = valid ? acc[a][b] * nscale : 0.f;
          float* A = const_cast<float*>(Am);
          if (split) {   // the finish kernel sums the parts and writes A and its mirror
            split_ws[(size_t)(t.slot - 1) * (BM * BN) + (size_t)(i - i0) * BN + (j - j0)] = v;
            continue;
          }
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

int simt_pad(int x) { return (x + BM - 1) / BM * BM; }

cudaError_t launch_ns_simt(NsPhase ph, int iter, int ngroups, const NsGroup* dgroups,
                           const NsTile* tiles, int ntiles, const double* norm2, NsCoeffs co,
                           cudaStream_t st, const unsigned char* active, float* split_ws, const unsigned* flags) {
  (void)ngroups;
  if (ntiles <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int grid = sms * 2;
  if (grid > ntiles) grid = ntiles;
  count_launch();
  ns_simt_kernel<<<grid, kThreads, 0, st>>>((int)ph, iter, dgroups, tiles, ntiles, norm2, co, active,
                                            split_ws, flags);
  return cudaGetLastError();
}

namespace {
// fp32 A from the parts of split Gram tiles, summed in part order; the tile
// and its mirror (a diagonal tile: its upper triangle and the mirror of it).
__global__ void __launch_bounds__(256) ns_split_finish_f32_kernel(const NsSplitTarget* __restrict__ targets,
                                                                  const float* __restrict__ ws,
                                                                  const unsigned* flags) {
  if (lm_stopped(flags)) return;
  const NsSplitTarget T = targets[blockIdx.y];
  float* dst = static_cast<float*>(T.a_tile);
  float* mir = static_cast<float*>(T.a_mirror);
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < BM * BN; e += gridDim.x * blockDim.x) {
    const int r = e / BN, c = e % BN;
    if (r >= T.nr || c >= T.nc || (T.diag && c < r)) continue;
    float sum = 0.f;
    for (int k = 0; k < T.nparts; ++k) sum += ws[(size_t)(T.first + k) * (BM * BN) + e];
    dst[(size_t)r * T.ld + c] = sum;
    mir[(size_t)c * T.ld + r] = sum;
  }
}
}  // namespace

cudaError_t launch_ns_split_finish_f32(const NsSplitTarget* targets, int n, const float* ws, const unsigned* flags,
                                       cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  count_launch();
  ns_split_finish_f32_kernel<<<dim3(16, n), 256, 0, st>>>(targets, ws, flags);
  return cudaGetLastError();
}

}  // namespace lm
