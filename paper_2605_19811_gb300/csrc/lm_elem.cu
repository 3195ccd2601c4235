// Element-wise kernels of the LionMuon step (arXiv 2605.19811, Algorithm 1):
//   * lion_kernel           : Lion branch + momentum update, multi-tensor,
//                             one pass over W, G, M with 16-byte vector I/O.
//   * momentum_norm_kernel  : Muon steps, first half: G_hat, ||G_hat||_F^2
//                             (warp shuffle -> CTA -> cluster DSMEM -> one
//                             fp64 atomic per cluster), M update, and
//                             X0 = G_hat in the wide orientation.
//   * finalize_kernel       : Muon steps, last part: W <- W - eta_M (0.2
//                             sqrt(max(m,n)) X_K + lambda W) (Table 5 scaling),
//                             or the plain msign output.
// All arithmetic is fp32 with each product and sum rounded separately
// (__fmul_rn / __fadd_rn / __fsub_rn): no contraction into FMA, so the Lion
// step is reproducible bit for bit by a same-order float32 evaluation.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include "lm_internal.h"

namespace cg = cooperative_groups;

namespace lm {
namespace {

// ---------------------------------------------------------------------------
// 8-element vector I/O (16-byte transactions), streaming cache hints
// ---------------------------------------------------------------------------
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  uint4 u = __ldcs(reinterpret_cast<const uint4*>(p));
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  float4 a = __ldcs(reinterpret_cast<const float4*>(p));
  float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float (&v)[8]) {
  uint4 u;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
  __stcs(reinterpret_cast<uint4*>(p), u);
}
__device__ __forceinline__ void store8(float* p, const float (&v)[8]) {
  __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
  __stcs(reinterpret_cast<float4*>(p) + 1, make_float4(v[4], v[5], v[6], v[7]));
}
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float to_f(float x) { return x; }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }

// sign with sign(+-0) = 0 and sign(NaN) = NaN.
__device__ __forceinline__ float sign_of(float x) {
  return x > 0.f ? 1.f : (x < 0.f ? -1.f : (x == 0.f ? 0.f : x));
}

// One Lion element: direction from the pre-update buffer, sign step with
// decoupled decay, then the momentum EMA (Algorithm 1, Lion branch).
__device__ __forceinline__ void lion_elem(float& w, float& m, float g, const LionConsts& k) {
  const float gh = __fadd_rn(__fmul_rn(k.b1, m), __fmul_rn(k.c1, g));
  const float u = sign_of(gh);
  w = __fsub_rn(w, __fmul_rn(k.eL, __fadd_rn(u, __fmul_rn(k.lam, w))));
  m = __fadd_rn(__fmul_rn(k.b2, m), __fmul_rn(k.c2, g));
}

template <typename T>
__device__ __forceinline__ void lion_vec(T* w, const T* g, float* m, const LionConsts& k) {
  float wv[8], gv[8], mv[8];
  load8(w, wv);
  load8(g, gv);
  load8(m, mv);
#pragma unroll
  for (int e = 0; e < 8; ++e) lion_elem(wv[e], mv[e], gv[e], k);
  store8(w, wv);
  store8(m, mv);
}

constexpr int kLionThreads = 256;

template <typename T>
__global__ void __launch_bounds__(kLionThreads)
    lion_kernel(const LionTensor* __restrict__ tensors, const LionChunk* __restrict__ chunks,
                int nchunks, const void* const* __restrict__ grads, LionConsts k) {
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const LionChunk ch = chunks[c];
    const LionTensor t = tensors[ch.tensor];
    T* w = static_cast<T*>(t.w) + ch.begin;
    const T* g = static_cast<const T*>(grads[t.grad_slot]) + ch.begin;
    float* m = t.m + ch.begin;
    const int64_t nvec = ch.count >> 3;
    int64_t v = threadIdx.x;
    // two independent vectors per trip keep more loads in flight
    for (; v + kLionThreads < nvec; v += 2 * kLionThreads) {
      float wa[8], ga[8], ma[8], wb[8], gb[8], mb[8];
      const int64_t ia = v * 8, ib = (v + kLionThreads) * 8;
      load8(w + ia, wa); load8(g + ia, ga); load8(m + ia, ma);
      load8(w + ib, wb); load8(g + ib, gb); load8(m + ib, mb);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        lion_elem(wa[e], ma[e], ga[e], k);
        lion_elem(wb[e], mb[e], gb[e], k);
      }
      store8(w + ia, wa); store8(m + ia, ma);
      store8(w + ib, wb); store8(m + ib, mb);
    }
    if (v < nvec) lion_vec(w + v * 8, g + v * 8, m + v * 8, k);
    for (int64_t e = (nvec << 3) + threadIdx.x; e < ch.count; e += kLionThreads) {
      float wf = to_f(w[e]), mf = m[e];
      lion_elem(wf, mf, to_f(g[e]), k);
      w[e] = from_f<T>(wf);
      m[e] = mf;
    }
  }
}

// ---------------------------------------------------------------------------
// Muon: momentum + Frobenius norm + X0
// ---------------------------------------------------------------------------
constexpr int kElemThreads = 256;
constexpr int kSmPitch = kElemTileR + 1;   // transposing tile [kElemTileC][kElemTileR + 1]
static_assert(kElemTileR * kElemTileC == 32 * kElemThreads, "4 vectors of 8 per thread");

template <typename XT, typename GT>
__device__ float momentum_norm_tile(const MatDesc& d, int tile, const GT* g, const MuonConsts& k,
                                    int mode, float* sm) {
  const int tr = tile / d.tiles_c, tcol = tile - tr * d.tiles_c;
  const int64_t r0 = (int64_t)tr * kElemTileR, c0 = (int64_t)tcol * kElemTileC;
  XT* x = static_cast<XT*>(d.x);
  const bool vec = (d.cols & 7) == 0;
  float acc = 0.f;
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int slot = threadIdx.x + it * kElemThreads;
    const int rr = slot >> 4, vv = slot & 15;
    const int64_t r = r0 + rr, c = c0 + vv * 8;
    if (r >= d.rows || c >= d.cols) continue;
    const int cnt = (int)min((int64_t)8, d.cols - c);
    const int64_t off = r * d.cols + c;
    float gv[8], mv[8], gh[8];
    if (vec) {
      load8(g + off, gv);
      if (mode == 0) load8(d.m + off, mv);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        gv[e] = e < cnt ? to_f(g[off + e]) : 0.f;
        mv[e] = (e < cnt && mode == 0) ? d.m[off + e] : 0.f;
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      if (mode == 0) {
        gh[e] = __fadd_rn(__fmul_rn(k.b1, mv[e]), __fmul_rn(k.c1, gv[e]));
        mv[e] = __fadd_rn(__fmul_rn(k.b2, mv[e]), __fmul_rn(k.c2, gv[e]));
      } else {
        gh[e] = gv[e];
      }
      if (e < cnt) acc = fmaf(gh[e], gh[e], acc);
    }
    if (mode == 0) {
      if (vec) {
        store8(d.m + off, mv);
      } else {
        for (int e = 0; e < cnt; ++e) d.m[off + e] = mv[e];
      }
    }
    if (!d.transposed) {
      XT* xp = x + r * d.ldx + c;
      if (vec) {
        store8(xp, gh);
      } else {
        for (int e = 0; e < cnt; ++e) xp[e] = from_f<XT>(gh[e]);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) sm[(vv * 8 + e) * kSmPitch + rr] = gh[e];
    }
  }
  if (d.transposed) {
    __syncthreads();
    // X0[c][r] = G_hat[r][c]: consecutive threads write consecutive r.
    for (int it = 0; it < (kElemTileR * kElemTileC) / kElemThreads; ++it) {
      const int slot = threadIdx.x + it * kElemThreads;
      const int cc = slot / kElemTileR, rr = slot % kElemTileR;
      const int64_t r = r0 + rr, c = c0 + cc;
      if (r < d.rows && c < d.cols) x[c * d.ldx + r] = from_f<XT>(sm[cc * kSmPitch + rr]);
    }
  }
  return acc;
}

template <typename XT>
__global__ void __cluster_dims__(kNormCluster, 1, 1) __launch_bounds__(kElemThreads)
    momentum_norm_kernel(const MatDesc* __restrict__ mats, const ElemTile* __restrict__ tiles,
                         const void* const* __restrict__ grads, MuonConsts k, int mode) {
  __shared__ float sm[kElemTileC * kSmPitch];
  __shared__ float red[kElemThreads / 32];
  __shared__ float cta_sum;
  const ElemTile et = tiles[blockIdx.x];
  float acc = 0.f;
  if (et.tile >= 0) {
    const MatDesc& d = mats[et.mat];
    const void* src = mode == 0 ? grads[d.grad_slot] : d.w;
    if (d.wdt == LM_BF16)
      acc = momentum_norm_tile<XT>(d, et.tile, static_cast<const __nv_bfloat16*>(src), k, mode, sm);
    else
      acc = momentum_norm_tile<XT>(d, et.tile, static_cast<const float*>(src), k, mode, sm);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kElemThreads / 32; ++i) s += red[i];
    cta_sum = s;
  }
  // Every CTA of a cluster works on the same matrix: reduce the cluster's
  // partial sums through distributed shared memory, one atomic per cluster.
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();
  if (cluster.block_rank() == 0 && threadIdx.x == 0) {
    double s = 0.0;
    for (unsigned r = 0; r < cluster.num_blocks(); ++r) s += (double)*cluster.map_shared_rank(&cta_sum, r);
    atomicAdd(mats[et.mat].norm2, s);
  }
  cluster.sync();
}

// ---------------------------------------------------------------------------
// Muon: finalize (parameter write) / msign output
// ---------------------------------------------------------------------------
template <typename XT, typename PT>
__device__ void finalize_tile(const MatDesc& d, int tile, const MuonConsts& k, int mode, float xs,
                              bool scale_x, float* sm) {
  const int tr = tile / d.tiles_c, tcol = tile - tr * d.tiles_c;
  const int64_t r0 = (int64_t)tr * kElemTileR, c0 = (int64_t)tcol * kElemTileC;
  const XT* x = static_cast<const XT*>(d.x_final);
  if (d.transposed) {
    // stage X_K[c][r] (r contiguous in memory) into sm[cc][rr]
    for (int it = 0; it < (kElemTileR * kElemTileC) / kElemThreads; ++it) {
      const int slot = threadIdx.x + it * kElemThreads;
      const int cc = slot / kElemTileR, rr = slot % kElemTileR;
      const int64_t r = r0 + rr, c = c0 + cc;
      sm[cc * kSmPitch + rr] = (r < d.rows && c < d.cols) ? to_f(x[c * d.ldx + r]) : 0.f;
    }
    __syncthreads();
  }
  PT* p = static_cast<PT*>(mode == 0 ? d.w : d.out);
  const bool vec = (d.cols & 7) == 0;
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int slot = threadIdx.x + it * kElemThreads;
    const int rr = slot >> 4, vv = slot & 15;
    const int64_t r = r0 + rr, c = c0 + vv * 8;
    if (r >= d.rows || c >= d.cols) continue;
    const int cnt = (int)min((int64_t)8, d.cols - c);
    const int64_t off = r * d.cols + c;
    float xv[8];
    if (d.transposed) {
#pragma unroll
      for (int e = 0; e < 8; ++e) xv[e] = sm[(vv * 8 + e) * kSmPitch + rr];
    } else if (vec) {
      load8(x + r * d.ldx + c, xv);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) xv[e] = e < cnt ? to_f(x[r * d.ldx + c + e]) : 0.f;
    }
    if (scale_x) {
#pragma unroll
      for (int e = 0; e < 8; ++e) xv[e] = __fmul_rn(xv[e], xs);
    }
    float pv[8];
    if (mode == 0) {
      if (vec) {
        load8(p + off, pv);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) pv[e] = e < cnt ? to_f(p[off + e]) : 0.f;
      }
#pragma unroll
      for (int e = 0; e < 8; ++e)
        pv[e] = __fsub_rn(pv[e], __fmul_rn(k.eM, __fadd_rn(__fmul_rn(d.shape_scale, xv[e]),
                                                           __fmul_rn(k.lam, pv[e]))));
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) pv[e] = xv[e];
    }
    if (vec) {
      store8(p + off, pv);
    } else {
      for (int e = 0; e < cnt; ++e) p[off + e] = from_f<PT>(pv[e]);
    }
  }
}

template <typename XT>
__global__ void __launch_bounds__(kElemThreads)
    finalize_kernel(const MatDesc* __restrict__ mats, const ElemTile* __restrict__ tiles,
                    MuonConsts k, int mode, unsigned* flags) {
  __shared__ float sm[kElemTileC * kSmPitch];
  const ElemTile et = tiles[blockIdx.x];
  if (et.tile < 0) return;
  const MatDesc& d = mats[et.mat];
  const double n2 = *d.norm2;
  const float nrm = (float)sqrt(n2);
  if (threadIdx.x == 0 && et.tile == 0 && !isfinite(nrm)) atomicOr(flags, LM_FLAG_NONFINITE);
  const bool scale_x = k.ns_steps == 0;
  const float xs = scale_x ? 1.f / __fadd_rn(nrm, k.eps) : 1.f;
  const int pdt = mode == 0 ? d.wdt : d.odt;
  if (pdt == LM_BF16)
    finalize_tile<XT, __nv_bfloat16>(d, et.tile, k, mode, xs, scale_x, sm);
  else
    finalize_tile<XT, float>(d, et.tile, k, mode, xs, scale_x, sm);
}

__global__ void upload_ptrs_kernel(const void** dst, const __grid_constant__ PtrUpload src,
                                   int count) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < count) dst[i] = src.p[i];
}

}  // namespace

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
int lion_grid_size(lm_dtype dt) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (dt == LM_BF16)
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lion_kernel<__nv_bfloat16>, kLionThreads, 0);
  else
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lion_kernel<float>, kLionThreads, 0);
  if (per_sm < 1) per_sm = 1;
  if (sms < 1) sms = 1;
  return sms * per_sm;
}

cudaError_t launch_lion(lm_dtype dt, const LionTensor* tensors, const LionChunk* chunks,
                        int nchunks, const void* const* grads, LionConsts k, int grid,
                        cudaStream_t st) {
  if (nchunks <= 0) return cudaSuccess;
  if (grid > nchunks) grid = nchunks;
  count_launch();
  if (dt == LM_BF16)
    lion_kernel<__nv_bfloat16><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  else
    lion_kernel<float><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  return cudaGetLastError();
}

cudaError_t launch_momentum_norm(lm_dtype xdt, const MatDesc* mats, const ElemTile* tiles,
                                 int ntiles, const void* const* grads, MuonConsts k, int mode,
                                 cudaStream_t st) {
  if (ntiles <= 0) return cudaSuccess;
  if (ntiles % kNormCluster != 0) return cudaErrorInvalidValue;
  count_launch();
  if (xdt == LM_BF16)
    momentum_norm_kernel<__nv_bfloat16><<<ntiles, kElemThreads, 0, st>>>(mats, tiles, grads, k, mode);
  else
    momentum_norm_kernel<float><<<ntiles, kElemThreads, 0, st>>>(mats, tiles, grads, k, mode);
  return cudaGetLastError();
}

cudaError_t launch_finalize(lm_dtype xdt, const MatDesc* mats, const ElemTile* tiles, int ntiles,
                            MuonConsts k, int mode, unsigned* flags, cudaStream_t st) {
  if (ntiles <= 0) return cudaSuccess;
  count_launch();
  if (xdt == LM_BF16)
    finalize_kernel<__nv_bfloat16><<<ntiles, kElemThreads, 0, st>>>(mats, tiles, k, mode, flags);
  else
    finalize_kernel<float><<<ntiles, kElemThreads, 0, st>>>(mats, tiles, k, mode, flags);
  return cudaGetLastError();
}

cudaError_t launch_upload_ptrs(const void** dst, const PtrUpload& src, int count, cudaStream_t st) {
  if (count <= 0) return cudaSuccess;
  count_launch();
  upload_ptrs_kernel<<<(count + 255) / 256, 256, 0, st>>>(dst, src, count);
  return cudaGetLastError();
}

}  // namespace lm
