// Element-wise kernels of the LionMuon step (arXiv 2605.19811, Algorithm 1):
//   * lion_kernel           : Lion branch + momentum update, multi-tensor,
//                             one pass over W, G, M with 16-byte vector I/O.
//   * momentum_norm_kernel  : Muon steps, first part: G_hat, ||G_hat||_F^2
//                             (warp shuffle, one fp64 atomic per warp and
//                             32K-element chunk), M update, X0 = G_hat.
//   * finalize_kernel       : Muon steps, last part: W <- W - eta_M (0.2
//                             sqrt(max(m,n)) X_K + lambda W) (Table 5 scaling),
//                             or the plain msign output.
// All arithmetic is fp32 with each product and sum rounded separately
// (__fmul_rn / __fadd_rn / __fsub_rn): no contraction into FMA, so the Lion
// step is reproducible bit for bit by a same-order float32 evaluation.
#include <cuda_bf16.h>

#include "lm_internal.h"

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
  if (lm_stopped(k.flags)) return;
  // the next kernel on the stream may start its set-up (programmatic launch)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const LionChunk ch = chunks[c];
    const LionTensor t = tensors[ch.tensor];
    if (k.skip != nullptr && k.skip[t.pad]) continue;   // this matrix takes the Muon step
    T* w = static_cast<T*>(t.w) + ch.begin;
    const T* g = static_cast<const T*>(grads[t.grad_slot]) + ch.begin;
    float* m = t.m + ch.begin;
    const int64_t nvec = ch.count >> 3;
    int64_t v = threadIdx.x;
    // four independent vectors per trip keep enough loads in flight to run
    // at the copy bandwidth; then pairs and a single vector for the tail
    for (; v + 3 * kLionThreads < nvec; v += 4 * kLionThreads) {
      float w0[8], g0[8], m0[8], w1[8], g1[8], m1[8], w2[8], g2[8], m2[8], w3[8], g3[8], m3[8];
      const int64_t i0 = v * 8, i1 = i0 + kLionThreads * 8, i2 = i1 + kLionThreads * 8,
                    i3 = i2 + kLionThreads * 8;
      load8(w + i0, w0); load8(g + i0, g0); load8(m + i0, m0);
      load8(w + i1, w1); load8(g + i1, g1); load8(m + i1, m1);
      load8(w + i2, w2); load8(g + i2, g2); load8(m + i2, m2);
      load8(w + i3, w3); load8(g + i3, g3); load8(m + i3, m3);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        lion_elem(w0[e], m0[e], g0[e], k);
        lion_elem(w1[e], m1[e], g1[e], k);
        lion_elem(w2[e], m2[e], g2[e], k);
        lion_elem(w3[e], m3[e], g3[e], k);
      }
      store8(w + i0, w0); store8(m + i0, m0);
      store8(w + i1, w1); store8(m + i1, m1);
      store8(w + i2, w2); store8(m + i2, m2);
      store8(w + i3, w3); store8(m + i3, m3);
    }
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

// Momentum update alone, M <- beta2 M + (1 - beta2) G (the last line of
// Algorithm 1's loop body), for the matrices another rank owns on a layer-
// sharded Muon step: the same float32 operations as lion_elem, so every
// rank's momentum stays equal to the owner's bit for bit.
template <typename T>
__global__ void __launch_bounds__(kLionThreads)
    ema_kernel(const LionTensor* __restrict__ tensors, const LionChunk* __restrict__ chunks, int nchunks,
               const void* const* __restrict__ grads, LionConsts k) {
  if (lm_stopped(k.flags)) return;
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const LionChunk ch = chunks[c];
    const LionTensor t = tensors[ch.tensor];
    const T* g = static_cast<const T*>(grads[t.grad_slot]) + ch.begin;
    float* m = t.m + ch.begin;
    const int64_t nvec = ch.count >> 3;
    for (int64_t v = threadIdx.x; v < nvec; v += kLionThreads) {
      float gv[8], mv[8];
      load8(g + v * 8, gv);
      load8(m + v * 8, mv);
#pragma unroll
      for (int e = 0; e < 8; ++e) mv[e] = __fadd_rn(__fmul_rn(k.b2, mv[e]), __fmul_rn(k.c2, gv[e]));
      store8(m + v * 8, mv);
    }
    for (int64_t e = (nvec << 3) + threadIdx.x; e < ch.count; e += kLionThreads)
      m[e] = __fadd_rn(__fmul_rn(k.b2, m[e]), __fmul_rn(k.c2, to_f(g[e])));
  }
}

// ---------------------------------------------------------------------------
// AdamW for 1-D parameters (Section 3's fallback for biases and norm gains).
// The same fixed operation order as the float32 reference: every product,
// sum, square root and quotient rounded once (IEEE __fsqrt_rn / __fdiv_rn).
// 1-D parameters are a small share of any set (0.02% of the 720M-shaped one),
// so the kernel streams one element per thread per trip.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void adamw_elem(float& w, float& m, float& v, float g, const AdamConsts& k) {
  m = __fadd_rn(__fmul_rn(k.b1, m), __fmul_rn(k.c1, g));
  v = __fadd_rn(__fmul_rn(k.b2, v), __fmul_rn(k.c2, __fmul_rn(g, g)));
  w = __fsub_rn(w, __fmul_rn(k.lrwd, w));
  const float den = __fadd_rn(__fmul_rn(__fsqrt_rn(v), k.rbc2), k.eps);
  w = __fsub_rn(w, __fmul_rn(k.step, __fdiv_rn(m, den)));
}

template <typename T>
__global__ void __launch_bounds__(kLionThreads)
    adamw_kernel(const AdamTensor* __restrict__ tensors, const LionChunk* __restrict__ chunks, int nchunks,
                 const void* const* __restrict__ grads, AdamConsts k) {
  if (lm_stopped(k.flags)) return;
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const LionChunk ch = chunks[c];
    const AdamTensor t = tensors[ch.tensor];
    T* w = static_cast<T*>(t.w) + ch.begin;
    const T* g = static_cast<const T*>(grads[t.grad_slot]) + ch.begin;
    float* m = t.m + ch.begin;
    float* v = t.v + ch.begin;
    for (int64_t e = threadIdx.x; e < ch.count; e += kLionThreads) {
      float wf = to_f(w[e]), mf = m[e], vf = v[e];
      adamw_elem(wf, mf, vf, to_f(g[e]), k);
      w[e] = from_f<T>(wf);
      m[e] = mf;
      v[e] = vf;
    }
  }
}

// ---------------------------------------------------------------------------
// Muon: momentum + Frobenius norm + X0, and finalize.  X keeps the
// parameter's orientation (row pitch ldx), so both kernels stream element
// ranges of a matrix: element e = r * cols + c of W, G, M is element
// r * ldx + c of X.
// ---------------------------------------------------------------------------
constexpr int kElemThreads = 256;

__device__ __forceinline__ int64_t x_index(const MatDesc& d, int64_t e) {
  // matrices in a state have fewer than 2^32 elements per row-block here;
  // 32-bit division when the element index fits
  if (e < 0xFFFFFFFFll && d.cols < 0xFFFFFFFFll) {
    const uint32_t r = (uint32_t)e / (uint32_t)d.cols;
    return (int64_t)r * d.ldx + (e - (int64_t)r * d.cols);
  }
  const int64_t r = e / d.cols;
  return r * d.ldx + (e - r * d.cols);
}

// Muon direction for 8 elements: G_hat = b1 M + c1 G (fp32, same operation
// order as the Lion step), M <- b2 M + c2 G; returns sum G_hat^2.
__device__ __forceinline__ float momentum_math(float (&gv)[8], float (&mv)[8], float (&gh)[8],
                                               const MuonConsts& k, int mode) {
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (mode == 0) {
      gh[j] = __fadd_rn(__fmul_rn(k.b1, mv[j]), __fmul_rn(k.c1, gv[j]));
      mv[j] = __fadd_rn(__fmul_rn(k.b2, mv[j]), __fmul_rn(k.c2, gv[j]));
    } else {
      gh[j] = gv[j];
    }
    acc = fmaf(gh[j], gh[j], acc);
  }
  return acc;
}

// 8-element vectors in flight per thread and trip, and CTAs per SM, as
// measured best on the 720M-shaped set (momentum 3 / 2, finalize 2 / 3)
constexpr int kMomVec = 3, kMomCtas = 2;
constexpr int kFinVec = 2, kFinCtas = 3;

template <typename XT, typename GT>
__device__ float momentum_chunk(const MatDesc& d, int64_t begin, int64_t count, const GT* g,
                                const MuonConsts& k, int mode) {
  float acc = 0.f;
  XT* x = static_cast<XT*>(d.x);
  if ((d.cols & 7) == 0) {
    // rows hold whole vectors; count is a multiple of 8.  kMomVec vectors
    // per trip, all loaded before anything is stored.
    const int64_t nvec = count >> 3;
    int64_t v = threadIdx.x;
    for (; v + (kMomVec - 1) * kElemThreads < nvec; v += kMomVec * kElemThreads) {
      float gv[kMomVec][8], mv[kMomVec][8], hv[kMomVec][8];
#pragma unroll
      for (int u = 0; u < kMomVec; ++u) {
        const int64_t e = begin + (v + u * kElemThreads) * 8;
        load8(g + e, gv[u]);
        if (mode == 0) load8(d.m + e, mv[u]);
      }
#pragma unroll
      for (int u = 0; u < kMomVec; ++u) acc += momentum_math(gv[u], mv[u], hv[u], k, mode);
#pragma unroll
      for (int u = 0; u < kMomVec; ++u) {
        const int64_t e = begin + (v + u * kElemThreads) * 8;
        if (mode == 0) store8(d.m + e, mv[u]);
        store8(x + x_index(d, e), hv[u]);
      }
    }
    for (; v < nvec; v += kElemThreads) {
      const int64_t ea = begin + v * 8;
      float ga[8], ma[8], ha[8];
      load8(g + ea, ga);
      if (mode == 0) load8(d.m + ea, ma);
      acc += momentum_math(ga, ma, ha, k, mode);
      if (mode == 0) store8(d.m + ea, ma);
      store8(x + x_index(d, ea), ha);
    }
  } else {
    for (int64_t e = begin + threadIdx.x; e < begin + count; e += kElemThreads) {
      const float gv = to_f(g[e]);
      float gh = gv;
      if (mode == 0) {
        const float mv = d.m[e];
        gh = __fadd_rn(__fmul_rn(k.b1, mv), __fmul_rn(k.c1, gv));
        d.m[e] = __fadd_rn(__fmul_rn(k.b2, mv), __fmul_rn(k.c2, gv));
      }
      acc = fmaf(gh, gh, acc);
      x[x_index(d, e)] = from_f<XT>(gh);
    }
  }
  return acc;
}

template <typename XT, typename GT, int MODE>
__global__ void __launch_bounds__(kElemThreads, kMomCtas)
    momentum_norm_kernel(const MatDesc* __restrict__ mats, const ElemChunk* __restrict__ chunks,
                         int nchunks, const void* const* __restrict__ grads, MuonConsts k) {
  if (lm_stopped(k.flags)) return;
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const ElemChunk ch = chunks[c];
    if (k.active != nullptr && !k.active[ch.mat]) continue;   // this matrix takes the Lion step
    const MatDesc& d = mats[ch.mat];
    const GT* src = static_cast<const GT*>(MODE == 0 ? grads[d.grad_slot] : d.w);
    float acc = momentum_chunk<XT>(d, ch.begin, ch.count, src, k, MODE);
    // ||G_hat||_F^2: warp shuffle, then one fp64 atomic per warp and chunk
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) atomicAdd(d.norm2, (double)acc);
  }
}

// W <- W - eta_M (s X_K + lambda W), or out = X_K (msign); X_K is scaled by
// 1/(||G_hat|| + eps) when no NS iteration ran.
__device__ __forceinline__ void finalize_math(float (&xv)[8], float (&pv)[8], float shape_scale,
                                              const MuonConsts& k, int mode, float xs, bool scale_x) {
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (scale_x) xv[j] = __fmul_rn(xv[j], xs);
    pv[j] = mode == 0 ? __fsub_rn(pv[j], __fmul_rn(k.eM, __fadd_rn(__fmul_rn(shape_scale, xv[j]),
                                                                   __fmul_rn(k.lam, pv[j]))))
                      : xv[j];
  }
}

template <typename XT, typename PT>
__device__ void finalize_chunk(const MatDesc& d, int64_t begin, int64_t count, const MuonConsts& k,
                               int mode, float xs, bool scale_x) {
  PT* p = static_cast<PT*>(mode == 0 ? d.w : d.out);
  const XT* x = static_cast<const XT*>(d.x_final);
  if ((d.cols & 7) == 0) {
    const int64_t nvec = count >> 3;
    int64_t v = threadIdx.x;
    for (; v + (kFinVec - 1) * kElemThreads < nvec; v += kFinVec * kElemThreads) {
      float xv[kFinVec][8], pv[kFinVec][8];
#pragma unroll
      for (int u = 0; u < kFinVec; ++u) {
        const int64_t e = begin + (v + u * kElemThreads) * 8;
        load8(x + x_index(d, e), xv[u]);
        if (mode == 0) load8(p + e, pv[u]);
      }
#pragma unroll
      for (int u = 0; u < kFinVec; ++u) finalize_math(xv[u], pv[u], d.shape_scale, k, mode, xs, scale_x);
#pragma unroll
      for (int u = 0; u < kFinVec; ++u) store8(p + begin + (v + u * kElemThreads) * 8, pv[u]);
    }
    for (; v < nvec; v += kElemThreads) {
      const int64_t ea = begin + v * 8;
      float xa[8], pa[8];
      load8(x + x_index(d, ea), xa);
      if (mode == 0) load8(p + ea, pa);
      finalize_math(xa, pa, d.shape_scale, k, mode, xs, scale_x);
      store8(p + ea, pa);
    }
  } else {
    for (int64_t e = begin + threadIdx.x; e < begin + count; e += kElemThreads) {
      float xv = to_f(x[x_index(d, e)]);
      if (scale_x) xv = __fmul_rn(xv, xs);
      float pv = mode == 0 ? to_f(p[e]) : 0.f;
      pv = mode == 0 ? __fsub_rn(pv, __fmul_rn(k.eM, __fadd_rn(__fmul_rn(d.shape_scale, xv),
                                                              __fmul_rn(k.lam, pv))))
                     : xv;
      p[e] = from_f<PT>(pv);
    }
  }
}

template <typename XT, typename PT, int MODE>
__global__ void __launch_bounds__(kElemThreads, kFinCtas)
    finalize_kernel(const MatDesc* __restrict__ mats, const ElemChunk* __restrict__ chunks, int nchunks,
                    MuonConsts k, unsigned* flags) {
  // the NS launches before it may be programmatic: wait for their results
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (lm_stopped(flags)) return;
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const ElemChunk ch = chunks[c];
    if (k.active != nullptr && !k.active[ch.mat]) continue;
    const MatDesc& d = mats[ch.mat];
    const float nrm = (float)sqrt(*d.norm2);
    if (threadIdx.x == 0 && ch.begin == 0 && !isfinite(nrm)) atomicOr(flags, LM_FLAG_NONFINITE);
    const bool scale_x = k.ns_steps == 0;
    const float xs = scale_x ? 1.f / __fadd_rn(nrm, k.eps) : 1.f;
    finalize_chunk<XT, PT>(d, ch.begin, ch.count, k, MODE, xs, scale_x);
  }
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

cudaError_t launch_ema(lm_dtype dt, const LionTensor* tensors, const LionChunk* chunks, int nchunks,
                       const void* const* grads, LionConsts k, int grid, cudaStream_t st) {
  if (nchunks <= 0) return cudaSuccess;
  if (grid > nchunks) grid = nchunks;
  count_launch();
  if (dt == LM_BF16)
    ema_kernel<__nv_bfloat16><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  else
    ema_kernel<float><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  return cudaGetLastError();
}

cudaError_t launch_adamw(lm_dtype dt, const AdamTensor* tensors, const LionChunk* chunks, int nchunks,
                         const void* const* grads, AdamConsts k, cudaStream_t st) {
  if (nchunks <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = nchunks < 4 * sms ? nchunks : 4 * sms;
  count_launch();
  if (dt == LM_BF16)
    adamw_kernel<__nv_bfloat16><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  else
    adamw_kernel<float><<<grid, kLionThreads, 0, st>>>(tensors, chunks, nchunks, grads, k);
  return cudaGetLastError();
}

template <typename K>
int elem_grid_size(K kernel) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kElemThreads, 0);
  if (per_sm < 1) per_sm = 1;
  if (sms < 1) sms = 1;
  return sms * per_sm;
}

namespace {
template <typename XT, typename GT>
void mn_launch(int grid, cudaStream_t st, const MatDesc* mats, const ElemChunk* chunks, int nchunks,
               const void* const* grads, MuonConsts k, int mode) {
  if (mode == 0)
    momentum_norm_kernel<XT, GT, 0><<<grid, kElemThreads, 0, st>>>(mats, chunks, nchunks, grads, k);
  else
    momentum_norm_kernel<XT, GT, 1><<<grid, kElemThreads, 0, st>>>(mats, chunks, nchunks, grads, k);
}
template <typename XT, typename PT>
void fin_launch(int grid, cudaStream_t st, const MatDesc* mats, const ElemChunk* chunks, int nchunks,
                MuonConsts k, int mode, unsigned* flags) {
  if (mode == 0)
    finalize_kernel<XT, PT, 0><<<grid, kElemThreads, 0, st>>>(mats, chunks, nchunks, k, flags);
  else
    finalize_kernel<XT, PT, 1><<<grid, kElemThreads, 0, st>>>(mats, chunks, nchunks, k, flags);
}
}  // namespace

cudaError_t launch_momentum_norm(lm_dtype xdt, lm_dtype gdt, const MatDesc* mats, const ElemChunk* chunks,
                                 int nchunks, const void* const* grads, MuonConsts k, int mode,
                                 cudaStream_t st) {
  if (nchunks <= 0) return cudaSuccess;
  static int grid_caps[kMaxDevices] = {};
  const int slot = device_slot();
  int grid_cap = slot >= 0 ? grid_caps[slot] : 0;
  if (grid_cap == 0) grid_cap = elem_grid_size(momentum_norm_kernel<__nv_bfloat16, __nv_bfloat16, 0>);
  if (slot >= 0) grid_caps[slot] = grid_cap;
  const int grid = nchunks < grid_cap ? nchunks : grid_cap;
  count_launch();
  if (xdt == LM_BF16) {
    if (gdt == LM_BF16) mn_launch<__nv_bfloat16, __nv_bfloat16>(grid, st, mats, chunks, nchunks, grads, k, mode);
    else mn_launch<__nv_bfloat16, float>(grid, st, mats, chunks, nchunks, grads, k, mode);
  } else {
    if (gdt == LM_BF16) mn_launch<float, __nv_bfloat16>(grid, st, mats, chunks, nchunks, grads, k, mode);
    else mn_launch<float, float>(grid, st, mats, chunks, nchunks, grads, k, mode);
  }
  return cudaGetLastError();
}

cudaError_t launch_finalize(lm_dtype xdt, lm_dtype pdt, const MatDesc* mats, const ElemChunk* chunks,
                            int nchunks, MuonConsts k, int mode, unsigned* flags, cudaStream_t st) {
  if (nchunks <= 0) return cudaSuccess;
  static int grid_caps[kMaxDevices] = {};
  const int slot = device_slot();
  int grid_cap = slot >= 0 ? grid_caps[slot] : 0;
  if (grid_cap == 0) grid_cap = elem_grid_size(finalize_kernel<__nv_bfloat16, __nv_bfloat16, 0>);
  if (slot >= 0) grid_caps[slot] = grid_cap;
  const int grid = nchunks < grid_cap ? nchunks : grid_cap;
  count_launch();
  if (xdt == LM_BF16) {
    if (pdt == LM_BF16) fin_launch<__nv_bfloat16, __nv_bfloat16>(grid, st, mats, chunks, nchunks, k, mode, flags);
    else fin_launch<__nv_bfloat16, float>(grid, st, mats, chunks, nchunks, k, mode, flags);
  } else {
    if (pdt == LM_BF16) fin_launch<float, __nv_bfloat16>(grid, st, mats, chunks, nchunks, k, mode, flags);
    else fin_launch<float, float>(grid, st, mats, chunks, nchunks, k, mode, flags);
  }
  return cudaGetLastError();
}

cudaError_t launch_upload_ptrs(const void** dst, const PtrUpload& src, int count, cudaStream_t st) {
  if (count <= 0) return cudaSuccess;
  count_launch();
  upload_ptrs_kernel<<<(count + 255) / 256, 256, 0, st>>>(dst, src, count);
  return cudaGetLastError();
}

}  // namespace lm
