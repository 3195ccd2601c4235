// Stable-rank selection between the Muon and Lion steps (Appendix G): for
// every matrix, the stable rank of its momentum buffer, ||M||_F^2 /
// sigma_1_hat^2, with sigma_1_hat from a few power-iteration passes; the
// matrix takes the Muon step iff that is at most alpha * min(m, n).
//
// One pass is one read of M from HBM (4 B per element): a block owns a run
// of rows and all columns.  Thread t holds columns j * 4 * TPB + 4 t + e of
// the normalised input vector v in registers; for a batch of RB rows it
// loads the row segments once, forms the partial dot products, reduces them
// across the block (warp shuffles, then one shared-memory exchange), and
// from the same registers accumulates u_r * M[r, :] into its share of
// M^T u.  At the end of the run each thread adds its columns into the
// pass's output vector (one atomic per column and run).  ||u||^2 and, in the
// first pass, ||M||_F^2 go to per-matrix fp64 accumulators.
//
// Matrices whose rows are 16-byte multiples (columns divisible by 4) go
// through the ring kernel instead: a producer warp streams whole rows into a
// shared-memory ring with 1-D bulk copies (cp.async.bulk, completion on an
// mbarrier per stage), and eight or ten consumer warps read their columns of
// each staged row twice from shared memory (dot product, then the M^T u
// update).
// Loads are thus decoupled from the per-batch reductions, and a batch can
// hold many rows without using registers.  Every mbarrier wait is bounded;
// a wait that gives up sets LM_FLAG_TIMEOUT and the block stops.
#include <algorithm>

#include "lm_internal.h"

namespace lm {
namespace {

// ------------------------------- PTX wrappers -------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void bar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}
__device__ __forceinline__ void bar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ void bar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool bar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with this parity; false if limit_ns passed or *stop is set.
__device__ __noinline__ bool bar_wait_bounded(uint64_t* bar, uint32_t parity, volatile int* stop,
                                              uint64_t limit_ns) {
  const uint64_t t0 = gtimer();
  for (uint32_t i = 1;; ++i) {
    if (bar_try_wait(bar, parity)) return true;
    if ((i & 127u) == 0) {
      if (*stop) return false;
      if (gtimer() - t0 > limit_ns) return false;
    }
  }
}
__device__ __forceinline__ bool bar_wait(uint64_t* bar, uint32_t parity, volatile int* stop, uint64_t limit_ns) {
  if (bar_try_wait(bar, parity)) return true;
  return bar_wait_bounded(bar, parity, stop, limit_ns);
}
// 1-D bulk copy global -> shared, completion counted on bar (bytes: multiple
// of 16, both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}
// barrier over the NC consumer warps only (the producer warp stays out)
template <int NC>
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(32 * NC) : "memory"); }

template <int TPB>
__device__ __forceinline__ double block_sum(double x, double* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[warp] = x;
  __syncthreads();
  double s = 0.0;
#pragma unroll
  for (int w = 0; w < TPB / 32; ++w) s += red[w];   // same order in every thread
  __syncthreads();
  return s;
}

// Sum of squares of this thread's entries of v, returned in fp64 but formed
// in fp32 (this GPU's fp64 rate is a small fraction of its fp32 rate): the
// entries are first scaled by the power of two that brings the largest to
// [1, 2), so no square overflows or underflows.  Zero, infinite or NaN
// entries take the plain fp64 sum.
template <int S>
__device__ __forceinline__ double sumsq_scaled(const float (&v)[S][4]) {
  float mx = 0.f;
#pragma unroll
  for (int j = 0; j < S; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) mx = fmaxf(mx, fabsf(v[j][e]));
  bool plain = !(mx > 0.f) || !isfinite(mx);
#pragma unroll
  for (int j = 0; j < S; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) plain = plain || isnan(v[j][e]);
  if (plain) {
    double s = 0.0;
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) s += (double)v[j][e] * v[j][e];
    return s;
  }
  const int ex = ilogbf(mx);
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < S; ++j)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float x = scalbnf(v[j][e], -ex);
      s = fmaf(x, x, s);
    }
  return ldexp((double)s, 2 * ex);
}

// Rows [r0, r0 + RB) of the item (zeros past nrows), this thread's columns.
template <int S, int TPB, int RB, bool VEC>
__device__ __forceinline__ void load_rows(float (&m)[RB][S][4], const float* M, int64_t cols, int row0, int r0,
                                          int nrows, int tid) {
#pragma unroll
  for (int b = 0; b < RB; ++b) {
    const bool rv = r0 + b < nrows;
    const float* row = M + (int64_t)(row0 + r0 + b) * cols;
#pragma unroll
    for (int j = 0; j < S; ++j) {
      const int64_t c0 = (int64_t)j * 4 * TPB + 4 * tid;
      if (VEC && rv && c0 + 3 < cols) {
        const float4 q = __ldcs(reinterpret_cast<const float4*>(row + c0));
        m[b][j][0] = q.x; m[b][j][1] = q.y; m[b][j][2] = q.z; m[b][j][3] = q.w;
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) m[b][j][e] = (rv && c0 + e < cols) ? row[c0 + e] : 0.f;
      }
    }
  }
}

// One batch: u_r = M_r . v for the RB rows (block reduction through red[buf]),
// ||u||^2, ||M||_F^2 (pass 0), and w += u_r M_r (unless last).
template <int S, int TPB, int RB>
__device__ __forceinline__ void row_batch(const float (&m)[RB][S][4], const float (&v)[S][4], float (&w)[S][4],
                                          float (*red)[RB][TPB / 32], int& buf, int r0, int nrows, int pass,
                                          int last, double& f2, double& u2) {
  constexpr int NW = TPB / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float sq = 0.f;   // this batch's squares: one fp64 addition per batch
#pragma unroll
  for (int b = 0; b < RB; ++b) {
    float ps = 0.f;
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        ps = fmaf(m[b][j][e], v[j][e], ps);
        sq = fmaf(m[b][j][e], m[b][j][e], sq);
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
    if (lane == 0) red[buf][b][warp] = ps;
  }
  if (pass == 0) f2 += (double)sq;
  __syncthreads();
  float u[RB];
#pragma unroll
  for (int b = 0; b < RB; ++b) {
    float x = 0.f;
#pragma unroll
    for (int q = 0; q < NW; ++q) x += red[buf][b][q];
    u[b] = x;
  }
  buf ^= 1;   // the next batch writes the other buffer: no second barrier
  if (threadIdx.x == 0) {
    float us = 0.f;
#pragma unroll
    for (int b = 0; b < RB; ++b)
      if (r0 + b < nrows) us = fmaf(u[b], u[b], us);
    u2 += (double)us;
  }
  if (!last)
#pragma unroll
    for (int b = 0; b < RB; ++b)
#pragma unroll
      for (int j = 0; j < S; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) w[j][e] = fmaf(u[b], m[b][j][e], w[j][e]);
}

template <int S, int TPB, int RB, bool VEC>
__global__ void __launch_bounds__(TPB)
    srank_pass_kernel(const SrMat* __restrict__ mats, const SrItem* __restrict__ items, int nitems, int pass,
                      int last, const unsigned* flags) {
  if (lm_stopped(flags)) return;
  constexpr int NW = TPB / 32;
  __shared__ float red[2][RB][NW];
  __shared__ double dred[NW];
  const int tid = threadIdx.x;
  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const SrItem I = items[it];
    const SrMat d = mats[I.m];
    const float* vin = pass == 0 ? d.v0 : ((pass & 1) ? d.wa : d.wb);
    float* wout = (pass & 1) ? d.wb : d.wa;
    const int64_t cols = d.cols;

    // normalised input vector, this thread's columns
    float v[S][4];
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int64_t c = (int64_t)j * 4 * TPB + 4 * tid + e;
        v[j][e] = c < cols ? vin[c] : 0.f;
      }
    const double ss = block_sum<TPB>(sumsq_scaled<S>(v), dred);
    const float inv = ss > 0.0 ? (float)(1.0 / sqrt(ss)) : 0.f;
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) v[j][e] *= inv;

    float w[S][4];
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) w[j][e] = 0.f;
    double f2 = 0.0, u2 = 0.0;
    int buf = 0;
    // Two register sets of RB rows: the loads of one batch are in flight
    // while the other is reduced and accumulated.
    float mA[RB][S][4], mB[RB][S][4];
    load_rows<S, TPB, RB, VEC>(mA, d.M, cols, I.row0, 0, I.nrows, tid);
    for (int r0 = 0; r0 < I.nrows; r0 += 2 * RB) {
      load_rows<S, TPB, RB, VEC>(mB, d.M, cols, I.row0, r0 + RB, I.nrows, tid);
      row_batch<S, TPB, RB>(mA, v, w, red, buf, r0, I.nrows, pass, last, f2, u2);
      if (r0 + RB >= I.nrows) break;
      load_rows<S, TPB, RB, VEC>(mA, d.M, cols, I.row0, r0 + 2 * RB, I.nrows, tid);
      row_batch<S, TPB, RB>(mB, v, w, red, buf, r0 + RB, I.nrows, pass, last, f2, u2);
    }
    if (!last)
#pragma unroll
      for (int j = 0; j < S; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int64_t c = (int64_t)j * 4 * TPB + 4 * tid + e;
          if (c < cols) atomicAdd(&wout[c], w[j][e]);
        }
    if (pass == 0) {
      f2 = block_sum<TPB>(f2, dred);
      if (tid == 0) atomicAdd(&d.acc[0], f2);
    }
    if (tid == 0) atomicAdd(&d.acc[1 + pass], u2);
    __syncthreads();   // red / dred are reused by the next item
  }
}

constexpr int kRingMaxStages = 4;
constexpr size_t kRingBudget = 104 * 1024;      // ring bytes per block: two blocks per SM

template <int NC>
__device__ __forceinline__ double consumer_sum(double x, double* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = x;
  consumers_sync<NC>();
  double s = 0.0;
#pragma unroll
  for (int w = 0; w < NC; ++w) s += red[w];
  consumers_sync<NC>();
  return s;
}

// One pass over the items of this launch (all matrices have cols % 4 == 0 and
// at most 128 * NC * S columns: consumer thread t holds columns
// 128 NC j + 4 t .. + 3, j < S; NC = 10 splits 1280 columns evenly).  The ring holds nst stages of RB rows, each row at
// a pitch of `stride` floats; RB is a compile-time constant so that the RB
// rows' dot products, shuffles and updates interleave.
template <int S, int RB, int NC>
__global__ void __launch_bounds__(32 * (NC + 1), (S <= 8 ? 2 : 1))
    srank_ring_kernel(const SrMat* __restrict__ mats, const SrItem* __restrict__ items, int nitems, int pass,
                      int last, int nst, int stride, unsigned* flags, uint64_t wait_ns) {
  extern __shared__ __align__(128) unsigned char ring_raw[];
  float* ring = reinterpret_cast<float*>(ring_raw);
  __shared__ uint64_t full[kRingMaxStages], empty[kRingMaxStages];
  __shared__ float red[2][RB][NC];
  __shared__ double dred[NC];
  __shared__ int stop;
  if (lm_stopped(flags)) return;   // block-uniform: before any barrier
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int k = 0; k < nst; ++k) {
      bar_init(&full[k], 1);
      bar_init(&empty[k], NC);
    }
    stop = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  volatile int* vstop = &stop;

  if (warp == NC) {
    // ------------------------------ producer ------------------------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int armed[kRingMaxStages];
      for (int k = 0; k < kRingMaxStages; ++k) armed[k] = -1;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < nitems; it += gridDim.x) {
        const SrItem I = items[it];
        const SrMat& d = mats[I.m];
        for (int r0 = 0; r0 < I.nrows; r0 += RB) {
          if (!bar_wait(&empty[stage], ph ^ 1u, vstop, wait_ns)) {
            ok = false;
            break;
          }
          const int n = min(RB, I.nrows - r0);
          const uint32_t row_bytes = (uint32_t)(d.cols * 4);
          bar_expect_tx(&full[stage], row_bytes * (uint32_t)n);
          armed[stage] = (int)ph;
          float* dst = ring + (size_t)stage * RB * stride;
          for (int b = 0; b < n; ++b)
            bulk_g2s(dst + (size_t)b * stride, d.M + (int64_t)(I.row0 + r0 + b) * d.cols, row_bytes, &full[stage]);
          if (++stage == nst) {
            stage = 0;
            ph ^= 1u;
          }
        }
      }
      if (!ok) {
        *vstop = 1;
        atomicOr(flags, LM_FLAG_TIMEOUT);
        // copies already issued land before the block exits
        volatile int never = 0;
        for (int k = 0; k < nst; ++k)
          if (armed[k] >= 0) bar_wait(&full[k], (uint32_t)armed[k], &never, 100000000ull);
      }
    }
    return;
  }

  // ------------------------------ consumers -------------------------------
  int stage = 0, buf = 0;
  uint32_t ph = 0;
  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const SrItem I = items[it];
    const SrMat d = mats[I.m];
    const float* vin = pass == 0 ? d.v0 : ((pass & 1) ? d.wa : d.wb);
    float* wout = (pass & 1) ? d.wb : d.wa;
    const int cols = (int)d.cols;
    float v[S][4], w[S][4];
#pragma unroll
    for (int j = 0; j < S; ++j) {
      const int c0 = j * 128 * NC + 4 * tid;
      if (c0 < cols) {
        const float4 q = *reinterpret_cast<const float4*>(vin + c0);
        v[j][0] = q.x; v[j][1] = q.y; v[j][2] = q.z; v[j][3] = q.w;
      } else {
        v[j][0] = v[j][1] = v[j][2] = v[j][3] = 0.f;
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) w[j][e] = 0.f;
    }
    const double ss = consumer_sum<NC>(sumsq_scaled<S>(v), dred);
    const float inv = ss > 0.0 ? (float)(1.0 / sqrt(ss)) : 0.f;
#pragma unroll
    for (int j = 0; j < S; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) v[j][e] *= inv;
    float f2 = 0.f;
    double u2 = 0.0;
    bool aborted = false;
    for (int r0 = 0; r0 < I.nrows; r0 += RB) {
      const int n = min(RB, I.nrows - r0);
      bool ok = true;
      if (lane == 0) ok = bar_wait(&full[stage], ph, vstop, wait_ns);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok && lane == 0) {
        *vstop = 1;
        atomicOr(flags, LM_FLAG_TIMEOUT);
      }
      const float* st = ring + (size_t)stage * RB * stride;
      float ps[RB];
#pragma unroll
      for (int b = 0; b < RB; ++b) {
        ps[b] = 0.f;
        if (b < n) {
#pragma unroll
          for (int j = 0; j < S; ++j) {
            const int c0 = j * 128 * NC + 4 * tid;
            if (c0 < cols) {
              const float4 q = *reinterpret_cast<const float4*>(st + (size_t)b * stride + c0);
              ps[b] = fmaf(q.x, v[j][0], ps[b]); ps[b] = fmaf(q.y, v[j][1], ps[b]);
              ps[b] = fmaf(q.z, v[j][2], ps[b]); ps[b] = fmaf(q.w, v[j][3], ps[b]);
              if (pass == 0) f2 += q.x * q.x + q.y * q.y + q.z * q.z + q.w * q.w;
            }
          }
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int b = 0; b < RB; ++b) ps[b] += __shfl_xor_sync(0xffffffffu, ps[b], o);
      if (lane == 0)
#pragma unroll
        for (int b = 0; b < RB; ++b) red[buf][b][warp] = ps[b];
      consumers_sync<NC>();
      if (*vstop) {        // every consumer reads the same value after the barrier
        aborted = true;
        break;
      }
      float u[RB];
#pragma unroll
      for (int b = 0; b < RB; ++b) {
        u[b] = 0.f;
#pragma unroll
        for (int q = 0; q < NC; ++q) u[b] += red[buf][b][q];
        if (b >= n) u[b] = 0.f;
      }
      if (tid == 0) {   // one fp64 addition per stage (this GPU's fp64 rate is a
                        // small fraction of its fp32 rate); u_b^2 is of the order
                        // of the squares in ||M||_F^2, which are summed in fp32
        float us = 0.f;
#pragma unroll
        for (int b = 0; b < RB; ++b) us = fmaf(u[b], u[b], us);
        u2 += (double)us;
      }
      if (!last) {
#pragma unroll
        for (int b = 0; b < RB; ++b) {
          if (b < n) {
#pragma unroll
            for (int j = 0; j < S; ++j) {
              const int c0 = j * 128 * NC + 4 * tid;
              if (c0 < cols) {
                const float4 q = *reinterpret_cast<const float4*>(st + (size_t)b * stride + c0);
                w[j][0] = fmaf(u[b], q.x, w[j][0]); w[j][1] = fmaf(u[b], q.y, w[j][1]);
                w[j][2] = fmaf(u[b], q.z, w[j][2]); w[j][3] = fmaf(u[b], q.w, w[j][3]);
              }
            }
          }
        }
      }
      buf ^= 1;   // the next batch writes the other buffer of red
      __syncwarp();
      if (lane == 0) bar_arrive(&empty[stage]);
      if (++stage == nst) {
        stage = 0;
        ph ^= 1u;
      }
    }
    if (aborted) break;
    if (!last)
#pragma unroll
      for (int j = 0; j < S; ++j) {
        const int c0 = j * 128 * NC + 4 * tid;
        if (c0 < cols)
#pragma unroll
          for (int e = 0; e < 4; ++e) atomicAdd(&wout[c0 + e], w[j][e]);
      }
    if (pass == 0) {
      const double f2s = consumer_sum<NC>((double)f2, dred);
      if (tid == 0) atomicAdd(&d.acc[0], f2s);
    }
    if (tid == 0) atomicAdd(&d.acc[1 + pass], u2);
  }
}

__global__ void srank_decide_kernel(const SrMat* __restrict__ mats, int nmat, double alpha, int last_pass,
                                    unsigned char* active, unsigned char* skip, double* srank,
                                    const unsigned* flags) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nmat || lm_stopped(flags)) return;
  const SrMat d = mats[i];
  const double f2 = d.acc[0], s2 = d.acc[1 + last_pass];
  const double smin = (double)(d.rows < d.cols ? d.rows : d.cols);
  const bool muon = f2 == 0.0 || f2 <= alpha * smin * s2;
  active[d.mat] = muon ? 1 : 0;
  skip[d.param] = muon ? 1 : 0;
  srank[d.mat] = f2 == 0.0 ? 0.0 : (s2 > 0.0 ? f2 / s2 : __longlong_as_double(0x7ff0000000000000ll));
}

template <int S, int TPB, int RB, bool VEC>
cudaError_t launch_one(const SrMat* mats, const SrItem* items, int nitems, int pass, bool last,
                       const unsigned* flags, cudaStream_t st) {
  auto kern = srank_pass_kernel<S, TPB, RB, VEC>;
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, TPB, 0);
  int grid = sms * (per_sm > 0 ? per_sm : 1);
  if (grid > nitems) grid = nitems;
  count_launch();
  kern<<<grid, TPB, 0, st>>>(mats, items, nitems, pass, last ? 1 : 0, flags);
  return cudaGetLastError();
}

template <bool VEC>
cudaError_t dispatch(int slots, int threads, const SrMat* mats, const SrItem* items, int nitems, int pass,
                     bool last, const unsigned* flags, cudaStream_t st) {
  // rows per batch: about 8 floats x 4 per thread in each of the two sets
  if (threads == 512) return launch_one<8, 512, 1, VEC>(mats, items, nitems, pass, last, flags, st);
  switch (slots) {
    case 1: return launch_one<1, 256, 8, VEC>(mats, items, nitems, pass, last, flags, st);
    case 2: return launch_one<2, 256, 4, VEC>(mats, items, nitems, pass, last, flags, st);
    case 3: return launch_one<3, 256, 2, VEC>(mats, items, nitems, pass, last, flags, st);
    case 4: return launch_one<4, 256, 2, VEC>(mats, items, nitems, pass, last, flags, st);
    case 5: return launch_one<5, 256, 1, VEC>(mats, items, nitems, pass, last, flags, st);
    case 6: return launch_one<6, 256, 1, VEC>(mats, items, nitems, pass, last, flags, st);
    case 7: return launch_one<7, 256, 1, VEC>(mats, items, nitems, pass, last, flags, st);
    case 8: return launch_one<8, 256, 1, VEC>(mats, items, nitems, pass, last, flags, st);
    default: return cudaErrorInvalidValue;
  }
}

template <int S, int RB, int NC = 8>
cudaError_t ring_launch(const SrMat* mats, const SrItem* items, int nitems, int pass, bool last, int max_cols,
                        unsigned* flags, uint64_t wait_ns, cudaStream_t st) {
  auto kern = srank_ring_kernel<S, RB, NC>;
  constexpr int kThreads = 32 * (NC + 1);   // NC consumer warps + 1 producer warp
  // three or four stages of RB rows (at most 32 KB each), four where they
  // fit the per-block budget: more rows in flight per block (a fifth stage
  // measured slower at 5120 columns)
  const int stride = (max_cols + 3) / 4 * 4;
  const size_t stage_bytes = (size_t)RB * stride * 4;
  const int nst = (int)std::min<size_t>(kRingMaxStages, std::max<size_t>(3, kRingBudget / stage_bytes));
  const size_t smem = (size_t)nst * stage_bytes;
  static bool attr_set[kMaxDevices] = {};   // per instantiation and device
  const int slot = device_slot();
  if (slot < 0 || !attr_set[slot]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (e != cudaSuccess) return e;
    if (slot >= 0) attr_set[slot] = true;
  }
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem);
  int grid = sms * (per_sm > 0 ? per_sm : 1);
  if (grid > nitems) grid = nitems;
  count_launch();
  kern<<<grid, kThreads, smem, st>>>(mats, items, nitems, pass, last ? 1 : 0, nst, stride, flags, wait_ns);
  return cudaGetLastError();
}

// Rows per stage for S slots of NC consumer warps: the largest of 1, 2, 3,
// 4, 6, 8 whose stage (rows of the full slot width, S * NC * 512 bytes) stays
// within 32 KB, so that three stages of two blocks fit an SM.
constexpr int ring_rows(int s, int nc) {
  return 64 / (s * nc) >= 8 ? 8 : 64 / (s * nc) >= 6 ? 6 : 64 / (s * nc) >= 4 ? 4
       : 64 / (s * nc) >= 3 ? 3 : 64 / (s * nc) >= 2 ? 2 : 1;
}

template <int S, int NC>
cudaError_t ring_go(const SrMat* mats, const SrItem* items, int nitems, int pass, bool last, int max_cols,
                    unsigned* flags, uint64_t wait_ns, cudaStream_t st) {
  return ring_launch<S, ring_rows(S, NC), NC>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
}

// Launch shape of the ring kernel for rows of max_cols columns, as
// (slots per thread S, consumer warps NC).
struct RingShape {
  int s, nc;
};
RingShape ring_shape(int max_cols) {
  // Six consumer warps for rows of at most 768 columns: every thread holds
  // a float4 (eight warps would leave a quarter of them idle at 768).
  if (max_cols <= 768) return {1, 6};
  // Ten consumer warps where they need fewer slots per thread than eight, up
  // to three slots (1280 columns: one float4 per thread instead of two for a
  // quarter of them); at 5120 columns four slots of ten warps measured no
  // faster than five of eight.
  const int s8 = (max_cols + 1023) / 1024, s10 = (max_cols + 1279) / 1280;
  if (s10 < s8 && s10 <= 3) return {s10, 10};
  return {s8 <= 6 ? s8 : s8 <= 8 ? 8 : s8 <= 12 ? 12 : 16, 8};
}

cudaError_t ring_dispatch(int max_cols, const SrMat* mats, const SrItem* items, int nitems, int pass, bool last,
                          unsigned* flags, uint64_t wait_ns, cudaStream_t st) {
  if (max_cols > 16 * 1024) return cudaErrorInvalidValue;
  const RingShape sh = ring_shape(max_cols);
  if (sh.nc == 6) return ring_go<1, 6>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
  if (sh.nc == 10) {
    switch (sh.s) {
      case 1: return ring_go<1, 10>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
      case 2: return ring_go<2, 10>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
      case 3: return ring_go<3, 10>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (sh.s) {
    case 1: return ring_go<1, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 2: return ring_go<2, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 3: return ring_go<3, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 4: return ring_go<4, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 5: return ring_go<5, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 6: return ring_go<6, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 8: return ring_go<8, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 12: return ring_go<12, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    case 16: return ring_go<16, 8>(mats, items, nitems, pass, last, max_cols, flags, wait_ns, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int srank_ring_shape(int64_t cols) {
  if (cols <= 0 || cols > 16 * 1024) return 0;
  const RingShape sh = ring_shape((int)cols);
  return sh.nc * 100 + sh.s;
}

cudaError_t launch_srank_ring(int max_cols, const SrMat* mats, const SrItem* items, int nitems, int pass, bool last,
                              unsigned* flags, uint64_t wait_ns, cudaStream_t st) {
  if (nitems <= 0) return cudaSuccess;
  return ring_dispatch(max_cols, mats, items, nitems, pass, last, flags, wait_ns, st);
}

int srank_slots(int64_t cols, int* threads) {
  if (cols <= 0) return 0;
  if (cols <= 8 * 1024) {
    *threads = 256;
    return (int)((cols + 1023) / 1024);
  }
  if (cols <= 8 * 2048) {
    *threads = 512;
    return 8;
  }
  return 0;
}

cudaError_t launch_srank_pass(int slots, int threads, bool vec4, const SrMat* mats, const SrItem* items,
                              int nitems, int pass, bool last, const unsigned* flags, cudaStream_t st) {
  if (nitems <= 0) return cudaSuccess;
  return vec4 ? dispatch<true>(slots, threads, mats, items, nitems, pass, last, flags, st)
              : dispatch<false>(slots, threads, mats, items, nitems, pass, last, flags, st);
}

cudaError_t launch_srank_decide(const SrMat* mats, int nmat, double alpha, int last_pass, unsigned char* active,
                                unsigned char* skip, double* srank, const unsigned* flags, cudaStream_t st) {
  if (nmat <= 0) return cudaSuccess;
  count_launch();
  srank_decide_kernel<<<(nmat + 127) / 128, 128, 0, st>>>(mats, nmat, alpha, last_pass, active, skip, srank, flags);
  return cudaGetLastError();
}

}  // namespace lm
