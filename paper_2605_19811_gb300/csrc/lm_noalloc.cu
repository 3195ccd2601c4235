// lm_msign_ns_noalloc: the Newton-Schulz msign approximation of lm_msign_ns,
// run in a fixed scratch area that is part of the library image instead of
// memory allocated per call.
//
// The scratch is a file-scope __device__ array of kNoAllocScratchBytes.  Every
// GPU that loads this library holds it until the process exits.  Host code
// cannot use the array's name as a device address (on the host it names a
// stand-in object), so the device address is looked up with
// cudaGetSymbolAddress, with that device current, on the first call made on
// that device, and cached together with the device's current context: a call
// that finds another context (the old one destroyed and a new one made, as
// by cudaDeviceReset, which reloads the module) looks the address up again.
//
// All calls share the array and it keeps what the last call left there: the
// parts that must start at zero (the padded X0 buffer, the norm accumulator,
// the status word) are cleared on every call, and calls whose GPU work
// overlaps (different streams, or different host threads, without ordering
// between them) race on it.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include <cudaTypedefs.h>

#include "lm_internal.h"

namespace lm {
namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)64 << 20;   // 64 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mu;
struct ScratchSlot {
  CUcontext ctx;   // context the address was looked up in
  char* addr;
};
ScratchSlot g_scratch[kMaxDevices] = {};

// The calling thread's current context (the device's primary context for
// runtime-API callers), through the driver entry point the runtime exposes.
CUcontext current_context() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static bool looked = false;
  if (!looked) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f);
    looked = true;
  }
  CUcontext c = nullptr;
  if (fn != nullptr && fn(&c) != CUDA_SUCCESS) c = nullptr;
  return c;
}

cudaError_t scratch_address(int dev, char** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  // the pointer checks before this made the device's context current
  const CUcontext ctx = current_context();
  ScratchSlot& sl = g_scratch[dev];
  if (sl.addr == nullptr || ctx == nullptr || sl.ctx != ctx) {   // no context handle: look up every call
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    sl.addr = static_cast<char*>(p);
    sl.ctx = ctx;
  }
  *out = sl.addr;
  return cudaSuccess;
}

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// Number of tiles of one Newton-Schulz phase for a single matrix, and the
// (tm, tn) of tile k in the same order the allocating path builds them
// (row-major; symmetric phases keep tiles that reach the diagonal).
__host__ __device__ inline int phase_tiles(int phase, int s_pad, int l_pad, int tall, int bm, int bn) {
  const int nrow = (phase == NS_APPLY && tall) ? l_pad : s_pad;
  const int ncol = phase == NS_APPLY ? (tall ? s_pad : l_pad) : s_pad;
  const int tms = (nrow + bm - 1) / bm;
  const int tns = (ncol + bn - 1) / bn;
  if (phase == NS_APPLY) return tms * tns;
  int n = 0;
  for (int tm = 0; tm < tms; ++tm)
    for (int tn = 0; tn < tns; ++tn)
      if ((int64_t)(tn + 1) * bn > (int64_t)tm * bm) ++n;
  return n;
}

struct BuildArgs {
  MatDesc mat;
  NsGroup group;
  MatDesc* d_mat;
  NsGroup* d_group;
  ElemChunk* d_chunks;
  int n_chunks;
  NsTile* d_tiles[3];
  int bm, bn;
  double* d_norm2;
  unsigned* d_flags;
};

// Writes the descriptor tables of one msign call into the scratch area.
__global__ void build_tables_kernel(BuildArgs a) {
  if (blockIdx.x != 0) return;
  if (threadIdx.x == 0) {
    *a.d_mat = a.mat;
    *a.d_group = a.group;
    *a.d_norm2 = 0.0;
    *a.d_flags = 0u;
  }
  const int64_t numel = a.mat.rows * a.mat.cols;
  for (int i = threadIdx.x; i < a.n_chunks; i += blockDim.x) {
    const int64_t b = (int64_t)i * kElemChunk;
    a.d_chunks[i] = ElemChunk{0, 0, b, numel - b < kElemChunk ? numel - b : kElemChunk};
  }
  if (threadIdx.x < 3) {
    const int ph = threadIdx.x;
    const NsGroup& g = a.group;
    const int nrow = (ph == NS_APPLY && g.tall) ? g.l_pad : g.s_pad;
    const int ncol = ph == NS_APPLY ? (g.tall ? g.s_pad : g.l_pad) : g.s_pad;
    const int tms = (nrow + a.bm - 1) / a.bm;
    const int tns = (ncol + a.bn - 1) / a.bn;
    int k = 0;
    for (int tm = 0; tm < tms; ++tm)
      for (int tn = 0; tn < tns; ++tn) {
        if (ph != NS_APPLY && (int64_t)(tn + 1) * a.bn <= (int64_t)tm * a.bm) continue;
        a.d_tiles[ph][k++] = NsTile{0, 0, (uint16_t)tm, (uint16_t)tn};
      }
  }
}

}  // namespace
}  // namespace lm

using namespace lm;

extern "C" lm_status lm_msign_ns_noalloc(const lm_tensor* in, lm_tensor* out, int steps, double a,
                                         double b, double c, double eps, int precision,
                                         void* cuda_stream) {
  if (in == nullptr || out == nullptr) return set_error(LM_ERR_INVALID_ARG, "in/out is NULL");
  for (const lm_tensor* t : {in, static_cast<const lm_tensor*>(out)}) {
    if (t->dtype != LM_BF16 && t->dtype != LM_F32) return set_error(LM_ERR_DTYPE, "unsupported dtype");
    if (t->rows < 2 || t->cols < 2) return set_error(LM_ERR_INVALID_ARG, "msign needs rows, cols >= 2");
    if (t->data == nullptr) return set_error(LM_ERR_INVALID_ARG, "NULL data");
    if (reinterpret_cast<uintptr_t>(t->data) % 16 != 0)
      return set_error(LM_ERR_ALIGN, "data pointer not 16-byte aligned");
  }
  if (out->rows != in->rows || out->cols != in->cols)
    return set_error(LM_ERR_INVALID_ARG, "out shape differs from in");
  if (steps < 0 || steps > 64) return set_error(LM_ERR_INVALID_ARG, "steps must be in [0, 64]");
  if (!std::isfinite(a) || !std::isfinite(b) || !std::isfinite(c) || !std::isfinite(eps) || eps < 0)
    return set_error(LM_ERR_INVALID_ARG, "coefficients must be finite, eps >= 0");
  if (precision != LM_BF16 && precision != LM_F32)
    return set_error(LM_ERR_INVALID_ARG, "precision must be LM_BF16 or LM_F32");
  if (in->rows > 65536 || in->cols > 65536)
    return set_error(LM_ERR_UNSUPPORTED, "lm_msign_ns_noalloc: matrix dimension above 65536");

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return set_error(LM_ERR_CUDA, "no CUDA device");
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return set_error(LM_ERR_UNSUPPORTED, "device is not sm_103");
  if (dev >= kMaxDevices) return set_error(LM_ERR_UNSUPPORTED, "device ordinal above 63");
  // in and out must be memory of this device (a host pointer would reach the kernels)
  for (const lm_tensor* t : {in, static_cast<const lm_tensor*>(out)}) {
    cudaPointerAttributes pa{};
    if (cudaPointerGetAttributes(&pa, t->data) != cudaSuccess) {
      cudaGetLastError();
      return set_error(LM_ERR_INVALID_ARG, "in/out is not a CUDA pointer");
    }
    if (!(pa.type == cudaMemoryTypeManaged || (pa.type == cudaMemoryTypeDevice && pa.device == dev)))
      return set_error(LM_ERR_INVALID_ARG, "in/out is not device memory of the current device");
  }

  // Layout of this call inside the scratch area.
  const lm_dtype xdt = precision == LM_F32 ? LM_F32 : LM_BF16;
  const int s = (int)std::min(in->rows, in->cols), l = (int)std::max(in->rows, in->cols);
  const int s_pad = xdt == LM_BF16 ? tc_pad_s(s) : simt_pad(s);
  const int l_pad = xdt == LM_BF16 ? tc_pad_l(l) : simt_pad(l);
  const int bm = xdt == LM_BF16 ? kTcBM : kSimtBM, bn = xdt == LM_BF16 ? kTcBN : kSimtBN;
  const size_t es = xdt == LM_BF16 ? 2 : 4;
  const int tall = in->rows > in->cols ? 1 : 0;
  const int64_t numel = in->rows * in->cols;
  const int n_et = (int)((numel + kElemChunk - 1) / kElemChunk);
  int ntiles[3];
  for (int ph = 0; ph < 3; ++ph) ntiles[ph] = phase_tiles(ph, s_pad, l_pad, tall, bm, bn);

  size_t off = 0;
  const size_t off_flags = off;   off = align256(off + sizeof(unsigned));
  const size_t off_norm = off;    off = align256(off + sizeof(double));
  const size_t off_mat = off;     off = align256(off + sizeof(MatDesc));
  const size_t off_group = off;   off = align256(off + sizeof(NsGroup));
  const size_t off_et = off;      off = align256(off + (size_t)n_et * sizeof(ElemChunk));
  size_t off_tiles[3];
  for (int ph = 0; ph < 3; ++ph) {
    off_tiles[ph] = off;
    off = align256(off + (size_t)ntiles[ph] * sizeof(NsTile));
  }
  const size_t xbytes = (size_t)s_pad * l_pad * es, abytes = (size_t)s_pad * s_pad * es;
  const size_t off_x0 = off;  off = align256(off + xbytes);
  const size_t off_x1 = off;  off = align256(off + xbytes);
  const size_t off_a = off;   off = align256(off + abytes);
  const size_t off_b = off;   off = align256(off + abytes);
  if (off > kNoAllocScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "lm_msign_ns_noalloc: a %lldx%lld matrix needs %zu bytes of scratch; the limit is %zu "
             "(64 MiB)", (long long)in->rows, (long long)in->cols, off, kNoAllocScratchBytes);
    return set_error(LM_ERR_UNSUPPORTED, msg);
  }

  char* base = nullptr;
  cudaError_t e = scratch_address(dev, &base);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);

  NsGroup g;
  memset(&g, 0, sizeof(g));
  g.count = 1;
  g.s = s;
  g.l = l;
  g.s_pad = s_pad;
  g.l_pad = l_pad;
  g.first_mat = 0;
  g.tall = tall;
  g.X[0] = base + off_x0;
  g.X[1] = base + off_x1;
  g.A = base + off_a;
  g.B = base + off_b;

  BuildArgs ba;
  memset(&ba, 0, sizeof(ba));
  MatDesc& d = ba.mat;
  d.w = in->data;
  d.m = nullptr;
  d.x = g.X[0];
  d.x_final = g.X[steps & 1];
  d.out = out->data;
  d.norm2 = reinterpret_cast<double*>(base + off_norm);
  d.rows = in->rows;
  d.cols = in->cols;
  d.ldx = tall ? s_pad : l_pad;
  d.grad_slot = 0;
  d.wdt = in->dtype;
  d.odt = out->dtype;
  d.shape_scale = 1.f;
  ba.group = g;
  ba.d_mat = reinterpret_cast<MatDesc*>(base + off_mat);
  ba.d_group = reinterpret_cast<NsGroup*>(base + off_group);
  ba.d_chunks = reinterpret_cast<ElemChunk*>(base + off_et);
  ba.n_chunks = n_et;
  for (int ph = 0; ph < 3; ++ph) ba.d_tiles[ph] = reinterpret_cast<NsTile*>(base + off_tiles[ph]);
  ba.bm = bm;
  ba.bn = bn;
  ba.d_norm2 = d.norm2;
  ba.d_flags = reinterpret_cast<unsigned*>(base + off_flags);

  TcGroupMaps maps;
  if (xdt == LM_BF16) {
    e = tc_encode_group_maps(g, &maps);
    if (e != cudaSuccess) return set_error(LM_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  }

  // X0's padding must read as zero; the other buffers are fully written
  // before they are read.
  e = cudaMemsetAsync(g.X[0], 0, xbytes, stream);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  count_launch();
  build_tables_kernel<<<1, 256, 0, stream>>>(ba);
  if ((e = cudaGetLastError()) != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));

  MuonConsts mk;
  memset(&mk, 0, sizeof(mk));
  mk.eps = (float)eps;
  mk.ns_steps = steps;
  mk.flags = ba.d_flags;
  e = launch_momentum_norm(xdt, in->dtype, ba.d_mat, ba.d_chunks, n_et, nullptr, mk, 1, stream);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  const NsCoeffs co{(float)a, (float)b, (float)c, (float)eps};
  // c = 0 (a cubic): B = b A is not formed, APPLY reads A and scales by b;
  // otherwise, where |a| < 4, a is folded into B's diagonal (as lm_msign_ns
  // does, unless LM_NS_FOLD=0)
  const bool from_a = xdt == LM_BF16 && co.c == 0.f;
  const char* fold_env = std::getenv("LM_NS_FOLD");
  const bool fold = xdt == LM_BF16 && !from_a && std::fabs(co.a) < 4.f &&
                    !(fold_env != nullptr && std::strcmp(fold_env, "0") == 0);
  for (int it = 0; it < steps; ++it)
    for (int ph = 0; ph < 3; ++ph) {
      if (ph == NS_POLY && from_a) continue;
      if (xdt == LM_BF16)
        e = launch_ns_tc((NsPhase)ph, it, 1, &g, &maps, ba.d_tiles[ph], ntiles[ph], nullptr, 0,
                         d.norm2, co, ba.d_flags, nullptr, stream, nullptr, nullptr, 1, 0, false, false,
                         env_wait_limit_ns(), ph == NS_APPLY && from_a, ph != NS_GRAM && fold);
      else
        e = launch_ns_simt((NsPhase)ph, it, 1, ba.d_group, ba.d_tiles[ph], ntiles[ph], d.norm2, co,
                           stream, nullptr, nullptr, ba.d_flags);
      if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
    }
  e = launch_finalize(xdt, out->dtype, ba.d_mat, ba.d_chunks, n_et, mk, 1, ba.d_flags, stream);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  return LM_OK;
}

extern "C" lm_status lm_msign_ns_noalloc_status(uint32_t* device_flags, void* cuda_stream) {
  if (device_flags == nullptr) return set_error(LM_ERR_INVALID_ARG, "device_flags is NULL");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return set_error(LM_ERR_CUDA, "no CUDA device");
  if (dev >= kMaxDevices) return set_error(LM_ERR_UNSUPPORTED, "device ordinal above 63");
  char* base = nullptr;
  cudaError_t e = scratch_address(dev, &base);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  unsigned h = 0;   // the status word sits at offset 0 of every call's layout
  e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess) e = cudaMemcpy(&h, base, sizeof(unsigned), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return set_error(LM_ERR_CUDA, cudaGetErrorString(e));
  *device_flags = h;
  if (h & LM_FLAG_TIMEOUT)
    return set_error(LM_ERR_TIMEOUT, "a bounded device wait of the last lm_msign_ns_noalloc call gave up");
  return LM_OK;
}
